// egmla_aux.cu - the small kernels around the tensor-core decode kernel:
//   append_latent_kernel   cache write of the new token (bit-exact copy)
//   prologue_*_kernel      per-step query absorption q^ = W_UK,h^T q^C, the
//                          page prefix sums and split start records of the
//                          split-KV schedule, and (in eg_mla_step) the append
//   combine_kernel         log-sum-exp merge of the split partials and the
//                          W_UV,h up-projection of the latent output, for the
//                          launches whose decode kernel does not fuse it
//   decode_f32_kernel      the fp32 specialisation of the split-KV decode
//                          (exact fp32 arithmetic on CUDA cores; bf16 runs on
//                          tcgen05 in egmla_decode_tc.cu)
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <cmath>
#include <cstdint>
#include <cstring>

#include "egmla_common.cuh"
#include "egmla_kernels.h"
#include "egmla_ptx.cuh"

namespace egmla {

// ------------------------------------------------------------------ append
// The new token's rows of sequence b, copied by the calling block; the row
// copies are 16-byte vectors (the row byte counts allow it for every
// supported shape).
__device__ void append_row(const AppendArgs& a, int b) {
  const int pos = a.positions[b];
  if (pos < 0) return;
  const int lp = pos / a.page_size;
  if (lp >= a.max_pages) {
    if (threadIdx.x == 0) report_status(a.status, kStatusOutOfRange);
    return;
  }
  const int page = a.block_table[static_cast<size_t>(b) * a.max_pages + lp];
  if (page < 0 || page >= a.num_pages) {
    if (threadIdx.x == 0) report_status(a.status, kStatusOutOfRange);
    return;
  }
  const size_t row = static_cast<size_t>(page) * a.page_size + pos % a.page_size;
  uint4* cd = reinterpret_cast<uint4*>(static_cast<uint8_t*>(a.c_pool) + row * a.c_row_bytes);
  const uint4* cs = reinterpret_cast<const uint4*>(static_cast<const uint8_t*>(a.c_new) +
                                                   static_cast<size_t>(b) * a.c_row_bytes);
  for (int i = threadIdx.x; i < a.c_row_bytes / 16; i += blockDim.x) cd[i] = cs[i];
  uint4* kd = reinterpret_cast<uint4*>(static_cast<uint8_t*>(a.kr_pool) + row * a.kr_row_bytes);
  const uint4* ks = reinterpret_cast<const uint4*>(static_cast<const uint8_t*>(a.kr_new) +
                                                   static_cast<size_t>(b) * a.kr_row_bytes);
  for (int i = threadIdx.x; i < a.kr_row_bytes / 16; i += blockDim.x) kd[i] = ks[i];
  if (a.id_pool != nullptr && a.ids_new != nullptr && threadIdx.x == 0) a.id_pool[row] = a.ids_new[b];
}

// one block per sequence
__global__ void append_latent_kernel(const AppendArgs a) { append_row(a, blockIdx.x); }

// ------------------------------------------------------------------ helpers
// eight bf16 (or four fp32) of a 16-byte piece as floats
__device__ __forceinline__ void unpack16(const uint4& raw, float (&w)[8]) {
  const __nv_bfloat162* e = reinterpret_cast<const __nv_bfloat162*>(&raw);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const float2 f = __bfloat1622float2(e[i]);
    w[2 * i] = f.x;
    w[2 * i + 1] = f.y;
  }
}
__device__ __forceinline__ void unpack16(const uint4& raw, float (&w)[4]) {
  w[0] = __uint_as_float(raw.x);
  w[1] = __uint_as_float(raw.y);
  w[2] = __uint_as_float(raw.z);
  w[3] = __uint_as_float(raw.w);
}

// ------------------------------------------------------------------ prologue
// Exclusive prefix sum of the schedule units per sequence (its pages plus
// kSegCost when it has any): cu[b] = sum_{b'<b} units_b', cu[batch] = total; a
// scan by the block's first warp, 32 sequences per pass.
__device__ void page_prefix_sums(const int32_t* seq_lens, int batch, int page_size, int32_t* cu) {
  if (threadIdx.x >= 32) return;
  const int lane = threadIdx.x;
  int32_t carry = 0;
  for (int base = 0; base < batch; base += 32) {
    const int b = base + lane;
    const int L = b < batch ? seq_lens[b] : 0;
    const int np = L > 0 ? (L + page_size - 1) / page_size + kSegCost : 0;
    int incl = np;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int t = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += t;
    }
    if (b < batch) cu[b] = carry + incl - np;
    carry += __shfl_sync(0xffffffffu, incl, 31);
  }
  if (lane == 0) cu[batch] = carry;
}

// The same prefix sums by a whole block of 256 threads (a warp scan per 256
// sequences, the warps' totals through shared memory), written to global
// memory and to the block's shared copy cu_s (batch + 1 entries); one load
// round trip per 256 sequences.
__device__ void page_prefix_sums_block(const int32_t* seq_lens, int batch, int page_size, int32_t* cu,
                                       int32_t* cu_s, int32_t* wsum) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5, nw = blockDim.x / 32;
  int32_t carry = 0;
  for (int base = 0; base < batch; base += blockDim.x) {
    const int b = base + tid;
    const int L = b < batch ? seq_lens[b] : 0;
    const int np = L > 0 ? (L + page_size - 1) / page_size + kSegCost : 0;
    int incl = np;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int t = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += t;
    }
    if (lane == 31) wsum[warp] = incl;
    __syncthreads();
    int before = 0, total = 0;
    for (int w = 0; w < nw; ++w) {
      const int v = wsum[w];
      before += w < warp ? v : 0;
      total += v;
    }
    if (b < batch) {
      const int32_t e = carry + before + incl - np;
      cu[b] = e;
      cu_s[b] = e;
    }
    carry += total;
    __syncthreads();   // wsum is rewritten by the next pass
  }
  if (tid == 0) {
    cu[batch] = carry;
    cu_s[batch] = carry;
  }
}

// Start record of every split (see SplitStart), from the prefix sums this
// block just wrote (its shared copy).  Split c
// owns units [c chunk, (c + 1) chunk); its first sequence is the last one whose
// first unit is at most c chunk (empty sequences skipped), as in the decode
// kernel's walk.
__device__ void split_starts(const int32_t* cu, const int32_t* seq_lens, int batch, int num_splits,
                             const int32_t* __restrict__ block_table, int max_pages, SplitStart* starts) {
  const int total = cu[batch];
  const int chunk = split_chunk(total, num_splits);
  for (int c = threadIdx.x; c < num_splits; c += blockDim.x) {
    SplitStart st;
    const int g0 = c * chunk;
    st.g1 = min(g0 + chunk, total);
    st.b = st.lp = st.lp_end = st.L = st.npages = st.pad = 0;
    st.done = g0 >= st.g1;
    if (!st.done) {
      int lo = 0, hi = batch - 1;
      while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (cu[mid] <= g0) lo = mid; else hi = mid - 1;
      }
      while (lo < batch - 1 && cu[lo + 1] <= g0) ++lo;
      const int base = cu[lo] + kSegCost;   // unit of the sequence's first page
      st.b = lo;
      st.lp = max(g0 - base, 0);
      st.lp_end = min(st.g1, cu[lo + 1]) - base;
      st.L = seq_lens[lo];
      st.done = st.lp_end <= st.lp;
      if (!st.done) st.npages = min(kStartPages, min(st.lp_end, max_pages) - st.lp);
    }
    for (int i = 0; i < kStartPages; ++i)
      st.page[i] = i < st.npages ? block_table[static_cast<size_t>(st.b) * max_pages + st.lp + i] : -1;
    const int4* src = reinterpret_cast<const int4*>(&st);
    int4* dst = reinterpret_cast<int4*>(starts + c);
#pragma unroll
    for (int k = 0; k < 4; ++k) dst[k] = src[k];
  }
}

// Tensor-core path: block (head h, chunk of kSumFeatures = 32 latent features,
// group of up to kPBatch sequences) computes q^_{b,h}[f] = sum_n W_UK,h[n][f] q^C_{b,h}[n]
// in fp32 and stores (q^ (*) gamma) rounded to bf16 in the prepared query
// block (qop_offset layout).  Its per-chunk partials of w_h = sum_f bf16(q^ gamma)_f
// and b_h = q^_h . beta go to the block's slots of the sums area.  Chunk-0
// blocks also copy q^R.  Block 0 computes the page prefix sums and the
// splits' start records.
//  - All 16-byte global loads of a thread are issued before any is stored
//    (W_UK with an L2 evict-last hint: it stays in L2 across steps).
//  - W_UK (bf16) and q^C (converted to fp32 once, as it is staged) are held
//    row-major; a warp takes a quad of sequences and a part of the n range,
//    reading per 8 n the lane's feature of 8 W rows and 8 n of each q^C row
//    (two 16-byte broadcasts per sequence) for 32 FMAs.  With few sequences
//    the spare warps split n further; the parts are added in shared memory.
constexpr int kPBatch = 32;
constexpr int kPMaxNope = 256;
constexpr int kPThreads = 256;
constexpr int kPLoads = kPMaxNope * kSumFeatures * 2 / 16 / kPThreads;   // 16-byte pieces per thread and array

// (no launch bound: with one, ptxas trims the kernel to 48 registers and spills)
__global__ void prologue_tc_kernel(const __nv_bfloat16* __restrict__ q, const __nv_bfloat16* __restrict__ w_uk,
                       const float* __restrict__ gamma, const float* __restrict__ beta,
                       const int32_t* __restrict__ seq_lens, int batch, int d_nope, int d_rope, int d_c,
                       int page_size, uint8_t* __restrict__ qprep, size_t qstride, int32_t* __restrict__ cu,
                       uint32_t* __restrict__ seq_done, int num_splits, const int32_t* __restrict__ block_table,
                       int max_pages, SplitStart* __restrict__ starts, const AppendArgs app) {
  __shared__ __align__(16) __nv_bfloat16 ws[kPMaxNope][kSumFeatures];  // W_UK,h[n][f0 + f]
  __shared__ __align__(16) float qs[kPBatch][kPMaxNope];              // q^C_{b0 + j, h}[n]
  // partial sums [n part * 4 quads + j][f], written once every warp is done with ws
  float (*red)[kSumFeatures] = reinterpret_cast<float (*)[kSumFeatures]>(&ws[0][0]);
  static_assert(sizeof(ws) >= 32 * kSumFeatures * sizeof(float), "reduction buffer aliases ws");
  constexpr int H = 16;
  const int nchunk = d_c / kSumFeatures;
  const int ngroups = (batch + kPBatch - 1) / kPBatch;
  // the decode kernel after this one may begin its setup (it waits for this
  // kernel's completion before it reads anything written here)
  grid_launch_dependents();
  // block 0: the schedule (dispatched first, so that it never waits for a
  // second wave of the grid); blocks 1 .. A: the absorption items; then the
  // append blocks
  const int nabs = H * nchunk * ngroups;
  if (blockIdx.x > static_cast<unsigned>(nabs)) {
    // blocks after the schedule block: the new token of one sequence (a step
    // that appends before it attends); no block of this kernel reads the pools
    append_row(app, blockIdx.x - (nabs + 1));
    return;
  }
  if (blockIdx.x == 0) {
    if (seq_done != nullptr)
      for (int i = threadIdx.x; i <= batch; i += blockDim.x) seq_done[i] = 0u;
    // the prefix sums in shared memory too (the W_UK staging area is idle in
    // this block), so that the splits' searches read them there
    int32_t* cu_s = reinterpret_cast<int32_t*>(&ws[0][0]);
    int32_t* wsum = reinterpret_cast<int32_t*>(&qs[0][0]);
    constexpr int kCuSmem = static_cast<int>(sizeof(ws) / sizeof(int32_t));
    if (batch + 1 <= kCuSmem) {
      page_prefix_sums_block(seq_lens, batch, page_size, cu, cu_s, wsum);
      __syncthreads();   // the prefix sums are visible to the whole block
      split_starts(cu_s, seq_lens, batch, num_splits, block_table, max_pages, starts);
    } else {
      page_prefix_sums(seq_lens, batch, page_size, cu);
      __syncthreads();
      split_starts(cu, seq_lens, batch, num_splits, block_table, max_pages, starts);
    }
    return;
  }
  if (q == nullptr) return;  // cache-read test entry: prefix sums only
  const int item = static_cast<int>(blockIdx.x) - 1;
  const int h = item % H, fc = (item / H) % nchunk, bg = item / (H * nchunk);
  const int b0 = bg * kPBatch, nb = min(kPBatch, batch - b0);
  const int f0 = fc * kSumFeatures;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int qrow = d_nope + d_rope;
  // W piece i: row n = i / 4, features 8 (i % 4) ..; q piece i: sequence j = i / (d_nope / 8), columns 8 (i % ..)
  const int wpieces = d_nope * (kSumFeatures / 8), qpr = d_nope / 8, qpieces = kPBatch * qpr;
  const uint64_t keep = policy_evict_last();
  uint4 wv[kPLoads], qv[kPLoads];
#pragma unroll
  for (int k = 0; k < kPLoads; ++k) {
    const int i = tid + k * kPThreads;
    wv[k] = make_uint4(0, 0, 0, 0);
    qv[k] = make_uint4(0, 0, 0, 0);
    if (i < wpieces)
      wv[k] = ldg_16_na_hint(w_uk + (static_cast<size_t>(h) * d_nope + i / 4) * d_c + f0 + 8 * (i % 4), keep);
    if (i < qpieces && i / qpr < nb)
      qv[k] = *reinterpret_cast<const uint4*>(q + (static_cast<size_t>(b0 + i / qpr) * H + h) * qrow + 8 * (i % qpr));
  }
#pragma unroll
  for (int k = 0; k < kPLoads; ++k) {
    const int i = tid + k * kPThreads;
    if (i < wpieces) *reinterpret_cast<uint4*>(&ws[i / 4][8 * (i % 4)]) = wv[k];
    if (i < qpieces) {
      float x[8];
      unpack16(qv[k], x);
      float4* d = reinterpret_cast<float4*>(&qs[i / qpr][8 * (i % qpr)]);
      d[0] = make_float4(x[0], x[1], x[2], x[3]);
      d[1] = make_float4(x[4], x[5], x[6], x[7]);
    }
  }
  __syncthreads();
  // warp -> (sequence quad sq, n part kp); nq quads, ks parts of the n range
  const int nq = (nb + 3) / 4, nblk = d_nope / 8;
  int ks = 8 / nq;
  ks = ks >= 8 ? 8 : ks >= 4 ? 4 : ks >= 2 ? 2 : 1;
  while (nblk % ks) ks >>= 1;
  float acc[4] = {0.f, 0.f, 0.f, 0.f};
  const int sq = warp % nq, kp = warp / nq, bpk = nblk / ks;
  if (warp < nq * ks) {
    for (int blk = kp * bpk; blk < (kp + 1) * bpk; ++blk) {
      float w[8];
#pragma unroll
      for (int e = 0; e < 8; ++e) w[e] = __bfloat162float(ws[blk * 8 + e][lane]);
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const float4 x0 = *reinterpret_cast<const float4*>(&qs[4 * sq + i][blk * 8]);
        const float4 x1 = *reinterpret_cast<const float4*>(&qs[4 * sq + i][blk * 8 + 4]);
        acc[i] = fmaf(w[0], x0.x, acc[i]);
        acc[i] = fmaf(w[1], x0.y, acc[i]);
        acc[i] = fmaf(w[2], x0.z, acc[i]);
        acc[i] = fmaf(w[3], x0.w, acc[i]);
        acc[i] = fmaf(w[4], x1.x, acc[i]);
        acc[i] = fmaf(w[5], x1.y, acc[i]);
        acc[i] = fmaf(w[6], x1.z, acc[i]);
        acc[i] = fmaf(w[7], x1.w, acc[i]);
      }
    }
  }
  const int f = f0 + lane;
  const float gm = gamma ? gamma[f] : 1.f;
  const float bt = beta ? beta[f] : 0.f;
  // q^ of sequence j (its 32 features over the warp's lanes) -> prepared query block
  auto emit = [&](int j, float a) {
    const __nv_bfloat16 bq = __float2bfloat16_rn(a * gm);
    float wpart = __bfloat162float(bq), bpart = a * bt;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      wpart += __shfl_xor_sync(0xffffffffu, wpart, o);
      bpart += __shfl_xor_sync(0xffffffffu, bpart, o);
    }
    uint8_t* qb = qprep + static_cast<size_t>(b0 + j) * qstride;
    *reinterpret_cast<__nv_bfloat16*>(qb + qop_offset(h, f)) = bq;
    if (lane == 0) {
      float* sums = reinterpret_cast<float*>(qb + qprep_lat_bytes(d_c) + qprep_rope_bytes(d_rope));
      sums[(fc * 2) * 16 + h] = wpart;
      sums[(fc * 2 + 1) * 16 + h] = bpart;
    }
  };
  if (ks == 1) {
    // each warp holds whole sums: emit from registers
    if (warp < nq) {
#pragma unroll
      for (int i = 0; i < 4; ++i)
        if (4 * sq + i < nb) emit(4 * sq + i, acc[i]);
    }
  } else {
    __syncthreads();   // every warp is done with ws, which red aliases
    if (warp < nq * ks) {
#pragma unroll
      for (int i = 0; i < 4; ++i) red[kp * 4 * nq + 4 * sq + i][lane] = acc[i];
    }
    __syncthreads();
    for (int j = warp; j < nb; j += kPThreads / 32) {
      float a = 0.f;
      for (int k = 0; k < ks; ++k) a += red[k * 4 * nq + j][lane];
      emit(j, a);
    }
  }
  if (fc == 0) {
    for (int i = tid; i < nb * d_rope; i += kPThreads) {
      const int j = i / d_rope, r = i % d_rope;
      *reinterpret_cast<__nv_bfloat16*>(qprep + static_cast<size_t>(b0 + j) * qstride + qprep_lat_bytes(d_c) +
                                        qop_offset(h, r)) = q[(static_cast<size_t>(b0 + j) * H + h) * qrow + d_nope + r];
    }
  }
}

// fp32 path: q^ [H, d_c] and q^R [H, d_rope] in fp32, row-major.
__global__ void prologue_f32_kernel(const float* __restrict__ q, const float* __restrict__ w_uk,
                                    const int32_t* __restrict__ seq_lens, int batch, int H, int d_nope,
                                    int d_rope, int d_c, int page_size, uint8_t* __restrict__ qprep,
                                    size_t qstride, int32_t* __restrict__ cu) {
  __shared__ float qn[256];
  if (blockIdx.x == static_cast<unsigned>(batch * H)) {
    page_prefix_sums(seq_lens, batch, page_size, cu);
    return;
  }
  const int b = blockIdx.x / H, h = blockIdx.x % H;
  const float* qv = q + (static_cast<size_t>(b) * H + h) * (d_nope + d_rope);
  for (int n = threadIdx.x; n < d_nope; n += blockDim.x) qn[n] = qv[n];
  __syncthreads();
  float* qh = reinterpret_cast<float*>(qprep + static_cast<size_t>(b) * qstride);
  const float* w = w_uk + static_cast<size_t>(h) * d_nope * d_c;
  for (int f = threadIdx.x; f < d_c; f += blockDim.x) {
    float acc = 0.f;
    for (int n = 0; n < d_nope; ++n) acc = fmaf(w[static_cast<size_t>(n) * d_c + f], qn[n], acc);
    qh[static_cast<size_t>(h) * d_c + f] = acc;
  }
  float* qr = qh + static_cast<size_t>(H) * d_c;
  for (int r = threadIdx.x; r < d_rope; r += blockDim.x) qr[static_cast<size_t>(h) * d_rope + r] = qv[d_nope + r];
}

// ------------------------------------------------------------------ combine
template <typename T>
__device__ __forceinline__ float to_f(T v);
template <>
__device__ __forceinline__ float to_f<float>(float v) { return v; }
template <>
__device__ __forceinline__ float to_f<__nv_bfloat16>(__nv_bfloat16 v) { return __bfloat162float(v); }
template <typename T>
__device__ __forceinline__ T from_f(float v);
template <>
__device__ __forceinline__ float from_f<float>(float v) { return v; }
template <>
__device__ __forceinline__ __nv_bfloat16 from_f<__nv_bfloat16>(float v) { return __float2bfloat16_rn(v); }

// Block per (head h, group of kCombineGroup sequences), 256 threads: the
// sequences of a group share one pass over W_UV,h.  The splits that covered
// sequence b are the CTAs c0..c1 of the page schedule; their partials sit in
// slots c + b.  M = max_s m_s; o = sum_s 2^(m_s - M) O_s / sum_s 2^(m_s - M)
// l_s (m in log2 units); then u = W_UV,h o.  A sequence of length 0 gets
// u = 0.
//  - merge: warp j takes sequence b0 + j: lane k holds slot k's (m, l) of
//    each group of 32 slots, and every lane the O values of its features
//    (f = lane + 32 i) for one slot at a time, the slot's weight broadcast
//    from the lane that holds it;
//  - u: warp w takes groups of four W_UV,h rows; a lane loads its 16-byte
//    pieces of the four rows once and multiplies them into all the group's
//    merged vectors (shared memory), then the 32 sums (sequence, row) are
//    reduced across the lanes by a transposing butterfly (31 shuffles), after
//    which lane t holds sequence t / 4, row t % 4.
constexpr int kCombineThreads = 256;
constexpr int kCombineGroup = 8;        // sequences per block (one warp each in the merge)
constexpr int kCombineMaxDc = 512;
constexpr int kCombineFeat = kCombineMaxDc / 32;   // features per lane in the merge, at most

// v[i] (i < 32) summed over the warp; lane t returns the sum of v[t]
__device__ __forceinline__ float reduce32_transpose(float (&v)[32], int lane) {
#pragma unroll
  for (int o = 16, len = 32; o > 0; o >>= 1, len >>= 1) {
    const bool up = (lane & o) != 0;
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      if (i < len / 2) {
        const float keep = up ? v[i + len / 2] : v[i];
        const float send = up ? v[i] : v[i + len / 2];
        v[i] = keep + __shfl_xor_sync(0xffffffffu, send, o);
      }
    }
  }
  return v[0];
}

template <typename T>
__global__ void __launch_bounds__(kCombineThreads)
combine_kernel(const int32_t* __restrict__ cu, const float* __restrict__ part_ml, const float* __restrict__ part_o,
               const T* __restrict__ w_uv, T* __restrict__ out, int batch, int H, int d_c, int d_v,
               int num_splits) {
  __shared__ __align__(16) float olat[kCombineGroup][kCombineMaxDc];
  const int h = blockIdx.x % H, b0 = (blockIdx.x / H) * kCombineGroup;
  const int nb = min(kCombineGroup, batch - b0);
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  constexpr int kWarps = kCombineThreads / 32;
  const int total = cu[batch];
  const int chunk = split_chunk(total, num_splits);
  if (warp < nb) {
    const int b = b0 + warp;
    const int p0 = cu[b] + kSegCost, p1 = cu[b + 1];   // units of the sequence's pages
    const int c0 = p0 / chunk;
    const int n = p1 > p0 ? (p1 - 1) / chunk - c0 + 1 : 0;
    float* ol = olat[warp];
    if (n == 0) {
      for (int f = lane; f < d_c; f += 32) ol[f] = 0.f;
    } else {
      const size_t mlstride = static_cast<size_t>(H) * 2, sstride = static_cast<size_t>(H) * d_c;
      const float* pml = part_ml + (static_cast<size_t>(c0 + b) * H + h) * 2;
      const float* po = part_o + (static_cast<size_t>(c0 + b) * H + h) * d_c;
      float M = -INFINITY;
      for (int k = lane; k < n; k += 32) M = fmaxf(M, pml[k * mlstride]);
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, o));
      float acc[kCombineFeat];
#pragma unroll
      for (int i = 0; i < kCombineFeat; ++i) acc[i] = 0.f;
      float lsum = 0.f;
      for (int k0 = 0; k0 < n; k0 += 32) {
        const int kn = min(32, n - k0);
        float wk = 0.f;
        if (lane < kn) {
          const float2 ml = *reinterpret_cast<const float2*>(pml + (k0 + lane) * mlstride);
          wk = exp2f(ml.x - M);
          lsum = fmaf(wk, ml.y, lsum);
        }
#pragma unroll 2
        for (int kk = 0; kk < kn; ++kk) {
          const float w = __shfl_sync(0xffffffffu, wk, kk);
          const float* ps = po + (k0 + kk) * sstride;
#pragma unroll
          for (int i = 0; i < kCombineFeat; ++i) {
            const int f = lane + 32 * i;
            if (f < d_c) acc[i] = fmaf(w, ps[f], acc[i]);
          }
        }
      }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) lsum += __shfl_xor_sync(0xffffffffu, lsum, o);
      const float invL = 1.f / lsum;
#pragma unroll
      for (int i = 0; i < kCombineFeat; ++i) {
        const int f = lane + 32 * i;
        if (f < d_c) ol[f] = acc[i] * invL;
      }
    }
  }
  __syncthreads();
  // u[j][v] = sum_f W_UV[h][v][f] olat[j][f]
  constexpr int VEC = 16 / sizeof(T);
  const int npieces = d_c / VEC;   // d_c is a multiple of VEC for both element types
  const T* wh = w_uv + static_cast<size_t>(h) * d_v * d_c;
  for (int v0 = 4 * warp; v0 < d_v; v0 += 4 * kWarps) {
    float acc[32];
#pragma unroll
    for (int i = 0; i < 32; ++i) acc[i] = 0.f;
    for (int pc = lane; pc < npieces; pc += 32) {
      float wf[4][VEC];
#pragma unroll
      for (int r = 0; r < 4; ++r) {
        uint4 raw = make_uint4(0, 0, 0, 0);
        if (v0 + r < d_v) raw = *reinterpret_cast<const uint4*>(wh + static_cast<size_t>(v0 + r) * d_c + pc * VEC);
        const T* e = reinterpret_cast<const T*>(&raw);
#pragma unroll
        for (int i = 0; i < VEC; ++i) wf[r][i] = to_f<T>(e[i]);
      }
#pragma unroll
      for (int j = 0; j < kCombineGroup; ++j) {
        if (j < nb) {
          float o[VEC];
#pragma unroll
          for (int i = 0; i < VEC; i += 4) {
            const float4 q = *reinterpret_cast<const float4*>(&olat[j][pc * VEC + i]);
            o[i] = q.x;
            o[i + 1] = q.y;
            o[i + 2] = q.z;
            o[i + 3] = q.w;
          }
#pragma unroll
          for (int r = 0; r < 4; ++r)
#pragma unroll
            for (int i = 0; i < VEC; ++i) acc[4 * j + r] = fmaf(wf[r][i], o[i], acc[4 * j + r]);
        }
      }
    }
    const float sum = reduce32_transpose(acc, lane);
    const int j = lane >> 2, v = v0 + (lane & 3);
    if (j < nb && v < d_v) out[(static_cast<size_t>(b0 + j) * H + h) * d_v + v] = from_f<T>(sum);
  }
}

// ------------------------------------------------------------------ fp32 decode
// One block per split, 128 threads.  Each cached token of the block's page
// range is processed in order: c~ = LN(c (*) G[id]) with a two-pass mean and
// variance, per-head scores against q^ and q^R, online softmax, and the
// running latent output sum_j p_j c~_j.  Writes the same partials as the
// tensor-core kernel.
constexpr int kF32Threads = 128;

__device__ __forceinline__ float block_sum_128(float v, float* red, int slot) {
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  if ((threadIdx.x & 31) == 0) red[slot * 4 + (threadIdx.x >> 5)] = v;
  __syncthreads();
  const float s = red[slot * 4] + red[slot * 4 + 1] + red[slot * 4 + 2] + red[slot * 4 + 3];
  __syncthreads();
  return s;
}

__global__ void __launch_bounds__(kF32Threads)
decode_f32_kernel(const float* __restrict__ c_pool, const float* __restrict__ kr_pool,
                  const int32_t* __restrict__ id_pool, const int32_t* __restrict__ block_table,
                  int max_pages, const int32_t* __restrict__ seq_lens, int batch, int num_pages,
                  const float* __restrict__ gate_table, const float* __restrict__ gamma,
                  const float* __restrict__ beta, const uint8_t* __restrict__ qprep, size_t qstride,
                  const int32_t* __restrict__ cu, float* __restrict__ part_ml, float* __restrict__ part_o,
                  int H, int d_c, int d_rope, int vocab, int gate, int gate_add, int gate_ln, float scale_log2,
                  float eps,
                  int32_t* status) {
  extern __shared__ float sm[];
  float* qh = sm;                               // [H][d_c]
  float* qr = qh + H * d_c;                     // [H][d_rope]
  float* acc = qr + H * d_rope;                 // [H][d_c]
  float* ct = acc + H * d_c;                    // [d_c]
  float* krs = ct + d_c;                        // [d_rope]
  float* red = krs + 64;                        // [20][4]
  __shared__ float mrun[16], lrun[16], pcur[16], alph[16];

  const int total = cu[batch];
  const int chunk = split_chunk(total, gridDim.x);
  const int g0 = blockIdx.x * chunk;
  const int g1 = min(g0 + chunk, total);
  if (g0 >= g1) return;
  int b = find_sequence(cu, batch, g0);
  int g = g0;
  while (g < g1) {
    const int pend = min(g1, cu[b + 1]);
    const int L = seq_lens[b];
    const int s = cu[b] + kSegCost;   // unit of the sequence's first page
    const int tok0 = max(g - s, 0) * kPage;
    const int tok1 = min((pend - s) * kPage, L);
    if (tok1 <= tok0) break;   // the range ends inside the sequence's start cost
    const float* qsrc = reinterpret_cast<const float*>(qprep + static_cast<size_t>(b) * qstride);
    for (int i = threadIdx.x; i < H * (d_c + d_rope); i += blockDim.x) qh[i] = qsrc[i];
    for (int i = threadIdx.x; i < H * d_c; i += blockDim.x) acc[i] = 0.f;
    if (threadIdx.x < 16) { mrun[threadIdx.x] = -INFINITY; lrun[threadIdx.x] = 0.f; }
    __syncthreads();
    for (int j = tok0; j < tok1; ++j) {
      const int page = block_table[static_cast<size_t>(b) * max_pages + j / kPage];
      const bool page_ok = page >= 0 && page < num_pages;
      const size_t row = static_cast<size_t>(page_ok ? page : 0) * kPage + j % kPage;
      if (!page_ok && threadIdx.x == 0) report_status(status, kStatusOutOfRange);
      int id = 0;
      if (gate) {
        id = id_pool[row];
        if (id < 0 || id >= vocab) {
          if (threadIdx.x == 0) report_status(status, kStatusOutOfRange);
          id = 0;
        }
      }
      // gate and LayerNorm (two-pass statistics)
      float s1 = 0.f;
      for (int f = threadIdx.x; f < d_c; f += blockDim.x) {
        float z = c_pool[row * d_c + f];
        if (gate) {
          const float g = gate_table[static_cast<size_t>(id) * d_c + f];
          z = gate_add ? z + g : z * g;
        }
        ct[f] = z;
        s1 += z;
      }
      for (int r = threadIdx.x; r < d_rope; r += blockDim.x) krs[r] = kr_pool[row * d_rope + r];
      if (gate && gate_ln) {
        const float mean = block_sum_128(s1, red, 0) / d_c;
        float s2 = 0.f;
        for (int f = threadIdx.x; f < d_c; f += blockDim.x) {
          const float dz = ct[f] - mean;
          s2 = fmaf(dz, dz, s2);
        }
        const float var = block_sum_128(s2, red, 1) / d_c;
        const float rstd = rsqrtf(var + eps);
        for (int f = threadIdx.x; f < d_c; f += blockDim.x)
          ct[f] = (ct[f] - mean) * rstd * (gamma ? gamma[f] : 1.f) + (beta ? beta[f] : 0.f);
      }
      __syncthreads();
      // scores of every head
      for (int h = 0; h < H; ++h) {
        float part = 0.f;
        for (int f = threadIdx.x; f < d_c; f += blockDim.x) part = fmaf(qh[h * d_c + f], ct[f], part);
        for (int r = threadIdx.x; r < d_rope; r += blockDim.x) part = fmaf(qr[h * d_rope + r], krs[r], part);
        const float s = block_sum_128(part, red, 2 + h) * scale_log2;
        if (threadIdx.x == 0) {
          const float mn = fmaxf(mrun[h], s);
          const float a = exp2f(mrun[h] - mn);
          const float p = exp2f(s - mn);
          lrun[h] = lrun[h] * a + p;
          mrun[h] = mn;
          alph[h] = a;
          pcur[h] = p;
        }
      }
      __syncthreads();
      for (int i = threadIdx.x; i < H * d_c; i += blockDim.x) {
        const int h = i / d_c;
        acc[i] = fmaf(acc[i], alph[h], pcur[h] * ct[i - h * d_c]);
      }
      __syncthreads();
    }
    const int slot = blockIdx.x + b;
    for (int i = threadIdx.x; i < H * d_c; i += blockDim.x) part_o[static_cast<size_t>(slot) * H * d_c + i] = acc[i];
    if (threadIdx.x < H) {
      part_ml[(static_cast<size_t>(slot) * H + threadIdx.x) * 2] = mrun[threadIdx.x];
      part_ml[(static_cast<size_t>(slot) * H + threadIdx.x) * 2 + 1] = lrun[threadIdx.x];
    }
    __syncthreads();
    g = pend;
    ++b;
    while (b < batch && cu[b + 1] <= g) ++b;
  }
}

// ------------------------------------------------------------------ launchers
cudaError_t launch_append(const AppendArgs& a, cudaStream_t st) {
  if (a.batch == 0) return cudaSuccess;
  append_latent_kernel<<<a.batch, 64, 0, st>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_prologue_tc(const DecodeArgs& a, const AppendArgs* app, cudaStream_t st) {
  const WorkspaceLayout wl = workspace_layout(a.batch, a.num_splits, 16, a.d_c, a.d_rope, true);
  uint8_t* ws = static_cast<uint8_t*>(a.workspace);
  // with the gate off the latent is used as cached: no LayerNorm affine to fold into q^
  const float* gamma = a.gate && a.gate_ln ? a.ln_gamma : nullptr;
  const float* beta = a.gate && a.gate_ln ? a.ln_beta : nullptr;
  const int ngroups = (a.batch + kPBatch - 1) / kPBatch;
  AppendArgs none;
  std::memset(&none, 0, sizeof(none));
  const AppendArgs& ap = app != nullptr ? *app : none;
  prologue_tc_kernel<<<16 * (a.d_c / kSumFeatures) * ngroups + 1 + ap.batch, 256, 0, st>>>(
      static_cast<const __nv_bfloat16*>(a.q), static_cast<const __nv_bfloat16*>(a.w_uk), gamma, beta,
      a.seq_lens, a.batch, a.d_nope, a.d_rope, a.d_c, a.page_size, ws + wl.off_qprep, wl.qprep_stride,
      reinterpret_cast<int32_t*>(ws + wl.off_cu), reinterpret_cast<uint32_t*>(ws + wl.off_done), a.num_splits,
      a.block_table, a.max_pages, reinterpret_cast<SplitStart*>(ws + wl.off_start), ap);
  return cudaGetLastError();
}

cudaError_t launch_decode_f32(const DecodeArgs& a, cudaStream_t st) {
  const WorkspaceLayout wl = workspace_layout(a.batch, a.num_splits, a.H, a.d_c, a.d_rope, false);
  uint8_t* ws = static_cast<uint8_t*>(a.workspace);
  prologue_f32_kernel<<<a.batch * a.H + 1, 256, 0, st>>>(
      static_cast<const float*>(a.q), static_cast<const float*>(a.w_uk), a.seq_lens, a.batch, a.H, a.d_nope,
      a.d_rope, a.d_c, a.page_size, ws + wl.off_qprep, wl.qprep_stride,
      reinterpret_cast<int32_t*>(ws + wl.off_cu));
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  const size_t smem = (static_cast<size_t>(a.H) * (2 * a.d_c + a.d_rope) + a.d_c + 64 + 80) * sizeof(float);
  if (smem > 48 * 1024) {
    e = cudaFuncSetAttribute(decode_f32_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
  }
  decode_f32_kernel<<<a.num_splits, kF32Threads, smem, st>>>(
      static_cast<const float*>(a.c_pool), static_cast<const float*>(a.kr_pool), a.id_pool, a.block_table,
      a.max_pages, a.seq_lens, a.batch, a.num_pages, static_cast<const float*>(a.gate_table), a.ln_gamma,
      a.ln_beta, ws + wl.off_qprep, wl.qprep_stride, reinterpret_cast<const int32_t*>(ws + wl.off_cu),
      reinterpret_cast<float*>(ws + wl.off_ml), reinterpret_cast<float*>(ws + wl.off_o), a.H, a.d_c, a.d_rope,
      a.vocab, a.gate, a.gate_add, a.gate_ln, a.scale_log2, a.eps, a.status);
  return cudaGetLastError();
}

namespace {
template <typename T>
void launch_combine_t(const DecodeArgs& a, const int32_t* cu, const float* ml, const float* po, cudaStream_t st) {
  const int grid = a.H * ((a.batch + kCombineGroup - 1) / kCombineGroup);
  combine_kernel<T><<<grid, kCombineThreads, 0, st>>>(cu, ml, po, static_cast<const T*>(a.w_uv),
                                                      static_cast<T*>(a.out), a.batch, a.H, a.d_c, a.d_v,
                                                      a.num_splits);
}
}  // namespace

cudaError_t launch_combine(const DecodeArgs& a, bool tc_path, cudaStream_t st) {
  const WorkspaceLayout wl = workspace_layout(a.batch, a.num_splits, a.H, a.d_c, a.d_rope, tc_path);
  uint8_t* ws = static_cast<uint8_t*>(a.workspace);
  const int32_t* cu = reinterpret_cast<const int32_t*>(ws + wl.off_cu);
  const float* ml = reinterpret_cast<const float*>(ws + wl.off_ml);
  const float* po = reinterpret_cast<const float*>(ws + wl.off_o);
  if (a.dtype == 0)
    launch_combine_t<__nv_bfloat16>(a, cu, ml, po, st);
  else
    launch_combine_t<float>(a, cu, ml, po, st);
  return cudaGetLastError();
}

}  // namespace egmla
