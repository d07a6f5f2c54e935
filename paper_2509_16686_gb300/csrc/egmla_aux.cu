// egmla_aux.cu - the small kernels around the tensor-core decode kernel:
//   append_latent_kernel   cache write of the new token (bit-exact copy)
//   prologue_*_kernel      per-step query absorption q^ = W_UK,h^T q^C and the
//                          page prefix sums the split-KV schedule needs
//   combine_*_kernel       log-sum-exp merge of the split partials and the
//                          W_UV,h up-projection of the latent output
//   decode_f32_kernel      the fp32 specialisation of the split-KV decode
//                          (exact fp32 arithmetic on CUDA cores; bf16 runs on
//                          tcgen05 in egmla_decode_tc.cu)
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <cmath>
#include <cstdint>

#include "egmla_common.cuh"
#include "egmla_kernels.h"
#include "egmla_ptx.cuh"

namespace egmla {

// ------------------------------------------------------------------ append
// One block per sequence; the row copies are 16-byte vectors when the row
// byte counts allow it (they do for every supported shape).
__global__ void append_latent_kernel(uint8_t* __restrict__ c_pool, uint8_t* __restrict__ kr_pool,
                                     int32_t* __restrict__ id_pool, const uint8_t* __restrict__ c_new,
                                     const uint8_t* __restrict__ kr_new,
                                     const int32_t* __restrict__ ids_new,
                                     const int32_t* __restrict__ block_table, int max_pages,
                                     const int32_t* __restrict__ positions, int num_pages, int page_size,
                                     int c_row_bytes, int kr_row_bytes, int32_t* status) {
  const int b = blockIdx.x;
  const int pos = positions[b];
  if (pos < 0) return;
  const int lp = pos / page_size;
  if (lp >= max_pages) {
    if (threadIdx.x == 0) report_status(status, kStatusOutOfRange);
    return;
  }
  const int page = block_table[static_cast<size_t>(b) * max_pages + lp];
  if (page < 0 || page >= num_pages) {
    if (threadIdx.x == 0) report_status(status, kStatusOutOfRange);
    return;
  }
  const size_t row = static_cast<size_t>(page) * page_size + pos % page_size;
  uint8_t* cd = c_pool + row * c_row_bytes;
  const uint8_t* cs = c_new + static_cast<size_t>(b) * c_row_bytes;
  for (int i = threadIdx.x; i < c_row_bytes / 16; i += blockDim.x)
    reinterpret_cast<uint4*>(cd)[i] = reinterpret_cast<const uint4*>(cs)[i];
  uint8_t* kd = kr_pool + row * kr_row_bytes;
  const uint8_t* ks = kr_new + static_cast<size_t>(b) * kr_row_bytes;
  for (int i = threadIdx.x; i < kr_row_bytes / 16; i += blockDim.x)
    reinterpret_cast<uint4*>(kd)[i] = reinterpret_cast<const uint4*>(ks)[i];
  if (id_pool != nullptr && ids_new != nullptr && threadIdx.x == 0) id_pool[row] = ids_new[b];
}

// ------------------------------------------------------------------ prologue
// Exclusive prefix sum of pages per sequence: cu[b] = sum_{b'<b} ceil(L_b'/P).
__device__ void page_prefix_sums(const int32_t* seq_lens, int batch, int page_size, int32_t* cu) {
  if (threadIdx.x == 0) {
    int32_t acc = 0;
    for (int b = 0; b < batch; ++b) {
      cu[b] = acc;
      int L = seq_lens[b];
      acc += L > 0 ? (L + page_size - 1) / page_size : 0;
    }
    cu[batch] = acc;
  }
}

__device__ __forceinline__ float block_sum_256(float v, float* red) {
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  __syncthreads();
  if (lane == 0) red[w] = v;
  __syncthreads();
  float s = 0.f;
  for (int i = 0; i < (int)(blockDim.x >> 5); ++i) s += red[i];
  return s;
}

// Tensor-core path: block (h, group of up to kQGroup sequences) computes
// q^_{b,h} = W_UK,h^T q^C_{b,h} in fp32 (one latent feature per thread, W_UK,h
// read once per group) and stores (q^ (*) gamma) as the bf16 B operand of the
// score MMA, laid out in 8x8 core matrices (no swizzle, K-major): element
// (head n, feature k) at byte (k/8)*256 + (n/8)*128 + (n%8)*16 + (k%8)*2.  q^R
// goes to the same layout.  The per-head sums w_h = sum_f bf16(q^ gamma)_f and
// b_h = q^_h . beta are the terms the LayerNorm contributes after the MMA.
constexpr int kQGroup = 8;

__global__ void __launch_bounds__(256)
prologue_tc_kernel(const __nv_bfloat16* __restrict__ q, const __nv_bfloat16* __restrict__ w_uk,
                   const float* __restrict__ gamma, const float* __restrict__ beta,
                   const int32_t* __restrict__ seq_lens, int batch, int d_nope, int d_rope, int d_c,
                   int page_size, uint8_t* __restrict__ qprep, size_t qstride, int32_t* __restrict__ cu) {
  __shared__ float qn[kQGroup][256];
  __shared__ float red[2][kQGroup][8];
  const int H = 16;
  const int ngroups = (batch + kQGroup - 1) / kQGroup;
  if (blockIdx.x == static_cast<unsigned>(ngroups * H)) {
    page_prefix_sums(seq_lens, batch, page_size, cu);
    return;
  }
  if (q == nullptr) return;  // cache-read test entry: prefix sums only
  const int h = blockIdx.x % H, b0 = (blockIdx.x / H) * kQGroup;
  const int nb = min(kQGroup, batch - b0);
  for (int i = threadIdx.x; i < kQGroup * d_nope; i += blockDim.x) {
    const int j = i / d_nope, n = i % d_nope;
    qn[j][n] = j < nb ? __bfloat162float(q[(static_cast<size_t>(b0 + j) * H + h) * (d_nope + d_rope) + n]) : 0.f;
  }
  __syncthreads();
  const __nv_bfloat16* w = w_uk + static_cast<size_t>(h) * d_nope * d_c;
  float wpart[kQGroup], bpart[kQGroup];
#pragma unroll
  for (int j = 0; j < kQGroup; ++j) wpart[j] = bpart[j] = 0.f;
  for (int f = threadIdx.x; f < d_c; f += blockDim.x) {
    float acc[kQGroup];
#pragma unroll
    for (int j = 0; j < kQGroup; ++j) acc[j] = 0.f;
#pragma unroll 8
    for (int n = 0; n < d_nope; ++n) {
      const float wv = __bfloat162float(w[static_cast<size_t>(n) * d_c + f]);
#pragma unroll
      for (int j = 0; j < kQGroup; ++j) acc[j] = fmaf(wv, qn[j][n], acc[j]);
    }
    const float gm = gamma ? gamma[f] : 1.f;
    const float bt = beta ? beta[f] : 0.f;
    const size_t off = qop_offset(h, f);
#pragma unroll
    for (int j = 0; j < kQGroup; ++j) {
      if (j >= nb) break;
      const __nv_bfloat16 bq = __float2bfloat16_rn(acc[j] * gm);
      *reinterpret_cast<__nv_bfloat16*>(qprep + static_cast<size_t>(b0 + j) * qstride + off) = bq;
      wpart[j] += __bfloat162float(bq);
      bpart[j] = fmaf(acc[j], bt, bpart[j]);
    }
  }
  for (int i = threadIdx.x; i < nb * d_rope; i += blockDim.x) {
    const int j = i / d_rope, r = i % d_rope;
    const size_t off = qprep_lat_bytes(d_c) + qop_offset(h, r);
    *reinterpret_cast<__nv_bfloat16*>(qprep + static_cast<size_t>(b0 + j) * qstride + off) = q[(static_cast<size_t>(b0 + j) * H + h) * (d_nope + d_rope) + d_nope + r];
  }
  // per-sequence block sums of w and b
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int j = 0; j < kQGroup; ++j) {
    float a = wpart[j], c = bpart[j];
    for (int o = 16; o > 0; o >>= 1) {
      a += __shfl_xor_sync(0xffffffffu, a, o);
      c += __shfl_xor_sync(0xffffffffu, c, o);
    }
    if (lane == 0) {
      red[0][j][warp] = a;
      red[1][j][warp] = c;
    }
  }
  __syncthreads();
  if (threadIdx.x < nb) {
    const int j = threadIdx.x;
    float a = 0.f, c = 0.f;
    for (int k = 0; k < (int)(blockDim.x >> 5); ++k) {
      a += red[0][j][k];
      c += red[1][j][k];
    }
    float* sums = reinterpret_cast<float*>(qprep + static_cast<size_t>(b0 + j) * qstride + qprep_lat_bytes(d_c) +
                                           qprep_rope_bytes(d_rope));
    sums[h] = a;
    sums[16 + h] = c;
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
// Block (h, group of 8 sequences).  For each sequence: M = max_s m_s,
// o = sum_s 2^(m_s - M) O_s / sum_s 2^(m_s - M) l_s (m in log2 units), then
// u = W_UV,h o.  Sequences of length 0 get u = 0.
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

// Block per (sequence b, head h), 256 threads.  The splits that covered b are
// the CTAs c0..c1 of the page schedule; their partials sit in slots c + b.
// M = max_s m_s; o = sum_s 2^(m_s - M) O_s / sum_s 2^(m_s - M) l_s (m in log2
// units); then u = W_UV,h o with two threads per output row.  A sequence of
// length 0 gets u = 0.
constexpr int kCombineThreads = 256;
constexpr int kMaxSlotsSmem = 512;

template <typename T>
__global__ void __launch_bounds__(kCombineThreads)
combine_kernel(const int32_t* __restrict__ cu, const float* __restrict__ part_ml, const float* __restrict__ part_o,
               const T* __restrict__ w_uv, T* __restrict__ out, int batch, int H, int d_c, int d_v,
               int num_splits) {
  extern __shared__ float olat[];  // [d_c]
  __shared__ float wts[kMaxSlotsSmem];
  __shared__ float red[32];
  const int b = blockIdx.x / H, h = blockIdx.x % H;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int total = cu[batch];
  const int chunk = split_chunk(total, num_splits);
  const int p0 = cu[b], p1 = cu[b + 1];
  const int c0 = p0 / chunk;
  const int n = p1 > p0 ? (p1 - 1) / chunk - c0 + 1 : 0;
  if (n == 0) {
    for (int f = tid; f < d_c; f += blockDim.x) olat[f] = 0.f;
  } else {
    // running max and denominator over the slots (n <= num_splits)
    float mloc = -INFINITY;
    for (int k = tid; k < n; k += blockDim.x) mloc = fmaxf(mloc, part_ml[(static_cast<size_t>(c0 + k + b) * H + h) * 2]);
    for (int o = 16; o > 0; o >>= 1) mloc = fmaxf(mloc, __shfl_xor_sync(0xffffffffu, mloc, o));
    if (lane == 0) red[warp] = mloc;
    __syncthreads();
    float M = red[0];
    for (int k = 1; k < (int)(blockDim.x >> 5); ++k) M = fmaxf(M, red[k]);
    __syncthreads();
    float lloc = 0.f;
    for (int k = tid; k < n; k += blockDim.x) {
      const float* ml = part_ml + (static_cast<size_t>(c0 + k + b) * H + h) * 2;
      const float wk = exp2f(ml[0] - M);
      if (k < kMaxSlotsSmem) wts[k] = wk;
      lloc = fmaf(wk, ml[1], lloc);
    }
    for (int o = 16; o > 0; o >>= 1) lloc += __shfl_xor_sync(0xffffffffu, lloc, o);
    if (lane == 0) red[warp] = lloc;
    __syncthreads();
    float L = 0.f;
    for (int k = 0; k < (int)(blockDim.x >> 5); ++k) L += red[k];
    const float invL = 1.f / L;
    for (int f = tid; f < d_c; f += blockDim.x) {
      float acc = 0.f;
#pragma unroll 8
      for (int k = 0; k < n; ++k) {
        const size_t s = static_cast<size_t>(c0 + k + b) * H + h;
        const float wk = k < kMaxSlotsSmem ? wts[k] : exp2f(part_ml[s * 2] - M);
        acc = fmaf(wk, part_o[s * d_c + f], acc);
      }
      olat[f] = acc * invL;
    }
  }
  __syncthreads();
  // u[v] = sum_f W_UV[h][v][f] olat[f]: a thread pair per row v, halves of f
  const T* wh = w_uv + static_cast<size_t>(h) * d_v * d_c;
  const int half = tid & 1;
  for (int base = 0; base < d_v; base += blockDim.x >> 1) {
    const int v = base + (tid >> 1);
    float acc = 0.f;
    if (v < d_v) {
      const T* row = wh + static_cast<size_t>(v) * d_c;
#pragma unroll 8
      for (int f = half; f < d_c; f += 2) acc = fmaf(to_f<T>(row[f]), olat[f], acc);
    }
    acc += __shfl_xor_sync(0xffffffffu, acc, 1);
    if (half == 0 && v < d_v) out[(static_cast<size_t>(b) * H + h) * d_v + v] = from_f<T>(acc);
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
                  int H, int d_c, int d_rope, int vocab, int gate, float scale_log2, float eps,
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
    const int tok0 = (g - cu[b]) * kPage;
    const int tok1 = min((pend - cu[b]) * kPage, L);
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
        if (gate) z *= gate_table[static_cast<size_t>(id) * d_c + f];
        ct[f] = z;
        s1 += z;
      }
      for (int r = threadIdx.x; r < d_rope; r += blockDim.x) krs[r] = kr_pool[row * d_rope + r];
      if (gate) {
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
  append_latent_kernel<<<a.batch, 64, 0, st>>>(
      static_cast<uint8_t*>(a.c_pool), static_cast<uint8_t*>(a.kr_pool), a.id_pool,
      static_cast<const uint8_t*>(a.c_new), static_cast<const uint8_t*>(a.kr_new), a.ids_new, a.block_table,
      a.max_pages, a.positions, a.num_pages, a.page_size, a.c_row_bytes, a.kr_row_bytes, a.status);
  return cudaGetLastError();
}

cudaError_t launch_prologue_tc(const DecodeArgs& a, cudaStream_t st) {
  const WorkspaceLayout wl = workspace_layout(a.batch, a.num_splits, 16, a.d_c, a.d_rope, true);
  uint8_t* ws = static_cast<uint8_t*>(a.workspace);
  // with the gate off the latent is used as cached: no LayerNorm affine to fold into q^
  const float* gamma = a.gate ? a.ln_gamma : nullptr;
  const float* beta = a.gate ? a.ln_beta : nullptr;
  const int ngroups = (a.batch + kQGroup - 1) / kQGroup;
  prologue_tc_kernel<<<ngroups * 16 + 1, 256, 0, st>>>(
      static_cast<const __nv_bfloat16*>(a.q), static_cast<const __nv_bfloat16*>(a.w_uk), gamma, beta,
      a.seq_lens, a.batch, a.d_nope, a.d_rope, a.d_c, a.page_size, ws + wl.off_qprep, wl.qprep_stride,
      reinterpret_cast<int32_t*>(ws + wl.off_cu));
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
      a.vocab, a.gate, a.scale_log2, a.eps, a.status);
  return cudaGetLastError();
}

cudaError_t launch_combine(const DecodeArgs& a, bool tc_path, cudaStream_t st) {
  const WorkspaceLayout wl = workspace_layout(a.batch, a.num_splits, a.H, a.d_c, a.d_rope, tc_path);
  uint8_t* ws = static_cast<uint8_t*>(a.workspace);
  const size_t smem = static_cast<size_t>(a.d_c) * sizeof(float);
  const int32_t* cu = reinterpret_cast<const int32_t*>(ws + wl.off_cu);
  const float* ml = reinterpret_cast<const float*>(ws + wl.off_ml);
  const float* po = reinterpret_cast<const float*>(ws + wl.off_o);
  const int grid = a.batch * a.H;
  if (a.dtype == 0) {
    combine_kernel<__nv_bfloat16><<<grid, kCombineThreads, smem, st>>>(
        cu, ml, po, static_cast<const __nv_bfloat16*>(a.w_uv), static_cast<__nv_bfloat16*>(a.out), a.batch, a.H,
        a.d_c, a.d_v, a.num_splits);
  } else {
    combine_kernel<float><<<grid, kCombineThreads, smem, st>>>(cu, ml, po, static_cast<const float*>(a.w_uv),
                                                                static_cast<float*>(a.out), a.batch, a.H, a.d_c,
                                                                a.d_v, a.num_splits);
  }
  return cudaGetLastError();
}

}  // namespace egmla
