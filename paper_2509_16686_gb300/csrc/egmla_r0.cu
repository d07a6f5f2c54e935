// egmla_r0.cu - decode with the paper-literal gate placement (R0): the gate
// and the LayerNorm act on the up-projected keys and values of all heads,
// kv~ = LN_{H(d_n + d_v)}((W^UKV c) (*) g) (Section 3 Eq. 5 applied after
// Eq. 2, as the Appendix E listing does), split per head into k^C, v^C
// (Eq. 6), then attention as in Eqs. 11-13 without absorption (the gate in
// the 4096-wide space cannot be folded into the query).
//
// Two kernels:
//   r0_project_kernel  (tcgen05) every row of the latent pool, 128 rows per
//                      CTA: for each head h, D = C W^UKV_h^T (M = 128 rows,
//                      N = 256 = d_n + d_v features, K = d_c) in a TMEM
//                      accumulator (two buffers, so the epilogue of head h
//                      overlaps the MMAs of head h + 1); the epilogue warps
//                      (one row each) gate the features with the row's R0
//                      gate G_R0[id], round z to bf16, store it, and add z and
//                      z^2 of the rounded values into the row's statistics;
//                      after the last head, (mu, 1/sqrt(var + eps)) per row.
//   r0_attend_kernel   one block per (sequence, head): the sequence's rows
//                      through its block table, LN applied on the fly
//                      (k~ = gamma (z - mu) r + beta), s = scale (q . k~ +
//                      q^R . k^R), an online softmax per warp (sixteen warps,
//                      four rows in flight each), merged at the end.
// z of the whole pool is materialised in the workspace (H (d_n + d_v) bf16
// per pool row); rows the attention never reads (free cache slots) are
// projected too, with their ids clamped, and never read.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <cmath>
#include <cstdint>
#include <cstring>
#include <mutex>

#include "egmla_common.cuh"
#include "egmla_kernels.h"
#include "egmla_ptx.cuh"

namespace egmla {
namespace {

constexpr int kR0Heads = 16;
constexpr int kR0Feat = 256;                    // d_n + d_v per head
constexpr int kR0Width = kR0Heads * kR0Feat;    // 4096
constexpr int kR0Rows = 128;                    // pool rows per CTA (the MMA's M)
constexpr int kR0Chunk = 64;                    // K elements per operand chunk (128-byte swizzle atom)
constexpr uint32_t kR0AChunkBytes = kR0Rows * kR0Chunk * 2;   // 16 KB
constexpr uint32_t kR0BChunkBytes = kR0Feat * kR0Chunk * 2;   // 32 KB
constexpr int kR0BStages = 3;
constexpr int kR0EpiWarps = 8;                  // two per TMEM lane quadrant, half of each head's columns each
constexpr int kR0Threads = 32 * (2 + kR0EpiWarps);   // warp 0 TMA, warp 1 MMA, warps 2-9 epilogue
constexpr uint32_t kR0TmemCols = 512;           // two 256-column accumulators

struct R0Bars {
  float2 half_sums[kR0Rows];   // the second column half's (sum z, sum z^2) per row
  uint64_t afull;
  uint64_t bfull[kR0BStages], bempty[kR0BStages];
  uint64_t dfull[2], dfree[2];
  uint64_t drain;
  uint32_t tmem_base;
  int abort;
};

struct R0ProjParams {
  const int32_t* id_pool;
  const __nv_bfloat16* gate;   // [vocab, 4096]
  __nv_bfloat16* z;            // [pool rows, 4096]
  float2* stats;               // [pool rows]: (mu, r)
  int pool_rows, vocab, nkc;   // nkc = d_c / 64
  float eps;
  uint64_t wait_ns;
  int32_t* status;
};

__device__ __forceinline__ bool warp_all_wait(uint32_t bar, uint32_t parity, volatile int* abort_flag,
                                              uint64_t limit_ns) {
  __syncwarp();
  const bool ok = mbar_wait(bar, parity, abort_flag, limit_ns);
  return __all_sync(0xffffffffu, ok);
}

__global__ void __launch_bounds__(kR0Threads, 1)
    r0_project_kernel(const __grid_constant__ CUtensorMap cmap, const __grid_constant__ CUtensorMap wmap,
                      const R0ProjParams p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  const uint32_t sbase = smem_u32(smem);
  const uint32_t b_off = static_cast<uint32_t>(p.nkc) * kR0AChunkBytes;
  R0Bars& bars = *reinterpret_cast<R0Bars*>(smem + b_off + kR0BStages * kR0BChunkBytes);
  volatile int* abort_flag = &bars.abort;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int row0 = blockIdx.x * kR0Rows;
  const int nsteps = kR0Heads * p.nkc;   // (head, K chunk) steps of the B stream

  if (tid == 0) {
    mbar_init(smem_u32(&bars.afull), 1);
    for (int s = 0; s < kR0BStages; ++s) {
      mbar_init(smem_u32(&bars.bfull[s]), 1);
      mbar_init(smem_u32(&bars.bempty[s]), 1);
    }
    for (int s = 0; s < 2; ++s) {
      mbar_init(smem_u32(&bars.dfull[s]), 1);
      mbar_init(smem_u32(&bars.dfree[s]), kR0EpiWarps);
    }
    mbar_init(smem_u32(&bars.drain), 1);
    bars.abort = 0;
    fence_mbar_init();
    prefetch_tensormap(&cmap);
    prefetch_tensormap(&wmap);
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(&bars.tmem_base), kR0TmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = bars.tmem_base;

  bool epi_ok = false, epi_first_half = false;
  float epi_s1 = 0.f, epi_s2 = 0.f;
  int epi_row = 0;
  if (warp == 0) {
    // ---- TMA: the CTA's 128 latent rows (all K chunks), then W^UKV_h chunk by chunk
    if (elect_one()) {
      const uint64_t pol_stream = policy_evict_first(), pol_keep = policy_evict_last();
      mbar_arrive_expect_tx(smem_u32(&bars.afull), static_cast<uint32_t>(p.nkc) * kR0AChunkBytes);
      for (int kc = 0; kc < p.nkc; ++kc)
        tma_load_2d(sbase + kc * kR0AChunkBytes, &cmap, kc * kR0Chunk, row0, smem_u32(&bars.afull), pol_stream);
      int issued = 0;
      for (int i = 0; i < nsteps; ++i) {
        const int s = i % kR0BStages;
        if (i >= kR0BStages &&
            !mbar_wait(smem_u32(&bars.bempty[s]), ((i / kR0BStages) & 1) ^ 1, abort_flag, p.wait_ns))
          break;
        const int h = i / p.nkc, kc = i % p.nkc;
        mbar_arrive_expect_tx(smem_u32(&bars.bfull[s]), kR0BChunkBytes);
        tma_load_2d(sbase + b_off + s * kR0BChunkBytes, &wmap, kc * kR0Chunk, h * kR0Feat, smem_u32(&bars.bfull[s]),
                    pol_keep);
        issued = i + 1;
      }
      // every copy issued lands before the CTA can leave (own flag: bounded, not cut short)
      volatile int own = 0;
      if (!mbar_wait(smem_u32(&bars.afull), 0, &own, p.wait_ns)) *abort_flag = 1;
      for (int i = issued > kR0BStages ? issued - kR0BStages : 0; i < issued; ++i)
        if (!mbar_wait(smem_u32(&bars.bfull[i % kR0BStages]), (i / kR0BStages) & 1, &own, p.wait_ns))
          *abort_flag = 1;
    }
    __syncwarp();
  } else if (warp == 1) {
    // ---- MMA: head h into accumulator h % 2 once the epilogue has read it out
    constexpr uint32_t idesc = idesc_bf16(kR0Rows, kR0Feat, 0, 0);
    bool ok = warp_all_wait(smem_u32(&bars.afull), 0, abort_flag, p.wait_ns);
    bool issued = false;
    for (int h = 0; ok && h < kR0Heads; ++h) {
      const int db = h & 1;
      if (h >= 2) ok = warp_all_wait(smem_u32(&bars.dfree[db]), ((h - 2) >> 1) & 1, abort_flag, p.wait_ns);
      for (int kc = 0; ok && kc < p.nkc; ++kc) {
        const int i = h * p.nkc + kc, s = i % kR0BStages;
        ok = warp_all_wait(smem_u32(&bars.bfull[s]), (i / kR0BStages) & 1, abort_flag, p.wait_ns);
        if (!ok) break;
        tc_fence_after();
        if (elect_one()) {
          const uint64_t ad = smem_desc(sbase + kc * kR0AChunkBytes, 16, 1024, kSwizzle128B);
          const uint64_t bd = smem_desc(sbase + b_off + s * kR0BChunkBytes, 16, 1024, kSwizzle128B);
#pragma unroll
          for (int kk = 0; kk < kR0Chunk / 16; ++kk)
            mma_bf16_ss(tmem + db * kR0Feat, ad + ((kk * 32) >> 4), bd + ((kk * 32) >> 4), idesc,
                        (kc > 0 || kk > 0) ? 1u : 0u);
          mma_commit(smem_u32(&bars.bempty[s]));
          if (kc == p.nkc - 1) mma_commit(smem_u32(&bars.dfull[db]));
        }
        __syncwarp();
        issued = true;
      }
    }
    // every MMA issued completes before TMEM is released
    if (issued) {
      if (elect_one()) mma_commit(smem_u32(&bars.drain));
      __syncwarp();
      volatile int own = 0;
      if (!mbar_wait(smem_u32(&bars.drain), 0, &own, p.wait_ns)) *abort_flag = 1;
    }
    __syncwarp();
  } else {
    // ---- epilogue: row r of the tile is TMEM lane r (warp w reads lane
    // quadrant w % 4); warps 2-5 take columns 0-127 of every head, warps 6-9
    // columns 128-255
    const int quad = warp & 3, half = (warp - 2) / 4;
    const int r = 32 * quad + lane, row = row0 + r;
    const bool in_pool = row < p.pool_rows;
    int id = in_pool ? p.id_pool[row] : 0;
    if (static_cast<unsigned>(id) >= static_cast<unsigned>(p.vocab)) id = 0;   // free slot: never read
    const int cbase = half * (kR0Feat / 2);
    const __nv_bfloat16* grow = p.gate + static_cast<size_t>(id) * kR0Width + cbase;
    const uint64_t pol_gate = policy_evict_last();
    __nv_bfloat16* zrow = p.z + static_cast<size_t>(in_pool ? row : 0) * kR0Width + cbase;
    float s1 = 0.f, s2 = 0.f;
    bool ok = true;
    for (int h = 0; h < kR0Heads; ++h) {
      const int db = h & 1;
      // this half of the row's gate values of the head, requested at once
      // (one round trip per head) while the head's MMAs may still run
      uint4 g[kR0Feat / 16];
#pragma unroll
      for (int i = 0; i < kR0Feat / 16; ++i) g[i] = ldg_16_na_hint(grow + h * kR0Feat + 8 * i, pol_gate);
      ok = ok && warp_all_wait(smem_u32(&bars.dfull[db]), (h >> 1) & 1, abort_flag, p.wait_ns);
      if (!ok) break;
      tc_fence_after();
#pragma unroll
      for (int c0 = 0; c0 < kR0Feat / 2; c0 += 16) {
        float v[16];
        tmem_ld16(tmem + (static_cast<uint32_t>(32 * quad) << 16) + db * kR0Feat + cbase + c0, v);
        tmem_wait_ld();
        const __nv_bfloat162* ge0 = reinterpret_cast<const __nv_bfloat162*>(&g[c0 / 8]);
        const __nv_bfloat162* ge1 = reinterpret_cast<const __nv_bfloat162*>(&g[c0 / 8 + 1]);
        uint32_t packed[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          const float2 gf = __bfloat1622float2(i < 4 ? ge0[i] : ge1[i - 4]);
          const __nv_bfloat162 zb = __floats2bfloat162_rn(v[2 * i] * gf.x, v[2 * i + 1] * gf.y);
          const float2 zr = __bfloat1622float2(zb);   // statistics of the stored values
          s1 += zr.x + zr.y;
          s2 = fmaf(zr.x, zr.x, fmaf(zr.y, zr.y, s2));
          packed[i] = *reinterpret_cast<const uint32_t*>(&zb);
        }
        if (in_pool) {
          uint4* dst = reinterpret_cast<uint4*>(zrow + h * kR0Feat + c0);
          dst[0] = make_uint4(packed[0], packed[1], packed[2], packed[3]);
          dst[1] = make_uint4(packed[4], packed[5], packed[6], packed[7]);
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_u32(&bars.dfree[db]));
    }
    if (half == 1) bars.half_sums[r] = make_float2(s1, s2);
    // the two halves of a row meet below (the first half adds the second's sums
    // after the block barrier)
    epi_ok = ok;
    epi_s1 = s1;
    epi_s2 = s2;
    epi_row = row;
    epi_first_half = half == 0 && in_pool;
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (epi_first_half && epi_ok && !bars.abort) {
    const float2 o = bars.half_sums[epi_row - row0];
    const float mu = (epi_s1 + o.x) / kR0Width;
    const float var = fmaxf((epi_s2 + o.y) / kR0Width - mu * mu, 0.f);
    p.stats[epi_row] = make_float2(mu, rsqrtf(var + p.eps));
  }
  if (warp == 1) tmem_dealloc(tmem, kR0TmemCols);
  if (tid == 0 && bars.abort) report_status(p.status, kStatusTimeout);
}

struct R0AttnParams {
  const __nv_bfloat16* q;       // [B, H, d_n + d_r]
  const __nv_bfloat16* kr_pool; // [pool rows, d_r]
  const int32_t* id_pool;
  const int32_t* block_table;
  const int32_t* seq_lens;
  const __nv_bfloat16* z;
  const float2* stats;
  const float* gamma;           // [4096] or null
  const float* beta;
  __nv_bfloat16* out;           // [B, H, d_v]
  int max_pages, num_pages, vocab;
  float scale_log2;
  int32_t* status;
};

constexpr int kR0AttnWarps = 16;
constexpr int kR0AttnThreads = 32 * kR0AttnWarps;
constexpr int kR0AttnBatch = 4;   // rows a warp has in flight at once

// One block per (sequence, head); warp w takes rows w + 16 i, four at a time
// (their loads issued together); lane l holds key features 4l .. 4l + 3 and
// value features 4l .. 4l + 3 of the head.  Each warp keeps its own online
// softmax (m, l, o); the warps are merged at the end.
__global__ void __launch_bounds__(kR0AttnThreads) r0_attend_kernel(const R0AttnParams p) {
  __shared__ float part[kR0AttnWarps][2 + 128];
  const int b = blockIdx.x / kR0Heads, h = blockIdx.x % kR0Heads;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int L = p.seq_lens[b];
  const int fk = h * kR0Feat + 4 * lane, fv = fk + 128;
  // q (gamma folded into the key part), w = sum q gamma, bq = q . beta
  const __nv_bfloat16* qh = p.q + (static_cast<size_t>(b) * kR0Heads + h) * 192;
  float qg[4], gv[4], bv[4], qr[2];
  float wpart = 0.f, bpart = 0.f;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const float qf = __bfloat162float(qh[4 * lane + i]);
    const float gk = p.gamma ? p.gamma[fk + i] : 1.f, bk = p.beta ? p.beta[fk + i] : 0.f;
    qg[i] = qf * gk;
    wpart += qg[i];
    bpart = fmaf(qf, bk, bpart);
    gv[i] = p.gamma ? p.gamma[fv + i] : 1.f;
    bv[i] = p.beta ? p.beta[fv + i] : 0.f;
  }
  qr[0] = __bfloat162float(qh[128 + 2 * lane]);
  qr[1] = __bfloat162float(qh[128 + 2 * lane + 1]);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    wpart += __shfl_xor_sync(0xffffffffu, wpart, o);
    bpart += __shfl_xor_sync(0xffffffffu, bpart, o);
  }
  float m = -INFINITY, l = 0.f, o4[4] = {0.f, 0.f, 0.f, 0.f};
  bool bad = false;
  for (int j0 = warp; j0 < L; j0 += kR0AttnWarps * kR0AttnBatch) {
    // the rows' addresses, then all their loads, then the arithmetic
    size_t row[kR0AttnBatch];
    bool valid[kR0AttnBatch];
#pragma unroll
    for (int t = 0; t < kR0AttnBatch; ++t) {
      const int j = j0 + t * kR0AttnWarps;
      valid[t] = j < L;
      row[t] = 0;
      if (valid[t]) {
        const int lp = j / kPage;
        const int page = lp < p.max_pages ? p.block_table[static_cast<size_t>(b) * p.max_pages + lp] : -1;
        if (page < 0 || page >= p.num_pages) {
          bad = true;
          valid[t] = false;
        } else {
          row[t] = static_cast<size_t>(page) * kPage + j % kPage;
        }
      }
    }
    float2 st[kR0AttnBatch];
    uint2 zk[kR0AttnBatch], zv[kR0AttnBatch];
    __nv_bfloat162 kr2[kR0AttnBatch];
    int id[kR0AttnBatch];
#pragma unroll
    for (int t = 0; t < kR0AttnBatch; ++t) {
      if (valid[t]) {
        id[t] = p.id_pool[row[t]];
        st[t] = p.stats[row[t]];
        zk[t] = *reinterpret_cast<const uint2*>(p.z + row[t] * kR0Width + fk);
        zv[t] = *reinterpret_cast<const uint2*>(p.z + row[t] * kR0Width + fv);
        kr2[t] = *reinterpret_cast<const __nv_bfloat162*>(p.kr_pool + row[t] * 64 + 2 * lane);
      }
    }
#pragma unroll
    for (int t = 0; t < kR0AttnBatch; ++t) {
      if (!valid[t]) continue;   // uniform in the warp
      if (static_cast<unsigned>(id[t]) >= static_cast<unsigned>(p.vocab)) bad = true;   // the gate used row 0
      const float2 k01 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&zk[t].x));
      const float2 k23 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&zk[t].y));
      const float2 krf = __bfloat1622float2(kr2[t]);
      const float dz = qg[0] * k01.x + qg[1] * k01.y + qg[2] * k23.x + qg[3] * k23.y;
      float part_s = fmaf(st[t].y, dz, qr[0] * krf.x + qr[1] * krf.y);
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) part_s += __shfl_xor_sync(0xffffffffu, part_s, o);
      // s (log2 units) = scale log2(e) (r (q gamma . z - mu w) + q . beta + q^R . k^R)
      const float s = p.scale_log2 * (part_s - st[t].y * st[t].x * wpart + bpart);
      const float mn = fmaxf(m, s);
      const float alpha = exp2f(m - mn), pj = exp2f(s - mn);
      l = fmaf(l, alpha, pj);
      const float2 v01 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&zv[t].x));
      const float2 v23 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&zv[t].y));
      const float vz[4] = {v01.x, v01.y, v23.x, v23.y};
#pragma unroll
      for (int i = 0; i < 4; ++i)
        o4[i] = fmaf(o4[i], alpha, pj * fmaf(gv[i], (vz[i] - st[t].x) * st[t].y, bv[i]));
      m = mn;
    }
  }
  if (bad && lane == 0) report_status(p.status, kStatusOutOfRange);
  if (lane == 0) {
    part[warp][0] = m;
    part[warp][1] = l;
  }
#pragma unroll
  for (int i = 0; i < 4; ++i) part[warp][2 + 4 * lane + i] = o4[i];
  __syncthreads();
  if (warp == 0) {
    float M = -INFINITY;
    for (int w = 0; w < kR0AttnWarps; ++w) M = fmaxf(M, part[w][0]);
    float Ls = 0.f, acc[4] = {0.f, 0.f, 0.f, 0.f};
    for (int w = 0; w < kR0AttnWarps; ++w) {
      const float sc = part[w][0] == -INFINITY ? 0.f : exp2f(part[w][0] - M);
      Ls = fmaf(part[w][1], sc, Ls);
#pragma unroll
      for (int i = 0; i < 4; ++i) acc[i] = fmaf(part[w][2 + 4 * lane + i], sc, acc[i]);
    }
    __nv_bfloat16* ob = p.out + (static_cast<size_t>(b) * kR0Heads + h) * 128 + 4 * lane;
#pragma unroll
    for (int i = 0; i < 4; ++i) ob[i] = __float2bfloat16_rn(L > 0 && Ls > 0.f ? acc[i] / Ls : 0.f);
  }
}

using EncodeFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                              const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                              CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeFn r0_encode_fn() {
  static EncodeFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeFn>(p);
  });
  return fn;
}

// row-major bf16 [rows, cols], boxes of 64 columns x box_rows rows, 128-byte swizzle
bool r0_encode(CUtensorMap* map, const void* base, uint64_t rows, uint64_t cols, uint32_t box_rows) {
  EncodeFn enc = r0_encode_fn();
  if (enc == nullptr) return false;
  std::memset(map, 0, sizeof(*map));
  const cuuint64_t dims[2] = {cols, rows};
  const cuuint64_t strides[1] = {cols * 2};
  const cuuint32_t box[2] = {static_cast<cuuint32_t>(kR0Chunk), box_rows};
  const cuuint32_t estr[2] = {1, 1};
  return enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace

size_t r0_workspace_bytes(int num_pages) {
  const size_t rows = static_cast<size_t>(num_pages) * kPage;
  return align_up(rows * kR0Width * 2, 256) + align_up(rows * sizeof(float2), 256);
}

cudaError_t launch_decode_r0(const R0Args& a, cudaStream_t st) {
  const size_t rows = static_cast<size_t>(a.num_pages) * kPage;
  uint8_t* ws = static_cast<uint8_t*>(a.workspace);
  __nv_bfloat16* z = reinterpret_cast<__nv_bfloat16*>(ws);
  float2* stats = reinterpret_cast<float2*>(ws + align_up(rows * kR0Width * 2, 256));
  CUtensorMap cmap, wmap;
  if (!r0_encode(&cmap, a.c_pool, rows, static_cast<uint64_t>(a.d_c), kR0Rows)) return cudaErrorInvalidValue;
  if (!r0_encode(&wmap, a.w_ukv, kR0Width, static_cast<uint64_t>(a.d_c), kR0Feat)) return cudaErrorInvalidValue;
  const int nkc = a.d_c / kR0Chunk;
  const int smem = static_cast<int>(nkc * kR0AChunkBytes + kR0BStages * kR0BChunkBytes + sizeof(R0Bars) + 1024);
  cudaError_t e = cudaFuncSetAttribute(r0_project_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  R0ProjParams pp;
  pp.id_pool = a.id_pool;
  pp.gate = static_cast<const __nv_bfloat16*>(a.gate_r0);
  pp.z = z;
  pp.stats = stats;
  pp.pool_rows = static_cast<int>(rows);
  pp.vocab = a.vocab;
  pp.nkc = nkc;
  pp.eps = a.eps;
  pp.wait_ns = kWaitLimitNs;
  pp.status = a.status;
  const int tiles = static_cast<int>((rows + kR0Rows - 1) / kR0Rows);
  r0_project_kernel<<<tiles, kR0Threads, smem, st>>>(cmap, wmap, pp);
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  R0AttnParams ap;
  ap.q = static_cast<const __nv_bfloat16*>(a.q);
  ap.kr_pool = static_cast<const __nv_bfloat16*>(a.kr_pool);
  ap.id_pool = a.id_pool;
  ap.block_table = a.block_table;
  ap.seq_lens = a.seq_lens;
  ap.z = z;
  ap.stats = stats;
  ap.gamma = a.ln_gamma;
  ap.beta = a.ln_beta;
  ap.out = static_cast<__nv_bfloat16*>(a.out);
  ap.max_pages = a.max_pages;
  ap.num_pages = a.num_pages;
  ap.vocab = a.vocab;
  ap.scale_log2 = a.scale_log2;
  ap.status = a.status;
  r0_attend_kernel<<<a.batch * kR0Heads, kR0AttnThreads, 0, st>>>(ap);
  return cudaGetLastError();
}

}  // namespace egmla
