// egmla_prefill.cu - prompt processing (prefill): every position t of a prompt
// attends causally to positions 0..t of the same prompt (Appendix C Eq. 13,
// whose sum stops at the query's own position), and the prompt is written into
// the paged latent cache for the decode steps that follow.
//
// Prefill is compute-bound (every query meets every earlier key), so it runs
// in the unabsorbed per-head form of the Appendix E listing, which needs
// 2 (d_n + d_r + d_v) = 640 flops per (query, key, head) instead of the
// absorbed form's 2 (d_c + d_r + d_c) = 1152:
//   prefill_gate_kernel  one warp per prompt token: c~ = LN(c (*) G[id]) (or the
//                        gate mode's variant; Section 3 Eq. 5 in latent space),
//                        rounded to bf16, and the raw c, k^R and id written to
//                        the token's cache slot through the block table; its
//                        first block also ranks the prompts by length (the
//                        attention's launch order) and zeroes the attention's
//                        work counter.
//   prefill_kv_kernel    (tcgen05) [k^C_h ; v^C_h] = [W_UK,h ; W_UV,h] c~ for
//                        128 tokens per CTA (RT = 1; RT = 2 row tiles share each
//                        weight chunk in the gate-table mode) and every head h
//                        (Eqs. 2 and 6): per output block of 128 columns (the
//                        key or the value rows of a head) M = 128 tokens per
//                        row tile, N = 128, K = d_c; two TMEM accumulators so
//                        the epilogue of one block overlaps the MMAs of the
//                        next; the output leaves through TMA tensor stores.
//                        The same kernel in plain x W^T mode computes the gate
//                        table E W^UE^T (eg_mla_gate_table).
//   prefill_attn_kernel  (tcgen05) causal flash attention, persistent: one CTA
//                        per SM takes (prompt, head, 256-query block) items,
//                        two query tiles of 128 rows each sharing every key and
//                        value tile (see the kernel's own header).
//
// Online softmax with a lazily moved reference: a row keeps the reference
// maximum m of its exponentials until a tile's maximum exceeds it by more than
// 2^8 (in log2 units 8); only then is O rescaled in TMEM.  Until then every
// exponential is at most 2^8, exact enough in fp32 and bf16.
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

constexpr int kPfRows = 128;                                // tokens per tile (the MMAs' M)
constexpr int kPfChunk = 64;                                // elements per 128-byte swizzle row
constexpr uint32_t kPfAtom = kPfRows * kPfChunk * 2;        // 16 KB: 128 rows x 64 bf16
constexpr int kPfDn = 128, kPfDr = 64, kPfDv = 128;
constexpr int kPfDqk = kPfDn + kPfDr;                       // 192: three 64-element chunks

__device__ __forceinline__ float pf_ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  const __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<const uint32_t*>(&v);
}

__device__ __forceinline__ bool pf_warp_wait(uint32_t bar, uint32_t parity, volatile int* abort_flag,
                                             uint64_t limit_ns) {
  __syncwarp();
  const bool ok = mbar_wait(bar, parity, abort_flag, limit_ns);
  return __all_sync(0xffffffffu, ok);
}

// prompt b of packed row t: the largest b with cu[b] <= t (empty prompts,
// whose start equals the next one's, are passed over)
__device__ __forceinline__ int prompt_of_row(const int32_t* cu, int batch, int t) {
  int lo = 0, hi = batch - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (__ldg(cu + mid) <= t) lo = mid; else hi = mid - 1;
  }
  return lo;
}

// ============================================================================ 1. gate, LayerNorm, cache write
struct PfGateParams {
  int32_t* order;              // [batch]: prompts by decreasing length (written by block 0)
  int32_t* next_item;          // the attention's work counter, zeroed by block 0
  const __nv_bfloat16* c;      // [T, d_c]
  const __nv_bfloat16* kr;     // [T, d_r]
  const int32_t* ids;          // [T] (null with the gate off)
  const int32_t* cu;           // [batch + 1]
  const __nv_bfloat16* gate_table;   // [vocab, d_c]
  const float* gamma;                // [d_c] or null
  const float* beta;
  __nv_bfloat16* ctil;         // [T, d_c]
  __nv_bfloat16* c_pool;       // null: no cache write
  __nv_bfloat16* kr_pool;
  int32_t* id_pool;
  const int32_t* block_table;
  int batch, total, d_c, d_r, vocab, max_pages, num_pages;
  int gate, gate_add, gate_ln;
  float eps;
  int32_t* status;
};

constexpr int kGateWarps = 8;

// c~ of one row from its loaded c and g units, stored, and the row's cache write
__device__ __forceinline__ void gate_row(const PfGateParams& p, int t, int b, int pos, int lane, int nu,
                                         const uint4 (&craw)[2], const uint4 (&graw)[2], bool& bad) {
  float z[2][8];
#pragma unroll
  for (int i = 0; i < 2; ++i) {
    const int u = lane + 32 * i;
    const __nv_bfloat162* c2 = reinterpret_cast<const __nv_bfloat162*>(&craw[i]);
    const __nv_bfloat162* g2 = reinterpret_cast<const __nv_bfloat162*>(&graw[i]);
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const float2 cf = __bfloat1622float2(c2[e]);
      float2 v = cf;
      if (p.gate) {
        const float2 gf = __bfloat1622float2(g2[e]);
        v = p.gate_add ? make_float2(cf.x + gf.x, cf.y + gf.y) : make_float2(cf.x * gf.x, cf.y * gf.y);
      }
      z[i][2 * e] = u < nu ? v.x : 0.f;
      z[i][2 * e + 1] = u < nu ? v.y : 0.f;
    }
  }
  if (p.gate && p.gate_ln) {
    float s = 0.f;
#pragma unroll
    for (int i = 0; i < 2; ++i)
#pragma unroll
      for (int e = 0; e < 8; ++e) s += z[i][e];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
    const float mu = s / p.d_c;
    float q = 0.f;
#pragma unroll
    for (int i = 0; i < 2; ++i)
      if (lane + 32 * i < nu)
#pragma unroll
        for (int e = 0; e < 8; ++e) q = fmaf(z[i][e] - mu, z[i][e] - mu, q);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) q += __shfl_xor_sync(0xffffffffu, q, o);
    const float r = rsqrtf(q / p.d_c + p.eps);
#pragma unroll
    for (int i = 0; i < 2; ++i) {
      const int u = lane + 32 * i;
      if (u >= nu) continue;
#pragma unroll
      for (int e = 0; e < 8; ++e) {
        const float gm = p.gamma ? __ldg(p.gamma + 8 * u + e) : 1.f;
        const float bt = p.beta ? __ldg(p.beta + 8 * u + e) : 0.f;
        z[i][e] = fmaf((z[i][e] - mu) * r, gm, bt);
      }
    }
  }
#pragma unroll
  for (int i = 0; i < 2; ++i) {
    const int u = lane + 32 * i;
    if (u >= nu) continue;
    uint4 o;
    o.x = pack_bf16x2(z[i][0], z[i][1]);
    o.y = pack_bf16x2(z[i][2], z[i][3]);
    o.z = pack_bf16x2(z[i][4], z[i][5]);
    o.w = pack_bf16x2(z[i][6], z[i][7]);
    reinterpret_cast<uint4*>(p.ctil + static_cast<size_t>(t) * p.d_c)[u] = o;
  }
  if (p.c_pool) {
    const int lp = pos / kPage;
    const int page = lp < p.max_pages ? __ldg(p.block_table + static_cast<size_t>(b) * p.max_pages + lp) : -1;
    if (page < 0 || page >= p.num_pages) {
      bad = true;
    } else {
      const size_t slot = static_cast<size_t>(page) * kPage + pos % kPage;
#pragma unroll
      for (int i = 0; i < 2; ++i) {
        const int u = lane + 32 * i;
        if (u < nu) reinterpret_cast<uint4*>(p.c_pool + slot * p.d_c)[u] = craw[i];
      }
      if (lane < p.d_r / 8)
        reinterpret_cast<uint4*>(p.kr_pool + slot * p.d_r)[lane] =
            __ldg(reinterpret_cast<const uint4*>(p.kr + static_cast<size_t>(t) * p.d_r) + lane);
      if (lane == 0 && p.id_pool && p.ids) p.id_pool[slot] = __ldg(p.ids + t);
    }
  }
}

constexpr int kSortMaxBatch = 2048;   // larger batches keep the given order

// One warp per token row.
__global__ void __launch_bounds__(32 * kGateWarps) prefill_gate_kernel(const PfGateParams p) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (blockIdx.x == 0) {
    if (threadIdx.x == 0) *p.next_item = 0;
    // the attention's launch order: longest prompts first (rank of each prompt
    // among all by length, ties by index), so that the longest prompts'
    // query blocks do not start last
    for (int b = threadIdx.x; b < p.batch; b += blockDim.x) {
      int rank = b;
      if (p.batch <= kSortMaxBatch) {
        const int Lb = __ldg(p.cu + b + 1) - __ldg(p.cu + b);
        rank = 0;
        for (int o = 0; o < p.batch; ++o) {
          const int Lo = __ldg(p.cu + o + 1) - __ldg(p.cu + o);
          rank += (Lo > Lb || (Lo == Lb && o < b)) ? 1 : 0;
        }
      }
      p.order[rank] = b;
    }
  }
  const int t = blockIdx.x * kGateWarps + warp;
  if (t >= p.total) return;
  const int nu = p.d_c / 8;   // 16-byte units of a row (at most 64: two per lane)
  const int b = prompt_of_row(p.cu, p.batch, t);
  const int pos = t - __ldg(p.cu + b);
  bool bad = false;
  int id = p.ids ? __ldg(p.ids + t) : 0;
  if (p.gate && static_cast<unsigned>(id) >= static_cast<unsigned>(p.vocab)) {
    bad = true;
    id = 0;
  }
  uint4 craw[2], graw[2];
#pragma unroll
  for (int i = 0; i < 2; ++i) {
    const int u = lane + 32 * i;
    craw[i] = make_uint4(0u, 0u, 0u, 0u);
    graw[i] = make_uint4(0u, 0u, 0u, 0u);
    if (u < nu) craw[i] = __ldg(reinterpret_cast<const uint4*>(p.c + static_cast<size_t>(t) * p.d_c) + u);
    if (p.gate && u < nu)
      graw[i] = __ldg(reinterpret_cast<const uint4*>(p.gate_table + static_cast<size_t>(id) * p.d_c) + u);
  }
  gate_row(p, t, b, pos, lane, nu, craw, graw, bad);
  if (bad && lane == 0) report_status(p.status, kStatusOutOfRange);
}

// ============================================================================ 2. key/value up-projection
// Each CTA owns RT tiles of 128 token rows and walks the output blocks
// (head h, key rows or value rows) in order; every 16 KB chunk of W (128
// output rows x 64 of d_c) that it pulls in feeds the MMAs of all RT row
// tiles, so the weights cross into the SM once per RT x 128 tokens (the
// weight stream, not the tensor pipe, bounds a CTA of one row tile).
constexpr int kKvFeat = kPfDn + kPfDv;                      // 256 output features per head
constexpr int kKvBlock = 128;                               // output columns per block (key or value rows)
constexpr uint32_t kKvBBytes = kKvBlock * kPfChunk * 2;     // 16 KB: one K chunk of a block's W rows
constexpr int kKvMaxStages = 4;
constexpr int kKvEpiWarps = 8;
// output staging: per epilogue warp two 4 KB buffers of 32 rows x 64 columns
// (128-byte swizzle), each stored to global memory by one TMA box
constexpr uint32_t kKvStageOut = 32 * kPfChunk * 2;         // 4 KB
constexpr uint32_t kKvOutBytes = kKvEpiWarps * 2 * kKvStageOut;   // 64 KB
constexpr int kKvThreads = 32 * (2 + kKvEpiWarps);          // warp 0 TMA, warp 1 MMA

struct KvBars {
  uint64_t afull;
  uint64_t bfull[kKvMaxStages], bempty[kKvMaxStages];
  uint64_t dfull[2], dfree[2];
  uint64_t drain;
  uint32_t tmem_base;
  int abort;
};

struct KvParams {
  __nv_bfloat16* kv;   // [T, H, 256]
  int total, H, nkc, stages;
  // kv_mode 1: block b is the key (b even) or value (b odd) rows of head b / 2
  // from the two weight maps; kv_mode 0: block b is rows 128 b .. 128 b + 127
  // of the first map (a plain x W^T, e.g. the gate table E W^UE^T)
  int nblocks, kv_mode;
  int out_cols;   // output row width (elements): stores of chunks past it are skipped
  uint64_t wait_ns;
  int32_t* status;
};

// weight stages that fit next to RT x nkc latent atoms and the output staging
template <int RT>
__host__ __device__ constexpr int kv_stages(int nkc) {
  const long long room = 227LL * 1024 - 2048 - static_cast<long long>(RT * nkc) * kPfAtom - kKvOutBytes;
  const long long st = room / kKvBBytes;
  return st > kKvMaxStages ? kKvMaxStages : static_cast<int>(st);
}
template <int RT>
__host__ __device__ constexpr uint32_t kv_smem_bytes(int nkc) {
  return static_cast<uint32_t>(RT * nkc) * kPfAtom + kKvOutBytes + kv_stages<RT>(nkc) * kKvBBytes + sizeof(KvBars) +
         1024;
}

template <int RT>
__global__ void __launch_bounds__(kKvThreads, 1)
    prefill_kv_kernel(const __grid_constant__ CUtensorMap cmap, const __grid_constant__ CUtensorMap wkmap,
                      const __grid_constant__ CUtensorMap wvmap, const __grid_constant__ CUtensorMap omap,
                      const KvParams p) {
  constexpr uint32_t kTmemCols = 2 * RT * kKvBlock;          // two accumulators of RT x 128 columns
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  const uint32_t sbase = smem_u32(smem);
  const int kKvStages = p.stages;
  const uint32_t o_off = static_cast<uint32_t>(RT * p.nkc) * kPfAtom;
  const uint32_t b_off = o_off + kKvOutBytes;
  KvBars& bars = *reinterpret_cast<KvBars*>(smem + b_off + kKvStages * kKvBBytes);
  volatile int* abort_flag = &bars.abort;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int row0 = blockIdx.x * RT * kPfRows;
  const int nblocks = p.nblocks;
  const int nsteps = nblocks * p.nkc;

  if (tid == 0) {
    mbar_init(smem_u32(&bars.afull), 1);
    for (int s = 0; s < kKvStages; ++s) {
      mbar_init(smem_u32(&bars.bfull[s]), 1);
      mbar_init(smem_u32(&bars.bempty[s]), 1);
    }
    for (int s = 0; s < 2; ++s) {
      mbar_init(smem_u32(&bars.dfull[s]), 1);
      mbar_init(smem_u32(&bars.dfree[s]), kKvEpiWarps);
    }
    mbar_init(smem_u32(&bars.drain), 1);
    bars.abort = 0;
    fence_mbar_init();
    prefetch_tensormap(&cmap);
    prefetch_tensormap(&wkmap);
    prefetch_tensormap(&wvmap);
    prefetch_tensormap(&omap);
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(&bars.tmem_base), kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = bars.tmem_base;

  if (warp == 0) {
    if (elect_one()) {
      const uint64_t pol_stream = policy_evict_first(), pol_keep = policy_evict_last();
      mbar_arrive_expect_tx(smem_u32(&bars.afull), static_cast<uint32_t>(RT * p.nkc) * kPfAtom);
      for (int t = 0; t < RT; ++t)
        for (int kc = 0; kc < p.nkc; ++kc)
          tma_load_2d(sbase + (t * p.nkc + kc) * kPfAtom, &cmap, kc * kPfChunk, row0 + t * kPfRows,
                      smem_u32(&bars.afull), pol_stream);
      int issued = 0;
      for (int i = 0; i < nsteps; ++i) {
        const int s = i % kKvStages;
        if (i >= kKvStages &&
            !mbar_wait(smem_u32(&bars.bempty[s]), ((i / kKvStages) & 1) ^ 1, abort_flag, p.wait_ns))
          break;
        const int blk = i / p.nkc, kc = i % p.nkc;
        mbar_arrive_expect_tx(smem_u32(&bars.bfull[s]), kKvBBytes);
        tma_load_2d(sbase + b_off + s * kKvBBytes, (p.kv_mode && (blk & 1)) ? &wvmap : &wkmap, kc * kPfChunk,
                    (p.kv_mode ? blk >> 1 : blk) * kKvBlock, smem_u32(&bars.bfull[s]), pol_keep);
        issued = i + 1;
      }
      // every copy issued lands before the CTA can leave
      volatile int own = 0;
      if (!mbar_wait(smem_u32(&bars.afull), 0, &own, p.wait_ns)) *abort_flag = 1;
      for (int i = issued > kKvStages ? issued - kKvStages : 0; i < issued; ++i)
        if (!mbar_wait(smem_u32(&bars.bfull[i % kKvStages]), (i / kKvStages) & 1, &own, p.wait_ns))
          *abort_flag = 1;
    }
    __syncwarp();
  } else if (warp == 1) {
    constexpr uint32_t idesc = idesc_bf16(kPfRows, kKvBlock, 0, 0);
    bool ok = pf_warp_wait(smem_u32(&bars.afull), 0, abort_flag, p.wait_ns);
    bool issued = false;
    for (int blk = 0; ok && blk < nblocks; ++blk) {
      const int db = blk & 1;
      if (blk >= 2) ok = pf_warp_wait(smem_u32(&bars.dfree[db]), ((blk - 2) >> 1) & 1, abort_flag, p.wait_ns);
      for (int kc = 0; ok && kc < p.nkc; ++kc) {
        const int i = blk * p.nkc + kc, s = i % kKvStages;
        ok = pf_warp_wait(smem_u32(&bars.bfull[s]), (i / kKvStages) & 1, abort_flag, p.wait_ns);
        if (!ok) break;
        tc_fence_after();
        if (elect_one()) {
          const uint64_t bd = smem_desc(sbase + b_off + s * kKvBBytes, 16, 1024, kSwizzle128B);
#pragma unroll
          for (int t = 0; t < RT; ++t) {
            const uint64_t ad = smem_desc(sbase + (t * p.nkc + kc) * kPfAtom, 16, 1024, kSwizzle128B);
#pragma unroll
            for (int kk = 0; kk < kPfChunk / 16; ++kk)
              mma_bf16_ss(tmem + db * (RT * kKvBlock) + t * kKvBlock, ad + ((kk * 32) >> 4), bd + ((kk * 32) >> 4),
                          idesc, (kc > 0 || kk > 0) ? 1u : 0u);
          }
          mma_commit(smem_u32(&bars.bempty[s]));
          if (kc == p.nkc - 1) mma_commit(smem_u32(&bars.dfull[db]));
        }
        __syncwarp();
        issued = true;
      }
    }
    if (issued) {
      if (elect_one()) mma_commit(smem_u32(&bars.drain));
      __syncwarp();
      volatile int own = 0;
      if (!mbar_wait(smem_u32(&bars.drain), 0, &own, p.wait_ns)) *abort_flag = 1;
    }
    __syncwarp();
  } else {
    // token row = TMEM lane of its row tile; RT = 2: warps 2-5 store row tile
    // 0, warps 6-9 row tile 1 (all 128 columns of a block); RT = 1: warps 2-5
    // store the block's first 64 columns, warps 6-9 the last 64.  Each warp
    // writes its 32 rows x 64 columns into one of its two staging buffers
    // (128-byte swizzle) and its lane 0 stores them with one TMA box.
    const int quad = warp & 3, g = (warp - 2) / 4;
    const int t = RT == 2 ? g : 0;
    constexpr int kCols = RT == 2 ? kKvBlock : kKvBlock / 2;
    const int cbase = RT == 2 ? 0 : g * kCols;
    const int y0 = row0 + t * kPfRows + 32 * quad;           // the warp's first token row
    const uint32_t stg = sbase + o_off + (warp - 2) * 2 * kKvStageOut;
    const uint32_t rowoff = (lane >> 3) * 1024 + (lane & 7) * 128;
    bool ok = true;
    int nst = 0;   // boxes stored so far (buffer nst % 2)
    for (int blk = 0; blk < nblocks; ++blk) {
      const int db = blk & 1;
      ok = ok && pf_warp_wait(smem_u32(&bars.dfull[db]), (blk >> 1) & 1, abort_flag, p.wait_ns);
      if (!ok) break;
      tc_fence_after();
#pragma unroll
      for (int c0 = 0; c0 < kCols; c0 += kPfChunk, ++nst) {
        float v[kPfChunk];
        const uint32_t ta =
            tmem + (static_cast<uint32_t>(32 * quad) << 16) + db * (RT * kKvBlock) + t * kKvBlock + cbase + c0;
#pragma unroll
        for (int c = 0; c < kPfChunk; c += 16) tmem_ld16(ta + c, *reinterpret_cast<float(*)[16]>(&v[c]));
        tmem_wait_ld();
        // the store that last read this buffer (two boxes ago) has read it
        if (lane == 0 && nst >= 2) bulk_wait_group_read<1>();
        __syncwarp();
        const uint32_t buf = stg + (nst & 1) * kKvStageOut + rowoff;
#pragma unroll
        for (int u = 0; u < 8; ++u)
          asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(buf + ((u ^ (lane & 7)) << 4)),
                       "r"(pack_bf16x2(v[8 * u], v[8 * u + 1])), "r"(pack_bf16x2(v[8 * u + 2], v[8 * u + 3])),
                       "r"(pack_bf16x2(v[8 * u + 4], v[8 * u + 5])), "r"(pack_bf16x2(v[8 * u + 6], v[8 * u + 7]))
                       : "memory");
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) {
          // every chunk commits a group (possibly empty), so the buffer
          // rotation above stays in step
          if (blk * kKvBlock + cbase + c0 < p.out_cols)
            tma_store_2d(&omap, blk * kKvBlock + cbase + c0, y0, stg + (nst & 1) * kKvStageOut);
          bulk_commit_group();
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_u32(&bars.dfree[db]));
    }
    if (lane == 0) bulk_wait_group_all();
    __syncwarp();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tmem, kTmemCols);
  if (tid == 0 && bars.abort) report_status(p.status, kStatusTimeout);
}

// ============================================================================ 3. causal flash attention
// Work item (prompt, head, block of 256 queries): two query tiles X = A
// (queries q0 .. q0 + 127) and B (q0 + 128 .. q0 + 255) share every key and
// value tile copied into shared memory, which halves the bytes a CTA pulls in
// per flop (the per-SM copy rate into shared memory, not the tensor pipe,
// bounds a CTA that owns one query tile).  Key tiles are 128 keys; A meets
// tiles 0 .. 2 qb, B tiles 0 .. 2 qb + 1 (qb = q0 / 256).
//
// Tensor memory holds S_X (128 fp32 columns) and O_X (128) of both tiles.
// The softmax threads write P_X in bf16 over the first 64 columns of S_X
// once they have read S_X, and the MMA issuer orders, per key tile j,
//   O_A += P_A(j - 1) V(j - 1);  S_A(j) = Q_A K(j)^T;
//   O_B += P_B(j - 1) V(j - 1);  S_B(j) = Q_B K(j)^T
// in one thread: the MMAs of one issuing thread run in order, so S_X(j)
// overwrites P_X(j - 1) only after the PV MMA has read it, and the commit
// after S_X(j) also covers that PV MMA (O_X is current when the softmax of
// tile j sees S_X(j)).  While the softmax threads of one query tile work, the
// tensor pipe runs the other tile's MMAs.
constexpr int kAttnKeys = 128;                              // keys per tile
constexpr uint32_t kAttnQBytes = 3 * kPfAtom;               // 48 KB: one query tile [128 x 192]
constexpr uint32_t kAttnVBytes = 2 * kPfAtom;               // 32 KB: V [128 keys x 128]
// key tiles arrive as three 16 KB chunks (k^C columns 0-63, 64-127, k^R)
// in a ring of four chunk slots, so the next tile's first chunks land while
// the last score MMAs of the current tile still read it; values in two stages
constexpr int kAttnKSlots = 4;
constexpr int kAttnVStages = 2;
constexpr uint32_t kOffQ = 0;
constexpr uint32_t kOffK = kOffQ + 2 * kAttnQBytes;
constexpr uint32_t kOffV = kOffK + kAttnKSlots * kPfAtom;
constexpr uint32_t kOffBars = kOffV + kAttnVStages * kAttnVBytes;
// warp 0: work items, query and key copies; warp 1: MMAs; warps 2-9: softmax
// and epilogue (2-5 tile A, 6-9 tile B, warp w reading TMEM lane quadrant
// w % 4); warp 10: value copies
constexpr int kAttnSoftWarp0 = 2;
constexpr int kAttnVWarp = 10;
constexpr int kAttnThreads = 32 * (kAttnVWarp + 1);
// TMEM columns: S_X (P_X over its first 64 columns) and O_X
__host__ __device__ constexpr uint32_t col_s(int x) { return x * kAttnKeys; }
__host__ __device__ constexpr uint32_t col_o(int x) { return 256 + x * kPfDv; }
constexpr float kRescaleLog2 = 8.f;

struct AttnItem {
  int b, h, qb, start, L;   // b < 0: no more work
};

struct AttnBars {
  uint64_t qfull, qempty;
  uint64_t kfull[kAttnKSlots], kempty[kAttnKSlots];
  uint64_t vfull[kAttnVStages], vempty[kAttnVStages];
  uint64_t sfull[2], pfull[2], odone[2], ofree[2];   // per query tile
  uint64_t ifull[2], iempty[2];                      // the work-item ring
  uint64_t drain;
  AttnItem item[2];
  uint32_t tmem_base;
  int abort;
};
constexpr uint32_t kAttnSmem = kOffBars + sizeof(AttnBars) + 1024;
constexpr int kAttnItemReaders = 2 + 8;   // MMA warp, value loader, eight softmax warps

struct AttnParams {
  const int32_t* cu;
  const int32_t* order;   // prompts in launch order
  int32_t* next_item;     // work counter, zeroed by the gate kernel
  __nv_bfloat16* out;     // [T, H, d_v]
  int batch, H, qblocks, total, items;
  float scale_log2;
  uint64_t wait_ns;
  int32_t* status;
};

// Persistent: one CTA per SM takes (prompt, head, 256-query block) items from
// a counter, in launch order (prompts longest first, heads, blocks heaviest
// first), so that the next item's query and key copies overlap the current
// item's last tiles and epilogue.  Every barrier's phases run on across items.
__global__ void __launch_bounds__(kAttnThreads, 1)
    prefill_attn_kernel(const __grid_constant__ CUtensorMap qmap, const __grid_constant__ CUtensorMap kvmap,
                        const __grid_constant__ CUtensorMap krmap, const AttnParams p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  const uint32_t sbase = smem_u32(smem);
  AttnBars& bars = *reinterpret_cast<AttnBars*>(smem + kOffBars);
  volatile int* abort_flag = &bars.abort;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

  if (tid == 0) {
    mbar_init(smem_u32(&bars.qfull), 1);
    mbar_init(smem_u32(&bars.qempty), 1);
    for (int s = 0; s < kAttnKSlots; ++s) {
      mbar_init(smem_u32(&bars.kfull[s]), 1);
      mbar_init(smem_u32(&bars.kempty[s]), 1);
    }
    for (int s = 0; s < kAttnVStages; ++s) {
      mbar_init(smem_u32(&bars.vfull[s]), 1);
      mbar_init(smem_u32(&bars.vempty[s]), 1);
    }
    for (int x = 0; x < 2; ++x) {
      mbar_init(smem_u32(&bars.sfull[x]), 1);
      mbar_init(smem_u32(&bars.pfull[x]), 4);
      mbar_init(smem_u32(&bars.odone[x]), 1);
      mbar_init(smem_u32(&bars.ofree[x]), 4);
      mbar_init(smem_u32(&bars.ifull[x]), 1);
      mbar_init(smem_u32(&bars.iempty[x]), kAttnItemReaders);
    }
    mbar_init(smem_u32(&bars.drain), 1);
    bars.abort = 0;
    fence_mbar_init();
    prefetch_tensormap(&qmap);
    prefetch_tensormap(&kvmap);
    prefetch_tensormap(&krmap);
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(&bars.tmem_base), 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = bars.tmem_base;

  // item n of this CTA sits in ring slot n % 2; a reader copies it out, then frees the slot
  auto read_item = [&](int n, AttnItem& it, bool arrive) -> bool {
    if (!pf_warp_wait(smem_u32(&bars.ifull[n & 1]), (n >> 1) & 1, abort_flag, p.wait_ns)) return false;
    it = bars.item[n & 1];
    __syncwarp();
    if (arrive && lane == 0) mbar_arrive(smem_u32(&bars.iempty[n & 1]));
    return true;
  };
  auto tiles_of = [&](const AttnItem& it, int (&nt)[2]) {
    const int q0 = it.qb * 2 * kPfRows;
    const bool has_b = q0 + kPfRows < it.L;
    nt[0] = 2 * it.qb + 1;
    nt[1] = has_b ? 2 * it.qb + 2 : 0;
  };

  if (warp == 0) {
    // ---- work items, the query tiles of each, and the key tiles: k^C of
    // head h (two 64-column chunks of the kv buffer) and the shared k^R rows
    if (elect_one()) {
      const uint64_t pol_q = policy_evict_first(), pol_k = policy_evict_last();
      int g = 0;       // key chunks issued (chunk g in slot g % 4)
      int n = 0;       // items published
      bool ok = true;
      while (ok) {
        // the next non-empty item, or the end
        AttnItem it;
        it.b = -1;
        for (;;) {
          const int i = atomicAdd(p.next_item, 1);
          if (i >= p.items) break;
          const int group = i / p.qblocks;
          const int qb = p.qblocks - 1 - i % p.qblocks;
          const int b = __ldg(p.order + group / p.H), h = group % p.H;
          const int start = __ldg(p.cu + b);
          const int L = __ldg(p.cu + b + 1) - start;
          // prompt offsets that do not fit the packed rows, or a prompt longer
          // than the host bound: report, compute nothing past it
          if (start < 0 || L < 0 || start > p.total - L) {
            report_status(p.status, kStatusOutOfRange);
            continue;
          }
          if (qb == p.qblocks - 1 && L > p.qblocks * 2 * kPfRows) report_status(p.status, kStatusOutOfRange);
          if (qb * 2 * kPfRows >= L) continue;
          it.b = b; it.h = h; it.qb = qb; it.start = start; it.L = L;
          break;
        }
        if (n >= 2 && !mbar_wait(smem_u32(&bars.iempty[n & 1]), ((n >> 1) & 1) ^ 1, abort_flag, p.wait_ns)) break;
        bars.item[n & 1] = it;
        mbar_arrive(smem_u32(&bars.ifull[n & 1]));
        if (it.b < 0) break;
        int nt[2];
        tiles_of(it, nt);
        const int nkt = nt[1] > 0 ? nt[1] : nt[0];
        // the query tiles once the previous item's score MMAs are done with them
        if (n >= 1 && !mbar_wait(smem_u32(&bars.qempty), (n - 1) & 1, abort_flag, p.wait_ns)) break;
        const int nq = nt[1] > 0 ? 2 : 1;
        mbar_arrive_expect_tx(smem_u32(&bars.qfull), nq * kAttnQBytes);
        for (int x = 0; x < nq; ++x)
          for (int c = 0; c < 3; ++c)
            tma_load_2d(sbase + kOffQ + x * kAttnQBytes + c * kPfAtom, &qmap, it.h * kPfDqk + c * kPfChunk,
                        it.start + it.qb * 2 * kPfRows + x * kPfRows, smem_u32(&bars.qfull), pol_q);
        for (int j = 0; ok && j < nkt; ++j) {
          const int y = it.start + j * kAttnKeys;
          for (int c = 0; c < 3; ++c, ++g) {
            const int s = g % kAttnKSlots;
            if (g >= kAttnKSlots &&
                !mbar_wait(smem_u32(&bars.kempty[s]), ((g / kAttnKSlots) & 1) ^ 1, abort_flag, p.wait_ns)) {
              ok = false;
              break;
            }
            mbar_arrive_expect_tx(smem_u32(&bars.kfull[s]), kPfAtom);
            if (c < 2)
              tma_load_2d(sbase + kOffK + s * kPfAtom, &kvmap, it.h * kKvFeat + c * kPfChunk, y,
                          smem_u32(&bars.kfull[s]), pol_k);
            else
              tma_load_2d(sbase + kOffK + s * kPfAtom, &krmap, 0, y, smem_u32(&bars.kfull[s]), pol_k);
          }
        }
        ++n;
      }
      // every copy issued lands before the CTA can leave (own flag: bounded, not cut short)
      volatile int own = 0;
      for (int q = g > kAttnKSlots ? g - kAttnKSlots : 0; q < g; ++q)
        if (!mbar_wait(smem_u32(&bars.kfull[q % kAttnKSlots]), (q / kAttnKSlots) & 1, &own, p.wait_ns))
          *abort_flag = 1;
      if (n >= 1 && !mbar_wait(smem_u32(&bars.qfull), (n - 1) & 1, &own, p.wait_ns)) *abort_flag = 1;
    }
    __syncwarp();
  } else if (warp == kAttnVWarp) {
    // ---- value tiles: v^C of head h, two stages, each refilled once both
    // PV MMAs that read it have completed
    // (lane 0 issues; the whole warp reads the items)
    int vt = 0;   // value tiles issued (tile vt in stage vt % 2), kept by lane 0
    const uint64_t pol_v = policy_evict_last();
    for (int n = 0;; ++n) {
      AttnItem it;
      if (!read_item(n, it, true) || it.b < 0) break;
      int nt[2];
      tiles_of(it, nt);
      const int nkt = nt[1] > 0 ? nt[1] : nt[0];
      int ok = 1;
      if (lane == 0) {
        for (int j = 0; j < nkt; ++j, ++vt) {
          const int s = vt % kAttnVStages;
          if (vt >= kAttnVStages &&
              !mbar_wait(smem_u32(&bars.vempty[s]), ((vt / kAttnVStages) & 1) ^ 1, abort_flag, p.wait_ns)) {
            ok = 0;
            break;
          }
          const int y = it.start + j * kAttnKeys;
          const uint32_t dst = sbase + kOffV + s * kAttnVBytes;
          mbar_arrive_expect_tx(smem_u32(&bars.vfull[s]), kAttnVBytes);
          tma_load_2d(dst, &kvmap, it.h * kKvFeat + kPfDn, y, smem_u32(&bars.vfull[s]), pol_v);
          tma_load_2d(dst + kPfAtom, &kvmap, it.h * kKvFeat + kPfDn + kPfChunk, y, smem_u32(&bars.vfull[s]),
                      pol_v);
        }
      }
      if (!__shfl_sync(0xffffffffu, ok, 0)) break;
    }
    if (lane == 0) {
      volatile int own = 0;
      for (int q = vt > kAttnVStages ? vt - kAttnVStages : 0; q < vt; ++q)
        if (!mbar_wait(smem_u32(&bars.vfull[q % kAttnVStages]), (q / kAttnVStages) & 1, &own, p.wait_ns))
          *abort_flag = 1;
    }
    __syncwarp();
  } else if (warp == 1) {
    // ---- MMAs.  Per key tile j and query tile X: O_X += P_X(j - 1) V(j - 1),
    // then S_X(j) = Q_X K(j)^T (see the header for why in this order)
    constexpr uint32_t idesc_s = idesc_bf16(kPfRows, kAttnKeys, 0, 0);
    constexpr uint32_t idesc_o = idesc_bf16(kPfRows, kPfDv, 0, 1);
    const uint64_t qdesc = smem_desc(sbase + kOffQ, 16, 1024, kSwizzle128B);
    const uint64_t kdesc = smem_desc(sbase + kOffK, 16, 1024, kSwizzle128B);
    // V [keys x features] is the B operand MN-major: 64-feature atoms 16 KB
    // apart, 8-key groups 1 KB apart
    const uint64_t vdesc = smem_desc(sbase + kOffV, kPfAtom, 1024, kSwizzle128B);
    bool ok = true, issued = false;
    int g0 = 0, v0 = 0;              // first key chunk and value tile of the item
    int tx[2] = {0, 0};              // tiles of query tile X before this item
    int kx[2] = {0, 0};              // items in which query tile X had rows
    int kseen = -1;                  // the last key chunk whose arrival was waited for
    for (int n = 0; ok; ++n) {
      AttnItem it;
      if (!read_item(n, it, true) || it.b < 0) break;
      int ntile[2];
      tiles_of(it, ntile);
      const int nkt = ntile[1] > 0 ? ntile[1] : ntile[0];
      ok = pf_warp_wait(smem_u32(&bars.qfull), n & 1, abort_flag, p.wait_ns);
      auto wait_k = [&](int g) {
        if (kseen < g) {
          ok = ok && pf_warp_wait(smem_u32(&bars.kfull[g % kAttnKSlots]), (g / kAttnKSlots) & 1, abort_flag,
                                  p.wait_ns);
          kseen = g;
        }
      };
      // O_X += P_X(i) V(i); the last reader of V(i) frees it, the last PV of X signals its epilogue
      auto issue_pv = [&](int x, int i) {
        const int vi = v0 + i, vs = vi % kAttnVStages;
        if (x == 0 || ntile[0] <= i)   // first reader of V(i)
          ok = ok && pf_warp_wait(smem_u32(&bars.vfull[vs]), (vi / kAttnVStages) & 1, abort_flag, p.wait_ns);
        // the first PV MMA of X in this item overwrites O_X: its last item's epilogue has read it
        if (i == 0 && kx[x] >= 1)
          ok = ok && pf_warp_wait(smem_u32(&bars.ofree[x]), (kx[x] - 1) & 1, abort_flag, p.wait_ns);
        ok = ok && pf_warp_wait(smem_u32(&bars.pfull[x]), (tx[x] + i) & 1, abort_flag, p.wait_ns);
        if (!ok) return;
        tc_fence_after();
        if (elect_one()) {
          const uint64_t vd = vdesc + ((vs * kAttnVBytes) >> 4);
          // A = P_X from tensor memory: 16 keys per MMA are 8 columns of bf16 pairs
#pragma unroll
          for (int ks = 0; ks < kAttnKeys / 16; ++ks)
            mma_bf16_ts(tmem + col_o(x), tmem + col_s(x) + ks * 8, vd + ((ks * 2048) >> 4), idesc_o,
                        (i > 0 || ks > 0) ? 1u : 0u);
          if (x == 1 || ntile[1] <= i) mma_commit(smem_u32(&bars.vempty[vs]));
          if (i == ntile[x] - 1) mma_commit(smem_u32(&bars.odone[x]));
        }
        __syncwarp();
        issued = true;
      };
      auto issue_s = [&](int x, int j) {
        const uint64_t qd = qdesc + ((x * kAttnQBytes) >> 4);
        // the last reader of a key chunk (B, or A when B has no tile j) frees its slot
        const bool last_reader = x == 1 || ntile[1] <= j;
        for (int c = 0; c < 3; ++c) {
          const int g = g0 + 3 * j + c, s = g % kAttnKSlots;
          wait_k(g);
          if (!ok) return;
          tc_fence_after();
          if (elect_one()) {
            const uint64_t kd = kdesc + ((s * kPfAtom) >> 4);
#pragma unroll
            for (int kk = 0; kk < 4; ++kk)
              mma_bf16_ss(tmem + col_s(x), qd + ((c * kPfAtom + kk * 32) >> 4), kd + ((kk * 32) >> 4), idesc_s,
                          (c > 0 || kk > 0) ? 1u : 0u);
            if (c == 2) mma_commit(smem_u32(&bars.sfull[x]));
            if (last_reader) mma_commit(smem_u32(&bars.kempty[s]));
            // the item's last score MMAs done: the query tiles may be refilled
            if (c == 2 && last_reader && j == nkt - 1) mma_commit(smem_u32(&bars.qempty));
          }
          __syncwarp();
        }
        issued = true;
      };
      for (int j = 0; ok && j <= nkt; ++j) {
        for (int x = 0; ok && x < 2; ++x) {
          if (j >= 1 && j - 1 < ntile[x]) issue_pv(x, j - 1);
          if (ok && j < ntile[x]) issue_s(x, j);
        }
      }
      g0 += 3 * nkt;
      v0 += nkt;
      for (int x = 0; x < 2; ++x) {
        tx[x] += ntile[x];
        if (ntile[x] > 0) ++kx[x];
      }
    }
    if (issued) {
      if (elect_one()) mma_commit(smem_u32(&bars.drain));
      __syncwarp();
      volatile int own = 0;
      if (!mbar_wait(smem_u32(&bars.drain), 0, &own, p.wait_ns)) *abort_flag = 1;
    }
    __syncwarp();
  } else {
    // ---- softmax and epilogue of query tile x: query row r = TMEM lane r
    const int x = (warp - kAttnSoftWarp0) >> 2;
    const int quad = warp & 3;
    const int r = 32 * quad + lane;
    const uint32_t lane_base = tmem + (static_cast<uint32_t>(32 * quad) << 16);
    const float sl2 = p.scale_log2;
    int tx = 0, kx = 0;   // tiles and items of X before this item
    bool ok = true;
    for (int n = 0; ok; ++n) {
      AttnItem it;
      if (!read_item(n, it, true) || it.b < 0) break;
      int ntile[2];
      tiles_of(it, ntile);
      const int nx = ntile[x];
      if (nx == 0) continue;
      const int qrow = it.qb * 2 * kPfRows + x * kPfRows + r;   // this row's position in the prompt
      float m_ref = 0.f, l = 0.f;
      for (int j = 0; ok && j < nx; ++j) {
        // S_X(j) complete (and with it every earlier MMA: O_X is current)
        ok = pf_warp_wait(smem_u32(&bars.sfull[x]), (tx + j) & 1, abort_flag, p.wait_ns);
        if (!ok) break;
        tc_fence_after();
        float sv[kAttnKeys];
#pragma unroll
        for (int c = 0; c < kAttnKeys; c += 16)
          tmem_ld16(lane_base + col_s(x) + c, *reinterpret_cast<float(*)[16]>(&sv[c]));
        tmem_wait_ld();
        const int k0 = j * kAttnKeys;
        if (k0 + kAttnKeys - 1 > qrow) {
          // keys after the query (the tile on the diagonal)
#pragma unroll
          for (int c = 0; c < kAttnKeys; ++c)
            if (k0 + c > qrow) sv[c] = -INFINITY;
        }
        // row maximum and sum as eight interleaved chains (short dependencies)
        float m8[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) m8[e] = sv[e];
#pragma unroll
        for (int c = 8; c < kAttnKeys; ++c) m8[c & 7] = fmaxf(m8[c & 7], sv[c]);
        float mx =
            fmaxf(fmaxf(fmaxf(m8[0], m8[1]), fmaxf(m8[2], m8[3])), fmaxf(fmaxf(m8[4], m8[5]), fmaxf(m8[6], m8[7])));
        mx *= sl2;
        float alpha = 1.f;
        if (j == 0) {
          m_ref = mx;
        } else if (mx > m_ref + kRescaleLog2) {
          alpha = pf_ex2(m_ref - mx);
          m_ref = mx;
        }
        float pk[kAttnKeys / 2];   // bf16 pairs, kept as 32-bit words for the TMEM store
        float r8[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int c = 0; c < kAttnKeys; c += 2) {
          const float p0 = pf_ex2(fmaf(sv[c], sl2, -m_ref));
          const float p1 = pf_ex2(fmaf(sv[c + 1], sl2, -m_ref));
          r8[(c >> 1) & 7] += p0 + p1;
          pk[c / 2] = __uint_as_float(pack_bf16x2(p0, p1));
        }
        const float rs = ((r8[0] + r8[1]) + (r8[2] + r8[3])) + ((r8[4] + r8[5]) + (r8[6] + r8[7]));
        l = fmaf(l, alpha, rs);
        if (__any_sync(0xffffffffu, alpha != 1.f)) {
#pragma unroll
          for (int c = 0; c < kPfDv; c += 16) {
            float o[16];
            tmem_ld16(lane_base + col_o(x) + c, o);
            tmem_wait_ld();
#pragma unroll
            for (int e = 0; e < 16; ++e) o[e] *= alpha;
            tmem_st16(lane_base + col_o(x) + c, o);
          }
        }
        // P_X over the first 64 columns of S_X
#pragma unroll
        for (int c = 0; c < kAttnKeys / 2; c += 16)
          tmem_st16(lane_base + col_s(x) + c, *reinterpret_cast<const float(*)[16]>(&pk[c]));
        tmem_wait_st();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(smem_u32(&bars.pfull[x]));
      }
      // ---- epilogue: O_X / l of the live rows, then O_X is free for the next item
      if (ok) ok = pf_warp_wait(smem_u32(&bars.odone[x]), kx & 1, abort_flag, p.wait_ns);
      if (!ok) break;
      tc_fence_after();
      const float inv = 1.f / l;
      const bool live = qrow < it.L;
      __nv_bfloat16* orow = p.out + (static_cast<size_t>(it.start + (live ? qrow : 0)) * p.H + it.h) * kPfDv;
      float o[kPfDv];
#pragma unroll
      for (int c = 0; c < kPfDv; c += 16) tmem_ld16(lane_base + col_o(x) + c, *reinterpret_cast<float(*)[16]>(&o[c]));
      tmem_wait_ld();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_u32(&bars.ofree[x]));
      if (live) {
        uint4* d = reinterpret_cast<uint4*>(orow);
#pragma unroll
        for (int q = 0; q < kPfDv / 8; ++q)
          d[q] = make_uint4(pack_bf16x2(o[8 * q] * inv, o[8 * q + 1] * inv),
                            pack_bf16x2(o[8 * q + 2] * inv, o[8 * q + 3] * inv),
                            pack_bf16x2(o[8 * q + 4] * inv, o[8 * q + 5] * inv),
                            pack_bf16x2(o[8 * q + 6] * inv, o[8 * q + 7] * inv));
      }
      tx += nx;
      ++kx;
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tmem, 512);
  if (tid == 0 && bars.abort) report_status(p.status, kStatusTimeout);
}

// ---------------------------------------------------------------- host
using EncodeFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                              const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                              CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeFn pf_encode_fn() {
  static EncodeFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeFn>(ptr);
  });
  return fn;
}

// row-major bf16 [rows, cols] with row stride `ld` elements; boxes of 64
// columns x box_rows rows, 128-byte swizzle, rows past the end read as zero
bool pf_encode(CUtensorMap* map, const void* base, uint64_t rows, uint64_t cols, uint64_t ld,
               uint32_t box_rows = kPfRows) {
  EncodeFn enc = pf_encode_fn();
  if (enc == nullptr) return false;
  std::memset(map, 0, sizeof(*map));
  const cuuint64_t dims[2] = {cols, rows};
  const cuuint64_t strides[1] = {ld * 2};
  const cuuint32_t box[2] = {static_cast<cuuint32_t>(kPfChunk), box_rows};
  const cuuint32_t estr[2] = {1, 1};
  return enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

struct PfWorkspace {
  size_t off_order, off_ctil, off_kv, total;
};

PfWorkspace pf_layout(int batch, int total, int H, int d_c) {
  PfWorkspace w;
  size_t off = 0;
  w.off_order = off;   // the prompt order, then the attention's work counter
  off = align_up(off + static_cast<size_t>(batch + 1) * 4, 256);
  w.off_ctil = off;
  off = align_up(off + static_cast<size_t>(total) * d_c * 2, 256);
  w.off_kv = off;
  off = align_up(off + static_cast<size_t>(total) * H * kKvFeat * 2, 256);
  w.total = off;
  return w;
}

}  // namespace

size_t prefill_workspace_bytes(int batch, int total_tokens, int H, int d_c) {
  return pf_layout(batch, total_tokens, H, d_c).total;
}

bool prefill_supported(int d_nope, int d_rope, int d_v, int d_c) {
  return d_nope == kPfDn && d_rope == kPfDr && d_v == kPfDv && d_c % kPfChunk == 0 && d_c >= kPfChunk &&
         d_c <= 512;
}

cudaError_t launch_prefill(const PrefillArgs& a, cudaStream_t st, void (*mark)(cudaStream_t, bool)) {
  if (a.total <= 0 || a.batch <= 0) return cudaSuccess;
  const PfWorkspace w = pf_layout(a.batch, a.total, a.H, a.d_c);
  uint8_t* ws = static_cast<uint8_t*>(a.workspace);
  int32_t* order = reinterpret_cast<int32_t*>(ws + w.off_order);
  __nv_bfloat16* ctil = reinterpret_cast<__nv_bfloat16*>(ws + w.off_ctil);
  __nv_bfloat16* kv = reinterpret_cast<__nv_bfloat16*>(ws + w.off_kv);

  // 1. gate, LayerNorm, cache write
  PfGateParams gp;
  gp.order = order;
  gp.next_item = order + a.batch;
  gp.c = static_cast<const __nv_bfloat16*>(a.c);
  gp.kr = static_cast<const __nv_bfloat16*>(a.kr);
  gp.ids = a.ids;
  gp.cu = a.cu_seqlens;
  gp.gate_table = static_cast<const __nv_bfloat16*>(a.gate_table);
  gp.gamma = a.ln_gamma;
  gp.beta = a.ln_beta;
  gp.ctil = ctil;
  gp.c_pool = static_cast<__nv_bfloat16*>(a.c_pool);
  gp.kr_pool = static_cast<__nv_bfloat16*>(a.kr_pool);
  gp.id_pool = a.id_pool;
  gp.block_table = a.block_table;
  gp.batch = a.batch;
  gp.total = a.total;
  gp.d_c = a.d_c;
  gp.d_r = kPfDr;
  gp.vocab = a.vocab;
  gp.max_pages = a.max_pages;
  gp.num_pages = a.num_pages;
  gp.gate = a.gate;
  gp.gate_add = a.gate_add;
  gp.gate_ln = a.gate_ln;
  gp.eps = a.eps;
  gp.status = a.status;
  prefill_gate_kernel<<<(a.total + kGateWarps - 1) / kGateWarps, 32 * kGateWarps, 0, st>>>(gp);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;

  // 2. keys and values of every head: one 128-row tile per CTA.  Its output
  // stores and its weight copies bound it about equally per SM, so spreading
  // the stores over more CTAs beats reading the weights fewer times (measured:
  // two tiles per CTA took 114 us against 109 at 8 x 4096)
  CUtensorMap cmap, wkmap, wvmap;
  if (!pf_encode(&cmap, ctil, a.total, a.d_c, a.d_c)) return cudaErrorInvalidValue;
  if (!pf_encode(&wkmap, a.w_uk, static_cast<uint64_t>(a.H) * kPfDn, a.d_c, a.d_c)) return cudaErrorInvalidValue;
  if (!pf_encode(&wvmap, a.w_uv, static_cast<uint64_t>(a.H) * kPfDv, a.d_c, a.d_c)) return cudaErrorInvalidValue;
  const int nkc = a.d_c / kPfChunk;
  CUtensorMap omap;   // the kv buffer, stored in boxes of 64 columns x 32 rows
  if (!pf_encode(&omap, kv, a.total, static_cast<uint64_t>(a.H) * kKvFeat, static_cast<uint64_t>(a.H) * kKvFeat, 32))
    return cudaErrorInvalidValue;
  KvParams kp;
  kp.kv = kv;
  kp.total = a.total;
  kp.H = a.H;
  kp.nkc = nkc;
  kp.wait_ns = kWaitLimitNs;
  kp.status = a.status;
  kp.nblocks = 2 * a.H;
  kp.kv_mode = 1;
  kp.out_cols = a.H * kKvFeat;
  {
    kp.stages = kv_stages<1>(nkc);
    const int kv_smem = static_cast<int>(kv_smem_bytes<1>(nkc));
    e = cudaFuncSetAttribute(prefill_kv_kernel<1>, cudaFuncAttributeMaxDynamicSharedMemorySize, kv_smem);
    if (e != cudaSuccess) return e;
    prefill_kv_kernel<1><<<(a.total + kPfRows - 1) / kPfRows, kKvThreads, kv_smem, st>>>(cmap, wkmap, wvmap, omap,
                                                                                         kp);
  }
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;

  // 3. causal attention
  CUtensorMap qmap, kvmap, krmap;
  if (!pf_encode(&qmap, a.q, a.total, static_cast<uint64_t>(a.H) * kPfDqk, static_cast<uint64_t>(a.H) * kPfDqk))
    return cudaErrorInvalidValue;
  if (!pf_encode(&kvmap, kv, a.total, static_cast<uint64_t>(a.H) * kKvFeat, static_cast<uint64_t>(a.H) * kKvFeat))
    return cudaErrorInvalidValue;
  if (!pf_encode(&krmap, a.kr, a.total, kPfDr, kPfDr)) return cudaErrorInvalidValue;
  e = cudaFuncSetAttribute(prefill_attn_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           static_cast<int>(kAttnSmem));
  if (e != cudaSuccess) return e;
  AttnParams ap;
  ap.cu = a.cu_seqlens;
  ap.order = order;
  ap.next_item = order + a.batch;
  ap.out = static_cast<__nv_bfloat16*>(a.out);
  ap.batch = a.batch;
  ap.H = a.H;
  ap.total = a.total;
  ap.qblocks = (a.max_seq_len + 2 * kPfRows - 1) / (2 * kPfRows);
  ap.scale_log2 = a.scale_log2;
  ap.wait_ns = kWaitLimitNs;
  ap.status = a.status;
  if (ap.qblocks == 0) return cudaSuccess;
  const long long items = static_cast<long long>(a.batch) * a.H * ap.qblocks;
  if (items > 0x7fffffffLL) return cudaErrorInvalidValue;
  ap.items = static_cast<int>(items);
  int dev = 0, sms = 0;
  e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (e != cudaSuccess) return e;
  const int grid = static_cast<int>(items < sms ? items : sms);
  if (mark) mark(st, true);
  prefill_attn_kernel<<<grid, kAttnThreads, kAttnSmem, st>>>(qmap, kvmap, krmap, ap);
  e = cudaGetLastError();
  if (mark) mark(st, false);
  return e;
}

cudaError_t launch_gate_table(const void* emb, const void* w_ue, int vocab, int d_e, int d_c, void* table,
                              int32_t* status, cudaStream_t st) {
  if (vocab <= 0) return cudaSuccess;
  CUtensorMap amap, wmap, omap;
  if (!pf_encode(&amap, emb, vocab, d_e, d_e)) return cudaErrorInvalidValue;
  if (!pf_encode(&wmap, w_ue, d_c, d_e, d_e)) return cudaErrorInvalidValue;
  if (!pf_encode(&omap, table, vocab, d_c, d_c, 32)) return cudaErrorInvalidValue;
  const int nkc = d_e / kPfChunk;
  KvParams kp;
  kp.kv = static_cast<__nv_bfloat16*>(table);
  kp.total = vocab;
  kp.H = 0;
  kp.nkc = nkc;
  kp.wait_ns = kWaitLimitNs;
  kp.status = status;
  kp.nblocks = (d_c + kKvBlock - 1) / kKvBlock;   // the last block's rows past d_c read as zero
  kp.kv_mode = 0;
  kp.out_cols = d_c;
  cudaError_t e;
  if (nkc <= 4) {
    kp.stages = kv_stages<2>(nkc);
    const int smem = static_cast<int>(kv_smem_bytes<2>(nkc));
    e = cudaFuncSetAttribute(prefill_kv_kernel<2>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    prefill_kv_kernel<2><<<(vocab + 2 * kPfRows - 1) / (2 * kPfRows), kKvThreads, smem, st>>>(amap, wmap, wmap, omap,
                                                                                              kp);
  } else {
    kp.stages = kv_stages<1>(nkc);
    const int smem = static_cast<int>(kv_smem_bytes<1>(nkc));
    e = cudaFuncSetAttribute(prefill_kv_kernel<1>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    prefill_kv_kernel<1><<<(vocab + kPfRows - 1) / kPfRows, kKvThreads, smem, st>>>(amap, wmap, wmap, omap, kp);
  }
  return cudaGetLastError();
}

}  // namespace egmla
