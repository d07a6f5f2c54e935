// egmla_r0.cu - decode with the paper-literal gate placement (R0): the gate
// and the LayerNorm act on the up-projected keys and values of all heads,
// kv~ = LN_{H(d_n + d_v)}((W^UKV c) (*) g) (Section 3 Eq. 5 applied after
// Eq. 2, as the Appendix E listing does), split per head into k^C, v^C
// (Eq. 6), then attention as in Eqs. 11-13 without absorption (the gate in
// the 4096-wide space cannot be folded into the query).
//
// The LayerNorm needs all 4096 features of a token before any head's key or
// value is final, but the scores do not need the normalised keys:
//   q . k~ = r (q gamma) . z_k - r mu sum(q gamma) + q . beta,
// so the up-projection computes every head's raw dot (q gamma) . z_k while
// it has z_k in registers and keeps only the gated values.  Two kernels:
//   r0_project_kernel  (tcgen05) one tile of two cache pages (128 tokens,
//                      the MMA's M) of the walk over every sequence's pages:
//                      for each head h, D = C W^UKV_h^T (N = 256 = d_n + d_v
//                      features, K = d_c) in one of two TMEM accumulators, so
//                      that the epilogue of head h overlaps the MMAs of head
//                      h + 1.  Epilogue warps, one row each (their R0 gate
//                      values G_R0[id] of head h + 1 requested a quarter at a
//                      time while head h is processed): the key half gates
//                      its 128 features, rounds z to bf16 and adds
//                      (q gamma) . z to the row's head dots; the value half
//                      gates and rounds its 128 features and stores them
//                      head-major through a per-warp shared-memory tile (two
//                      256-byte rows, 512 contiguous bytes, per store
//                      instruction).  Both
//                      add z and z^2 of the rounded values into the row's
//                      statistics.  After the last head: (mu, 1/sqrt(var +
//                      eps)) and every head's logit
//                        s = scale log2(e) (r ((q gamma) . z_k - mu sum(q gamma)) + q . beta + q^R . k^R).
//   r0_attend_kernel   one block per (sequence, head): an online softmax over
//                      the logits and, with P' = p r,
//                        o = gamma_v ((sum P' z_v - sum P' mu) / sum p) + beta_v,
//                      streaming 256 bytes of gated values per token.
// The gated values (H d_v bf16 per pool row, head-major) are identical for
// every sequence that holds a page, so a page shared by two sequences is
// written twice with the same bytes; the logits are per (sequence, position).
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
constexpr int kR0Half = 128;                    // d_n = d_v
constexpr int kR0Rope = 64;
constexpr int kR0Width = kR0Heads * kR0Feat;    // 4096
constexpr int kR0Rows = 2 * kPage;              // tile rows: two pages (the MMA's M)
constexpr int kR0Chunk = 64;                    // K elements per operand chunk (128-byte swizzle atom)
constexpr uint32_t kR0AChunkBytes = kR0Rows * kR0Chunk * 2;   // 16 KB
constexpr uint32_t kR0APageBytes = kPage * kR0Chunk * 2;      // 8 KB: one page's rows of a chunk
constexpr uint32_t kR0BChunkBytes = kR0Feat * kR0Chunk * 2;   // 32 KB
constexpr int kR0BStages = 3;
constexpr int kR0EpiWarps = 8;                  // warps 2-5 key half, 6-9 value half (one TMEM lane quadrant each)
constexpr int kR0Threads = 32 * (2 + kR0EpiWarps);   // warp 0 TMA, warp 1 MMA, warps 2-9 epilogue
constexpr uint32_t kR0TmemCols = 512;           // two 256-column accumulators
constexpr int kR0S1Stride = kR0Heads + 1;       // row stride of the head dots (no bank conflicts)
constexpr int kR0EpiBar = 1;                    // named barrier of the epilogue warps
constexpr uint32_t kR0RowBytes = kR0Half * 2;   // one row's gated values of a head: 256 bytes

// shared memory after the latent tile and the W^UKV stages
struct R0Smem {
  float qg[2][kR0Heads][kR0Half];       // q_h (*) gamma_k,h of the tile's two sequences
  __nv_bfloat16 qr[2][kR0Heads][kR0Rope];   // q^R_h
  float2 wb[2][kR0Heads];               // (sum_f q gamma, q . beta)
  float s1[kR0Rows][kR0S1Stride];       // (q gamma) . z_k per row and head
  float2 half_sums[kR0Rows];            // the value half's (sum z, sum z^2) per row
  uint8_t vstage[4][32 * kR0RowBytes];  // per value-half warp: its 32 rows, 16-byte chunks swizzled by row
  int tile_b[2], tile_lp[2], tile_page[2], tile_n[2];
  uint64_t afull;
  uint64_t bfull[kR0BStages], bempty[kR0BStages];
  uint64_t dfull[2], dfree[2];
  uint64_t drain;
  uint32_t tmem_base;
  int abort;
};

struct R0ProjParams {
  const __nv_bfloat16* q;        // [B, 16, d_n + d_r]
  const __nv_bfloat16* kr_pool;  // [pool rows, d_r]
  const int32_t* id_pool;
  const int32_t* block_table;
  const int32_t* seq_lens;
  const __nv_bfloat16* gate;     // [vocab, 4096]
  const float* gamma;            // [4096] or null
  const float* beta;
  __nv_bfloat16* zv;             // [16][pool rows][d_v]
  float2* stats;                 // [pool rows]: (mu, r)
  float* logit;                  // [B][max_pages * 64][16]
  int batch, max_pages, pool_rows, num_pages, vocab, nkc;
  float eps, scale_log2;
  uint64_t wait_ns;
  int32_t* status;
};

__device__ __forceinline__ bool warp_all_wait(uint32_t bar, uint32_t parity, volatile int* abort_flag,
                                              uint64_t limit_ns) {
  __syncwarp();
  const bool ok = mbar_wait(bar, parity, abort_flag, limit_ns);
  return __all_sync(0xffffffffu, ok);
}

__device__ __forceinline__ void epi_sync() {
  asm volatile("barrier.cta.sync %0, %1;" ::"r"(kR0EpiBar), "r"(32 * kR0EpiWarps) : "memory");
}

__device__ __forceinline__ void prefetch_l2(const void* p) {
  asm volatile("prefetch.global.L2::evict_last [%0];" ::"l"(reinterpret_cast<uint64_t>(p)));
}

__device__ __forceinline__ float bf(const __nv_bfloat16 x) { return __bfloat162float(x); }

// Pages 2t and 2t + 1 (t = blockIdx.x) of the walk over the sequences' pages
// (sequence by sequence, each in logical order), found by warp 0: a prefix
// sum of the page counts over the lanes, 32 sequences at a time.  A half with
// no page (past the last) has n = 0 and repeats the other half's page.
__device__ void find_tile(const R0ProjParams& p, R0Smem& sm, int lane) {
  const int g0 = 2 * static_cast<int>(blockIdx.x);
  int fb[2] = {-1, -1}, flp[2] = {0, 0}, fl[2] = {0, 0};
  int base = 0;
  const int max_len = p.max_pages * kPage;
  for (int b0 = 0; b0 < p.batch && fb[1] < 0; b0 += 32) {
    const int b = b0 + lane;
    // positions past the block table are not read (the attention kernel reports them)
    const int L = b < p.batch ? min(p.seq_lens[b], max_len) : 0;
    const int np = L > 0 ? (L + kPage - 1) / kPage : 0;
    int inc = np;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int t = __shfl_up_sync(0xffffffffu, inc, o);
      if (lane >= o) inc += t;
    }
    const int excl = base + inc - np;
#pragma unroll
    for (int k = 0; k < 2; ++k) {
      if (fb[k] >= 0) continue;   // uniform
      const int g = g0 + k;
      const unsigned m = __ballot_sync(0xffffffffu, np > 0 && g >= excl && g < excl + np);
      if (m != 0u) {
        const int src = __ffs(m) - 1;
        fb[k] = b0 + src;
        flp[k] = g - __shfl_sync(0xffffffffu, excl, src);
        fl[k] = __shfl_sync(0xffffffffu, L, src);
      }
    }
    base += __shfl_sync(0xffffffffu, inc, 31);
  }
  if (lane == 0) {
#pragma unroll
    for (int k = 0; k < 2; ++k) {
      int page = -1, n = 0;
      if (fb[k] >= 0) {
        page = p.block_table[static_cast<size_t>(fb[k]) * p.max_pages + flp[k]];
        if (page < 0 || page >= p.num_pages) {
          report_status(p.status, kStatusOutOfRange);
          page = -1;
        } else {
          n = min(kPage, fl[k] - flp[k] * kPage);
        }
      }
      sm.tile_b[k] = fb[k];
      sm.tile_lp[k] = flp[k];
      sm.tile_page[k] = page;
      sm.tile_n[k] = n;
    }
    // a half without a page of its own reads the other's (its results are not stored)
    if (sm.tile_page[0] < 0) sm.tile_page[0] = sm.tile_page[1];
    if (sm.tile_page[1] < 0) sm.tile_page[1] = sm.tile_page[0];
    if (sm.tile_b[0] < 0) sm.tile_b[0] = sm.tile_b[1];
    if (sm.tile_b[1] < 0) sm.tile_b[1] = sm.tile_b[0];
  }
}

__global__ void __launch_bounds__(kR0Threads, 1)
    r0_project_kernel(const __grid_constant__ CUtensorMap cmap, const __grid_constant__ CUtensorMap wmap,
                      const R0ProjParams p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  const uint32_t sbase = smem_u32(smem);
  const uint32_t b_off = static_cast<uint32_t>(p.nkc) * kR0AChunkBytes;
  R0Smem& sm = *reinterpret_cast<R0Smem*>(smem + b_off + kR0BStages * kR0BChunkBytes);
  volatile int* abort_flag = &sm.abort;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

  if (tid == 0) {
    mbar_init(smem_u32(&sm.afull), 1);
    for (int s = 0; s < kR0BStages; ++s) {
      mbar_init(smem_u32(&sm.bfull[s]), 1);
      mbar_init(smem_u32(&sm.bempty[s]), 1);
    }
    for (int s = 0; s < 2; ++s) {
      mbar_init(smem_u32(&sm.dfull[s]), 1);
      mbar_init(smem_u32(&sm.dfree[s]), kR0EpiWarps);
    }
    mbar_init(smem_u32(&sm.drain), 1);
    sm.abort = 0;
    fence_mbar_init();
    prefetch_tensormap(&cmap);
    prefetch_tensormap(&wmap);
  }
  if (warp == 0) find_tile(p, sm, lane);
  __syncthreads();
  if (sm.tile_n[0] == 0 && sm.tile_n[1] == 0) return;   // past the last page (uniform)
  if (warp == 1) {
    tmem_alloc(smem_u32(&sm.tmem_base), kR0TmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = sm.tmem_base;
  const int nsteps = kR0Heads * p.nkc;   // (head, K chunk) steps of the B stream

  bool epi_key = false, epi_ok = false;
  float epi_s1 = 0.f, epi_s2 = 0.f;
  if (warp == 0) {
    // ---- TMA: the tile's two pages (all K chunks), then W^UKV_h chunk by chunk
    if (elect_one()) {
      const uint64_t pol_stream = policy_evict_first(), pol_keep = policy_evict_last();
      mbar_arrive_expect_tx(smem_u32(&sm.afull), static_cast<uint32_t>(p.nkc) * kR0AChunkBytes);
      for (int kc = 0; kc < p.nkc; ++kc)
#pragma unroll
        for (int k = 0; k < 2; ++k)
          tma_load_2d(sbase + kc * kR0AChunkBytes + k * kR0APageBytes, &cmap, kc * kR0Chunk, sm.tile_page[k] * kPage,
                      smem_u32(&sm.afull), pol_stream);
      int issued = 0;
      for (int i = 0; i < nsteps; ++i) {
        const int s = i % kR0BStages;
        if (i >= kR0BStages &&
            !mbar_wait(smem_u32(&sm.bempty[s]), ((i / kR0BStages) & 1) ^ 1, abort_flag, p.wait_ns))
          break;
        const int h = i / p.nkc, kc = i % p.nkc;
        mbar_arrive_expect_tx(smem_u32(&sm.bfull[s]), kR0BChunkBytes);
        tma_load_2d(sbase + b_off + s * kR0BChunkBytes, &wmap, kc * kR0Chunk, h * kR0Feat, smem_u32(&sm.bfull[s]),
                    pol_keep);
        issued = i + 1;
      }
      // every copy issued lands before the CTA can leave (own flag: bounded, not cut short)
      volatile int own = 0;
      if (!mbar_wait(smem_u32(&sm.afull), 0, &own, p.wait_ns)) *abort_flag = 1;
      for (int i = issued > kR0BStages ? issued - kR0BStages : 0; i < issued; ++i)
        if (!mbar_wait(smem_u32(&sm.bfull[i % kR0BStages]), (i / kR0BStages) & 1, &own, p.wait_ns))
          *abort_flag = 1;
    }
    __syncwarp();
  } else if (warp == 1) {
    // ---- MMA: head h into accumulator h % 2 once the epilogue has read it out
    constexpr uint32_t idesc = idesc_bf16(kR0Rows, kR0Feat, 0, 0);
    bool ok = warp_all_wait(smem_u32(&sm.afull), 0, abort_flag, p.wait_ns);
    bool issued = false;
    for (int h = 0; ok && h < kR0Heads; ++h) {
      const int db = h & 1;
      if (h >= 2) ok = warp_all_wait(smem_u32(&sm.dfree[db]), ((h - 2) >> 1) & 1, abort_flag, p.wait_ns);
      for (int kc = 0; ok && kc < p.nkc; ++kc) {
        const int i = h * p.nkc + kc, s = i % kR0BStages;
        ok = warp_all_wait(smem_u32(&sm.bfull[s]), (i / kR0BStages) & 1, abort_flag, p.wait_ns);
        if (!ok) break;
        tc_fence_after();
        if (elect_one()) {
          const uint64_t ad = smem_desc(sbase + kc * kR0AChunkBytes, 16, 1024, kSwizzle128B);
          const uint64_t bd = smem_desc(sbase + b_off + s * kR0BChunkBytes, 16, 1024, kSwizzle128B);
#pragma unroll
          for (int kk = 0; kk < kR0Chunk / 16; ++kk)
            mma_bf16_ss(tmem + db * kR0Feat, ad + ((kk * 32) >> 4), bd + ((kk * 32) >> 4), idesc,
                        (kc > 0 || kk > 0) ? 1u : 0u);
          mma_commit(smem_u32(&sm.bempty[s]));
          if (kc == p.nkc - 1) mma_commit(smem_u32(&sm.dfull[db]));
        }
        __syncwarp();
        issued = true;
      }
    }
    // every MMA issued completes before TMEM is released
    if (issued) {
      if (elect_one()) mma_commit(smem_u32(&sm.drain));
      __syncwarp();
      volatile int own = 0;
      if (!mbar_wait(smem_u32(&sm.drain), 0, &own, p.wait_ns)) *abort_flag = 1;
    }
    __syncwarp();
  } else {
    // ---- epilogue: tile row r is TMEM lane r (warp w reads lane quadrant
    // w % 4); rows 0-63 are the first page, 64-127 the second.  Warps 2-5
    // take the key features (columns 0-127) of every head, warps 6-9 the
    // value features (columns 128-255).
    const int quad = warp & 3, half = (warp - 2) / 4;
    const int r = 32 * quad + lane, k = r >> 6, jrow = r & (kPage - 1);
    const int n = sm.tile_n[k], page = sm.tile_page[k];
    const bool valid = jrow < n;
    const size_t prow = static_cast<size_t>(page) * kPage + jrow;
    int id = p.id_pool[prow];
    if (static_cast<unsigned>(id) >= static_cast<unsigned>(p.vocab)) {
      if (valid && half == 0) report_status(p.status, kStatusOutOfRange);   // the gate uses row 0
      id = 0;
    }
    // the query terms of the tile's two sequences: q gamma (key features),
    // q^R, sum q gamma and q . beta per head
    const int et = tid - 64;
    for (int i = et; i < 2 * kR0Heads * kR0Half; i += 32 * kR0EpiWarps) {
      const int s = i / (kR0Heads * kR0Half), h = (i / kR0Half) % kR0Heads, f = i % kR0Half;
      const float qf = bf(p.q[(static_cast<size_t>(sm.tile_b[s]) * kR0Heads + h) * (kR0Half + kR0Rope) + f]);
      sm.qg[s][h][f] = qf * (p.gamma ? p.gamma[h * kR0Feat + f] : 1.f);
    }
    for (int i = et; i < 2 * kR0Heads * kR0Rope; i += 32 * kR0EpiWarps) {
      const int s = i / (kR0Heads * kR0Rope), h = (i / kR0Rope) % kR0Heads, d = i % kR0Rope;
      sm.qr[s][h][d] = p.q[(static_cast<size_t>(sm.tile_b[s]) * kR0Heads + h) * (kR0Half + kR0Rope) + kR0Half + d];
    }
    for (int pr = 0; pr < 4; ++pr) {
      const int pidx = 4 * (warp - 2) + pr, s = pidx / kR0Heads, h = pidx % kR0Heads;
      const __nv_bfloat16* qh = p.q + (static_cast<size_t>(sm.tile_b[s]) * kR0Heads + h) * (kR0Half + kR0Rope);
      float w = 0.f, bq = 0.f;
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const int f = 4 * lane + i;
        const float qf = bf(qh[f]);
        w += qf * (p.gamma ? p.gamma[h * kR0Feat + f] : 1.f);
        bq = fmaf(qf, p.beta ? p.beta[h * kR0Feat + f] : 0.f, bq);
      }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        w += __shfl_xor_sync(0xffffffffu, w, o);
        bq += __shfl_xor_sync(0xffffffffu, bq, o);
      }
      if (lane == 0) sm.wb[s][h] = make_float2(w, bq);
    }
    epi_sync();

    const __nv_bfloat16* grow = p.gate + static_cast<size_t>(id) * kR0Width + half * kR0Half;
    const uint64_t pol_gate = policy_evict_last();
    uint8_t* vst = sm.vstage[quad];
    const bool store_v = half == 1 && n > 0;   // uniform in the warp
    float s1 = 0.f, s2 = 0.f;
    bool ok = true;
    // this half of the row's gate values of a head (128 bf16): each quarter
    // of them is requested for head h + 1 as soon as head h has used it, so
    // that the loads run while the rest of head h is processed
    uint4 g[kR0Half / 8];
    auto load_g = [&](int hh, int i) { ldg_32_na_hint(grow + hh * kR0Feat + 16 * i, pol_gate, g[2 * i], g[2 * i + 1]); };
#pragma unroll
    for (int i = 0; i < kR0Half / 16; ++i) load_g(0, i);
    for (int h = 0; h < kR0Heads; ++h) {
      const int db = h & 1;
      if (h + 2 < kR0Heads) {   // two heads ahead into L2
        prefetch_l2(grow + (h + 2) * kR0Feat);
        prefetch_l2(grow + (h + 2) * kR0Feat + 64);
      }
      ok = ok && warp_all_wait(smem_u32(&sm.dfull[db]), (h >> 1) & 1, abort_flag, p.wait_ns);
      if (!ok) break;
      tc_fence_after();
      const float* qgh = &sm.qg[k][h][0];
      float dot = 0.f;
#pragma unroll
      for (int c0 = 0; c0 < kR0Half; c0 += 16) {
        float v[16];
        tmem_ld16(tmem + (static_cast<uint32_t>(32 * quad) << 16) + db * kR0Feat + half * kR0Half + c0, v);
        tmem_wait_ld();
        const __nv_bfloat162* ge0 = reinterpret_cast<const __nv_bfloat162*>(&g[c0 / 8]);
        const __nv_bfloat162* ge1 = reinterpret_cast<const __nv_bfloat162*>(&g[c0 / 8 + 1]);
        uint32_t packed[8];
        float zf[16];
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          const float2 gf = __bfloat1622float2(i < 4 ? ge0[i] : ge1[i - 4]);
          const __nv_bfloat162 zb = __floats2bfloat162_rn(v[2 * i] * gf.x, v[2 * i + 1] * gf.y);
          const float2 zr = __bfloat1622float2(zb);   // statistics and dots of the rounded values
          s1 += zr.x + zr.y;
          s2 = fmaf(zr.x, zr.x, fmaf(zr.y, zr.y, s2));
          zf[2 * i] = zr.x;
          zf[2 * i + 1] = zr.y;
          packed[i] = *reinterpret_cast<const uint32_t*>(&zb);
        }
        if (half == 0) {
#pragma unroll
          for (int i = 0; i < 4; ++i) {
            const float4 qv = *reinterpret_cast<const float4*>(qgh + c0 + 4 * i);
            dot = fmaf(qv.x, zf[4 * i], dot);
            dot = fmaf(qv.y, zf[4 * i + 1], dot);
            dot = fmaf(qv.z, zf[4 * i + 2], dot);
            dot = fmaf(qv.w, zf[4 * i + 3], dot);
          }
        } else {
          // chunks c0/8 and c0/8 + 1 of this row, at (chunk ^ (row % 16)) in its 256-byte row
          const int ch = c0 / 8;
          *reinterpret_cast<uint4*>(vst + lane * kR0RowBytes + ((ch ^ (lane & 15)) << 4)) =
              make_uint4(packed[0], packed[1], packed[2], packed[3]);
          *reinterpret_cast<uint4*>(vst + lane * kR0RowBytes + (((ch + 1) ^ (lane & 15)) << 4)) =
              make_uint4(packed[4], packed[5], packed[6], packed[7]);
        }
        if (c0 % 32 == 16 && h + 1 < kR0Heads) {   // columns c0 - 16 .. c0 + 15 done
          load_g(h + 1, c0 / 16 - 1);
          load_g(h + 1, c0 / 16);
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_u32(&sm.dfree[db]));
      if (half == 0) {
        sm.s1[r][h] = dot;
      } else if (store_v) {
        // the warp's 32 rows of head h are 8 KB in one piece (head-major):
        // two whole rows per store instruction
        uint8_t* dst = reinterpret_cast<uint8_t*>(
            p.zv + (static_cast<size_t>(h) * p.pool_rows + static_cast<size_t>(page) * kPage + 32 * (quad & 1)) *
                       kR0Half);
#pragma unroll
        for (int i = 0; i < 16; ++i) {
          const int rr = 2 * i + (lane >> 4), c = lane & 15;
          *reinterpret_cast<uint4*>(dst + rr * kR0RowBytes + c * 16) =
              *reinterpret_cast<const uint4*>(vst + rr * kR0RowBytes + ((c ^ (rr & 15)) << 4));
        }
        __syncwarp();   // the tile is read before the next head rewrites it
      }
    }
    if (half == 1) sm.half_sums[r] = make_float2(s1, s2);
    epi_key = half == 0 && n > 0;
    epi_ok = ok;
    epi_s1 = s1;
    epi_s2 = s2;
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (epi_key && epi_ok && !sm.abort) {
    // the row's statistics over all 4096 features, then every head's logit
    const int r = 32 * (warp & 3) + lane, k = r >> 6, jrow = r & (kPage - 1);
    const size_t prow = static_cast<size_t>(sm.tile_page[k]) * kPage + jrow;
    const float2 o = sm.half_sums[r];
    const float mu = (epi_s1 + o.x) / kR0Width;
    const float var = fmaxf((epi_s2 + o.y) / kR0Width - mu * mu, 0.f);
    const float rinv = rsqrtf(var + p.eps);
    p.stats[prow] = make_float2(mu, rinv);
    if (jrow < sm.tile_n[k]) {
      float kr[kR0Rope];
      const uint4* kr4 = reinterpret_cast<const uint4*>(p.kr_pool + prow * kR0Rope);
#pragma unroll
      for (int i = 0; i < kR0Rope / 8; ++i) {
        const uint4 u = kr4[i];
        const __nv_bfloat162* e = reinterpret_cast<const __nv_bfloat162*>(&u);
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const float2 f = __bfloat1622float2(e[j]);
          kr[8 * i + 2 * j] = f.x;
          kr[8 * i + 2 * j + 1] = f.y;
        }
      }
      float lg[kR0Heads];
#pragma unroll
      for (int h = 0; h < kR0Heads; ++h) {
        const __nv_bfloat162* qr2 = reinterpret_cast<const __nv_bfloat162*>(&sm.qr[k][h][0]);
        float sr = 0.f;
#pragma unroll
        for (int d = 0; d < kR0Rope / 2; ++d) {
          const float2 qf = __bfloat1622float2(qr2[d]);
          sr = fmaf(qf.x, kr[2 * d], fmaf(qf.y, kr[2 * d + 1], sr));
        }
        const float2 wb = sm.wb[k][h];
        lg[h] = p.scale_log2 * (rinv * (sm.s1[r][h] - mu * wb.x) + wb.y + sr);
      }
      const size_t pos = static_cast<size_t>(sm.tile_b[k]) * p.max_pages * kPage +
                         static_cast<size_t>(sm.tile_lp[k]) * kPage + jrow;
      float4* dst = reinterpret_cast<float4*>(p.logit + pos * kR0Heads);
#pragma unroll
      for (int i = 0; i < kR0Heads / 4; ++i) dst[i] = make_float4(lg[4 * i], lg[4 * i + 1], lg[4 * i + 2], lg[4 * i + 3]);
    }
  }
  if (warp == 1) tmem_dealloc(tmem, kR0TmemCols);
  if (tid == 0 && sm.abort) report_status(p.status, kStatusTimeout);
}

struct R0AttnParams {
  const int32_t* block_table;
  const int32_t* seq_lens;
  const __nv_bfloat16* zv;      // [16][pool rows][d_v]
  const float2* stats;          // [pool rows]
  const float* logit;           // [B][max_pages * 64][16]
  const float* gamma;           // [4096] or null
  const float* beta;
  __nv_bfloat16* out;           // [B, H, d_v]
  int max_pages, num_pages, pool_rows;
  int32_t* status;
};

constexpr int kR0AttnWarps = 16;
constexpr int kR0AttnThreads = 32 * kR0AttnWarps;
constexpr int kR0AttnPairs = 12;   // row pairs a warp has in flight at once (24 rows, 6 KB)

// One block per (sequence, head).  Warp w takes the sequence's pages w, w +
// 16, ...: a page's 64 rows of the head's gated values are 16 KB in one piece
// (head-major), read as two rows per load instruction (lane l: row 2i + l/16,
// features 8 (l % 16) .. + 7), 24 rows in flight.  Each half-warp keeps its
// own online softmax over its rows (m, l = sum p, the sums of P' z and P' mu
// with P' = p r); the 32 half-warps are merged at the end.
__global__ void __launch_bounds__(kR0AttnThreads) r0_attend_kernel(const R0AttnParams p) {
  __shared__ float part[2 * kR0AttnWarps][3 + kR0Half];
  const int b = blockIdx.x / kR0Heads, h = blockIdx.x % kR0Heads;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int hw = lane >> 4, c8 = 8 * (lane & 15);   // half-warp, first feature of the lane
  const int max_len = p.max_pages * kPage;
  const int L = min(p.seq_lens[b], max_len);
  if (threadIdx.x == 0 && h == 0 && p.seq_lens[b] > max_len) report_status(p.status, kStatusOutOfRange);
  const float* lgb = p.logit + static_cast<size_t>(b) * max_len * kR0Heads + h;
  const __nv_bfloat16* zh = p.zv + static_cast<size_t>(h) * p.pool_rows * kR0Half + c8;
  const int npages = L > 0 ? (L + kPage - 1) / kPage : 0;
  float m = -INFINITY, l = 0.f, bm = 0.f, acc[8];
#pragma unroll
  for (int i = 0; i < 8; ++i) acc[i] = 0.f;
  bool bad = false;
  int lp = warp;
  int page = lp < npages ? p.block_table[static_cast<size_t>(b) * p.max_pages + lp] : -1;
  while (lp < npages) {
    // the next page of this warp, requested before this one's rows
    const int lp_next = lp + kR0AttnWarps;
    const int page_next = lp_next < npages ? p.block_table[static_cast<size_t>(b) * p.max_pages + lp_next] : -1;
    if (page < 0 || page >= p.num_pages) {
      bad = true;
    } else {
      const int nrow = min(kPage, L - lp * kPage);
      const size_t row0 = static_cast<size_t>(page) * kPage;
#pragma unroll 1
      for (int r0 = 0; r0 < nrow; r0 += 2 * kR0AttnPairs) {
        uint4 zv[kR0AttnPairs];
        float s[kR0AttnPairs];
        float2 st[kR0AttnPairs];
#pragma unroll
        for (int i = 0; i < kR0AttnPairs; ++i) {
          const int r = r0 + 2 * i + hw;
          if (r < nrow) {
            zv[i] = *reinterpret_cast<const uint4*>(zh + (row0 + r) * kR0Half);
            s[i] = lgb[static_cast<size_t>(lp * kPage + r) * kR0Heads];
            st[i] = p.stats[row0 + r];
          }
        }
#pragma unroll
        for (int i = 0; i < kR0AttnPairs; ++i) {
          if (r0 + 2 * i + hw >= nrow) continue;   // uniform in the half-warp
          const float mn = fmaxf(m, s[i]);
          const float alpha = exp2f(m - mn), pj = exp2f(s[i] - mn);
          const float w = pj * st[i].y;
          l = fmaf(l, alpha, pj);
          bm = fmaf(bm, alpha, w * st[i].x);
          const __nv_bfloat162* z2 = reinterpret_cast<const __nv_bfloat162*>(&zv[i]);
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            const float2 zf = __bfloat1622float2(z2[j]);
            acc[2 * j] = fmaf(acc[2 * j], alpha, w * zf.x);
            acc[2 * j + 1] = fmaf(acc[2 * j + 1], alpha, w * zf.y);
          }
          m = mn;
        }
      }
    }
    lp = lp_next;
    page = page_next;
  }
  if (bad) report_status(p.status, kStatusOutOfRange);
  const int slot = 2 * warp + hw;
  if ((lane & 15) == 0) {
    part[slot][0] = m;
    part[slot][1] = l;
    part[slot][2] = bm;
  }
#pragma unroll
  for (int i = 0; i < 8; ++i) part[slot][3 + c8 + i] = acc[i];
  __syncthreads();
  if (warp == 0) {
    // lane l: value features 4l .. 4l + 3
    const int fv = h * kR0Feat + kR0Half + 4 * lane;
    float M = -INFINITY;
    for (int w = 0; w < 2 * kR0AttnWarps; ++w) M = fmaxf(M, part[w][0]);
    float Ls = 0.f, Bs = 0.f, a[4] = {0.f, 0.f, 0.f, 0.f};
    for (int w = 0; w < 2 * kR0AttnWarps; ++w) {
      const float sc = part[w][0] == -INFINITY ? 0.f : exp2f(part[w][0] - M);
      Ls = fmaf(part[w][1], sc, Ls);
      Bs = fmaf(part[w][2], sc, Bs);
#pragma unroll
      for (int i = 0; i < 4; ++i) a[i] = fmaf(part[w][3 + 4 * lane + i], sc, a[i]);
    }
    __nv_bfloat16* ob = p.out + (static_cast<size_t>(b) * kR0Heads + h) * kR0Half + 4 * lane;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const float gv = p.gamma ? p.gamma[fv + i] : 1.f, bv = p.beta ? p.beta[fv + i] : 0.f;
      ob[i] = __float2bfloat16_rn(L > 0 && Ls > 0.f ? fmaf(gv, (a[i] - Bs) / Ls, bv) : 0.f);
    }
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

size_t r0_workspace_bytes(int batch, int max_pages, int num_pages) {
  const size_t rows = static_cast<size_t>(num_pages) * kPage;
  const size_t positions = static_cast<size_t>(batch) * max_pages * kPage;
  return align_up(rows * kR0Heads * kR0Half * 2, 256) + align_up(rows * sizeof(float2), 256) +
         align_up(positions * kR0Heads * sizeof(float), 256);
}

cudaError_t launch_decode_r0(const R0Args& a, cudaStream_t st) {
  const size_t rows = static_cast<size_t>(a.num_pages) * kPage;
  uint8_t* ws = static_cast<uint8_t*>(a.workspace);
  __nv_bfloat16* zv = reinterpret_cast<__nv_bfloat16*>(ws);
  size_t off = align_up(rows * kR0Heads * kR0Half * 2, 256);
  float2* stats = reinterpret_cast<float2*>(ws + off);
  off += align_up(rows * sizeof(float2), 256);
  float* logit = reinterpret_cast<float*>(ws + off);
  CUtensorMap cmap, wmap;
  if (!r0_encode(&cmap, a.c_pool, rows, static_cast<uint64_t>(a.d_c), kPage)) return cudaErrorInvalidValue;
  if (!r0_encode(&wmap, a.w_ukv, kR0Width, static_cast<uint64_t>(a.d_c), kR0Feat)) return cudaErrorInvalidValue;
  const int nkc = a.d_c / kR0Chunk;
  const int smem = static_cast<int>(nkc * kR0AChunkBytes + kR0BStages * kR0BChunkBytes + sizeof(R0Smem) + 1024);
  cudaError_t e = cudaFuncSetAttribute(r0_project_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  R0ProjParams pp;
  pp.q = static_cast<const __nv_bfloat16*>(a.q);
  pp.kr_pool = static_cast<const __nv_bfloat16*>(a.kr_pool);
  pp.id_pool = a.id_pool;
  pp.block_table = a.block_table;
  pp.seq_lens = a.seq_lens;
  pp.gate = static_cast<const __nv_bfloat16*>(a.gate_r0);
  pp.gamma = a.ln_gamma;
  pp.beta = a.ln_beta;
  pp.zv = zv;
  pp.stats = stats;
  pp.logit = logit;
  pp.batch = a.batch;
  pp.max_pages = a.max_pages;
  pp.pool_rows = static_cast<int>(rows);
  pp.num_pages = a.num_pages;
  pp.vocab = a.vocab;
  pp.nkc = nkc;
  pp.eps = a.eps;
  pp.scale_log2 = a.scale_log2;
  pp.wait_ns = kWaitLimitNs;
  pp.status = a.status;
  // one CTA per two pages of the walk: the block table bounds the pages in use
  const int tiles = static_cast<int>((static_cast<int64_t>(a.batch) * a.max_pages + 1) / 2);
  r0_project_kernel<<<tiles, kR0Threads, smem, st>>>(cmap, wmap, pp);
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  R0AttnParams ap;
  ap.block_table = a.block_table;
  ap.seq_lens = a.seq_lens;
  ap.zv = zv;
  ap.stats = stats;
  ap.logit = logit;
  ap.gamma = a.ln_gamma;
  ap.beta = a.ln_beta;
  ap.out = static_cast<__nv_bfloat16*>(a.out);
  ap.max_pages = a.max_pages;
  ap.num_pages = a.num_pages;
  ap.pool_rows = static_cast<int>(rows);
  ap.status = a.status;
  r0_attend_kernel<<<a.batch * kR0Heads, kR0AttnThreads, 0, st>>>(ap);
  return cudaGetLastError();
}

}  // namespace egmla
