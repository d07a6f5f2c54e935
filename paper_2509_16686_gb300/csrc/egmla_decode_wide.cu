// egmla_decode_wide.cu - split-KV decode for the widest latent (d_c = 512, plain
// MLA without the gate), where the transposed layout of egmla_decode_tc.cu does
// not fit in tensor memory (two score buffers of 128 columns plus a 512-column
// output accumulator).  Here the latent output is accumulated transposed, latent
// features in TMEM lanes (M = 128) and heads in columns (N = 16), which needs
// only 16 columns per 128 features.
//
// One CTA per split-KV work unit (see egmla_common.cuh for the schedule).  The
// CTA streams its cache pages, one 64-token page per tile, through a ring of
// shared-memory slots:
//
//   TMA (warp 0)      latent page [64 tok x d_c] and RoPE-key page [64 x 64] as
//                     128-byte-swizzled boxes.
//   MMA (warp 1)      S_lat = Z Q^T and S_rope = K^R Q^R^T on tcgen05 with fp32
//                     accumulators in TMEM (M = 64 tokens, N = 16 heads, S
//                     double-buffered so the next tile's scores overlap the
//                     current softmax); O_tile = Z^T P' (M = 128 latent
//                     features, N = 16 heads, K = 64 tokens).
//   zero fill (warps 4-7)  rows past the end of a partial page are cleared so
//                     that the weighted sum never touches unused cache slots.
//   softmax (warps 8-11)
//                     s = scale * (S_lat + S_rope); online softmax with a
//                     lazily moved reference max per head (cross-warp max
//                     through shared memory); P' (bf16) is written as the B
//                     operand of the PV MMA.
//
// At the end of each sequence segment the un-normalised latent output O, the
// running max m and the denominator l are written as this split's partial
// result.  Everything the kernel waits on has a time limit: on expiry it
// records EG_MLA_ERR_TIMEOUT, drains its own copies and MMAs, frees TMEM and
// exits.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <cmath>
#include <cstdint>

#include "egmla_common.cuh"
#include "egmla_kernels.h"
#include "egmla_ptx.cuh"

namespace egmla {

namespace {

constexpr int kHeads = 16;
constexpr int kRope = 64;
constexpr int kThreads = 384;  // warp 0 TMA, warp 1 MMA + TMEM owner, 2-3 spare, 4-7 zero fill, 8-11 softmax
constexpr int kGateWarp0 = 4;
constexpr int kSoftWarp0 = 8;
constexpr uint32_t kSmemLimit = 232448;
// registers per thread: 384 threads x 168 at launch; warps 0-3 give theirs up
// to the gate and softmax warpgroups (128 x 56 + 256 x 224 = 384 x 168)
constexpr int kProducerRegs = 56;
constexpr int kConsumerRegs = 224;
// a head's reference max moves only when a tile exceeds it by 2^8
constexpr float kLazyLog2 = 8.f;

template <int D_C>
struct Cfg {
  static constexpr int NCH = D_C / 64;                  // 64-feature swizzle-atom columns
  static constexpr int NMC = (D_C + 127) / 128;         // 128-feature M chunks of the PV MMA
  static constexpr uint32_t PCHUNK = kPage * 128;       // one atom column of a page: 8 KB
  static constexpr uint32_t KR_OFF = NCH * PCHUNK;
  static constexpr uint32_t SLOT = KR_OFF + PCHUNK;     // latent + RoPE key of one page
  static constexpr uint32_t QB_LAT = qprep_lat_bytes(D_C);
  static constexpr uint32_t QPREP = qprep_bytes_tc(D_C, kRope);
  static constexpr uint32_t QBUF = (QPREP + 127) / 128 * 128;
  static constexpr uint32_t PBUF = kPage * kHeads * 2;
  static constexpr uint32_t MISC = 2048;
  static constexpr int NS_FIT = (int)((kSmemLimit - 1024 - 2 * QBUF - PBUF - MISC) / SLOT);
  static constexpr int NS = NS_FIT > 6 ? 6 : NS_FIT;
  static constexpr uint32_t OFF_QBUF = NS * SLOT;
  static constexpr uint32_t OFF_PBUF = OFF_QBUF + 2 * QBUF;
  static constexpr uint32_t OFF_MISC = OFF_PBUF + PBUF;
  static constexpr uint32_t SMEM = OFF_MISC + MISC + 1024;
  // TMEM columns: two score buffers of (latent 16 + RoPE 16) columns, then the
  // latent-output accumulator (16 columns per 128-feature chunk), which stays
  // in TMEM across the tiles of a sequence segment
  static constexpr uint32_t S_COLS = 32;
  static constexpr uint32_t COL_S = 0, COL_O = 2 * S_COLS;
  static constexpr uint32_t TMEM_COLS = 128;
  static constexpr uint32_t PAGE_TX = NCH * PCHUNK + PCHUNK;
  static_assert(NS >= 2, "the ring needs two page slots");
  static_assert(SMEM <= kSmemLimit, "shared memory");
  static_assert(D_C % 64 == 0 && D_C >= 128, "d_c");
  // first latent feature of PV M-chunk j; the last chunk is shifted back so that
  // it ends at D_C (for D_C = 192 it overlaps the previous one by 64 features)
  __host__ __device__ static constexpr int mc_start(int j) {
    return (128 * j + 128 <= D_C) ? 128 * j : D_C - 128;
  }
};

struct TcParams {
  const int32_t* block_table;
  const int32_t* seq_lens;
  const uint8_t* qprep;
  const int32_t* cu;
  float* part_ml;
  float* part_o;
  int32_t* status;
  int batch, max_pages, num_pages;
  float scale_log2;
};

// shared-memory barrier block (inside MISC, after 1 KB of reduction scratch)
struct Bars {
  uint64_t full[6], empty[6], zready[6];
  uint64_t qfull[2], qempty[2];
  uint64_t s_ready[2];
  uint64_t sp_done, o_ready;
  uint64_t red[2], sum;
  uint32_t tmem_base;
  int abort;
};

struct Tile {
  int b, lp, ntok, tok0;
  bool first, last;
};

// Walks this CTA's pages one at a time, segment by segment (identically in
// every role, so no per-tile metadata needs to be exchanged).
struct Walker {
  const int32_t* cu;
  const int32_t* lens;
  int batch, g1, b, lp, lp_end, L;
  bool first, done;

  __device__ void start(const int32_t* cu_, const int32_t* lens_, int batch_) {
    cu = cu_;
    lens = lens_;
    batch = batch_;
    const int total = __ldg(cu + batch);
    const int chunk = split_chunk(total, gridDim.x);
    const int g0 = blockIdx.x * chunk;
    g1 = min(g0 + chunk, total);
    done = g0 >= g1;
    if (done) return;
    b = find_sequence(cu, batch, g0);
    enter(g0);
  }
  __device__ void enter(int g) {
    const int base = __ldg(cu + b) + kSegCost;   // unit of the sequence's first page
    lp = max(g - base, 0);
    lp_end = min(g1, __ldg(cu + b + 1)) - base;
    L = __ldg(lens + b);
    first = true;
    if (lp_end <= lp) done = true;   // the range ends inside the sequence's start cost
  }
  __device__ bool next(Tile& t) {
    if (done) return false;
    t.b = b;
    t.lp = lp;
    t.tok0 = lp * kPage;
    t.ntok = min(kPage, L - t.tok0);
    t.first = first;
    first = false;
    lp += 1;
    t.last = lp >= lp_end;
    if (t.last) {
      const int g = __ldg(cu + b) + kSegCost + lp_end;
      if (g >= g1) {
        done = true;
      } else {
        ++b;
        while (b < batch - 1 && __ldg(cu + b + 1) <= g) ++b;
        enter(g);
      }
    }
    return true;
  }
};

// mbarrier wait taken by a whole warp: every lane polls, then the warp agrees,
// so that a timeout never splits the warp before a .sync.aligned instruction
__device__ __forceinline__ bool warp_wait(uint32_t bar, uint32_t parity, volatile int* abort_flag) {
  const bool ok = mbar_wait(bar, parity, abort_flag);
  return __all_sync(0xffffffffu, ok);
}

__device__ __forceinline__ float2 unpack_bf16x2(uint32_t w) {
  return make_float2(__uint_as_float(w << 16), __uint_as_float(w & 0xffff0000u));
}

// 2^x with the hardware approximation (max 2 ulp; the weights are rounded to
// bf16 right after, and -inf gives 0)
__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  __nv_bfloat162 z = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&z);
}

// Reduce 16 per-lane values over the 32 lanes of a warp; lane l ends with the
// result for index (l >> 1) & 15.  Each step hands half of the remaining
// values to the partner lane, so 16 shuffles replace 80.
template <bool MAX>
__device__ __forceinline__ float warp_reduce16(const float (&v)[16], int lane) {
  auto op = [](float a, float b) { return MAX ? fmaxf(a, b) : a + b; };
  float r8[8], r4[4], r2[2];
  const bool u16 = lane & 16, u8 = lane & 8, u4 = lane & 4, u2 = lane & 2;
#pragma unroll
  for (int k = 0; k < 8; ++k) {
    const float send = u16 ? v[k] : v[k + 8];
    const float keep = u16 ? v[k + 8] : v[k];
    r8[k] = op(keep, __shfl_xor_sync(0xffffffffu, send, 16));
  }
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    const float send = u8 ? r8[k] : r8[k + 4];
    const float keep = u8 ? r8[k + 4] : r8[k];
    r4[k] = op(keep, __shfl_xor_sync(0xffffffffu, send, 8));
  }
#pragma unroll
  for (int k = 0; k < 2; ++k) {
    const float send = u4 ? r4[k] : r4[k + 2];
    const float keep = u4 ? r4[k + 2] : r4[k];
    r2[k] = op(keep, __shfl_xor_sync(0xffffffffu, send, 4));
  }
  const float send = u2 ? r2[0] : r2[1];
  const float keep = u2 ? r2[1] : r2[0];
  const float r1 = op(keep, __shfl_xor_sync(0xffffffffu, send, 2));
  return op(r1, __shfl_xor_sync(0xffffffffu, r1, 1));
}

template <int D_C>
__global__ void __launch_bounds__(kThreads, 1)
    decode_tc_kernel(const __grid_constant__ CUtensorMap cmap, const __grid_constant__ CUtensorMap krmap,
                     const TcParams p) {
  using C = Cfg<D_C>;
  extern __shared__ uint8_t smem_raw[];
  // 1024-byte aligned base (128-byte swizzle atoms); derived by an offset from the
  // __shared__ array so that every access through it stays a shared-memory access
  uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  const uint32_t sbase = smem_u32(smem);
  float* red_max = reinterpret_cast<float*>(smem + C::OFF_MISC);         // [2][4][16]
  float* red_sum = red_max + 2 * 4 * 16;                                 // [4][32]
  Bars& bars = *reinterpret_cast<Bars*>(smem + C::OFF_MISC + 1024);
  volatile int* abort_flag = &bars.abort;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int s = 0; s < C::NS; ++s) {
      mbar_init(smem_u32(&bars.full[s]), 1);
      mbar_init(smem_u32(&bars.empty[s]), 1);
      mbar_init(smem_u32(&bars.zready[s]), 128);
    }
    for (int s = 0; s < 2; ++s) {
      mbar_init(smem_u32(&bars.qfull[s]), 1);
      mbar_init(smem_u32(&bars.qempty[s]), 1 + 128);
      mbar_init(smem_u32(&bars.s_ready[s]), 1);
      mbar_init(smem_u32(&bars.red[s]), 128);
    }
    mbar_init(smem_u32(&bars.sp_done), 128);
    mbar_init(smem_u32(&bars.o_ready), 1);
    mbar_init(smem_u32(&bars.sum), 128);
    bars.abort = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(&bars.tmem_base), C::TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = bars.tmem_base;
  // Everything above touches only this CTA's shared and tensor memory; what
  // follows reads the query-absorption kernel's outputs and the cache it may
  // have appended to (launched with programmatic stream serialisation).
  grid_dependency_wait();

  if (warp < kGateWarp0) regs_decrease<kProducerRegs>();
  if (warp == 0) {
    // ---------------------------------------------------------------- TMA producer
    // The whole warp walks the tiles; lane 0 waits and issues.  Block-table
    // entries are fetched 32 at a time (one per lane) so no page lookup sits on
    // the issue path.
    if (lane == 0) {
      prefetch_tensormap(&cmap);
      prefetch_tensormap(&krmap);
    }
    const uint64_t pol_stream = policy_evict_first();
    Walker w;
    w.start(p.cu, p.seq_lens, p.batch);
    Tile t;
    int it = 0, seg = -1;
    int last_it[6] = {-1, -1, -1, -1, -1, -1};
    int last_qseg[2] = {-1, -1};
    int bt_b = -1, bt_base = 0, bt_reg = -1;
    bool ok_loop = true;
    while (ok_loop && w.next(t)) {
      if (t.b != bt_b || t.lp >= bt_base + 32) {
        bt_b = t.b;
        bt_base = t.lp;
        const int lp = t.lp + lane;
        bt_reg = lp < p.max_pages ? __ldg(p.block_table + static_cast<size_t>(t.b) * p.max_pages + lp) : -1;
      }
      const int pg = __shfl_sync(0xffffffffu, bt_reg, t.lp - bt_base);
      if (t.first) ++seg;
      const int slot = it % C::NS;
      if (lane == 0) {
        if (t.first) {
          const int qb = seg & 1;
          if (mbar_wait(smem_u32(&bars.qempty[qb]), ((seg >> 1) & 1) ^ 1, abort_flag)) {
            mbar_arrive_expect_tx(smem_u32(&bars.qfull[qb]), C::QPREP);
            bulk_load(sbase + C::OFF_QBUF + qb * C::QBUF, p.qprep + static_cast<size_t>(t.b) * C::QPREP, C::QPREP,
                      smem_u32(&bars.qfull[qb]));
            last_qseg[qb] = seg;
          } else {
            ok_loop = false;
          }
        }
        if (ok_loop && !mbar_wait(smem_u32(&bars.empty[slot]), ((it / C::NS) & 1) ^ 1, abort_flag)) ok_loop = false;
        if (ok_loop) {
          const bool ok = pg >= 0 && pg < p.num_pages;
          if (!ok) report_status(p.status, kStatusOutOfRange);
          const uint32_t fb = smem_u32(&bars.full[slot]);
          mbar_arrive_expect_tx(fb, ok ? C::PAGE_TX : 0u);
          if (ok) {
            const uint32_t dst = sbase + slot * C::SLOT;
            const int y = pg * kPage;
#pragma unroll
            for (int fc = 0; fc < C::NCH; ++fc) tma_load_2d(dst + fc * C::PCHUNK, &cmap, fc * 64, y, fb, pol_stream);
            tma_load_2d(dst + C::KR_OFF, &krmap, 0, y, fb, pol_stream);
          }
          last_it[slot] = it;
        }
      }
      ok_loop = __shfl_sync(0xffffffffu, ok_loop, 0);
      ++it;
    }
    if (lane == 0) {
      // drain: every copy this thread issued must land before the CTA exits
      for (int s = 0; s < C::NS; ++s)
        if (last_it[s] >= 0) mbar_wait(smem_u32(&bars.full[s]), (last_it[s] / C::NS) & 1, abort_flag);
      for (int s = 0; s < 2; ++s)
        if (last_qseg[s] >= 0) mbar_wait(smem_u32(&bars.qfull[s]), (last_qseg[s] >> 1) & 1, abort_flag);
    }
    __syncwarp();
  } else if (warp == 1) {
    // ---------------------------------------------------------------- MMA issuer
    // Converged warp; one elected lane issues.  Order: scores(i + 1) before
    // PV(i), so the next tile's scores are ready when the softmax warps finish
    // tile i.  All loops are unrolled with compile-time accumulate flags.
    {
      constexpr uint32_t IDESC_QK = idesc_bf16(64, 16, 0, 0);
      constexpr uint32_t IDESC_PV = idesc_bf16(128, 16, 1, 1);
      Walker w;
      w.start(p.cu, p.seq_lens, p.batch);
      uint32_t last_bar = 0, last_par = 0;
      int seg = -1;
      // the query block as an N = 16 B operand: K cores 256 B apart, head halves 128 B apart
      const uint64_t qdesc0 = smem_desc(sbase + C::OFF_QBUF, kQGroupBytes, kQRowGroupBytes, kSwizzleNone);
      const uint64_t zdesc_k = smem_desc(sbase, 16, 1024, kSwizzle128B);         // K-major view of a slot
      const uint64_t zdesc_mn = smem_desc(sbase, C::PCHUNK, 1024, kSwizzle128B);  // MN-major view of a slot
      const uint64_t pdesc = smem_desc(sbase + C::OFF_PBUF, 256, 128, kSwizzleNone);
      Tile cur, nxt;
      bool have = w.next(cur);
      bool ok = true;
      int it = 0;
      // scores of tile j (t): S_lat = Z (q^ gamma)^T, S_rope = K^R (q^R)^T
      auto scores = [&](const Tile& t, int j) -> bool {
        if (t.first) {
          ++seg;
          if (!warp_wait(smem_u32(&bars.qfull[seg & 1]), (seg >> 1) & 1, abort_flag)) return false;
        }
        const int slot = j % C::NS;
        if (!warp_wait(smem_u32(&bars.zready[slot]), (j / C::NS) & 1, abort_flag)) return false;
        tc_fence_after();
        if (elect_one()) {
          const uint64_t za = zdesc_k + ((slot * C::SLOT) >> 4);
          const uint64_t qb = qdesc0 + (((seg & 1) * C::QBUF) >> 4);
          const uint32_t ds = tmem + C::COL_S + (j & 1) * C::S_COLS;
#pragma unroll
          for (int kk = 0; kk < D_C / 16; ++kk)
            mma_bf16_ss(ds, za + (((kk >> 2) * C::PCHUNK + (kk & 3) * 32) >> 4), qb + ((kk * 2 * kQGroupBytes) >> 4), IDESC_QK,
                        kk > 0);
#pragma unroll
          for (int kk = 0; kk < kRope / 16; ++kk)
            mma_bf16_ss(ds + 16, za + ((C::KR_OFF + kk * 32) >> 4), qb + ((C::QB_LAT + kk * 2 * kQGroupBytes) >> 4), IDESC_QK,
                        kk > 0);
          mma_commit(smem_u32(&bars.s_ready[j & 1]));
          if (t.last) mma_commit(smem_u32(&bars.qempty[seg & 1]));
        }
        __syncwarp();
        last_bar = smem_u32(&bars.s_ready[j & 1]);
        last_par = (j >> 1) & 1;
        return true;
      };
      if (have) ok = scores(cur, 0);
      while (have && ok) {
        const bool have_next = w.next(nxt);
        if (have_next && !scores(nxt, it + 1)) break;
        // latent output of tile it, accumulated in TMEM over the segment:
        // O^T[feature, head] += Z^T P'
        if (!warp_wait(smem_u32(&bars.sp_done), it & 1, abort_flag)) break;
        tc_fence_after();
        if (elect_one()) {
          const int slot = it % C::NS;
          const uint64_t za = zdesc_mn + ((slot * C::SLOT) >> 4);
          if (cur.first) {
#pragma unroll
            for (int ks = 0; ks < kPage / 16; ++ks)
#pragma unroll
              for (int mc = 0; mc < C::NMC; ++mc)
                mma_bf16_ss(tmem + C::COL_O + 16 * mc, za + (((C::mc_start(mc) / 64) * C::PCHUNK + ks * 2048) >> 4),
                            pdesc + ((ks * 512) >> 4), IDESC_PV, ks > 0);
          } else {
#pragma unroll
            for (int ks = 0; ks < kPage / 16; ++ks)
#pragma unroll
              for (int mc = 0; mc < C::NMC; ++mc)
                mma_bf16_ss(tmem + C::COL_O + 16 * mc, za + (((C::mc_start(mc) / 64) * C::PCHUNK + ks * 2048) >> 4),
                            pdesc + ((ks * 512) >> 4), IDESC_PV, 1);
          }
          mma_commit(smem_u32(&bars.o_ready));
          mma_commit(smem_u32(&bars.empty[slot]));
        }
        __syncwarp();
        last_bar = smem_u32(&bars.o_ready);
        last_par = it & 1;
        cur = nxt;
        have = have_next;
        ++it;
      }
      // drain: the last MMAs must finish before TMEM is released
      if (last_bar != 0) mbar_wait(last_bar, last_par, abort_flag);
    }
    __syncwarp();
  } else if (warp >= kGateWarp0 && warp < kGateWarp0 + 4) {
    // ---------------------------------------------------------------- zero fill of rows past a partial page
    regs_increase<kConsumerRegs>();
    const int gw = warp - kGateWarp0;
    const int row = gw * 16 + (lane & 15);    // token row of the page
    const int half = lane >> 4;               // 16-byte units 2k + half of every 128-byte chunk row
    Walker w;
    w.start(p.cu, p.seq_lens, p.batch);
    Tile t;
    int j = 0;
    while (w.next(t)) {
      const int slot = j % C::NS;
      if (!warp_wait(smem_u32(&bars.full[slot]), (j / C::NS) & 1, abort_flag)) break;
      uint8_t* crow = smem + slot * C::SLOT + row * 128;
      if (row >= t.ntok) {
#pragma unroll
        for (int fc = 0; fc < C::NCH; ++fc)
#pragma unroll
          for (int k = 0; k < 4; ++k)
            *reinterpret_cast<uint4*>(crow + fc * C::PCHUNK + (2 * k + half) * 16) = make_uint4(0, 0, 0, 0);
      }
      fence_proxy_async_smem();
      mbar_arrive(smem_u32(&bars.zready[slot]));
      ++j;
    }
  } else if (warp >= kSoftWarp0) {
    // ---------------------------------------------------------------- softmax, output read-out
    regs_increase<kConsumerRegs>();
    const int q4 = warp & 3;                   // TMEM lane quadrant of this warp
    const int srow = q4 * 16 + lane;           // token row of the M=64 score accumulator (lane < 16)
    const bool token_lane = lane < 16;
    const int frow = q4 * 32 + lane;           // latent feature row of the PV accumulator
    const uint32_t tl = tmem + (static_cast<uint32_t>(q4 * 32) << 16);
    // Online softmax with a lazily updated reference max m_ref per head: the
    // exponentials are taken against m_ref, which only moves (rescaling the
    // TMEM accumulator and l) when a tile's max exceeds it by more than
    // 2^kLazyLog2; otherwise the weights stay below 2^kLazyLog2.
    float m_ref[16], l_part[16];
    Walker w;
    w.start(p.cu, p.seq_lens, p.batch);
    Tile t;
    int it = 0, seg = -1, nseg_end = 0;
    while (w.next(t)) {
      if (t.first) {
        ++seg;
#pragma unroll
        for (int h = 0; h < 16; ++h) l_part[h] = 0.f;
        if (!warp_wait(smem_u32(&bars.qfull[seg & 1]), (seg >> 1) & 1, abort_flag)) break;
      }
      const int slot = it % C::NS;
      const int par = it & 1;
      if (!warp_wait(smem_u32(&bars.s_ready[par]), (it >> 1) & 1, abort_flag)) break;
      tc_fence_after();
      float sl[16], sr[16], s[16];
      tmem_ld16(tl + C::COL_S + par * C::S_COLS, sl);
      tmem_ld16(tl + C::COL_S + par * C::S_COLS + 16, sr);
      const bool valid = token_lane && srow < t.ntok;
      tmem_wait_ld();
#pragma unroll
      for (int h = 0; h < 16; ++h) s[h] = valid ? (sl[h] + sr[h]) * p.scale_log2 : -INFINITY;
      const float wmax = warp_reduce16<true>(s, lane);
      if ((lane & 1) == 0) red_max[(par * 16 + (lane >> 1)) * 4 + q4] = wmax;
      mbar_arrive(smem_u32(&bars.red[par]));
      if (!warp_wait(smem_u32(&bars.red[par]), (it >> 1) & 1, abort_flag)) break;
      // the previous tile's PV (same segment) must be complete before the
      // weight buffer is rewritten or the accumulator rescaled
      if (!t.first && !warp_wait(smem_u32(&bars.o_ready), (it - 1) & 1, abort_flag)) break;
      bool rescale = false;
      float alpha[16];
#pragma unroll
      for (int h = 0; h < 16; ++h) {
        const float4 rm = reinterpret_cast<const float4*>(red_max)[par * 16 + h];
        const float tmax = fmaxf(fmaxf(rm.x, rm.y), fmaxf(rm.z, rm.w));
        alpha[h] = 1.f;
        if (t.first) {
          m_ref[h] = tmax;
        } else if (tmax > m_ref[h] + kLazyLog2) {
          alpha[h] = exp2f(m_ref[h] - tmax);
          m_ref[h] = tmax;
          rescale = true;
        }
      }
      if (rescale) {
        // every thread saw the same maxima, so the branch is uniform
        tc_fence_after();
#pragma unroll
        for (int mc = 0; mc < C::NMC; ++mc) {
          float o[16];
          tmem_ld16(tl + C::COL_O + 16 * mc, o);
          tmem_wait_ld();
#pragma unroll
          for (int h = 0; h < 16; ++h) o[h] *= alpha[h];
          tmem_st16(tl + C::COL_O + 16 * mc, o);
        }
        tmem_wait_st();
#pragma unroll
        for (int h = 0; h < 16; ++h) l_part[h] *= alpha[h];
      }
      // The PV MMA sees the bf16-rounded weights P'; the denominator sums the
      // same rounded values, so their rounding cancels in o = sum P' z / l.
#pragma unroll
      for (int h = 0; h < 16; ++h) s[h] = ex2_approx(s[h] - m_ref[h]);
      uint32_t pw[8];
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        pw[k] = pack_bf16x2(s[2 * k], s[2 * k + 1]);
        const float2 pq = unpack_bf16x2(pw[k]);
        l_part[2 * k] += pq.x;
        l_part[2 * k + 1] += pq.y;
      }
      // P'[token][head] as an MN-major B operand: 8x8 core matrices, token group
      // stride 256 B, head group stride 128 B
      if (token_lane) {
        uint8_t* prow = smem + C::OFF_PBUF + (srow >> 3) * 256 + (srow & 7) * 16;
        *reinterpret_cast<uint4*>(prow) = make_uint4(pw[0], pw[1], pw[2], pw[3]);
        *reinterpret_cast<uint4*>(prow + 128) = make_uint4(pw[4], pw[5], pw[6], pw[7]);
      }
      fence_proxy_async_smem();
      tc_fence_before();
      mbar_arrive(smem_u32(&bars.sp_done));

      if (t.last) {
        mbar_arrive(smem_u32(&bars.qempty[seg & 1]));
        // ---- segment end: reduce l over the token rows
        const float lw = warp_reduce16<false>(l_part, lane);
        if ((lane & 1) == 0) red_sum[q4 * 32 + (lane >> 1)] = lw;
        mbar_arrive(smem_u32(&bars.sum));
        if (!warp_wait(smem_u32(&bars.sum), nseg_end & 1, abort_flag)) break;
        ++nseg_end;
        float lh[16];
#pragma unroll
        for (int h = 0; h < 16; ++h) lh[h] = red_sum[h] + red_sum[32 + h] + red_sum[64 + h] + red_sum[96 + h];
        // the segment's last PV, then the accumulated latent output
        if (!warp_wait(smem_u32(&bars.o_ready), it & 1, abort_flag)) break;
        tc_fence_after();
        const int slot_out = blockIdx.x + t.b;
        float* po = p.part_o + static_cast<size_t>(slot_out) * kHeads * D_C;
#pragma unroll
        for (int mc = 0; mc < C::NMC; ++mc) {
          float o[16];
          tmem_ld16(tl + C::COL_O + 16 * mc, o);
          tmem_wait_ld();
          const int f = C::mc_start(mc) + frow;
          if (mc == 0 || f >= 128 * mc) {
#pragma unroll
            for (int h = 0; h < 16; ++h)
              po[h * D_C + f] = o[h];
          }
        }
        tc_fence_before();
        if (frow < 16) {
          float mv = 0.f, lv = 0.f;
#pragma unroll
          for (int h = 0; h < 16; ++h)
            if (h == frow) {
              mv = m_ref[h];
              lv = lh[h];
            }
          float* ml = p.part_ml + (static_cast<size_t>(slot_out) * kHeads + frow) * 2;
          ml[0] = mv;
          ml[1] = lv;
        }
      }
      ++it;
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tmem, C::TMEM_COLS);
  if (threadIdx.x == 0 && bars.abort) report_status(p.status, kStatusTimeout);
}

template <int D_C>
cudaError_t launch_one(const DecodeArgs& a, const CUtensorMap* maps, cudaStream_t st) {
  using C = Cfg<D_C>;
  auto kern = decode_tc_kernel<D_C>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)C::SMEM);
  if (e != cudaSuccess) return e;
  const WorkspaceLayout wl = workspace_layout(a.batch, a.num_splits, kHeads, D_C, kRope, true);
  uint8_t* ws = static_cast<uint8_t*>(a.workspace);
  TcParams p;
  p.block_table = a.block_table;
  p.seq_lens = a.seq_lens;
  p.qprep = ws + wl.off_qprep;
  p.cu = reinterpret_cast<const int32_t*>(ws + wl.off_cu);
  p.part_ml = reinterpret_cast<float*>(ws + wl.off_ml);
  p.part_o = reinterpret_cast<float*>(ws + wl.off_o);
  p.status = a.status;
  p.batch = a.batch;
  p.max_pages = a.max_pages;
  p.num_pages = a.num_pages;
  p.scale_log2 = a.scale_log2;
  // set-up overlaps the query-absorption kernel before it on the stream
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(a.num_splits);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = C::SMEM;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, maps[0], maps[1], p);
}

}  // namespace

cudaError_t launch_decode_wide(const DecodeArgs& a, const CUtensorMap* maps, cudaStream_t st) {
  if (a.d_c == 512 && !a.gate) return launch_one<512>(a, maps, st);
  return cudaErrorInvalidValue;
}

}  // namespace egmla
