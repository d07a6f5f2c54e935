// egmla_decode_tc.cu - split-KV EG-MLA decode on sm_103a tensor cores.
//
// One CTA per split-KV work unit (see egmla_common.cuh for the schedule).  The
// CTA streams its cache pages two at a time (a 128-token tile) through a ring
// of shared-memory entries and runs, per tile:
//
//   TMA (warp 0)    latent page [64 tok x d_c] and RoPE-key page [64 x 64] as
//                   128-byte-swizzled boxes, plus the page's token ids.
//   gate (warps 2-5, one thread per token)
//                   g = G[id] gathered from global memory, z = c (*) g rounded
//                   to bf16 and written back in place, and the LayerNorm
//                   statistics mu, r = 1/sqrt(var + eps) of z (Eq. 5 over d_c).
//   MMA (warp 1)    S_lat = Z Bq^T and S_rope = K^R Q^R^T on tcgen05 with fp32
//                   accumulators in TMEM (M = 128 tokens, N = 16 heads).
//   softmax (warps 2-5)
//                   s = scale * (r (S_lat - mu w) + b + S_rope): the LayerNorm
//                   is applied after the MMA, because
//                   q^.LN(z) = r (q^ gamma).z - r mu sum(q^ gamma) + q^.beta;
//                   online softmax over the tile with a running max per head;
//                   P' = p r (bf16) is written as the B operand of the PV MMA.
//   MMA (warp 1)    O_tile = Z^T P' (M = 128 latent features, N = 16 heads).
//   accumulate (warps 2-5, one thread per latent feature)
//                   O = O alpha + O_tile in registers.
//
// At the end of each sequence segment the un-normalised latent output
// gamma (*) (O - sum_j P'_j mu_j) + beta l, the running max m and the
// denominator l are written as this split's partial result.
//
// The queries are absorbed before this kernel (q^ = W_UK^T q^C, with gamma
// folded in); W_UV is applied after the split merge.  Everything the kernel
// waits on has a time limit: on expiry it records EG_MLA_ERR_TIMEOUT, drains
// its own copies and MMAs, frees TMEM and exits.
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
constexpr int kTile = 128;
constexpr int kThreads = 192;  // warp 0 TMA, warp 1 MMA + TMEM owner, warps 2-5 gate/softmax
constexpr uint32_t kSmemLimit = 232448;
constexpr float kLog2e = 1.4426950408889634f;

template <int D_C, bool GATE>
struct Cfg {
  static constexpr int NCH = D_C / 64;                  // 64-feature swizzle-atom columns
  static constexpr int NMC = (D_C + 127) / 128;         // 128-feature M chunks of the PV MMA
  static constexpr uint32_t CHUNK = kTile * 128;        // one atom column of a tile: 16 KB
  static constexpr uint32_t PAGE_CHUNK = kPage * 128;   // one atom column of a page: 8 KB
  static constexpr uint32_t C_BYTES = NCH * CHUNK;
  static constexpr uint32_t KR_OFF = C_BYTES;
  static constexpr uint32_t ID_OFF = C_BYTES + CHUNK;
  static constexpr uint32_t ENTRY = (ID_OFF + kTile * 4 + 1023) / 1024 * 1024;
  static constexpr uint32_t QB_LAT = kHeads * D_C * 2;
  static constexpr uint32_t QB_ROPE = kHeads * kRope * 2;
  static constexpr uint32_t QPREP = QB_LAT + QB_ROPE + 128;
  static constexpr uint32_t QBUF = (QPREP + 1023) / 1024 * 1024;
  static constexpr uint32_t PBUF = kTile * kHeads * 2;
  static constexpr uint32_t MISC = 2048;
  static constexpr int NS_FIT = (int)((kSmemLimit - 1024 - 2 * QBUF - PBUF - MISC) / ENTRY);
  static constexpr int NS = NS_FIT > 4 ? 4 : NS_FIT;
  static constexpr uint32_t OFF_QBUF = NS * ENTRY;
  static constexpr uint32_t OFF_PBUF = OFF_QBUF + 2 * QBUF;
  static constexpr uint32_t OFF_MISC = OFF_PBUF + PBUF;
  static constexpr uint32_t SMEM = OFF_MISC + MISC + 1024;
  static constexpr uint32_t COL_SLAT = 0, COL_SROPE = 16, COL_O = 32;
  static constexpr uint32_t TMEM_COLS = 128;
  static constexpr uint32_t PAGE_TX = NCH * PAGE_CHUNK + PAGE_CHUNK + (GATE ? kPage * 4 : 0);
  static_assert(NS >= 1, "one ring entry must fit");
  static_assert(SMEM <= kSmemLimit, "shared memory");
  static_assert(COL_O + 16 * NMC <= TMEM_COLS, "TMEM columns");
  static_assert(D_C % 64 == 0 && D_C >= 128, "d_c");
  // first latent feature of PV M-chunk j; the last chunk is shifted back so that
  // it ends at D_C (for D_C = 192 it overlaps the previous one by 64 features)
  __host__ __device__ static constexpr int mc_start(int j) {
    return (128 * j + 128 <= D_C) ? 128 * j : D_C - 128;
  }
};

struct TcParams {
  const int32_t* id_pool;
  const int32_t* block_table;
  const int32_t* seq_lens;
  const __nv_bfloat16* gate_table;
  const float* gamma;
  const float* beta;
  const uint8_t* qprep;
  const int32_t* cu;
  float* part_ml;
  float* part_o;
  int32_t* status;
  int batch, max_pages, num_pages, vocab;
  float scale_log2, eps;
  __nv_bfloat16* dump_c;
  __nv_bfloat16* dump_kr;
  int32_t* dump_ids;
  __nv_bfloat16* dump_g;
  int dump_len;
};

// shared-memory barrier block (inside MISC, after 1 KB of reduction scratch)
struct Bars {
  uint64_t full[4], empty[4], qfull[2], qempty[2];
  uint64_t a_ready, s_ready, p_ready, o_ready;
  uint64_t red[2], sum;
  uint32_t tmem_base;
  int abort;
};

struct Tile {
  int b, lp, npg, ntok, tok0;
  bool first, last;
};

// Walks this CTA's pages in 2-page tiles, segment by segment (identically in
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
    const int base = __ldg(cu + b);
    lp = g - base;
    lp_end = min(g1, __ldg(cu + b + 1)) - base;
    L = __ldg(lens + b);
    first = true;
  }
  __device__ bool next(Tile& t) {
    if (done) return false;
    t.b = b;
    t.lp = lp;
    t.npg = min(2, lp_end - lp);
    t.tok0 = lp * kPage;
    t.ntok = min(t.npg * kPage, L - t.tok0);
    t.first = first;
    first = false;
    lp += t.npg;
    t.last = lp >= lp_end;
    if (t.last) {
      const int g = __ldg(cu + b) + lp_end;
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

__device__ __forceinline__ uint32_t mul_bf16x2(uint32_t a, uint32_t b) {
  __nv_bfloat162 x = *reinterpret_cast<__nv_bfloat162*>(&a);
  __nv_bfloat162 y = *reinterpret_cast<__nv_bfloat162*>(&b);
  __nv_bfloat162 z = __hmul2(x, y);
  return *reinterpret_cast<uint32_t*>(&z);
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

template <int D_C, bool GATE, bool DUMP>
__global__ void __launch_bounds__(kThreads, 1)
    decode_tc_kernel(const __grid_constant__ CUtensorMap cmap, const __grid_constant__ CUtensorMap krmap,
                     const TcParams p) {
  using C = Cfg<D_C, GATE>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const uint32_t sbase = smem_u32(smem);
  float* red_max = reinterpret_cast<float*>(smem + C::OFF_MISC);         // [2][4][16]
  float* red_sum = red_max + 2 * 4 * 16;                                 // [4][32]
  Bars& bars = *reinterpret_cast<Bars*>(smem + C::OFF_MISC + 1024);
  volatile int* abort_flag = &bars.abort;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int s = 0; s < C::NS; ++s) {
      mbar_init(smem_u32(&bars.full[s]), 1);
      mbar_init(smem_u32(&bars.empty[s]), DUMP ? 128 : 1);
    }
    for (int s = 0; s < 2; ++s) {
      mbar_init(smem_u32(&bars.qfull[s]), 1);
      mbar_init(smem_u32(&bars.qempty[s]), 1 + 128);
      mbar_init(smem_u32(&bars.red[s]), 128);
    }
    mbar_init(smem_u32(&bars.a_ready), 128);
    mbar_init(smem_u32(&bars.s_ready), 1);
    mbar_init(smem_u32(&bars.p_ready), 128);
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

  if (warp == 0) {
    // ---------------------------------------------------------------- TMA producer
    if (lane == 0) {
      prefetch_tensormap(&cmap);
      prefetch_tensormap(&krmap);
      const uint64_t pol_stream = policy_evict_first();
      Walker w;
      w.start(p.cu, p.seq_lens, p.batch);
      Tile t;
      int it = 0, seg = -1;
      int last_it[4] = {-1, -1, -1, -1};
      int last_qseg[2] = {-1, -1};
      while (w.next(t)) {
        if (t.first) {
          ++seg;
          if (!DUMP) {
            const int qb = seg & 1;
            if (!mbar_wait(smem_u32(&bars.qempty[qb]), ((seg >> 1) & 1) ^ 1, abort_flag)) break;
            mbar_arrive_expect_tx(smem_u32(&bars.qfull[qb]), C::QPREP);
            bulk_load(sbase + C::OFF_QBUF + qb * C::QBUF, p.qprep + static_cast<size_t>(t.b) * C::QPREP, C::QPREP,
                      smem_u32(&bars.qfull[qb]));
            last_qseg[qb] = seg;
          }
        }
        const int slot = it % C::NS;
        if (!mbar_wait(smem_u32(&bars.empty[slot]), ((it / C::NS) & 1) ^ 1, abort_flag)) break;
        int pg[2] = {-1, -1};
        uint32_t tx = 0;
        for (int pp = 0; pp < t.npg; ++pp) {
          const int v = __ldg(p.block_table + static_cast<size_t>(t.b) * p.max_pages + t.lp + pp);
          if (v >= 0 && v < p.num_pages) {
            pg[pp] = v;
            tx += C::PAGE_TX;
          } else {
            report_status(p.status, kStatusOutOfRange);
          }
        }
        const uint32_t fb = smem_u32(&bars.full[slot]);
        mbar_arrive_expect_tx(fb, tx);
        const uint32_t ent = sbase + slot * C::ENTRY;
        for (int pp = 0; pp < 2; ++pp) {
          if (pg[pp] < 0) continue;
          const int y = pg[pp] * kPage;
#pragma unroll
          for (int fc = 0; fc < C::NCH; ++fc)
            tma_load_2d(ent + fc * C::CHUNK + pp * C::PAGE_CHUNK, &cmap, fc * 64, y, fb, pol_stream);
          tma_load_2d(ent + C::KR_OFF + pp * C::PAGE_CHUNK, &krmap, 0, y, fb, pol_stream);
          if (GATE) bulk_load(ent + C::ID_OFF + pp * kPage * 4, p.id_pool + static_cast<size_t>(pg[pp]) * kPage,
                              kPage * 4, fb);
        }
        last_it[slot] = it;
        ++it;
      }
      // drain: every copy this thread issued must land before the CTA exits
      for (int s = 0; s < C::NS; ++s)
        if (last_it[s] >= 0) mbar_wait(smem_u32(&bars.full[s]), (last_it[s] / C::NS) & 1, abort_flag);
      for (int s = 0; s < 2; ++s)
        if (last_qseg[s] >= 0) mbar_wait(smem_u32(&bars.qfull[s]), (last_qseg[s] >> 1) & 1, abort_flag);
    }
    __syncwarp();
  } else if (warp == 1) {
    // ---------------------------------------------------------------- MMA issuer
    if (lane == 0) {
      constexpr uint32_t IDESC_QK = idesc_bf16(128, 16, 0, 0);
      constexpr uint32_t IDESC_PV = idesc_bf16(128, 16, 1, 1);
      Walker w;
      w.start(p.cu, p.seq_lens, p.batch);
      Tile t;
      int it = 0, seg = -1;
      uint32_t last_bar = 0, last_par = 0;
      while (w.next(t)) {
        if (t.first) {
          ++seg;
          if (!DUMP && !mbar_wait(smem_u32(&bars.qfull[seg & 1]), (seg >> 1) & 1, abort_flag)) break;
        }
        if (DUMP) break;  // the cache-read test entry issues no MMA
        const int slot = it % C::NS;
        if (!mbar_wait(smem_u32(&bars.a_ready), it & 1, abort_flag)) break;
        tc_fence_after();
        const uint32_t ent = sbase + slot * C::ENTRY;
        const uint32_t qbuf = sbase + C::OFF_QBUF + (seg & 1) * C::QBUF;
        // scores: latent part (K = d_c) and RoPE part (K = 64) into separate accumulators
#pragma unroll
        for (int kk = 0; kk < D_C / 16; ++kk) {
          const uint64_t a = smem_desc(ent + (kk >> 2) * C::CHUNK + (kk & 3) * 32, 16, 1024, kSwizzle128B);
          const uint64_t b = smem_desc(qbuf + kk * 512, 256, 128, kSwizzleNone);
          mma_bf16_ss(tmem + C::COL_SLAT, a, b, IDESC_QK, kk > 0);
        }
#pragma unroll
        for (int kk = 0; kk < kRope / 16; ++kk) {
          const uint64_t a = smem_desc(ent + C::KR_OFF + kk * 32, 16, 1024, kSwizzle128B);
          const uint64_t b = smem_desc(qbuf + C::QB_LAT + kk * 512, 256, 128, kSwizzleNone);
          mma_bf16_ss(tmem + C::COL_SROPE, a, b, IDESC_QK, kk > 0);
        }
        mma_commit(smem_u32(&bars.s_ready));
        last_bar = smem_u32(&bars.s_ready);
        last_par = it & 1;
        if (t.last) mma_commit(smem_u32(&bars.qempty[seg & 1]));
        if (!mbar_wait(smem_u32(&bars.p_ready), it & 1, abort_flag)) break;
        tc_fence_after();
        // latent output: O^T[feature, head] += Z^T P'
        const int nks = (t.ntok + 15) >> 4;
        const uint32_t pbuf = sbase + C::OFF_PBUF;
        for (int ks = 0; ks < nks; ++ks) {
          const uint64_t b = smem_desc(pbuf + ks * 512, 256, 128, kSwizzleNone);
#pragma unroll
          for (int mc = 0; mc < C::NMC; ++mc) {
            const uint64_t a = smem_desc(ent + (C::mc_start(mc) / 64) * C::CHUNK + ks * 2048, C::CHUNK, 1024,
                                         kSwizzle128B);
            mma_bf16_ss(tmem + C::COL_O + 16 * mc, a, b, IDESC_PV, ks > 0);
          }
        }
        mma_commit(smem_u32(&bars.o_ready));
        mma_commit(smem_u32(&bars.empty[slot]));
        last_bar = smem_u32(&bars.o_ready);
        last_par = it & 1;
        ++it;
      }
      // drain: the last MMAs must finish before TMEM is released
      if (last_bar != 0) mbar_wait(last_bar, last_par, abort_flag);
    }
    __syncwarp();
  } else {
    // ---------------------------------------------------------------- gate / softmax / accumulate
    const int q4 = warp & 3;                 // TMEM lane quadrant of this warp
    const int row = q4 * 32 + lane;          // token row of the tile; latent feature in O chunks
    const uint32_t tl = tmem + (static_cast<uint32_t>(q4 * 32) << 16);
    float m_run[16], l_part[16], bmu_part[16], alpha[16];
    float acc[C::NMC][16];
    float gam[C::NMC], bet[C::NMC];
#pragma unroll
    for (int mc = 0; mc < C::NMC; ++mc) {
      const int f = C::mc_start(mc) + row;
      gam[mc] = (GATE && p.gamma) ? p.gamma[f] : 1.f;
      bet[mc] = (GATE && p.beta) ? p.beta[f] : 0.f;
    }
    float wq[16], bq[16];
    const uint64_t pol_keep = policy_evict_last();
    Walker w;
    w.start(p.cu, p.seq_lens, p.batch);
    Tile t;
    int it = 0, seg = -1, nseg_end = 0;
    while (w.next(t)) {
      if (t.first) {
        ++seg;
#pragma unroll
        for (int h = 0; h < 16; ++h) {
          m_run[h] = -INFINITY;
          l_part[h] = 0.f;
          bmu_part[h] = 0.f;
#pragma unroll
          for (int mc = 0; mc < C::NMC; ++mc) acc[mc][h] = 0.f;
        }
        if (!DUMP) {
          const int qb = seg & 1;
          if (!warp_wait(smem_u32(&bars.qfull[qb]), (seg >> 1) & 1, abort_flag)) break;
          const float* sums = reinterpret_cast<const float*>(smem + C::OFF_QBUF + qb * C::QBUF + C::QB_LAT + C::QB_ROPE);
#pragma unroll
          for (int h = 0; h < 16; ++h) {
            wq[h] = GATE ? sums[h] : 0.f;
            bq[h] = GATE ? sums[16 + h] : 0.f;
          }
          mbar_arrive(smem_u32(&bars.qempty[qb]));
        }
      }
      const int slot = it % C::NS;
      if (!warp_wait(smem_u32(&bars.full[slot]), (it / C::NS) & 1, abort_flag)) break;
      uint8_t* ent = smem + slot * C::ENTRY;
      uint8_t* crow = ent + row * 128;
      const int sw = row & 7;
      const bool valid = row < t.ntok;
      const int32_t* ids = reinterpret_cast<const int32_t*>(ent + C::ID_OFF);

      if (DUMP) {
        if (valid) {
          int id = ids[row];
          const size_t o = static_cast<size_t>(t.b) * p.dump_len + t.tok0 + row;
          p.dump_ids[o] = id;
          if ((unsigned)id >= (unsigned)p.vocab) id = 0;
          const uint4* grow = reinterpret_cast<const uint4*>(p.gate_table + static_cast<size_t>(id) * D_C);
          uint4* dc = reinterpret_cast<uint4*>(p.dump_c + o * D_C);
          uint4* dg = reinterpret_cast<uint4*>(p.dump_g + o * D_C);
          uint4* dk = reinterpret_cast<uint4*>(p.dump_kr + o * kRope);
          for (int fc = 0; fc < C::NCH; ++fc)
            for (int u = 0; u < 8; ++u) {
              dc[fc * 8 + u] = *reinterpret_cast<const uint4*>(crow + fc * C::CHUNK + ((u ^ sw) << 4));
              dg[fc * 8 + u] = grow[fc * 8 + u];
            }
          for (int u = 0; u < 8; ++u)
            dk[u] = *reinterpret_cast<const uint4*>(ent + C::KR_OFF + row * 128 + ((u ^ sw) << 4));
        }
        mbar_arrive(smem_u32(&bars.empty[slot]));
        ++it;
        continue;
      }

      // ---- gate: z = c (*) G[id] in place (bf16), LayerNorm statistics of z
      float mu = 0.f, rstd = 1.f;
      if (GATE) {
        int id = 0;
        if (valid) {
          id = ids[row];
          if ((unsigned)id >= (unsigned)p.vocab) {
            report_status(p.status, kStatusOutOfRange);
            id = 0;
          }
        }
        const uint8_t* grow = reinterpret_cast<const uint8_t*>(p.gate_table) + static_cast<size_t>(id) * D_C * 2;
        float2 s1 = make_float2(0.f, 0.f), s2 = make_float2(0.f, 0.f);
        uint4 gv[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) gv[u] = valid ? ldg_16_hint(grow + u * 16, pol_keep) : make_uint4(0, 0, 0, 0);
#pragma unroll
        for (int fc = 0; fc < C::NCH; ++fc) {
          uint4 gn[8];
#pragma unroll
          for (int u = 0; u < 8; ++u)
            gn[u] = (valid && fc + 1 < C::NCH) ? ldg_16_hint(grow + (fc + 1) * 128 + u * 16, pol_keep)
                                               : make_uint4(0, 0, 0, 0);
#pragma unroll
          for (int u = 0; u < 8; ++u) {
            uint4* cp = reinterpret_cast<uint4*>(crow + fc * C::CHUNK + ((u ^ sw) << 4));
            const uint4 c = *cp;
            uint4 z;
            z.x = mul_bf16x2(c.x, gv[u].x);
            z.y = mul_bf16x2(c.y, gv[u].y);
            z.z = mul_bf16x2(c.z, gv[u].z);
            z.w = mul_bf16x2(c.w, gv[u].w);
            if (!valid) z = make_uint4(0, 0, 0, 0);
            const float2 f0 = unpack_bf16x2(z.x), f1 = unpack_bf16x2(z.y);
            const float2 f2 = unpack_bf16x2(z.z), f3 = unpack_bf16x2(z.w);
            s1 = __fadd2_rn(s1, f0);
            s1 = __fadd2_rn(s1, f1);
            s1 = __fadd2_rn(s1, f2);
            s1 = __fadd2_rn(s1, f3);
            s2 = __ffma2_rn(f0, f0, s2);
            s2 = __ffma2_rn(f1, f1, s2);
            s2 = __ffma2_rn(f2, f2, s2);
            s2 = __ffma2_rn(f3, f3, s2);
            *cp = z;
          }
#pragma unroll
          for (int u = 0; u < 8; ++u) gv[u] = gn[u];
        }
        constexpr float inv_dc = 1.f / D_C;
        mu = (s1.x + s1.y) * inv_dc;
        const float var = fmaxf((s2.x + s2.y) * inv_dc - mu * mu, 0.f);
        rstd = rsqrtf(var + p.eps);
      } else if (!valid) {
#pragma unroll
        for (int fc = 0; fc < C::NCH; ++fc)
#pragma unroll
          for (int u = 0; u < 8; ++u)
            *reinterpret_cast<uint4*>(crow + fc * C::CHUNK + u * 16) = make_uint4(0, 0, 0, 0);
      }
      fence_proxy_async_smem();
      mbar_arrive(smem_u32(&bars.a_ready));

      // ---- scores and online softmax over the tile
      if (!warp_wait(smem_u32(&bars.s_ready), it & 1, abort_flag)) break;
      tc_fence_after();
      float sl[16], sr[16], s[16];
      tmem_ld16(tl + C::COL_SLAT, sl);
      tmem_ld16(tl + C::COL_SROPE, sr);
      tmem_wait_ld();
#pragma unroll
      for (int h = 0; h < 16; ++h) {
        const float lat = GATE ? rstd * (sl[h] - mu * wq[h]) + bq[h] : sl[h];
        s[h] = valid ? (lat + sr[h]) * p.scale_log2 : -INFINITY;
      }
      const int par = it & 1;
      const float wmax = warp_reduce16<true>(s, lane);
      if ((lane & 1) == 0) red_max[(par * 4 + q4) * 16 + (lane >> 1)] = wmax;
      mbar_arrive(smem_u32(&bars.red[par]));
      if (!warp_wait(smem_u32(&bars.red[par]), (it >> 1) & 1, abort_flag)) break;
      uint32_t pw[8];
#pragma unroll
      for (int h = 0; h < 16; ++h) {
        const float* rm = red_max + par * 64 + h;
        const float tmax = fmaxf(fmaxf(rm[0], rm[16]), fmaxf(rm[32], rm[48]));
        const float mn = fmaxf(m_run[h], tmax);
        alpha[h] = exp2f(m_run[h] - mn);
        m_run[h] = mn;
        const float pr = exp2f(s[h] - mn);
        s[h] = GATE ? pr * rstd : pr;
      }
      // The PV MMA sees the bf16-rounded weights P'; the denominator and the mean
      // correction use the same rounded values (l = sum P'/r), so the rounding of
      // P' cancels in o = (sum P' z - sum P' mu) / l instead of biasing it.
      const float inv_r = GATE ? 1.f / rstd : 1.f;
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        pw[k] = pack_bf16x2(s[2 * k], s[2 * k + 1]);
        const float2 pq = unpack_bf16x2(pw[k]);
        l_part[2 * k] = fmaf(l_part[2 * k], alpha[2 * k], pq.x * inv_r);
        l_part[2 * k + 1] = fmaf(l_part[2 * k + 1], alpha[2 * k + 1], pq.y * inv_r);
        if (GATE) {
          bmu_part[2 * k] = fmaf(bmu_part[2 * k], alpha[2 * k], pq.x * mu);
          bmu_part[2 * k + 1] = fmaf(bmu_part[2 * k + 1], alpha[2 * k + 1], pq.y * mu);
        }
      }
      // P'[token][head] as an MN-major B operand: 8x8 core matrices, token group
      // stride 256 B, head group stride 128 B
      uint8_t* prow = smem + C::OFF_PBUF + (row >> 3) * 256 + (row & 7) * 16;
      *reinterpret_cast<uint4*>(prow) = make_uint4(pw[0], pw[1], pw[2], pw[3]);
      *reinterpret_cast<uint4*>(prow + 128) = make_uint4(pw[4], pw[5], pw[6], pw[7]);
      fence_proxy_async_smem();
      tc_fence_before();
      mbar_arrive(smem_u32(&bars.p_ready));

      // ---- accumulate the tile's latent output (this thread: one feature per M chunk)
      if (!warp_wait(smem_u32(&bars.o_ready), it & 1, abort_flag)) break;
      tc_fence_after();
#pragma unroll
      for (int mc = 0; mc < C::NMC; ++mc) {
        float o[16];
        tmem_ld16(tl + C::COL_O + 16 * mc, o);
        tmem_wait_ld();
#pragma unroll
        for (int h = 0; h < 16; ++h) acc[mc][h] = fmaf(acc[mc][h], alpha[h], o[h]);
      }
      tc_fence_before();

      if (t.last) {
        // ---- segment end: reduce l and sum_j P'_j mu_j over the 128 token rows
        const float lw = warp_reduce16<false>(l_part, lane);
        const float bw = GATE ? warp_reduce16<false>(bmu_part, lane) : 0.f;
        if ((lane & 1) == 0) {
          red_sum[q4 * 32 + (lane >> 1)] = lw;
          red_sum[q4 * 32 + 16 + (lane >> 1)] = bw;
        }
        mbar_arrive(smem_u32(&bars.sum));
        if (!warp_wait(smem_u32(&bars.sum), nseg_end & 1, abort_flag)) break;
        ++nseg_end;
        float lh[16], bh[16];
#pragma unroll
        for (int h = 0; h < 16; ++h) {
          lh[h] = red_sum[h] + red_sum[32 + h] + red_sum[64 + h] + red_sum[96 + h];
          bh[h] = red_sum[16 + h] + red_sum[48 + h] + red_sum[80 + h] + red_sum[112 + h];
        }
        const int slot_out = blockIdx.x + t.b;
        float* po = p.part_o + static_cast<size_t>(slot_out) * kHeads * D_C;
#pragma unroll
        for (int mc = 0; mc < C::NMC; ++mc) {
          const int f = C::mc_start(mc) + row;
          if (mc == 0 || f >= 128 * mc) {
#pragma unroll
            for (int h = 0; h < 16; ++h)
              po[h * D_C + f] = GATE ? fmaf(gam[mc], acc[mc][h] - bh[h], bet[mc] * lh[h]) : acc[mc][h];
          }
        }
        if (row < 16) {
          float mv = 0.f, lv = 0.f;
#pragma unroll
          for (int h = 0; h < 16; ++h)
            if (h == row) {
              mv = m_run[h];
              lv = lh[h];
            }
          float* ml = p.part_ml + (static_cast<size_t>(slot_out) * kHeads + row) * 2;
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

template <int D_C, bool GATE, bool DUMP>
cudaError_t launch_one(const DecodeArgs& a, const CUtensorMap* maps, cudaStream_t st) {
  using C = Cfg<D_C, GATE>;
  auto kern = decode_tc_kernel<D_C, GATE, DUMP>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)C::SMEM);
  if (e != cudaSuccess) return e;
  const WorkspaceLayout wl = workspace_layout(a.batch, a.num_splits, kHeads, D_C, kRope, true);
  uint8_t* ws = static_cast<uint8_t*>(a.workspace);
  TcParams p;
  p.id_pool = a.id_pool;
  p.block_table = a.block_table;
  p.seq_lens = a.seq_lens;
  p.gate_table = static_cast<const __nv_bfloat16*>(a.gate_table);
  p.gamma = a.ln_gamma;
  p.beta = a.ln_beta;
  p.qprep = ws + wl.off_qprep;
  p.cu = reinterpret_cast<const int32_t*>(ws + wl.off_cu);
  p.part_ml = reinterpret_cast<float*>(ws + wl.off_ml);
  p.part_o = reinterpret_cast<float*>(ws + wl.off_o);
  p.status = a.status;
  p.batch = a.batch;
  p.max_pages = a.max_pages;
  p.num_pages = a.num_pages;
  p.vocab = a.vocab;
  p.scale_log2 = a.scale_log2;
  p.eps = a.eps;
  p.dump_c = static_cast<__nv_bfloat16*>(a.dump_c);
  p.dump_kr = static_cast<__nv_bfloat16*>(a.dump_kr);
  p.dump_ids = a.dump_ids;
  p.dump_g = static_cast<__nv_bfloat16*>(a.dump_g);
  p.dump_len = a.max_seq_len;
  kern<<<a.num_splits, kThreads, C::SMEM, st>>>(maps[0], maps[1], p);
  return cudaGetLastError();
}

}  // namespace

bool tc_supported(int d_c, int gate) {
  if (gate) return d_c == 192 || d_c == 256;
  return d_c == 192 || d_c == 256 || d_c == 512;
}

cudaError_t launch_decode_tc(const DecodeArgs& a, const CUtensorMap* maps, bool dump, cudaStream_t st) {
  if (dump) {
    if (a.d_c == 192) return launch_one<192, true, true>(a, maps, st);
    if (a.d_c == 256) return launch_one<256, true, true>(a, maps, st);
    return cudaErrorInvalidValue;
  }
  if (a.gate) {
    if (a.d_c == 192) return launch_one<192, true, false>(a, maps, st);
    if (a.d_c == 256) return launch_one<256, true, false>(a, maps, st);
  } else {
    if (a.d_c == 192) return launch_one<192, false, false>(a, maps, st);
    if (a.d_c == 256) return launch_one<256, false, false>(a, maps, st);
    if (a.d_c == 512) return launch_one<512, false, false>(a, maps, st);
  }
  return cudaErrorInvalidValue;
}

}  // namespace egmla
