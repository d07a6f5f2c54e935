// egmla_decode_tc.cu - split-KV EG-MLA decode on sm_103a tensor cores for the
// latent widths 192 and 256 (gated or plain).
//
// One CTA per split-KV work unit (see egmla_common.cuh for the schedule).  The
// CTA streams its cache pages, one 64-token page per tile, through a ring of
// shared-memory slots.  Four roles run concurrently on different tiles:
//
//   TMA (warp 3)      latent page [64 tok x d_c] (one 3-D box: 64-feature
//                     columns x 64 rows) and RoPE-key page [64 x 64], both
//                     128-byte swizzled.
//   gate (warps 4-11; each quarter-warp owns two token rows, lane u the 16-byte
//                     unit u of every 64-feature column of them)
//                     the token ids (two tiles ahead) and the gate rows
//                     g = G[id] (EG-MLA-A table, Section 5.2; one tile ahead)
//                     from L2 into registers, every quarter-warp load reading
//                     one whole 128-byte line; z = c (*) g rounded to bf16 and
//                     written back in place, and the LayerNorm statistics
//                     mu, r = 1/sqrt(var + eps) of z (Eq. 5 over d_c).
//   scores (warp 2)   transposed scores S^T = Q Z^T and S_rope^T = Q^R K^R^T on
//                     tcgen05 (M = 64 rows, N = 64 tokens, fp32 in TMEM,
//                     double-buffered).  The operand rows of heads 0-7 and 8-15
//                     are placed so that their accumulator rows fall in TMEM lane
//                     quadrants 0 and 1.
//   output (warp 3, with the TMA loads) the latent output O += P' Z (M = 64
//                     rows, N = d_c features, K = 64 tokens), accumulated in
//                     TMEM over a sequence segment.  Issued by its own thread, so
//                     that the scores of later tiles never queue behind it.
//   softmax (warps 0 and 1, heads 0-7 and 8-15)
//                     reads its eight head rows of S^T spread over the 32
//                     threads (one head x 16 tokens each), s = scale * (r (S -
//                     mu w) + b + S_rope) -- the LayerNorm applied after the MMA,
//                     since q^.LN(z) = r (q^ gamma).z - r mu sum(q^ gamma) +
//                     q^.beta --, an online softmax whose per-head maxima need no
//                     exchange beyond the four threads of a head, and P' = p r
//                     (bf16) as the A operand of the output MMA.
//
// With heads in the accumulator rows, the running max, its lazy rescaling of
// O and the final read-out of a head all stay inside one softmax warp.  At the end of each
// sequence segment the un-normalised latent output gamma (*) (O - sum_j P'_j
// mu_j) + beta l, the running max m and the denominator l = sum_j P'_j / r_j are
// written as this split's partial result.
//
// The queries are absorbed before this kernel (q^ = W_UK^T q^C, with gamma
// folded in); W_UV is applied after the split merge.  Everything the kernel
// waits on has a time limit: on expiry it records EG_MLA_ERR_TIMEOUT, drains
// its own copies and MMAs, frees TMEM and exits.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdint>

#include "egmla_common.cuh"
#include "egmla_kernels.h"
#include "egmla_ptx.cuh"

namespace egmla {

namespace {

constexpr int kHeads = 16;
constexpr int kRope = 64;
constexpr int kThreads = 384;
constexpr int kSoftWarps = 2;    // warps 0 and 1: TMEM lane quadrants 0 and 1 hold heads 0-7 and 8-15
constexpr int kMmaWarp = 2;
constexpr int kTmaWarp = 3;
constexpr int kGateWarp0 = 4;
constexpr int kGateWarps = 8;
constexpr uint32_t kSmemLimit = 232448;
// sequences per unit of the fused combine
constexpr uint32_t kFusedMaxG = 16;
// a head's reference max moves only when a tile exceeds it by 2^8
constexpr float kLazyLog2 = 8.f;

template <int D_C, bool GATE>
struct Cfg {
  static constexpr int NCH = D_C / 64;                  // 64-feature swizzle-atom columns
  static constexpr uint32_t PCHUNK = kPage * 128;       // one atom column of a page: 8 KB
  static constexpr uint32_t KR_OFF = NCH * PCHUNK;
  static constexpr uint32_t SLOT = KR_OFF + PCHUNK;     // latent + RoPE key of one page
  static constexpr uint32_t QB_LAT = qprep_lat_bytes(D_C);
  static constexpr uint32_t QB_ROPE = qprep_rope_bytes(kRope);
  static constexpr uint32_t QPREP = qprep_bytes_tc(D_C, kRope);
  // two query blocks (the next sequence's loads while this one is in use)
  static constexpr uint32_t QBUF = (QPREP + 127) / 128 * 128;
  // P' [16 heads x 64 tokens] in the layout of the query block (qop_offset)
  static constexpr uint32_t PBUF = kPage / 8 * kQGroupBytes;
  static constexpr uint32_t STAT_BYTES = 3 * kPage * 4;   // per slot: mu[64], r[64], 1/r[64]
  static constexpr uint32_t MISC = 1024;
  // LayerNorm gamma and beta of the segment read-out, one copy per softmax warp
  static constexpr uint32_t GB_BYTES = 2 * D_C * 4;
  static constexpr int NS_FIT =
      (int)((kSmemLimit - 1024 - 2 * QBUF - 2 * PBUF - 2 * GB_BYTES - MISC) / (SLOT + STAT_BYTES));
  static constexpr int NS = NS_FIT > 6 ? 6 : NS_FIT;
  static constexpr uint32_t OFF_QBUF = NS * SLOT;
  static constexpr uint32_t OFF_PBUF = OFF_QBUF + 2 * QBUF;
  static constexpr uint32_t OFF_STAT = OFF_PBUF + 2 * PBUF;
  static constexpr uint32_t OFF_GB = OFF_STAT + NS * STAT_BYTES;
  static constexpr uint32_t OFF_MISC = OFF_GB + 2 * GB_BYTES;
  static constexpr uint32_t SMEM = OFF_MISC + MISC + 1024;
  // TMEM columns: two score buffers of (latent 64 + RoPE 64) token columns, then
  // the latent output (d_c columns), rows = heads
  static constexpr uint32_t S_COLS = 128;
  static constexpr uint32_t COL_S = 0, COL_O = 2 * S_COLS;
  static constexpr uint32_t TMEM_COLS = 512;
  static constexpr uint32_t PAGE_TX = SLOT;
  static_assert(NS >= 2, "the ring needs two page slots");
  static_assert(SMEM <= kSmemLimit, "shared memory");
  static_assert(D_C == 192 || D_C == 256, "latent widths of this kernel");
  static_assert(COL_O + D_C <= TMEM_COLS, "tensor memory");
  // The M = 64 MMAs read 64 operand rows (8 row groups 128 B apart in each of
  // the two 512-byte K groups of a step), 16 of which are heads: a step reads
  // up to 1536 bytes from its start (the other rows land in TMEM lanes nobody
  // reads).  Every such read stays inside the allocation:
  static constexpr uint32_t STEP_SPAN = kQGroupBytes + 8 * 128;
  static_assert(OFF_QBUF + QBUF + QB_LAT + (kRope / 16 - 1) * 2 * kQGroupBytes + STEP_SPAN <= OFF_MISC,
                "query over-read");
  static_assert(OFF_PBUF + PBUF + (kPage / 16 - 1) * 2 * kQGroupBytes + STEP_SPAN <= OFF_MISC + MISC,
                "weight over-read");
  // fused combine: W_UV,h (at most 256 rows) and up to kFusedMaxG merged
  // latent rows reuse the page-slot area
  static_assert(256u * D_C * 2 + kFusedMaxG * D_C * 4 + 128 <= OFF_QBUF, "fused combine area");
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
  // optional event trace (eg_mla_debug_set_trace): per traced CTA and role a
  // run of (tag, clock64) pairs; tag = event << 24 | tile
  unsigned long long* trace;
  int trace_ctas, trace_cap;
  // fused split combine (cooperative launch only): W_UV, output, grid counter,
  // and the (head, group of cmb_g sequences) units
  const __nv_bfloat16* w_uv;
  __nv_bfloat16* out;
  uint32_t* seq_done;   // [0] CTAs done, [1 + b] split partials of sequence b stored
  int d_v, cmb_groups, cmb_g;
  int fuse;
};

// Trace recorder of one role of one CTA.  Only the trace instantiation of the
// kernel records (ON); in the others every call compiles to nothing, since even
// untaken trace stores in the loops cost registers and instruction-cache room.
template <bool ON>
struct TracerT {
  unsigned long long* base;
  int n, cap;
  __device__ void init(const TcParams& p, int role) {
    base = nullptr;
    n = 0;
    cap = p.trace_cap;
    if (ON && p.trace != nullptr && static_cast<int>(blockIdx.x) < p.trace_ctas)
      base = p.trace + (static_cast<size_t>(blockIdx.x) * kTraceRoles + role) * p.trace_cap * 2;
  }
  __device__ __forceinline__ void mark(int event, int tile) {
    if (ON && base != nullptr && n < cap) {
      base[2 * n] = (static_cast<unsigned long long>(event) << 56) |
                    (static_cast<unsigned long long>(tile & 0xffffff) << 32) |
                    static_cast<uint32_t>(globaltimer());
      base[2 * n + 1] = clock64();
      ++n;
    }
  }
};

// Kernel phase `event` of this CTA into entry `event` of trace role 4 (thread 0;
// stateless, so that nothing stays live across the kernel for it).
template <bool ON>
__device__ __forceinline__ void phase_mark(const TcParams& p, int event) {
  if (ON && p.trace != nullptr && threadIdx.x == 0 && static_cast<int>(blockIdx.x) < p.trace_ctas && event < p.trace_cap) {
    unsigned long long* e = p.trace + ((static_cast<size_t>(blockIdx.x) * kTraceRoles + 4) * p.trace_cap + event) * 2;
    e[0] = (static_cast<unsigned long long>(event) << 56) | static_cast<uint32_t>(globaltimer());
    e[1] = clock64();
  }
}

// shared-memory barrier block (inside MISC)
struct Bars {
  uint64_t full[6], empty[6], zready[6];
  uint64_t qfull[2], qempty[2];
  uint64_t s_ready[2], pfree[2];
  // weights of tile j ready: sp_done[j & 1] (the two softmax warps may be one
  // tile apart, never two: tile j + 2's scores follow tile j's output MMA)
  uint64_t sp_done[2];
  uint64_t sfree[2];           // the softmax warps have read score buffer b
  uint64_t drain_s, drain_o;   // all MMAs of the score / output issuer done
  uint64_t wbar;               // W_UV rows of the fused combine landed
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

// Page of tile t through a 32-entry window of the block table held one entry per
// lane (whole warp; the window moves when the tile leaves it).
struct PageWindow {
  int b = -1, base = 0, reg = -1;
  __device__ __forceinline__ int page(const TcParams& p, const Tile& t, int lane) {
    if (t.b != b || t.lp >= base + 32) {
      b = t.b;
      base = t.lp;
      const int lp = t.lp + lane;
      reg = lp < p.max_pages ? __ldg(p.block_table + static_cast<size_t>(t.b) * p.max_pages + lp) : -1;
    }
    return __shfl_sync(0xffffffffu, reg, t.lp - base);
  }
};

// mbarrier wait taken by a whole warp: the warp first reconverges (a lane
// still on a divergent path would otherwise only resume after the others'
// suspended wait), every lane polls, then the warp agrees, so that a timeout
// never splits the warp before a .sync.aligned instruction
__device__ __forceinline__ bool warp_wait(uint32_t bar, uint32_t parity, volatile int* abort_flag) {
  __syncwarp();
  const bool ok = mbar_wait(bar, parity, abort_flag);
  return __all_sync(0xffffffffu, ok);
}

// one arrival per warp: the warp barrier orders every lane's earlier writes
// before lane 0's release arrival
__device__ __forceinline__ void warp_arrive(uint32_t bar) {
  __syncwarp();
  if ((threadIdx.x & 31) == 0) mbar_arrive(bar);
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

// 2^x with the hardware approximation (max 2 ulp; the weights are rounded to
// bf16 right after, and -inf gives 0)
__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// ---------------------------------------------------------------- fused split combine
// Eight bf16 of a 16-byte piece as floats.
__device__ __forceinline__ void bf16x8_to_float(const uint4& raw, float (&w)[8]) {
  const __nv_bfloat162* e = reinterpret_cast<const __nv_bfloat162*>(&raw);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const float2 f = __bfloat1622float2(e[i]);
    w[2 * i] = f.x;
    w[2 * i + 1] = f.y;
  }
}

// Sums of eight rows whose parts are spread over the warp (v[r] = this lane's
// part of row r): a transposing butterfly halves the rows a lane carries at
// each of the xor-16, -8 and -4 exchanges, then two plain steps finish; lane
// 4r + q (q < 4) ends with the sum of row r.
__device__ __forceinline__ float reduce8_rows(const float (&v)[8], int lane) {
  const bool b4 = (lane & 16) != 0, b3 = (lane & 8) != 0, b2 = (lane & 4) != 0;
  float a[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const float send = b4 ? v[i] : v[i + 4];
    const float keep = b4 ? v[i + 4] : v[i];
    a[i] = keep + __shfl_xor_sync(0xffffffffu, send, 16);
  }
  float c[2];
#pragma unroll
  for (int i = 0; i < 2; ++i) {
    const float send = b3 ? a[i] : a[i + 2];
    const float keep = b3 ? a[i + 2] : a[i];
    c[i] = keep + __shfl_xor_sync(0xffffffffu, send, 8);
  }
  const float send = b2 ? c[0] : c[1];
  float s = (b2 ? c[1] : c[0]) + __shfl_xor_sync(0xffffffffu, send, 4);
  s += __shfl_xor_sync(0xffffffffu, s, 2);
  s += __shfl_xor_sync(0xffffffffu, s, 1);
  return s;
}

// Split-KV combine inside the decode kernel (cooperative launch: every CTA is
// resident, so a wait on other CTAs cannot starve).  A CTA merges its units
// (head h, group of cmb_g sequences) once their split partials are stored:
// with one sequence per unit (small batches) as soon as the softmax warps of
// the splits that covered that sequence have counted their halves on its
// counter, otherwise after every CTA has arrived on a grid counter (both
// counters zeroed by the prologue kernel of the same call).  For each sequence
// b, over the splits s that covered it,
//   o = sum_s 2^(m_s - M) O_s / sum_s 2^(m_s - M) l_s,  M = max_s m_s,
//   u_{b,h} = W_UV,h o
// (a sequence of length 0 gets u = 0).  W_UV,h is bulk-copied into the free
// page-slot area while the CTA waits for the others.  Merge: a warp per
// (sequence, 32 features), lane k loading (m, l) of slot k0 + k and every lane
// O of 32 slots at once (online rescaling across groups of 32).  u: a warp per
// group of eight output rows (see below).
template <int D_C>
__device__ void fused_combine(const TcParams& p, uint8_t* smem, Bars& bars) {
  constexpr int kWarps = kThreads / 32;
  constexpr int NFB = D_C / 32;      // 32-feature blocks of a row
  constexpr int LANES = D_C / 8;     // lanes holding 8 features each
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int G = p.cmb_g, units = kHeads * p.cmb_groups;
  const uint32_t wbytes = static_cast<uint32_t>(p.d_v) * D_C * 2;
  uint8_t* wsm = smem;                                                    // [d_v][D_C] bf16
  float* olat = reinterpret_cast<float*>(smem + ((wbytes + 127u) & ~127u));   // [G][D_C]
  const uint32_t wbar = smem_u32(&bars.wbar);
  volatile int* abort_flag = &bars.abort;
  auto issue_w = [&](int h) {
    if (tid == 0) {
      fence_proxy_async_smem();   // the slot area was last used through the generic proxy too
      mbar_arrive_expect_tx(wbar, wbytes);
      bulk_load_hint(smem_u32(wsm), p.w_uv + static_cast<size_t>(h) * p.d_v * D_C, wbytes, wbar,
                     policy_evict_last());
    }
  };
  int u = blockIdx.x;
  if (u < units) issue_w(u % kHeads);
  const int total = p.cu[p.batch];
  const int chunk = split_chunk(total, gridDim.x);
  // splits that covered sequence b
  auto splits_of = [&](int b) -> int {
    const int q0 = p.cu[b] + kSegCost, q1 = p.cu[b + 1];   // units of the sequence's pages
    return q1 > q0 ? (q1 - 1) / chunk - q0 / chunk + 1 : 0;
  };
  if (G > 1 && tid == 0) {
    // units of several sequences wait for the whole grid: this CTA's partials
    // are stored (the kernel-end barrier ordered the other threads' stores
    // before this thread): release them, then wait for all
    __threadfence();
    atomicAdd(p.seq_done, 1u);
    const uint64_t t0 = globaltimer();
    while (ld_acquire_gpu(p.seq_done) < gridDim.x) {
      if (globaltimer() - t0 > kWaitLimitNs) {
        report_status(p.status, kStatusTimeout);
        *abort_flag = 1;
        break;
      }
      __nanosleep(32);
    }
  }
  int phase = 0;
  for (; u < units; u += gridDim.x) {
    const int h = u % kHeads, grp = u / kHeads;
    const int b0 = grp * G, nb = min(G, p.batch - b0);
    if (G == 1 && tid == 0 && !*abort_flag) {
      // a unit of one sequence: both halves of every split partial of it stored
      const uint32_t want = 2u * static_cast<uint32_t>(splits_of(b0));
      const uint64_t t0 = globaltimer();
      while (ld_acquire_gpu(p.seq_done + 1 + b0) < want) {
        if (*abort_flag) break;
        if (globaltimer() - t0 > kWaitLimitNs) {
          report_status(p.status, kStatusTimeout);
          *abort_flag = 1;
          break;
        }
        __nanosleep(32);
      }
    }
    __syncthreads();
    if (!*abort_flag) {
      for (int w = warp; w < nb * NFB; w += kWarps) {
        const int j = w / NFB, f = (w % NFB) * 32 + lane, b = b0 + j;
        const int q0 = p.cu[b] + kSegCost, q1 = p.cu[b + 1];   // units of the sequence's pages
        const int c0 = q0 / chunk;
        const int n = q1 > q0 ? (q1 - 1) / chunk - c0 + 1 : 0;
        const float* po = p.part_o + (static_cast<size_t>(c0 + b) * kHeads + h) * D_C + f;
        const float* pm = p.part_ml + (static_cast<size_t>(c0 + b) * kHeads + h) * 2;
        float M = -INFINITY, L = 0.f, acc = 0.f;
        for (int k0 = 0; k0 < n; k0 += 32) {
          const int kn = min(32, n - k0);
          float2 ml = make_float2(-INFINITY, 0.f);
          if (lane < kn) ml = __ldcg(reinterpret_cast<const float2*>(pm + static_cast<size_t>(k0 + lane) * kHeads * 2));
          float ov[32];
#pragma unroll
          for (int kk = 0; kk < 32; ++kk)
            ov[kk] = kk < kn ? __ldcg(po + static_cast<size_t>(k0 + kk) * kHeads * D_C) : 0.f;
          float mc = ml.x;
#pragma unroll
          for (int o = 16; o > 0; o >>= 1) mc = fmaxf(mc, __shfl_xor_sync(0xffffffffu, mc, o));
          const float Mn = fmaxf(M, mc);
          const float sc = exp2f(M - Mn);   // 0 on the first group (M = -inf)
          const float wk = lane < kn ? exp2f(ml.x - Mn) : 0.f;
          float lw = wk * ml.y;
#pragma unroll
          for (int o = 16; o > 0; o >>= 1) lw += __shfl_xor_sync(0xffffffffu, lw, o);
          L = fmaf(L, sc, lw);
          acc *= sc;
#pragma unroll
          for (int kk = 0; kk < 32; ++kk) acc = fmaf(__shfl_sync(0xffffffffu, wk, kk), ov[kk], acc);
          M = Mn;
        }
        olat[j * D_C + f] = n > 0 ? acc / L : 0.f;
      }
    }
    // the W_UV,h rows have landed: thread 0 waits on its own flag, so that the
    // copy is waited for even after an abort (no copy may outlive the CTA)
    if (tid == 0) {
      volatile int own = 0;
      if (!mbar_wait(wbar, phase, &own)) {
        report_status(p.status, kStatusTimeout);
        *abort_flag = 1;
      }
    }
    phase ^= 1;
    __syncthreads();
    if (*abort_flag) return;
    // u = W_UV,h o: a warp per group of 8 output rows (loaded once, lane l
    // holding features 8l .. 8l + 7 of each), then for each sequence the eight
    // row sums, reduced across the lanes by a transposing butterfly (9
    // shuffles) after which lane 4r holds row r
    const int nvg = (p.d_v + 7) / 8;
    for (int g = warp; g < nvg; g += kWarps) {
      uint4 wraw[8];
#pragma unroll
      for (int r = 0; r < 8; ++r) {
        const int v = 8 * g + r;
        wraw[r] = make_uint4(0, 0, 0, 0);
        if (lane < LANES && v < p.d_v)
          wraw[r] = *reinterpret_cast<const uint4*>(wsm + (static_cast<size_t>(v) * D_C + 8 * lane) * 2);
      }
      for (int j = 0; j < nb; ++j) {
        float o8[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
        if (lane < LANES) {
          const float4 x0 = *reinterpret_cast<const float4*>(olat + j * D_C + 8 * lane);
          const float4 x1 = *reinterpret_cast<const float4*>(olat + j * D_C + 8 * lane + 4);
          o8[0] = x0.x; o8[1] = x0.y; o8[2] = x0.z; o8[3] = x0.w;
          o8[4] = x1.x; o8[5] = x1.y; o8[6] = x1.z; o8[7] = x1.w;
        }
        float part[8];
#pragma unroll
        for (int r = 0; r < 8; ++r) {
          float wv[8];
          bf16x8_to_float(wraw[r], wv);
          part[r] = 0.f;
#pragma unroll
          for (int e = 0; e < 8; ++e) part[r] = fmaf(wv[e], o8[e], part[r]);
        }
        const float sum = reduce8_rows(part, lane);
        const int v = 8 * g + (lane >> 2);
        if ((lane & 3) == 0 && v < p.d_v)
          p.out[(static_cast<size_t>(b0 + j) * kHeads + h) * p.d_v + v] = __float2bfloat16_rn(sum);
      }
    }
    __syncthreads();   // W and olat are free for the next unit
    if (u + static_cast<int>(gridDim.x) < units) issue_w((u + gridDim.x) % kHeads);
  }
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  __nv_bfloat162 z = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&z);
}

// GM: gate mode (0 none, 1 LN(c (*) g), 2 c (*) g, 3 LN(c + g): eg_mla_gate_mode)
// DBG: 0 the decode, 1 the cache-read dump (raw pages and gate rows, no
// attention), 2 the decode with the pipeline trace
template <int D_C, int GM, int DBG>
__global__ void __launch_bounds__(kThreads, 1)
    decode_tc_kernel(const __grid_constant__ CUtensorMap cmap, const __grid_constant__ CUtensorMap krmap,
                     const TcParams p) {
  constexpr bool DUMP = DBG == 1;
  using Tracer = TracerT<DBG == 2>;
  constexpr bool GATE = GM != 0;
  constexpr bool GATE_ADD = GM == 3;             // ablation: c + g
  constexpr bool GATE_LN = GM == 1 || GM == 3;   // LayerNorm after the gate
  using C = Cfg<D_C, GATE>;
  extern __shared__ uint8_t smem_raw[];
  // 1024-byte aligned base (128-byte swizzle atoms); derived by an offset from the
  // __shared__ array so that every access through it stays a shared-memory access
  uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  const uint32_t sbase = smem_u32(smem);
  Bars& bars = *reinterpret_cast<Bars*>(smem + C::OFF_MISC);
  volatile int* abort_flag = &bars.abort;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  phase_mark<DBG == 2>(p, 0);

  if (threadIdx.x == 0) {
    for (int s = 0; s < C::NS; ++s) {
      mbar_init(smem_u32(&bars.full[s]), 1);
      mbar_init(smem_u32(&bars.empty[s]), DUMP ? kGateWarps : 1);
      mbar_init(smem_u32(&bars.zready[s]), kGateWarps);
    }
    for (int s = 0; s < 2; ++s) {
      mbar_init(smem_u32(&bars.qfull[s]), 1);
      mbar_init(smem_u32(&bars.qempty[s]), 1 + kSoftWarps);
      // the MMA commit plus a release arrival of the MMA warp after it saw the
      // gate's zready (so that the statistics are visible to the softmax warps)
      mbar_init(smem_u32(&bars.s_ready[s]), 2);
      mbar_init(smem_u32(&bars.pfree[s]), 1);
    }
    mbar_init(smem_u32(&bars.sp_done[0]), kSoftWarps);
    mbar_init(smem_u32(&bars.sp_done[1]), kSoftWarps);
    mbar_init(smem_u32(&bars.sfree[0]), kSoftWarps);
    mbar_init(smem_u32(&bars.sfree[1]), kSoftWarps);
    mbar_init(smem_u32(&bars.drain_s), 1);
    mbar_init(smem_u32(&bars.drain_o), 1);
    mbar_init(smem_u32(&bars.wbar), 1);
    bars.abort = 0;
    fence_mbar_init();
  }
  if (warp == kMmaWarp) {
    tmem_alloc(smem_u32(&bars.tmem_base), C::TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  phase_mark<DBG == 2>(p, 1);
  const uint32_t tmem = bars.tmem_base;

  constexpr uint32_t KSTEP = 2 * kQGroupBytes;   // bytes of 16 columns of an A operand
  if (warp == kTmaWarp) {
    // ---------------------------------------------------------------- TMA producer + output MMAs
    // The whole warp walks the tiles; lane 0 waits and issues the copies.
    // Before a page slot is reused the output MMA of the tile that held it is
    // issued here (it is what frees the slot), as soon as that tile's weights
    // are ready; the remaining ones after the last copy.
    if (lane == 0) {
      prefetch_tensormap(&cmap);
      prefetch_tensormap(&krmap);
    }
    const uint64_t pol_stream = policy_evict_first();
    constexpr uint32_t IDESC_PV = idesc_bf16(64, D_C, 0, 1);
    // A operand P' in 8x8 core matrices (K groups 512 B apart, row groups
    // 128 B); B operand: the page slot read MN-major (features along N, tokens
    // along K)
    const uint64_t pdesc0 = smem_desc(sbase + C::OFF_PBUF, kQGroupBytes, 128, kSwizzleNone);
    const uint64_t zdesc_mn = smem_desc(sbase, C::PCHUNK, 1024, kSwizzle128B);
    Walker w, wo;
    w.start(p.cu, p.seq_lens, p.batch);
    wo.start(p.cu, p.seq_lens, p.batch);
    PageWindow pw;
    Tile t, to;
    int it = 0, io = 0;
    int last_it[6] = {-1, -1, -1, -1, -1, -1};
    bool issued_o = false;
    Tracer tr;
    tr.init(p, 0);
    if (lane != 0) tr.base = nullptr;
    bool ok_loop = true;
    // output MMA of the next tile in order (O += P' Z); false on a timeout
    auto output = [&]() -> bool {
      if (!wo.next(to)) return true;
      if (!warp_wait(smem_u32(&bars.sp_done[io & 1]), (io >> 1) & 1, abort_flag)) return false;
      tc_fence_after();
      if (elect_one()) {
        const int slot = io % C::NS;
        const uint64_t zb = zdesc_mn + ((slot * C::SLOT) >> 4);
        const uint64_t pa = pdesc0 + (((io & 1) * C::PBUF) >> 4);
        if (to.first) {
#pragma unroll
          for (int ks = 0; ks < kPage / 16; ++ks)
            mma_bf16_ss(tmem + C::COL_O, pa + ((ks * KSTEP) >> 4), zb + ((ks * 2048) >> 4), IDESC_PV, ks > 0);
        } else {
#pragma unroll
          for (int ks = 0; ks < kPage / 16; ++ks)
            mma_bf16_ss(tmem + C::COL_O, pa + ((ks * KSTEP) >> 4), zb + ((ks * 2048) >> 4), IDESC_PV, 1);
        }
        mma_commit(smem_u32(&bars.empty[slot]));
        mma_commit(smem_u32(&bars.pfree[io & 1]));
      }
      __syncwarp();
      issued_o = true;
      ++io;
      return true;
    };
    while (ok_loop && w.next(t)) {
      const int pg = pw.page(p, t, lane);
      const int slot = it % C::NS;
      // the tile that held this slot must have had its output MMA issued
      if (!DUMP && it >= C::NS && !output()) break;
      if (lane == 0) {
        tr.mark(0, it);
        if (ok_loop && !mbar_wait(smem_u32(&bars.empty[slot]), ((it / C::NS) & 1) ^ 1, abort_flag)) ok_loop = false;
        if (ok_loop) {
          tr.mark(1, it);
          const bool ok = pg >= 0 && pg < p.num_pages;
          if (!ok) report_status(p.status, kStatusOutOfRange);
          const uint32_t fb = smem_u32(&bars.full[slot]);
          mbar_arrive_expect_tx(fb, ok ? C::PAGE_TX : 0u);
          tr.mark(3, it);
          if (ok) {
            const uint32_t dst = sbase + slot * C::SLOT;
            const int y = pg * kPage;
            tma_load_3d(dst, &cmap, 0, y, 0, fb, pol_stream);
            tma_load_2d(dst + C::KR_OFF, &krmap, 0, y, fb, pol_stream);
          }
          tr.mark(2, it);
          last_it[slot] = it;
        }
      }
      ok_loop = __shfl_sync(0xffffffffu, ok_loop, 0);
      ++it;
    }
    // the output MMAs of the last tiles
    if (!DUMP && ok_loop)
      while (io < it)
        if (!output()) break;
    if (!DUMP && issued_o) {
      // every output MMA must finish before TMEM is released
      if (elect_one()) mma_commit(smem_u32(&bars.drain_o));
      __syncwarp();
      mbar_wait(smem_u32(&bars.drain_o), 0, abort_flag);
    }
    if (lane == 0) {
      // drain: every copy this thread issued must land before the CTA exits
      for (int s = 0; s < C::NS; ++s)
        if (last_it[s] >= 0) mbar_wait(smem_u32(&bars.full[s]), (last_it[s] / C::NS) & 1, abort_flag);
    }
    __syncwarp();
  } else if (warp == kMmaWarp) {
    // ---------------------------------------------------------------- score MMAs
    // Converged warp; one elected lane issues.  Tile j's scores go out as soon
    // as its gated page is ready and the softmax warps have read the score
    // buffer two tiles back.  Loops are unrolled with compile-time accumulate
    // flags.  This warp also loads the sequences' query blocks (double-
    // buffered): the next segment's block as soon as its buffer is free (a
    // non-blocking test after every tile), blocking only at a segment start.
    if (!DUMP) {
      constexpr uint32_t IDESC_S = idesc_bf16(64, kPage, 0, 0);
      Walker w;
      w.start(p.cu, p.seq_lens, p.batch);
      int seg = -1;
      Tracer tr;
      tr.init(p, 1);
      if (lane != 0) tr.base = nullptr;
      // A operand: the query block in 8x8 core matrices, K groups 512 B apart,
      // row groups 128 B apart (heads 0-7 -> rows 0-7, heads 8-15 -> rows
      // 16-23).  B operand: the page slot, 128-byte swizzled, read K-major
      // (tokens x features).
      const uint64_t qdesc0 = smem_desc(sbase + C::OFF_QBUF, kQGroupBytes, 128, kSwizzleNone);
      const uint64_t zdesc_k = smem_desc(sbase, 16, 1024, kSwizzle128B);
      // segment starts ahead of the tile loop: wq sits on the first tile of
      // segment qn, the next one whose query block is to be loaded
      Walker wq;
      wq.start(p.cu, p.seq_lens, p.batch);
      Tile tq;
      bool q_more = wq.next(tq);
      int qn = 0;
      int last_q[2] = {-1, -1};
      // 1: issued, 0: buffer still in use (non-blocking call), -1: timed out
      auto load_query = [&](bool block) -> int {
        const int qb = qn & 1;
        if (qn >= 2) {
          const uint32_t qe = smem_u32(&bars.qempty[qb]);
          const uint32_t par = ((qn >> 1) & 1) ^ 1;
          if (block) {
            if (!warp_wait(qe, par, abort_flag)) return -1;
          } else if (!__all_sync(0xffffffffu, mbar_test_now(qe, par))) {
            return 0;
          }
        }
        if (lane == 0) {
          mbar_arrive_expect_tx(smem_u32(&bars.qfull[qb]), C::QPREP);
          bulk_load(sbase + C::OFF_QBUF + qb * C::QBUF, p.qprep + static_cast<size_t>(tq.b) * C::QPREP, C::QPREP,
                    smem_u32(&bars.qfull[qb]));
        }
        __syncwarp();
        last_q[qb] = qn;
        ++qn;
        do {
          q_more = wq.next(tq);
        } while (q_more && !tq.first);
        return 1;
      };
      Tile t;
      int j = 0;
      bool issued = false;
      bool ok_q = true;
      while (w.next(t)) {
        if (t.first) {
          ++seg;
          while (qn <= seg && (ok_q = load_query(true) > 0)) {
          }
          if (!ok_q) break;
          if (!warp_wait(smem_u32(&bars.qfull[seg & 1]), (seg >> 1) & 1, abort_flag)) break;
        }
        const int slot = j % C::NS;
        tr.mark(0, j);
        if (!warp_wait(smem_u32(&bars.zready[slot]), (j / C::NS) & 1, abort_flag)) break;
        if (j >= 2 && !warp_wait(smem_u32(&bars.sfree[j & 1]), ((j >> 1) & 1) ^ 1, abort_flag)) break;
        tr.mark(1, j);
        if (lane == 0) mbar_arrive(smem_u32(&bars.s_ready[j & 1]));
        tc_fence_after();
        if (elect_one()) {
          const uint64_t zb = zdesc_k + ((slot * C::SLOT) >> 4);
          const uint64_t qa = qdesc0 + (((seg & 1) * C::QBUF) >> 4);
          const uint32_t ds = tmem + C::COL_S + (j & 1) * C::S_COLS;
#pragma unroll
          for (int kk = 0; kk < D_C / 16; ++kk)
            mma_bf16_ss(ds, qa + ((kk * KSTEP) >> 4), zb + (((kk >> 2) * C::PCHUNK + (kk & 3) * 32) >> 4), IDESC_S,
                        kk > 0);
#pragma unroll
          for (int kk = 0; kk < kRope / 16; ++kk)
            mma_bf16_ss(ds + kPage, qa + ((C::QB_LAT + kk * KSTEP) >> 4), zb + ((C::KR_OFF + kk * 32) >> 4), IDESC_S,
                        kk > 0);
          mma_commit(smem_u32(&bars.s_ready[j & 1]));
          if (t.last) mma_commit(smem_u32(&bars.qempty[seg & 1]));
        }
        __syncwarp();
        tr.mark(2, j);
        issued = true;
        ++j;
        if (q_more && qn == seg + 1 && load_query(false) < 0) break;
      }
      if (lane == 0) {
        // drain: the query-block copies this warp issued must land before the CTA exits
        for (int b = 0; b < 2; ++b)
          if (last_q[b] >= 0) mbar_wait(smem_u32(&bars.qfull[b]), (last_q[b] >> 1) & 1, abort_flag);
      }
      __syncwarp();
      if (issued) {
        // every score MMA must finish before TMEM is released
        if (elect_one()) mma_commit(smem_u32(&bars.drain_s));
        __syncwarp();
        mbar_wait(smem_u32(&bars.drain_s), 0, abort_flag);
      }
    }
    __syncwarp();
  } else if (warp >= kGateWarp0) {
    // ---------------------------------------------------------------- gate: z = c (*) g, LN statistics
    // Quarter-warp k = 4 (warp - 4) + lane / 8 owns token rows 2k (lanes 0-3)
    // and 2k + 1 (lanes 4-7); lane p = lane % 4 of a row takes the 16-byte
    // units 2p and 2p + 1 of every 64-feature column.  The gate-row load of a
    // column is then one 32-byte load per lane and a whole 128-byte line per
    // row (the load/store data path pays per instruction and per line, so
    // fewer, wider loads are cheaper), and a quarter-warp's shared-memory
    // accesses to the swizzled page still hit eight distinct bank groups (the
    // two rows differ in swizzle parity).  The gate rows come from L2 (the
    // table stays there under an evict-last hint while the cache stream is
    // evict-first): each tile issues the id loads of the tile two ahead and the
    // gate-row loads of the next tile, so neither latency sits on the loop.
    const int gw = warp - kGateWarp0;
    const int pp = lane & 3;
    const int row = 2 * (gw * 4 + (lane >> 3)) + ((lane >> 2) & 1);
    const uint64_t pol_keep = policy_evict_last();
    constexpr bool gate_ln = GATE_LN;
    Walker w;
    w.start(p.cu, p.seq_lens, p.batch);
    PageWindow pw;
    // id of this thread's row of a tile (0 past the end of the page or for a
    // bad page, which the producer reports)
    auto load_id = [&](const Tile& tt) -> int {
      const int pg = pw.page(p, tt, lane);
      const int n = (pg >= 0 && pg < p.num_pages) ? tt.ntok : 0;
      return row < n ? __ldg(p.id_pool + static_cast<size_t>(pg) * kPage + row) : 0;
    };
    auto load_g = [&](int& id, uint4 (&gv)[C::NCH][2]) {
      if ((unsigned)id >= (unsigned)p.vocab) {
        report_status(p.status, kStatusOutOfRange);
        id = 0;
      }
      const __nv_bfloat16* src = p.gate_table + static_cast<size_t>(id) * D_C + pp * 16;
#pragma unroll
      for (int fc = 0; fc < C::NCH; ++fc) ldg_32_na_hint(src + fc * 64, pol_keep, gv[fc][0], gv[fc][1]);
    };
    // shared-memory offset of unit (2 pp + h) of column fc of this thread's row
    auto unit_off = [&](int fc, int h) -> uint32_t {
      return fc * C::PCHUNK + row * 128 + (((2 * pp + h) ^ (row & 7)) << 4);
    };
    Tracer tr;
    tr.init(p, 2);
    if (threadIdx.x != kGateWarp0 * 32) tr.base = nullptr;
    Tile t, t1, t2;
    bool have = w.next(t);
    bool have1 = have && w.next(t1);
    bool have2 = have1 && w.next(t2);
    int id0 = 0, id1 = 0, id2 = 0;   // ids of tiles j, j + 1, j + 2
    uint4 gcur[C::NCH][2], gnext[C::NCH][2];
    if (GATE) {
      if (have) id0 = load_id(t);
      if (have1) id1 = load_id(t1);
      if (have) load_g(id0, gcur);
    }
    int j = 0;
    while (have) {
      const int slot = j % C::NS;
      tr.mark(0, j);
      if (GATE) {
        // prefetch: ids of tile j + 2, gate rows of tile j + 1
        if (have2) id2 = load_id(t2);
        if (have1) load_g(id1, gnext);
      }
      if (!warp_wait(smem_u32(&bars.full[slot]), (j / C::NS) & 1, abort_flag)) break;
      tr.mark(1, j);
      uint8_t* cpage = smem + slot * C::SLOT;
      if (DUMP) {
        if (row < t.ntok) {
          const size_t o = static_cast<size_t>(t.b) * p.dump_len + t.tok0 + row;
          uint4* dc = reinterpret_cast<uint4*>(p.dump_c + o * D_C);
          uint4* dg = reinterpret_cast<uint4*>(p.dump_g + o * D_C);
#pragma unroll
          for (int fc = 0; fc < C::NCH; ++fc) {
#pragma unroll
            for (int h = 0; h < 2; ++h) {
              dc[fc * 8 + 2 * pp + h] = *reinterpret_cast<const uint4*>(cpage + unit_off(fc, h));
              dg[fc * 8 + 2 * pp + h] = gcur[fc][h];
            }
          }
#pragma unroll
          for (int h = 0; h < 2; ++h)
            reinterpret_cast<uint4*>(p.dump_kr + o * kRope)[2 * pp + h] = *reinterpret_cast<const uint4*>(
                cpage + C::KR_OFF + row * 128 + (((2 * pp + h) ^ (row & 7)) << 4));
          if (pp == 0) p.dump_ids[o] = id0;
        }
        warp_arrive(smem_u32(&bars.empty[slot]));
      } else {
        const bool full_page = t.ntok == kPage;   // uniform: no token masking needed
        if (GATE) {
          float* st = reinterpret_cast<float*>(smem + C::OFF_STAT + slot * C::STAT_BYTES);
          // all shared-memory reads of this thread's units first (the in-place
          // stores below would otherwise order every later load behind them)
          uint4 cv[C::NCH][2];
#pragma unroll
          for (int fc = 0; fc < C::NCH; ++fc)
#pragma unroll
            for (int h = 0; h < 2; ++h) cv[fc][h] = *reinterpret_cast<const uint4*>(cpage + unit_off(fc, h));
          tr.mark(5, j);
          const bool valid = row < t.ntok;
          if constexpr (GATE_ADD) {
            // ablation LN(c + g): c + g is exact in fp32; the row is centred by its
            // mean before the bf16 rounding (LN is shift-invariant), so the rounding
            // error is relative to the spread LN keeps, not to the gate's offset
            float2 s1 = make_float2(0.f, 0.f), s2 = make_float2(0.f, 0.f);
#pragma unroll
            for (int fc = 0; fc < C::NCH; ++fc) {
#pragma unroll
              for (int h = 0; h < 2; ++h) {
                const uint32_t* cw = reinterpret_cast<const uint32_t*>(&cv[fc][h]);
                const uint32_t* gw2 = reinterpret_cast<const uint32_t*>(&gcur[fc][h]);
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                  const float2 zf = __fadd2_rn(unpack_bf16x2(cw[k]), unpack_bf16x2(gw2[k]));
                  s1 = __fadd2_rn(s1, zf);
                  s2 = __ffma2_rn(zf, zf, s2);
                }
              }
            }
            float sum1 = s1.x + s1.y, sum2 = s2.x + s2.y;
#pragma unroll
            for (int o = 1; o < 4; o <<= 1) {
              sum1 += __shfl_xor_sync(0xffffffffu, sum1, o);
              sum2 += __shfl_xor_sync(0xffffffffu, sum2, o);
            }
            constexpr float inv_dc = 1.f / D_C;
            const float mu = sum1 * inv_dc;
            const float var = fmaxf(sum2 * inv_dc - mu * mu, 0.f);
            const float r = rsqrtf(var + p.eps);
            const float2 mu2v = make_float2(mu, mu);
#pragma unroll
            for (int fc = 0; fc < C::NCH; ++fc) {
#pragma unroll
              for (int h = 0; h < 2; ++h) {
                const uint32_t* cw = reinterpret_cast<const uint32_t*>(&cv[fc][h]);
                const uint32_t* gw2 = reinterpret_cast<const uint32_t*>(&gcur[fc][h]);
                uint4 z;
                uint32_t* zw = reinterpret_cast<uint32_t*>(&z);
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                  const float2 zf = __fadd2_rn(__fadd2_rn(unpack_bf16x2(cw[k]), unpack_bf16x2(gw2[k])),
                                               make_float2(-mu2v.x, -mu2v.y));
                  zw[k] = pack_bf16x2(zf.x, zf.y);
                }
                if (!full_page && !valid) z = make_uint4(0, 0, 0, 0);
                *reinterpret_cast<uint4*>(cpage + unit_off(fc, h)) = z;
              }
            }
            tr.mark(6, j);
            if (pp == 0) {
              st[row] = 0.f;   // the stored z is centred
              st[kPage + row] = valid ? r : 0.f;
              st[2 * kPage + row] = valid ? 1.f / r : 0.f;
            }
          } else {
            float2 s1 = make_float2(0.f, 0.f), s2 = make_float2(0.f, 0.f);
            float2 a1 = make_float2(0.f, 0.f), a2 = make_float2(0.f, 0.f);
#pragma unroll
            for (int fc = 0; fc < C::NCH; ++fc) {
#pragma unroll
              for (int h = 0; h < 2; ++h) {
                uint4 z;
                z.x = mul_bf16x2(cv[fc][h].x, gcur[fc][h].x);
                z.y = mul_bf16x2(cv[fc][h].y, gcur[fc][h].y);
                z.z = mul_bf16x2(cv[fc][h].z, gcur[fc][h].z);
                z.w = mul_bf16x2(cv[fc][h].w, gcur[fc][h].w);
                if (!full_page && !valid) z = make_uint4(0, 0, 0, 0);
                const float2 f0 = unpack_bf16x2(z.x), f1 = unpack_bf16x2(z.y);
                const float2 f2 = unpack_bf16x2(z.z), f3 = unpack_bf16x2(z.w);
                s1 = __fadd2_rn(s1, f0);
                a1 = __fadd2_rn(a1, f1);
                s1 = __fadd2_rn(s1, f2);
                a1 = __fadd2_rn(a1, f3);
                s2 = __ffma2_rn(f0, f0, s2);
                a2 = __ffma2_rn(f1, f1, a2);
                s2 = __ffma2_rn(f2, f2, s2);
                a2 = __ffma2_rn(f3, f3, a2);
                *reinterpret_cast<uint4*>(cpage + unit_off(fc, h)) = z;
              }
            }
            s1 = __fadd2_rn(s1, a1);
            s2 = __fadd2_rn(s2, a2);
            float sum1 = s1.x + s1.y, sum2 = s2.x + s2.y;
            tr.mark(6, j);
            // row sums over the four lanes of the row (without the LayerNorm
            // ablation's norm: mu = 0, r = 1)
            if (gate_ln) {
#pragma unroll
              for (int o = 1; o < 4; o <<= 1) {
                sum1 += __shfl_xor_sync(0xffffffffu, sum1, o);
                sum2 += __shfl_xor_sync(0xffffffffu, sum2, o);
              }
            }
            if (pp == 0) {
              constexpr float inv_dc = 1.f / D_C;
              const float mu = gate_ln ? sum1 * inv_dc : 0.f;
              const float var = fmaxf(sum2 * inv_dc - mu * mu, 0.f);
              const float r = gate_ln ? rsqrtf(var + p.eps) : 1.f;
              st[row] = valid ? mu : 0.f;
              st[kPage + row] = valid ? r : 0.f;
              st[2 * kPage + row] = valid ? 1.f / r : 0.f;
            }
          }
        } else if (!full_page) {
          if (row >= t.ntok) {
#pragma unroll
            for (int fc = 0; fc < C::NCH; ++fc)
#pragma unroll
              for (int h = 0; h < 2; ++h)
                *reinterpret_cast<uint4*>(cpage + unit_off(fc, h)) = make_uint4(0, 0, 0, 0);
          }
        }
        tr.mark(2, j);
        fence_proxy_async_smem();
        warp_arrive(smem_u32(&bars.zready[slot]));
      }
      tr.mark(3, j);
      ++j;
      t = t1;
      t1 = t2;
      have = have1;
      have1 = have2;
      have2 = have2 && w.next(t2);
      if (GATE) {
        id0 = id1;
        id1 = id2;
#pragma unroll
        for (int fc = 0; fc < C::NCH; ++fc) {
          gcur[fc][0] = gnext[fc][0];
          gcur[fc][1] = gnext[fc][1];
        }
      }
    }
  } else if (warp < kSoftWarps && !DUMP) {
    // ---------------------------------------------------------------- softmax, output read-out
    // Warp hw owns heads 8hw..8hw+7, whose rows of S^T and O sit in TMEM lanes
    // 32hw..32hw+7.  Thread t owns head hd = 8hw + t/4 and, in every 8-token
    // group k of a page, the tokens 8k + 2(t%4) and 8k + 2(t%4) + 1.  The
    // 16-lane TMEM loads also return lanes 32hw+8..32hw+15 (rows no head uses),
    // which are ignored.
    const int hw = warp, hd = 8 * hw + (lane >> 2), qq = lane & 3;
    const uint32_t tq = tmem + (static_cast<uint32_t>(32 * hw) << 16);
    const float scale = p.scale_log2;
    // Online softmax with a lazily updated reference max m_ref per head: the
    // exponentials are taken against m_ref, which only moves (rescaling the TMEM
    // accumulator, l and the mean correction) when a tile's max exceeds it by
    // more than 2^kLazyLog2; otherwise the weights stay below 2^kLazyLog2.
    float m_ref = 0.f, l_acc = 0.f, bmu_acc = 0.f, wq = 0.f, bsc = 0.f;
    // this warp's copy of gamma and beta (identity without a LayerNorm), so that
    // the segment read-out waits on no global load
    float* gb = reinterpret_cast<float*>(smem + C::OFF_GB + hw * C::GB_BYTES);
    if (GATE) {
      for (int f = lane; f < D_C; f += 32) {
        gb[f] = p.gamma ? __ldg(p.gamma + f) : 1.f;
        gb[D_C + f] = p.beta ? __ldg(p.beta + f) : 0.f;
      }
      __syncwarp();
    }
    Walker w;
    w.start(p.cu, p.seq_lens, p.batch);
    Tile t;
    int it = 0, seg = -1;
    Tracer tr;
    tr.init(p, 3);
    if (threadIdx.x != 0) tr.base = nullptr;
    while (w.next(t)) {
      if (t.first) {
        ++seg;
        if (!warp_wait(smem_u32(&bars.qfull[seg & 1]), (seg >> 1) & 1, abort_flag)) break;
        if (GATE) {
          // w_h = sum_f bf16(q^ gamma)_hf and b_h = q^_h . beta from their
          // per-chunk partials after the operands, added in chunk order
          const float* sums = reinterpret_cast<const float*>(smem + C::OFF_QBUF + (seg & 1) * C::QBUF + C::QB_LAT +
                                                             C::QB_ROPE);
          float wsum = 0.f, bsum = 0.f;
#pragma unroll
          for (int c = 0; c < D_C / kSumFeatures; ++c) {
            wsum += sums[c * 32 + hd];
            bsum += sums[c * 32 + 16 + hd];
          }
          wq = wsum;
          bsc = bsum * scale;
        }
        warp_arrive(smem_u32(&bars.qempty[seg & 1]));
        l_acc = 0.f;
        bmu_acc = 0.f;
      }
      const int slot = it % C::NS;
      const int par = it & 1;
      tr.mark(0, it);
      // Scores of this tile; the score warp's release arrival on the same
      // barrier orders the gate's statistics before it.
      if (!warp_wait(smem_u32(&bars.s_ready[par]), (it >> 1) & 1, abort_flag)) break;
      tr.mark(1, it);
      tc_fence_after();
      float sl[32], sr[32];
      tmem_ld_16x256b_x8(tq + C::COL_S + par * C::S_COLS, sl);
      tmem_ld_16x256b_x8(tq + C::COL_S + par * C::S_COLS + kPage, sr);
      const float* st = reinterpret_cast<const float*>(smem + C::OFF_STAT + slot * C::STAT_BYTES);
      float2 mu2[8], r2[8], ri2[8];
      if (GATE) {
#pragma unroll
        for (int k = 0; k < 8; ++k) {
          mu2[k] = *reinterpret_cast<const float2*>(st + 8 * k + 2 * qq);
          r2[k] = *reinterpret_cast<const float2*>(st + kPage + 8 * k + 2 * qq);
          ri2[k] = *reinterpret_cast<const float2*>(st + 2 * kPage + 8 * k + 2 * qq);
        }
      }
      tmem_wait_ld();
      tc_fence_before();
      warp_arrive(smem_u32(&bars.sfree[par]));   // score buffer read: tile it + 2 may overwrite it
      tr.mark(7, it);
      // s[2k + e]: token 8k + 2 qq + e of head hd (log2 units)
      float s[16];
      const bool full_page = t.ntok == kPage;
#pragma unroll
      for (int k = 0; k < 8; ++k) {
#pragma unroll
        for (int e = 0; e < 2; ++e) {
          const float lat = sl[4 * k + e], rope = sr[4 * k + e];
          float v;
          if (GATE) {
            const float mu = e ? mu2[k].y : mu2[k].x;
            const float rs = (e ? r2[k].y : r2[k].x) * scale;
            v = fmaf(rs, fmaf(-mu, wq, lat), fmaf(rope, scale, bsc));
          } else {
            v = (lat + rope) * scale;
          }
          const bool valid = full_page || (8 * k + 2 * qq + e) < t.ntok;
          s[2 * k + e] = valid ? v : -INFINITY;
        }
      }
      tr.mark(8, it);
      // tile max of the head: 16 tokens in-thread (a tree), then its four threads
      float m8[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) m8[i] = fmaxf(s[i], s[i + 8]);
#pragma unroll
      for (int i = 0; i < 4; ++i) m8[i] = fmaxf(m8[i], m8[i + 4]);
      float mx = fmaxf(fmaxf(m8[0], m8[2]), fmaxf(m8[1], m8[3]));
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 2));
      float alpha = 1.f;
      bool rescale = false;
      if (t.first) {
        m_ref = mx;
      } else if (mx > m_ref + kLazyLog2) {
        alpha = ex2_approx(m_ref - mx);
        m_ref = mx;
        rescale = true;
      }
      tr.mark(2, it);
      if (__any_sync(0xffffffffu, rescale)) {
        // The previous tile's output MMA must be complete before O is rescaled.
        // Phase n of pfree[b] completes with output MMA 2n + b; the wait below
        // on every tile keeps each buffer's phase count at most one behind, so
        // the parity wait is exact.
        if (!warp_wait(smem_u32(&bars.pfree[(it - 1) & 1]), ((it - 1) >> 1) & 1, abort_flag)) break;
        tc_fence_after();
#pragma unroll 1
        for (int c = 0; c < D_C / 64; ++c) {
          float o[32];
          tmem_ld_16x256b_x8(tq + C::COL_O + 64 * c, o);
          tmem_wait_ld();
#pragma unroll
          for (int k = 0; k < 8; ++k) {
            o[4 * k] *= alpha;
            o[4 * k + 1] *= alpha;
          }
          tmem_st_16x256b_x8(tq + C::COL_O + 64 * c, o);
        }
        tmem_wait_st();
        l_acc *= alpha;
        bmu_acc *= alpha;
      }
      // the weight buffer of this parity is free once the output MMA two tiles
      // back has read it
      if (!warp_wait(smem_u32(&bars.pfree[par]), ((it >> 1) & 1) ^ 1, abort_flag)) break;
      tr.mark(5, it);
      // The output MMA sees the bf16-rounded weights P'; the denominator and the
      // mean correction use the same rounded values (l = sum P'/r), so the
      // rounding of P' cancels in o = (sum P' z - sum P' mu) / l.
      uint8_t* pbuf = smem + C::OFF_PBUF + par * C::PBUF + qop_offset(hd, 2 * qq);
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        const float r0 = GATE ? r2[k].x : 1.f, r1 = GATE ? r2[k].y : 1.f;
        const float p0 = ex2_approx(s[2 * k] - m_ref) * r0;
        const float p1 = ex2_approx(s[2 * k + 1] - m_ref) * r1;
        const uint32_t pw = pack_bf16x2(p0, p1);
        const float2 pq = unpack_bf16x2(pw);
        if (GATE) {
          l_acc = fmaf(pq.x, ri2[k].x, fmaf(pq.y, ri2[k].y, l_acc));
          bmu_acc = fmaf(pq.x, mu2[k].x, fmaf(pq.y, mu2[k].y, bmu_acc));
        } else {
          l_acc += pq.x + pq.y;
        }
        *reinterpret_cast<uint32_t*>(pbuf + k * kQGroupBytes) = pw;
      }
      tr.mark(6, it);
      fence_proxy_async_smem();
      tc_fence_before();
      warp_arrive(smem_u32(&bars.sp_done[par]));
      tr.mark(3, it);

      if (t.last) {
        // ---- segment end: l and sum_j P'_j mu_j over the four threads of the head
        float lh = l_acc, bh = bmu_acc;
        lh += __shfl_xor_sync(0xffffffffu, lh, 1);
        bh += __shfl_xor_sync(0xffffffffu, bh, 1);
        lh += __shfl_xor_sync(0xffffffffu, lh, 2);
        bh += __shfl_xor_sync(0xffffffffu, bh, 2);
        // the segment's last output MMA (the earlier ones complete before it;
        // exact parity wait as for the rescale), then the accumulated output
        if (!warp_wait(smem_u32(&bars.pfree[par]), (it >> 1) & 1, abort_flag)) break;
        tc_fence_after();
        const int slot_out = blockIdx.x + t.b;
        float* po = p.part_o + (static_cast<size_t>(slot_out) * kHeads + hd) * D_C;
#pragma unroll 1
        for (int c = 0; c < D_C / 64; ++c) {
          float o[32];
          tmem_ld_16x256b_x8(tq + C::COL_O + 64 * c, o);
          tmem_wait_ld();
#pragma unroll
          for (int k = 0; k < 8; ++k) {
            const int f = 64 * c + 8 * k + 2 * qq;
            float2 v = make_float2(o[4 * k], o[4 * k + 1]);
            if (GATE) {
              const float2 gm = *reinterpret_cast<const float2*>(gb + f);
              const float2 bt = *reinterpret_cast<const float2*>(gb + D_C + f);
              v.x = fmaf(gm.x, v.x - bh, bt.x * lh);
              v.y = fmaf(gm.y, v.y - bh, bt.y * lh);
            }
            *reinterpret_cast<float2*>(po + f) = v;
          }
        }
        tc_fence_before();
        if (qq == 0) {
          float* ml = p.part_ml + (static_cast<size_t>(slot_out) * kHeads + hd) * 2;
          ml[0] = m_ref;
          ml[1] = lh;
        }
        if (p.fuse && p.cmb_g == 1) {
          // one sequence per combine unit: release this warp's half of the
          // partial to the wait on its sequence (the warp barrier orders every
          // lane's stores before lane 0's fence)
          __syncwarp();
          if (lane == 0) {
            __threadfence();
            atomicAdd(p.seq_done + 1 + t.b, 1u);
          }
        }

        tr.mark(4, it);
      }
      ++it;
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  phase_mark<DBG == 2>(p, 2);
  if (warp == kMmaWarp) tmem_dealloc(tmem, C::TMEM_COLS);
  if (threadIdx.x == 0 && bars.abort) report_status(p.status, kStatusTimeout);
  if (!DUMP && p.fuse) fused_combine<D_C>(p, smem, bars);
  phase_mark<DBG == 2>(p, 3);
}

// CTAs of `kern` that the current device holds at once (1 per SM here), cached per kernel
template <typename K>
int resident_ctas(K kern, uint32_t smem) {
  static int cached[64] = {0};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 0;
  if (cached[dev] == 0) {
    int per_sm = 0, sms = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, kThreads, smem) != cudaSuccess ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
      return 0;
    cached[dev] = std::max(0, per_sm) * sms;
  }
  return cached[dev];
}

template <int D_C, int GM, int DBG>
cudaError_t launch_one(const DecodeArgs& a, const CUtensorMap* maps, cudaStream_t st, bool* fused) {
  using C = Cfg<D_C, GM != 0>;
  auto kern = decode_tc_kernel<D_C, GM, DBG>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)C::SMEM);
  if (e != cudaSuccess) return e;
  const WorkspaceLayout wl = workspace_layout(a.batch, a.num_splits, kHeads, D_C, kRope, true);
  uint8_t* ws = static_cast<uint8_t*>(a.workspace);
  TcParams p;
  p.id_pool = a.id_pool;
  p.block_table = a.block_table;
  p.seq_lens = a.seq_lens;
  p.gate_table = static_cast<const __nv_bfloat16*>(a.gate_table);
  // gamma and beta belong to the LayerNorm (none in the "remove LayerNorm" ablation)
  p.gamma = a.gate_ln ? a.ln_gamma : nullptr;
  p.beta = a.gate_ln ? a.ln_beta : nullptr;

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
  p.trace = static_cast<unsigned long long*>(a.trace);
  p.trace_ctas = a.trace_ctas;
  p.trace_cap = a.trace_cap;
  // The split combine runs inside this kernel when every CTA of the grid can
  // be resident at once (a cooperative launch guarantees it, or fails).
  p.w_uv = static_cast<const __nv_bfloat16*>(a.w_uv);
  p.out = static_cast<__nv_bfloat16*>(a.out);
  p.seq_done = reinterpret_cast<uint32_t*>(ws + wl.off_done);
  p.d_v = a.d_v;
  int groups = std::max(1, std::min(a.batch, a.num_splits / kHeads));
  const int g = std::min(static_cast<int>(kFusedMaxG), (a.batch + groups - 1) / groups);
  p.cmb_g = g;
  p.cmb_groups = (a.batch + g - 1) / g;
  p.fuse = DBG != 1 && a.batch > 0 && a.num_splits <= resident_ctas(kern, C::SMEM);
  if (fused) *fused = p.fuse != 0;
  if (!p.fuse) {
    kern<<<a.num_splits, kThreads, C::SMEM, st>>>(maps[0], maps[1], p);
    return cudaGetLastError();
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(a.num_splits);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = C::SMEM;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeCooperative;
  attr[0].val.cooperative = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, maps[0], maps[1], p);
}

}  // namespace

bool tc_supported(int d_c, int gate) {
  if (gate) return d_c == 192 || d_c == 256;
  return d_c == 192 || d_c == 256 || d_c == 512;
}

// d_c-dispatch of one gate mode; the trace instantiation exists for the modes
// none and mul_ln (the others run untraced)
template <int GM>
cudaError_t launch_mode(const DecodeArgs& a, const CUtensorMap* maps, cudaStream_t st, bool* fused) {
  if constexpr (GM <= 1) {
    if (a.trace != nullptr) {
      if (a.d_c == 192) return launch_one<192, GM, 2>(a, maps, st, fused);
      if (a.d_c == 256) return launch_one<256, GM, 2>(a, maps, st, fused);
      return cudaErrorInvalidValue;
    }
  }
  if (a.d_c == 192) return launch_one<192, GM, 0>(a, maps, st, fused);
  if (a.d_c == 256) return launch_one<256, GM, 0>(a, maps, st, fused);
  return cudaErrorInvalidValue;
}

cudaError_t launch_decode_tc(const DecodeArgs& a, const CUtensorMap* maps, bool dump, cudaStream_t st,
                             bool* fused) {
  if (fused) *fused = false;
  if (dump) {   // cache-read test entry: the raw page and gate rows
    if (a.d_c == 192) return launch_one<192, 1, 1>(a, maps, st, nullptr);
    if (a.d_c == 256) return launch_one<256, 1, 1>(a, maps, st, nullptr);
    return cudaErrorInvalidValue;
  }
  if (!a.gate) {
    if (a.d_c == 512) return launch_decode_wide(a, maps, st);
    return launch_mode<0>(a, maps, st, fused);
  }
  if (a.gate_add) return launch_mode<3>(a, maps, st, fused);
  if (a.gate_ln) return launch_mode<1>(a, maps, st, fused);
  return launch_mode<2>(a, maps, st, fused);
}

}  // namespace egmla
