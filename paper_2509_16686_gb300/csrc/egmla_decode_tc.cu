// egmla_decode_tc.cu - split-KV EG-MLA decode on sm_103a tensor cores for the
// latent widths 192 and 256 (gated or plain).
//
// One CTA per split-KV work unit (see egmla_common.cuh for the schedule).  The
// CTA streams its cache pages, one 64-token page per tile, through a ring of
// shared-memory slots; the tiles are token rows of the tensor-core operations
// (M = 64 tokens), the 16 heads their columns (N = 16).  Roles:
//
//   TMA (warp 4)      latent page [64 tok x d_c] (one 3-D box: 64-feature
//                     columns x 64 rows) and RoPE-key page [64 x 64], both
//                     128-byte swizzled, and the page's token ids (a bulk copy
//                     into the slot's statistics area), as soon as the page
//                     slot is free; a CTA's first page is requested alone.
//                     The split's start comes from a record the
//                     query-absorption kernel wrote.
//   gate (warps 7-14; each quarter-warp owns two token rows, lane u the 16-byte
//                     units 2u, 2u + 1 of every 64-feature column of them)
//                     the gate rows g = G[id] (EG-MLA-A table, Section 5.2)
//                     of the next tile into registers, requested column by
//                     column between this tile's stores as soon as the next
//                     page (and so its ids) has landed, every quarter-warp
//                     load reading one whole 128-byte line from L2; z = c (*) g
//                     rounded to bf16 and written back in place, and the
//                     LayerNorm statistics mu, r = 1/sqrt(var + eps) of z
//                     (Eq. 5 over d_c).
//   scores (warp 5)   S = Z (q^ gamma)^T and S_rope = K^R q^R^T (M = 64 tokens,
//                     N = 16 heads, K = d_c and 64; fp32 in TMEM, four score
//                     buffers) as soon as a gated page and a score buffer are
//                     ready, and the query block of the next sequence segment;
//                     with no query block to load the warp sleeps in hardware
//                     on the gate's barrier.
//   output (warp 6)   O^T += Z^T P' (M = 128 latent features, N = 16 heads,
//                     K = 64 tokens; O^T stays in TMEM over a sequence
//                     segment).  An issuing thread stalls while the tensor
//                     pipe's queue is full, so the two MMA streams have a
//                     thread each.
//   softmax (warps 0-3, one per TMEM lane quadrant: tokens 16w .. 16w + 15)
//                     thread t reads two tokens x four heads of S; the
//                     LayerNorm is applied after the MMA, since
//                       q^.LN(z) = r (q^ gamma).z - r mu sum(q^ gamma) + q^.beta,
//                     s = scale (r (S - mu w) + b + S_rope); an online softmax
//                     whose per-head reference max moves only when a tile
//                     exceeds it by 2^8 (one barrier vote of the four warps per
//                     tile decides; the maxima are exchanged only then), and
//                     P' = p r (bf16) as the B operand of the output MMA.
//
// At the end of each sequence segment the four softmax warps read O^T (latent
// features in TMEM lanes) and write the split's partial result: the
// un-normalised latent output gamma (*) (O - sum_j P'_j mu_j) + beta l, the
// reference max m and the denominator l = sum_j P'_j / r_j.  With heads as
// the MMA columns, no tensor-core work is spent on padding rows, tensor
// memory holds four score buffers and the whole output in 160 columns, and the
// query block takes 10 KB, which leaves room for five page slots at d_c = 256.
//
// The queries are absorbed before this kernel (q^ = W_UK^T q^C, with gamma
// folded in); the kernel may start while that kernel runs (programmatic
// stream serialisation) and waits for it after its set-up.  The split merge
// and W_UV run at its end when the grid is cooperative (fused_combine).
// Everything the kernel waits on has a time limit: on expiry it records
// EG_MLA_ERR_TIMEOUT, drains its own copies and MMAs, frees TMEM and exits.
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

#ifndef EGMLA_GATE_WARPS
#define EGMLA_GATE_WARPS 8
#endif
constexpr int kHeads = 16;
constexpr int kRope = 64;
constexpr int kThreads = 32 * (7 + EGMLA_GATE_WARPS);
constexpr int kSoftWarps = 4;    // warps 0-3: TMEM lane quadrants 0-3
constexpr int kSoftThreads = 32 * kSoftWarps;
constexpr int kTmaWarp = 4;
constexpr int kMmaWarp = 5;      // score MMAs and query blocks; also allocates and frees TMEM
constexpr int kOutWarp = 6;      // output MMAs
constexpr int kGateWarp0 = 7;
constexpr int kGateWarps = EGMLA_GATE_WARPS;
// 16-byte units of each 64-feature column a gate thread takes (the 64 token
// rows of a page over the gate threads), and lanes per token row
constexpr int kGateUnits = 16 / kGateWarps;
constexpr int kGateLanesPerRow = 8 / kGateUnits;
static_assert(kGateWarps == 8 || kGateWarps == 16, "gate warps");
constexpr uint32_t kSmemLimit = 232448;
// named barriers of the softmax warps (0 is __syncthreads)
constexpr int kBarTile = 1;
constexpr int kBarXch = 2;
// sequences per unit of the fused combine
constexpr uint32_t kFusedMaxG = 16;
// W_UV,h rows per warp in the fused combine (the fused path needs d_v <= 9 x warps)
constexpr int kCombineRowsPerWarp = 9;
// a head's reference max moves only when a tile exceeds it by 2^8
constexpr float kLazyLog2 = 8.f;
// score buffers in TMEM and P' buffers in shared memory
constexpr int kNB = 4;
constexpr int kNP = 4;

template <int D_C, bool GATE>
struct Cfg {
  static constexpr int NCH = D_C / 64;                  // 64-feature swizzle-atom columns
  static constexpr uint32_t PCHUNK = kPage * 128;       // one atom column of a page: 8 KB
  static constexpr uint32_t KR_OFF = NCH * PCHUNK;
  static constexpr uint32_t SLOT = KR_OFF + PCHUNK;     // latent + RoPE key of one page
  static constexpr uint32_t STAT_BYTES = GATE ? 2 * kPage * 4 : 0;   // per slot: mu[64], r[64]
  static constexpr uint32_t QB_LAT = qprep_lat_bytes(D_C);
  static constexpr uint32_t QPREP = qprep_bytes_tc(D_C, kRope);
  static constexpr uint32_t QBUF = (QPREP + 127) / 128 * 128;
  // P' [64 tokens x 16 heads] as the MN-major B operand of the output MMA
  static constexpr uint32_t PBUF = kPage * kHeads * 2;
  // LayerNorm gamma and beta of the segment read-out
  static constexpr uint32_t GB_BYTES = GATE ? 2 * D_C * 4 : 0;
  // softmax exchange: tile maxima [4 warps][16], segment sums [4 warps][16][2]
  static constexpr uint32_t XCH = 1024;
  static constexpr uint32_t MISC = 1024;
  static constexpr uint32_t FIXED = kNP * PBUF + GB_BYTES + XCH + MISC + 1024;
  // slots with two query buffers (the next segment's loaded while this one is
  // in use) or with one; one buffer when a second would cost a slot below five
  static constexpr int NS2 = (int)((kSmemLimit - FIXED - 2 * QBUF) / (SLOT + STAT_BYTES));
  static constexpr int NS1 = (int)((kSmemLimit - FIXED - QBUF) / (SLOT + STAT_BYTES));
  static constexpr int NQ = (NS2 < 5 && NS1 > NS2) ? 1 : 2;
  static constexpr int NS_FIT = NQ == 2 ? NS2 : NS1;
  static constexpr int NS = NS_FIT > 6 ? 6 : NS_FIT;
  static constexpr uint32_t OFF_QBUF = NS * SLOT;
  static constexpr uint32_t OFF_PBUF = OFF_QBUF + NQ * QBUF;
  static constexpr uint32_t OFF_STAT = OFF_PBUF + kNP * PBUF;
  static constexpr uint32_t OFF_GB = OFF_STAT + NS * STAT_BYTES;
  static constexpr uint32_t OFF_XCH = OFF_GB + GB_BYTES;
  static constexpr uint32_t OFF_MISC = OFF_XCH + XCH;
  static constexpr uint32_t SMEM = OFF_MISC + MISC + 1024;
  // TMEM columns: kNB score buffers of (latent 16 + RoPE 16) head columns,
  // then the latent output O^T (16 head columns per 128-feature M chunk)
  static constexpr uint32_t S_COLS = 32;
  static constexpr uint32_t COL_S = 0, COL_O = kNB * S_COLS;
  static constexpr uint32_t TMEM_COLS = 256;
  static constexpr uint32_t PAGE_TX = SLOT;
  static constexpr uint32_t ID_TX = GATE ? kPage * 4 : 0;   // the page's token ids
  static_assert(NS >= 3, "the ring needs three page slots");
  static_assert(SMEM <= kSmemLimit, "shared memory");
  static_assert(D_C == 192 || D_C == 256, "latent widths of this kernel");
  static_assert(COL_O + 32 <= TMEM_COLS, "tensor memory");
  // first latent feature of output M chunk j (two chunks of 128 rows); for
  // D_C = 192 the second chunk starts at 64 and overlaps the first, so that no
  // MMA reads past the latent part of a slot (its rows 64..127 are not read out)
  __host__ __device__ static constexpr int mc_start(int j) { return j == 0 ? 0 : D_C - 128; }
  // fused combine: up to kFusedMaxG merged latent rows reuse the page-slot area
  static_assert(kFusedMaxG * D_C * 4 <= OFF_QBUF, "fused combine area");
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
  const SplitStart* starts;
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
  // limit of every wait (ns); a test entry lowers it, together with a
  // withheld page copy (stall_cta, stall_tile; stall_cta < 0: none)
  uint64_t wait_ns;
  int stall_cta, stall_tile;
};

// Trace recorder of one role of one CTA.  Only the trace instantiation of the
// kernel records (ON); in the others every call compiles to nothing, since even
// untaken trace stores in the loops cost registers and instruction-cache room.
template <bool ON>
struct TracerT {
  unsigned long long* base;
  int n, cap;
  // part 0 of 1 is the role's whole run; part k of 2 is half of it (two writers)
  __device__ void init(const TcParams& p, int role, int part = 0, int parts = 1) {
    base = nullptr;
    n = 0;
    cap = p.trace_cap / parts;
    if (ON && p.trace != nullptr && static_cast<int>(blockIdx.x) < p.trace_ctas)
      base = p.trace + ((static_cast<size_t>(blockIdx.x) * kTraceRoles + role) * p.trace_cap + part * cap) * 2;
  }
  // (tag, SM clock); the phase marks carry the global timer that maps the
  // clock of each CTA to time
  __device__ __forceinline__ void mark(int event, int tile) {
    if (ON && base != nullptr && n < cap) {
      base[2 * n] = (static_cast<unsigned long long>(event) << 56) |
                    (static_cast<unsigned long long>(tile & 0xffffff) << 32);
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
  uint64_t sready[kNB], sfree[kNB];
  uint64_t spdone[kNP], pfree[kNP];
  uint64_t drain_s, drain_o;   // all MMAs of the score / output issuer done
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

  // the split's start record (written by the prologue kernel): one round of loads
  __device__ void start(const TcParams& p) {
    cu = p.cu;
    lens = p.seq_lens;
    batch = p.batch;
    const int4* r = reinterpret_cast<const int4*>(p.starts + blockIdx.x);
    const int4 h0 = __ldg(r), h1 = __ldg(r + 1);
    b = h0.x;
    lp = h0.y;
    lp_end = h0.z;
    L = h0.w;
    g1 = h1.x;
    done = h1.y != 0;
    first = true;
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
// The window starts as the first pages of the split's start record.
struct PageWindow {
  int b = -1, base = 0, n = 0, reg = -1;
  __device__ __forceinline__ void init(const TcParams& p, int lane) {
    const SplitStart* r = p.starts + blockIdx.x;
    b = __ldg(&r->b);
    base = __ldg(&r->lp);
    n = __ldg(&r->npages);
    reg = lane < kStartPages ? __ldg(&r->page[lane]) : -1;
  }
  __device__ __forceinline__ int page(const TcParams& p, const Tile& t, int lane) {
    if (t.b != b || t.lp < base || t.lp >= base + n) {
      b = t.b;
      base = t.lp;
      n = 32;
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
__device__ __forceinline__ bool warp_wait(uint32_t bar, uint32_t parity, volatile int* abort_flag, uint64_t limit_ns) {
  __syncwarp();
  const bool ok = mbar_wait(bar, parity, abort_flag, limit_ns);
  return __all_sync(0xffffffffu, ok);
}

// one arrival per warp: the warp barrier orders every lane's earlier writes
// before lane 0's release arrival
__device__ __forceinline__ void warp_arrive(uint32_t bar) {
  __syncwarp();
  if ((threadIdx.x & 31) == 0) mbar_arrive(bar);
}

// lane 0's non-blocking test of a phase, the same answer in every lane
__device__ __forceinline__ bool warp_test(uint32_t bar, uint32_t parity) {
  return __shfl_sync(0xffffffffu, mbar_test_now(bar, parity) ? 1 : 0, 0) != 0;
}

// Named barrier of the softmax warps that also ORs a predicate over them: every
// participant gets the same answer, so a branch on it is uniform.
__device__ __forceinline__ bool soft_vote(int id, bool v) {
  uint32_t r;
  asm volatile(
      "{\n\t.reg .pred p, q;\n\t"
      "setp.ne.u32 p, %1, 0;\n\t"
      "barrier.cta.red.or.pred q, %2, %3, p;\n\t"
      "selp.u32 %0, 1, 0, q;\n\t}"
      : "=r"(r)
      : "r"(v ? 1u : 0u), "r"(id), "r"(kSoftThreads)
      : "memory");
  return r != 0;
}

__device__ __forceinline__ void soft_sync(int id) {
  asm volatile("barrier.cta.sync %0, %1;" ::"r"(id), "r"(kSoftThreads) : "memory");
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

// 2^x with the hardware approximation (max 2 ulp; the weights are rounded to
// bf16 right after, and -inf gives 0)
__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// 16 lanes x 32 columns of 32-bit (tcgen05.ld.16x256b.x4): thread t gets lanes
// t/4 and t/4 + 8 at columns 8k + 2(t%4) and 8k + 2(t%4) + 1 of every 8-column
// group k, as v[4k] = (t/4, 8k + 2(t%4)), v[4k + 1] = (t/4, +1),
// v[4k + 2] = (t/4 + 8, ...), v[4k + 3] = (t/4 + 8, +1)
__device__ __forceinline__ void tmem_ld_16x256b_x4(uint32_t taddr, float (&v)[16]) {
  uint32_t r[16];
  asm volatile(
      "tcgen05.ld.sync.aligned.16x256b.x4.b32 "
      "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
      : "r"(taddr)
      : "memory");
#pragma unroll
  for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}

// 32 lanes x 32 columns of 32-bit: thread i of the warp gets its lane's 32 values
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, float (&v)[32]) {
  uint32_t r[32];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16, %17, %18, %19, %20, %21, %22, "
      "%23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
        "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
        "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr)
      : "memory");
#pragma unroll
  for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}

// inverse of tmem_ld32 (same thread-to-element map)
__device__ __forceinline__ void tmem_st32(uint32_t taddr, const float (&v)[32]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], "
      "{%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16, %17, %18, %19, %20, %21, %22, %23, "
      "%24, %25, %26, %27, %28, %29, %30, %31, %32};" ::"r"(taddr),
      "r"(__float_as_uint(v[0])), "r"(__float_as_uint(v[1])), "r"(__float_as_uint(v[2])), "r"(__float_as_uint(v[3])),
      "r"(__float_as_uint(v[4])), "r"(__float_as_uint(v[5])), "r"(__float_as_uint(v[6])), "r"(__float_as_uint(v[7])),
      "r"(__float_as_uint(v[8])), "r"(__float_as_uint(v[9])), "r"(__float_as_uint(v[10])), "r"(__float_as_uint(v[11])),
      "r"(__float_as_uint(v[12])), "r"(__float_as_uint(v[13])), "r"(__float_as_uint(v[14])),
      "r"(__float_as_uint(v[15])), "r"(__float_as_uint(v[16])), "r"(__float_as_uint(v[17])),
      "r"(__float_as_uint(v[18])), "r"(__float_as_uint(v[19])), "r"(__float_as_uint(v[20])),
      "r"(__float_as_uint(v[21])), "r"(__float_as_uint(v[22])), "r"(__float_as_uint(v[23])),
      "r"(__float_as_uint(v[24])), "r"(__float_as_uint(v[25])), "r"(__float_as_uint(v[26])),
      "r"(__float_as_uint(v[27])), "r"(__float_as_uint(v[28])), "r"(__float_as_uint(v[29])),
      "r"(__float_as_uint(v[30])), "r"(__float_as_uint(v[31]))
      : "memory");
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
// the splits that covered that sequence have counted their parts on its
// counter, otherwise after every CTA has arrived on a grid counter (both
// counters zeroed by the prologue kernel of the same call).  For each sequence
// b, over the splits s that covered it,
//   o = sum_s 2^(m_s - M) O_s / sum_s 2^(m_s - M) l_s,  M = max_s m_s,
//   u_{b,h} = W_UV,h o
// (a sequence of length 0 gets u = 0).  Each warp loads its nine rows of
// W_UV,h (lane l holding features 8l .. 8l + 7) from global memory into
// registers before it waits, so that the loads overlap the wait.  Merge: a
// warp per (sequence, 32 features), lane k loading (m, l) of slot k0 + k and
// every lane O of 32 slots at once (online rescaling across groups of 32),
// into shared memory.  u: per sequence, the warp's first eight row sums
// reduced across the lanes by a transposing butterfly (9 shuffles, after
// which lane 4r holds row r) and the ninth by a plain warp sum.
template <int D_C, bool TRACE>
__device__ void fused_combine(const TcParams& p, uint8_t* smem, Bars& bars) {
  constexpr int kWarps = kThreads / 32;
  constexpr int NFB = D_C / 32;      // 32-feature blocks of a row
  constexpr int LANES = D_C / 8;     // lanes holding 8 features each
  constexpr int kRows = kCombineRowsPerWarp;   // output rows of W_UV,h per warp
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int G = p.cmb_g, units = kHeads * p.cmb_groups;
  float* olat = reinterpret_cast<float*>(smem);   // [G][D_C], in the free page-slot area
  volatile int* abort_flag = &bars.abort;
  const uint64_t wait_ns = p.wait_ns;
  const uint64_t keep = policy_evict_last();
  const int v0 = warp * kRows;   // this warp's first output row
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
      if (globaltimer() - t0 > wait_ns) {
        report_status(p.status, kStatusTimeout);
        *abort_flag = 1;
        break;
      }
      __nanosleep(32);
    }
  }
  for (int u = blockIdx.x; u < units; u += gridDim.x) {
    const int h = u % kHeads, grp = u / kHeads;
    const int b0 = grp * G, nb = min(G, p.batch - b0);
    // this warp's W_UV,h rows, requested before the wait
    uint4 wraw[kRows];
#pragma unroll
    for (int r = 0; r < kRows; ++r) {
      const int v = v0 + r;
      wraw[r] = make_uint4(0, 0, 0, 0);
      if (lane < LANES && v < p.d_v)
        wraw[r] = ldg_16_na_hint(p.w_uv + (static_cast<size_t>(h) * p.d_v + v) * D_C + 8 * lane, keep);
    }
    if (G == 1 && tid == 0 && !*abort_flag) {
      // a unit of one sequence: every softmax warp's part of every split partial of it stored
      const uint32_t want = static_cast<uint32_t>(kSoftWarps) * static_cast<uint32_t>(splits_of(b0));
      const uint64_t t0 = globaltimer();
      while (ld_acquire_gpu(p.seq_done + 1 + b0) < want) {
        if (*abort_flag) break;
        if (globaltimer() - t0 > wait_ns) {
          report_status(p.status, kStatusTimeout);
          *abort_flag = 1;
          break;
        }
        __nanosleep(32);
      }
    }
    __syncthreads();
    if (u == static_cast<int>(blockIdx.x)) phase_mark<TRACE>(p, 4);
    if (*abort_flag) return;
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
        // four independent sums over the slots (zero weight past kn)
        float a4[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int kk = 0; kk < 32; ++kk) a4[kk & 3] = fmaf(__shfl_sync(0xffffffffu, wk, kk), ov[kk], a4[kk & 3]);
        acc = fmaf(acc, sc, (a4[0] + a4[1]) + (a4[2] + a4[3]));
        M = Mn;
      }
      olat[j * D_C + f] = n > 0 ? acc / L : 0.f;
    }
    __syncthreads();
    if (u == static_cast<int>(blockIdx.x)) phase_mark<TRACE>(p, 5);
    // u = W_UV,h o from the registers loaded above: rows v0 .. v0 + 7 by the
    // butterfly, the ninth by a plain reduction
    if (v0 < p.d_v) {   // uniform in the warp
      for (int j = 0; j < nb; ++j) {
        float o8[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
        if (lane < LANES) {
          const float4 x0 = *reinterpret_cast<const float4*>(olat + j * D_C + 8 * lane);
          const float4 x1 = *reinterpret_cast<const float4*>(olat + j * D_C + 8 * lane + 4);
          o8[0] = x0.x; o8[1] = x0.y; o8[2] = x0.z; o8[3] = x0.w;
          o8[4] = x1.x; o8[5] = x1.y; o8[6] = x1.z; o8[7] = x1.w;
        }
        float part[kRows];
#pragma unroll
        for (int r = 0; r < kRows; ++r) {
          float wv[8];
          bf16x8_to_float(wraw[r], wv);
          part[r] = 0.f;
#pragma unroll
          for (int e = 0; e < 8; ++e) part[r] = fmaf(wv[e], o8[e], part[r]);
        }
        const float sum = reduce8_rows(reinterpret_cast<const float (&)[8]>(part), lane);
        float last = part[8];
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) last += __shfl_xor_sync(0xffffffffu, last, o);
        __nv_bfloat16* orow = p.out + (static_cast<size_t>(b0 + j) * kHeads + h) * p.d_v;
        const int v = v0 + (lane >> 2);
        if ((lane & 3) == 0 && v < p.d_v) orow[v] = __float2bfloat16_rn(sum);
        if (lane == 0 && v0 + 8 < p.d_v) orow[v0 + 8] = __float2bfloat16_rn(last);
      }
    }
    __syncthreads();   // olat is free for the next unit
    if (u == static_cast<int>(blockIdx.x)) phase_mark<TRACE>(p, 6);
  }
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
  const uint64_t wait_ns = p.wait_ns;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  phase_mark<DBG == 2>(p, 0);
  // a kernel launched after this one with programmatic stream serialisation
  // (the layer's output projection) may take each SM this kernel leaves
  grid_launch_dependents();

  if (threadIdx.x == 0) {
    for (int s = 0; s < C::NS; ++s) {
      mbar_init(smem_u32(&bars.full[s]), 1);
      mbar_init(smem_u32(&bars.empty[s]), DUMP ? kGateWarps : 1);
      mbar_init(smem_u32(&bars.zready[s]), kGateWarps);
    }
    for (int s = 0; s < 2; ++s) {
      mbar_init(smem_u32(&bars.qfull[s]), 1);
      // the last score MMA of the segment (commit) and the softmax warps' read of its sums
      mbar_init(smem_u32(&bars.qempty[s]), 1 + kSoftWarps);
    }
    for (int s = 0; s < kNB; ++s) {
      // the MMA commit plus a release arrival of the MMA warp after it saw the
      // gate's zready (so that the statistics are visible to the softmax warps)
      mbar_init(smem_u32(&bars.sready[s]), 2);
      mbar_init(smem_u32(&bars.sfree[s]), kSoftWarps);
    }
    for (int s = 0; s < kNP; ++s) {
      mbar_init(smem_u32(&bars.spdone[s]), kSoftWarps);
      mbar_init(smem_u32(&bars.pfree[s]), 1);
    }
    mbar_init(smem_u32(&bars.drain_s), 1);
    mbar_init(smem_u32(&bars.drain_o), 1);
    bars.abort = 0;
    fence_mbar_init();
  }
  if (warp == kMmaWarp) {
    tmem_alloc(smem_u32(&bars.tmem_base), C::TMEM_COLS);
    tmem_relinquish();
  }
  if (warp == kTmaWarp && lane == 0) {
    prefetch_tensormap(&cmap);
    prefetch_tensormap(&krmap);
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  phase_mark<DBG == 2>(p, 1);
  const uint32_t tmem = bars.tmem_base;
  // Everything above touches only this CTA's shared and tensor memory; what
  // follows reads the query-absorption kernel's outputs (prepared queries,
  // split schedule, zeroed counters) and the cache it may have appended to.
  grid_dependency_wait();

  if (warp == kTmaWarp) {
    // ---------------------------------------------------------------- TMA producer
    // The whole warp walks the tiles; lane 0 waits for the slot and issues the
    // copies.  A slot is free once the output MMA of the tile that held it is
    // complete.
    const uint64_t pol_stream = policy_evict_first();
    Walker w;
    w.start(p);
    PageWindow pw;
    pw.init(p, lane);
    Tile t;
    int it = 0;
    int last_it[6] = {-1, -1, -1, -1, -1, -1};
    Tracer tr;
    tr.init(p, 0);
    if (lane != 0) tr.base = nullptr;
    bool ok_loop = true;
    while (ok_loop && w.next(t)) {
      const int pg = pw.page(p, t, lane);
      const int slot = it % C::NS;
      if (lane == 0) {
        tr.mark(0, it);
        if (!mbar_wait(smem_u32(&bars.empty[slot]), ((it / C::NS) & 1) ^ 1, abort_flag, wait_ns)) ok_loop = false;
        if (ok_loop) {
          tr.mark(1, it);
          const bool ok = pg >= 0 && pg < p.num_pages;
          if (!ok) report_status(p.status, kStatusOutOfRange);
          // (test entry) a withheld page: no copy and no arrival, so that the
          // gate's wait on this slot runs out
          const bool withheld = static_cast<int>(blockIdx.x) == p.stall_cta && it == p.stall_tile;
          if (!withheld) {
            const uint32_t fb = smem_u32(&bars.full[slot]);
            mbar_arrive_expect_tx(fb, ok ? C::PAGE_TX + C::ID_TX : 0u);
            if (ok) {
              const uint32_t dst = sbase + slot * C::SLOT;
              const int y = pg * kPage;
              tma_load_3d(dst, &cmap, 0, y, 0, fb, pol_stream);
              tma_load_2d(dst + C::KR_OFF, &krmap, 0, y, fb, pol_stream);
              // the page's token ids, into the half of the slot's statistics that
              // holds r once the gate has read them
              if (C::ID_TX)
                bulk_load_hint(sbase + C::OFF_STAT + slot * C::STAT_BYTES + kPage * 4,
                               p.id_pool + static_cast<size_t>(pg) * kPage, C::ID_TX, fb, pol_stream);
            }
            last_it[slot] = it;
          }
          tr.mark(2, it);
        }
      }
      // The first page alone: every CTA asks for one page, and the rest only
      // once it has landed, so that the first pages of all CTAs land early
      // (one page per SM) instead of in a burst of all their slots.
      if (it == 0 && lane == 0 && ok_loop && last_it[0] == 0 &&
          !mbar_wait(smem_u32(&bars.full[0]), 0, abort_flag, wait_ns))
        ok_loop = false;
      ok_loop = __shfl_sync(0xffffffffu, ok_loop, 0);
      ++it;
    }
    if (lane == 0) {
      // drain: every copy this thread issued must land before the CTA exits,
      // also after an abort (own flag: the wait is bounded but not cut short)
      volatile int own = 0;
      for (int s = 0; s < C::NS; ++s)
        if (last_it[s] >= 0 && !mbar_wait(smem_u32(&bars.full[s]), (last_it[s] / C::NS) & 1, &own, wait_ns)) *abort_flag = 1;
    }
    __syncwarp();
  } else if (warp == kMmaWarp) {
    // ---------------------------------------------------------------- score MMAs, query blocks
    // Converged warp; one elected lane issues.  The warp polls two queues and
    // serves whichever is ready, so that neither waits for the other's
    // condition:
    //   query block of segment qn: its buffer's previous segment is done
    //     (last score MMA complete, sums read by the softmax warps);
    //   scores of tile js: its gated page (zready), a free score buffer (the
    //     softmax warps read tile js - kNB's), and at a segment start the
    //     segment's query block.
    // Loops are unrolled with compile-time accumulate flags.
    if (!DUMP) {
      constexpr uint32_t IDESC_S = idesc_bf16(64, kHeads, 0, 0);
      // A operand: the page slot, 128-byte swizzled, K-major (tokens x
      // features); B: the query block in 8x8 core matrices, K cores 256 B
      // apart, head halves 128 B apart
      const uint64_t zdesc_k = smem_desc(sbase, 16, 1024, kSwizzle128B);
      const uint64_t qdesc0 = smem_desc(sbase + C::OFF_QBUF, kQGroupBytes, kQRowGroupBytes, kSwizzleNone);
      Walker ws, wq;
      ws.start(p);
      wq.start(p);
      Tile ts, tq;
      bool s_more = ws.next(ts), q_more = wq.next(tq);
      int js = 0, qn = 0, seg_s = -1;
      int last_q[2] = {-1, -1};
      bool issued = false;
      Tracer tr;
      tr.init(p, 1, 0, 2);
      if (lane != 0) tr.base = nullptr;
      uint64_t idle_since = 0;
      while (s_more) {
        bool progress = false;
        // ---- query block of the next segment
        if (q_more && warp_test(smem_u32(&bars.qempty[qn % C::NQ]), ((qn / C::NQ) & 1) ^ 1)) {
          const int qb = qn % C::NQ;
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
          progress = true;
        }
        // ---- scores of tile js
        const int slot = js % C::NS, sb = js % kNB;
        const uint32_t zpar = (js / C::NS) & 1;
        const int sg = seg_s + (ts.first ? 1 : 0);
        bool ready = !ts.first || (qn > sg && warp_test(smem_u32(&bars.qfull[sg % C::NQ]), (sg / C::NQ) & 1));
        ready = ready && warp_test(smem_u32(&bars.sfree[sb]), ((js / kNB) & 1) ^ 1);
        if (ready && !(q_more && warp_test(smem_u32(&bars.qempty[qn % C::NQ]), ((qn / C::NQ) & 1) ^ 1))) {
          // nothing else to serve: sleep in hardware until the gate warps
          // release the slot (the gate waits on nothing this warp does)
          ready = warp_wait(smem_u32(&bars.zready[slot]), zpar, abort_flag, wait_ns);
          if (!ready) break;   // uniform: the wait ran out or another role aborted
        } else {
          ready = ready && warp_test(smem_u32(&bars.zready[slot]), zpar);
        }
        if (ready) {
          seg_s = sg;
          tr.mark(1, js);
          if (lane == 0) mbar_arrive(smem_u32(&bars.sready[sb]));
          tc_fence_after();
          if (elect_one()) {
            const uint64_t za = zdesc_k + ((slot * C::SLOT) >> 4);
            const uint64_t qb = qdesc0 + (((seg_s % C::NQ) * C::QBUF) >> 4);
            const uint32_t ds = tmem + C::COL_S + sb * C::S_COLS;
#pragma unroll
            for (int kk = 0; kk < D_C / 16; ++kk)
              mma_bf16_ss(ds, za + (((kk >> 2) * C::PCHUNK + (kk & 3) * 32) >> 4),
                          qb + ((kk * 2 * kQGroupBytes) >> 4), IDESC_S, kk > 0);
#pragma unroll
            for (int kk = 0; kk < kRope / 16; ++kk)
              mma_bf16_ss(ds + kHeads, za + ((C::KR_OFF + kk * 32) >> 4),
                          qb + ((C::QB_LAT + kk * 2 * kQGroupBytes) >> 4), IDESC_S, kk > 0);
            mma_commit(smem_u32(&bars.sready[sb]));
            if (ts.last) mma_commit(smem_u32(&bars.qempty[seg_s % C::NQ]));
          }
          __syncwarp();
          tr.mark(2, js);
          issued = true;
          ++js;
          s_more = ws.next(ts);
          progress = true;
        }
        if (progress) {
          idle_since = 0;
        } else {
          // nothing ready: bounded wait for the others (and their abort)
          const uint64_t now = globaltimer();
          if (idle_since == 0) idle_since = now;
          bool stop = *abort_flag != 0;
          if (!stop && now - idle_since > wait_ns) {
            *abort_flag = 1;
            stop = true;
          }
          if (__any_sync(0xffffffffu, stop)) break;
          __nanosleep(32);   // leave the issue slots to the warps that do the work
        }
      }
      if (lane == 0) {
        // drain: the query-block copies this warp issued must land, and every
        // MMA must finish, before the CTA exits and TMEM is released (own flag:
        // bounded but not cut short by an abort)
        volatile int own = 0;
        for (int b = 0; b < 2; ++b)
          if (last_q[b] >= 0 && !mbar_wait(smem_u32(&bars.qfull[b]), (last_q[b] / C::NQ) & 1, &own, wait_ns)) *abort_flag = 1;
      }
      __syncwarp();
      if (issued) {
        if (elect_one()) mma_commit(smem_u32(&bars.drain_s));
        __syncwarp();
        volatile int own = 0;
        if (!mbar_wait(smem_u32(&bars.drain_s), 0, &own, wait_ns)) *abort_flag = 1;
      }
    }
    __syncwarp();
  } else if (warp == kOutWarp) {
    // ---------------------------------------------------------------- output MMAs
    // O^T[feature, head] += Z^T P' for each tile in order, as soon as the
    // softmax warps wrote its P'; completion frees the page slot and the P'
    // buffer.  A operand: the page slot read MN-major (features along M,
    // 64-feature atoms PCHUNK apart; tokens along K, 8-row groups 1 KB apart);
    // B: P' MN-major in 8x8 core matrices (token groups 256 B, head halves
    // 128 B).
    if (!DUMP) {
      constexpr uint32_t IDESC_O = idesc_bf16(128, kHeads, 1, 1);
      const uint64_t zdesc_mn = smem_desc(sbase, C::PCHUNK, 1024, kSwizzle128B);
      const uint64_t pdesc0 = smem_desc(sbase + C::OFF_PBUF, 256, 128, kSwizzleNone);
      Walker wo;
      wo.start(p);
      Tile to;
      int jo = 0;
      bool issued = false;
      Tracer tr;
      tr.init(p, 1, 1, 2);   // second half of the MMA role's run
      if (lane != 0) tr.base = nullptr;
      while (wo.next(to)) {
        if (!warp_wait(smem_u32(&bars.spdone[jo % kNP]), (jo / kNP) & 1, abort_flag, wait_ns)) break;
        tr.mark(3, jo);
        tc_fence_after();
        if (elect_one()) {
          const int slot = jo % C::NS;
          const uint64_t za = zdesc_mn + ((slot * C::SLOT) >> 4);
          const uint64_t pb = pdesc0 + (((jo % kNP) * C::PBUF) >> 4);
          if (to.first) {
#pragma unroll
            for (int ks = 0; ks < kPage / 16; ++ks)
#pragma unroll
              for (int mc = 0; mc < 2; ++mc)
                mma_bf16_ss(tmem + C::COL_O + kHeads * mc, za + (((C::mc_start(mc) / 64) * C::PCHUNK + ks * 2048) >> 4),
                            pb + ((ks * 512) >> 4), IDESC_O, ks > 0);
          } else {
#pragma unroll
            for (int ks = 0; ks < kPage / 16; ++ks)
#pragma unroll
              for (int mc = 0; mc < 2; ++mc)
                mma_bf16_ss(tmem + C::COL_O + kHeads * mc, za + (((C::mc_start(mc) / 64) * C::PCHUNK + ks * 2048) >> 4),
                            pb + ((ks * 512) >> 4), IDESC_O, 1);
          }
          mma_commit(smem_u32(&bars.empty[slot]));
          mma_commit(smem_u32(&bars.pfree[jo % kNP]));
        }
        __syncwarp();
        tr.mark(4, jo);
        issued = true;
        ++jo;
      }
      if (issued) {
        if (elect_one()) mma_commit(smem_u32(&bars.drain_o));
        __syncwarp();
        volatile int own = 0;
        if (!mbar_wait(smem_u32(&bars.drain_o), 0, &own, wait_ns)) *abort_flag = 1;
      }
    }
    __syncwarp();
  } else if (warp >= kGateWarp0) {
    // ---------------------------------------------------------------- gate: z = c (*) g, LN statistics
    // Quarter-warp k = 4 (warp - 7) + lane / 8 owns token rows 2k (lanes 0-3)
    // and 2k + 1 (lanes 4-7); lane p = lane % 4 of a row takes the 16-byte
    // units 2p and 2p + 1 of every 64-feature column.  The gate-row load of a
    // column is then one 32-byte load per lane and a whole 128-byte line per
    // row (the load/store data path pays per instruction and per line, so
    // fewer, wider loads are cheaper), and a quarter-warp's shared-memory
    // accesses to the swizzled page still hit eight distinct bank groups (the
    // two rows differ in swizzle parity).  The gate rows come from L2 (the
    // table stays there under an evict-last hint while the cache stream is
    // evict-first).  The token ids come with the page (the producer copies them
    // into the slot), so the gate rows of the next tile are requested as soon
    // as its page has landed, while this tile is processed; no load sits on a
    // chain of dependent global accesses.
    const int gw = warp - kGateWarp0;
    const int pp = lane % kGateLanesPerRow;
    const int row = gw * (32 / kGateLanesPerRow) + lane / kGateLanesPerRow;
    const uint64_t pol_keep = policy_evict_last();
    constexpr bool gate_ln = GATE_LN;
    Walker w;
    w.start(p);
    // id of this thread's row of tile jj, from the slot that holds its page (0
    // past the end of the page)
    auto slot_id = [&](int jj, const Tile& tt) -> int {
      const int32_t* ids = reinterpret_cast<const int32_t*>(smem + C::OFF_STAT + (jj % C::NS) * C::STAT_BYTES + kPage * 4);
      return row < tt.ntok ? ids[row] : 0;
    };
    // this thread's part of the gate row of token id (row 0, reported, for an
    // id outside the vocabulary)
    auto g_row = [&](int id) -> const __nv_bfloat16* {
      if ((unsigned)id >= (unsigned)p.vocab) {
        report_status(p.status, kStatusOutOfRange);
        id = 0;
      }
      return p.gate_table + static_cast<size_t>(id) * D_C + pp * 8 * kGateUnits;
    };
    auto load_g = [&](int id, uint4 (&gv)[C::NCH][kGateUnits]) {
      const __nv_bfloat16* src = g_row(id);
#pragma unroll
      for (int fc = 0; fc < C::NCH; ++fc) {
        if constexpr (kGateUnits == 2)
          ldg_32_na_hint(src + fc * 64, pol_keep, gv[fc][0], gv[fc][1]);
        else
          gv[fc][0] = ldg_16_na_hint(src + fc * 64, pol_keep);
      }
    };
    // shared-memory offset of unit (kGateUnits pp + h) of column fc of this thread's row
    auto unit_off = [&](int fc, int h) -> uint32_t {
      return fc * C::PCHUNK + row * 128 + (((kGateUnits * pp + h) ^ (row & 7)) << 4);
    };
    Tracer tr;
    tr.init(p, 2);
    if (threadIdx.x != kGateWarp0 * 32) tr.base = nullptr;
    Tile t, t1;
    bool have = w.next(t);
    bool have1 = have && w.next(t1);
    uint4 gcur[C::NCH][kGateUnits], gnext[C::NCH][kGateUnits];
    int id0 = 0;
    if (GATE && have) {
      // the first tile's rows: its page must land first
      if (warp_wait(smem_u32(&bars.full[0]), 0, abort_flag, wait_ns)) {
        id0 = slot_id(0, t);
        load_g(id0, gcur);
      } else {
        have = false;
      }
    }
    int j = 0;
    while (have) {
      const int slot = j % C::NS;
      tr.mark(0, j);
      // The next tile's gate rows: if its page has landed, requested column by
      // column between this tile's shared-memory stores (spreading the loads
      // over the tile instead of one burst), otherwise after this tile.
      bool next_issued = false;
      const __nv_bfloat16* gsrc_next = p.gate_table;
      if (GATE && have1 && warp_test(smem_u32(&bars.full[(j + 1) % C::NS]), ((j + 1) / C::NS) & 1)) {
        gsrc_next = g_row(slot_id(j + 1, t1));
        next_issued = true;
      }
      auto load_next_column = [&](int fc) {
        if (next_issued) {
          if constexpr (kGateUnits == 2)
            ldg_32_na_hint(gsrc_next + fc * 64, pol_keep, gnext[fc][0], gnext[fc][1]);
          else
            gnext[fc][0] = ldg_16_na_hint(gsrc_next + fc * 64, pol_keep);
        }
      };
      if (!warp_wait(smem_u32(&bars.full[slot]), (j / C::NS) & 1, abort_flag, wait_ns)) break;
      tr.mark(1, j);
      if (DUMP) id0 = slot_id(j, t);
      uint8_t* cpage = smem + slot * C::SLOT;
      if (DUMP) {
        if (row < t.ntok) {
          const size_t o = static_cast<size_t>(t.b) * p.dump_len + t.tok0 + row;
          uint4* dc = reinterpret_cast<uint4*>(p.dump_c + o * D_C);
          uint4* dg = reinterpret_cast<uint4*>(p.dump_g + o * D_C);
#pragma unroll
          for (int fc = 0; fc < C::NCH; ++fc) {
#pragma unroll
            for (int h = 0; h < kGateUnits; ++h) {
              dc[fc * 8 + kGateUnits * pp + h] = *reinterpret_cast<const uint4*>(cpage + unit_off(fc, h));
              dg[fc * 8 + kGateUnits * pp + h] = gcur[fc][h];
            }
          }
#pragma unroll
          for (int h = 0; h < kGateUnits; ++h)
            reinterpret_cast<uint4*>(p.dump_kr + o * kRope)[kGateUnits * pp + h] = *reinterpret_cast<const uint4*>(
                cpage + C::KR_OFF + row * 128 + (((kGateUnits * pp + h) ^ (row & 7)) << 4));
          if (pp == 0) p.dump_ids[o] = id0;
        }
#pragma unroll
        for (int fc = 0; fc < C::NCH; ++fc) load_next_column(fc);
        warp_arrive(smem_u32(&bars.empty[slot]));
      } else {
        const bool full_page = t.ntok == kPage;   // uniform: no token masking needed
        if (GATE) {
          float* st = reinterpret_cast<float*>(smem + C::OFF_STAT + slot * C::STAT_BYTES);
          // all shared-memory reads of this thread's units first (the in-place
          // stores below would otherwise order every later load behind them)
          uint4 cv[C::NCH][kGateUnits];
#pragma unroll
          for (int fc = 0; fc < C::NCH; ++fc)
#pragma unroll
            for (int h = 0; h < kGateUnits; ++h) cv[fc][h] = *reinterpret_cast<const uint4*>(cpage + unit_off(fc, h));
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
              for (int h = 0; h < kGateUnits; ++h) {
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
            for (int o = 1; o < kGateLanesPerRow; o <<= 1) {
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
              for (int h = 0; h < kGateUnits; ++h) {
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
              load_next_column(fc);
            }
            tr.mark(6, j);
            if (pp == 0) {
              // the stored z is centred; rows past the page end get r = 1 (their
              // weight is 0, and l adds 0 / r)
              st[row] = 0.f;
              st[kPage + row] = valid ? r : 1.f;
            }
          } else {
            float2 s1 = make_float2(0.f, 0.f), s2 = make_float2(0.f, 0.f);
            float2 a1 = make_float2(0.f, 0.f), a2 = make_float2(0.f, 0.f);
#pragma unroll
            for (int fc = 0; fc < C::NCH; ++fc) {
#pragma unroll
              for (int h = 0; h < kGateUnits; ++h) {
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
              load_next_column(fc);
            }
            s1 = __fadd2_rn(s1, a1);
            s2 = __fadd2_rn(s2, a2);
            float sum1 = s1.x + s1.y, sum2 = s2.x + s2.y;
            tr.mark(6, j);
            // row sums over the four lanes of the row (without the LayerNorm
            // ablation's norm: mu = 0, r = 1)
            if (gate_ln) {
#pragma unroll
              for (int o = 1; o < kGateLanesPerRow; o <<= 1) {
                sum1 += __shfl_xor_sync(0xffffffffu, sum1, o);
                sum2 += __shfl_xor_sync(0xffffffffu, sum2, o);
              }
            }
            if (pp == 0) {
              constexpr float inv_dc = 1.f / D_C;
              const float mu = gate_ln ? sum1 * inv_dc : 0.f;
              const float var = fmaxf(sum2 * inv_dc - mu * mu, 0.f);
              const float r = gate_ln ? rsqrtf(var + p.eps) : 1.f;
              // rows past the page end: mu = 0, r = 1 (their weight is 0, and l adds 0 / r)
              st[row] = valid ? mu : 0.f;
              st[kPage + row] = valid ? r : 1.f;
            }
          }
        } else if (!full_page) {
          if (row >= t.ntok) {
#pragma unroll
            for (int fc = 0; fc < C::NCH; ++fc)
#pragma unroll
              for (int h = 0; h < kGateUnits; ++h)
                *reinterpret_cast<uint4*>(cpage + unit_off(fc, h)) = make_uint4(0, 0, 0, 0);
          }
        }
        tr.mark(2, j);
        fence_proxy_async_smem();
        warp_arrive(smem_u32(&bars.zready[slot]));
      }
      tr.mark(3, j);
      if (GATE && have1 && !next_issued) {
        // the next page landed only now
        if (!warp_wait(smem_u32(&bars.full[(j + 1) % C::NS]), ((j + 1) / C::NS) & 1, abort_flag, wait_ns)) break;
        load_g(slot_id(j + 1, t1), gnext);
      }
      ++j;
      t = t1;
      have = have1;
      have1 = have1 && w.next(t1);
      if (GATE) {
#pragma unroll
        for (int fc = 0; fc < C::NCH; ++fc) {
#pragma unroll
          for (int h = 0; h < kGateUnits; ++h) gcur[fc][h] = gnext[fc][h];
        }
      }
    }
  } else if (warp < kSoftWarps && !DUMP) {
    // ---------------------------------------------------------------- softmax, output read-out
    // Warp w reads TMEM lane quadrant w: tokens 16w .. 16w + 15 of a tile's
    // scores (rows of the M = 64 accumulator) and latent features 32w .. 32w +
    // 31 of each 128-feature chunk of O^T.  Thread t owns tokens r0 = 16w + t/4
    // and r1 = r0 + 8 and heads hh(k) = 2q, 2q + 1, 8 + 2q, 9 + 2q (q = t % 4).
    // Lane h < 16 of every warp also keeps head h's reference max (the same in
    // all four warps), which the rare slow path of the max update uses.
    const int q = lane & 3;
    const int r0 = 16 * warp + (lane >> 2), r1 = r0 + 8;
    const uint32_t tq = tmem + (static_cast<uint32_t>(32 * warp) << 16);
    const float scale = p.scale_log2;
    float* xmax = reinterpret_cast<float*>(smem + C::OFF_XCH);        // [4 warps][16 heads]
    float* xsum = xmax + kSoftWarps * kHeads;                         // [4 warps][16 heads][2]
    auto head_of = [&](int k) { return (k & 1) + 2 * q + 8 * (k >> 1); };
    // gamma and beta of the segment read-out in shared memory (written once by
    // the four warps; the first tile's barrier orders the writes before any read)
    float* gb = reinterpret_cast<float*>(smem + C::OFF_GB);
    if (GATE) {
      for (int f = threadIdx.x; f < D_C; f += kSoftThreads) {
        gb[f] = p.gamma ? __ldg(p.gamma + f) : 1.f;
        gb[D_C + f] = p.beta ? __ldg(p.beta + f) : 0.f;
      }
    }
    float m_ref[4], l_acc[4], bmu_acc[4], wq[4], bsc[4];
    float m16 = -INFINITY;   // head `lane` (lanes 0-15)
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      m_ref[k] = -INFINITY;
      l_acc[k] = 0.f;
      bmu_acc[k] = 0.f;
      wq[k] = 0.f;
      bsc[k] = 0.f;
    }
    Walker w;
    w.start(p);
    Tile t;
    int it = 0, seg = -1;
    Tracer tr;
    tr.init(p, 3);
    if (threadIdx.x != 0) tr.base = nullptr;
    while (w.next(t)) {
      bool ok = true;
      if (t.first) {
        ++seg;
        ok = warp_wait(smem_u32(&bars.qfull[seg % C::NQ]), (seg / C::NQ) & 1, abort_flag, wait_ns);
        if (ok && GATE) {
          // w_h = sum_f bf16(q^ gamma)_hf and b_h = q^_h . beta from their
          // per-chunk partials after the operands, added in chunk order
          const float* sums = reinterpret_cast<const float*>(smem + C::OFF_QBUF + (seg % C::NQ) * C::QBUF +
                                                             C::QB_LAT + qprep_rope_bytes(kRope));
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            const int h = head_of(k);
            float wsum = 0.f, bsum = 0.f;
#pragma unroll
            for (int c = 0; c < D_C / kSumFeatures; ++c) {
              wsum += sums[c * 32 + h];
              bsum += sums[c * 32 + 16 + h];
            }
            wq[k] = wsum;
            bsc[k] = bsum * scale;
          }
        }
        if (ok) warp_arrive(smem_u32(&bars.qempty[seg % C::NQ]));
      }
      const int slot = it % C::NS, sb = it % kNB, pb = it % kNP;
      tr.mark(0, it);
      // scores of this tile; the MMA warp's release arrival on the same barrier
      // orders the gate's statistics before them
      ok = ok && warp_wait(smem_u32(&bars.sready[sb]), (it / kNB) & 1, abort_flag, wait_ns);
      tr.mark(1, it);
      float s[2][4];
      float mu[2] = {0.f, 0.f}, rr[2] = {1.f, 1.f};
      bool exceed = false;
      if (ok) {
        tc_fence_after();
        float v[16];
        tmem_ld_16x256b_x4(tq + C::COL_S + sb * C::S_COLS, v);
        if (GATE) {
          const float* st = reinterpret_cast<const float*>(smem + C::OFF_STAT + slot * C::STAT_BYTES);
          mu[0] = st[r0];
          mu[1] = st[r1];
          rr[0] = st[kPage + r0];
          rr[1] = st[kPage + r1];
        }
        tmem_wait_ld();
        tc_fence_before();
        warp_arrive(smem_u32(&bars.sfree[sb]));   // score buffer read: tile it + kNB may overwrite it
        tr.mark(7, it);
        const bool full_page = t.ntok == kPage;
#pragma unroll
        for (int e = 0; e < 2; ++e) {
          const bool valid = full_page || (e ? r1 : r0) < t.ntok;
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            const float lat = v[(k >> 1) * 4 + 2 * e + (k & 1)];
            const float rope = v[8 + (k >> 1) * 4 + 2 * e + (k & 1)];
            float x;
            if (GATE) {
              x = fmaf(rr[e] * scale, fmaf(-mu[e], wq[k], lat), fmaf(rope, scale, bsc[k]));
            } else {
              x = (lat + rope) * scale;
            }
            s[e][k] = valid ? x : -INFINITY;
            exceed = exceed || (x > m_ref[k] + kLazyLog2 && valid);
          }
        }
      }
      tr.mark(8, it);
      // one vote of the four warps: a head's reference max must move (or a
      // wait failed somewhere)
      if (soft_vote(kBarTile, exceed || !ok)) {
        if (soft_vote(kBarTile, !ok)) break;   // uniform: every warp leaves
        // ---- slow path: tile maxima of the heads over the 64 tokens
        float tm[4];
#pragma unroll
        for (int k = 0; k < 4; ++k) tm[k] = fmaxf(s[0][k], s[1][k]);
#pragma unroll
        for (int o = 4; o < 32; o <<= 1)
#pragma unroll
          for (int k = 0; k < 4; ++k) tm[k] = fmaxf(tm[k], __shfl_xor_sync(0xffffffffu, tm[k], o));
        if (lane < 4) {
#pragma unroll
          for (int k = 0; k < 4; ++k) xmax[warp * kHeads + head_of(k)] = tm[k];
        }
        soft_sync(kBarXch);
        // lane h < 16: the new reference of head h and the factor for what was
        // accumulated against the old one (the same in every warp)
        float alpha = 1.f;
        if (lane < kHeads) {
          const float tmax = fmaxf(fmaxf(xmax[lane], xmax[kHeads + lane]),
                                   fmaxf(xmax[2 * kHeads + lane], xmax[3 * kHeads + lane]));
          if (m16 == -INFINITY) {
            m16 = tmax;
            alpha = 0.f;
          } else if (tmax > m16 + kLazyLog2) {
            alpha = ex2_approx(m16 - tmax);
            m16 = tmax;
          }
        }
#pragma unroll
        for (int k = 0; k < 4; ++k) m_ref[k] = __shfl_sync(0xffffffffu, m16, head_of(k));
        if (!t.first && __any_sync(0xffffffffu, lane < kHeads && alpha != 1.f)) {
          // O^T and the running sums were accumulated against the old
          // reference: the previous tile's output MMA must be complete first
          // (completion n of pfree[b] is output MMA n kNP + b)
          const int pv = (it - 1) % kNP;
          ok = warp_wait(smem_u32(&bars.pfree[pv]), ((it - 1) / kNP) & 1, abort_flag, wait_ns);
          if (ok) {
            tc_fence_after();
            float o[32];
            tmem_ld32(tq + C::COL_O, o);
            tmem_wait_ld();
#pragma unroll
            for (int c = 0; c < 32; ++c) o[c] *= __shfl_sync(0xffffffffu, alpha, c & 15);
            tmem_st32(tq + C::COL_O, o);
            tmem_wait_st();
#pragma unroll
            for (int k = 0; k < 4; ++k) {
              const float a = __shfl_sync(0xffffffffu, alpha, head_of(k));
              l_acc[k] *= a;
              bmu_acc[k] *= a;
            }
          }
        }
      }
      // the P' buffer of this tile is free once the output MMA kNP tiles back
      // has read it
      ok = ok && warp_wait(smem_u32(&bars.pfree[pb]), ((it / kNP) & 1) ^ 1, abort_flag, wait_ns);
      tr.mark(5, it);
      if (ok) {
        // The output MMA sees the bf16-rounded weights P'; the denominator and
        // the mean correction use the same rounded values (l = sum P'/r), so
        // the rounding of P' cancels in o = (sum P' z - sum P' mu) / l.
        // P'[token][head] as an MN-major B operand: element (head n, token k)
        // at (k / 8) 256 + (n / 8) 128 + (k % 8) 16 + (n % 8) 2.
        uint8_t* pbuf = smem + C::OFF_PBUF + pb * C::PBUF;
#pragma unroll
        for (int e = 0; e < 2; ++e) {
          const int r = e ? r1 : r0;
          const float ri = GATE ? 1.f / rr[e] : 1.f;
          float pq[4];
#pragma unroll
          for (int k = 0; k < 4; ++k) pq[k] = ex2_approx(s[e][k] - m_ref[k]) * rr[e];
#pragma unroll
          for (int hp = 0; hp < 2; ++hp) {
            const uint32_t pw = pack_bf16x2(pq[2 * hp], pq[2 * hp + 1]);
            const float2 pr = unpack_bf16x2(pw);
            if (GATE) {
              l_acc[2 * hp] = fmaf(pr.x, ri, l_acc[2 * hp]);
              l_acc[2 * hp + 1] = fmaf(pr.y, ri, l_acc[2 * hp + 1]);
              bmu_acc[2 * hp] = fmaf(pr.x, mu[e], bmu_acc[2 * hp]);
              bmu_acc[2 * hp + 1] = fmaf(pr.y, mu[e], bmu_acc[2 * hp + 1]);
            } else {
              l_acc[2 * hp] += pr.x;
              l_acc[2 * hp + 1] += pr.y;
            }
            *reinterpret_cast<uint32_t*>(pbuf + (r >> 3) * 256 + hp * 128 + (r & 7) * 16 + 4 * q) = pw;
          }
        }
        tr.mark(6, it);
        fence_proxy_async_smem();
        tc_fence_before();
        warp_arrive(smem_u32(&bars.spdone[pb]));
      }
      tr.mark(3, it);

      if (t.last) {
        // ---- segment end: l and sum_j P'_j mu_j of every head over the 64 token rows
#pragma unroll
        for (int o = 4; o < 32; o <<= 1)
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            l_acc[k] += __shfl_xor_sync(0xffffffffu, l_acc[k], o);
            bmu_acc[k] += __shfl_xor_sync(0xffffffffu, bmu_acc[k], o);
          }
        if (lane < 4) {
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            xsum[(warp * kHeads + head_of(k)) * 2] = l_acc[k];
            xsum[(warp * kHeads + head_of(k)) * 2 + 1] = bmu_acc[k];
          }
        }
        if (soft_vote(kBarXch, !ok)) break;   // uniform
        float lh = 0.f, bh = 0.f;   // head `lane` (lanes 0-15)
        if (lane < kHeads) {
#pragma unroll
          for (int ww = 0; ww < kSoftWarps; ++ww) {
            lh += xsum[(ww * kHeads + lane) * 2];
            bh += xsum[(ww * kHeads + lane) * 2 + 1];
          }
        }
        // the segment's last output MMA (the earlier ones complete before it;
        // completion n of pfree[b] is output MMA n kNP + b), then O^T
        ok = warp_wait(smem_u32(&bars.pfree[pb]), (it / kNP) & 1, abort_flag, wait_ns);
        if (ok) {
          tc_fence_after();
          float o[32];
          tmem_ld32(tq + C::COL_O, o);
          tmem_wait_ld();
          const int slot_out = blockIdx.x + t.b;
          float* po = p.part_o + static_cast<size_t>(slot_out) * kHeads * D_C;
#pragma unroll
          for (int mc = 0; mc < 2; ++mc) {
            const int f = C::mc_start(mc) + 32 * warp + lane;
            if (mc == 0 || C::mc_start(1) + 32 * warp >= 128) {   // uniform in the warp
              float gm = 1.f, bt = 0.f;
              if (GATE) {
                gm = gb[f];
                bt = gb[D_C + f];
              }
#pragma unroll
              for (int h = 0; h < kHeads; ++h) {
                float v = o[mc * kHeads + h];
                if (GATE) {
                  const float lhh = __shfl_sync(0xffffffffu, lh, h), bhh = __shfl_sync(0xffffffffu, bh, h);
                  v = fmaf(gm, v - bhh, bt * lhh);
                }
                po[h * D_C + f] = v;
              }
            }
          }
          tc_fence_before();
          if (warp == 0 && lane < kHeads) {
            float* ml = p.part_ml + (static_cast<size_t>(slot_out) * kHeads + lane) * 2;
            ml[0] = m16;
            ml[1] = lh;
          }
          if (p.fuse && p.cmb_g == 1) {
            // one sequence per combine unit: release this warp's part of the
            // partial to the wait on its sequence (the warp barrier orders every
            // lane's stores before lane 0's fence)
            __syncwarp();
            if (lane == 0) {
              __threadfence();
              atomicAdd(p.seq_done + 1 + t.b, 1u);
            }
          }
        }
        tr.mark(4, it);
        // the next segment starts from scratch
        m16 = -INFINITY;
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          m_ref[k] = -INFINITY;
          l_acc[k] = 0.f;
          bmu_acc[k] = 0.f;
        }
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
  if (!DUMP && p.fuse) fused_combine<D_C, DBG == 2>(p, smem, bars);
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
  p.starts = reinterpret_cast<const SplitStart*>(ws + wl.off_start);
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
  p.wait_ns = a.wait_ns;
  p.stall_cta = a.stall_cta;
  p.stall_tile = a.stall_tile;
  // (the fused combine holds kCombineRowsPerWarp rows of W_UV,h per warp)
  p.fuse = DBG != 1 && a.batch > 0 && a.d_v <= kCombineRowsPerWarp * (kThreads / 32) &&
           a.num_splits <= resident_ctas(kern, C::SMEM);
  if (fused) *fused = p.fuse != 0;
  // The kernel may start while the query-absorption kernel before it on the
  // stream still runs (programmatic stream serialisation): its setup then
  // overlaps that kernel's tail, and grid_dependency_wait orders the rest.
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(a.num_splits);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = C::SMEM;
  cfg.stream = st;
  cudaLaunchAttribute attr[2];
  int na = 0;
  if (p.fuse) {
    attr[na].id = cudaLaunchAttributeCooperative;
    attr[na].val.cooperative = 1;
    ++na;
  }
  attr[na].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[na].val.programmaticStreamSerializationAllowed = 1;
  ++na;
  cfg.attrs = attr;
  cfg.numAttrs = na;
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
