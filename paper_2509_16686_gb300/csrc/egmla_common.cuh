// egmla_common.cuh - launch-independent pieces shared by the decode kernels:
// the workspace layout and the split-KV work schedule.
//
// Split-KV schedule.  The work is counted in units: the cache pages of every
// sequence plus kSegCost per non-empty sequence (what a split pays to take in
// a sequence).  The units of all sequences are numbered globally in sequence
// order (prefix sums cu[b]) and cut into `num_splits` equal contiguous ranges
// of `chunk` units, one per CTA.  A
// CTA may therefore cover the tail of one sequence and the head of the next;
// it emits one partial result (running max m, denominator l, un-normalised
// latent output) per sequence it touches.  Partial slot of (CTA c, sequence b)
// is c + b: the CTA ranges of consecutive sequences overlap in at most one CTA,
// so these slots never collide and there are at most num_splits + batch of them.
#pragma once
#include <cstddef>
#include <cstdint>

namespace egmla {

constexpr int kPage = 64;

__host__ __device__ inline size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// Per-sequence prepared query block of the tensor-core path: q^ (*) gamma
// [16 heads x d_c] and q^R [16 x d_rope] as bf16 MMA operands in 8x8 core
// matrices, then, per chunk of kSumFeatures latent features, the per-head fp32
// partial sums of w_h = sum_f bf16(q^ gamma)_hf and b_h = q^_h . beta
// ([d_c / kSumFeatures][2][16] floats; the consumer adds the chunks in order,
// so the result does not depend on launch order).  Every group of 8 columns
// (one K core of the operand, 256 bytes) holds heads 0-7 in its first 128
// bytes and heads 8-15 in its second: read as the N = 16 B operand of the
// score MMA (K-major, no swizzle) the K cores are 256 B apart and the two
// 8-head row groups 128 B apart.
constexpr int kQGroupBytes = 256;
constexpr int kQRowGroupBytes = 128;
__host__ __device__ constexpr size_t qop_offset(int h, int k) {
  return static_cast<size_t>(k / 8) * kQGroupBytes + (h / 8) * kQRowGroupBytes + (h % 8) * 16 + (k % 8) * 2;
}
__host__ __device__ constexpr size_t qprep_lat_bytes(int d_c) { return static_cast<size_t>(d_c / 8) * kQGroupBytes; }
__host__ __device__ constexpr size_t qprep_rope_bytes(int d_rope) {
  return static_cast<size_t>(d_rope / 8) * kQGroupBytes;
}
constexpr int kSumFeatures = 32;
__host__ __device__ constexpr size_t qprep_sums_bytes(int d_c) {
  return static_cast<size_t>(d_c / kSumFeatures) * 2 * 16 * 4;
}
__host__ __device__ constexpr size_t qprep_bytes_tc(int d_c, int d_rope) {
  return qprep_lat_bytes(d_c) + qprep_rope_bytes(d_rope) + qprep_sums_bytes(d_c);
}

// fp32 path: q^ [H, d_c] and q^R [H, d_rope] in fp32.
__host__ __device__ inline size_t qprep_bytes_f32(int H, int d_c, int d_rope) {
  return align_up(static_cast<size_t>(H) * (d_c + d_rope) * 4, 16);
}

// Where a split's page walk starts, written by the prologue kernel, so that
// each role of the decode kernel reads it with one round of loads instead of
// searching the prefix sums: the sequence b, the split's first page lp and
// end lp_end in it, the sequence length L, the split's end unit g1, whether
// the split is empty, and the physical ids of the first npages pages of the
// walk (at most kStartPages, all in sequence b).
constexpr int kStartPages = 8;
struct alignas(16) SplitStart {
  int32_t b, lp, lp_end, L, g1, done, npages, pad;
  int32_t page[kStartPages];
};
static_assert(sizeof(SplitStart) == 64, "split start record");

struct WorkspaceLayout {
  size_t off_cu, off_done, off_start, off_qprep, off_ml, off_o, total;
  size_t qprep_stride;
  int num_slots;
};

__host__ __device__ inline WorkspaceLayout workspace_layout(int batch, int num_splits, int H, int d_c,
                                                            int d_rope, bool tc_path) {
  WorkspaceLayout w;
  w.num_slots = num_splits + batch;
  w.qprep_stride = tc_path ? qprep_bytes_tc(d_c, d_rope) : qprep_bytes_f32(H, d_c, d_rope);
  size_t off = 0;
  w.off_cu = off;
  off = align_up(off + static_cast<size_t>(batch + 1) * 4, 256);
  // the fused combine's counters (zeroed by the prologue each call): [0] the
  // CTAs done, [1 + b] the split partials of sequence b stored
  w.off_done = off;
  off = align_up(off + static_cast<size_t>(batch + 1) * 4, 256);
  w.off_start = off;
  off = align_up(off + static_cast<size_t>(num_splits) * sizeof(SplitStart), 256);
  w.off_qprep = off;
  off = align_up(off + static_cast<size_t>(batch) * w.qprep_stride, 256);
  w.off_ml = off;
  off = align_up(off + static_cast<size_t>(w.num_slots) * H * 2 * 4, 256);
  w.off_o = off;
  off = align_up(off + static_cast<size_t>(w.num_slots) * H * d_c * 4, 256);
  w.total = off;
  return w;
}

// Split-KV schedule.  The splits share the work in units: one per cache page,
// plus kSegCost for the start of every non-empty sequence (the per-sequence cost
// of a split: loading the query block, reading out and storing the partial
// output), so that splits that take in more sequences get fewer pages.  cu[b]
// is the first unit of sequence b; its pages are units cu[b] + kSegCost + i,
// i < ceil(L_b / page); split c owns units [c chunk, (c + 1) chunk).
constexpr int kSegCost = 1;

// units per split for the total unit count
__host__ __device__ inline int split_chunk(int total_pages, int num_splits) {
  int c = (total_pages + num_splits - 1) / num_splits;
  return c < 1 ? 1 : c;
}

// first sequence whose page range contains global page g (cu has batch+1 entries,
// non-decreasing, cu[0] = 0, g < cu[batch])
__device__ inline int find_sequence(const int32_t* cu, int batch, int g) {
  int lo = 0, hi = batch - 1;
  while (lo < hi) {
    int mid = (lo + hi + 1) >> 1;
    if (__ldg(cu + mid) <= g) lo = mid; else hi = mid - 1;
  }
  // skip empty sequences that share the same start
  while (lo < batch - 1 && __ldg(cu + lo + 1) <= g) ++lo;
  return lo;
}

}  // namespace egmla
