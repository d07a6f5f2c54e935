// egmla_kernels.h - internal launch interface between the C-ABI layer
// (egmla_api.cu) and the kernels.  Not part of the public ABI.
#pragma once
#include <cuda.h>
#include <cuda_runtime.h>

#include <cstddef>
#include <cstdint>

namespace egmla {

struct AppendArgs {
  void* c_pool;
  void* kr_pool;
  int32_t* id_pool;
  const void* c_new;
  const void* kr_new;
  const int32_t* ids_new;
  const int32_t* block_table;
  int max_pages;
  const int32_t* positions;
  int batch, num_pages, page_size;
  int c_row_bytes, kr_row_bytes;
  int32_t* status;
};

// roles recorded by the decode kernel's event trace (eg_mla_debug_set_trace)
constexpr int kTraceRoles = 5;

struct DecodeArgs {
  // shapes
  int H, d_nope, d_rope, d_v, d_c, page_size, vocab;
  int dtype;  // 0 bf16, 1 fp32
  int gate;      // 0 none, 1 gated (the three gate modes below)
  int gate_add;  // gate by c + g (EG_MLA_GATE_ADD_LN) instead of c (*) g
  int gate_ln;   // LayerNorm after the gate (EG_MLA_GATE_MUL_LN, EG_MLA_GATE_ADD_LN)
  float scale_log2;  // softmax scale * log2(e)
  float eps;
  // tensors
  const void* q;
  const void* c_pool;
  const void* kr_pool;
  const int32_t* id_pool;
  const int32_t* block_table;
  int max_pages;
  const int32_t* seq_lens;
  int max_seq_len;
  int batch, num_pages;
  const void* gate_table;
  const float* ln_gamma;
  const float* ln_beta;
  const void* w_uk;
  const void* w_uv;
  void* out;
  int num_splits;
  void* workspace;
  int32_t* status;
  // cache-read test entry outputs (eg_mla_debug_gather)
  void* dump_c;
  void* dump_kr;
  int32_t* dump_ids;
  void* dump_g;
  // pipeline event trace of the decode kernel (eg_mla_debug_set_trace)
  void* trace;
  int trace_ctas, trace_cap;
  // limit of every pipeline wait (ns), and a withheld page copy of the
  // tensor-core decode kernel (eg_mla_debug_set_fault; stall_cta < 0: none)
  uint64_t wait_ns;
  int stall_cta, stall_tile;
};

cudaError_t launch_append(const AppendArgs& a, cudaStream_t st);
// query absorption and split schedule; with `app` non-null its blocks also
// append the new token of every sequence (the pools are read by no block of it)
cudaError_t launch_prologue_tc(const DecodeArgs& a, const AppendArgs* app, cudaStream_t st);
cudaError_t launch_decode_f32(const DecodeArgs& a, cudaStream_t st);
cudaError_t launch_combine(const DecodeArgs& a, bool tc_path, cudaStream_t st);
// tensor-core split-KV kernel; `maps` = {c_pool map (3-D page box for d_c <= 256), kr_pool map}.
// *fused (may be null) is set when the split combine ran inside the kernel
// (cooperative launch); otherwise launch_combine must follow.
cudaError_t launch_decode_tc(const DecodeArgs& a, const CUtensorMap* maps, bool dump, cudaStream_t st,
                             bool* fused);
// d_c = 512 without the gate (output accumulated with latent features in TMEM lanes)
cudaError_t launch_decode_wide(const DecodeArgs& a, const CUtensorMap* maps, cudaStream_t st);
// true if the bf16 tensor-core path has a kernel for these shapes
bool tc_supported(int d_c, int gate);

// R0 decode (egmla_r0.cu): bf16, 16 heads, d_n = d_v = 128, d_r = 64,
// d_c in {192, 256}
struct R0Args {
  const void* q;
  const void* c_pool;
  const void* kr_pool;
  const int32_t* id_pool;
  const int32_t* block_table;
  const int32_t* seq_lens;
  const void* w_ukv;     // [16 * 256, d_c]: per head its 128 key rows, then its 128 value rows
  const void* gate_r0;   // [vocab, 4096]
  const float* ln_gamma;
  const float* ln_beta;
  void* out;
  void* workspace;
  int32_t* status;
  int d_c, vocab, batch, max_pages, num_pages;
  float eps, scale_log2;
};
size_t r0_workspace_bytes(int batch, int max_pages, int num_pages);
cudaError_t launch_decode_r0(const R0Args& a, cudaStream_t st);
// Prefill (egmla_prefill.cu): bf16, d_n = d_v = 128, d_r = 64, d_c a
// multiple of 64 up to 512, any head count.  Prompts packed row after row
// (cu_seqlens [batch + 1] on the device); the pool pointers may be null (no
// cache write).
struct PrefillArgs {
  const void* q;            // [total, H, d_n + d_r]
  const void* c;            // [total, d_c]
  const void* kr;           // [total, d_r]
  const int32_t* ids;       // [total]
  const int32_t* cu_seqlens;
  const void* gate_table;
  const float* ln_gamma;
  const float* ln_beta;
  const void* w_uk;
  const void* w_uv;
  void* out;                // [total, H, d_v]
  void* c_pool;
  void* kr_pool;
  int32_t* id_pool;
  const int32_t* block_table;
  void* workspace;
  int32_t* status;
  int H, d_c, vocab, batch, total, max_seq_len, max_pages, num_pages;
  int gate, gate_add, gate_ln;
  float eps, scale_log2;
};
size_t prefill_workspace_bytes(int batch, int total_tokens, int H, int d_c);
bool prefill_supported(int d_nope, int d_rope, int d_v, int d_c);
// `mark` (may be null) is called with (stream, true) just before the
// attention kernel's launch and (stream, false) just after it.
cudaError_t launch_prefill(const PrefillArgs& a, cudaStream_t st, void (*mark)(cudaStream_t, bool));
// The gate table G = E W^UE^T (Section 3 Eqs. 3-4 for every vocabulary
// entry): E [vocab, d_e], W^UE [d_c, d_e] bf16 row-major, G [vocab, d_c] bf16;
// d_e a multiple of 64 up to 512, d_c a multiple of 64 (egmla_prefill.cu).
cudaError_t launch_gate_table(const void* emb, const void* w_ue, int vocab, int d_e, int d_c, void* table,
                              int32_t* status, cudaStream_t st);
// out[b][n] = sum_k x[b][k] W[n][k] for b < batch, n < n_out: W [n_out, k] and
// x [batch, k] bf16 row-major (16-byte aligned, k % 8 == 0), out fp32 or
// bf16 with row stride ldo elements (egmla_linear.cu).  Launched with
// programmatic stream serialisation: the weight copies may start while the
// kernel before it on the stream still runs.
cudaError_t launch_linear_tc(const void* w, int n_out, int k, const void* x, int batch, void* out, int ldo,
                             bool out_f32, int32_t* status, cudaStream_t st);
// the launch shape launch_linear_tc picks: cluster size (CTAs splitting k),
// ring stages, and the clusters of that size the device holds at once
cudaError_t linear_tc_plan(int n_out, int k, int batch, int* cluster, int* stages, int* max_clusters);

}  // namespace egmla
