// egmla_api.cu - the C ABI of libegmla: argument validation, workspace
// carving, TMA descriptor encoding and kernel launches.  See include/egmla.h
// for the contract of every entry point.
#include <cuda.h>
#include <cuda_runtime.h>

#include <cmath>
#include <cstdint>
#include <cstring>
#include <mutex>
#include <vector>

#include "../../include/egmla.h"
#include "egmla_common.cuh"
#include "egmla_kernels.h"
#include "egmla_ptx.cuh"

namespace {

using egmla::DecodeArgs;

bool aligned(const void* p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

int elem_bytes(const eg_mla_dims* d) { return d->dtype == EG_MLA_BF16 ? 2 : 4; }

bool is_tc_path(const eg_mla_dims* d) { return d->dtype == EG_MLA_BF16; }

// shape support; returns EG_MLA_OK or the error code
int check_dims(const eg_mla_dims* d) {
  if (d == nullptr) return EG_MLA_ERR_INVALID_ARG;
  if (d->num_heads <= 0 || d->d_nope <= 0 || d->d_rope <= 0 || d->d_v <= 0 || d->d_c <= 0 ||
      d->page_size <= 0 || d->vocab <= 0)
    return EG_MLA_ERR_INVALID_ARG;
  if (d->gate_mode < EG_MLA_GATE_NONE || d->gate_mode > EG_MLA_GATE_ADD_LN) return EG_MLA_ERR_INVALID_ARG;
  if (d->page_size != egmla::kPage) return EG_MLA_ERR_UNSUPPORTED;
  if (d->dtype == EG_MLA_BF16) {
    if (d->num_heads != 16 || d->d_rope != 64) return EG_MLA_ERR_UNSUPPORTED;
    if (!egmla::tc_supported(d->d_c, d->gate_mode)) return EG_MLA_ERR_UNSUPPORTED;
    if (d->d_nope % 8 || d->d_nope > 256 || d->d_v % 8 || d->d_v > 256) return EG_MLA_ERR_UNSUPPORTED;
    return EG_MLA_OK;
  }
  if (d->dtype == EG_MLA_FP32) {
    if (d->num_heads > 16 || d->d_c > 512 || d->d_c % 4 || d->d_rope > 64 || d->d_rope % 4 ||
        d->d_nope > 256 || d->d_v > 256)
      return EG_MLA_ERR_UNSUPPORTED;
    return EG_MLA_OK;
  }
  return EG_MLA_ERR_INVALID_ARG;
}

int resolve_splits(int32_t num_splits, int32_t* out) {
  if (num_splits < 0) return EG_MLA_ERR_INVALID_ARG;
  if (num_splits > 0) {
    *out = num_splits;
    return EG_MLA_OK;
  }
  int dev = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return EG_MLA_ERR_CUDA;
  if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return EG_MLA_ERR_CUDA;
  *out = sms > 0 ? sms : 1;
  return EG_MLA_OK;
}

// cuTensorMapEncodeTiled through the runtime's driver entry point (no libcuda link)
using EncodeFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                              const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                              CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeFn get_encode() {
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

// 2D view [rows, cols] of a bf16 pool, boxes of 64 columns (128 bytes) x 64 rows,
// 128-byte swizzle (the layout the MMA descriptors of the decode kernel expect)
bool encode_pool_map(CUtensorMap* map, const void* base, uint64_t rows, uint64_t cols) {
  EncodeFn enc = get_encode();
  if (enc == nullptr) return false;
  const cuuint64_t dims[2] = {cols, rows};
  const cuuint64_t strides[1] = {cols * 2};
  const cuuint32_t box[2] = {64, 64};
  const cuuint32_t estr[2] = {1, 1};
  return enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Latent pool as one 3-D box per page for the d_c <= 256 kernel: dims
// {64 features, rows, d_c / 64 feature columns}, so that one copy writes the
// page as its 128-byte-swizzled 64-feature columns one after another.
bool encode_page_map_3d(CUtensorMap* map, const void* base, uint64_t rows, uint64_t cols) {
  EncodeFn enc = get_encode();
  if (enc == nullptr) return false;
  const cuuint64_t dims[3] = {64, rows, cols / 64};
  const cuuint64_t strides[2] = {cols * 2, 128};
  const cuuint32_t box[3] = {64, 64, static_cast<cuuint32_t>(cols / 64)};
  const cuuint32_t estr[3] = {1, 1, 1};
  return enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box, estr,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// maps = {latent pool (3-D page box for d_c <= 256, 64x64 boxes otherwise), RoPE-key pool}
bool encode_decode_maps(CUtensorMap (&maps)[2], const eg_mla_dims* d, const void* c_pool, const void* krope_pool,
                        int32_t num_pages) {
  std::memset(maps, 0, sizeof(maps));
  const uint64_t rows = static_cast<uint64_t>(num_pages) * d->page_size;
  const bool paged3d = d->d_c <= 256;
  if (!(paged3d ? encode_page_map_3d(&maps[0], c_pool, rows, d->d_c) : encode_pool_map(&maps[0], c_pool, rows, d->d_c)))
    return false;
  return encode_pool_map(&maps[1], krope_pool, rows, d->d_rope);
}

float resolve_scale(const eg_mla_dims* d) {
  return d->softmax_scale > 0.f ? d->softmax_scale : 1.0f / std::sqrt(static_cast<float>(d->d_nope + d->d_rope));
}

int fill_decode_args(DecodeArgs& a, const eg_mla_dims* d, const void* c_pool, const void* krope_pool,
                     const int32_t* id_pool, const int32_t* block_table, int32_t max_pages,
                     const int32_t* seq_lens, int32_t max_seq_len, int32_t batch, int32_t num_pages,
                     const void* gate_table, int32_t num_splits, void* workspace, size_t workspace_bytes,
                     int32_t* dev_status) {
  int rc = check_dims(d);
  if (rc != EG_MLA_OK) return rc;
  if (batch < 0 || num_pages <= 0 || max_pages <= 0 || max_seq_len < 0) return EG_MLA_ERR_INVALID_ARG;
  if (static_cast<int64_t>(max_seq_len) > static_cast<int64_t>(max_pages) * d->page_size)
    return EG_MLA_ERR_INVALID_ARG;
  if (static_cast<int64_t>(num_pages) * d->page_size > INT32_MAX) return EG_MLA_ERR_UNSUPPORTED;
  if (c_pool == nullptr || krope_pool == nullptr || block_table == nullptr || seq_lens == nullptr)
    return EG_MLA_ERR_INVALID_ARG;
  if (d->gate_mode != EG_MLA_GATE_NONE && (id_pool == nullptr || gate_table == nullptr))
    return EG_MLA_ERR_INVALID_ARG;
  // the bf16 kernels read gate rows in 32-byte pieces
  const size_t g_align = is_tc_path(d) ? 32 : 16;
  if (!aligned(c_pool, 16) || !aligned(krope_pool, 16) || (id_pool && !aligned(id_pool, 16)) ||
      (gate_table && d->gate_mode != EG_MLA_GATE_NONE && !aligned(gate_table, g_align)))
    return EG_MLA_ERR_INVALID_ARG;
  int32_t splits = 0;
  rc = resolve_splits(num_splits, &splits);
  if (rc != EG_MLA_OK) return rc;
  const egmla::WorkspaceLayout wl =
      egmla::workspace_layout(batch, splits, d->num_heads, d->d_c, d->d_rope, is_tc_path(d));
  if (workspace == nullptr || workspace_bytes < wl.total || !aligned(workspace, 256)) return EG_MLA_ERR_WORKSPACE;
  std::memset(&a, 0, sizeof(a));
  a.H = d->num_heads;
  a.d_nope = d->d_nope;
  a.d_rope = d->d_rope;
  a.d_v = d->d_v;
  a.d_c = d->d_c;
  a.page_size = d->page_size;
  a.vocab = d->vocab;
  a.dtype = d->dtype;
  a.gate = d->gate_mode != EG_MLA_GATE_NONE ? 1 : 0;
  a.gate_add = d->gate_mode == EG_MLA_GATE_ADD_LN ? 1 : 0;
  a.gate_ln = (d->gate_mode == EG_MLA_GATE_MUL_LN || d->gate_mode == EG_MLA_GATE_ADD_LN) ? 1 : 0;
  a.scale_log2 = resolve_scale(d) * 1.4426950408889634f;
  a.eps = d->ln_eps > 0.f ? d->ln_eps : 1e-5f;
  a.c_pool = c_pool;
  a.kr_pool = krope_pool;
  a.id_pool = id_pool;
  a.block_table = block_table;
  a.max_pages = max_pages;
  a.seq_lens = seq_lens;
  a.max_seq_len = max_seq_len;
  a.batch = batch;
  a.num_pages = num_pages;
  a.gate_table = gate_table;
  a.num_splits = splits;
  a.workspace = workspace;
  a.status = dev_status;
  a.wait_ns = egmla::kWaitLimitNs;
  a.stall_cta = a.stall_tile = -1;
  return EG_MLA_OK;
}

int to_status(cudaError_t e) { return e == cudaSuccess ? EG_MLA_OK : EG_MLA_ERR_CUDA; }

// per-launch event pairs around the split-KV kernel (eg_mla_profile_begin/end)
struct Profiler {
  std::mutex mu;
  bool active = false;
  std::vector<cudaEvent_t> ev;  // 2 per launch
  int used = 0;
} g_prof;

// optional pipeline trace buffer for the decode kernel (eg_mla_debug_set_trace)
struct TraceCfg {
  std::mutex mu;
  void* buf = nullptr;
  int ctas = 0, cap = 0;
} g_trace;

void apply_trace(DecodeArgs& a) {
  std::lock_guard<std::mutex> lk(g_trace.mu);
  a.trace = g_trace.buf;
  a.trace_ctas = g_trace.ctas;
  a.trace_cap = g_trace.cap;
}

// test entry eg_mla_debug_set_fault: a withheld page copy and a lowered wait limit
struct FaultCfg {
  std::mutex mu;
  int cta = -1, tile = -1;
  uint64_t wait_ns = egmla::kWaitLimitNs;
} g_fault;

void apply_fault(DecodeArgs& a) {
  std::lock_guard<std::mutex> lk(g_fault.mu);
  a.wait_ns = g_fault.wait_ns;
  a.stall_cta = g_fault.cta;
  a.stall_tile = g_fault.tile;
}

// Records a profiling event on the launching stream; under stream capture it
// becomes an event-record node of the graph (timestamped at each replay).
void prof_record(cudaEvent_t e, cudaStream_t st) {
  cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
  if (cudaStreamIsCapturing(st, &cs) == cudaSuccess && cs == cudaStreamCaptureStatusActive)
    cudaEventRecordWithFlags(e, st, cudaEventRecordExternal);
  else
    cudaEventRecord(e, st);
}

void prof_mark(cudaStream_t st, bool before) {
  std::lock_guard<std::mutex> lk(g_prof.mu);
  if (!g_prof.active) return;
  const int pairs = static_cast<int>(g_prof.ev.size() / 2);
  if (before) {
    if (g_prof.used < pairs) prof_record(g_prof.ev[2 * g_prof.used], st);
  } else if (g_prof.used < pairs) {
    prof_record(g_prof.ev[2 * g_prof.used + 1], st);
    ++g_prof.used;
  }
}

// Static scratch of eg_mla_decode_static.  Callers that cannot hand the
// decode a workspace (an engine that reserved all free HBM for the paged
// latent cache at start-up, or a C caller without a caching allocator, whose
// per-step cudaFree would synchronise the device inside the token loop) get
// this module-owned array instead; no call allocates or frees device memory.
// Nothing in it needs to start at zero: the prologue writes the page prefix
// sums and prepared queries, the split-KV kernel writes every partial slot the
// combine reads, all within the same call.  One array per device, so calls
// whose kernels overlap on one device race on it.
static __device__ __align__(256) unsigned char g_static_scratch[EG_MLA_STATIC_SCRATCH_BYTES];

constexpr int kMaxDevices = 64;

// device address of g_static_scratch, looked up with the device current and
// cached together with the id of the context it belongs to: a context made
// after cudaDeviceReset gets a new id (and possibly a new address), so the
// first call in it looks the address up again.  A lookup may load the module,
// so the first call in each context belongs before any stream capture.
using CtxGetCurrentFn = CUresult (*)(CUcontext*);
using CtxGetIdFn = CUresult (*)(CUcontext, unsigned long long*);

struct StaticScratch {
  std::mutex mu;
  void* ptr[kMaxDevices] = {};
  unsigned long long ctx_id[kMaxDevices] = {};
  CtxGetCurrentFn get_current = nullptr;
  CtxGetIdFn get_id = nullptr;
  bool resolved = false;
} g_static;

template <typename Fn>
Fn driver_fn(const char* name) {
  void* p = nullptr;
  cudaDriverEntryPointQueryResult q;
  if (cudaGetDriverEntryPointByVersion(name, &p, 12000, cudaEnableDefault, &q) != cudaSuccess ||
      q != cudaDriverEntryPointSuccess)
    return nullptr;
  return reinterpret_cast<Fn>(p);
}

int static_scratch(void** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return EG_MLA_ERR_CUDA;
  if (dev < 0 || dev >= kMaxDevices) return EG_MLA_ERR_UNSUPPORTED;
  std::lock_guard<std::mutex> lk(g_static.mu);
  if (!g_static.resolved) {
    g_static.get_current = driver_fn<CtxGetCurrentFn>("cuCtxGetCurrent");
    g_static.get_id = driver_fn<CtxGetIdFn>("cuCtxGetId");
    g_static.resolved = true;
  }
  if (g_static.get_current == nullptr || g_static.get_id == nullptr) return EG_MLA_ERR_CUDA;
  CUcontext ctx = nullptr;
  unsigned long long id = 0;
  if (g_static.get_current(&ctx) != CUDA_SUCCESS) return EG_MLA_ERR_CUDA;
  if (ctx == nullptr) {
    // no context on this thread yet: have the runtime make the device's
    // primary context current
    if (cudaFree(nullptr) != cudaSuccess || g_static.get_current(&ctx) != CUDA_SUCCESS || ctx == nullptr)
      return EG_MLA_ERR_CUDA;
  }
  if (g_static.get_id(ctx, &id) != CUDA_SUCCESS) return EG_MLA_ERR_CUDA;
  if (g_static.ptr[dev] == nullptr || g_static.ctx_id[dev] != id) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_static_scratch) != cudaSuccess || p == nullptr) return EG_MLA_ERR_CUDA;
    g_static.ptr[dev] = p;
    g_static.ctx_id[dev] = id;
  }
  *out = g_static.ptr[dev];
  return EG_MLA_OK;
}

// argument checks and launch record of one append (eg_mla_append_latent)
int fill_append_args(egmla::AppendArgs& a, const eg_mla_dims* dims, void* c_pool, void* krope_pool,
                     int32_t* id_pool, const void* c_new, const void* krope_new, const int32_t* ids_new,
                     const int32_t* block_table, int32_t max_pages_per_seq, const int32_t* positions,
                     int32_t batch, int32_t num_pages, int32_t* dev_status) {
  int rc = check_dims(dims);
  if (rc != EG_MLA_OK) return rc;
  if (batch < 0 || num_pages <= 0 || max_pages_per_seq <= 0) return EG_MLA_ERR_INVALID_ARG;
  std::memset(&a, 0, sizeof(a));
  if (batch == 0) return EG_MLA_OK;
  if (!c_pool || !krope_pool || !c_new || !krope_new || !block_table || !positions) return EG_MLA_ERR_INVALID_ARG;
  const int eb = elem_bytes(dims);
  const int crb = dims->d_c * eb, krb = dims->d_rope * eb;
  if (crb % 16 || krb % 16) return EG_MLA_ERR_UNSUPPORTED;
  if (!aligned(c_pool, 16) || !aligned(krope_pool, 16) || !aligned(c_new, 16) || !aligned(krope_new, 16))
    return EG_MLA_ERR_INVALID_ARG;
  a.c_pool = c_pool;
  a.kr_pool = krope_pool;
  a.id_pool = id_pool;
  a.c_new = c_new;
  a.kr_new = krope_new;
  a.ids_new = ids_new;
  a.block_table = block_table;
  a.max_pages = max_pages_per_seq;
  a.positions = positions;
  a.batch = batch;
  a.num_pages = num_pages;
  a.page_size = dims->page_size;
  a.c_row_bytes = crb;
  a.kr_row_bytes = krb;
  a.status = dev_status;
  return EG_MLA_OK;
}

// eg_mla_decode, preceded by the append of `app` when it is non-null (in the
// query-absorption kernel's grid on the tensor-core path; as its own launch
// otherwise).  Every argument is checked before anything is launched.
int decode_impl(const eg_mla_dims* dims, const void* q, const void* c_pool, const void* krope_pool,
                const int32_t* id_pool, const int32_t* block_table, int32_t max_pages_per_seq,
                const int32_t* seq_lens, int32_t max_seq_len, int32_t batch, int32_t num_pages,
                const void* gate_table, const float* ln_gamma, const float* ln_beta, const void* w_uk,
                const void* w_uv, void* out, int32_t num_splits, void* workspace, size_t workspace_bytes,
                int32_t* dev_status, const egmla::AppendArgs* app, cudaStream_t st) {
  DecodeArgs a;
  int rc = fill_decode_args(a, dims, c_pool, krope_pool, id_pool, block_table, max_pages_per_seq, seq_lens,
                            max_seq_len, batch, num_pages, gate_table, num_splits, workspace, workspace_bytes,
                            dev_status);
  if (rc != EG_MLA_OK) return rc;
  if (batch == 0) return EG_MLA_OK;
  if (q == nullptr || w_uk == nullptr || w_uv == nullptr || out == nullptr) return EG_MLA_ERR_INVALID_ARG;
  // q, W_UK and W_UV rows are read in 16-byte pieces
  if (!aligned(w_uv, 16) || !aligned(w_uk, 16) || !aligned(q, 16)) return EG_MLA_ERR_INVALID_ARG;
  a.q = q;
  a.ln_gamma = ln_gamma;
  a.ln_beta = ln_beta;
  a.w_uk = w_uk;
  a.w_uv = w_uv;
  a.out = out;
  if (is_tc_path(dims)) {
    CUtensorMap maps[2];
    if (!encode_decode_maps(maps, dims, c_pool, krope_pool, num_pages)) return EG_MLA_ERR_CUDA;
    apply_trace(a);
    apply_fault(a);
    cudaError_t e = egmla::launch_prologue_tc(a, app, st);
    bool fused = false;
    if (e == cudaSuccess) {
      prof_mark(st, true);
      e = egmla::launch_decode_tc(a, maps, false, st, &fused);
      prof_mark(st, false);
    }
    if (e == cudaSuccess && !fused) e = egmla::launch_combine(a, true, st);
    return to_status(e);
  }
  cudaError_t e = app != nullptr ? egmla::launch_append(*app, st) : cudaSuccess;
  if (e == cudaSuccess) e = egmla::launch_decode_f32(a, st);
  if (e == cudaSuccess) e = egmla::launch_combine(a, false, st);
  return to_status(e);
}

}  // namespace

namespace {
// shapes the prefill kernels cover; EG_MLA_OK or the error code
int check_prefill_dims(const eg_mla_dims* d) {
  if (d == nullptr) return EG_MLA_ERR_INVALID_ARG;
  if (d->num_heads <= 0 || d->d_nope <= 0 || d->d_rope <= 0 || d->d_v <= 0 || d->d_c <= 0 ||
      d->page_size <= 0 || d->vocab <= 0)
    return EG_MLA_ERR_INVALID_ARG;
  if (d->gate_mode < EG_MLA_GATE_NONE || d->gate_mode > EG_MLA_GATE_ADD_LN) return EG_MLA_ERR_INVALID_ARG;
  if (d->dtype != EG_MLA_BF16 || d->page_size != egmla::kPage) return EG_MLA_ERR_UNSUPPORTED;
  if (!egmla::prefill_supported(d->d_nope, d->d_rope, d->d_v, d->d_c)) return EG_MLA_ERR_UNSUPPORTED;
  return EG_MLA_OK;
}
}  // namespace

extern "C" {

const char* eg_mla_status_string(int status) {
  switch (status) {
    case EG_MLA_OK: return "ok";
    case EG_MLA_ERR_INVALID_ARG: return "invalid argument";
    case EG_MLA_ERR_UNSUPPORTED: return "unsupported shape";
    case EG_MLA_ERR_CUDA: return "CUDA runtime error";
    case EG_MLA_ERR_OUT_OF_RANGE: return "page id or token id out of range";
    case EG_MLA_ERR_TIMEOUT: return "device pipeline wait timed out";
    case EG_MLA_ERR_WORKSPACE: return "workspace too small or misaligned";
    case EG_MLA_ERR_SCRATCH_LIMIT:
      return "problem needs more scratch than the static scratch array (EG_MLA_STATIC_SCRATCH_BYTES) holds";
    default: return "unknown status";
  }
}

int eg_mla_kv_bytes_per_token(const eg_mla_dims* dims, int32_t n_layers, int64_t* bytes_out) {
  if (dims == nullptr || bytes_out == nullptr || n_layers < 0) return EG_MLA_ERR_INVALID_ARG;
  if (dims->d_c <= 0 || dims->d_rope < 0) return EG_MLA_ERR_INVALID_ARG;
  const int64_t per_layer = static_cast<int64_t>(dims->d_c + dims->d_rope) * elem_bytes(dims) +
                            (dims->gate_mode != EG_MLA_GATE_NONE ? 4 : 0);
  *bytes_out = per_layer * n_layers;
  return EG_MLA_OK;
}

int eg_mla_default_num_splits(int32_t* out_splits) {
  if (out_splits == nullptr) return EG_MLA_ERR_INVALID_ARG;
  return resolve_splits(0, out_splits);
}

size_t eg_mla_decode_workspace_size(const eg_mla_dims* dims, int32_t batch, int32_t num_splits) {
  if (check_dims(dims) != EG_MLA_OK || batch < 0) return 0;
  int32_t splits = 0;
  if (resolve_splits(num_splits, &splits) != EG_MLA_OK) return 0;
  return egmla::workspace_layout(batch, splits, dims->num_heads, dims->d_c, dims->d_rope, is_tc_path(dims)).total;
}

int eg_mla_append_latent(const eg_mla_dims* dims, void* c_pool, void* krope_pool, int32_t* id_pool,
                         const void* c_new, const void* krope_new, const int32_t* ids_new,
                         const int32_t* block_table, int32_t max_pages_per_seq, const int32_t* positions,
                         int32_t batch, int32_t num_pages, int32_t* dev_status, void* stream) {
  egmla::AppendArgs a;
  const int rc = fill_append_args(a, dims, c_pool, krope_pool, id_pool, c_new, krope_new, ids_new, block_table,
                                  max_pages_per_seq, positions, batch, num_pages, dev_status);
  if (rc != EG_MLA_OK || batch == 0) return rc;
  return to_status(egmla::launch_append(a, static_cast<cudaStream_t>(stream)));
}

int eg_mla_decode(const eg_mla_dims* dims, const void* q, const void* c_pool, const void* krope_pool,
                  const int32_t* id_pool, const int32_t* block_table, int32_t max_pages_per_seq,
                  const int32_t* seq_lens, int32_t max_seq_len, int32_t batch, int32_t num_pages,
                  const void* gate_table, const float* ln_gamma, const float* ln_beta, const void* w_uk,
                  const void* w_uv, void* out, int32_t num_splits, void* workspace, size_t workspace_bytes,
                  int32_t* dev_status, void* stream) {
  return decode_impl(dims, q, c_pool, krope_pool, id_pool, block_table, max_pages_per_seq, seq_lens, max_seq_len,
                     batch, num_pages, gate_table, ln_gamma, ln_beta, w_uk, w_uv, out, num_splits, workspace,
                     workspace_bytes, dev_status, nullptr, static_cast<cudaStream_t>(stream));
}

int eg_mla_step(const eg_mla_dims* dims, void* c_pool, void* krope_pool, int32_t* id_pool, const void* c_new,
                const void* krope_new, const int32_t* ids_new, const int32_t* positions, const void* q,
                const int32_t* block_table, int32_t max_pages_per_seq, const int32_t* seq_lens,
                int32_t max_seq_len, int32_t batch, int32_t num_pages, const void* gate_table,
                const float* ln_gamma, const float* ln_beta, const void* w_uk, const void* w_uv, void* out,
                int32_t num_splits, void* workspace, size_t workspace_bytes, int32_t* dev_status, void* stream) {
  egmla::AppendArgs app;
  const int rc = fill_append_args(app, dims, c_pool, krope_pool, id_pool, c_new, krope_new, ids_new, block_table,
                                  max_pages_per_seq, positions, batch, num_pages, dev_status);
  if (rc != EG_MLA_OK) return rc;
  return decode_impl(dims, q, c_pool, krope_pool, id_pool, block_table, max_pages_per_seq, seq_lens, max_seq_len,
                     batch, num_pages, gate_table, ln_gamma, ln_beta, w_uk, w_uv, out, num_splits, workspace,
                     workspace_bytes, dev_status, &app, static_cast<cudaStream_t>(stream));
}

int eg_mla_decode_static(const eg_mla_dims* dims, const void* q, const void* c_pool, const void* krope_pool,
                         const int32_t* id_pool, const int32_t* block_table, int32_t max_pages_per_seq,
                         const int32_t* seq_lens, int32_t max_seq_len, int32_t batch, int32_t num_pages,
                         const void* gate_table, const float* ln_gamma, const float* ln_beta, const void* w_uk,
                         const void* w_uv, void* out, int32_t num_splits, int32_t* dev_status, void* stream) {
  int rc = check_dims(dims);
  if (rc != EG_MLA_OK) return rc;
  if (batch < 0 || num_splits < 0) return EG_MLA_ERR_INVALID_ARG;
  const size_t need = eg_mla_decode_workspace_size(dims, batch, num_splits);
  if (need == 0) return EG_MLA_ERR_CUDA;  // dims were checked: only the SM-count query can fail
  if (need > EG_MLA_STATIC_SCRATCH_BYTES) return EG_MLA_ERR_SCRATCH_LIMIT;
  void* scratch = nullptr;
  rc = static_scratch(&scratch);
  if (rc != EG_MLA_OK) return rc;
  return eg_mla_decode(dims, q, c_pool, krope_pool, id_pool, block_table, max_pages_per_seq, seq_lens, max_seq_len,
                       batch, num_pages, gate_table, ln_gamma, ln_beta, w_uk, w_uv, out, num_splits, scratch,
                       EG_MLA_STATIC_SCRATCH_BYTES, dev_status, stream);
}

size_t eg_mla_decode_r0_workspace_size(const eg_mla_dims* dims, int32_t batch, int32_t max_pages_per_seq,
                                       int32_t num_pages) {
  if (check_dims(dims) != EG_MLA_OK || num_pages <= 0 || batch < 0 || max_pages_per_seq <= 0) return 0;
  if (dims->dtype != EG_MLA_BF16 || dims->d_nope != 128 || dims->d_v != 128 || (dims->d_c != 192 && dims->d_c != 256))
    return 0;
  return egmla::r0_workspace_bytes(batch, max_pages_per_seq, num_pages);
}

int eg_mla_decode_r0(const eg_mla_dims* dims, const void* q, const void* c_pool, const void* krope_pool,
                     const int32_t* id_pool, const int32_t* block_table, int32_t max_pages_per_seq,
                     const int32_t* seq_lens, int32_t batch, int32_t num_pages, const void* w_ukv,
                     const void* gate_r0, const float* ln_gamma_r0, const float* ln_beta_r0, void* out,
                     void* workspace, size_t workspace_bytes, int32_t* dev_status, void* stream) {
  int rc = check_dims(dims);
  if (rc != EG_MLA_OK) return rc;
  if (dims->dtype != EG_MLA_BF16 || dims->d_nope != 128 || dims->d_v != 128 || (dims->d_c != 192 && dims->d_c != 256))
    return EG_MLA_ERR_UNSUPPORTED;
  if (batch < 0 || num_pages <= 0 || max_pages_per_seq <= 0) return EG_MLA_ERR_INVALID_ARG;
  if (batch == 0) return EG_MLA_OK;
  if (!q || !c_pool || !krope_pool || !id_pool || !block_table || !seq_lens || !w_ukv || !gate_r0 || !out)
    return EG_MLA_ERR_INVALID_ARG;
  if (!aligned(q, 16) || !aligned(c_pool, 16) || !aligned(krope_pool, 16) || !aligned(w_ukv, 16) ||
      !aligned(gate_r0, 16) || !aligned(out, 16))
    return EG_MLA_ERR_INVALID_ARG;
  if (static_cast<int64_t>(num_pages) * dims->page_size > INT32_MAX) return EG_MLA_ERR_UNSUPPORTED;
  if (workspace == nullptr || !aligned(workspace, 256) || workspace_bytes < egmla::r0_workspace_bytes(batch, max_pages_per_seq, num_pages))
    return EG_MLA_ERR_WORKSPACE;
  egmla::R0Args a;
  a.q = q;
  a.c_pool = c_pool;
  a.kr_pool = krope_pool;
  a.id_pool = id_pool;
  a.block_table = block_table;
  a.seq_lens = seq_lens;
  a.w_ukv = w_ukv;
  a.gate_r0 = gate_r0;
  a.ln_gamma = ln_gamma_r0;
  a.ln_beta = ln_beta_r0;
  a.out = out;
  a.workspace = workspace;
  a.status = dev_status;
  a.d_c = dims->d_c;
  a.vocab = dims->vocab;
  a.batch = batch;
  a.max_pages = max_pages_per_seq;
  a.num_pages = num_pages;
  a.eps = dims->ln_eps > 0.f ? dims->ln_eps : 1e-5f;
  a.scale_log2 = resolve_scale(dims) * 1.4426950408889634f;
  return to_status(egmla::launch_decode_r0(a, static_cast<cudaStream_t>(stream)));
}

size_t eg_mla_prefill_workspace_size(const eg_mla_dims* dims, int32_t batch, int32_t total_tokens) {
  if (check_prefill_dims(dims) != EG_MLA_OK || total_tokens < 0 || batch < 0) return 0;
  return egmla::prefill_workspace_bytes(batch, total_tokens, dims->num_heads, dims->d_c);
}

int eg_mla_prefill(const eg_mla_dims* dims, const void* q, const void* c_new, const void* krope_new,
                   const int32_t* ids_new, const int32_t* cu_seqlens, int32_t batch, int32_t total_tokens,
                   int32_t max_seq_len, const void* gate_table, const float* ln_gamma, const float* ln_beta,
                   const void* w_uk, const void* w_uv, void* out, void* c_pool, void* krope_pool,
                   int32_t* id_pool, const int32_t* block_table, int32_t max_pages_per_seq, int32_t num_pages,
                   void* workspace, size_t workspace_bytes, int32_t* dev_status, void* stream) {
  int rc = check_prefill_dims(dims);
  if (rc != EG_MLA_OK) return rc;
  if (batch < 0 || total_tokens < 0 || max_seq_len < 0) return EG_MLA_ERR_INVALID_ARG;
  if (batch == 0 || total_tokens == 0) return EG_MLA_OK;
  if (max_seq_len == 0 || max_seq_len > total_tokens) return EG_MLA_ERR_INVALID_ARG;
  const bool gated = dims->gate_mode != EG_MLA_GATE_NONE;
  if (!q || !c_new || !krope_new || !cu_seqlens || !w_uk || !w_uv || !out) return EG_MLA_ERR_INVALID_ARG;
  if (gated && (!ids_new || !gate_table)) return EG_MLA_ERR_INVALID_ARG;
  if (!aligned(q, 16) || !aligned(c_new, 16) || !aligned(krope_new, 16) || !aligned(w_uk, 16) ||
      !aligned(w_uv, 16) || !aligned(out, 16) || (gated && !aligned(gate_table, 16)))
    return EG_MLA_ERR_INVALID_ARG;
  if (c_pool != nullptr) {
    if (!krope_pool || !block_table || (gated && !id_pool) || max_pages_per_seq <= 0 || num_pages <= 0)
      return EG_MLA_ERR_INVALID_ARG;
    if (!aligned(c_pool, 16) || !aligned(krope_pool, 16)) return EG_MLA_ERR_INVALID_ARG;
    if (static_cast<int64_t>(num_pages) * dims->page_size > INT32_MAX) return EG_MLA_ERR_UNSUPPORTED;
  }
  const int64_t qtiles = (static_cast<int64_t>(max_seq_len) + 127) / 128;
  if (static_cast<int64_t>(batch) * dims->num_heads * qtiles > INT32_MAX) return EG_MLA_ERR_UNSUPPORTED;
  if (workspace == nullptr || !aligned(workspace, 256) ||
      workspace_bytes < egmla::prefill_workspace_bytes(batch, total_tokens, dims->num_heads, dims->d_c))
    return EG_MLA_ERR_WORKSPACE;
  egmla::PrefillArgs a;
  std::memset(&a, 0, sizeof(a));
  a.q = q;
  a.c = c_new;
  a.kr = krope_new;
  a.ids = ids_new;
  a.cu_seqlens = cu_seqlens;
  a.gate_table = gate_table;
  a.ln_gamma = ln_gamma;
  a.ln_beta = ln_beta;
  a.w_uk = w_uk;
  a.w_uv = w_uv;
  a.out = out;
  a.c_pool = c_pool;
  a.kr_pool = c_pool ? krope_pool : nullptr;
  a.id_pool = c_pool ? id_pool : nullptr;
  a.block_table = block_table;
  a.workspace = workspace;
  a.status = dev_status;
  a.H = dims->num_heads;
  a.d_c = dims->d_c;
  a.vocab = dims->vocab;
  a.batch = batch;
  a.total = total_tokens;
  a.max_seq_len = max_seq_len;
  a.max_pages = max_pages_per_seq;
  a.num_pages = num_pages;
  a.gate = gated ? 1 : 0;
  a.gate_add = dims->gate_mode == EG_MLA_GATE_ADD_LN ? 1 : 0;
  a.gate_ln = (dims->gate_mode == EG_MLA_GATE_MUL_LN || dims->gate_mode == EG_MLA_GATE_ADD_LN) ? 1 : 0;
  a.eps = dims->ln_eps > 0.f ? dims->ln_eps : 1e-5f;
  a.scale_log2 = resolve_scale(dims) * 1.4426950408889634f;
  return to_status(egmla::launch_prefill(a, static_cast<cudaStream_t>(stream), prof_mark));
}

int eg_mla_gate_table(const eg_mla_dims* dims, int32_t d_e, const void* emb, const void* w_ue, void* gate_table,
                      int32_t* dev_status, void* stream) {
  if (dims == nullptr || d_e <= 0 || dims->vocab <= 0 || dims->d_c <= 0) return EG_MLA_ERR_INVALID_ARG;
  if (dims->dtype != EG_MLA_BF16 || d_e % 64 != 0 || d_e > 512 || dims->d_c % 64 != 0) return EG_MLA_ERR_UNSUPPORTED;
  if (!emb || !w_ue || !gate_table || !aligned(emb, 16) || !aligned(w_ue, 16) || !aligned(gate_table, 16))
    return EG_MLA_ERR_INVALID_ARG;
  return to_status(egmla::launch_gate_table(emb, w_ue, dims->vocab, d_e, dims->d_c, gate_table, dev_status,
                                            static_cast<cudaStream_t>(stream)));
}

int eg_mla_debug_linear(const void* w, int32_t n_out, int32_t k, const void* x, int32_t batch, void* out,
                        int32_t ldo, int32_t out_f32, int32_t* dev_status, void* stream) {
  if (n_out <= 0 || k <= 0 || batch < 0 || ldo < n_out || k % 8 != 0) return EG_MLA_ERR_INVALID_ARG;
  if (batch == 0) return EG_MLA_OK;
  if (!w || !x || !out || !aligned(w, 16) || !aligned(x, 16) || !aligned(out, out_f32 ? 4 : 2))
    return EG_MLA_ERR_INVALID_ARG;
  return to_status(egmla::launch_linear_tc(w, n_out, k, x, batch, out, ldo, out_f32 != 0, dev_status,
                                           static_cast<cudaStream_t>(stream)));
}

int eg_mla_debug_linear_plan(int32_t n_out, int32_t k, int32_t batch, int32_t* cluster, int32_t* stages,
                             int32_t* max_clusters) {
  if (!cluster || !stages || !max_clusters || n_out <= 0 || k <= 0 || batch <= 0 || k % 8 != 0)
    return EG_MLA_ERR_INVALID_ARG;
  int c = 0, s = 0, m = 0;
  const cudaError_t e = egmla::linear_tc_plan(n_out, k, batch, &c, &s, &m);
  *cluster = c;
  *stages = s;
  *max_clusters = m;
  return to_status(e);
}

int eg_mla_debug_set_trace(void* dev_buf, int64_t bytes, int32_t ctas) {
  std::lock_guard<std::mutex> lk(g_trace.mu);
  if (dev_buf == nullptr || bytes <= 0 || ctas <= 0) {
    g_trace.buf = nullptr;
    g_trace.ctas = g_trace.cap = 0;
    return EG_MLA_OK;
  }
  const int64_t cap = bytes / (static_cast<int64_t>(ctas) * egmla::kTraceRoles * 16);
  if (cap < 1 || !aligned(dev_buf, 16)) return EG_MLA_ERR_INVALID_ARG;
  g_trace.buf = dev_buf;
  g_trace.ctas = ctas;
  g_trace.cap = static_cast<int>(cap > (1 << 20) ? (1 << 20) : cap);
  return EG_MLA_OK;
}

int eg_mla_debug_set_fault(int32_t cta, int32_t tile, int64_t wait_limit_ns) {
  std::lock_guard<std::mutex> lk(g_fault.mu);
  if (cta < 0) {
    g_fault.cta = g_fault.tile = -1;
    g_fault.wait_ns = egmla::kWaitLimitNs;
    return EG_MLA_OK;
  }
  if (tile < 0 || wait_limit_ns < 1000 || wait_limit_ns > static_cast<int64_t>(egmla::kWaitLimitNs))
    return EG_MLA_ERR_INVALID_ARG;
  g_fault.cta = cta;
  g_fault.tile = tile;
  g_fault.wait_ns = static_cast<uint64_t>(wait_limit_ns);
  return EG_MLA_OK;
}

int eg_mla_profile_begin(int32_t max_launches) {
  if (max_launches <= 0) return EG_MLA_ERR_INVALID_ARG;
  std::lock_guard<std::mutex> lk(g_prof.mu);
  for (cudaEvent_t e : g_prof.ev) cudaEventDestroy(e);
  g_prof.ev.assign(2 * static_cast<size_t>(max_launches), nullptr);
  for (auto& e : g_prof.ev)
    if (cudaEventCreate(&e) != cudaSuccess) {
      g_prof.ev.clear();
      g_prof.active = false;
      return EG_MLA_ERR_CUDA;
    }
  g_prof.used = 0;
  g_prof.active = true;
  return EG_MLA_OK;
}

int eg_mla_profile_end(double* ms_sum, int32_t* launches) {
  if (ms_sum == nullptr || launches == nullptr) return EG_MLA_ERR_INVALID_ARG;
  std::lock_guard<std::mutex> lk(g_prof.mu);
  double total = 0.0;
  int rc = EG_MLA_OK;
  for (int i = 0; i < g_prof.used; ++i) {
    float ms = 0.f;
    if (cudaEventSynchronize(g_prof.ev[2 * i + 1]) != cudaSuccess ||
        cudaEventElapsedTime(&ms, g_prof.ev[2 * i], g_prof.ev[2 * i + 1]) != cudaSuccess) {
      rc = EG_MLA_ERR_CUDA;
      break;
    }
    total += ms;
  }
  *ms_sum = total;
  *launches = g_prof.used;
  for (cudaEvent_t e : g_prof.ev) cudaEventDestroy(e);
  g_prof.ev.clear();
  g_prof.used = 0;
  g_prof.active = false;
  return rc;
}

int eg_mla_debug_gather(const eg_mla_dims* dims, const void* c_pool, const void* krope_pool,
                        const int32_t* id_pool, const int32_t* block_table, int32_t max_pages_per_seq,
                        const int32_t* seq_lens, int32_t max_seq_len, int32_t batch, int32_t num_pages,
                        const void* gate_table, void* c_out, void* kr_out, int32_t* ids_out, void* g_out,
                        int32_t num_splits, void* workspace, size_t workspace_bytes, int32_t* dev_status,
                        void* stream) {
  if (dims == nullptr || dims->dtype != EG_MLA_BF16 || dims->gate_mode == EG_MLA_GATE_NONE ||
      (dims->d_c != 192 && dims->d_c != 256))
    return EG_MLA_ERR_UNSUPPORTED;
  DecodeArgs a;
  int rc = fill_decode_args(a, dims, c_pool, krope_pool, id_pool, block_table, max_pages_per_seq, seq_lens,
                            max_seq_len, batch, num_pages, gate_table, num_splits, workspace, workspace_bytes,
                            dev_status);
  if (rc != EG_MLA_OK) return rc;
  if (batch == 0) return EG_MLA_OK;
  if (!c_out || !kr_out || !ids_out || !g_out) return EG_MLA_ERR_INVALID_ARG;
  a.dump_c = c_out;
  a.dump_kr = kr_out;
  a.dump_ids = ids_out;
  a.dump_g = g_out;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  CUtensorMap maps[2];
  if (!encode_decode_maps(maps, dims, c_pool, krope_pool, num_pages)) return EG_MLA_ERR_CUDA;
  a.q = nullptr;  // prologue computes the page prefix sums only
  cudaError_t e = egmla::launch_prologue_tc(a, nullptr, st);
  if (e == cudaSuccess) e = egmla::launch_decode_tc(a, maps, true, st, nullptr);
  return to_status(e);
}

}  // extern "C"
