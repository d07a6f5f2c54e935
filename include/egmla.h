/*
 * egmla.h - C ABI of libegmla, the GB300 (sm_103a) decode hot path of EG-MLA
 * (Embedding-Gated Multi-head Latent Attention, arXiv 2509.16686).
 *
 * The library implements one decode step of an EG-MLA attention layer over a
 * paged latent KV cache:
 *   - eg_mla_append_latent writes each sequence's new compressed latent c^KV
 *     (Appendix C Eq. 1) and its rotated RoPE key k^R (Eq. 10), plus the token
 *     id, into the cache.  The cache keeps (d_c + d_h^R) values per token per
 *     layer (Table 5).
 *   - eg_mla_decode reads the cache, gathers each cached token's gate row
 *     g = G[id] (Section 3 Eqs. 3-4 in the table form of EG-MLA-A, Section 5.2),
 *     applies the gate and LayerNorm to the latent as it is read,
 *     c~ = LN(c (*) g) (Eq. 5 in latent space), and runs weight-absorbed MLA
 *     (Eqs. 11-13): q^ = W_UK,h^T q^C scores the shared latent plus the shared
 *     RoPE key with scale 1/sqrt(d_h + d_h^R), an online softmax with split-KV
 *     partials is merged by log-sum-exp, and the latent-space output is
 *     up-projected through W_UV,h.  It returns the per-head outputs u_{t,i}.
 *   - eg_mla_layer_decode runs the same step from the layer's hidden state:
 *     the query and latent projections (Eqs. 1, 8-10), the latent's RMSNorm
 *     and the rotary embedding, the append and the decode above, and the
 *     output projection (Eq. 14).
 *
 * Conventions shared by every call:
 *   - Every pointer argument except `dims`, `bytes_out` and `out_splits` is a
 *     DEVICE pointer to caller-owned memory.  The library never allocates,
 *     frees or keeps device memory between calls; the device memory it owns
 *     is the fixed static scratch array of eg_mla_decode_static, which is
 *     part of the loaded module.
 *   - `stream` is a cudaStream_t passed as void* (NULL = legacy default
 *     stream).  Calls are asynchronous on that stream and never synchronise
 *     the host.
 *   - Host-side argument errors return a negative eg_mla_status and launch
 *     nothing.  Errors found on the device (out-of-range page id or token id,
 *     a pipeline wait that timed out) are written to *dev_status (a device
 *     int32 that the caller zeroes; the first error wins); the host reads it
 *     after synchronising.  dev_status may be NULL, in which case device
 *     errors are not reported.
 *   - Layouts are row-major and densely packed unless stated.  Model-dtype
 *     tensors hold bf16 (EG_MLA_BF16) or fp32 (EG_MLA_FP32) elements;
 *     ln_gamma/ln_beta are always fp32.
 */
#ifndef EGMLA_H
#define EGMLA_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  EG_MLA_OK = 0,
  EG_MLA_ERR_INVALID_ARG = -1,   /* null pointer, bad size, misaligned buffer */
  EG_MLA_ERR_UNSUPPORTED = -2,   /* dims outside the compiled kernel shapes */
  EG_MLA_ERR_CUDA = -3,          /* a CUDA runtime call failed (launch, attribute) */
  EG_MLA_ERR_OUT_OF_RANGE = -4,  /* device: page id >= num_pages or token id >= vocab */
  EG_MLA_ERR_TIMEOUT = -5,       /* device: a pipeline wait exceeded its limit */
  EG_MLA_ERR_WORKSPACE = -6,     /* workspace too small or misaligned */
  EG_MLA_ERR_SCRATCH_LIMIT = -7  /* needs more than EG_MLA_STATIC_SCRATCH_BYTES of static scratch */
} eg_mla_status;

typedef enum { EG_MLA_BF16 = 0, EG_MLA_FP32 = 1 } eg_mla_dtype;

typedef enum {
  EG_MLA_GATE_NONE = 0,    /* plain MLA: the latent is used as cached (baseline) */
  EG_MLA_GATE_MUL_LN = 1,  /* EG-MLA: c~ = LN(c (*) G[id]) with affine gamma/beta */
  EG_MLA_GATE_MUL = 2,     /* ablation "remove LayerNorm" (Section 4.4): c~ = c (*) G[id] */
  EG_MLA_GATE_ADD_LN = 3   /* ablation "replace (*) with addition" (Section 4.4): c~ = LN(c + G[id]) */
} eg_mla_gate_mode;

/* Shapes of one attention layer.  d_v = value head dim (= d_nope in the paper's
 * models, Appendix A).  softmax_scale <= 0 selects 1/sqrt(d_nope + d_rope)
 * (Eq. 13); ln_eps <= 0 selects 1e-5 (nn.LayerNorm's default, listing of
 * Appendix E). */
typedef struct {
  int32_t num_heads;
  int32_t d_nope;
  int32_t d_rope;
  int32_t d_v;
  int32_t d_c;
  int32_t page_size;
  int32_t vocab;
  int32_t dtype;      /* eg_mla_dtype */
  int32_t gate_mode;  /* eg_mla_gate_mode */
  float softmax_scale;
  float ln_eps;
} eg_mla_dims;

/* Supported shapes.
 *   bf16 (tensor-core path): num_heads 16, d_rope 64, page_size 64,
 *        d_c in {192, 256} with any gate mode, d_c 512 with EG_MLA_GATE_NONE;
 *        d_nope, d_v multiples of 8 up to 256.
 *   fp32: num_heads <= 16, d_c <= 512 and a multiple of 4, d_rope <= 64,
 *        d_nope, d_v <= 256, page_size 64.
 * Other shapes return EG_MLA_ERR_UNSUPPORTED. */

/*
 * eg_mla_append_latent - write one new token per sequence into the paged cache.
 *
 * Cache content per token is the compressed latent c^KV [d_c] (Appendix C
 * Eq. 1), the rotated shared RoPE key k^R [d_rope] (Eq. 10; the listing of
 * Appendix E rotates k_pe before it is used), and the token id i_t that the
 * gate needs at read time (Section 3, Eq. 3).  Nothing is gated here: with
 * latent-space gating the gate is applied when the latent is read.
 *
 *   c_pool       [num_pages, page_size, d_c]   model dtype, written
 *   krope_pool   [num_pages, page_size, d_rope] model dtype, written
 *   id_pool      [num_pages, page_size] int32, written; may be NULL (then
 *                ids_new is ignored)
 *   c_new        [batch, d_c], krope_new [batch, d_rope], ids_new [batch]
 *   block_table  [batch, max_pages_per_seq] int32: logical page -> physical page
 *   positions    [batch] int32: logical slot of the new token (= seq_len-1);
 *                a negative position skips that sequence
 * Device errors: a position whose page index is >= max_pages_per_seq or whose
 * physical page is outside [0, num_pages) is skipped and reported as
 * EG_MLA_ERR_OUT_OF_RANGE.  The copy is bit-exact.
 */
int eg_mla_append_latent(const eg_mla_dims* dims, void* c_pool, void* krope_pool,
                         int32_t* id_pool, const void* c_new, const void* krope_new,
                         const int32_t* ids_new, const int32_t* block_table,
                         int32_t max_pages_per_seq, const int32_t* positions,
                         int32_t batch, int32_t num_pages, int32_t* dev_status,
                         void* stream);

/*
 * eg_mla_default_num_splits - the split count eg_mla_decode uses for
 * num_splits = 0: one split-KV work unit per SM of the current device.
 */
int eg_mla_default_num_splits(int32_t* out_splits);

/*
 * eg_mla_decode_workspace_size - bytes of device workspace eg_mla_decode needs
 * for this batch and split count (0 = default).  The workspace holds the page
 * prefix sums, the absorbed queries q^ = W_UK,h^T q^C and the split-KV partial
 * results (running max, denominator and un-normalised latent output per
 * split, sequence and head).  Returns 0 for unsupported dims.
 */
size_t eg_mla_decode_workspace_size(const eg_mla_dims* dims, int32_t batch, int32_t num_splits);

/*
 * eg_mla_decode - one decode step of EG-MLA attention for `batch` sequences.
 *
 * For each sequence b and head h, with L_b = seq_lens[b] cached tokens
 * (including the one just appended) and c~_j = LN(c_j (*) G[id_j]) over d_c
 * (EG_MLA_GATE_MUL_LN), c_j (*) G[id_j] (EG_MLA_GATE_MUL), LN(c_j + G[id_j])
 * (EG_MLA_GATE_ADD_LN) or c~_j = c_j (EG_MLA_GATE_NONE); gamma and beta apply
 * only with a LayerNorm:
 *   s_j   = scale * (q^_h . c~_j + q^R_h . k^R_j),  q^_h = W_UK,h^T q^C_h   (Eqs. 11-13)
 *   u_b,h = W_UV,h sum_j softmax(s)_j c~_j                                    (Eq. 13, Eq. 6)
 * which equals the paper's per-head attention with k^C = W_UK c~ and
 * v^C = W_UV c~ (weight absorption).  A sequence with L_b = 0 gets u = 0.
 *
 *   q            [batch, num_heads, d_nope + d_rope] model dtype; RoPE already
 *                applied to the last d_rope entries; 16-byte aligned
 *   c_pool, krope_pool, id_pool: the paged cache (see eg_mla_append_latent);
 *                id_pool may be NULL for EG_MLA_GATE_NONE.  c_pool and
 *                krope_pool must be 16-byte aligned.
 *   block_table  [batch, max_pages_per_seq] int32
 *   seq_lens     [batch] int32 (device), each <= max_seq_len
 *   max_seq_len  host-side upper bound of seq_lens (<= max_pages_per_seq*page_size)
 *   gate_table   [vocab, d_c] model dtype: G[i] = W^UE Emb(i) precomputed per
 *                vocabulary entry (EG-MLA-A); ignored for EG_MLA_GATE_NONE;
 *                32-byte aligned for bf16 (read in 32-byte pieces), 16-byte
 *                aligned for fp32
 *   ln_gamma, ln_beta  [d_c] fp32, may be NULL (gamma = 1, beta = 0)
 *   w_uk         [num_heads, d_nope, d_c] model dtype (the key rows of the
 *                joint key/value up-projection W^UKV, Appendix C Eq. 2,
 *                viewed per head), 16-byte aligned
 *   w_uv         [num_heads, d_v, d_c] model dtype (its value rows),
 *                16-byte aligned
 *   out          [batch, num_heads, d_v] model dtype, written
 *   num_splits   number of split-KV work units (0 = eg_mla_default_num_splits);
 *                the cache pages of all sequences are divided into this many
 *                equal contiguous ranges
 *   workspace    device buffer of at least eg_mla_decode_workspace_size()
 *                bytes, 256-byte aligned; its content is scratch
 * Returns EG_MLA_OK once the kernels are queued.  Device errors go to
 * *dev_status; the content of `out` is then unspecified.
 */
int eg_mla_decode(const eg_mla_dims* dims, const void* q, const void* c_pool,
                  const void* krope_pool, const int32_t* id_pool,
                  const int32_t* block_table, int32_t max_pages_per_seq,
                  const int32_t* seq_lens, int32_t max_seq_len, int32_t batch,
                  int32_t num_pages, const void* gate_table, const float* ln_gamma,
                  const float* ln_beta, const void* w_uk, const void* w_uv, void* out,
                  int32_t num_splits, void* workspace, size_t workspace_bytes,
                  int32_t* dev_status, void* stream);

/*
 * eg_mla_step - one decode step: eg_mla_append_latent, then eg_mla_decode, in
 * one call (the method's decode step: the new token is cached, Appendix C
 * Eq. 1 and Eq. 10, and attends over the cache including itself, Eq. 13).
 *
 * Arguments: the union of the two calls', with the same meaning, layout,
 * ownership and alignment rules (c_new, krope_new, ids_new and positions as
 * for eg_mla_append_latent; seq_lens must already count the new token).
 * Results: bit-identical to eg_mla_append_latent followed by eg_mla_decode on
 * the same stream with the same arguments.  Every argument of both parts is
 * checked before anything is launched; host errors return the same codes as
 * the two calls, device errors go to *dev_status.
 *
 * On the bf16 path the append runs inside the grid of the query-absorption
 * kernel (which reads no pool), one launch fewer per step; the split-KV
 * kernel starts its setup while that kernel finishes and waits for its
 * completion before it reads the cache.
 */
int eg_mla_step(const eg_mla_dims* dims, void* c_pool, void* krope_pool, int32_t* id_pool,
                const void* c_new, const void* krope_new, const int32_t* ids_new,
                const int32_t* positions, const void* q, const int32_t* block_table,
                int32_t max_pages_per_seq, const int32_t* seq_lens, int32_t max_seq_len,
                int32_t batch, int32_t num_pages, const void* gate_table,
                const float* ln_gamma, const float* ln_beta, const void* w_uk,
                const void* w_uv, void* out, int32_t num_splits, void* workspace,
                size_t workspace_bytes, int32_t* dev_status, void* stream);

/* Size of the static device scratch array behind eg_mla_decode_static. */
#define EG_MLA_STATIC_SCRATCH_BYTES ((size_t)16 << 20)

/*
 * eg_mla_decode_static - eg_mla_decode without a caller workspace.  The paper
 * has no counterpart to this call: it is an interface choice of this library.
 *
 * Same arguments, results, validation and device-error reporting as
 * eg_mla_decode, minus `workspace` and `workspace_bytes`: the scratch is a
 * file-scope static device array of EG_MLA_STATIC_SCRATCH_BYTES (16 MiB),
 * 256-byte aligned, compiled into the library.  The call allocates no device
 * or pinned memory: no cudaMalloc/cudaFree and no allocating library routine.
 * It serves callers that have no device memory to hand out per step, such as
 * an engine that reserved all free HBM for the paged latent cache at start-up,
 * or a C caller without a caching allocator that would otherwise pay a
 * device-synchronising cudaFree inside the token loop.
 *
 *   - Size limit: if eg_mla_decode_workspace_size(dims, batch, num_splits)
 *     exceeds EG_MLA_STATIC_SCRATCH_BYTES the call returns
 *     EG_MLA_ERR_SCRATCH_LIMIT and launches nothing; use eg_mla_decode with a
 *     workspace, or fewer splits, instead.  The limit covers, for example,
 *     batch 128 at d_c = 512 with 301 splits (16,754,944 bytes).
 *   - Start-up: the first call on each device, with that device current,
 *     looks up the array's device address (cudaGetSymbolAddress) and caches
 *     it with the id of the current context; make that first call before any
 *     stream capture begins.  After cudaDeviceReset the next call sees a new
 *     context id and looks the address up again (the same rule applies to
 *     that call).  A failed lookup returns EG_MLA_ERR_CUDA.
 *   - Zeroing: no part of the scratch needs to start at zero (every word the
 *     kernels read from it is written earlier in the same call), so the call
 *     runs no clearing pass.  *dev_status is the caller's, zeroed by the
 *     caller, as for eg_mla_decode.
 *   - Concurrency: there is one scratch array per device.  Calls on the same
 *     device whose kernels may overlap (different streams without ordering,
 *     or different host threads) race on it and corrupt each other's
 *     results; serialise them, e.g. on one stream.
 */
int eg_mla_decode_static(const eg_mla_dims* dims, const void* q, const void* c_pool,
                         const void* krope_pool, const int32_t* id_pool,
                         const int32_t* block_table, int32_t max_pages_per_seq,
                         const int32_t* seq_lens, int32_t max_seq_len, int32_t batch,
                         int32_t num_pages, const void* gate_table, const float* ln_gamma,
                         const float* ln_beta, const void* w_uk, const void* w_uv, void* out,
                         int32_t num_splits, int32_t* dev_status, void* stream);

/*
 * One decode step through a whole EG-MLA attention layer (Appendix C Eqs. 1,
 * 8-14 with the q-LoRA rank 0 of every model in Appendix A; the listing of
 * Appendix E for kv_norm and the rotary embedding).  For every sequence b:
 *
 *   q      = W^Q x_b                    [H (d_nope + d_rope)], split per head
 *                                        into [q^C ; q^R]   (Eqs. 8-9, 11)
 *   [c ; k] = W^{DKV,KR} x_b            [d_c + d_rope]      (Eqs. 1, 10)
 *   c^KV   = RMSNorm(c) * kv_norm_w     (the listing's kv_norm; what the cache keeps)
 *   q^R, k^R rotated at position L_b - 1: pair (2i, 2i + 1) by the angle
 *            pos * theta^(-2i / d_rope) (the listing's apply_rotary_emb)
 *   append (c^KV, k^R, id) to the cache; u = eg_mla_decode(q, cache)  (Eqs. 2-13)
 *   y_b    = W^O [u_b,1 ; ... ; u_b,H]  [n_embd]             (Eq. 14)
 *
 * bf16 only.  q, c^KV, k^R and u are rounded to bf16 once, from fp32, where
 * the layer stores them; y is written in bf16.
 */
typedef struct {
  int32_t n_embd;     /* model width E (a multiple of 8) */
  float rope_theta;   /* rotary base; <= 0 selects 10000 */
  float rms_eps;      /* kv_norm epsilon; <= 0 selects 2^-23 (the fp32 machine epsilon) */
  int32_t share_kv;   /* nonzero: a later layer of a layer group (Section 5 inter-layer
                         sharing, Appendix H "layer group size"): the group shares the
                         first half of the KV projection, W^{DKV,KR}, and its activations,
                         so the group's first layer already projected, normalised, rotated
                         and appended this step's c^KV, k^R and id to the cache the group
                         shares.  This layer projects only its q (only the W^Q rows of
                         w_qkv_a are read), appends nothing and attends over the shared
                         cache with its own W_UK, W_UV, gate table and LayerNorm */
} eg_mla_layer_dims;

/* Device pointers of one layer's weights, each 16-byte aligned, in the
 * PyTorch Linear layout [out, in] of the model dtype (bf16) unless stated. */
typedef struct {
  const void* w_qkv_a;      /* [H (d_nope + d_rope) + d_c + d_rope, E]: the rows of
                               W^Q, then those of W^{DKV,KR} (one projection GEMM) */
  const void* kv_norm_w;    /* [d_c] */
  const void* w_o;          /* [E, H d_v] */
  const void* gate_table;   /* [vocab, d_c]  as for eg_mla_decode */
  const float* ln_gamma;    /* [d_c] fp32 or NULL, as for eg_mla_decode */
  const float* ln_beta;     /* [d_c] fp32 or NULL */
  const void* w_uk;         /* [H, d_nope, d_c] */
  const void* w_uv;         /* [H, d_v, d_c] */
} eg_mla_layer_weights;

/* Workspace bytes eg_mla_layer_decode needs (0 on invalid arguments): the
 * projections' outputs, u and the decode workspace of eg_mla_decode. */
size_t eg_mla_layer_workspace_size(const eg_mla_dims* dims, const eg_mla_layer_dims* layer,
                                   int32_t batch, int32_t num_splits);

/*
 * eg_mla_layer_attn_offset - byte offset, within the workspace of an
 * eg_mla_layer_decode call with these arguments, of the step's attention
 * output u [batch, num_heads, d_v] (bf16, Eq. 13), which the call leaves there
 * after it completes (the input of the output projection, Eq. 14): a testing
 * and debugging aid.  Returns 0 on invalid arguments (a valid offset for
 * batch >= 1 is never 0: the projections' outputs come first).
 */
size_t eg_mla_layer_attn_offset(const eg_mla_dims* dims, const eg_mla_layer_dims* layer, int32_t batch,
                                int32_t num_splits);

/*
 * eg_mla_layer_decode - the step above for `batch` sequences, on `stream`.
 *
 *   x          [batch, E] bf16 hidden states of the new tokens
 *   ids_new    [batch] int32 token ids of the new tokens (their gate rows)
 *   positions  [batch] int32 = seq_lens[b] - 1: the new token's slot and its
 *              rotation position
 *   c_pool, krope_pool, id_pool, block_table, max_pages_per_seq, seq_lens,
 *   max_seq_len, num_pages, num_splits, dev_status: as for
 *              eg_mla_append_latent and eg_mla_decode (seq_lens include the
 *              new token, so every sequence has L_b >= 1)
 *   y          [batch, E] bf16 output, caller-owned
 *   workspace  >= eg_mla_layer_workspace_size(...) bytes, 256-byte aligned
 *
 The projections run in this library's weight-streaming tcgen05 GEMM
 * (fp32 accumulation, the reduction dimension split over the CTAs of a
 * thread-block cluster and summed in rank order, so results do not depend on
 * timing).  The call allocates nothing.  The first call with a given shape
 * runs a host-side occupancy query for the GEMM's cluster size (cached
 * afterwards); make it before any stream capture.  Host-side argument errors
 * return a negative status and launch nothing; device errors go to
 * *dev_status as for eg_mla_decode.
 */
int eg_mla_layer_decode(const eg_mla_dims* dims, const eg_mla_layer_dims* layer,
                        const eg_mla_layer_weights* weights, const void* x, const int32_t* ids_new,
                        const int32_t* positions, void* c_pool, void* krope_pool, int32_t* id_pool,
                        const int32_t* block_table, int32_t max_pages_per_seq, const int32_t* seq_lens,
                        int32_t max_seq_len, int32_t batch, int32_t num_pages, void* y,
                        int32_t num_splits, void* workspace, size_t workspace_bytes,
                        int32_t* dev_status, void* stream);

/*
 * eg_mla_kv_bytes_per_token - bytes the paged cache keeps per token over
 * n_layers layers: (d_c + d_rope) elements of the model dtype per layer
 * (Table 5 with d_c the cached latent width), plus a 4-byte token id per
 * layer when gating is on (read-time gating needs the id).  Host only.
 */
int eg_mla_kv_bytes_per_token(const eg_mla_dims* dims, int32_t n_layers, int64_t* bytes_out);

/* eg_mla_status_string - static text for a status code. */
const char* eg_mla_status_string(int status);

/*
 * eg_mla_debug_gather - test entry: runs the decode kernel's cache-read stage
 * (TMA page loads through the block table and the token-id gate-row gather)
 * and writes what it read for every cached position instead of attending.
 * bf16 path only.  Outputs are dense per (sequence, logical position):
 *   c_out [batch, max_seq_len, d_c], kr_out [batch, max_seq_len, d_rope],
 *   ids_out [batch, max_seq_len] int32, g_out [batch, max_seq_len, d_c]
 * Positions >= seq_lens[b] are left untouched.  Same argument rules and
 * workspace as eg_mla_decode.
 */
int eg_mla_debug_gather(const eg_mla_dims* dims, const void* c_pool, const void* krope_pool,
                        const int32_t* id_pool, const int32_t* block_table,
                        int32_t max_pages_per_seq, const int32_t* seq_lens,
                        int32_t max_seq_len, int32_t batch, int32_t num_pages,
                        const void* gate_table, void* c_out, void* kr_out, int32_t* ids_out,
                        void* g_out, int32_t num_splits, void* workspace,
                        size_t workspace_bytes, int32_t* dev_status, void* stream);

/*
 * eg_mla_profile_begin / eg_mla_profile_end - per-launch timing of the split-KV
 * decode kernel (the one that streams the latent cache) and of the prefill's
 * attention kernel.  After begin, every eg_mla_decode (eg_mla_step) call
 * records a CUDA event pair around the decode kernel's launch on its stream,
 * and every eg_mla_prefill call one around its attention kernel's launch, for
 * at most max_launches launches in all.  end synchronises on the
 * events, returns the summed kernel time in milliseconds and the number of
 * launches timed, releases the events and stops recording.  During stream
 * capture the pair becomes event-record nodes of the graph
 * (cudaEventRecordExternal): replay the graph, synchronise, then call end,
 * which reads the last replay's timestamps.
 * Returns EG_MLA_ERR_CUDA if event creation fails, EG_MLA_ERR_INVALID_ARG for
 * max_launches <= 0 or null outputs.
 */
int eg_mla_profile_begin(int32_t max_launches);
int eg_mla_profile_end(double* ms_sum, int32_t* launches);

/*
 * eg_mla_decode_r0 - decode with the paper-literal gate placement (R0): the
 * gate and the LayerNorm act on the up-projected keys and values of all heads
 * at once (Section 3 Eq. 5 applied after Eq. 2, as the Appendix E listing
 * does), kv~_j = LN_{H(d_n + d_v)}((W^UKV c_j) (*) G_R0[id_j]), split per head
 * into k^C_j, v^C_j (Eq. 6); then u_h = sum_j softmax_j(s_j) v^C_j,h with
 * s_j = ([k^C_j,h ; k^R_j] . q_h) / sqrt(d_n + d_r) (Eqs. 11-13, without
 * weight absorption: the gate in this space cannot be folded into q).
 *
 * Supported: bf16, 16 heads, d_nope = d_v = 128, d_rope = 64, d_c in
 * {192, 256} (EG_MLA_ERR_UNSUPPORTED otherwise).  dims->gate_mode is ignored;
 * dims->ln_eps is the LayerNorm's epsilon (<= 0: 1e-5).
 *
 *   q, c_pool, krope_pool, id_pool, block_table, max_pages_per_seq,
 *   seq_lens, batch, num_pages: as for eg_mla_decode (the cache after the
 *              step's append; seq_lens include the new token)
 *   w_ukv      [16 * 256, d_c] bf16: per head h its 128 key rows (W_UK,h),
 *              then its 128 value rows (W_UV,h), the row order of the joint
 *              up-projection in Appendix E
 *   gate_r0    [vocab, 4096] bf16: the gate in that space per token id
 *   ln_gamma_r0, ln_beta_r0  [4096] fp32, may be NULL (1, 0)
 *   out        [batch, 16, 128] bf16
 *   workspace  >= eg_mla_decode_r0_workspace_size(dims, batch,
 *              max_pages_per_seq, num_pages) bytes, 256-byte aligned: the
 *              gated values of every pool row (16 x 128 bf16, head-major),
 *              the rows' LayerNorm statistics, and the logits of every
 *              (sequence, position) the block table can hold (16 fp32 each)
 *
 * Device errors: a page id outside [0, num_pages), a sequence longer than
 * its block table (positions past it are not read), or a token id outside
 * [0, vocab) of a cached token is reported as EG_MLA_ERR_OUT_OF_RANGE (the
 * gate then uses row 0); a timed-out pipeline wait as EG_MLA_ERR_TIMEOUT.
 * All 16-byte-read arguments must be 16-byte aligned.
 */
size_t eg_mla_decode_r0_workspace_size(const eg_mla_dims* dims, int32_t batch, int32_t max_pages_per_seq,
                                       int32_t num_pages);
int eg_mla_decode_r0(const eg_mla_dims* dims, const void* q, const void* c_pool, const void* krope_pool,
                     const int32_t* id_pool, const int32_t* block_table, int32_t max_pages_per_seq,
                     const int32_t* seq_lens, int32_t batch, int32_t num_pages, const void* w_ukv,
                     const void* gate_r0, const float* ln_gamma_r0, const float* ln_beta_r0, void* out,
                     void* workspace, size_t workspace_bytes, int32_t* dev_status, void* stream);

/*
 * eg_mla_prefill - prompt processing: causal attention of every prompt
 * position over the prompt up to and including itself, and the prompt written
 * into the paged latent cache for the decode steps that follow.
 *
 * For prompt b (packed rows cu_seqlens[b] .. cu_seqlens[b+1] - 1), position t
 * and head h, with c~_j the gated latent of position j as in eg_mla_decode
 * (the gate mode's form of Section 3 Eq. 5 in latent space):
 *   k_j,h = [W_UK,h c~_j ; k^R_j],  v_j,h = W_UV,h c~_j        (Eqs. 2, 6, 12)
 *   u_t,h = sum_{j <= t} softmax_j(q_t,h . k_j,h * scale) v_j,h  (Eq. 13)
 * computed without weight absorption (the per-head keys and values are
 * materialised once per token; Appendix E's form).  The new tokens' raw c,
 * k^R and id are written to logical positions 0 .. L_b - 1 of prompt b.
 *
 * Supported: bf16, d_nope = d_v = 128, d_rope = 64, d_c a multiple of 64 up
 * to 512, any number of heads, any gate mode, page size 64
 * (EG_MLA_ERR_UNSUPPORTED otherwise).
 *
 *   q            [total_tokens, num_heads, d_nope + d_rope] bf16, RoPE already
 *                applied to the last d_rope entries of every row
 *   c_new        [total_tokens, d_c] bf16: each prompt token's c^KV (Eq. 1)
 *   krope_new    [total_tokens, d_rope] bf16: its rotated k^R (Eq. 10)
 *   ids_new      [total_tokens] int32 token ids (may be NULL with
 *                EG_MLA_GATE_NONE)
 *   cu_seqlens   [batch + 1] int32 on the device: cu_seqlens[0] = 0,
 *                non-decreasing, cu_seqlens[batch] = total_tokens
 *   max_seq_len  host-side bound of every prompt length (1 .. total_tokens)
 *   gate_table, ln_gamma, ln_beta, w_uk, w_uv: as for eg_mla_decode
 *   out          [total_tokens, num_heads, d_v] bf16, written
 *   c_pool, krope_pool, id_pool, block_table, max_pages_per_seq, num_pages:
 *                the paged cache as for eg_mla_append_latent; c_pool NULL
 *                skips the cache write (the other four are then ignored);
 *                id_pool may be NULL with EG_MLA_GATE_NONE
 *   workspace    >= eg_mla_prefill_workspace_size(dims, batch, total_tokens)
 *                bytes, 256-byte aligned: the prompts' launch order (longest
 *                first; batch int32), c~ of every token (d_c bf16) and its
 *                per-head keys and values (num_heads * 256 bf16)
 * All tensor arguments read or written in 16-byte pieces must be 16-byte
 * aligned.  Host errors return at once (nothing launched).  Device errors go
 * to *dev_status (may be NULL): a token id outside [0, vocab) (the gate then
 * uses row 0), a page id outside [0, num_pages), a prompt past
 * max_pages_per_seq pages, cu_seqlens inconsistent with total_tokens, or a
 * prompt longer than max_seq_len (its rows past the bound are not computed)
 * as EG_MLA_ERR_OUT_OF_RANGE; a timed-out pipeline wait as EG_MLA_ERR_TIMEOUT.
 */
size_t eg_mla_prefill_workspace_size(const eg_mla_dims* dims, int32_t batch, int32_t total_tokens);
int eg_mla_prefill(const eg_mla_dims* dims, const void* q, const void* c_new, const void* krope_new,
                   const int32_t* ids_new, const int32_t* cu_seqlens, int32_t batch, int32_t total_tokens,
                   int32_t max_seq_len, const void* gate_table, const float* ln_gamma, const float* ln_beta,
                   const void* w_uk, const void* w_uv, void* out, void* c_pool, void* krope_pool,
                   int32_t* id_pool, const int32_t* block_table, int32_t max_pages_per_seq, int32_t num_pages,
                   void* workspace, size_t workspace_bytes, int32_t* dev_status, void* stream);

/*
 * eg_mla_gate_table - the gate table of every vocabulary entry,
 * G[i] = W^UE Emb(i) (Section 3 Eqs. 3-4), computed on the GPU:
 * G [vocab, d_c] = E [vocab, d_e] W^UE^T with fp32 accumulation, rounded to
 * bf16.  EG-MLA-A keeps G from model load on; calling this before each
 * eg_mla_step instead gates the decode with the embedding's projection
 * computed in the step (the EG-MLA form without a stored table), at
 * vocab x d_e x d_c MACs per call.
 *
 *   dims        dtype bf16; dims->vocab rows, dims->d_c a multiple of 64
 *   d_e         embedding width, a multiple of 64 up to 512
 *   emb         [vocab, d_e] bf16 row-major, 16-byte aligned
 *   w_ue        [d_c, d_e] bf16 row-major (the Linear weight layout), 16-byte aligned
 *   gate_table  [vocab, d_c] bf16 row-major, written; 16-byte aligned
 * Returns EG_MLA_ERR_UNSUPPORTED for other shapes or dtypes,
 * EG_MLA_ERR_INVALID_ARG for null or misaligned pointers; a timed-out
 * pipeline wait is reported in *dev_status (may be NULL).
 */
int eg_mla_gate_table(const eg_mla_dims* dims, int32_t d_e, const void* emb, const void* w_ue, void* gate_table,
                      int32_t* dev_status, void* stream);

/*
 * eg_mla_debug_linear - the projection GEMM of eg_mla_layer_decode on its own
 * (a testing aid): out[b][n] = sum_j x[b][j] w[n][j] for b < batch,
 * n < n_out (Eq. 14 and the projections of Appendix C Eqs. 1, 8-10 are of
 * this form).
 *
 *   w     [n_out, k] bf16 row-major, 16-byte aligned
 *   x     [batch, k] bf16 row-major, 16-byte aligned; k % 8 == 0
 *   out   [batch, ldo] fp32 (out_f32 != 0) or bf16, ldo >= n_out; columns
 *         n_out .. ldo - 1 are left untouched
 * fp32 accumulation; the sum over k is split over the CTAs of a cluster and
 * added in rank order.  Returns EG_MLA_ERR_INVALID_ARG for bad sizes, strides
 * or alignment, EG_MLA_ERR_CUDA if the launch fails; a timed-out pipeline
 * wait is reported in *dev_status (may be NULL) as EG_MLA_ERR_TIMEOUT.
 */
int eg_mla_debug_linear(const void* w, int32_t n_out, int32_t k, const void* x, int32_t batch, void* out,
                        int32_t ldo, int32_t out_f32, int32_t* dev_status, void* stream);

/*
 * eg_mla_debug_linear_plan - the launch shape eg_mla_debug_linear (and the
 * projections of eg_mla_layer_decode) use for these sizes on the current
 * device: *cluster CTAs split the reduction dimension of each 128-row tile,
 * *stages shared-memory stages, and *max_clusters clusters of that size the
 * device holds at once (host-side queries; no launch).  Returns
 * EG_MLA_ERR_INVALID_ARG for bad sizes or null outputs, EG_MLA_ERR_CUDA if a
 * query fails.
 */
int eg_mla_debug_linear_plan(int32_t n_out, int32_t k, int32_t batch, int32_t* cluster, int32_t* stages,
                             int32_t* max_clusters);

/*
 * eg_mla_debug_set_trace - pipeline event trace of the split-KV decode kernel
 * (a debugging aid, off by default).  With a device buffer set, later calls of
 * eg_mla_decode at d_c 192 or 256 in the gate modes none and mul_ln run a
 * separately compiled traced build of the kernel (same results; the untraced
 * build carries no trace code), whose first `ctas` CTAs record, per role (0 TMA producer,
 * 1 MMA issuers: the score issuer in the first half of the run, the output
 * issuer in the second, 2 gate, 3 softmax, 4 at d_c 192/256 the kernel phases:
 * entry, set-up done, tile loops done, split combine done), a run of (tag, SM clock) pairs of 8-byte
 * words, tag = event << 56 | tile index << 32, whose low 32 bits hold, in the
 * kernel phases only, the low 32 bits of the global nanosecond timer (which
 * maps each CTA's clock to time); run r of CTA c starts at word
 * (c * 5 + r) * cap * 2 with cap = bytes / (ctas * 5 * 16).  The caller zeroes
 * the buffer; unused entries stay zero.  NULL or bytes <= 0 turns tracing off.
 */
int eg_mla_debug_set_trace(void* dev_buf, int64_t bytes, int32_t ctas);

/*
 * eg_mla_debug_set_fault - test entry for the failure path of the split-KV
 * decode kernel (d_c 192 and 256, bf16).  With cta >= 0, later eg_mla_decode
 * calls withhold one page copy: CTA `cta` skips the copy of its tile `tile`
 * (0-based in its walk) and its arrival, and every pipeline wait of those
 * launches gives up after wait_limit_ns (1 us .. 2 s) instead of the default
 * 2 s.  The wait on the withheld page then runs out: the kernel records
 * EG_MLA_ERR_TIMEOUT in *dev_status, every role leaves its loop, the copies
 * and MMAs already issued are waited for, TMEM is freed and the kernel
 * returns; the rest of the grid reports the same status when its split merge
 * waits for the missing partial.  No fault, trap or hang is involved, and the
 * device stays usable.  cta < 0 restores normal operation.  Returns
 * EG_MLA_ERR_INVALID_ARG for a negative tile or a limit out of range.
 */
int eg_mla_debug_set_fault(int32_t cta, int32_t tile, int64_t wait_limit_ns);

#ifdef __cplusplus
}
#endif

#endif /* EGMLA_H */
