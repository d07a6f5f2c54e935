// egmla_layer.cu - one decode step through a whole EG-MLA attention layer:
// the query and latent projections, the latent's RMSNorm and the rotary
// embedding of q^R and k^R (one fused kernel), the cache append and the
// gated latent attention of egmla_api.cu, and the output projection.  The two
// projection GEMMs (the stacked query/latent weight, and W^O) run in the
// weight-streaming tcgen05 kernel of egmla_linear.cu.  See include/egmla.h
// for the contract.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <cmath>
#include <cstdint>
#include <mutex>

#include "../../include/egmla.h"
#include "egmla_kernels.h"

namespace {

constexpr int kQkvThreads = 256;

size_t up256(size_t x) { return (x + 255) / 256 * 256; }

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15) == 0; }

struct LayerWorkspace {
  size_t off_qkv32, off_q, off_c, off_kr, off_u, off_dec, dec_bytes, total;
};

// carve of the layer workspace (every piece 256-byte aligned); dec_bytes = 0 on
// invalid decode arguments
LayerWorkspace layer_workspace(const eg_mla_dims* d, int32_t batch, int32_t num_splits) {
  LayerWorkspace w{};
  const size_t B = static_cast<size_t>(batch > 0 ? batch : 0);
  const size_t nq = static_cast<size_t>(d->num_heads) * (d->d_nope + d->d_rope);
  const size_t nkv = static_cast<size_t>(d->d_c + d->d_rope);
  size_t off = 0;
  w.off_qkv32 = off;
  off = up256(off + B * (nq + nkv) * 4);
  w.off_q = off;
  off = up256(off + B * nq * 2);
  w.off_c = off;
  off = up256(off + B * d->d_c * 2);
  w.off_kr = off;
  off = up256(off + B * d->d_rope * 2);
  w.off_u = off;
  off = up256(off + B * d->num_heads * d->d_v * 2);
  w.off_dec = off;
  w.dec_bytes = eg_mla_decode_workspace_size(d, batch, num_splits);
  w.total = up256(off + w.dec_bytes);
  return w;
}

// The new token's kv_norm and rotary embedding (one CTA per sequence):
//   c^KV = c / sqrt(mean(c^2) + eps) * w,  k^R and every head's q^R rotated,
//   pair (2i, 2i + 1) by the angle pos * theta^(-2i / d_rope).
// Inputs are the fp32 GEMM outputs; each result is rounded to bf16 once.  The
// d_rope / 2 angles are formed and reduced to [-pi, pi] in double precision
// (the frequencies theta^(-2i/d_rope) come from the host in double), so that
// positions in the tens of thousands keep full fp32 accuracy in the rotation;
// sine and cosine of the reduced angle are taken in fp32, once per sequence,
// and shared through shared memory.  The rotations of the heads' q^R and of
// k^R are spread over all threads.
constexpr int kMaxRopePairs = 64;

struct RopeFreqs {
  double f[kMaxRopePairs];
};

__global__ void __launch_bounds__(kQkvThreads) layer_qkv_kernel(
    const float* __restrict__ qkv32, const int32_t* __restrict__ positions,
    const __nv_bfloat16* __restrict__ kv_norm_w, int H, int dn, int dr, int dc, const RopeFreqs freqs, float eps,
    int do_kv, __nv_bfloat16* __restrict__ q_out, __nv_bfloat16* __restrict__ c_out,
    __nv_bfloat16* __restrict__ kr_out) {
  __shared__ float red[kQkvThreads / 32];
  __shared__ float cs_s[kMaxRopePairs], sn_s[kMaxRopePairs];
  const int b = blockIdx.x, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int dq = dn + dr, np = dr / 2;
  const float* q = qkv32 + static_cast<size_t>(b) * (H * dq + dc + dr);   // [q (H dq) | c (dc) | k^R (dr)]
  const float* kv = q + H * dq;
  __nv_bfloat16* qo = q_out + static_cast<size_t>(b) * H * dq;

  if (tid < np) {
    constexpr double kTwoPi = 6.283185307179586, kInvTwoPi = 0.15915494309189535;
    const double ang = static_cast<double>(positions[b]) * freqs.f[tid];
    const double red_ang = fma(-rint(ang * kInvTwoPi), kTwoPi, ang);
    float sn, cs;
    sincosf(static_cast<float>(red_ang), &sn, &cs);
    sn_s[tid] = sn;
    cs_s[tid] = cs;
  }
  // kv_norm: the mean of c^2 over d_c (warp sums, then the warps' sums in order)
  float ss = 0.f;
  if (do_kv)
    for (int f = tid; f < dc; f += blockDim.x) ss = fmaf(kv[f], kv[f], ss);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
  if (lane == 0) red[warp] = ss;
  // q^C of every head, rounded
  for (int e = tid; e < H * dq; e += blockDim.x)
    if (e % dq < dn) qo[e] = __float2bfloat16_rn(q[e]);
  __syncthreads();
  float tot = 0.f;
  for (int i = 0; i < static_cast<int>(blockDim.x / 32); ++i) tot += red[i];
  const float r = 1.f / sqrtf(tot / static_cast<float>(dc) + eps);
  if (do_kv)
    for (int f = tid; f < dc; f += blockDim.x)
      c_out[static_cast<size_t>(b) * dc + f] = __float2bfloat16_rn(kv[f] * r * __bfloat162float(kv_norm_w[f]));
  // rotations: item (h, i) for h < H is pair i of head h's q^R, h = H is k^R
  for (int it = tid; it < (H + (do_kv ? 1 : 0)) * np; it += blockDim.x) {
    const int h = it / np, i = it % np;
    const float cs = cs_s[i], sn = sn_s[i];
    const float* src = h < H ? q + h * dq + dn : kv + dc;
    __nv_bfloat16* dst = h < H ? qo + h * dq + dn : kr_out + static_cast<size_t>(b) * dr;
    const float x0 = src[2 * i], x1 = src[2 * i + 1];
    dst[2 * i] = __float2bfloat16_rn(x0 * cs - x1 * sn);
    dst[2 * i + 1] = __float2bfloat16_rn(x0 * sn + x1 * cs);
  }
}

}  // namespace

extern "C" {

size_t eg_mla_layer_workspace_size(const eg_mla_dims* dims, const eg_mla_layer_dims* layer, int32_t batch,
                                   int32_t num_splits) {
  if (dims == nullptr || layer == nullptr || batch < 0 || layer->n_embd <= 0) return 0;
  if (dims->dtype != EG_MLA_BF16) return 0;
  const LayerWorkspace w = layer_workspace(dims, batch, num_splits);
  return w.dec_bytes == 0 ? 0 : w.total;
}

size_t eg_mla_layer_attn_offset(const eg_mla_dims* dims, const eg_mla_layer_dims* layer, int32_t batch,
                                int32_t num_splits) {
  if (eg_mla_layer_workspace_size(dims, layer, batch, num_splits) == 0) return 0;
  return layer_workspace(dims, batch, num_splits).off_u;
}

int eg_mla_layer_decode(const eg_mla_dims* dims, const eg_mla_layer_dims* layer, const eg_mla_layer_weights* wt,
                        const void* x, const int32_t* ids_new, const int32_t* positions, void* c_pool,
                        void* krope_pool, int32_t* id_pool, const int32_t* block_table, int32_t max_pages_per_seq,
                        const int32_t* seq_lens, int32_t max_seq_len, int32_t batch, int32_t num_pages, void* y,
                        int32_t num_splits, void* workspace, size_t workspace_bytes, int32_t* dev_status,
                        void* stream) {
  if (dims == nullptr || layer == nullptr || wt == nullptr) return EG_MLA_ERR_INVALID_ARG;
  if (dims->dtype != EG_MLA_BF16) return EG_MLA_ERR_UNSUPPORTED;
  if (batch < 0 || num_splits < 0 || layer->n_embd <= 0) return EG_MLA_ERR_INVALID_ARG;
  if (layer->n_embd % 8 || dims->d_rope % 2 || dims->d_rope > 2 * kMaxRopePairs) return EG_MLA_ERR_UNSUPPORTED;
  if (batch == 0) return EG_MLA_OK;
  if (!x || !positions || !y || !workspace || !wt->w_qkv_a || (layer->share_kv == 0 && !wt->kv_norm_w) || !wt->w_o)
    return EG_MLA_ERR_INVALID_ARG;
  if (!aligned16(x) || !aligned16(y) || !aligned16(wt->w_qkv_a) || !aligned16(wt->w_o)) return EG_MLA_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(workspace) & 255) != 0) return EG_MLA_ERR_INVALID_ARG;
  const LayerWorkspace ws = layer_workspace(dims, batch, num_splits);
  if (ws.dec_bytes == 0) return EG_MLA_ERR_INVALID_ARG;
  if (workspace_bytes < ws.total) return EG_MLA_ERR_WORKSPACE;
  uint8_t* base = static_cast<uint8_t*>(workspace);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const int H = dims->num_heads, E = layer->n_embd;
  const int nq = H * (dims->d_nope + dims->d_rope), nkv = dims->d_c + dims->d_rope, nu = H * dims->d_v;
  const double theta = layer->rope_theta > 0.f ? static_cast<double>(layer->rope_theta) : 10000.0;
  RopeFreqs freqs{};
  for (int i = 0; i < dims->d_rope / 2; ++i) freqs.f[i] = std::pow(theta, -2.0 * i / dims->d_rope);
  const float eps = layer->rms_eps > 0.f ? layer->rms_eps : 1.1920928955078125e-07f;
  void* qkv32 = base + ws.off_qkv32;
  auto* qb = reinterpret_cast<__nv_bfloat16*>(base + ws.off_q);
  auto* cb = reinterpret_cast<__nv_bfloat16*>(base + ws.off_c);
  auto* krb = reinterpret_cast<__nv_bfloat16*>(base + ws.off_kr);
  void* ub = base + ws.off_u;

  // the query and latent projections, fp32 out (a later layer of a layer
  // group projects only its query)
  const bool do_kv = layer->share_kv == 0;
  if (egmla::launch_linear_tc(wt->w_qkv_a, do_kv ? nq + nkv : nq, E, x, batch, qkv32, nq + nkv, true, dev_status,
                              st) != cudaSuccess)
    return EG_MLA_ERR_CUDA;
  layer_qkv_kernel<<<batch, kQkvThreads, 0, st>>>(
      static_cast<const float*>(qkv32), positions,
      static_cast<const __nv_bfloat16*>(wt->kv_norm_w), H, dims->d_nope, dims->d_rope, dims->d_c, freqs, eps,
      do_kv ? 1 : 0, qb, cb, krb);
  if (cudaGetLastError() != cudaSuccess) return EG_MLA_ERR_CUDA;
  // the append (first layer of a group) and the decode as one step
  const int rc = do_kv ? eg_mla_step(dims, c_pool, krope_pool, id_pool, cb, krb, ids_new, positions, qb, block_table,
                                     max_pages_per_seq, seq_lens, max_seq_len, batch, num_pages, wt->gate_table,
                                     wt->ln_gamma, wt->ln_beta, wt->w_uk, wt->w_uv, ub, num_splits, base + ws.off_dec,
                                     ws.dec_bytes, dev_status, stream)
                       : eg_mla_decode(dims, qb, c_pool, krope_pool, id_pool, block_table, max_pages_per_seq,
                                       seq_lens, max_seq_len, batch, num_pages, wt->gate_table, wt->ln_gamma,
                                       wt->ln_beta, wt->w_uk, wt->w_uv, ub, num_splits, base + ws.off_dec,
                                       ws.dec_bytes, dev_status, stream);
  if (rc != EG_MLA_OK) return rc;
  // Eq. 14: the output projection of the heads' concatenated outputs
  if (egmla::launch_linear_tc(wt->w_o, E, nu, ub, batch, y, E, false, dev_status, st) != cudaSuccess)
    return EG_MLA_ERR_CUDA;
  return EG_MLA_OK;
}

}  // extern "C"
