// egmla_linear.cu - the layer's projection GEMMs on tcgen05: out = x W^T for a
// Linear weight W [n_out, k] (bf16, row-major) and a small batch of rows x
// [batch, k] (decode: one token per sequence), fp32 or bf16 out.
//
// Decode projections are weight-streaming: every weight byte is used once per
// step, by at most 256 batch rows, so the kernel is bound by the HBM read of
// W.  Layout:
//   - a tile is 128 output features (the MMA's M, rows of W in TMEM lanes)
//     by the whole batch (the MMA's N, padded to a multiple of 16);
//   - the reduction dimension k is split over the CTAs of a thread-block
//     cluster (one CTA per SM); each CTA streams its k range of the tile's
//     weight rows in 64-element chunks by TMA (128-byte swizzle, the MMA's
//     K-major operand layout) through a ring of shared-memory stages, and one
//     elected thread issues four K = 16 MMAs per chunk into a TMEM
//     accumulator;
//   - the cluster's partial sums meet in distributed shared memory: batch
//     row b belongs to one rank; every rank bulk-copies its partials of the
//     owner's rows into a slot of the owner's shared memory (one copy per
//     owner, completing on the owner's mbarrier), and the owner adds the
//     slots in rank order (the result does not depend on timing) and writes
//     the rows out.
// The weight copies do not depend on the kernel before this one on the
// stream, so with programmatic stream serialisation they start before it has
// finished; the copies of x (its output) wait for it.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cstdint>
#include <cstring>
#include <mutex>

#include "egmla_kernels.h"
#include "egmla_ptx.cuh"

namespace egmla {
namespace {

constexpr int kLinThreads = 128;            // four warps: TMA, MMA, and all four in the epilogue
constexpr int kTileM = 128;                 // output features per tile
constexpr int kChunkK = 64;                 // k elements per stage (one 128-byte swizzle atom)
constexpr uint32_t kATileBytes = kTileM * kChunkK * 2;
constexpr int kMaxBatch = 128;              // batch rows per launch (partials and slots fit the stages)
constexpr int kMaxStages = 8;
constexpr int kMaxCluster = 8;
constexpr uint32_t kLinSmemLimit = 227 * 1024;

struct LinParams {
  void* out;
  int ldo;          // row stride of out, elements
  int out_f32;      // 1: fp32 out, 0: bf16 out
  int n_out, k, batch, bp;   // bp: batch padded to a multiple of 16
  int kchunks;      // ceil(k / 64)
  int stages;
  uint32_t stage_bytes;
  uint32_t slots_off;  // incoming partials of this CTA's batch rows, past the ring
  uint32_t bars_off;   // barrier block, past the slots
  uint64_t wait_ns;
  int32_t* status;
};

__device__ __forceinline__ uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}

__device__ __forceinline__ uint32_t cluster_size() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_nctarank;" : "=r"(r));
  return r;
}

__device__ __forceinline__ void cluster_sync() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}

// address of the same shared-memory location in CTA `rank` of the cluster
__device__ __forceinline__ uint32_t map_to_rank(uint32_t saddr, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(saddr), "r"(rank));
  return r;
}

// bulk copy of `bytes` from this CTA's shared memory to a shared::cluster
// address (another CTA's), completing as transaction bytes on the mbarrier at
// the shared::cluster address `bar` (in the destination CTA)
__device__ __forceinline__ void bulk_copy_to_rank(uint32_t dst, uint32_t src, uint32_t bytes, uint32_t bar) {
  asm volatile("cp.async.bulk.shared::cluster.shared::cta.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
               "r"(src), "r"(bytes), "r"(bar)
               : "memory");
}

// wait until every bulk copy this thread issued has finished reading its source
__device__ __forceinline__ void bulk_wait_reads() {
  asm volatile("cp.async.bulk.commit_group;\n\tcp.async.bulk.wait_group.read 0;" ::: "memory");
}

// every lane waits for the phase; false in all lanes if any lane's wait ran out
__device__ __forceinline__ bool warp_all_wait(uint32_t bar, uint32_t parity, volatile int* abort_flag,
                                              uint64_t limit_ns) {
  __syncwarp();
  const bool ok = mbar_wait(bar, parity, abort_flag, limit_ns);
  return __all_sync(0xffffffffu, ok);
}

struct LinBars {
  uint64_t full[kMaxStages], empty[kMaxStages];
  uint64_t done;
  uint64_t slots;   // every rank's partial of this CTA's batch rows landed
  uint32_t tmem_base;
  int abort;
};

__global__ void __launch_bounds__(kLinThreads, 1)
    linear_tc_kernel(const __grid_constant__ CUtensorMap wmap, const __grid_constant__ CUtensorMap xmap,
                     const LinParams p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  const uint32_t sbase = smem_u32(smem);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const uint32_t rank = cluster_rank(), nrank = cluster_size();
  const int n0 = blockIdx.y * kTileM;
  // the next projection (or kernel) on the stream may start streaming its
  // own weights as this kernel's CTAs leave the SMs
  grid_launch_dependents();
  // this CTA's chunks of the reduction dimension
  const int c_lo = static_cast<int>(rank) * p.kchunks / static_cast<int>(nrank);
  const int c_hi = (static_cast<int>(rank) + 1) * p.kchunks / static_cast<int>(nrank);
  const int nck = c_hi - c_lo;
  LinBars& bars = *reinterpret_cast<LinBars*>(smem + p.bars_off);
  volatile int* abort_flag = &bars.abort;
  uint32_t tmem_cols = 32;
  while (tmem_cols < static_cast<uint32_t>(p.bp)) tmem_cols <<= 1;

  // batch rows [b_first(o), b_first(o + 1)) belong to rank o
  const int share = (p.batch + static_cast<int>(nrank) - 1) / static_cast<int>(nrank);
  auto b_first = [&](int o) { return o * p.batch / static_cast<int>(nrank); };
  const int b_lo = b_first(static_cast<int>(rank)), b_hi = b_first(static_cast<int>(rank) + 1);
  const uint32_t xbytes = static_cast<uint32_t>(p.bp) * kChunkK * 2;
  const int first = nck < p.stages ? nck : p.stages;
  if (tid == 0) {
    for (int s = 0; s < p.stages; ++s) {
      mbar_init(smem_u32(&bars.full[s]), 1);
      mbar_init(smem_u32(&bars.empty[s]), 1);
    }
    mbar_init(smem_u32(&bars.done), 1);
    mbar_init(smem_u32(&bars.slots), 1);
    bars.abort = 0;
    fence_mbar_init();
    // what every rank will send here: its partial of this CTA's batch rows
    mbar_arrive_expect_tx(smem_u32(&bars.slots), static_cast<uint32_t>(nrank) * (b_hi - b_lo) * kTileM * 4);
    prefetch_tensormap(&wmap);
    prefetch_tensormap(&xmap);
    // the weight chunks of the first ring pass need nothing from the kernel
    // before this one (nor from the other ranks)
    const uint64_t pol_w = policy_evict_first();
    for (int i = 0; i < first; ++i) {
      mbar_arrive_expect_tx(smem_u32(&bars.full[i]), kATileBytes + xbytes);
      tma_load_2d(sbase + i * p.stage_bytes, &wmap, (c_lo + i) * kChunkK, n0, smem_u32(&bars.full[i]), pol_w);
    }
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(&bars.tmem_base), tmem_cols);
    tmem_relinquish();
  }
  tc_fence_before();
  // every rank's barriers are initialised (and expecting) before any rank's
  // copy can reach them
  cluster_sync();
  tc_fence_after();
  const uint32_t tmem = bars.tmem_base;

  if (warp == 0) {
    // ---- TMA producer: x (the kernel before this one wrote it) after the
    // wait, then the rest of the ring
    if (elect_one()) {
      const uint64_t pol_w = policy_evict_first();
      const uint64_t pol_x = policy_evict_last();
      grid_dependency_wait();
      for (int i = 0; i < first; ++i)
        tma_load_2d(sbase + i * p.stage_bytes + kATileBytes, &xmap, (c_lo + i) * kChunkK, 0,
                    smem_u32(&bars.full[i]), pol_x);
      int issued = first;
      for (int i = first; i < nck; ++i) {
        const int s = i % p.stages;
        if (!mbar_wait(smem_u32(&bars.empty[s]), ((i / p.stages) & 1) ^ 1, abort_flag, p.wait_ns)) break;
        mbar_arrive_expect_tx(smem_u32(&bars.full[s]), kATileBytes + xbytes);
        tma_load_2d(sbase + s * p.stage_bytes, &wmap, (c_lo + i) * kChunkK, n0, smem_u32(&bars.full[s]), pol_w);
        tma_load_2d(sbase + s * p.stage_bytes + kATileBytes, &xmap, (c_lo + i) * kChunkK, 0,
                    smem_u32(&bars.full[s]), pol_x);
        issued = i + 1;
      }
      // every copy issued must have landed before the stages are reused or the
      // CTA exits, also after an abort (own flag: bounded, not cut short)
      volatile int own = 0;
      for (int i = issued > p.stages ? issued - p.stages : 0; i < issued; ++i)
        if (!mbar_wait(smem_u32(&bars.full[i % p.stages]), (i / p.stages) & 1, &own, p.wait_ns)) *abort_flag = 1;
    }
    __syncwarp();
  } else if (warp == 1) {
    // ---- MMA issuer: D[n, b] += W[n, k] x[b, k] over this CTA's chunks
    const uint32_t idesc = idesc_bf16(kTileM, p.bp, 0, 0);
    for (int i = 0; i < nck; ++i) {
      const int s = i % p.stages;
      if (!warp_all_wait(smem_u32(&bars.full[s]), (i / p.stages) & 1, abort_flag, p.wait_ns)) break;
      tc_fence_after();
      if (elect_one()) {
        const uint64_t ad = smem_desc(sbase + s * p.stage_bytes, 16, 1024, kSwizzle128B);
        const uint64_t bd = smem_desc(sbase + s * p.stage_bytes + kATileBytes, 16, 1024, kSwizzle128B);
#pragma unroll
        for (int kk = 0; kk < kChunkK / 16; ++kk)
          mma_bf16_ss(tmem, ad + ((kk * 32) >> 4), bd + ((kk * 32) >> 4), idesc, (i > 0 || kk > 0) ? 1u : 0u);
        mma_commit(smem_u32(&bars.empty[s]));
      }
      __syncwarp();
    }
    if (elect_one()) mma_commit(smem_u32(&bars.done));
    __syncwarp();
  }
  // out may still be read by the kernel before this one (a no-op wait once
  // that kernel is done; taken here, off the epilogue's path)
  grid_dependency_wait();

  // ---- epilogue: this rank's accumulator into its stages as [batch][128]
  // fp32 (`part`), one bulk copy of owner o's rows into slot [this rank] of
  // o's slots ([cluster][rows per owner][128]); each owner adds its slots in
  // rank order and writes its rows out
  const int row = 32 * warp + lane;
  float* part = reinterpret_cast<float*>(smem);
  const float* slots = reinterpret_cast<const float*>(smem + p.slots_off);
  bool ok = true;
  if (nck > 0) ok = warp_all_wait(smem_u32(&bars.done), 0, abort_flag, p.wait_ns);
  // the producer's drain (every copy landed) and the done barrier (every MMA
  // finished reading) come before the stages are rewritten
  __syncthreads();
  ok = ok && *abort_flag == 0;
  tc_fence_after();
  for (int c0 = 0; c0 < p.batch; c0 += 16) {
    float v[16];
    if (nck > 0 && ok) {
      tmem_ld16(tmem + (static_cast<uint32_t>(32 * warp) << 16) + c0, v);
      tmem_wait_ld();
    } else {
#pragma unroll
      for (int j = 0; j < 16; ++j) v[j] = 0.f;
    }
#pragma unroll
    for (int j = 0; j < 16; ++j)
      if (c0 + j < p.batch) part[(c0 + j) * kTileM + row] = v[j];
  }
  tc_fence_before();
  fence_proxy_async_smem();   // the copies below read `part` through the async proxy
  __syncthreads();
  if (warp == 1) tmem_dealloc(tmem, tmem_cols);
  if (tid == 0) {
    for (uint32_t o = 0; o < nrank; ++o) {
      const int lo = b_first(static_cast<int>(o)), hi = b_first(static_cast<int>(o) + 1);
      if (hi > lo) {
        const uint32_t dst = smem_u32(smem + p.slots_off) + (rank * static_cast<uint32_t>(share)) * kTileM * 4;
        bulk_copy_to_rank(map_to_rank(dst, o), smem_u32(part + lo * kTileM), (hi - lo) * kTileM * 4,
                          map_to_rank(smem_u32(&bars.slots), o));
      }
    }
  }
  // every rank's slot of this CTA's rows (bounded: a missing copy is reported)
  if (!warp_all_wait(smem_u32(&bars.slots), 0, abort_flag, p.wait_ns)) ok = false;
  if (tid == 0 && *abort_flag) report_status(p.status, kStatusTimeout);
  const int n = n0 + row;
  for (int b = b_lo; b < b_hi; b += 4) {
    float acc[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
    for (int r = 0; r < kMaxCluster; ++r) {
      if (r < static_cast<int>(nrank)) {
#pragma unroll
        for (int j = 0; j < 4; ++j)
          if (b + j < b_hi) acc[j] += slots[(r * static_cast<uint32_t>(share) + (b + j - b_lo)) * kTileM + row];
      }
    }
    if (n < p.n_out) {
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        if (b + j < b_hi) {
          if (p.out_f32)
            static_cast<float*>(p.out)[static_cast<size_t>(b + j) * p.ldo + n] = acc[j];
          else
            static_cast<__nv_bfloat16*>(p.out)[static_cast<size_t>(b + j) * p.ldo + n] = __float2bfloat16_rn(acc[j]);
        }
      }
    }
  }
  // this CTA's outgoing copies have read `part` before it exits
  if (tid == 0) bulk_wait_reads();
  __syncthreads();
}

using EncodeFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                              const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                              CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeFn encode_fn() {
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

// row-major bf16 [rows, cols] with boxes of 64 columns x box_rows rows,
// 128-byte swizzle; rows past the end read as zero
bool encode_rows(CUtensorMap* map, const void* base, uint64_t rows, uint64_t cols, uint32_t box_rows) {
  EncodeFn enc = encode_fn();
  if (enc == nullptr) return false;
  const cuuint64_t dims[2] = {cols, rows};
  const cuuint64_t strides[1] = {cols * 2};
  const cuuint32_t box[2] = {static_cast<cuuint32_t>(kChunkK), box_rows};
  const cuuint32_t estr[2] = {1, 1};
  return enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// cluster size per (device, tiles, chunks, smem bytes): the largest that
// splits the reduction dimension, keeps one wave of CTAs on the SMs and lets
// every cluster be resident at once (a host-side occupancy query, cached)
struct ClusterEntry {
  int dev, tiles, kchunks, smem, choice;
};
struct ClusterCache {
  std::mutex mu;
  ClusterEntry e[16];
  int n = 0;
} g_cluster;

int pick_cluster(int tiles, int kchunks, int smem, int sms) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 1;
  std::lock_guard<std::mutex> lk(g_cluster.mu);
  for (int i = 0; i < g_cluster.n; ++i) {
    const ClusterEntry& c = g_cluster.e[i];
    if (c.dev == dev && c.tiles == tiles && c.kchunks == kchunks && c.smem == smem) return c.choice;
  }
  int best = 1;
  for (int s = std::min(kMaxCluster, kchunks); s > 1; --s) {
    if (tiles * s > sms) continue;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(s, tiles);
    cfg.blockDim = dim3(kLinThreads);
    cfg.dynamicSmemBytes = smem;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = s;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int nclusters = 0;
    if (cudaOccupancyMaxActiveClusters(&nclusters, linear_tc_kernel, &cfg) != cudaSuccess) {
      cudaGetLastError();
      continue;
    }
    if (nclusters >= tiles) {
      best = s;
      break;
    }
  }
  ClusterEntry& c = g_cluster.e[g_cluster.n < 16 ? g_cluster.n++ : 15];
  c = ClusterEntry{dev, tiles, kchunks, smem, best};
  return best;
}

// shared-memory plan for a launch of nb batch rows (padded to bp): the ring of
// stages (which the outgoing partials [nb][128] fp32 reuse), then the
// incoming slots ([cluster][rows per owner][128] fp32, at most nb + 8 rows),
// then the barrier block; false if two stages do not fit
struct SmemPlan {
  int stages;
  uint32_t stage_bytes, slots_off, bars_off;
  int smem;
};

bool plan_smem(int nb, int bp, SmemPlan& sp) {
  sp.stage_bytes = kATileBytes + static_cast<uint32_t>(bp) * kChunkK * 2;
  const uint32_t part_bytes = static_cast<uint32_t>(nb) * kTileM * 4;
  const uint32_t slot_bytes = static_cast<uint32_t>(nb + kMaxCluster) * kTileM * 4;
  const uint32_t fixed = slot_bytes + static_cast<uint32_t>(sizeof(LinBars)) + 16 + 1024;
  if (fixed >= kLinSmemLimit) return false;
  sp.stages = std::min(kMaxStages, static_cast<int>((kLinSmemLimit - fixed) / sp.stage_bytes));
  if (sp.stages < 2) return false;
  sp.slots_off = std::max(static_cast<uint32_t>(sp.stages) * sp.stage_bytes, part_bytes);
  sp.bars_off = (sp.slots_off + slot_bytes + 15u) & ~15u;
  sp.smem = static_cast<int>(sp.bars_off + sizeof(LinBars) + 1024);
  return sp.smem <= static_cast<int>(kLinSmemLimit);
}

}  // namespace

bool linear_tc_supported(int n_out, int k, int batch) {
  return n_out > 0 && k > 0 && k % 8 == 0 && batch >= 0;
}

cudaError_t linear_tc_plan(int n_out, int k, int batch, int* cluster, int* stages, int* max_clusters) {
  *cluster = *stages = *max_clusters = 0;
  if (n_out <= 0 || k <= 0 || batch <= 0) return cudaErrorInvalidValue;
  cudaError_t e = cudaFuncSetAttribute(linear_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(kLinSmemLimit));
  if (e != cudaSuccess) return e;
  int dev = 0, sms = 0;
  e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (e != cudaSuccess) return e;
  const int nb = std::min(kMaxBatch, batch);
  const int bp = (nb + 15) / 16 * 16;
  SmemPlan sp;
  if (!plan_smem(nb, bp, sp)) return cudaErrorInvalidConfiguration;
  const int st = sp.stages, smem = sp.smem;
  const int tiles = (n_out + kTileM - 1) / kTileM;
  const int kchunks = (k + kChunkK - 1) / kChunkK;
  *cluster = pick_cluster(tiles, kchunks, smem, sms);
  *stages = st;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(*cluster, tiles);
  cfg.blockDim = dim3(kLinThreads);
  cfg.dynamicSmemBytes = smem;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = *cluster;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  e = cudaOccupancyMaxActiveClusters(max_clusters, linear_tc_kernel, &cfg);
  return e;
}

cudaError_t launch_linear_tc(const void* w, int n_out, int k, const void* x, int batch, void* out, int ldo,
                             bool out_f32, int32_t* status, cudaStream_t st) {
  if (batch == 0) return cudaSuccess;
  static bool attr_set = false;
  if (!attr_set) {
    cudaError_t e = cudaFuncSetAttribute(linear_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(kLinSmemLimit));
    if (e != cudaSuccess) return e;
    attr_set = true;
  }
  int dev = 0, sms = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (e != cudaSuccess) return e;
  CUtensorMap wmap;
  std::memset(&wmap, 0, sizeof(wmap));
  if (!encode_rows(&wmap, w, static_cast<uint64_t>(n_out), static_cast<uint64_t>(k), kTileM))
    return cudaErrorInvalidValue;
  const int tiles = (n_out + kTileM - 1) / kTileM;
  const int kchunks = (k + kChunkK - 1) / kChunkK;
  for (int b0 = 0; b0 < batch; b0 += kMaxBatch) {
    const int nb = std::min(kMaxBatch, batch - b0);
    const int bp = (nb + 15) / 16 * 16;
    CUtensorMap xmap;
    std::memset(&xmap, 0, sizeof(xmap));
    const auto* xb = static_cast<const __nv_bfloat16*>(x) + static_cast<size_t>(b0) * k;
    if (!encode_rows(&xmap, xb, static_cast<uint64_t>(nb), static_cast<uint64_t>(k), static_cast<uint32_t>(bp)))
      return cudaErrorInvalidValue;
    LinParams p;
    p.out = out_f32 ? static_cast<void*>(static_cast<float*>(out) + static_cast<size_t>(b0) * ldo)
                    : static_cast<void*>(static_cast<__nv_bfloat16*>(out) + static_cast<size_t>(b0) * ldo);
    p.ldo = ldo;
    p.out_f32 = out_f32 ? 1 : 0;
    p.n_out = n_out;
    p.k = k;
    p.batch = nb;
    p.bp = bp;
    p.kchunks = kchunks;
    p.wait_ns = kWaitLimitNs;
    p.status = status;
    SmemPlan sp;
    if (!plan_smem(nb, bp, sp)) return cudaErrorInvalidConfiguration;
    p.stages = sp.stages;
    p.stage_bytes = sp.stage_bytes;
    p.slots_off = sp.slots_off;
    p.bars_off = sp.bars_off;
    const int smem = sp.smem;
    const int cl = pick_cluster(tiles, kchunks, smem, sms);
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(cl, tiles);
    cfg.blockDim = dim3(kLinThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = cl;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 2;
    e = cudaLaunchKernelEx(&cfg, linear_tc_kernel, wmap, xmap, p);
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

}  // namespace egmla
