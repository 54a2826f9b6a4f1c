// Platform floors for the chained verify layers: what a chain of dependent
// launches costs with no work in it, and how fast a chain of launches that
// only stream one layer's K/V bytes through shared memory (TMA) can go. These
// bound the fused layer kernel from below; they are measurement kernels, not
// part of the verify path, and live in their own library (libsdfloor.so).
//
// Both entry points capture `layers` launches into a CUDA graph on a stream of
// their own, replay it three times untimed, then time `reps` replays with CUDA
// events on that stream and return the mean time per launch.
#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace {

__device__ int g_floor_error;  // set by a wait that gave up (never in a healthy run)

constexpr int kWaitLimit = 1 << 22;  // try_wait rounds before a wait gives up

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}
__device__ __forceinline__ bool mbar_try(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n.reg .pred p;\nmbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\nselp.u32 %0, 1, 0, p;\n}"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}
// bounded wait: false (and the error word set) when the phase never completed
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity) {
  for (int i = 0; i < kWaitLimit; ++i)
    if (mbar_try(bar, parity)) return true;
  atomicExch(&g_floor_error, 1);
  return false;
}
__device__ __forceinline__ void griddep_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void griddep_launch() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

// An empty launch: the dependent-launch trigger, the dependency wait and, when
// tmem_cols > 0, the tensor-memory allocation and release of the layer kernel.
__global__ void floor_empty_kernel(int tmem_cols) {
  __shared__ uint32_t slot;
  griddep_launch();
  griddep_wait();
  if (tmem_cols > 0 && threadIdx.x < 32) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     static_cast<uint32_t>(__cvta_generic_to_shared(&slot))),
                 "r"(tmem_cols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncwarp();
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(slot), "r"(tmem_cols) : "memory");
  }
}

constexpr int kStageRows = 128;                  // 128 rows of 256 B: two 64-column boxes
constexpr int kStageBytes = kStageRows * 256;    // 32 KB
constexpr int kStreamThreads = 160;              // 4 consumer warps + 1 producer warp

// One CTA streams rows [blockIdx.x * rows_per_cta, +rows_per_cta) of a
// [rows][128] bf16 tensor through a ring of `stages` 32 KB slots: warp 4's
// elected lane issues the TMA boxes, the other four warps wait for each slot
// and hand it back. waitpos: 0 = dependency wait at the start, 1 = after the
// first ring fill is issued (the layer kernel's early prefix), 2 = at the end.
__global__ void __launch_bounds__(kStreamThreads, 1)
    floor_stream_kernel(const __grid_constant__ CUtensorMap tm, int rows_per_cta, int stages, int waitpos) {
  griddep_launch();
  if (waitpos == 0) griddep_wait();
  extern __shared__ uint8_t raw[];
  uint8_t* ring_ptr = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(raw) + 1023) & ~uintptr_t(1023));
  const uint32_t ring = static_cast<uint32_t>(__cvta_generic_to_shared(ring_ptr));
  const uint32_t full = ring + stages * kStageBytes;  // [stages] full barriers, then [stages] empty ones
  const uint32_t empty = full + 8 * stages;
  if (threadIdx.x == 0) {
    for (int s = 0; s < stages; ++s) {
      mbar_init(full + 8 * s, 1);
      mbar_init(empty + 8 * s, 4);
    }
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncthreads();
  const int n_tiles = rows_per_cta / kStageRows;
  const int row0 = blockIdx.x * rows_per_cta;
  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  if (warp == 4) {
    if (lane == 0) {
      for (int t = 0; t < n_tiles; ++t) {
        const int s = t % stages;
        if (t == stages && waitpos == 1) griddep_wait();
        if (t >= stages && !mbar_wait(empty + 8 * s, ((t / stages) - 1) & 1)) break;
        mbar_expect_tx(full + 8 * s, kStageBytes);
        const int y = row0 + t * kStageRows;
        for (int h = 0; h < 2; ++h)
          asm volatile(
              "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
              " [%0], [%1, {%3, %4}], [%2];" ::"r"(ring + s * kStageBytes + h * kStageRows * 128),
              "l"(reinterpret_cast<uint64_t>(&tm)), "r"(full + 8 * s), "r"(h * 64), "r"(y)
              : "memory");
      }
      if (waitpos == 1 && n_tiles <= stages) griddep_wait();
    }
    __syncwarp();
  } else {
    // the consumers see every slot complete, so no copy is in flight at exit
    for (int t = 0; t < n_tiles; ++t) {
      const int s = t % stages;
      if (!mbar_wait(full + 8 * s, (t / stages) & 1)) break;
      __syncwarp();
      if (lane == 0) mbar_arrive(empty + 8 * s);
    }
  }
  if (waitpos == 2) griddep_wait();
}

typedef CUresult (*EncodeTiled)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiled encoder() {
  static EncodeTiled fn = nullptr;
  if (!fn) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiled>(p);
  }
  return fn;
}

// Replays `graph` 3 times, then times `reps` replays; *us = mean per launch.
int time_graph(cudaGraph_t graph, cudaStream_t s, int layers, int reps, float* us) {
  cudaGraphExec_t exec;
  if (cudaGraphInstantiate(&exec, graph, 0) != cudaSuccess) return 3;
  cudaEvent_t e0, e1;
  cudaEventCreate(&e0);
  cudaEventCreate(&e1);
  int rc = 0;
  for (int i = 0; i < 3 && rc == 0; ++i)
    if (cudaGraphLaunch(exec, s) != cudaSuccess) rc = 4;
  if (rc == 0 && cudaStreamSynchronize(s) != cudaSuccess) rc = 5;
  if (rc == 0) {
    cudaEventRecord(e0, s);
    for (int i = 0; i < reps; ++i) cudaGraphLaunch(exec, s);
    cudaEventRecord(e1, s);
    if (cudaEventSynchronize(e1) != cudaSuccess) rc = 5;
  }
  float ms = 0.f;
  if (rc == 0) cudaEventElapsedTime(&ms, e0, e1);
  *us = ms * 1000.f / static_cast<float>(reps) / static_cast<float>(layers);
  cudaEventDestroy(e0);
  cudaEventDestroy(e1);
  cudaGraphExecDestroy(exec);
  return rc;
}

}  // namespace

extern "C" {

// The word set by a floor kernel's wait that gave up (0: none); cleared.
int sdfloor_take_error() {
  int v = 0, z = 0;
  if (cudaMemcpyFromSymbol(&v, g_floor_error, sizeof(int)) != cudaSuccess) return -1;
  cudaMemcpyToSymbol(g_floor_error, &z, sizeof(int));
  return v;
}

// `layers` chained empty launches of `ctas` CTAs of `threads` threads in
// clusters of `cluster`, each holding `smem_bytes` of dynamic shared memory
// and (tmem_cols > 0) allocating that many tensor-memory columns; every launch
// after the first is a programmatic dependent launch when pdl != 0.
// Returns 0, or a nonzero step code (1 bad arguments, 2 launch, 3-5 graph).
int sdfloor_empty_chain(int layers, int ctas, int cluster, int threads, int smem_bytes, int tmem_cols, int pdl,
                        int reps, float* us_per_launch) {
  if (layers <= 0 || ctas <= 0 || cluster <= 0 || ctas % cluster != 0 || threads <= 0 || threads > 1024 ||
      smem_bytes < 0 || smem_bytes > 227 * 1024 || reps <= 0 || !us_per_launch)
    return 1;
  if (tmem_cols != 0 && (tmem_cols < 32 || tmem_cols > 512 || (tmem_cols & (tmem_cols - 1)) != 0)) return 1;
  if (cudaFuncSetAttribute(floor_empty_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem_bytes) !=
      cudaSuccess)
    return 2;
  if (cluster > 8) cudaFuncSetAttribute(floor_empty_kernel, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
  cudaStream_t s;
  if (cudaStreamCreateWithFlags(&s, cudaStreamNonBlocking) != cudaSuccess) return 2;
  int rc = 0;
  cudaGraph_t graph = nullptr;
  cudaStreamBeginCapture(s, cudaStreamCaptureModeThreadLocal);
  for (int l = 0; l < layers && rc == 0; ++l) {
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute at[2];
    int na = 0;
    at[na].id = cudaLaunchAttributeClusterDimension;
    at[na].val.clusterDim.x = cluster;
    at[na].val.clusterDim.y = 1;
    at[na].val.clusterDim.z = 1;
    ++na;
    if (pdl && l > 0) {
      at[na].id = cudaLaunchAttributeProgrammaticStreamSerialization;
      at[na].val.programmaticStreamSerializationAllowed = 1;
      ++na;
    }
    cfg.gridDim = dim3(ctas, 1, 1);
    cfg.blockDim = dim3(threads, 1, 1);
    cfg.dynamicSmemBytes = smem_bytes;
    cfg.stream = s;
    cfg.attrs = at;
    cfg.numAttrs = na;
    if (cudaLaunchKernelEx(&cfg, floor_empty_kernel, tmem_cols) != cudaSuccess) rc = 2;
  }
  if (cudaStreamEndCapture(s, &graph) != cudaSuccess) {
    graph = nullptr;
    if (rc == 0) rc = 3;
  }
  if (rc == 0) rc = time_graph(graph, s, layers, reps, us_per_launch);
  if (graph) cudaGraphDestroy(graph);
  cudaStreamDestroy(s);
  return rc;
}

// `layers` chained launches, launch l streaming rows [l * rows_per_layer,
// (l + 1) * rows_per_layer) of the [layers * rows_per_layer][128] bf16 tensor
// at `base` (device memory, 16-byte aligned) over `ctas` CTAs (one or two a
// SM), 128-byte swizzled TMA boxes of 64 columns x 128 rows; every launch
// after the first is a programmatic dependent launch unless waitpos < 0, and
// waitpos = 0 / 1 / 2 places the dependency wait at the start / after the
// first ring fill / at the end. Rows past a layer's end read as zeros (a CTA's
// range is rounded up to whole 128-row stages). Return codes as above.
int sdfloor_stream_chain(void* base, long long rows_per_layer, int layers, int ctas, int waitpos, int reps,
                         float* us_per_launch) {
  if (!base || (reinterpret_cast<uintptr_t>(base) & 15) != 0 || rows_per_layer <= 0 ||
      rows_per_layer > (1ll << 31) - 1 || layers <= 0 || ctas <= 0 || ctas > 4096 || waitpos < -1 ||
      waitpos > 2 || reps <= 0 || !us_per_launch)
    return 1;
  EncodeTiled enc = encoder();
  if (!enc) return 2;
  int nsm = 0;
  cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, 0);
  long long per = (rows_per_layer + ctas - 1) / ctas;
  per = (per + kStageRows - 1) / kStageRows * kStageRows;
  const int tiles = static_cast<int>(per / kStageRows);
  const int max_stages = (ctas > nsm ? 96 : 192) * 1024 / kStageBytes;
  const int stages = tiles < max_stages ? tiles : max_stages;
  const int smem = stages * kStageBytes + 1024 + 16 * stages;
  if (cudaFuncSetAttribute(floor_stream_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) != cudaSuccess)
    return 2;
  cudaStream_t s;
  if (cudaStreamCreateWithFlags(&s, cudaStreamNonBlocking) != cudaSuccess) return 2;
  int rc = 0;
  cudaGraph_t graph = nullptr;
  cudaStreamBeginCapture(s, cudaStreamCaptureModeThreadLocal);
  for (int l = 0; l < layers && rc == 0; ++l) {
    CUtensorMap tm;
    const cuuint64_t dims[2] = {128, static_cast<cuuint64_t>(rows_per_layer)};
    const cuuint64_t strides[1] = {256};
    const cuuint32_t box[2] = {64, kStageRows}, es[2] = {1, 1};
    void* layer_base = static_cast<char*>(base) + static_cast<size_t>(l) * static_cast<size_t>(rows_per_layer) * 256;
    if (enc(&tm, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, layer_base, dims, strides, box, es,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS) {
      rc = 2;
      break;
    }
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.gridDim = dim3(ctas, 1, 1);
    cfg.blockDim = dim3(kStreamThreads, 1, 1);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cfg.attrs = at;
    cfg.numAttrs = (waitpos >= 0 && l > 0) ? 1 : 0;
    if (cudaLaunchKernelEx(&cfg, floor_stream_kernel, tm, static_cast<int>(per), stages,
                           waitpos < 0 ? 0 : waitpos) != cudaSuccess)
      rc = 2;
  }
  if (cudaStreamEndCapture(s, &graph) != cudaSuccess) {
    graph = nullptr;
    if (rc == 0) rc = 3;
  }
  if (rc == 0) rc = time_graph(graph, s, layers, reps, us_per_launch);
  if (graph) cudaGraphDestroy(graph);
  cudaStreamDestroy(s);
  return rc;
}

}  // extern "C"
