// K4: greedy acceptance (Eqs. verify, accept, commit, Sec. 3.2; Eq.
// accept-length, Sec. 4.3).
//
//   r*_j = argmax_v logits[b][j][v]   (lowest index among equal maxima)
//   l    = number of leading drafts equal to r*   (draft[j] vs r*_j, j < K)
//   emit draft[0..l-1], r*_l            n_emit = l + 1
//
// Cluster kernel (rows whose bytes are 16-byte aligned, the usual case): one
// thread-block cluster of up to 16 CTAs per (scene, row). CTA c scans the c-th
// slice of the row with 16-byte loads and sends its (value, index) to rank 0
// through distributed shared memory; rank 0 writes the row's argmax and takes
// the scene's ticket (one atomic per row); the scene's last row reads every
// row's argmax, compares with the drafts (read at kernel start) and writes
// the outputs. Other shapes take the chunked kernel: a CTA per (scene, row,
// chunk) writes a partial, and the last CTA of each scene (atomic ticket, no
// spin) reduces them. The (value desc, index asc) order is total, so both
// results do not depend on the order candidates are combined in: bit-exact
// and deterministic.
#include "common.cuh"

#include <mutex>

SD_DEFINE_ERROR_ACCESSOR(sd_take_error_greedy)

namespace {

constexpr int kThreads = 256;
constexpr int kMaxChunks = 1024;

struct Best {
  float v;
  int i;
};

// a beats b: larger value, or equal value (numerically: +0 == -0) and lower index.
__device__ __forceinline__ bool beats(float av, int ai, float bv, int bi) {
  return av > bv || (av == bv && ai < bi);
}

__device__ __forceinline__ void take(Best& best, float v, int i) {
  if (beats(v, i, best.v, best.i)) {
    best.v = v;
    best.i = i;
  }
}

__device__ __forceinline__ Best warp_best(Best b) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float ov = __shfl_xor_sync(0xffffffffu, b.v, o);
    const int oi = __shfl_xor_sync(0xffffffffu, b.i, o);
    take(b, ov, oi);
  }
  return b;
}

template <typename T>
__device__ __forceinline__ float load_one(const T* p, long long i);
template <>
__device__ __forceinline__ float load_one<float>(const float* p, long long i) { return p[i]; }
template <>
__device__ __forceinline__ float load_one<__nv_bfloat16>(const __nv_bfloat16* p, long long i) {
  return __bfloat162float(p[i]);
}

// Scan [lo, hi) of one row. Each thread keeps the first maximum of its own
// ascending subsequence; the cross-thread combine uses the full order.
template <typename T>
__device__ Best scan_chunk(const T* row, int lo, int hi, bool vec_ok) {
  Best best{-INFINITY, 0x7fffffff};
  constexpr int kPer = 16 / sizeof(T);  // elements per 16-byte vector
  int start = lo;
  if (vec_ok) {
    const int vlo = (lo + kPer - 1) / kPer * kPer;
    const int vhi = hi / kPer * kPer;
    // head and tail elements outside the aligned body
    for (int i = lo + threadIdx.x; i < min(vlo, hi); i += blockDim.x) take(best, load_one(row, i), i);
    for (int i = max(vhi, vlo) + threadIdx.x; i < hi; i += blockDim.x) take(best, load_one(row, i), i);
    for (int v = vlo / kPer + threadIdx.x; v < vhi / kPer; v += blockDim.x) {
      const uint4 w = __ldg(reinterpret_cast<const uint4*>(row) + v);
      const int base = v * kPer;
      if (sizeof(T) == 4) {
        take(best, __uint_as_float(w.x), base + 0);
        take(best, __uint_as_float(w.y), base + 1);
        take(best, __uint_as_float(w.z), base + 2);
        take(best, __uint_as_float(w.w), base + 3);
      } else {
        const uint32_t ws[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          take(best, sd_bf16_lo(ws[j]), base + 2 * j);
          take(best, sd_bf16_hi(ws[j]), base + 2 * j + 1);
        }
      }
    }
    start = hi;  // everything covered
  }
  for (int i = start + threadIdx.x; i < hi; i += blockDim.x) take(best, load_one(row, i), i);
  return best;
}

__device__ Best block_best(Best b) {
  __shared__ float sv[kThreads / 32];
  __shared__ int si[kThreads / 32];
  b = warp_best(b);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (lane == 0) {
    sv[warp] = b.v;
    si[warp] = b.i;
  }
  __syncthreads();
  if (warp == 0) {
    Best c{-INFINITY, 0x7fffffff};
    if (lane < kThreads / 32) c = Best{sv[lane], si[lane]};
    b = warp_best(c);
  }
  return b;  // valid in warp 0
}

template <typename T>
__global__ void __launch_bounds__(kThreads) greedy_kernel(const T* __restrict__ logits, int R, int V,
                                                          int chunk, int n_chunks,
                                                          const int32_t* __restrict__ draft,
                                                          int32_t* __restrict__ n_emit,
                                                          int32_t* __restrict__ tokens,
                                                          int32_t* __restrict__ argmax_out,
                                                          float2* __restrict__ part,
                                                          uint32_t* __restrict__ ticket) {
  const int c = blockIdx.x, r = blockIdx.y, b = blockIdx.z;
  sd_pdl_enter();  // a plain launch: no wait; a programmatic successor may become resident
  const T* row = logits + (static_cast<long long>(b) * R + r) * V;
  const bool vec_ok = ((static_cast<long long>(V) * sizeof(T)) % 16 == 0) &&
                      ((reinterpret_cast<uintptr_t>(logits) & 15) == 0);
  const int lo = c * chunk, hi = min(V, lo + chunk);
  Best best = block_best(scan_chunk(row, lo, hi, vec_ok));
  __shared__ bool s_last;
  if (threadIdx.x == 0) {
    part[(static_cast<long long>(b) * R + r) * n_chunks + c] = make_float2(best.v, __int_as_float(best.i));
    __threadfence();
    const uint32_t prev = atomicAdd(&ticket[b], 1u);
    s_last = prev == static_cast<uint32_t>(R * n_chunks - 1);
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  // ---- last CTA of scene b: reduce every row's partials, then accept
  __shared__ int s_star[32 * 4];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  for (int rr = warp; rr < R; rr += kThreads / 32) {
    Best w{-INFINITY, 0x7fffffff};
    const float2* pr = part + (static_cast<long long>(b) * R + rr) * n_chunks;
    for (int k = lane; k < n_chunks; k += 32) {
      const float2 e = __ldcg(pr + k);
      take(w, e.x, __float_as_int(e.y));
    }
    w = warp_best(w);
    if (lane == 0) {
      const int star = w.i == 0x7fffffff ? 0 : w.i;
      s_star[rr] = star;
      if (argmax_out) argmax_out[static_cast<long long>(b) * R + rr] = star;
    }
  }
  const int K = R - 1;
  __shared__ int s_draft[128];
  for (int j = threadIdx.x; j < K; j += kThreads) s_draft[j] = draft[static_cast<long long>(b) * K + j];
  __syncthreads();
  if (threadIdx.x == 0) {
    int ell = K;
    bool range_ok = true;
    for (int j = 0; j < K; ++j) {
      const int d = s_draft[j];
      if (d < 0 || d >= V) range_ok = false;
      if (ell == K && d != s_star[j]) ell = j;
    }
    if (!range_ok) sd_set_error(SD_DEVERR_TOKEN_RANGE);
    int32_t* tk = tokens + static_cast<long long>(b) * R;
    for (int j = 0; j < R; ++j) {
      int v = -1;
      if (j < ell) v = s_draft[j];
      else if (j == ell) v = s_star[ell];
      tk[j] = v;
    }
    n_emit[b] = ell + 1;
    ticket[b] = 0;  // re-arm for the next call
  }
}

// ------------------------------------------------------------ cluster kernel
constexpr int kCThreads = 512;
constexpr int kCWarps = kCThreads / 32;

// One cluster of csize CTAs per (scene b, row r): CTA c scans elements
// [c * slice, (c + 1) * slice) of the row with 16-byte loads, its best goes
// to rank 0's shared memory; rank 0 writes the row's best to rowbest[b][r]
// and takes the scene's ticket; the last row of the scene to finish reads
// every row's best and accepts. R atomics per scene.
template <typename T>
__global__ void __launch_bounds__(kCThreads, 1)
    greedy_cluster_kernel(const T* __restrict__ logits, int R, int V, int slice,
                          const int32_t* __restrict__ draft, int32_t* __restrict__ n_emit,
                          int32_t* __restrict__ tokens, int32_t* __restrict__ argmax_out,
                          float2* __restrict__ rowbest, uint32_t* __restrict__ ticket) {
  __shared__ float2 s_wbest[kCWarps];
  __shared__ float2 s_cand[16];
  __shared__ int s_draft[128];
  __shared__ int s_star[128];
  __shared__ bool s_last;
  const int rank = blockIdx.x, csize = gridDim.x, r = blockIdx.y, b = blockIdx.z;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int K = R - 1;
  sd_pdl_enter();  // a plain launch: no wait; a programmatic successor may become resident
  if (rank == 0)  // read early: only the scene's last row uses them
    for (int j = threadIdx.x; j < K; j += kCThreads) s_draft[j] = __ldg(draft + static_cast<long long>(b) * K + j);
  const T* row = logits + (static_cast<long long>(b) * R + r) * V;
  const int lo = rank * slice, hi = min(V, lo + slice);
  Best best = warp_best(scan_chunk(row, lo, hi, true));
  if (lane == 0) s_wbest[warp] = make_float2(best.v, __int_as_float(best.i));
  __syncthreads();
  if (warp == 0) {
    Best c{-INFINITY, 0x7fffffff};
    if (lane < kCWarps) c = Best{s_wbest[lane].x, __float_as_int(s_wbest[lane].y)};
    c = warp_best(c);
    if (lane == 0) {
      uint32_t dst;
      asm volatile("mapa.shared::cluster.u32 %0, %1, 0;"
                   : "=r"(dst)
                   : "r"(static_cast<uint32_t>(__cvta_generic_to_shared(s_cand + rank))));
      asm volatile("st.shared::cluster.v2.f32 [%0], {%1, %2};" ::"r"(dst), "f"(c.v), "f"(__int_as_float(c.i))
                   : "memory");
    }
  }
  asm volatile("barrier.cluster.arrive.release.aligned;" ::: "memory");
  asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory");
  if (rank != 0 || warp != 0) return;
  // ---- rank 0, warp 0: the row's best, then the scene's ticket
  Best w{-INFINITY, 0x7fffffff};
  if (lane < csize) w = Best{s_cand[lane].x, __float_as_int(s_cand[lane].y)};
  w = warp_best(w);
  if (lane == 0) {
    const int star = w.i == 0x7fffffff ? 0 : w.i;
    if (argmax_out) argmax_out[static_cast<long long>(b) * R + r] = star;
    rowbest[static_cast<long long>(b) * R + r] = make_float2(0.f, __int_as_float(star));
    __threadfence();
    s_last = atomicAdd(&ticket[b], 1u) == static_cast<uint32_t>(R - 1);
  }
  __syncwarp();
  if (!s_last) return;
  __threadfence();
  for (int j = lane; j < R; j += 32) s_star[j] = __float_as_int(__ldcg(rowbest + static_cast<long long>(b) * R + j).y);
  __syncwarp();
  // l = first j < K with draft[j] != r*_j (K when none): one ballot per 32 drafts
  int ell = K;
  bool range_ok = true;
  for (int j0 = 0; j0 < K && ell == K; j0 += 32) {
    const int j = j0 + lane;
    const bool live = j < K;
    const int d = live ? s_draft[j] : 0;
    range_ok &= !live || (d >= 0 && d < V);
    const uint32_t miss = __ballot_sync(0xffffffffu, live && d != s_star[live ? j : 0]);
    if (miss) ell = j0 + __ffs(miss) - 1;
  }
  for (int j = ell + 1 + lane; j < K; j += 32) {  // drafts past the first mismatch: range only
    const int d = s_draft[j];
    range_ok &= d >= 0 && d < V;
  }
  if (!__all_sync(0xffffffffu, range_ok) && lane == 0) sd_set_error(SD_DEVERR_TOKEN_RANGE);
  int32_t* tk = tokens + static_cast<long long>(b) * R;
  for (int j = lane; j < R; j += 32) tk[j] = j < ell ? s_draft[j] : (j == ell ? s_star[ell] : -1);
  if (lane == 0) {
    n_emit[b] = ell + 1;
    ticket[b] = 0;  // re-arm for the next call
  }
}

// Cluster size (rows of about 16 KB per CTA, at most 16) and the slice each
// CTA scans (a multiple of 16 bytes); 0 when the shape is left to the chunked
// kernel.
int max_cluster();

int cluster_slice(int R, int V, int elem_bytes, int* slice) {
  if ((static_cast<long long>(V) * elem_bytes) % 16 != 0 || R > 128) return 0;
  const int per = 16 / elem_bytes;
  long long cs = (static_cast<long long>(V) * elem_bytes + 16383) / 16384;
  cs = cs < 1 ? 1 : (cs > 16 ? 16 : cs);
  const int cmax = max_cluster();
  if (cmax <= 0) return 0;
  if (cs > cmax) cs = cmax;
  *slice = static_cast<int>(((V + cs - 1) / cs + per - 1) / per * per);
  return static_cast<int>(cs);
}

// Largest cluster size (16 or 8) that can run on this device; 0 when neither
// (or the attribute calls fail).
int max_cluster() {
  static int cache[64];
  static bool done[64];
  static std::mutex mu;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) {
    (void)cudaGetLastError();
    return 0;
  }
  std::lock_guard<std::mutex> lock(mu);
  if (!done[dev]) {
    done[dev] = true;
    const void* kerns[2] = {reinterpret_cast<const void*>(greedy_cluster_kernel<float>),
                            reinterpret_cast<const void*>(greedy_cluster_kernel<__nv_bfloat16>)};
    bool ok = true;
    for (const void* k : kerns)
      ok = ok && cudaFuncSetAttribute(k, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) == cudaSuccess;
    int best = 0;
    if (ok) {
      for (int cs : {16, 8}) {
        cudaLaunchConfig_t cfg = {};
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeClusterDimension;
        attr[0].val.clusterDim.x = cs;
        attr[0].val.clusterDim.y = 1;
        attr[0].val.clusterDim.z = 1;
        cfg.gridDim = dim3(cs, 1, 1);
        cfg.blockDim = dim3(kCThreads, 1, 1);
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        int nclusters = 0;
        if (cudaOccupancyMaxActiveClusters(&nclusters, kerns[1], &cfg) == cudaSuccess && nclusters > 0) {
          best = cs;
          break;
        }
        (void)cudaGetLastError();
      }
    } else {
      (void)cudaGetLastError();
    }
    cache[dev] = best;
  }
  return cache[dev];
}

// Chunking depends on V only (never on the device), so the workspace size
// is the same wherever it is queried: 4096 elements per CTA, more when the
// row would need over kMaxChunks chunks.
void plan(int B, int R, int V, int* chunk, int* n_chunks) {
  (void)B;
  (void)R;
  long long ch = 4096;
  while ((V + ch - 1) / ch > kMaxChunks) ch *= 2;
  *chunk = static_cast<int>(ch);
  *n_chunks = static_cast<int>((V + ch - 1) / ch);
}

size_t ws_bytes_for(int B, int R, int n_chunks) {
  return static_cast<size_t>(B) * R * n_chunks * sizeof(float2) + static_cast<size_t>(B) * 4 + 256;
}

}  // namespace

extern "C" size_t sd_accept_greedy_workspace(int B, int K, int V) {
  if (B <= 0 || K < 0 || V <= 0) return 0;
  int chunk, n_chunks;
  plan(B, K + 1, V, &chunk, &n_chunks);
  return ws_bytes_for(B, K + 1, n_chunks);
}

// Host-side argument checks shared by both entry points.
static sd_status check_args(const void* logits, sd_dtype dtype, int B, int K, int V,
                            const int32_t* draft, int32_t* n_emit, int32_t* tokens) {
  if (B < 0 || K < 0 || V <= 0) return SD_ERR_INVALID_ARG;
  if (dtype != SD_BF16 && dtype != SD_F32) return SD_ERR_INVALID_ARG;
  if (K + 1 > 128 || B > 65535) return SD_ERR_UNSUPPORTED;
  if (B == 0) return SD_OK;
  if (!logits || !n_emit || !tokens || (K > 0 && !draft)) return SD_ERR_INVALID_ARG;
  return SD_OK;
}

// The cluster kernel when the shape allows it; true when it was launched (or
// the launch failed: *status says which). rowbest takes the first B * R
// entries of the partials.
static bool launch_cluster(const void* logits, sd_dtype dtype, int B, int K, int V,
                           const int32_t* draft, int32_t* n_emit, int32_t* tokens, int32_t* argmax,
                           float2* rowbest, uint32_t* ticket, cudaStream_t st, sd_status* status) {
  const int R = K + 1;
  const int eb = dtype == SD_BF16 ? 2 : 4;
  if ((reinterpret_cast<uintptr_t>(logits) & 15) != 0) return false;
  int slice = 0;
  const int cs = cluster_slice(R, V, eb, &slice);
  if (cs <= 0) return false;
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = cs;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.gridDim = dim3(cs, R, B);
  cfg.blockDim = dim3(kCThreads, 1, 1);
  cfg.stream = st;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  cudaError_t e;
  if (dtype == SD_BF16)
    e = cudaLaunchKernelEx(&cfg, greedy_cluster_kernel<__nv_bfloat16>, static_cast<const __nv_bfloat16*>(logits),
                           R, V, slice, draft, n_emit, tokens, argmax, rowbest, ticket);
  else
    e = cudaLaunchKernelEx(&cfg, greedy_cluster_kernel<float>, static_cast<const float*>(logits), R, V, slice,
                           draft, n_emit, tokens, argmax, rowbest, ticket);
  if (e != cudaSuccess) {
    (void)cudaGetLastError();
    *status = SD_ERR_CUDA;
  } else {
    *status = SD_OK;
  }
  return true;
}

static sd_status launch(const void* logits, sd_dtype dtype, int B, int K, int V,
                        const int32_t* draft, int32_t* n_emit, int32_t* tokens, int32_t* argmax,
                        float2* part, uint32_t* ticket, int chunk, int n_chunks,
                        cudaStream_t st) {
  sd_status cs_status;
  if (launch_cluster(logits, dtype, B, K, V, draft, n_emit, tokens, argmax, part, ticket, st, &cs_status))
    return cs_status;
  const int R = K + 1;
  const dim3 grid(n_chunks, R, B);
  if (dtype == SD_BF16)
    greedy_kernel<__nv_bfloat16><<<grid, kThreads, 0, st>>>(
        static_cast<const __nv_bfloat16*>(logits), R, V, chunk, n_chunks, draft, n_emit, tokens,
        argmax, part, ticket);
  else
    greedy_kernel<float><<<grid, kThreads, 0, st>>>(static_cast<const float*>(logits), R, V, chunk,
                                                    n_chunks, draft, n_emit, tokens, argmax, part,
                                                    ticket);
  SD_CHECK_LAUNCH();
  return SD_OK;
}

extern "C" sd_status sd_accept_greedy(const void* logits, sd_dtype dtype, int B, int K, int V,
                                      const int32_t* draft, int32_t* n_emit, int32_t* tokens,
                                      int32_t* argmax, void* ws, size_t ws_bytes,
                                      sd_stream_t stream) {
  const sd_status chk = check_args(logits, dtype, B, K, V, draft, n_emit, tokens);
  if (chk != SD_OK || B == 0) return chk;
  const int R = K + 1;
  int chunk, n_chunks;
  plan(B, R, V, &chunk, &n_chunks);
  const size_t need = ws_bytes_for(B, R, n_chunks);
  if (!ws || ws_bytes < need || !sd_aligned16(ws)) return SD_ERR_WORKSPACE;
  auto* part = static_cast<float2*>(ws);
  auto* ticket = reinterpret_cast<uint32_t*>(static_cast<char*>(ws) +
                                             static_cast<size_t>(B) * R * n_chunks * sizeof(float2));
  return launch(logits, dtype, B, K, V, draft, n_emit, tokens, argmax, part, ticket, chunk, n_chunks,
                reinterpret_cast<cudaStream_t>(stream));
}

// ---------------------------------------------------------------------------
// Allocation-free variant. Some callers cannot allocate device memory at the
// point where they accept drafts: a serving loop whose memory pool is owned
// and fully carved up by another runtime, a pre-planned inference graph that
// forbids allocation once it runs, or an embedded host that has no device
// allocator at all. For them the scratch this kernel needs lives in a
// file-scope device array of fixed size, loaded with the library (every GPU
// that loads it holds these bytes until the process exits).
//
// Layout: tickets of up to kNoAllocMaxB scenes at the front, so their place
// never moves with the call's shape and no partial result lands on them; the
// per-chunk partials follow. The array starts zeroed when the module loads,
// and every completed call leaves the tickets at zero again; the partials
// need no clearing. All calls share the array: calls that overlap on the GPU
// (other streams, other threads) race and must not be issued.
// ---------------------------------------------------------------------------
constexpr size_t kNoAllocBytes = size_t(1) << 20;  // 1 MiB
constexpr int kNoAllocMaxB = 4096;
constexpr size_t kNoAllocTicketBytes = kNoAllocMaxB * sizeof(uint32_t);
static __device__ __align__(256) unsigned char g_greedy_scratch[kNoAllocBytes];

// Device address of the array on the current device, resolved once per device
// (host code cannot use the symbol itself: it is a host-side stand-in).
static void* noalloc_scratch() {
  static void* ptrs[64] = {nullptr};
  static std::mutex mu;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) {
    (void)cudaGetLastError();
    return nullptr;
  }
  std::lock_guard<std::mutex> lock(mu);
  if (!ptrs[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_greedy_scratch) != cudaSuccess || !p) {
      (void)cudaGetLastError();
      return nullptr;
    }
    ptrs[dev] = p;
  }
  return ptrs[dev];
}

extern "C" size_t sd_accept_greedy_noalloc_max_bytes(void) { return kNoAllocBytes; }

extern "C" sd_status sd_accept_greedy_noalloc(const void* logits, sd_dtype dtype, int B, int K,
                                              int V, const int32_t* draft, int32_t* n_emit,
                                              int32_t* tokens, int32_t* argmax,
                                              sd_stream_t stream) {
  const sd_status chk = check_args(logits, dtype, B, K, V, draft, n_emit, tokens);
  if (chk != SD_OK || B == 0) return chk;
  const int R = K + 1;
  int chunk, n_chunks;
  plan(B, R, V, &chunk, &n_chunks);
  const size_t part_bytes = static_cast<size_t>(B) * R * n_chunks * sizeof(float2);
  if (B > kNoAllocMaxB || kNoAllocTicketBytes + part_bytes > kNoAllocBytes) return SD_ERR_WORKSPACE;
  void* scratch = noalloc_scratch();
  if (!scratch) return SD_ERR_CUDA;
  auto* ticket = static_cast<uint32_t*>(scratch);
  auto* part = reinterpret_cast<float2*>(static_cast<char*>(scratch) + kNoAllocTicketBytes);
  return launch(logits, dtype, B, K, V, draft, n_emit, tokens, argmax, part, ticket, chunk, n_chunks,
                reinterpret_cast<cudaStream_t>(stream));
}
