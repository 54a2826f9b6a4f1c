// Attention budget of the verify rows (Sec. 4.2 "Empirical confirmation",
// Table tab:attn-budget): for every (scene, row, query head), the share of
// the row's softmax mass on the visual keys, on the trajectory / prompt-text
// keys and on the rows generated in this step, and the entropy of the
// attention among the non-visual keys (renormalised), divided by the log of
// their number.
//
// A diagnostic beside the verify path. One thread-block cluster per (KV head,
// scene) splits the visible keys over its S CTAs; the G * R query rows of the
// KV head (packed row p = i * G + j: new row i, query head j of the group)
// take their scores from bf16 tensor-core products (mma.sync m16n8k16, fp32
// accumulation), 16 rows by 8 keys a product, the keys' fragments read
// straight from the cache. Every thread folds the scores it holds into an
// online state per row, relative to a running maximum m:
//   v, t, g = sum of exp(y - m) over the visual, trajectory / prompt-text and
//             generated keys, n = sum over the non-visual keys of
//             exp(y - m) (y - m),        y = q . k * scale,
// the states merge in a fixed order over the lanes and warps, then over the
// cluster's CTAs through distributed shared memory (rank 0 takes the S
// partials), and
//
//   entropy = (ln l' - n / l') / ln N'     l' = t + g, N' = number of
//                                          non-visual keys the row sees
#include "common.cuh"

#include <cuda.h>  // CUtensorMap and its enums (header only; no libcuda link)

#include <math.h>
#include <mutex>

SD_DEFINE_ERROR_ACCESSOR(sd_take_error_budget)

namespace {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr float kLog2e = 1.4426950408889634f;

__device__ __forceinline__ float ex2f(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Online state of one row (see the header): sums relative to the maximum m.
struct RowState {
  float m, v, t, g, n;
};

__device__ __forceinline__ RowState row_empty() { return RowState{-INFINITY, 0.f, 0.f, 0.f, 0.f}; }

// fold two scores (y[e] of segment seg[e]; -inf: masked) whose block
// maximum over the row's lanes is bm: one rescale of the state at most
__device__ __forceinline__ void row_block(RowState& s, const float (&y)[2], const int (&seg)[2], float bm) {
  if (bm == -INFINITY) return;
  if (bm > s.m) {
    if (s.m != -INFINITY) {
      const float a = ex2f((s.m - bm) * kLog2e);
      s.n = a * fmaf(s.m - bm, s.t + s.g, s.n);
      s.v *= a;
      s.t *= a;
      s.g *= a;
    }
    s.m = bm;
  }
#pragma unroll
  for (int e = 0; e < 2; ++e) {
    const float d = y[e] - s.m, w = ex2f(d * kLog2e);  // masked: ex2(-inf) = 0
    if (seg[e] == 0) {
      s.v += w;
    } else {
      if (seg[e] == 1) s.t += w;
      else s.g += w;
      if (w > 0.f) s.n = fmaf(w, d, s.n);
    }
  }
}

// a := merge(a, b), both relative to their own maxima
__device__ __forceinline__ void row_merge(RowState& a, const RowState& b) {
  if (b.m == -INFINITY) return;
  if (a.m == -INFINITY) {
    a = b;
    return;
  }
  const float M = fmaxf(a.m, b.m);
  const float fa = ex2f((a.m - M) * kLog2e), fb = ex2f((b.m - M) * kLog2e);
  const float n = fa * fmaf(a.m - M, a.t + a.g, a.n) + fb * fmaf(b.m - M, b.t + b.g, b.n);
  a.v = fa * a.v + fb * b.v;
  a.t = fa * a.t + fb * b.t;
  a.g = fa * a.g + fb * b.g;
  a.n = n;
  a.m = M;
}

__device__ __forceinline__ RowState row_shfl(const RowState& s, int o) {
  return RowState{__shfl_xor_sync(0xffffffffu, s.m, o), __shfl_xor_sync(0xffffffffu, s.v, o),
                  __shfl_xor_sync(0xffffffffu, s.t, o), __shfl_xor_sync(0xffffffffu, s.g, o),
                  __shfl_xor_sync(0xffffffffu, s.n, o)};
}

__device__ __forceinline__ uint32_t cta_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
// 8 floats (two 16-byte loads) of CTA `rank`'s copy of p
__device__ __forceinline__ void ld_cluster8(const float* p, uint32_t rank, float (&v)[8]) {
  uint32_t a;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(a) : "r"(static_cast<uint32_t>(__cvta_generic_to_shared(p))), "r"(rank));
  asm volatile("ld.shared::cluster.v4.f32 {%0,%1,%2,%3}, [%4];" : "=f"(v[0]), "=f"(v[1]), "=f"(v[2]), "=f"(v[3]) : "r"(a) : "memory");
  asm volatile("ld.shared::cluster.v4.f32 {%0,%1,%2,%3}, [%4];" : "=f"(v[4]), "=f"(v[5]), "=f"(v[6]), "=f"(v[7]) : "r"(a + 16) : "memory");
}
__device__ __forceinline__ void cluster_sync_all() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}

__device__ __forceinline__ void mma_bf16(float (&c)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
  asm(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// grid (S, Hkv, B), clusters of S CTAs along x: CTA `rank` of the cluster of
// (KV head kvh, scene b) takes keys [rank * n / S, (rank + 1) * n / S) of the
// n = len[b] keys the scene holds, for the M = G * R packed rows in passes of
// kTiles tiles of 16 rows (lane l of a warp holds rows l / 4 and l / 4 + 8 of
// a tile, keys 2 (l % 4) and 2 (l % 4) + 1 of every 8-key block); a block's
// key fragments serve every tile of the pass.
constexpr int kTiles = 2;
constexpr int kPassRows = 16 * kTiles;
constexpr int kChunkKeys = 320;  // keys a CTA stages at once (10 boxes of 32)

// two CTAs an SM (at most 128 registers a thread), so that clusters of 16
// need only 8 SMs of a GPC and every cluster of a launch fits in one wave
template <int D>
__global__ void __launch_bounds__(kThreads, 2)
    budget_kernel(const __grid_constant__ CUtensorMap tm_k, const __nv_bfloat16* __restrict__ q,
                  const int32_t* __restrict__ len, const int32_t* __restrict__ n_visual, int R, int Hq,
                  int Hkv, int cap, float scale, float* __restrict__ mass, float* __restrict__ entropy) {
  __shared__ RowState red[kWarps][kPassRows];
  __shared__ __align__(16) float part[kPassRows][8];  // this CTA's state per row of the pass (read by rank 0)
  __shared__ RowState gath[kPassRows][16];           // rank 0: every CTA's state per row
  const int kvh = blockIdx.y, b = blockIdx.z;
  const int S = gridDim.x;
  const uint32_t rank = cta_rank();
  // a programmatic dependent launch: resident while the kernel before it
  // runs, reading nothing before it has completed
  sd_pdl_enter();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int gq = lane >> 2, tq = lane & 3;
  const int G = Hq / Hkv, M = G * R;
  const int n_keys = len[b], L = n_keys - R;
  int nv = n_visual[b];
  // every CTA of a cluster runs the same barriers, so a bad length only
  // empties the key ranges (and writes nothing)
  const bool ok = L >= 0 && n_keys <= cap;
  if (!ok && threadIdx.x == 0 && kvh == 0 && rank == 0) sd_set_error(SD_DEVERR_LENGTH);
  if (ok && (nv < 0 || nv > L)) {
    if (threadIdx.x == 0 && kvh == 0 && rank == 0) sd_set_error(SD_DEVERR_LENGTH);
    nv = nv < 0 ? 0 : L;
  }
  const int k_lo = ok ? static_cast<int>(static_cast<long long>(rank) * n_keys / S) : 0;
  const int k_hi = ok ? static_cast<int>(static_cast<long long>(rank + 1) * n_keys / S) : 0;
  // the CTA's keys are staged in shared memory a chunk of up to kChunkKeys at
  // a time (one TMA round trip a chunk): 32-key boxes of 64 columns with the
  // 128-byte swizzle, one region per 64-column half
  extern __shared__ uint8_t smem_raw[];
  const uint32_t kbuf = (static_cast<uint32_t>(__cvta_generic_to_shared(smem_raw)) + 1023u) & ~1023u;
  __shared__ __align__(8) uint64_t chunk_bar;
  const uint32_t bar = static_cast<uint32_t>(__cvta_generic_to_shared(&chunk_bar));
  if (threadIdx.x == 0) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(bar) : "memory");
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncthreads();
  const int n_chunks = (k_hi - k_lo + kChunkKeys - 1) / kChunkKeys;
  int loaded = -1;
  uint32_t phase = 0;
  for (int m0 = 0; m0 < M; m0 += kPassRows) {
    // query fragments of rows m0 + 16 u + gq and + 8 (zero past M); the keys
    // each row sees (causal over the new rows); one state per row
    uint32_t af[kTiles][D / 16][4];
    int lim[kTiles][2];
    RowState st[kTiles][2];
#pragma unroll
    for (int u = 0; u < kTiles; ++u)
#pragma unroll
      for (int h2 = 0; h2 < 2; ++h2) {
        const int p = m0 + 16 * u + gq + 8 * h2, i = p / G;
        const __nv_bfloat16* qr = q + ((static_cast<long long>(b) * R + i) * Hq + kvh * G + (p - i * G)) * D;
#pragma unroll
        for (int ks = 0; ks < D / 16; ++ks) {
          const int d0 = ks * 16 + 2 * tq;
          af[u][ks][h2] = p < M ? *reinterpret_cast<const uint32_t*>(qr + d0) : 0u;
          af[u][ks][h2 + 2] = p < M ? *reinterpret_cast<const uint32_t*>(qr + d0 + 8) : 0u;
        }
        lim[u][h2] = p < M ? L + i : -1;
        st[u][h2] = row_empty();
      }
#pragma unroll 1
    for (int ci = 0; ci < n_chunks; ++ci) {  // block-uniform
      const int c0 = k_lo + ci * kChunkKeys, nk = min(kChunkKeys, k_hi - c0);
      if (loaded != ci) {
        __syncthreads();  // every warp is done with the chunk in place
        if (threadIdx.x == 0) {
          const int nbox = (nk + 31) / 32;
          asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar),
                       "r"(static_cast<uint32_t>(nbox * 32 * 128 * (D / 64)))
                       : "memory");
          for (int bx = 0; bx < nbox; ++bx)
#pragma unroll
            for (int hf = 0; hf < D / 64; ++hf)
              asm volatile(
                  "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
                  " [%0], [%1, {%3, %4, %5}], [%2];" ::"r"(kbuf + hf * kChunkKeys * 128 + bx * 32 * 128),
                  "l"(reinterpret_cast<uint64_t>(&tm_k)), "r"(bar), "r"(hf * 64), "r"(c0 + bx * 32),
                  "r"(b * Hkv + kvh)
                  : "memory");
        }
        // bounded wait on the chunk's copies
        uint32_t done = 0;
        for (uint32_t it = 0; it < (1u << 22) && !done; ++it)
          asm volatile(
              "{\n\t.reg .pred p;\n\tmbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
              "selp.u32 %0, 1, 0, p;\n\t}"
              : "=r"(done)
              : "r"(bar), "r"(phase)
              : "memory");
        if (!done && threadIdx.x == 0) sd_set_error(SD_DEVERR_TIMEOUT);
        phase ^= 1u;
        loaded = ci;
      }
#pragma unroll 1
    for (int kb = 8 * warp; kb < nk; kb += 8 * kWarps) {
      const int kb0 = c0 + kb;  // the block's first key
      // B fragments of the block's 8 keys from the staged rows: ldmatrix of
      // (8 keys x 8 d) matrices, two k16 steps a load
      uint32_t bf[D / 16][2];
#pragma unroll
      for (int ks = 0; ks < D / 16; ks += 2) {
        const int row = kb + (lane & 7), chunk = 2 * ks + (lane >> 3);
        const uint32_t addr = kbuf + (chunk >> 3) * kChunkKeys * 128 + row * 128 + (((chunk & 7) ^ (row & 7)) << 4);
        asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
                     : "=r"(bf[ks][0]), "=r"(bf[ks][1]), "=r"(bf[ks + 1][0]), "=r"(bf[ks + 1][1])
                     : "r"(addr));
      }
      int seg[2];
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        const int key = kb0 + 2 * tq + e;
        seg[e] = key < nv ? 0 : (key < L ? 1 : 2);
      }
#pragma unroll
      for (int u = 0; u < kTiles; ++u) {
        float c[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int ks = 0; ks < D / 16; ++ks) mma_bf16(c, af[u][ks], bf[ks][0], bf[ks][1]);
        // scaled, masked scores; the block's maximum per row over the quad of
        // lanes that holds the row (all four then share the running maximum)
#pragma unroll
        for (int h2 = 0; h2 < 2; ++h2) {
          float y[2];
#pragma unroll
          for (int e = 0; e < 2; ++e) {
            const int key = kb0 + 2 * tq + e;
            y[e] = (key < k_hi && key <= lim[u][h2]) ? c[2 * h2 + e] * scale : -INFINITY;
          }
          float bm = fmaxf(y[0], y[1]);
#pragma unroll
          for (int o = 1; o < 4; o <<= 1) bm = fmaxf(bm, __shfl_xor_sync(0xffffffffu, bm, o));
          row_block(st[u][h2], y, seg, bm);
        }
      }
    }
    }
    // the four lanes of a row (fixed butterfly), then the warps in order
#pragma unroll
    for (int u = 0; u < kTiles; ++u)
#pragma unroll
      for (int h2 = 0; h2 < 2; ++h2) {
#pragma unroll
        for (int o = 1; o < 4; o <<= 1) row_merge(st[u][h2], row_shfl(st[u][h2], o));
        if (tq == 0) red[warp][16 * u + gq + 8 * h2] = st[u][h2];
      }
    __syncthreads();
    if (threadIdx.x < kPassRows) {
      RowState a = red[0][threadIdx.x];
      for (int w = 1; w < kWarps; ++w) row_merge(a, red[w][threadIdx.x]);
      part[threadIdx.x][0] = a.m;
      part[threadIdx.x][1] = a.v;
      part[threadIdx.x][2] = a.t;
      part[threadIdx.x][3] = a.g;
      part[threadIdx.x][4] = a.n;
    }
    cluster_sync_all();  // every CTA's part is written
    const int nr = min(kPassRows, M - m0);
    if (rank == 0) {
      // one lane a (row, CTA): the S partial states travel at once and merge
      // over the row's S lanes (S a power of two, so a row's lanes are an
      // aligned group of one warp) in a fixed butterfly
      for (int base0 = 0; base0 < kPassRows * S; base0 += kThreads) {  // block-uniform
        const int idx = base0 + threadIdx.x;
        const int r = idx / S, cc = idx % S;
        RowState a = row_empty();
        if (r < nr) {
          float v[8];
          ld_cluster8(&part[r][0], cc, v);
          a = RowState{v[0], v[1], v[2], v[3], v[4]};
        }
        for (int o = 1; o < S; o <<= 1) row_merge(a, row_shfl(a, o));
        if (cc == 0 && r < kPassRows) gath[r][0] = a;
      }
      __syncthreads();
    }
    if (rank == 0 && threadIdx.x < nr && ok) {
      const int p = m0 + threadIdx.x, i = p / G, h = kvh * G + (p - i * G);
      const RowState a = gath[threadIdx.x][0];
      const float tot = a.v + a.t + a.g;
      const long long o = (static_cast<long long>(b) * R + i) * Hq + h;
      mass[o * 3 + 0] = a.v / tot;
      mass[o * 3 + 1] = a.t / tot;
      mass[o * 3 + 2] = a.g / tot;
      const float lnv = a.t + a.g;
      const int n_rest = (L - nv) + i + 1;
      entropy[o] = (n_rest > 1 && lnv > 0.f) ? (logf(lnv) - a.n / lnv) / logf(static_cast<float>(n_rest)) : 0.f;
    }
    cluster_sync_all();  // rank 0 has read every part; red and part may be rewritten
  }
}

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult qres;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &qres) == cudaSuccess &&
        qres == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  });
  return fn;
}

// [B*Hkv][cap][D] bf16 keys as a 3-D tensor; boxes of 64 columns x 32 rows,
// 128-byte swizzle (the layout the kernel's ldmatrix reads)
bool make_key_map(CUtensorMap* map, void* base, int D, int cap, int planes) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[3] = {static_cast<cuuint64_t>(D), static_cast<cuuint64_t>(cap), static_cast<cuuint64_t>(planes)};
  cuuint64_t strides[2] = {static_cast<cuuint64_t>(D) * 2, static_cast<cuuint64_t>(cap) * static_cast<cuuint64_t>(D) * 2};
  cuuint32_t box[3] = {64, 32, 1};
  cuuint32_t estr[3] = {1, 1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, base, dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
            CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int D>
constexpr int smem_bytes() { return kChunkKeys * 128 * (D / 64) + 1024; }

}  // namespace

extern "C" sd_status sd_attention_budget(const void* q, const sd_kv_cache* cache, int R, int Hq, float scale,
                                         const int32_t* n_visual, float* mass, float* entropy,
                                         sd_stream_t stream) {
  if (!cache) return SD_ERR_INVALID_ARG;
  const int B = cache->batch, Hkv = cache->n_kv_heads, D = cache->head_dim, cap = cache->capacity;
  if (B < 0 || R <= 0 || Hq <= 0 || Hkv <= 0 || cap <= 0 || Hq % Hkv) return SD_ERR_INVALID_ARG;
  if (D != 64 && D != 128) return SD_ERR_UNSUPPORTED;
  if (B > 65535 || Hq > 65535) return SD_ERR_UNSUPPORTED;
  if (B == 0) return SD_OK;
  if (!q || !cache->k || !cache->len || !n_visual || !mass || !entropy) return SD_ERR_INVALID_ARG;
  if (!sd_aligned16(cache->k)) return SD_ERR_INVALID_ARG;
  if (!(scale >= 0.f) || !isfinite(scale)) return SD_ERR_INVALID_ARG;
  const float sc = scale > 0.f ? scale : static_cast<float>(1.0 / sqrt(static_cast<double>(D)));
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  // cluster size: the smallest power of two (up to 16) that leaves each CTA
  // at most 256 keys of the largest scene (32 keys a warp)
  int S = 1;
  while (S < 16 && static_cast<long long>(cap) > 256LL * S) S *= 2;
  const auto* qq = static_cast<const __nv_bfloat16*>(q);
  CUtensorMap tk;
  if (!make_key_map(&tk, cache->k, D, cap, B * Hkv)) return SD_ERR_CUDA;
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = S;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.gridDim = dim3(S, Hkv, B);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = D == 128 ? smem_bytes<128>() : smem_bytes<64>();
  cfg.stream = st;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  cudaError_t e;
  // clusters of 16 are non-portable and the staging buffer passes 48 KB:
  // both allowed once per device and kernel
  static bool allowed[64][2];
  int dev = 0;
  if (cudaGetDevice(&dev) == cudaSuccess && dev >= 0 && dev < 64 && !allowed[dev][D == 128]) {
    if (D == 128) {
      cudaFuncSetAttribute(budget_kernel<128>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
      cudaFuncSetAttribute(budget_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem_bytes<128>());
    } else {
      cudaFuncSetAttribute(budget_kernel<64>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
      cudaFuncSetAttribute(budget_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem_bytes<64>());
    }
    (void)cudaGetLastError();
    allowed[dev][D == 128] = true;
  }
  if (D == 128) {
    e = cudaLaunchKernelEx(&cfg, budget_kernel<128>, tk, qq, static_cast<const int32_t*>(cache->len), n_visual, R, Hq,
                           Hkv, cap, sc, mass, entropy);
  } else {
    e = cudaLaunchKernelEx(&cfg, budget_kernel<64>, tk, qq, static_cast<const int32_t*>(cache->len), n_visual, R, Hq,
                           Hkv, cap, sc, mass, entropy);
  }
  if (e != cudaSuccess) {
    (void)cudaGetLastError();
    return SD_ERR_CUDA;
  }
  SD_CHECK_LAUNCH();
  return SD_OK;
}
