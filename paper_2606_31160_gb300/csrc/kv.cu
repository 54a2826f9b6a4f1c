// K2: KV-cache append and rollback (sm_103a).
//
// Eq. commit (Sec. 3.2): an iteration commits l + 1 tokens, t <- t + l + 1.
// The verify pass appends the keys/values of all R = K + 1 rows before the
// acceptance is known; afterwards the length moves back to keep only the
// n_emit = l + 1 committed rows. Nothing is erased: later appends overwrite.
//
// Append: one CTA per scene reads len[b] once, copies the R x Hkv rows with
// 16-byte vector stores, then advances len[b]; keeping the scene in one CTA
// makes the read-then-advance of len race-free without a grid-wide ticket.
// Rollback: one thread per length entry, no host synchronisation.
#include "common.cuh"

SD_DEFINE_ERROR_ACCESSOR(sd_take_error_kv)

namespace {

__global__ void __launch_bounds__(512) kv_append_kernel(uint4* __restrict__ kc, uint4* __restrict__ vc,
                                                        int32_t* __restrict__ len,
                                                        const uint4* __restrict__ kn,
                                                        const uint4* __restrict__ vn, int R, int hkv,
                                                        int cap, int vec_per_row) {
  sd_pdl_enter();
  const int b = blockIdx.x;
  __shared__ int s_len;
  if (threadIdx.x == 0) {
    const int l = len[b];
    const bool ok = l >= 0 && (long long)l + R <= cap;
    if (!ok) sd_set_error(SD_DEVERR_KV_OVERFLOW);
    s_len = ok ? l : -1;
  }
  __syncthreads();
  const int l0 = s_len;
  if (l0 < 0) return;
  const int per_scene = R * hkv * vec_per_row;
  for (int i = threadIdx.x; i < per_scene; i += blockDim.x) {
    const int vec = i % vec_per_row;
    const int t = i / vec_per_row;
    const int g = t % hkv;
    const int r = t / hkv;
    const long long src = ((long long)b * per_scene) + i;                 // [b][r][g][vec]
    const long long dst = (((long long)b * hkv + g) * cap + (l0 + r)) * vec_per_row + vec;
    kc[dst] = kn[src];
    vc[dst] = vn[src];
  }
  __syncthreads();
  if (threadIdx.x == 0) len[b] = l0 + R;
}

__global__ void kv_rollback_kernel(int32_t* __restrict__ len, int count, int B,
                                   const int32_t* __restrict__ committed, int n_appended) {
  sd_pdl_enter();
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= count) return;
  const int c = committed[i % B];
  const int l = len[i];
  const int nl = l - n_appended + c;
  if (c < 0 || c > n_appended || nl < 0) {
    sd_set_error(SD_DEVERR_ROLLBACK);
    return;
  }
  len[i] = nl;
}

}  // namespace

extern "C" sd_status sd_kv_append(const sd_kv_cache* cache, const void* k_new, const void* v_new,
                                  int R, sd_stream_t stream) {
  if (!cache) return SD_ERR_INVALID_ARG;
  const int B = cache->batch, hkv = cache->n_kv_heads, cap = cache->capacity, D = cache->head_dim;
  if (B < 0 || hkv <= 0 || cap <= 0 || R < 0) return SD_ERR_INVALID_ARG;
  if (D <= 0 || (D * 2) % 16) return SD_ERR_UNSUPPORTED;
  if (B == 0 || R == 0) return SD_OK;
  if (!cache->k || !cache->v || !cache->len || !k_new || !v_new) return SD_ERR_INVALID_ARG;
  if (!sd_aligned16(cache->k) || !sd_aligned16(cache->v) || !sd_aligned16(k_new) ||
      !sd_aligned16(v_new))
    return SD_ERR_INVALID_ARG;
  if (sd_launch_pdl(kv_append_kernel, dim3(B), dim3(512), 0, reinterpret_cast<cudaStream_t>(stream),
                    static_cast<uint4*>(cache->k), static_cast<uint4*>(cache->v), cache->len,
                    static_cast<const uint4*>(k_new), static_cast<const uint4*>(v_new), R, hkv, cap,
                    D / 8) != cudaSuccess) {
    (void)cudaGetLastError();
    return SD_ERR_CUDA;
  }
  return SD_OK;
}

extern "C" sd_status sd_kv_rollback(int32_t* len, int count, int B, const int32_t* committed,
                                    int n_appended, sd_stream_t stream) {
  if (count < 0 || B <= 0 || n_appended < 0) return SD_ERR_INVALID_ARG;
  if (count % B) return SD_ERR_INVALID_ARG;
  if (count == 0) return SD_OK;
  if (!len || !committed) return SD_ERR_INVALID_ARG;
  const int threads = 128;
  if (sd_launch_pdl(kv_rollback_kernel, dim3((count + threads - 1) / threads), dim3(threads), 0,
                    reinterpret_cast<cudaStream_t>(stream), len, count, B, committed,
                    n_appended) != cudaSuccess) {
    (void)cudaGetLastError();
    return SD_ERR_CUDA;
  }
  return SD_OK;
}
