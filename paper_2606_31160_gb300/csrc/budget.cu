// Attention budget of the verify rows (Sec. 4.2 "Empirical confirmation",
// Table tab:attn-budget): for every (scene, row, query head), the share of
// the row's softmax mass on the visual keys, on the trajectory / prompt-text
// keys and on the rows generated in this step, and the entropy of the
// attention among the non-visual keys (renormalised), divided by the log of
// their number.
//
// A diagnostic beside the verify path, exact rather than fast: one CTA per
// (query head, scene) takes the rows in groups of 8; for each group it makes
// two passes over the visible keys on the CUDA cores (fp32 dot products of the
// bf16 rows): the row maxima, then the weights exp(s - max) summed per segment
// together with the entropy term sum w (s - max). Block reductions run in a
// fixed order.
//
//   entropy = (ln l' - T' / l') / ln N'     l' = sum of the non-visual weights,
//                                           T' = sum over them of w (s - max),
//                                           N' = number of non-visual keys
#include "common.cuh"

#include <math.h>

SD_DEFINE_ERROR_ACCESSOR(sd_take_error_budget)

namespace {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr int kGroup = 8;  // rows per group
constexpr float kLog2e = 1.4426950408889634f;

// scores of key row kr (D bf16, 16-byte aligned) against the group's rows
template <int D>
__device__ __forceinline__ void key_scores(const __nv_bfloat16* kr, const float (*qs)[D], float (&acc)[kGroup]) {
#pragma unroll
  for (int r = 0; r < kGroup; ++r) acc[r] = 0.f;
#pragma unroll 4
  for (int c = 0; c < D / 8; ++c) {
    const uint4 w = __ldg(reinterpret_cast<const uint4*>(kr) + c);
    const uint32_t ws[4] = {w.x, w.y, w.z, w.w};
    float kf[8];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      kf[2 * j] = sd_bf16_lo(ws[j]);
      kf[2 * j + 1] = sd_bf16_hi(ws[j]);
    }
#pragma unroll
    for (int r = 0; r < kGroup; ++r)
#pragma unroll
      for (int e = 0; e < 8; ++e) acc[r] = fmaf(qs[r][c * 8 + e], kf[e], acc[r]);
  }
}

// block-wide reduction of v[r] (max or sum), fixed order; result in out[r]
template <bool kMax>
__device__ __forceinline__ void block_reduce(float (&v)[kGroup], float (*red)[kGroup], float* out) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
#pragma unroll
  for (int r = 0; r < kGroup; ++r)
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const float x = __shfl_xor_sync(0xffffffffu, v[r], o);
      v[r] = kMax ? fmaxf(v[r], x) : v[r] + x;
    }
  if (lane == 0)
#pragma unroll
    for (int r = 0; r < kGroup; ++r) red[warp][r] = v[r];
  __syncthreads();
  if (threadIdx.x < kGroup) {
    float a = red[0][threadIdx.x];
    for (int w = 1; w < kWarps; ++w) a = kMax ? fmaxf(a, red[w][threadIdx.x]) : a + red[w][threadIdx.x];
    out[threadIdx.x] = a;
  }
  __syncthreads();
}

template <int D>
__global__ void __launch_bounds__(kThreads)
    budget_kernel(const __nv_bfloat16* __restrict__ q, const __nv_bfloat16* __restrict__ kc,
                  const int32_t* __restrict__ len, const int32_t* __restrict__ n_visual, int R, int Hq,
                  int Hkv, int cap, float scale, float* __restrict__ mass, float* __restrict__ entropy) {
  __shared__ float qs[kGroup][D];
  __shared__ float red[kWarps][kGroup];
  __shared__ float s_max[kGroup], s_lv[kGroup], s_lt[kGroup], s_lg[kGroup], s_tn[kGroup];
  const int h = blockIdx.x, b = blockIdx.y;
  const int g = h / (Hq / Hkv);
  const int n_keys = len[b], L = n_keys - R;
  int nv = n_visual[b];
  if (L < 0 || n_keys > cap) {
    if (threadIdx.x == 0 && h == 0) sd_set_error(SD_DEVERR_LENGTH);
    return;
  }
  if (nv < 0 || nv > L) {
    if (threadIdx.x == 0 && h == 0) sd_set_error(SD_DEVERR_LENGTH);
    nv = nv < 0 ? 0 : L;
  }
  const __nv_bfloat16* kb = kc + (static_cast<long long>(b) * Hkv + g) * cap * D;
  for (int r0 = 0; r0 < R; r0 += kGroup) {
    const int nr = min(kGroup, R - r0);
    for (int idx = threadIdx.x; idx < kGroup * D; idx += kThreads) {
      const int r = idx / D, d = idx % D;
      qs[r][d] = r < nr ? __bfloat162float(q[((static_cast<long long>(b) * R + r0 + r) * Hq + h) * D + d]) : 0.f;
    }
    __syncthreads();
    const int last = L + r0 + nr;  // keys visible to the group's last row
    // pass 1: row maxima of the scaled scores
    float v[kGroup];
#pragma unroll
    for (int r = 0; r < kGroup; ++r) v[r] = -INFINITY;
    for (int k = threadIdx.x; k < last; k += kThreads) {
      float acc[kGroup];
      key_scores<D>(kb + static_cast<long long>(k) * D, qs, acc);
#pragma unroll
      for (int r = 0; r < kGroup; ++r)
        if (r < nr && k <= L + r0 + r) v[r] = fmaxf(v[r], acc[r] * scale);
    }
    block_reduce<true>(v, red, s_max);
    // pass 2: weights per segment and the non-visual entropy term
    float lv[kGroup], lt[kGroup], lg[kGroup], tn[kGroup];
#pragma unroll
    for (int r = 0; r < kGroup; ++r) lv[r] = lt[r] = lg[r] = tn[r] = 0.f;
    for (int k = threadIdx.x; k < last; k += kThreads) {
      float acc[kGroup];
      key_scores<D>(kb + static_cast<long long>(k) * D, qs, acc);
#pragma unroll
      for (int r = 0; r < kGroup; ++r) {
        if (r < nr && k <= L + r0 + r) {
          const float y = acc[r] * scale - s_max[r];
          const float w = exp2f(y * kLog2e);
          if (k < nv) {
            lv[r] += w;
          } else {
            if (k < L) lt[r] += w;
            else lg[r] += w;
            tn[r] = fmaf(w, y, tn[r]);
          }
        }
      }
    }
    block_reduce<false>(lv, red, s_lv);
    block_reduce<false>(lt, red, s_lt);
    block_reduce<false>(lg, red, s_lg);
    block_reduce<false>(tn, red, s_tn);
    if (threadIdx.x < nr) {
      const int r = threadIdx.x, i = r0 + r;
      const float tot = s_lv[r] + s_lt[r] + s_lg[r];
      const long long o = (static_cast<long long>(b) * R + i) * Hq + h;
      mass[o * 3 + 0] = s_lv[r] / tot;
      mass[o * 3 + 1] = s_lt[r] / tot;
      mass[o * 3 + 2] = s_lg[r] / tot;
      const float lnv = s_lt[r] + s_lg[r];
      const int n_rest = (L - nv) + i + 1;
      entropy[o] = (n_rest > 1 && lnv > 0.f) ? (logf(lnv) - s_tn[r] / lnv) / logf(static_cast<float>(n_rest)) : 0.f;
    }
    __syncthreads();  // qs is rewritten by the next group
  }
}

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
  const dim3 grid(Hq, B);
  const auto* qq = static_cast<const __nv_bfloat16*>(q);
  const auto* kk = static_cast<const __nv_bfloat16*>(cache->k);
  if (D == 128)
    budget_kernel<128><<<grid, kThreads, 0, st>>>(qq, kk, cache->len, n_visual, R, Hq, Hkv, cap, sc, mass, entropy);
  else
    budget_kernel<64><<<grid, kThreads, 0, st>>>(qq, kk, cache->len, n_visual, R, Hq, Hkv, cap, sc, mass, entropy);
  SD_CHECK_LAUNCH();
  return SD_OK;
}
