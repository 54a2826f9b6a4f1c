// The fused verify layer: M-RoPE of the new query and key rows (Sec. 3.3,
// Sec. 4.2), the KV append (Eq. commit) and the verify attention (Eq. verify,
// Sec. 3.2) of one attention layer as one call.
//
// On the tcgen05 path (head_dim 128, G * R <= 128, R <= 31) it is one kernel launch that
// may overlap the previous layer: the cached prefix of a layer does not
// depend on the layer before it, so with SD_LAYER_PREFIX_EARLY the kernel is
// a programmatic dependent launch that starts streaming that prefix while the
// preceding kernel is still running, and waits only before it reads the new
// rows. Other shapes run the three kernels in sequence.
#include "common.cuh"

#include <math.h>

namespace {
// per-scene tickets [B], then per-(scene, KV head) tickets [B][Hkv] (the
// tcgen05 kernel's read-before-write-back count when a head spans several
// clusters)
constexpr size_t kTicketBytes(int B, int Hkv) {
  return (static_cast<size_t>(B) * (1 + static_cast<size_t>(Hkv)) * 4 + 255) / 256 * 256;
}
}  // namespace

extern "C" size_t sd_verify_layer_workspace(int B, int R, int Hq, int Hkv, int D, int capacity) {
  if (B <= 0) return 0;
  const size_t attn = sd_verify_attention_workspace(B, R, Hq, Hkv, D, capacity);
  return kTicketBytes(B, Hkv) + attn;
}

extern "C" sd_status sd_verify_layer(void* q, void* k_new, const void* v_new, const int32_t* pos,
                                     const int32_t sections[3], int interleaved, float base,
                                     const sd_kv_cache* cache, void* out, int R, int Hq,
                                     float scale, void* workspace, size_t ws_bytes, int flags,
                                     sd_stream_t stream) {
  if (!cache) return SD_ERR_INVALID_ARG;
  const int B = cache->batch, Hkv = cache->n_kv_heads, D = cache->head_dim, cap = cache->capacity;
  if (B < 0 || R <= 0 || Hq <= 0 || Hkv <= 0 || cap <= 0 || Hq % Hkv) return SD_ERR_INVALID_ARG;
  if (D != 64 && D != 128) return SD_ERR_UNSUPPORTED;
  if (interleaved != 0 && interleaved != 1) return SD_ERR_INVALID_ARG;
  if (flags & ~(SD_LAYER_PREFIX_EARLY | SD_LAYER_BLOCK_MASK)) return SD_ERR_INVALID_ARG;
  const int block = (flags & SD_LAYER_BLOCK_MASK) ? 1 : 0;
  if (B == 0) return SD_OK;
  if (!q || !k_new || !v_new || !pos || !sections || !out || !cache->k || !cache->v || !cache->len)
    return SD_ERR_INVALID_ARG;
  if (!sd_aligned16(q) || !sd_aligned16(k_new) || !sd_aligned16(v_new) || !sd_aligned16(out) ||
      !sd_aligned16(cache->k) || !sd_aligned16(cache->v))
    return SD_ERR_INVALID_ARG;
  if (!(scale >= 0.f) || !isfinite(scale) || !(base > 1.f) || !isfinite(base)) return SD_ERR_INVALID_ARG;
  const size_t need = sd_verify_layer_workspace(B, R, Hq, Hkv, D, cap);
  if (!workspace || ws_bytes < need || !sd_aligned16(workspace)) return SD_ERR_WORKSPACE;
  RopeTable tab;
  if (!sd_internal_rope_table(D, sections, interleaved, base, &tab)) return SD_ERR_INVALID_ARG;
  const float sc = scale > 0.f ? scale : static_cast<float>(1.0 / sqrt(static_cast<double>(D)));
  const float scale_log2 = static_cast<float>(static_cast<double>(sc) * 1.4426950408889634);
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  auto* ticket = static_cast<uint32_t*>(workspace);
  bool handled = false;
  const sd_status s = sd_internal_verify_layer_tc(q, k_new, v_new, pos, tab, cache, out, R, Hq,
                                                  scale_log2, ticket, flags & SD_LAYER_PREFIX_EARLY,
                                                  block, st, &handled);
  if (handled) return s;
  // other shapes: the same three steps as separate kernels
  sd_status r = sd_rope_apply(q, k_new, B, R, Hq, Hkv, D, pos, sections, interleaved, base, stream);
  if (r != SD_OK) return r;
  r = sd_kv_append(cache, k_new, v_new, R, stream);
  if (r != SD_OK) return r;
  return sd_verify_attention_ex(q, cache, out, R, Hq, scale, block ? SD_ATTN_BLOCK_MASK : 0,
                                static_cast<char*>(workspace) + kTicketBytes(B, Hkv),
                                ws_bytes - kTicketBytes(B, Hkv), stream);
}

extern "C" const char* sd_verify_kernel(int B, int R, int Hq, int Hkv, int D, int capacity, int layer) {
  if (B <= 0 || R <= 0 || Hq <= 0 || Hkv <= 0 || capacity <= 0 || Hq % Hkv || (D != 64 && D != 128) ||
      static_cast<long long>(Hq / Hkv) * R > 128)
    return "unsupported";
  if (layer) return sd_internal_tc_serves_layer(B, R, Hq, Hkv, D, capacity, layer > 1) ? "tcgen05" : "three kernels";
  return sd_internal_tc_serves(B, R, Hq, Hkv, D, capacity) ? "tcgen05" : "mma.sync";
}
