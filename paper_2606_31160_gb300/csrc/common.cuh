// Shared device and host helpers of libsd.so (sm_103a). Included by every
// translation unit; holds no part of the method's arithmetic.
#pragma once

#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <stdint.h>

#include "../../include/sd.h"

// ---------------------------------------------------------------------------
// Device error word. Each translation unit owns one (file-scope static), and
// exposes a host accessor that sd_get_device_error() calls. A kernel that
// meets a device-side problem ORs a bit in and skips the affected work; none
// traps.
// ---------------------------------------------------------------------------
static __device__ uint32_t sd_err_word;

__device__ __forceinline__ void sd_set_error(uint32_t bits) { atomicOr(&sd_err_word, bits); }

#define SD_DEFINE_ERROR_ACCESSOR(NAME)                                          \
  cudaError_t NAME(uint32_t* bits) {                                            \
    uint32_t v = 0, zero = 0;                                                   \
    cudaError_t e = cudaMemcpyFromSymbol(&v, sd_err_word, sizeof(v));           \
    if (e != cudaSuccess) return e;                                             \
    if (v) e = cudaMemcpyToSymbol(sd_err_word, &zero, sizeof(zero));            \
    *bits |= v;                                                                 \
    return e;                                                                   \
  }

// Host accessors, one per translation unit (defined with the macro above).
cudaError_t sd_take_error_rope(uint32_t* bits);
cudaError_t sd_take_error_kv(uint32_t* bits);
cudaError_t sd_take_error_attention(uint32_t* bits);
cudaError_t sd_take_error_attention_tc(uint32_t* bits);
cudaError_t sd_take_error_greedy(uint32_t* bits);
cudaError_t sd_take_error_sample(uint32_t* bits);

// Verify attention on the tcgen05 path (attention_tc.cu). Sets *handled when
// the shape is one it serves (head_dim 128, G * R <= 32) and it launched.
sd_status sd_internal_verify_attention_tc(const void* q, const sd_kv_cache* cache, void* out,
                                          int R, int Hq, float scale_log2, cudaStream_t stream,
                                          bool* handled);
// Whether the tcgen05 path serves this shape on the current device.
bool sd_internal_tc_serves(int B, int R, int Hq, int Hkv, int D, int cap);

// ---------------------------------------------------------------------------
// Host helpers
// ---------------------------------------------------------------------------
static inline bool sd_aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

static inline int sd_num_sms() {
  static int cached[64] = {0};
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev < 0 || dev >= 64) dev = 0;
  if (!cached[dev]) {
    int n = 0;
    cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    cached[dev] = n > 0 ? n : 1;
  }
  return cached[dev];
}

#define SD_CHECK_LAUNCH()                                   \
  do {                                                      \
    if (cudaPeekAtLastError() != cudaSuccess) {             \
      (void)cudaGetLastError();                             \
      return SD_ERR_CUDA;                                   \
    }                                                       \
  } while (0)

// ---------------------------------------------------------------------------
// Device helpers
// ---------------------------------------------------------------------------
__device__ __forceinline__ float sd_bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float sd_bf16_hi(uint32_t w) { return __uint_as_float(w & 0xffff0000u); }

// Two floats -> packed bf16x2 (round to nearest even), lo in the low half.
__device__ __forceinline__ uint32_t sd_pack_bf16x2(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}
