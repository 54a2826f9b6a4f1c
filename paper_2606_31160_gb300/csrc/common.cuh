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
cudaError_t sd_take_error_budget(uint32_t* bits);

// Verify attention on the tcgen05 path (attention_tc.cu). Sets *handled when
// the shape is one it serves (head_dim 128, G * R <= 32) and it launched.
sd_status sd_internal_verify_attention_tc(const void* q, const sd_kv_cache* cache, void* out,
                                          int R, int Hq, float scale_log2, int flags, cudaStream_t stream,
                                          bool* handled);
// Whether the tcgen05 path serves this shape on the current device: the
// attention, and the fused layer without the block mask.
bool sd_internal_tc_serves(int B, int R, int Hq, int Hkv, int D, int cap);
bool sd_internal_tc_serves_layer(int B, int R, int Hq, int Hkv, int D, int cap, bool block);

struct RopeTable;
// The fused verify layer on the tcgen05 path (attention_tc.cu); *handled is
// set when the shape is served and the kernel launched.
sd_status sd_internal_verify_layer_tc(void* q, void* k_new, const void* v_new, const int32_t* pos,
                                      const RopeTable& tab, const sd_kv_cache* cache, void* out,
                                      int R, int Hq, float scale_log2, uint32_t* ticket, int early,
                                      int block, cudaStream_t stream, bool* handled);

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

// Programmatic dependent launch of a kernel that begins with sd_pdl_enter():
// it may become resident while the previous kernel on the stream finishes,
// but reaches no global memory before that kernel has completed.
template <typename... P, typename... A>
static inline cudaError_t sd_launch_pdl(void (*kernel)(P...), dim3 grid, dim3 block, size_t smem,
                                        cudaStream_t stream, A... args) {
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, args...);
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
// First statement of a kernel launched by sd_launch_pdl: wait until the
// previous kernel on the stream has completed (its writes visible), then let
// the next kernel launch. Waiting first keeps a successor's pre-wait phase
// from overlapping anything but this kernel.
__device__ __forceinline__ void sd_pdl_enter() {
  asm volatile("griddepcontrol.wait;" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

__device__ __forceinline__ float sd_bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float sd_bf16_hi(uint32_t w) { return __uint_as_float(w & 0xffff0000u); }

// ---------------------------------------------------------------------------
// RoPE (Sec. 3.3 Eq. rope-1d, Sec. 4.2 Eqs. axis-assign, mrope-phase) shared by
// the standalone rotation kernel and the fused verify-layer kernel, so both
// produce identical bits. The angle theta_d * p is carried in TURNS:
// tau_d = theta_d / (2 pi) as an fp32 hi/lo pair; p * tau_d is formed with an
// exact fma split, whole turns are dropped (an exact subtraction) and
// sincospif evaluates the remaining fraction, so the reduced angle is
// accurate to ~1e-7 rad for any |p| < 2^24.
// ---------------------------------------------------------------------------
constexpr int kRopeMaxPairs = 64;  // D <= 128

struct RopeTable {
  float tau_hi[kRopeMaxPairs];  // fp32 part of theta_d / (2 pi)
  float tau_lo[kRopeMaxPairs];  // remainder theta_d / (2 pi) - tau_hi
  int8_t axis[kRopeMaxPairs];   // a(d) in {0 = T, 1 = H, 2 = W}
};

// Fills the table for head dim D; sections == nullptr gives the 1-D table.
// Returns false for sections that do not sum to D / 2.
bool sd_internal_rope_table(int D, const int32_t* sections, int interleaved, float base,
                            RopeTable* tab);

// Fractional turns of p * tau, in [-0.5, 0.5] up to rounding.
__device__ __forceinline__ float sd_frac_turns(float p, float hi, float lo) {
  const float a = p * hi;          // rounded product
  const float e = fmaf(p, hi, -a); // its exact rounding error
  const float f = a - rintf(a);    // exact: whole turns removed
  return f + fmaf(p, lo, e);
}

// (cos, sin) of the rotation angle theta_d * p of pair d at coordinate p.
__device__ __forceinline__ float2 sd_rope_cs(float p, int d, const RopeTable& tab) {
  float s, c;
  sincospif(2.0f * sd_frac_turns(p, tab.tau_hi[d], tab.tau_lo[d]), &s, &c);
  return make_float2(c, s);
}

// Two floats -> packed bf16x2 (round to nearest even), lo in the low half.
__device__ __forceinline__ uint32_t sd_pack_bf16x2(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

// Rotate one pair (x, y) packed as bf16x2 by the angle with cosine c, sine s.
__device__ __forceinline__ uint32_t sd_rope_pair(uint32_t w, float c, float s) {
  const float x = sd_bf16_lo(w);
  const float y = sd_bf16_hi(w);
  return sd_pack_bf16x2(fmaf(x, c, -y * s), fmaf(x, s, y * c));
}

// Rotate 4 adjacent pairs (8 bf16 packed in w[4]) of head-vector chunk `vec`
// (pairs 4*vec .. 4*vec+3) at coordinates p3 (t, h, w).
__device__ __forceinline__ void sd_rope_rotate8(uint32_t (&w)[4], int vec, const int (&p3)[3],
                                                const RopeTable& tab) {
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    const int d = vec * 4 + j;
    const float2 cs = sd_rope_cs(static_cast<float>(p3[tab.axis[d]]), d, tab);
    w[j] = sd_rope_pair(w[j], cs.x, cs.y);
  }
}
