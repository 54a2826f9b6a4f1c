// K1: rotary position encoding of the new verify rows (sm_103a).
//
// Sec. 3.3 Eq. rope-1d: each adjacent pair (2d, 2d+1) of a head vector
// rotates by phi_d; Sec. 3.3 Eq. rope-3d with Sec. 4.2 Eqs. axis-assign and
// mrope-phase: phi_d = theta_d * p_{a(d)}, theta_d = base^(-2d/D), a(d)
// blocked over (s_T, s_H, s_W) or (T,H,W)[d mod 3]; Sec. 4.2 Eq.
// flatrope-proj: FlatRoPE puts every axis at the sequence index.
//
// Layout: one thread rotates 4 pairs (8 bf16 = one 16-byte load/store) of
// one head row; the whole launch is a few thousand threads and is bound by
// launch latency, not bandwidth.
//
// Angle precision: theta_d * p reaches ~1.6e4 rad at the positions of the
// longest workloads, where an fp32 product alone is off by ~1e-3 rad; the
// turn-based reduction in common.cuh keeps it at ~1e-7 rad.
#include "common.cuh"

#include <math.h>

SD_DEFINE_ERROR_ACCESSOR(sd_take_error_rope)

namespace {

// One thread: 8 consecutive elements (4 pairs) of one head row.
template <int D, bool kFlat>
__global__ void __launch_bounds__(256) rope_kernel(__nv_bfloat16* __restrict__ q,
                                                   __nv_bfloat16* __restrict__ k,
                                                   int rows, int hq, int hkv,
                                                   const int32_t* __restrict__ pos,
                                                   RopeTable tab) {
  sd_pdl_enter();
  constexpr int kVecPerHead = D / 8;
  const int heads = hq + hkv;
  const long long total = (long long)rows * heads * kVecPerHead;
  for (long long idx = blockIdx.x * (long long)blockDim.x + threadIdx.x; idx < total;
       idx += (long long)gridDim.x * blockDim.x) {
    const int vec = (int)(idx % kVecPerHead);
    const long long t = idx / kVecPerHead;
    const int head = (int)(t % heads);
    const long long row = t / heads;  // flattened (b, r)
    __nv_bfloat16* base = head < hq ? q + ((row * hq + head) * D)
                                    : k + ((row * hkv + (head - hq)) * D);
    uint4* ptr = reinterpret_cast<uint4*>(base) + vec;
    const uint4 v = *ptr;
    uint32_t words[4] = {v.x, v.y, v.z, v.w};
    int p3[3];
    if (kFlat) {
      p3[0] = p3[1] = p3[2] = pos[row];
    } else {
      p3[0] = pos[row * 3 + 0];
      p3[1] = pos[row * 3 + 1];
      p3[2] = pos[row * 3 + 2];
    }
    sd_rope_rotate8(words, vec, p3, tab);
    *ptr = make_uint4(words[0], words[1], words[2], words[3]);
  }
}

sd_status launch(void* q, void* k, int B, int R, int Hq, int Hkv, int D, const int32_t* pos,
                 const int32_t* sections, int interleaved, float base, bool flat,
                 cudaStream_t stream) {
  if (B < 0 || R < 0 || Hq < 0 || Hkv < 0) return SD_ERR_INVALID_ARG;
  if (D != 64 && D != 128) return SD_ERR_UNSUPPORTED;
  if (!(base > 1.0f) || !isfinite(base)) return SD_ERR_INVALID_ARG;
  if ((Hq > 0 && (!q || !sd_aligned16(q))) || (Hkv > 0 && (!k || !sd_aligned16(k))))
    return SD_ERR_INVALID_ARG;
  const long long rows = (long long)B * R;
  if (rows == 0 || Hq + Hkv == 0) return SD_OK;
  if (!pos) return SD_ERR_INVALID_ARG;
  if (!flat && !sections) return SD_ERR_INVALID_ARG;
  RopeTable tab;
  if (!sd_internal_rope_table(D, flat ? nullptr : sections, interleaved, base, &tab))
    return SD_ERR_INVALID_ARG;
  const long long total = rows * (Hq + Hkv) * (D / 8);
  const int threads = 256;
  long long blocks = (total + threads - 1) / threads;
  const long long cap = (long long)sd_num_sms() * 8;
  if (blocks > cap) blocks = cap;
  auto* qp = static_cast<__nv_bfloat16*>(q);
  auto* kp = static_cast<__nv_bfloat16*>(k);
  auto* kern = D == 64 ? (flat ? rope_kernel<64, true> : rope_kernel<64, false>)
                       : (flat ? rope_kernel<128, true> : rope_kernel<128, false>);
  if (sd_launch_pdl(kern, dim3((unsigned)blocks), dim3(threads), 0, stream, qp, kp, (int)rows, Hq, Hkv,
                    pos, tab) != cudaSuccess) {
    (void)cudaGetLastError();
    return SD_ERR_CUDA;
  }
  return SD_OK;
}

}  // namespace

bool sd_internal_rope_table(int D, const int32_t* sections, int interleaved, float base,
                            RopeTable* tab) {
  const int pairs = D / 2;
  if (pairs > kRopeMaxPairs) return false;
  if (sections) {
    if (sections[0] < 0 || sections[1] < 0 || sections[2] < 0) return false;
    if (sections[0] + sections[1] + sections[2] != pairs) return false;
  }
  const double two_pi = 6.283185307179586476925286766559;
  for (int d = 0; d < pairs; ++d) {
    const double theta = pow((double)base, -2.0 * d / (double)D);
    const double tau = theta / two_pi;
    tab->tau_hi[d] = (float)tau;
    tab->tau_lo[d] = (float)(tau - (double)tab->tau_hi[d]);
    int a = 0;
    if (sections) {
      if (interleaved) a = d % 3;
      else if (d < sections[0]) a = 0;
      else if (d < sections[0] + sections[1]) a = 1;
      else a = 2;
    }
    tab->axis[d] = (int8_t)a;
  }
  for (int d = pairs; d < kRopeMaxPairs; ++d) {
    tab->tau_hi[d] = tab->tau_lo[d] = 0.f;
    tab->axis[d] = 0;
  }
  return true;
}

extern "C" sd_status sd_rope_apply(void* q, void* k, int B, int R, int Hq, int Hkv, int D,
                                   const int32_t* pos, const int32_t sections[3],
                                   int interleaved, float base, sd_stream_t stream) {
  if (interleaved != 0 && interleaved != 1) return SD_ERR_INVALID_ARG;
  return launch(q, k, B, R, Hq, Hkv, D, pos, sections, interleaved, base, false,
                reinterpret_cast<cudaStream_t>(stream));
}

extern "C" sd_status sd_rope_apply_1d(void* q, void* k, int B, int R, int Hq, int Hkv, int D,
                                      const int32_t* pos1d, float base, sd_stream_t stream) {
  return launch(q, k, B, R, Hq, Hkv, D, pos1d, nullptr, 0, base, true,
                reinterpret_cast<cudaStream_t>(stream));
}
