// K5: rejection-sampling acceptance (Leviathan et al. / Chen et al., cited
// in Sec. 1-2 of the paper, which evaluates the greedy rule only).
//
//   p_j = softmax(z_T[j] / T), q_j = softmax(z_D[j] / T)
//   draft j (token x) accepted iff u_j * q_j(x) <= p_j(x)
//   first rejection at j: draw from (p_j - q_j)+ with u_K
//   all K accepted:       draw the bonus from p_K with u_K
//   draw from w with u:   smallest v with sum_{v' <= v} w(v') > u * sum(w)
//
// Two launches:
//   stats:  grid (chunk, row, scene) over the 2K + 1 rows; each CTA writes
//           (max, sum exp2((z - max) * log2e / T)) of one chunk of 16384
//           (rows of 16-byte multiples: 32 values per thread from eight
//           16-byte loads, kept in registers for both) or 4096 elements, and
//           the CTA whose chunk holds a draft token records its logit. The
//           last CTA of a scene (atomic ticket, no spin) merges the chunks of
//           every row in a fixed order, runs the K acceptance tests and
//           records l and the normalisers of the row to draw from.
//   draw:   grid (chunk of 4096 values, scene) over that one row, a thread
//           owning 16 consecutive values of both logit rows (16-byte loads
//           when the rows are aligned); each CTA writes the chunk sums of the
//           residual weights and of the target weights; the last CTA of a
//           scene finds the chunk where the running sum passes u_K * S and
//           re-scans the same per-thread runs inside it. A programmatic
//           dependent launch: its CTAs are resident once every statistics CTA
//           runs, and wait for the statistics to complete before they read.
// All reductions run in a fixed order (deterministic), the weight formula
// uses non-contractible intrinsics so both passes of the draw evaluate
// identical values, and every spin-free ticket is re-armed after use.
#include "common.cuh"

#include <mutex>

SD_DEFINE_ERROR_ACCESSOR(sd_take_error_sample)

namespace {

constexpr int kThreads = 256;
constexpr int kMaxChunks = 1024;
constexpr float kLog2e = 1.4426950408889634f;

struct DrawInfo {
  int ell;
  float mt, inv_zt;  // target row l (or K): max and 1 / sum
  float md, inv_zd;  // draft row l (when l < K)
  float pad[3];
};

// exp2((z - m) * c2) with a fixed rounding sequence
__device__ __forceinline__ float wexp(float z, float m, float c2) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(__fmul_rn(__fsub_rn(z, m), c2)));
  return y;
}

// (max, sum) pair merge: sum rescaled to the larger max
__device__ __forceinline__ void merge_ms(float& m, float& s, float m2, float s2, float c2) {
  if (m2 == -INFINITY) return;
  if (m == -INFINITY) {
    m = m2;
    s = s2;
    return;
  }
  if (m2 > m) {
    s = __fadd_rn(__fmul_rn(s, wexp(m, m2, c2)), s2);
    m = m2;
  } else {
    s = __fadd_rn(s, __fmul_rn(s2, wexp(m2, m, c2)));
  }
}

__device__ __forceinline__ const float* row_ptr(const float* zt, const float* zd, int b, int rr,
                                                int K, int V) {
  if (rr <= K) return zt + (static_cast<long long>(b) * (K + 1) + rr) * V;
  return zd + (static_cast<long long>(b) * K + (rr - K - 1)) * V;
}

// The last CTA of scene b (all of its chunk partials are in): merge the
// chunks of every row in a fixed order, run the K acceptance tests, record l
// and the normalisers of the row to draw from, write n_emit and the accepted
// tokens, re-arm the ticket. Called by all nthreads threads of that CTA.
__device__ __noinline__ void accept_tail(const float* __restrict__ zt, const float* __restrict__ zd, int K,
                                         int V, float c2, int n_chunks, int b, const int* s_x,
                                         const float* __restrict__ u, int32_t* __restrict__ n_emit,
                                         int32_t* __restrict__ tokens, const float2* __restrict__ part,
                                         const float* __restrict__ dlogit, uint32_t* __restrict__ ticket,
                                         DrawInfo* __restrict__ info, int nthreads) {
  const int rows = 2 * K + 1;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int kT = nthreads;
  __shared__ float row_m[2 * 128 + 1], row_s[2 * 128 + 1];
  // every load of the tail is issued before any result is used (one memory
  // round trip): the K draft tokens' two logits, recorded by the CTAs holding
  // them, the scene's K acceptance uniforms, and the rows' chunk partials,
  // two rows a warp at a time
  __shared__ float s_zt[128], s_zd[128], s_u[128];
  for (int j = threadIdx.x; j < K; j += kT) {
    const int x = s_x[j];
    const bool ok = x >= 0 && x < V;
    s_zt[j] = ok ? __ldcg(dlogit + static_cast<long long>(b) * rows + j) : 0.f;
    s_zd[j] = ok ? __ldcg(dlogit + static_cast<long long>(b) * rows + K + 1 + j) : 0.f;
    s_u[j] = u[static_cast<long long>(b) * (K + 1) + j];
  }
  const int nw = kT / 32;
  for (int r0 = warp; r0 < rows; r0 += 2 * nw) {
    const int r1 = r0 + nw;
    float rm[2] = {-INFINITY, -INFINITY}, rs[2] = {0.f, 0.f};
    const float2* p0 = part + (static_cast<long long>(b) * rows + r0) * n_chunks;
    const float2* p1 = part + (static_cast<long long>(b) * rows + (r1 < rows ? r1 : r0)) * n_chunks;
    for (int k = lane; k < n_chunks; k += 32) {
      const float2 e0 = __ldcg(p0 + k);
      const float2 e1 = __ldcg(p1 + k);
      merge_ms(rm[0], rs[0], e0.x, e0.y, c2);
      merge_ms(rm[1], rs[1], e1.x, e1.y, c2);
    }
#pragma unroll
    for (int h = 0; h < 2; ++h) {
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        const float m2 = __shfl_xor_sync(0xffffffffu, rm[h], o);
        const float s2 = __shfl_xor_sync(0xffffffffu, rs[h], o);
        merge_ms(rm[h], rs[h], m2, s2, c2);
      }
    }
    if (lane == 0) {
      row_m[r0] = rm[0];
      row_s[r0] = rs[0];
      if (r1 < rows) {
        row_m[r1] = rm[1];
        row_s[r1] = rs[1];
      }
    }
  }
  __syncthreads();
  if (warp == 0) {
    // the K acceptance tests side by side (lane j of a 32-draft group), the
    // first stop by ballot: l = the first j whose token is out of range or
    // whose test fails, as a sequential scan would find it
    int ell = K;
    bool range_bad = false;
    for (int j0 = 0; j0 < K; j0 += 32) {  // warp-uniform
      const int j = j0 + lane;
      bool stop = false, bad = false;
      if (j < K) {
        const int x = s_x[j];
        bad = x < 0 || x >= V;
        if (bad) {
          stop = true;
        } else {
          const float p = __fdiv_rn(wexp(s_zt[j], row_m[j], c2), row_s[j]);
          const float q = __fdiv_rn(wexp(s_zd[j], row_m[K + 1 + j], c2), row_s[K + 1 + j]);
          stop = !(__fmul_rn(s_u[j], q) <= p);
        }
      }
      const unsigned hit = __ballot_sync(0xffffffffu, stop);
      if (hit) {
        const int first = __ffs(hit) - 1;
        ell = j0 + first;
        range_bad = __shfl_sync(0xffffffffu, bad, first);
        break;
      }
    }
    if (lane == 0) {
      if (range_bad) sd_set_error(SD_DEVERR_TOKEN_RANGE);
      DrawInfo di;
      di.ell = ell;
      di.mt = row_m[ell];
      di.inv_zt = __fdiv_rn(1.f, row_s[ell]);
      di.md = ell < K ? row_m[K + 1 + ell] : 0.f;
      di.inv_zd = ell < K ? __fdiv_rn(1.f, row_s[K + 1 + ell]) : 0.f;
      di.pad[0] = di.pad[1] = di.pad[2] = 0.f;
      info[b] = di;
      n_emit[b] = ell + 1;
      ticket[b] = 0;
    }
    int32_t* tk = tokens + static_cast<long long>(b) * (K + 1);
    for (int j = lane; j <= K; j += 32) tk[j] = j < ell ? s_x[j] : -1;
  }
}

// ------------------------------------------------------------------ stats
constexpr int kVecThreads = 512;       // threads of the vectorised stats kernel
constexpr int kVecPer = 32;            // values per thread (eight 16-byte loads)
constexpr int kVecChunk = kVecThreads * kVecPer;

template <bool kVec>
__global__ void __launch_bounds__(kVec ? kVecThreads : kThreads)
    sample_stats_kernel(const float* __restrict__ zt, const float* __restrict__ zd, int K, int V,
                        float c2, int chunk, int n_chunks, const int32_t* __restrict__ draft,
                        const float* __restrict__ u, int32_t* __restrict__ n_emit,
                        int32_t* __restrict__ tokens, float2* __restrict__ part,
                        float* __restrict__ dlogit, uint32_t* __restrict__ ticket,
                        DrawInfo* __restrict__ info) {
  constexpr int kT = kVec ? kVecThreads : kThreads;
  const int c = blockIdx.x, rr = blockIdx.y, b = blockIdx.z;
  if (threadIdx.x == 0) asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  const int rows = 2 * K + 1;
  const float* row = row_ptr(zt, zd, b, rr, K, V);
  const int lo = c * chunk, hi = min(V, lo + chunk);
  // the drafts, read early (only the scene's last CTA needs them all); the
  // CTA whose chunk holds the draft token of its row records that logit
  __shared__ int s_x[128];
  for (int j = threadIdx.x; j < K; j += kT) s_x[j] = __ldg(draft + static_cast<long long>(b) * K + j);
  if (threadIdx.x == 0 && rr != K) {
    const int j = rr < K ? rr : rr - K - 1;
    const int x = __ldg(draft + static_cast<long long>(b) * K + j);
    if (x >= lo && x < hi) dlogit[static_cast<long long>(b) * rows + rr] = __ldg(row + x);
  }
  float m = -INFINITY, s = 0.f;
  if (kVec) {
    // values lo + 4 (t + kT k) + e, k < 8, e < 4: one fixed order for both passes
    float x[kVecPer];
#pragma unroll
    for (int k = 0; k < kVecPer / 4; ++k) {
      const int i = lo + 4 * (threadIdx.x + kT * k);
      const float4 v = i < hi ? __ldg(reinterpret_cast<const float4*>(row + i))
                              : make_float4(-INFINITY, -INFINITY, -INFINITY, -INFINITY);
      x[4 * k + 0] = v.x;
      x[4 * k + 1] = v.y;
      x[4 * k + 2] = v.z;
      x[4 * k + 3] = v.w;
    }
#pragma unroll
    for (int e = 0; e < kVecPer; ++e) m = fmaxf(m, x[e]);
    if (m != -INFINITY)
#pragma unroll
      for (int e = 0; e < kVecPer; ++e) s = __fadd_rn(s, x[e] == -INFINITY ? 0.f : wexp(x[e], m, c2));
  } else {
    // thread max, then thread sum, over a fixed strided subset of the chunk
    for (int i = lo + threadIdx.x; i < hi; i += kT) m = fmaxf(m, __ldg(row + i));
    if (m != -INFINITY)
      for (int i = lo + threadIdx.x; i < hi; i += kT) s = __fadd_rn(s, wexp(__ldg(row + i), m, c2));
  }
  // warp then block merge, fixed tree
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float m2 = __shfl_xor_sync(0xffffffffu, m, o);
    const float s2 = __shfl_xor_sync(0xffffffffu, s, o);
    merge_ms(m, s, m2, s2, c2);
  }
  __shared__ float sm[kT / 32], ss[kT / 32];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (lane == 0) {
    sm[warp] = m;
    ss[warp] = s;
  }
  __syncthreads();
  __shared__ bool s_last;
  if (threadIdx.x == 0) {
    float bm = sm[0], bs = ss[0];
    for (int w = 1; w < kT / 32; ++w) merge_ms(bm, bs, sm[w], ss[w], c2);
    part[(static_cast<long long>(b) * rows + rr) * n_chunks + c] = make_float2(bm, bs);
    __threadfence();
    s_last = atomicAdd(&ticket[b], 1u) == static_cast<uint32_t>(rows * n_chunks - 1);
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  accept_tail(zt, zd, K, V, c2, n_chunks, b, s_x, u, n_emit, tokens, part, dlogit, ticket, info, kT);
}

// Streaming stats: one CTA per (segment, row, scene) moves its segment of the
// row through a ring of kStages 16 KB shared-memory stages with bulk copies
// (warp 8 produces, warps 0-7 consume); a consumer thread keeps an online
// (max, sum) over its 16 values of every stage in a fixed order. Rows must
// start on 16-byte boundaries (V % 4 == 0, aligned bases).
constexpr int kStreamConsumers = 256;
constexpr int kStreamThreads = kStreamConsumers + 32;
constexpr int kStageFloats = 4096;
constexpr int kStreamStages = 4;
constexpr uint32_t kStreamSpin = 1u << 22;

__device__ __forceinline__ bool st_try_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\tmbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}
// bounded wait; false after the limit (the caller records a timeout)
__device__ __forceinline__ bool st_wait(uint32_t bar, uint32_t parity) {
#pragma unroll 1
  for (uint32_t i = 0; i < kStreamSpin; ++i)
    if (st_try_wait(bar, parity)) return true;
  return false;
}

__global__ void __launch_bounds__(kStreamThreads)
    sample_stats_stream_kernel(const float* __restrict__ zt, const float* __restrict__ zd, int K, int V,
                               float c2, int seg, int n_seg, const int32_t* __restrict__ draft,
                               const float* __restrict__ u, int32_t* __restrict__ n_emit,
                               int32_t* __restrict__ tokens, float2* __restrict__ part,
                               float* __restrict__ dlogit, uint32_t* __restrict__ ticket,
                               DrawInfo* __restrict__ info) {
  extern __shared__ __align__(128) float stage_raw[];  // [kStreamStages][kStageFloats]
  float (*stage)[kStageFloats] = reinterpret_cast<float (*)[kStageFloats]>(stage_raw);
  __shared__ __align__(8) uint64_t full[kStreamStages], empty[kStreamStages];
  __shared__ int s_x[128];
  __shared__ int s_timeout;
  const int c = blockIdx.x, rr = blockIdx.y, b = blockIdx.z;
  const int rows = 2 * K + 1;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const float* row = row_ptr(zt, zd, b, rr, K, V);
  const int lo = c * seg, hi = min(V, lo + seg);
  if (threadIdx.x == 0) asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  const int n_st = hi > lo ? (hi - lo + kStageFloats - 1) / kStageFloats : 0;
  if (threadIdx.x == 0) {
    for (int i = 0; i < kStreamStages; ++i) {
      asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(static_cast<uint32_t>(__cvta_generic_to_shared(&full[i]))));
      asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(static_cast<uint32_t>(__cvta_generic_to_shared(&empty[i]))),
                   "r"(kStreamConsumers / 32));
    }
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    s_timeout = 0;
  }
  __syncthreads();
  // the drafts (for the scene's last CTA; read after the barriers below), by
  // the consumers: the producer's first copies do not wait for them
  if (warp < kStreamConsumers / 32)
    for (int j = threadIdx.x; j < K; j += kStreamConsumers) s_x[j] = __ldg(draft + static_cast<long long>(b) * K + j);
  float m = -INFINITY, s = 0.f;
  if (warp == kStreamConsumers / 32) {
    // ---- producer: thread 0 of warp 8; the first copies go out before it
    //      records the draft token's logit (a load it then waits for)
    if (lane == 0) {
      for (int t = 0; t < n_st; ++t) {
        const int st = t % kStreamStages;
        if (t >= kStreamStages &&
            !st_wait(static_cast<uint32_t>(__cvta_generic_to_shared(&empty[st])),
                     static_cast<uint32_t>(((t / kStreamStages) - 1) & 1))) {
          s_timeout = 1;
          break;
        }
        const int p0 = lo + t * kStageFloats;
        const uint32_t bytes = static_cast<uint32_t>(min(kStageFloats, hi - p0) * 4);
        const uint32_t fb = static_cast<uint32_t>(__cvta_generic_to_shared(&full[st]));
        asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(fb), "r"(bytes) : "memory");
        asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                         static_cast<uint32_t>(__cvta_generic_to_shared(&stage[st][0]))),
                     "l"(row + p0), "r"(bytes), "r"(fb)
                     : "memory");
      }
      if (rr != K) {
        const int j = rr < K ? rr : rr - K - 1;
        const int x = __ldg(draft + static_cast<long long>(b) * K + j);
        if (x >= lo && x < hi) dlogit[static_cast<long long>(b) * rows + rr] = __ldg(row + x);
      }
    }
  } else {
    // ---- consumers: thread t takes float4 t + 256 k (k < 4) of every stage
    for (int t = 0; t < n_st; ++t) {
      const int st = t % kStreamStages;
      if (!st_wait(static_cast<uint32_t>(__cvta_generic_to_shared(&full[st])),
                   static_cast<uint32_t>((t / kStreamStages) & 1))) {
        s_timeout = 1;
        break;
      }
      const int p0 = lo + t * kStageFloats;
      const int nv = min(kStageFloats, hi - p0) / 4;  // float4s in this stage
      float x[16];
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const int v = threadIdx.x + kStreamConsumers * k;
        const float4 f = v < nv ? reinterpret_cast<const float4*>(stage[st])[v]
                                : make_float4(-INFINITY, -INFINITY, -INFINITY, -INFINITY);
        x[4 * k + 0] = f.x;
        x[4 * k + 1] = f.y;
        x[4 * k + 2] = f.z;
        x[4 * k + 3] = f.w;
      }
      __syncwarp();
      if (lane == 0)
        asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(static_cast<uint32_t>(__cvta_generic_to_shared(&empty[st])))
                     : "memory");
      float mx = x[0];
#pragma unroll
      for (int e = 1; e < 16; ++e) mx = fmaxf(mx, x[e]);
      if (mx != -INFINITY) {
        if (mx > m) {
          if (m != -INFINITY) s = __fmul_rn(s, wexp(m, mx, c2));
          m = mx;
        }
#pragma unroll
        for (int e = 0; e < 16; ++e) s = __fadd_rn(s, wexp(x[e], m, c2));
      }
    }
  }
  // warp then block merge (consumer warps), fixed tree
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float m2 = __shfl_xor_sync(0xffffffffu, m, o);
    const float s2 = __shfl_xor_sync(0xffffffffu, s, o);
    merge_ms(m, s, m2, s2, c2);
  }
  __shared__ float sm[kStreamConsumers / 32], ss[kStreamConsumers / 32];
  if (lane == 0 && warp < kStreamConsumers / 32) {
    sm[warp] = m;
    ss[warp] = s;
  }
  __syncthreads();
  __shared__ bool s_last;
  if (threadIdx.x == 0) {
    if (s_timeout) sd_set_error(SD_DEVERR_TIMEOUT);
    float bm = sm[0], bs = ss[0];
    for (int w = 1; w < kStreamConsumers / 32; ++w) merge_ms(bm, bs, sm[w], ss[w], c2);
    part[(static_cast<long long>(b) * rows + rr) * n_seg + c] = make_float2(bm, bs);
    __threadfence();
    s_last = atomicAdd(&ticket[b], 1u) == static_cast<uint32_t>(rows * n_seg - 1);
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  accept_tail(zt, zd, K, V, c2, n_seg, b, s_x, u, n_emit, tokens, part, dlogit, ticket, info,
              kStreamThreads);
}

// ------------------------------------------------------------------ draw
// Weights of one element of the draw row from its two logits: residual
// (p - q)+ (l < K) and the unnormalised target weight exp2((z_T - m_T) * c2).
__device__ __forceinline__ void weights(float zt_v, float zd_v, const DrawInfo& di, int K, float c2, float& w_res,
                                        float& w_tgt) {
  const float et = wexp(zt_v, di.mt, c2);
  w_tgt = et;
  if (di.ell < K) {
    const float p = __fmul_rn(et, di.inv_zt);
    const float q = __fmul_rn(wexp(zd_v, di.md, c2), di.inv_zd);
    w_res = fmaxf(__fsub_rn(p, q), 0.f);
  } else {
    w_res = 0.f;
  }
}

constexpr int kDrawPer = 16;                     // consecutive values a thread owns
constexpr int kDrawChunk = kThreads * kDrawPer;  // values a CTA owns

// this thread's kDrawPer logits of both rows (missing values: -inf, weight 0)
__device__ __forceinline__ void draw_load(const float* rt, const float* rd, int v0, int V, bool vec, float (&xt)[kDrawPer],
                                          float (&xd)[kDrawPer]) {
  if (vec && v0 + kDrawPer <= V) {
#pragma unroll
    for (int q = 0; q < kDrawPer / 4; ++q) {
      const float4 a = __ldg(reinterpret_cast<const float4*>(rt + v0) + q);
      xt[4 * q] = a.x, xt[4 * q + 1] = a.y, xt[4 * q + 2] = a.z, xt[4 * q + 3] = a.w;
      const float4 d = rd ? __ldg(reinterpret_cast<const float4*>(rd + v0) + q) : make_float4(0.f, 0.f, 0.f, 0.f);
      xd[4 * q] = d.x, xd[4 * q + 1] = d.y, xd[4 * q + 2] = d.z, xd[4 * q + 3] = d.w;
    }
  } else {
#pragma unroll
    for (int e = 0; e < kDrawPer; ++e) {
      const bool in = v0 + e < V;
      xt[e] = in ? __ldg(rt + v0 + e) : -INFINITY;
      xd[e] = (in && rd) ? __ldg(rd + v0 + e) : 0.f;
    }
  }
}

__device__ float block_sum(float x, float* red) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) x = __fadd_rn(x, __shfl_xor_sync(0xffffffffu, x, o));
  __syncthreads();
  if (lane == 0) red[warp] = x;
  __syncthreads();
  float t = 0.f;
  if (threadIdx.x == 0)
    for (int w = 0; w < kThreads / 32; ++w) t = __fadd_rn(t, red[w]);
  return t;  // valid in thread 0
}

// grid (chunk, scene): chunk c of the draw row holds values [c * kDrawChunk,
// (c + 1) * kDrawChunk), thread t the kDrawPer consecutive values from
// c * kDrawChunk + t * kDrawPer, summed in order.
__global__ void __launch_bounds__(kThreads)
    sample_draw_kernel(const float* __restrict__ zt, const float* __restrict__ zd, int K, int V,
                       float c2, int n_chunks, bool vec, const float* __restrict__ u,
                       int32_t* __restrict__ tokens, const DrawInfo* __restrict__ info,
                       float2* __restrict__ sums, uint32_t* __restrict__ ticket) {
  const int c = blockIdx.x, b = blockIdx.y;
  // a programmatic dependent launch: resident while the statistics finish,
  // reading nothing they write before they have completed
  asm volatile("griddepcontrol.wait;" ::: "memory");
  const DrawInfo di = info[b];
  const float* rt = zt + (static_cast<long long>(b) * (K + 1) + di.ell) * V;
  const float* rd = di.ell < K ? zd + (static_cast<long long>(b) * K + di.ell) * V : nullptr;
  float xt[kDrawPer], xd[kDrawPer];
  draw_load(rt, rd, c * kDrawChunk + threadIdx.x * kDrawPer, V, vec, xt, xd);
  float sr = 0.f, sp = 0.f;
#pragma unroll
  for (int e = 0; e < kDrawPer; ++e) {
    float wr, wt;
    weights(xt[e], xd[e], di, K, c2, wr, wt);
    sr = __fadd_rn(sr, wr);
    sp = __fadd_rn(sp, wt);
  }
  __shared__ float red[kThreads / 32];
  const float tr = block_sum(sr, red);
  const float tp = block_sum(sp, red);
  __shared__ bool s_last;
  if (threadIdx.x == 0) {
    sums[static_cast<long long>(b) * n_chunks + c] = make_float2(tr, tp);
    __threadfence();
    s_last = atomicAdd(&ticket[b], 1u) == static_cast<uint32_t>(n_chunks - 1);
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  // ---- last CTA of scene b: choose the weights, locate the chunk, scan it
  __shared__ float s_sr[kMaxChunks], s_sp[kMaxChunks];
  for (int k = threadIdx.x; k < n_chunks; k += kThreads) {
    const float2 e = __ldcg(sums + static_cast<long long>(b) * n_chunks + k);
    s_sr[k] = e.x;
    s_sp[k] = e.y;
  }
  __syncthreads();
  __shared__ int s_chunk, s_use_res;
  __shared__ float s_base, s_target;
  if (threadIdx.x < 32) {
    const int lane = threadIdx.x;
    // lane l owns chunks [l*per, (l+1)*per): sequential lane sums, warp scan
    const int per = (n_chunks + 31) / 32;
    const int k0 = min(n_chunks, lane * per), k1 = min(n_chunks, k0 + per);
    float lr = 0.f, lp = 0.f;
    for (int k = k0; k < k1; ++k) {
      lr = __fadd_rn(lr, s_sr[k]);
      lp = __fadd_rn(lp, s_sp[k]);
    }
    float ir = lr, ip = lp;  // inclusive warp scan
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const float xr = __shfl_up_sync(0xffffffffu, ir, o);
      const float xp = __shfl_up_sync(0xffffffffu, ip, o);
      if (lane >= o) {
        ir = __fadd_rn(xr, ir);
        ip = __fadd_rn(xp, ip);
      }
    }
    const float tot_r = __shfl_sync(0xffffffffu, ir, 31);
    const float tot_p = __shfl_sync(0xffffffffu, ip, 31);
    const int use_res = (di.ell < K && tot_r > 0.f) ? 1 : 0;
    const float total = use_res ? tot_r : tot_p;
    const float target = __fmul_rn(u[static_cast<long long>(b) * (K + 1) + K], total);
    const float incl = use_res ? ir : ip;
    float run = __shfl_up_sync(0xffffffffu, incl, 1);
    if (lane == 0) run = 0.f;
    int found = -1, last_nz = -1;
    float base = 0.f;
    for (int k = k0; k < k1; ++k) {
      const float w = use_res ? s_sr[k] : s_sp[k];
      if (w > 0.f) last_nz = k;
      const float nxt = __fadd_rn(run, w);
      if (found < 0 && nxt > target) {
        found = k;
        base = run;
      }
      run = nxt;
    }
    const unsigned hit = __ballot_sync(0xffffffffu, found >= 0);
    int lnz = last_nz;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) lnz = max(lnz, __shfl_xor_sync(0xffffffffu, lnz, o));
    if (hit) {
      const int src = __ffs(hit) - 1;
      found = __shfl_sync(0xffffffffu, found, src);
      base = __shfl_sync(0xffffffffu, base, src);
    } else {
      // u * S at or above the rounded total: the draw is the last positive
      // weight, found by the in-chunk fallback below
      found = lnz >= 0 ? lnz : 0;
      base = -INFINITY;
    }
    if (lane == 0) {
      s_chunk = found;
      s_base = base;
      s_target = target;
      s_use_res = use_res;
    }
  }
  __syncthreads();
  // in-chunk scan: thread t owns the same kDrawPer consecutive values as in
  // the chunk sums above
  const int my_lo = s_chunk * kDrawChunk + threadIdx.x * kDrawPer;
  const bool use_res = s_use_res != 0;
  draw_load(rt, rd, my_lo, V, vec, xt, xd);
  float w[kDrawPer];
  float tsum = 0.f;
#pragma unroll
  for (int e = 0; e < kDrawPer; ++e) {
    float wr, wt;
    weights(xt[e], xd[e], di, K, c2, wr, wt);
    w[e] = use_res ? wr : wt;
    tsum = __fadd_rn(tsum, w[e]);
  }
  // exclusive prefix of the thread sums: warp scan + warp offsets (fixed)
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  float incl = tsum;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const float x = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl = __fadd_rn(x, incl);
  }
  float excl = __shfl_up_sync(0xffffffffu, incl, 1);
  if (lane == 0) excl = 0.f;
  __shared__ float s_wtot[kThreads / 32];
  if (lane == 31) s_wtot[warp] = incl;
  __syncthreads();
  float woff = 0.f;
  for (int q = 0; q < warp; ++q) woff = __fadd_rn(woff, s_wtot[q]);
  float run = __fadd_rn(s_base, __fadd_rn(woff, excl));
  int cand = 0x7fffffff, last_pos = -1;
#pragma unroll
  for (int e = 0; e < kDrawPer; ++e) {
    const int v = my_lo + e;
    if (w[e] > 0.f) last_pos = v;
    run = __fadd_rn(run, w[e]);
    if (cand == 0x7fffffff && run > s_target) cand = v;
  }
  // block min of candidates, block max of the last positive weight
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    cand = min(cand, __shfl_xor_sync(0xffffffffu, cand, o));
    last_pos = max(last_pos, __shfl_xor_sync(0xffffffffu, last_pos, o));
  }
  __shared__ int s_cand[kThreads / 32], s_lastp[kThreads / 32];
  if (lane == 0) {
    s_cand[warp] = cand;
    s_lastp[warp] = last_pos;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    int best = 0x7fffffff, lp = -1;
    for (int q = 0; q < kThreads / 32; ++q) {
      best = min(best, s_cand[q]);
      lp = max(lp, s_lastp[q]);
    }
    const int tok = best != 0x7fffffff ? best : (lp >= 0 ? lp : s_chunk * kDrawChunk);
    tokens[static_cast<long long>(b) * (K + 1) + di.ell] = tok;
    ticket[b] = 0;
  }
}

struct Plan {
  int chunk1, n1, chunk2, n2;
  bool vec;
  int chunk_scalar, n_scalar;  // the scalar stats kernel's chunking (unaligned rows)
};

// Vectorised stats when every row starts on a 16-byte boundary (V a multiple
// of 4 and a 16-byte-aligned base, checked at the call).
Plan plan(int V) {
  Plan p;
  p.vec = V % 4 == 0;
  p.chunk1 = p.vec ? kVecChunk : 4096;
  while ((V + p.chunk1 - 1) / p.chunk1 > kMaxChunks) p.chunk1 *= 2;
  p.n1 = (V + p.chunk1 - 1) / p.chunk1;
  p.chunk_scalar = 4096;
  while ((V + p.chunk_scalar - 1) / p.chunk_scalar > kMaxChunks) p.chunk_scalar *= 2;
  p.n_scalar = (V + p.chunk_scalar - 1) / p.chunk_scalar;
  p.chunk2 = kDrawChunk;
  p.n2 = (V + p.chunk2 - 1) / p.chunk2;
  return p;
}

struct Layout {
  size_t part, dlogit, ticket1, info, sums, ticket2, total;
};

Layout layout(int B, int K, const Plan& p) {
  Layout l;
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t at = off;
    off += (bytes + 255) / 256 * 256;
    return at;
  };
  // room for the scalar chunking's partials too (rows found unaligned at the call)
  l.part = take(static_cast<size_t>(B) * (2 * K + 1) * (p.n_scalar > p.n1 ? p.n_scalar : p.n1) * sizeof(float2));
  l.dlogit = take(static_cast<size_t>(B) * (2 * K + 1) * sizeof(float));
  l.ticket1 = take(static_cast<size_t>(B) * 4);
  l.info = take(static_cast<size_t>(B) * sizeof(DrawInfo));
  l.sums = take(static_cast<size_t>(B) * p.n2 * sizeof(float2));
  l.ticket2 = take(static_cast<size_t>(B) * 4);
  l.total = off;
  return l;
}

constexpr int kStreamSmem = kStreamStages * kStageFloats * 4;

// SMs of the current device, once the streaming kernel's shared-memory
// attribute is set there; 0 when either call fails (the one-shot kernel runs).
int stream_sms() {
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
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
        cudaFuncSetAttribute(sample_stats_stream_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             kStreamSmem) != cudaSuccess) {
      (void)cudaGetLastError();
      n = 0;
    }
    cache[dev] = n;
  }
  return cache[dev];
}

}  // namespace

extern "C" size_t sd_accept_sample_workspace(int B, int K, int V) {
  if (B <= 0 || K < 0 || V <= 0) return 0;
  return layout(B, K, plan(V)).total;
}

extern "C" sd_status sd_accept_sample(const float* z_target, const float* z_draft, int B, int K,
                                      int V, float temperature, const int32_t* draft,
                                      const float* u, int32_t* n_emit, int32_t* tokens, void* ws,
                                      size_t ws_bytes, sd_stream_t stream) {
  if (B < 0 || K < 0 || V <= 0) return SD_ERR_INVALID_ARG;
  if (!(temperature > 0.f) || !isfinite(temperature)) return SD_ERR_INVALID_ARG;
  if (K > 128 || B > 65535 || (V + kDrawChunk - 1) / kDrawChunk > kMaxChunks) return SD_ERR_UNSUPPORTED;
  if (B == 0) return SD_OK;
  if (!z_target || !u || !n_emit || !tokens || (K > 0 && (!z_draft || !draft)))
    return SD_ERR_INVALID_ARG;
  Plan p = plan(V);
  const Layout l = layout(B, K, p);
  // the vectorised stats also need 16-byte-aligned rows (same workspace either way)
  if ((reinterpret_cast<uintptr_t>(z_target) & 15) || (K > 0 && (reinterpret_cast<uintptr_t>(z_draft) & 15))) {
    p.vec = false;
    p.chunk1 = p.chunk_scalar;
    p.n1 = p.n_scalar;
  }
  if (!ws || ws_bytes < l.total || !sd_aligned16(ws)) return SD_ERR_WORKSPACE;
  char* w = static_cast<char*>(ws);
  auto* part = reinterpret_cast<float2*>(w + l.part);
  auto* dlogit = reinterpret_cast<float*>(w + l.dlogit);
  auto* ticket1 = reinterpret_cast<uint32_t*>(w + l.ticket1);
  auto* info = reinterpret_cast<DrawInfo*>(w + l.info);
  auto* sums = reinterpret_cast<float2*>(w + l.sums);
  auto* ticket2 = reinterpret_cast<uint32_t*>(w + l.ticket2);
  const float c2 = static_cast<float>(kLog2e / static_cast<double>(temperature));
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  const int n_sm = stream_sms();
  if (p.vec && n_sm > 0) {
    // segments of whole stages, about two CTAs per SM over all (row, scene) pairs
    const long long rows_all = static_cast<long long>(2 * K + 1) * B;
    long long n_seg = (2LL * n_sm + rows_all - 1) / rows_all;
    n_seg = n_seg < 1 ? 1 : (n_seg > p.n1 ? p.n1 : n_seg);
    const int seg = static_cast<int>(((V + n_seg - 1) / n_seg + kStageFloats - 1) / kStageFloats * kStageFloats);
    const int ns = (V + seg - 1) / seg;
    sample_stats_stream_kernel<<<dim3(ns, 2 * K + 1, B), kStreamThreads, kStreamSmem, st>>>(
        z_target, z_draft, K, V, c2, seg, ns, draft, u, n_emit, tokens, part, dlogit, ticket1, info);
  } else if (p.vec)
    sample_stats_kernel<true><<<dim3(p.n1, 2 * K + 1, B), kVecThreads, 0, st>>>(
        z_target, z_draft, K, V, c2, p.chunk1, p.n1, draft, u, n_emit, tokens, part, dlogit, ticket1, info);
  else
    sample_stats_kernel<false><<<dim3(p.n1, 2 * K + 1, B), kThreads, 0, st>>>(
        z_target, z_draft, K, V, c2, p.chunk1, p.n1, draft, u, n_emit, tokens, part, dlogit, ticket1, info);
  SD_CHECK_LAUNCH();
  // the draw is a programmatic dependent launch (it waits for the
  // statistics before its first read of their results)
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.gridDim = dim3(p.n2, B, 1);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.stream = st;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  const bool vec = p.vec;
  if (cudaLaunchKernelEx(&cfg, sample_draw_kernel, z_target, z_draft, K, V, c2, p.n2, vec, u, static_cast<int32_t*>(tokens),
                         static_cast<const DrawInfo*>(info), sums, ticket2) != cudaSuccess) {
    (void)cudaGetLastError();
    return SD_ERR_CUDA;
  }
  return SD_OK;
}
