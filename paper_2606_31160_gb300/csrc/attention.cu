// K3: verify attention of the K + 1 new rows against the cached prefix
// (Eq. verify, Sec. 2.2), GQA, causal, bf16 in / bf16 out, fp32 softmax.
//
// Work decomposition (one launch, no workspace, no second pass):
//   * One thread-block CLUSTER per (scene b, KV head g, block of packed query
//     rows). The G query heads of KV head g times the R verify rows are packed
//     into one M = G*R row tile ("packed rows", p = i*G + gq), so every K/V row
//     of that head is fetched from HBM exactly once.
//   * The C CTAs of a cluster split the valid keys 0..len[b]-1 into C
//     contiguous, 16-key-aligned ranges (split-L / flash-decoding).
//   * Inside a CTA a producer warp streams its range with TMA tensor loads
//     (cp.async.bulk.tensor, 128-byte swizzle, 16-row boxes) into a ring of
//     64-key stages guarded by mbarriers; every stage holds K and V.
//   * Four consumer warps per 16*MT-row group each own one 16-key block of
//     every stage: S = Q K^T and O += P V on mma.sync m16n8k16 bf16 tensor
//     cores with fp32 accumulators, online softmax kept per warp in
//     registers (P never leaves registers).
//   * End: the warps' (m, l, O) partials merge in shared memory, then the
//     cluster's CTA partials merge through distributed shared memory
//     (mapa + ld.shared::cluster); each CTA finalises a slice of the rows and
//     writes bf16 output. Every merge runs in a fixed order, so results are
//     deterministic.
//
// Masking: row i of scene b is the token at position L_b + i, L_b = len[b] - R,
// and sees keys 0 .. L_b + i. Keys past len[b] (stale cache rows, TMA
// out-of-bounds fill) are excluded by selection, and the V rows of the final
// partial block are zeroed in shared memory before the P V product, so stale
// NaN/Inf in the cache never reaches the output.
//
// Every mbarrier wait is bounded; a wait that runs out sets
// SD_DEVERR_TIMEOUT and the CTA carries on to the cluster barriers instead of
// hanging.
#include "common.cuh"

#include <cuda.h>  // CUtensorMap and its enums (header only; no libcuda link)

#include <math.h>
#include <mutex>

SD_DEFINE_ERROR_ACCESSOR(sd_take_error_attention)

namespace {

constexpr int kBlockKeys = 16;             // keys per consumer warp per stage
constexpr int kTileKeys = 4 * kBlockKeys;  // keys per stage
constexpr uint32_t kSpinLimit = 1u << 20;  // bounded mbarrier polls (well under a second)

// --------------------------------------------------------------------------
// PTX wrappers
// --------------------------------------------------------------------------
__device__ __forceinline__ uint32_t smem_addr(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}

__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes)
               : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}

// Bounded wait: false (and the timeout bit) when the phase never completes.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity) {
  for (uint32_t i = 0; i < kSpinLimit; ++i)
    if (mbar_try_wait(bar, parity)) return true;
  sd_set_error(SD_DEVERR_TIMEOUT);
  return false;
}

__device__ __forceinline__ void tma_load_3d(uint32_t dst, const CUtensorMap* map, uint32_t bar,
                                            int x, int y, int z) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%3, %4, %5}], [%2];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(bar), "r"(x), "r"(y), "r"(z)
      : "memory");
}

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                        uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}

__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                          uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}

__device__ __forceinline__ void mma_bf16(float (&c)[4], uint32_t a0, uint32_t a1, uint32_t a2,
                                         uint32_t a3, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
      "{%8,%9}, {%0,%1,%2,%3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ void named_bar_sync(int id, int threads) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(threads) : "memory");
}

__device__ __forceinline__ void cluster_sync_all() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::
                   : "memory");
}

__device__ __forceinline__ uint32_t cluster_map(uint32_t addr, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(addr), "r"(rank));
  return r;
}

__device__ __forceinline__ float ld_cluster_f32(uint32_t addr) {
  float v;
  asm volatile("ld.shared::cluster.f32 %0, [%1];" : "=f"(v) : "r"(addr) : "memory");
  return v;
}

__device__ __forceinline__ float4 ld_cluster_f32x4(uint32_t addr) {
  float4 v;
  asm volatile("ld.shared::cluster.v4.f32 {%0,%1,%2,%3}, [%4];"
               : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
               : "r"(addr)
               : "memory");
  return v;
}

// 128-byte swizzle of a [rows][128 B] region whose base is 1024-byte aligned:
// 16-byte chunk c of row r sits at chunk c ^ (r & 7). TMA's SWIZZLE_128B mode
// writes this layout and every ldmatrix below reads it.
__device__ __forceinline__ uint32_t swz(int row, int chunk) {
  return static_cast<uint32_t>(row * 128 + ((chunk ^ (row & 7)) << 4));
}

// --------------------------------------------------------------------------
// Configuration
// --------------------------------------------------------------------------
template <int D, int MT, int NMG>
struct Cfg {
  static constexpr int kHalves = D / 64;                  // 128-byte column halves
  static constexpr int kRowsW = 16 * MT;                  // packed rows per consumer warp
  static constexpr int kRows = kRowsW * NMG;              // packed rows per CTA
  static constexpr int kConsumerWarps = 4 * NMG;
  static constexpr int kConsumerThreads = 32 * kConsumerWarps;
  static constexpr int kThreads = kConsumerThreads + 32;  // + producer warp
  static constexpr int kHalfTileBytes = kTileKeys * 128;
  static constexpr int kKVTileBytes = kHalves * kHalfTileBytes;
  static constexpr int kStageBytes = 2 * kKVTileBytes;
  static constexpr int kStages = D == 128 ? 6 : 10;
  static constexpr int kRingBytes = kStages * kStageBytes;
  static constexpr int kQHalfBytes = kRows * 128;
  static constexpr int kQBytes = kHalves * kQHalfBytes;
  static constexpr int kLd = D + 4;                       // padded fp32 row stride
  static constexpr int kWarpPartFloats = kRowsW * kLd + 2 * kRowsW;
  static constexpr int kWarpPartBytes = kConsumerWarps * kWarpPartFloats * 4;
  static constexpr int kCtaPartFloats = kRows * kLd + 2 * kRows;
  static constexpr int kCtaPartBytes = kCtaPartFloats * 4;
  static constexpr int kBarBytes = 2 * kStages * 8;
  static constexpr int kSmemBytes = kRingBytes + kQBytes + kBarBytes + 1024;
  static_assert(kWarpPartBytes + kCtaPartBytes <= kRingBytes, "merge areas must fit in the ring");
  static_assert(kSmemBytes <= 227 * 1024, "shared memory budget");
};

struct AttnArgs {
  const __nv_bfloat16* q;
  __nv_bfloat16* out;
  const int32_t* len;
  int R, Hq, Hkv, G, M, cap;
  float scale_log2;  // softmax scale * log2(e)
};

// --------------------------------------------------------------------------
// Kernel
// --------------------------------------------------------------------------
template <int D, int MT, int NMG>
__global__ void __launch_bounds__(Cfg<D, MT, NMG>::kThreads, 1)
    verify_attn_kernel(const __grid_constant__ CUtensorMap tm_k,
                       const __grid_constant__ CUtensorMap tm_v, const AttnArgs a) {
  using C = Cfg<D, MT, NMG>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  const uint32_t ring = smem_addr(smem);
  const uint32_t qs = ring + C::kRingBytes;
  const uint32_t bars = qs + C::kQBytes;  // full[kStages], then empty[kStages]
  auto full_bar = [&](int s) { return bars + 8u * s; };
  auto empty_bar = [&](int s) { return bars + 8u * (C::kStages + s); };
  auto k_stage = [&](int s) { return ring + s * C::kStageBytes; };
  auto v_stage = [&](int s) { return ring + s * C::kStageBytes + C::kKVTileBytes; };

  const int rank = blockIdx.x;  // cluster rank: the cluster spans the grid's x extent
  const int csize = gridDim.x;
  const int kvh = blockIdx.y % a.Hkv;
  const int mblock = blockIdx.y / a.Hkv;
  const int b = blockIdx.z;
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int s = 0; s < C::kStages; ++s) {
      mbar_init(full_bar(s), 1);
      mbar_init(empty_bar(s), C::kConsumerWarps);
    }
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncthreads();

  const int n_keys = a.len[b];
  const bool valid = n_keys >= a.R && n_keys <= a.cap;
  if (!valid && rank == 0 && threadIdx.x == 0 && blockIdx.y == 0) sd_set_error(SD_DEVERR_LENGTH);
  const int nblk = valid ? (n_keys + kBlockKeys - 1) / kBlockKeys : 0;
  const int blk_begin = static_cast<int>((static_cast<long long>(rank) * nblk) / csize);
  const int blk_end = static_cast<int>((static_cast<long long>(rank + 1) * nblk) / csize);
  const int n_tiles = (blk_end - blk_begin + 3) / 4;

  float* cta_part = reinterpret_cast<float*>(smem + C::kWarpPartBytes);

  if (warp == C::kConsumerWarps) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      const int z = b * a.Hkv + kvh;
      for (int t = 0; t < n_tiles; ++t) {
        const int s = t % C::kStages;
        if (t >= C::kStages) mbar_wait(empty_bar(s), ((t / C::kStages) - 1) & 1);
        const int nb = min(4, blk_end - blk_begin - 4 * t);
        mbar_expect_tx(full_bar(s), static_cast<uint32_t>(nb * C::kHalves * 2 * kBlockKeys * 128));
        for (int j = 0; j < nb; ++j) {
          const int y = (blk_begin + 4 * t + j) * kBlockKeys;
#pragma unroll
          for (int h = 0; h < C::kHalves; ++h) {
            const uint32_t off = h * C::kHalfTileBytes + j * kBlockKeys * 128;
            tma_load_3d(k_stage(s) + off, &tm_k, full_bar(s), h * 64, y, z);
            tma_load_3d(v_stage(s) + off, &tm_v, full_bar(s), h * 64, y, z);
          }
        }
      }
    }
    __syncwarp();
  } else {
    // ------------------------------------------------------------ consumers
    const int tid = threadIdx.x;
    // packed query rows of this CTA -> shared memory (swizzled like the K tiles)
    for (int idx = tid; idx < C::kRows * (D / 8); idx += C::kConsumerThreads) {
      const int row = idx / (D / 8);
      const int chunk = idx % (D / 8);
      const int p = mblock * C::kRows + row;
      uint4 val = make_uint4(0, 0, 0, 0);
      if (valid && p < a.M) {
        const int i = p / a.G, gq = p % a.G;
        const long long off = ((static_cast<long long>(b) * a.R + i) * a.Hq + kvh * a.G + gq) * D;
        val = *reinterpret_cast<const uint4*>(a.q + off + chunk * 8);
      }
      const uint32_t dst = qs + (chunk >> 3) * C::kQHalfBytes + swz(row, chunk & 7);
      asm volatile("st.shared.v4.u32 [%0], {%1,%2,%3,%4};" ::"r"(dst), "r"(val.x), "r"(val.y),
                   "r"(val.z), "r"(val.w)
                   : "memory");
    }
    named_bar_sync(1, C::kConsumerThreads);

    const int mg = warp >> 2;  // row group of this warp
    const int ks = warp & 3;   // 16-key block of every stage owned by this warp
    const int g8 = lane >> 2;
    const int t4 = lane & 3;
    const int L_prefix = n_keys - a.R;

    // last visible key of each of this thread's rows
    int lim[MT][2];
#pragma unroll
    for (int mt = 0; mt < MT; ++mt)
#pragma unroll
      for (int hh = 0; hh < 2; ++hh) {
        const int p = mblock * C::kRows + mg * C::kRowsW + mt * 16 + g8 + 8 * hh;
        lim[mt][hh] = min(L_prefix + p / a.G, n_keys - 1);
      }

    float o[MT][D / 8][4];
    float m_run[MT][2], l_run[MT][2];
#pragma unroll
    for (int mt = 0; mt < MT; ++mt) {
#pragma unroll
      for (int nd = 0; nd < D / 8; ++nd)
#pragma unroll
        for (int c = 0; c < 4; ++c) o[mt][nd][c] = 0.f;
      m_run[mt][0] = m_run[mt][1] = -INFINITY;
      l_run[mt][0] = l_run[mt][1] = 0.f;
    }

    // ldmatrix lane roles
    const int a_row = (lane & 7) + ((lane >> 3) & 1) * 8;  // A (Q) and trans-B (V): row in 16
    const int a_chk = lane >> 4;                             // A: +0 / +1 chunk
    const int b_row = (lane & 7) + (lane >> 4) * 8;          // B (K): key row in 16
    const int b_chk = (lane >> 3) & 1;                       // B: +0 / +1 chunk

    for (int t = 0; t < n_tiles; ++t) {
      const int s = t % C::kStages;
      mbar_wait(full_bar(s), (t / C::kStages) & 1);
      const int blk = blk_begin + 4 * t + ks;
      if (blk < blk_end) {
        const int key0 = blk * kBlockKeys;
        const uint32_t kb = k_stage(s);
        const uint32_t vb = v_stage(s);
        // ---- S = Q K^T over this warp's 16 keys
        float sc[MT][2][4];
#pragma unroll
        for (int mt = 0; mt < MT; ++mt)
#pragma unroll
          for (int nt = 0; nt < 2; ++nt)
#pragma unroll
            for (int c = 0; c < 4; ++c) sc[mt][nt][c] = 0.f;
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
          const int half = kk >> 2;
          const int chunk = (kk & 3) * 2;
          uint32_t kf0, kf1, kf2, kf3;
          ldsm_x4(kb + half * C::kHalfTileBytes + swz(ks * 16 + b_row, chunk + b_chk), kf0, kf1,
                  kf2, kf3);
#pragma unroll
          for (int mt = 0; mt < MT; ++mt) {
            uint32_t qa0, qa1, qa2, qa3;
            ldsm_x4(qs + half * C::kQHalfBytes +
                        swz(mg * C::kRowsW + mt * 16 + a_row, chunk + a_chk),
                    qa0, qa1, qa2, qa3);
            mma_bf16(sc[mt][0], qa0, qa1, qa2, qa3, kf0, kf1);
            mma_bf16(sc[mt][1], qa0, qa1, qa2, qa3, kf2, kf3);
          }
        }
        // ---- scale, causal / length mask, online softmax, P -> bf16 fragments
        uint32_t pa[MT][4];
#pragma unroll
        for (int mt = 0; mt < MT; ++mt) {
#pragma unroll
          for (int hh = 0; hh < 2; ++hh) {
            float v[4];
#pragma unroll
            for (int nt = 0; nt < 2; ++nt)
#pragma unroll
              for (int c = 0; c < 2; ++c) {
                const int key = key0 + nt * 8 + 2 * t4 + c;
                const float x = sc[mt][nt][2 * hh + c] * a.scale_log2;
                v[nt * 2 + c] = key <= lim[mt][hh] ? x : -INFINITY;
              }
            float mx = fmaxf(fmaxf(v[0], v[1]), fmaxf(v[2], v[3]));
            mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
            mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 2));
            const float m_new = fmaxf(m_run[mt][hh], mx);
            const float m_base = m_new == -INFINITY ? 0.f : m_new;
            const float corr = ex2(m_run[mt][hh] - m_base);
            m_run[mt][hh] = m_new;
            const uint32_t w0 = sd_pack_bf16x2(ex2(v[0] - m_base), ex2(v[1] - m_base));
            const uint32_t w1 = sd_pack_bf16x2(ex2(v[2] - m_base), ex2(v[3] - m_base));
            // the normaliser sums the same bf16-rounded weights the MMA uses
            const float rs = (sd_bf16_lo(w0) + sd_bf16_hi(w0)) + (sd_bf16_lo(w1) + sd_bf16_hi(w1));
            l_run[mt][hh] = fmaf(l_run[mt][hh], corr, rs);
#pragma unroll
            for (int nd = 0; nd < D / 8; ++nd) {
              o[mt][nd][2 * hh] *= corr;
              o[mt][nd][2 * hh + 1] *= corr;
            }
            pa[mt][hh] = w0;      // a0 / a1: keys 0..7 of the block
            pa[mt][2 + hh] = w1;  // a2 / a3: keys 8..15
          }
        }
        // ---- the scene's last block: zero V rows past len (stale cache data)
        if (key0 + kBlockKeys > n_keys) {
          const int first = n_keys - key0;
          const int n_chunks = (kBlockKeys - first) * C::kHalves * 8;
          for (int cidx = lane; cidx < n_chunks; cidx += 32) {
            const int r = first + cidx / (C::kHalves * 8);
            const int rem = cidx % (C::kHalves * 8);
            const uint32_t addr = vb + (rem >> 3) * C::kHalfTileBytes + (ks * 16 + r) * 128 +
                                  (rem & 7) * 16;
            asm volatile("st.shared.v4.u32 [%0], {%1,%1,%1,%1};" ::"r"(addr), "r"(0) : "memory");
          }
          __syncwarp();
        }
        // ---- O += P V
#pragma unroll
        for (int dp = 0; dp < D / 16; ++dp) {
          const int chunk = dp * 2;  // d chunks 2dp, 2dp+1 (8 values each)
          uint32_t v0, v1, v2, v3;
          ldsm_x4_t(vb + (chunk >> 3) * C::kHalfTileBytes +
                        swz(ks * 16 + a_row, (chunk & 7) + a_chk),
                    v0, v1, v2, v3);
#pragma unroll
          for (int mt = 0; mt < MT; ++mt) {
            mma_bf16(o[mt][2 * dp], pa[mt][0], pa[mt][1], pa[mt][2], pa[mt][3], v0, v1);
            mma_bf16(o[mt][2 * dp + 1], pa[mt][0], pa[mt][1], pa[mt][2], pa[mt][3], v2, v3);
          }
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(empty_bar(s));
    }

    // ---- per-warp partial -> shared memory (the ring is free: every tile landed
    //      and was consumed by every consumer warp)
    named_bar_sync(1, C::kConsumerThreads);
    float* wp = reinterpret_cast<float*>(smem) + warp * C::kWarpPartFloats;
#pragma unroll
    for (int mt = 0; mt < MT; ++mt) {
#pragma unroll
      for (int hh = 0; hh < 2; ++hh) {
        float l = l_run[mt][hh];
        l += __shfl_xor_sync(0xffffffffu, l, 1);
        l += __shfl_xor_sync(0xffffffffu, l, 2);
        const int r = mt * 16 + g8 + 8 * hh;
#pragma unroll
        for (int nd = 0; nd < D / 8; ++nd)
          *reinterpret_cast<float2*>(wp + r * C::kLd + nd * 8 + 2 * t4) =
              make_float2(o[mt][nd][2 * hh], o[mt][nd][2 * hh + 1]);
        if (t4 == 0) {
          wp[C::kRowsW * C::kLd + r] = m_run[mt][hh];
          wp[C::kRowsW * C::kLd + C::kRowsW + r] = l;
        }
      }
    }
    named_bar_sync(1, C::kConsumerThreads);
    // ---- merge the four key-slice warps of each row group (fixed order)
    for (int idx = tid; idx < C::kRows * (D / 4); idx += C::kConsumerThreads) {
      const int row = idx / (D / 4);
      const int col = (idx % (D / 4)) * 4;
      const int g = row / C::kRowsW;
      const int rw = row % C::kRowsW;
      float mw[4], mmax = -INFINITY;
#pragma unroll
      for (int w = 0; w < 4; ++w) {
        const float* part = reinterpret_cast<float*>(smem) + (g * 4 + w) * C::kWarpPartFloats;
        mw[w] = part[C::kRowsW * C::kLd + rw];
        mmax = fmaxf(mmax, mw[w]);
      }
      float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
      float lsum = 0.f;
#pragma unroll
      for (int w = 0; w < 4; ++w) {
        const float* part = reinterpret_cast<float*>(smem) + (g * 4 + w) * C::kWarpPartFloats;
        const float f = mw[w] == -INFINITY ? 0.f : ex2(mw[w] - mmax);
        const float4 ov = *reinterpret_cast<const float4*>(part + rw * C::kLd + col);
        acc.x = fmaf(f, ov.x, acc.x);
        acc.y = fmaf(f, ov.y, acc.y);
        acc.z = fmaf(f, ov.z, acc.z);
        acc.w = fmaf(f, ov.w, acc.w);
        lsum = fmaf(f, part[C::kRowsW * C::kLd + C::kRowsW + rw], lsum);
      }
      *reinterpret_cast<float4*>(cta_part + row * C::kLd + col) = acc;
      if (col == 0) {
        cta_part[C::kRows * C::kLd + row] = mmax;
        cta_part[C::kRows * C::kLd + C::kRows + row] = lsum;
      }
    }
  }

  // ---- cluster merge through distributed shared memory
  __syncthreads();
  cluster_sync_all();
  {
    const int rpc = C::kRows / csize;  // rows finalised by this CTA
    const uint32_t part_local = smem_addr(cta_part);
    for (int idx = threadIdx.x; idx < rpc * (D / 4); idx += C::kThreads) {
      const int row = rank * rpc + idx / (D / 4);
      const int col = (idx % (D / 4)) * 4;
      const int p = mblock * C::kRows + row;
      float mmax = -INFINITY;
      for (int c = 0; c < csize; ++c) {
        const uint32_t base = cluster_map(part_local, c);
        mmax = fmaxf(mmax, ld_cluster_f32(base + 4u * (C::kRows * C::kLd + row)));
      }
      float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
      float lsum = 0.f;
      for (int c = 0; c < csize; ++c) {
        const uint32_t base = cluster_map(part_local, c);
        const float mc = ld_cluster_f32(base + 4u * (C::kRows * C::kLd + row));
        const float f = mc == -INFINITY ? 0.f : ex2(mc - mmax);
        const float lc = ld_cluster_f32(base + 4u * (C::kRows * C::kLd + C::kRows + row));
        const float4 oc = ld_cluster_f32x4(base + 4u * (row * C::kLd + col));
        acc.x = fmaf(f, oc.x, acc.x);
        acc.y = fmaf(f, oc.y, acc.y);
        acc.z = fmaf(f, oc.z, acc.z);
        acc.w = fmaf(f, oc.w, acc.w);
        lsum = fmaf(f, lc, lsum);
      }
      if (valid && p < a.M && lsum > 0.f) {
        const float inv = 1.f / lsum;
        const int i = p / a.G, gq = p % a.G;
        const long long off =
            ((static_cast<long long>(b) * a.R + i) * a.Hq + kvh * a.G + gq) * D + col;
        uint2 packed = make_uint2(sd_pack_bf16x2(acc.x * inv, acc.y * inv),
                                  sd_pack_bf16x2(acc.z * inv, acc.w * inv));
        *reinterpret_cast<uint2*>(a.out + off) = packed;
      }
    }
  }
  cluster_sync_all();  // no CTA leaves while a peer still reads its shared memory
}

// --------------------------------------------------------------------------
// Host side
// --------------------------------------------------------------------------
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

// [B*Hkv][cap][D] bf16 viewed as a 3-D tensor; boxes of 64 columns x 16 rows.
bool make_kv_map(CUtensorMap* map, void* base, int D, int cap, int planes) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[3] = {static_cast<cuuint64_t>(D), static_cast<cuuint64_t>(cap),
                        static_cast<cuuint64_t>(planes)};
  cuuint64_t strides[2] = {static_cast<cuuint64_t>(D) * 2,
                           static_cast<cuuint64_t>(cap) * static_cast<cuuint64_t>(D) * 2};
  cuuint32_t box[3] = {64, kBlockKeys, 1};
  cuuint32_t estr[3] = {1, 1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, base, dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

constexpr int kClusterSizes[5] = {1, 2, 4, 8, 16};

template <int D, int MT, int NMG>
struct Launcher {
  using C = Cfg<D, MT, NMG>;
  // per device: attributes set, and the number of co-resident clusters per size
  struct DevState {
    bool ready = false;
    int active[5] = {0, 0, 0, 0, 0};
  };

  static DevState* state() {
    static DevState st[16];
    static std::mutex mu;
    int dev = 0;
    cudaGetDevice(&dev);
    if (dev < 0 || dev >= 16) return nullptr;
    std::lock_guard<std::mutex> lock(mu);
    DevState& s = st[dev];
    if (!s.ready) {
      auto kern = verify_attn_kernel<D, MT, NMG>;
      if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, C::kSmemBytes) !=
              cudaSuccess ||
          cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) !=
              cudaSuccess) {
        (void)cudaGetLastError();
        return nullptr;
      }
      for (int i = 0; i < 5; ++i) {
        cudaLaunchConfig_t cfg = {};
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeClusterDimension;
        attr[0].val.clusterDim.x = kClusterSizes[i];
        attr[0].val.clusterDim.y = 1;
        attr[0].val.clusterDim.z = 1;
        cfg.gridDim = dim3(kClusterSizes[i], 1, 1);
        cfg.blockDim = dim3(C::kThreads, 1, 1);
        cfg.dynamicSmemBytes = C::kSmemBytes;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        int n = 0;
        if (cudaOccupancyMaxActiveClusters(&n, reinterpret_cast<const void*>(kern), &cfg) !=
            cudaSuccess) {
          (void)cudaGetLastError();
          n = 0;
        }
        s.active[i] = n;
      }
      s.ready = true;
    }
    return &s;
  }

  // Cluster size: minimise waves x (16-key blocks per CTA + a fixed per-CTA cost).
  static int pick_cluster(const DevState& s, long long units, int cap) {
    const long long nblk = (cap + kBlockKeys - 1) / kBlockKeys;
    long long best_cost = -1;
    int best = 0;
    for (int i = 0; i < 5; ++i) {
      const int cs = kClusterSizes[i];
      if (s.active[i] <= 0) continue;
      if (cs > 1 && nblk < 4LL * cs) continue;
      if (cs > C::kRows) continue;
      const long long waves = (units + s.active[i] - 1) / s.active[i];
      const long long cost = waves * ((nblk + cs - 1) / cs + 8);
      if (best_cost < 0 || cost < best_cost) {
        best_cost = cost;
        best = cs;
      }
    }
    return best;
  }

  static sd_status run(const CUtensorMap& tk, const CUtensorMap& tv, const AttnArgs& a, int B,
                       int n_mblocks, cudaStream_t stream) {
    DevState* s = state();
    if (!s) return SD_ERR_CUDA;
    const long long units = static_cast<long long>(B) * a.Hkv * n_mblocks;
    const int cs = pick_cluster(*s, units, a.cap);
    if (cs <= 0) return SD_ERR_UNSUPPORTED;
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = cs;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.gridDim = dim3(cs, a.Hkv * n_mblocks, B);
    cfg.blockDim = dim3(C::kThreads, 1, 1);
    cfg.dynamicSmemBytes = C::kSmemBytes;
    cfg.stream = stream;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    if (cudaLaunchKernelEx(&cfg, verify_attn_kernel<D, MT, NMG>, tk, tv, a) != cudaSuccess) {
      (void)cudaGetLastError();
      return SD_ERR_CUDA;
    }
    return SD_OK;
  }
};

template <int D>
sd_status dispatch_rows(const CUtensorMap& tk, const CUtensorMap& tv, const AttnArgs& a, int B,
                        cudaStream_t stream) {
  if (a.M <= 16) return Launcher<D, 1, 1>::run(tk, tv, a, B, 1, stream);
  if (a.M <= 32) return Launcher<D, 2, 1>::run(tk, tv, a, B, 1, stream);
  return Launcher<D, 2, 2>::run(tk, tv, a, B, (a.M + 63) / 64, stream);
}

}  // namespace

extern "C" sd_status sd_verify_attention(const void* q, const sd_kv_cache* cache, void* out,
                                         int R, int Hq, float scale, sd_stream_t stream) {
  if (!cache) return SD_ERR_INVALID_ARG;
  const int B = cache->batch, Hkv = cache->n_kv_heads, cap = cache->capacity, D = cache->head_dim;
  if (B < 0 || R <= 0 || Hq <= 0 || Hkv <= 0 || cap <= 0) return SD_ERR_INVALID_ARG;
  if (Hq % Hkv) return SD_ERR_INVALID_ARG;
  if (D != 64 && D != 128) return SD_ERR_UNSUPPORTED;
  const int G = Hq / Hkv;
  if (static_cast<long long>(G) * R > 128) return SD_ERR_UNSUPPORTED;
  if (B == 0) return SD_OK;
  if (B > 65535 || Hkv * ((G * R + 63) / 64) > 65535) return SD_ERR_UNSUPPORTED;
  if (!q || !out || !cache->k || !cache->v || !cache->len) return SD_ERR_INVALID_ARG;
  if (!sd_aligned16(q) || !sd_aligned16(out) || !sd_aligned16(cache->k) || !sd_aligned16(cache->v))
    return SD_ERR_INVALID_ARG;
  if (!(scale >= 0.f) || !isfinite(scale)) return SD_ERR_INVALID_ARG;
  CUtensorMap tk, tv;
  if (!make_kv_map(&tk, cache->k, D, cap, B * Hkv) || !make_kv_map(&tv, cache->v, D, cap, B * Hkv))
    return SD_ERR_CUDA;
  AttnArgs a;
  a.q = static_cast<const __nv_bfloat16*>(q);
  a.out = static_cast<__nv_bfloat16*>(out);
  a.len = cache->len;
  a.R = R;
  a.Hq = Hq;
  a.Hkv = Hkv;
  a.G = G;
  a.M = G * R;
  a.cap = cap;
  const float sc = scale > 0.f ? scale : static_cast<float>(1.0 / sqrt(static_cast<double>(D)));
  a.scale_log2 = static_cast<float>(static_cast<double>(sc) * 1.4426950408889634);
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  return D == 64 ? dispatch_rows<64>(tk, tv, a, B, st) : dispatch_rows<128>(tk, tv, a, B, st);
}
