// K3: verify attention of the K + 1 new rows against the cached prefix
// (Eq. verify, Sec. 3.2), GQA, causal, bf16 in / bf16 out, fp32 softmax.
//
// Work decomposition (one launch):
//   * A "unit" is (scene b, KV head g, block of packed query rows). The G
//     query heads of KV head g times the R verify rows are packed into one
//     M = G*R row tile (packed row p = i*G + gq), so every K/V row of the head
//     is fetched from HBM exactly once.
//   * Each unit's valid keys 0..len[b]-1 are split into n_sp contiguous,
//     32-key-aligned ranges, one CTA each (split-L / flash-decoding); n_sp is
//     chosen so the grid fills the GPU in one wave.
//   * Inside a CTA a producer warp streams its range with TMA tensor loads
//     (cp.async.bulk.tensor, 128-byte swizzle, 32-row boxes) into a ring of
//     128-key stages guarded by mbarriers; every stage holds K and V.
//   * Four consumer warps per 16*MT-row group each own one 32-key block of
//     every stage: S = Q K^T and O += P V on mma.sync m16n8k16 bf16 tensor
//     cores with fp32 accumulators; online softmax per warp in registers (P
//     never leaves registers), the causal mask only on the blocks that reach
//     past the prefix, and the O rescale only when a row maximum grows.
//   * End: the warps' (m, l, O) partials merge in shared memory. With one
//     split the CTA writes the output; otherwise every CTA publishes its
//     partial to the workspace, the unit's CTAs meet at an arrival counter
//     (cooperative launch: all CTAs are co-resident; the wait is bounded) and
//     each finalises a slice of the unit's rows. All merges run in a fixed
//     order, so results are deterministic.
//
// Masking: row i of scene b is the token at position L_b + i, L_b = len[b] - R,
// and sees keys 0 .. L_b + i. Keys past len[b] (stale cache rows, TMA
// out-of-bounds fill) are excluded by selection, and the V rows of the final
// partial block are zeroed in shared memory before the P V product, so stale
// NaN/Inf in the cache never reaches the output.
//
// Every wait is bounded; a wait that runs out sets SD_DEVERR_TIMEOUT and the
// CTA carries on without hanging.
#include "common.cuh"

#include <cuda.h>  // CUtensorMap and its enums (header only; no libcuda link)

#include <math.h>
#include <mutex>

SD_DEFINE_ERROR_ACCESSOR(sd_take_error_attention)

namespace {

constexpr int kBlk = 32;                   // keys per consumer warp per stage (one TMA box)
constexpr int kStageKeys = 4 * kBlk;       // keys per stage
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

// 16-byte asynchronous global -> shared copy; src_bytes = 0 zero-fills
__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src, int src_bytes) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(src_bytes)
               : "memory");
}

__device__ __forceinline__ void cp_async_wait_all() {
  asm volatile("cp.async.wait_all;" ::: "memory");
}

__device__ __forceinline__ void named_bar_sync(int id, int threads) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(threads) : "memory");
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
  static constexpr int kHalfStageBytes = kStageKeys * 128;
  static constexpr int kKVStageBytes = kHalves * kHalfStageBytes;
  static constexpr int kStageBytes = 2 * kKVStageBytes;
  static constexpr int kStages = (192 * 1024) / kStageBytes;
  static constexpr int kRingBytes = kStages * kStageBytes;
  static constexpr int kQHalfBytes = kRows * 128;
  static constexpr int kQBytes = kHalves * kQHalfBytes;
  static constexpr int kLd = D + 4;                       // padded fp32 row stride
  static constexpr int kWarpPartFloats = kRowsW * kLd + 2 * kRowsW;
  static constexpr int kWarpPartBytes = kConsumerWarps * kWarpPartFloats * 4;
  static constexpr int kPartFloats = kRows * kLd + 2 * kRows;  // one CTA's (O, m, l)
  static constexpr int kPartBytes = kPartFloats * 4;
  static constexpr int kBarBytes = 2 * kStages * 8;
  static constexpr int kSmemBytes = kRingBytes + kQBytes + kBarBytes + 16 + 1024;
  static_assert(kWarpPartBytes + kPartBytes <= kRingBytes, "merge areas must fit in the ring");
  static_assert(kSmemBytes <= 227 * 1024, "shared memory budget");
  static_assert(kPartFloats % 4 == 0, "float4 copies of the partial");
  static_assert((kRows + 256) * (D + 2) * 4 <= kRingBytes, "merge staging must fit in the ring");
};

struct AttnArgs {
  const __nv_bfloat16* q;
  __nv_bfloat16* out;
  const int32_t* len;
  float* part;    // [units][n_sp][kPartFloats] split partials (n_sp > 1)
  uint32_t* cnt;  // [units][2] arrival / departure counters (n_sp > 1)
  int R, Hq, Hkv, G, M, cap, n_sp;
  int block;         // block mask: every new row sees all R new rows
  float scale_log2;  // softmax scale * log2(e)
};

__device__ __forceinline__ uint32_t ld_acquire_gpu(const uint32_t* p) {
  uint32_t v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

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
  int* s_flag = reinterpret_cast<int*>(smem + C::kRingBytes + C::kQBytes + C::kBarBytes);
  auto full_bar = [&](int s) { return bars + 8u * s; };
  auto empty_bar = [&](int s) { return bars + 8u * (C::kStages + s); };
  auto k_stage = [&](int s) { return ring + s * C::kStageBytes; };
  auto v_stage = [&](int s) { return ring + s * C::kStageBytes + C::kKVStageBytes; };

  const int sp = blockIdx.x;  // split index within the unit
  const int n_sp = a.n_sp;
  const int kvh = blockIdx.y % a.Hkv;
  const int mblock = blockIdx.y / a.Hkv;
  const int b = blockIdx.z;
  const long long unit = (static_cast<long long>(b) * gridDim.y + blockIdx.y);
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
  if (!valid && sp == 0 && threadIdx.x == 0 && blockIdx.y == 0) sd_set_error(SD_DEVERR_LENGTH);
  const int nblk = valid ? (n_keys + kBlk - 1) / kBlk : 0;
  const int blk_begin = static_cast<int>((static_cast<long long>(sp) * nblk) / n_sp);
  const int blk_end = static_cast<int>((static_cast<long long>(sp + 1) * nblk) / n_sp);
  const int n_tiles = (blk_end - blk_begin + 3) / 4;

  float* part_smem = reinterpret_cast<float*>(smem + C::kWarpPartBytes);

  if (warp == C::kConsumerWarps) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      const int z = b * a.Hkv + kvh;
      asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tm_k)) : "memory");
      asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tm_v)) : "memory");
      for (int t = 0; t < n_tiles; ++t) {
        const int s = t % C::kStages;
        if (t >= C::kStages) mbar_wait(empty_bar(s), ((t / C::kStages) - 1) & 1);
        const int nb = min(4, blk_end - blk_begin - 4 * t);
        mbar_expect_tx(full_bar(s), static_cast<uint32_t>(nb * C::kHalves * 2 * kBlk * 128));
        for (int j = 0; j < nb; ++j) {
          const int y = (blk_begin + 4 * t + j) * kBlk;
#pragma unroll
          for (int h = 0; h < C::kHalves; ++h) {
            const uint32_t off = h * C::kHalfStageBytes + j * kBlk * 128;
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
    // packed query rows of this CTA -> shared memory (swizzled like the K
    // tiles), all 16-byte copies in flight at once; padding rows zero-fill
    for (int idx = tid; idx < C::kRows * (D / 8); idx += C::kConsumerThreads) {
      const int row = idx / (D / 8);
      const int chunk = idx % (D / 8);
      const int p = mblock * C::kRows + row;
      const bool live = valid && p < a.M;
      const int i = live ? p / a.G : 0, gq = live ? p % a.G : 0;
      const __nv_bfloat16* src =
          a.q + ((static_cast<long long>(b) * a.R + i) * a.Hq + kvh * a.G + gq) * D + chunk * 8;
      cp_async16(qs + (chunk >> 3) * C::kQHalfBytes + swz(row, chunk & 7), src, live ? 16 : 0);
    }
    cp_async_wait_all();
    named_bar_sync(1, C::kConsumerThreads);

    const int mg = warp >> 2;  // row group of this warp
    const int ks = warp & 3;   // 32-key block of every stage owned by this warp
    const int g8 = lane >> 2;
    const int t4 = lane & 3;
    const int L_prefix = n_keys - a.R;
    const float sl = a.scale_log2;

    // last visible key of each of this thread's rows
    int lim[MT][2];
#pragma unroll
    for (int mt = 0; mt < MT; ++mt)
#pragma unroll
      for (int hh = 0; hh < 2; ++hh) {
        const int p = mblock * C::kRows + mg * C::kRowsW + mt * 16 + g8 + 8 * hh;
        lim[mt][hh] = a.block ? n_keys - 1 : min(L_prefix + p / a.G, n_keys - 1);
      }

    float o[MT][D / 8][4];
    float m_run[MT][2], l_run[MT][2];  // m in raw score units
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
        const int key0 = blk * kBlk;
        const uint32_t kb = k_stage(s) + ks * kBlk * 128;  // this warp's 32 rows
        const uint32_t vb = v_stage(s) + ks * kBlk * 128;
        // ---- S = Q K^T over this warp's 32 keys (4 n8 tiles)
        float sc[MT][4][4];
#pragma unroll
        for (int mt = 0; mt < MT; ++mt)
#pragma unroll
          for (int nt = 0; nt < 4; ++nt)
#pragma unroll
            for (int c = 0; c < 4; ++c) sc[mt][nt][c] = 0.f;
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
          const int half = kk >> 2;
          const int chunk = (kk & 3) * 2;
          uint32_t kf[2][4];
#pragma unroll
          for (int np = 0; np < 2; ++np)
            ldsm_x4(kb + half * C::kHalfStageBytes + swz(np * 16 + b_row, chunk + b_chk), kf[np][0],
                    kf[np][1], kf[np][2], kf[np][3]);
#pragma unroll
          for (int mt = 0; mt < MT; ++mt) {
            uint32_t qa0, qa1, qa2, qa3;
            ldsm_x4(qs + half * C::kQHalfBytes +
                        swz(mg * C::kRowsW + mt * 16 + a_row, chunk + a_chk),
                    qa0, qa1, qa2, qa3);
#pragma unroll
            for (int np = 0; np < 2; ++np) {
              mma_bf16(sc[mt][2 * np], qa0, qa1, qa2, qa3, kf[np][0], kf[np][1]);
              mma_bf16(sc[mt][2 * np + 1], qa0, qa1, qa2, qa3, kf[np][2], kf[np][3]);
            }
          }
        }
        // ---- causal / length mask: only blocks reaching past the prefix
        if (key0 + kBlk - 1 > L_prefix) {
#pragma unroll
          for (int mt = 0; mt < MT; ++mt)
#pragma unroll
            for (int nt = 0; nt < 4; ++nt)
#pragma unroll
              for (int c = 0; c < 4; ++c) {
                const int key = key0 + nt * 8 + 2 * t4 + (c & 1);
                if (key > lim[mt][c >> 1]) sc[mt][nt][c] = -INFINITY;
              }
        }
        // ---- online softmax (row max over the block; lazy O rescale)
        float m_new[MT][2];
        bool grow = false;
#pragma unroll
        for (int mt = 0; mt < MT; ++mt)
#pragma unroll
          for (int hh = 0; hh < 2; ++hh) {
            float mx = -INFINITY;
#pragma unroll
            for (int nt = 0; nt < 4; ++nt)
              mx = fmaxf(mx, fmaxf(sc[mt][nt][2 * hh], sc[mt][nt][2 * hh + 1]));
            mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
            mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 2));
            m_new[mt][hh] = fmaxf(m_run[mt][hh], mx);
            grow |= (m_run[mt][hh] != -INFINITY) && (m_new[mt][hh] > m_run[mt][hh]);
          }
        if (__any_sync(0xffffffffu, grow)) {
#pragma unroll
          for (int mt = 0; mt < MT; ++mt)
#pragma unroll
            for (int hh = 0; hh < 2; ++hh) {
              const float corr = m_run[mt][hh] == -INFINITY
                                     ? 1.f
                                     : ex2((m_run[mt][hh] - m_new[mt][hh]) * sl);
              l_run[mt][hh] *= corr;
#pragma unroll
              for (int nd = 0; nd < D / 8; ++nd) {
                o[mt][nd][2 * hh] *= corr;
                o[mt][nd][2 * hh + 1] *= corr;
              }
            }
        }
        uint32_t pa[2][MT][4];  // [k16 step][m tile][a0..a3]
#pragma unroll
        for (int mt = 0; mt < MT; ++mt)
#pragma unroll
          for (int hh = 0; hh < 2; ++hh) {
            m_run[mt][hh] = m_new[mt][hh];
            const float mb = m_new[mt][hh] == -INFINITY ? 0.f : m_new[mt][hh] * sl;
            float rs = 0.f;
#pragma unroll
            for (int nt = 0; nt < 4; ++nt) {
              const uint32_t w = sd_pack_bf16x2(ex2(fmaf(sc[mt][nt][2 * hh], sl, -mb)),
                                                ex2(fmaf(sc[mt][nt][2 * hh + 1], sl, -mb)));
              rs += sd_bf16_lo(w) + sd_bf16_hi(w);  // normaliser of the bf16 weights used
              pa[nt >> 1][mt][(nt & 1) * 2 + hh] = w;
            }
            l_run[mt][hh] += rs;
          }
        // ---- the scene's last block: zero V rows past len (stale cache data)
        if (key0 + kBlk > n_keys) {
          const int first = n_keys - key0;
          const int n_chunks = (kBlk - first) * C::kHalves * 8;
          for (int cidx = lane; cidx < n_chunks; cidx += 32) {
            const int r = first + cidx / (C::kHalves * 8);
            const int rem = cidx % (C::kHalves * 8);
            const uint32_t addr = vb + (rem >> 3) * C::kHalfStageBytes + r * 128 + (rem & 7) * 16;
            asm volatile("st.shared.v4.u32 [%0], {%1,%1,%1,%1};" ::"r"(addr), "r"(0) : "memory");
          }
          __syncwarp();
        }
        // ---- O += P V (two k16 steps)
#pragma unroll
        for (int k2 = 0; k2 < 2; ++k2) {
#pragma unroll
          for (int dp = 0; dp < D / 16; ++dp) {
            const int chunk = dp * 2;  // d chunks 2dp, 2dp+1 (8 values each)
            uint32_t v0, v1, v2, v3;
            ldsm_x4_t(vb + (chunk >> 3) * C::kHalfStageBytes +
                          swz(k2 * 16 + a_row, (chunk & 7) + a_chk),
                      v0, v1, v2, v3);
#pragma unroll
            for (int mt = 0; mt < MT; ++mt) {
              mma_bf16(o[mt][2 * dp], pa[k2][mt][0], pa[k2][mt][1], pa[k2][mt][2], pa[k2][mt][3],
                       v0, v1);
              mma_bf16(o[mt][2 * dp + 1], pa[k2][mt][0], pa[k2][mt][1], pa[k2][mt][2],
                       pa[k2][mt][3], v2, v3);
            }
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
          wp[C::kRowsW * C::kLd + r] = m_run[mt][hh] == -INFINITY ? -INFINITY : m_run[mt][hh] * sl;
          wp[C::kRowsW * C::kLd + C::kRowsW + r] = l;
        }
      }
    }
    named_bar_sync(1, C::kConsumerThreads);
    // ---- merge the four key-slice warps of each row group (fixed order);
    //      m is kept in log2-scaled units from here on
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
      if (n_sp == 1) {
        // single split: this CTA owns the unit -> normalise and write out
        const int p = mblock * C::kRows + row;
        if (valid && p < a.M && lsum > 0.f) {
          const float inv = 1.f / lsum;
          const int i = p / a.G, gq = p % a.G;
          const long long off =
              ((static_cast<long long>(b) * a.R + i) * a.Hq + kvh * a.G + gq) * D + col;
          *reinterpret_cast<uint2*>(a.out + off) =
              make_uint2(sd_pack_bf16x2(acc.x * inv, acc.y * inv), sd_pack_bf16x2(acc.z * inv, acc.w * inv));
        }
      } else {
        *reinterpret_cast<float4*>(part_smem + row * C::kLd + col) = acc;
        if (col == 0) {
          part_smem[C::kRows * C::kLd + row] = mmax;
          part_smem[C::kRows * C::kLd + C::kRows + row] = lsum;
        }
      }
    }
    if (n_sp > 1) {
      named_bar_sync(1, C::kConsumerThreads);
      float4* dst = reinterpret_cast<float4*>(a.part + (unit * n_sp + sp) * C::kPartFloats);
      const float4* src = reinterpret_cast<const float4*>(part_smem);
      for (int i = tid; i < C::kPartFloats / 4; i += C::kConsumerThreads) __stcg(dst + i, src[i]);
    }
  }
  if (n_sp == 1) return;  // uniform across the grid

  // ---- cross-split merge: meet at the unit's arrival counter (release /
  //      acquire), then each CTA finalises a slice of the unit's rows from the
  //      partials of every split, staged in shared memory with all copies in
  //      flight at once
  __syncthreads();
  uint32_t* arrive = a.cnt + 2 * unit;
  uint32_t* depart = arrive + 1;
  if (threadIdx.x == 0) {
    asm volatile("red.release.gpu.global.add.u32 [%0], 1;" ::"l"(arrive) : "memory");
    int ok = 1;
    for (uint32_t it = 0; ld_acquire_gpu(arrive) < static_cast<uint32_t>(n_sp); ++it) {
      if (it >= kSpinLimit) {
        sd_set_error(SD_DEVERR_TIMEOUT);
        ok = 0;
        break;
      }
      __nanosleep(20);
    }
    *s_flag = ok;
  }
  __syncthreads();
  const int r0 = static_cast<int>((static_cast<long long>(sp) * C::kRows) / n_sp);
  const int r1 = static_cast<int>((static_cast<long long>(sp + 1) * C::kRows) / n_sp);
  const int nr = r1 - r0;
  if (*s_flag && nr > 0) {
    // stage: for every split c, rows [r0, r1) of O plus their m and l
    const float* base = a.part + unit * n_sp * C::kPartFloats;
    float* st = reinterpret_cast<float*>(smem);          // [n_sp][nr][D]
    float* st_ml = st + static_cast<size_t>(n_sp) * nr * D;  // [n_sp][2][nr]
    const int vec_per_split = nr * (D / 4);
    for (int idx = threadIdx.x; idx < n_sp * vec_per_split; idx += C::kThreads) {
      const int c = idx / vec_per_split;
      const int rem = idx % vec_per_split;
      const int row = r0 + rem / (D / 4);
      const int col = (rem % (D / 4)) * 4;
      cp_async16(smem_addr(st + (static_cast<size_t>(c) * nr + (row - r0)) * D + col),
                 base + c * C::kPartFloats + row * C::kLd + col, 16);
    }
    for (int idx = threadIdx.x; idx < n_sp * 2 * nr; idx += C::kThreads) {
      const int c = idx / (2 * nr);
      const int which = (idx / nr) & 1;
      const int row = r0 + idx % nr;
      st_ml[idx] = __ldcg(base + c * C::kPartFloats + C::kRows * C::kLd + which * C::kRows + row);
    }
    cp_async_wait_all();
    __syncthreads();
    for (int idx = threadIdx.x; idx < nr * (D / 4); idx += C::kThreads) {
      const int rr = idx / (D / 4);
      const int col = (idx % (D / 4)) * 4;
      const int p = mblock * C::kRows + r0 + rr;
      if (!valid || p >= a.M) continue;
      float mmax = -INFINITY;
      for (int c = 0; c < n_sp; ++c) mmax = fmaxf(mmax, st_ml[(c * 2 + 0) * nr + rr]);
      float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
      float lsum = 0.f;
      for (int c = 0; c < n_sp; ++c) {
        const float mc = st_ml[(c * 2 + 0) * nr + rr];
        const float f = mc == -INFINITY ? 0.f : ex2(mc - mmax);
        const float4 oc = *reinterpret_cast<const float4*>(st + (static_cast<size_t>(c) * nr + rr) * D + col);
        acc.x = fmaf(f, oc.x, acc.x);
        acc.y = fmaf(f, oc.y, acc.y);
        acc.z = fmaf(f, oc.z, acc.z);
        acc.w = fmaf(f, oc.w, acc.w);
        lsum = fmaf(f, st_ml[(c * 2 + 1) * nr + rr], lsum);
      }
      if (lsum > 0.f) {
        const float inv = 1.f / lsum;
        const int i = p / a.G, gq = p % a.G;
        const long long off =
            ((static_cast<long long>(b) * a.R + i) * a.Hq + kvh * a.G + gq) * D + col;
        *reinterpret_cast<uint2*>(a.out + off) =
            make_uint2(sd_pack_bf16x2(acc.x * inv, acc.y * inv), sd_pack_bf16x2(acc.z * inv, acc.w * inv));
      }
    }
  }
  __syncthreads();
  if (threadIdx.x == 0 && *s_flag) {
    // the last CTA to leave re-arms both counters for the next call
    if (atomicAdd(depart, 1u) == static_cast<uint32_t>(n_sp - 1)) {
      *arrive = 0;
      *depart = 0;
      __threadfence();
    }
  }
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

// [B*Hkv][cap][D] bf16 viewed as a 3-D tensor; boxes of 64 columns x 32 rows.
bool make_kv_map(CUtensorMap* map, void* base, int D, int cap, int planes) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[3] = {static_cast<cuuint64_t>(D), static_cast<cuuint64_t>(cap),
                        static_cast<cuuint64_t>(planes)};
  cuuint64_t strides[2] = {static_cast<cuuint64_t>(D) * 2,
                           static_cast<cuuint64_t>(cap) * static_cast<cuuint64_t>(D) * 2};
  cuuint32_t box[3] = {64, kBlk, 1};
  cuuint32_t estr[3] = {1, 1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, base, dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Launch plan of one call: splits per unit, workspace bytes.
struct Plan {
  int n_sp = 1;
  int n_mblocks = 1;
  int rows = 0;  // packed rows per CTA
  size_t ws_bytes = 0;
  int mt = 1, nmg = 1;
};

template <int D, int MT, int NMG>
struct Launcher {
  using C = Cfg<D, MT, NMG>;
  // per device: attributes set, co-resident CTAs per SM
  static int ctas_per_sm() {
    static int st[16] = {0};
    static std::mutex mu;
    int dev = 0;
    cudaGetDevice(&dev);
    if (dev < 0 || dev >= 16) return 0;
    std::lock_guard<std::mutex> lock(mu);
    if (!st[dev]) {
      auto kern = verify_attn_kernel<D, MT, NMG>;
      if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, C::kSmemBytes) !=
          cudaSuccess) {
        (void)cudaGetLastError();
        return 0;
      }
      int n = 0;
      if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, kern, C::kThreads, C::kSmemBytes) !=
          cudaSuccess) {
        (void)cudaGetLastError();
        n = 0;
      }
      st[dev] = n > 0 ? n : -1;
    }
    return st[dev] > 0 ? st[dev] : 0;
  }

  static bool plan(int B, int Hkv, int n_mblocks, int cap, Plan* p) {
    const int occ = ctas_per_sm();
    if (occ <= 0) return false;
    const long long units = static_cast<long long>(B) * Hkv * n_mblocks;
    const long long slots = static_cast<long long>(occ) * sd_num_sms();
    const long long nblk = (cap + kBlk - 1) / kBlk;
    long long n_sp = 1;
    if (units < slots) {
      n_sp = slots / units;
      if (n_sp > nblk) n_sp = nblk;
      // the merge stages n_sp x ceil(rows / n_sp) partial rows in the ring:
      // at most (rows + 256) x D floats
      if (n_sp > 256) n_sp = 256;
      if (n_sp < 1) n_sp = 1;
    }
    p->n_sp = static_cast<int>(n_sp);
    p->n_mblocks = n_mblocks;
    p->rows = C::kRows;
    p->mt = MT;
    p->nmg = NMG;
    p->ws_bytes = n_sp > 1 ? static_cast<size_t>(units) * n_sp * C::kPartBytes +
                                 static_cast<size_t>(units) * 8 + 256
                           : 0;
    return true;
  }

  static sd_status run(const CUtensorMap& tk, const CUtensorMap& tv, AttnArgs a, int B,
                       const Plan& p, void* ws, cudaStream_t stream) {
    a.n_sp = p.n_sp;
    const long long units = static_cast<long long>(B) * a.Hkv * p.n_mblocks;
    if (p.n_sp > 1) {
      a.part = static_cast<float*>(ws);
      a.cnt = reinterpret_cast<uint32_t*>(static_cast<char*>(ws) +
                                          static_cast<size_t>(units) * p.n_sp * C::kPartBytes);
    } else {
      a.part = nullptr;
      a.cnt = nullptr;
    }
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeCooperative;  // all splits of a unit co-resident
    attr[0].val.cooperative = 1;
    cfg.gridDim = dim3(p.n_sp, a.Hkv * p.n_mblocks, B);
    cfg.blockDim = dim3(C::kThreads, 1, 1);
    cfg.dynamicSmemBytes = C::kSmemBytes;
    cfg.stream = stream;
    cfg.attrs = attr;
    cfg.numAttrs = p.n_sp > 1 ? 1 : 0;
    if (cudaLaunchKernelEx(&cfg, verify_attn_kernel<D, MT, NMG>, tk, tv, a) != cudaSuccess) {
      (void)cudaGetLastError();
      return SD_ERR_CUDA;
    }
    return SD_OK;
  }
};

template <int D>
bool plan_rows(int M, int B, int Hkv, int cap, Plan* p) {
  if (M <= 16) return Launcher<D, 1, 1>::plan(B, Hkv, 1, cap, p);
  if (M <= 32) return Launcher<D, 2, 1>::plan(B, Hkv, 1, cap, p);
  return Launcher<D, 2, 2>::plan(B, Hkv, (M + 63) / 64, cap, p);
}

template <int D>
sd_status run_rows(const CUtensorMap& tk, const CUtensorMap& tv, const AttnArgs& a, int B,
                   const Plan& p, void* ws, cudaStream_t stream) {
  if (a.M <= 16) return Launcher<D, 1, 1>::run(tk, tv, a, B, p, ws, stream);
  if (a.M <= 32) return Launcher<D, 2, 1>::run(tk, tv, a, B, p, ws, stream);
  return Launcher<D, 2, 2>::run(tk, tv, a, B, p, ws, stream);
}

bool make_plan(int B, int R, int Hq, int Hkv, int D, int cap, Plan* p) {
  const int M = (Hq / Hkv) * R;
  return D == 64 ? plan_rows<64>(M, B, Hkv, cap, p) : plan_rows<128>(M, B, Hkv, cap, p);
}

}  // namespace

static sd_status check_shape(int B, int R, int Hq, int Hkv, int D, int cap) {
  if (B < 0 || R <= 0 || Hq <= 0 || Hkv <= 0 || cap <= 0) return SD_ERR_INVALID_ARG;
  if (Hq % Hkv) return SD_ERR_INVALID_ARG;
  if (D != 64 && D != 128) return SD_ERR_UNSUPPORTED;
  const int G = Hq / Hkv;
  if (static_cast<long long>(G) * R > 128) return SD_ERR_UNSUPPORTED;
  if (B > 65535 || Hkv * ((G * R + 63) / 64) > 65535) return SD_ERR_UNSUPPORTED;
  return SD_OK;
}

extern "C" size_t sd_verify_attention_workspace(int B, int R, int Hq, int Hkv, int D, int capacity) {
  if (check_shape(B, R, Hq, Hkv, D, capacity) != SD_OK || B == 0) return 0;
  if (sd_internal_tc_serves(B, R, Hq, Hkv, D, capacity)) return 0;
  Plan p;
  if (!make_plan(B, R, Hq, Hkv, D, capacity, &p)) return 0;
  return p.ws_bytes;
}

extern "C" sd_status sd_verify_attention(const void* q, const sd_kv_cache* cache, void* out,
                                         int R, int Hq, float scale, void* workspace,
                                         size_t ws_bytes, sd_stream_t stream) {
  return sd_verify_attention_ex(q, cache, out, R, Hq, scale, 0, workspace, ws_bytes, stream);
}

extern "C" sd_status sd_verify_attention_ex(const void* q, const sd_kv_cache* cache, void* out,
                                            int R, int Hq, float scale, int flags, void* workspace,
                                            size_t ws_bytes, sd_stream_t stream) {
  if (!cache) return SD_ERR_INVALID_ARG;
  if (flags & ~(SD_ATTN_BLOCK_MASK | SD_ATTN_PREFIX_EARLY)) return SD_ERR_INVALID_ARG;
  const int block = (flags & SD_ATTN_BLOCK_MASK) ? 1 : 0;
  const int B = cache->batch, Hkv = cache->n_kv_heads, cap = cache->capacity, D = cache->head_dim;
  const sd_status shape = check_shape(B, R, Hq, Hkv, D, cap);
  if (shape != SD_OK) return shape;
  if (B == 0) return SD_OK;
  if (!q || !out || !cache->k || !cache->v || !cache->len) return SD_ERR_INVALID_ARG;
  if (!sd_aligned16(q) || !sd_aligned16(out) || !sd_aligned16(cache->k) || !sd_aligned16(cache->v))
    return SD_ERR_INVALID_ARG;
  if (!(scale >= 0.f) || !isfinite(scale)) return SD_ERR_INVALID_ARG;
  const float sc = scale > 0.f ? scale : static_cast<float>(1.0 / sqrt(static_cast<double>(D)));
  const float scale_log2 = static_cast<float>(static_cast<double>(sc) * 1.4426950408889634);
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  {
    bool handled = false;
    const sd_status s = sd_internal_verify_attention_tc(q, cache, out, R, Hq, scale_log2, flags, st, &handled);
    if (handled) return s;
  }
  Plan p;
  if (!make_plan(B, R, Hq, Hkv, D, cap, &p)) return SD_ERR_CUDA;
  if (p.ws_bytes > 0 && (!workspace || ws_bytes < p.ws_bytes || !sd_aligned16(workspace)))
    return SD_ERR_WORKSPACE;
  CUtensorMap tk, tv;
  if (!make_kv_map(&tk, cache->k, D, cap, B * Hkv) || !make_kv_map(&tv, cache->v, D, cap, B * Hkv))
    return SD_ERR_CUDA;
  AttnArgs a;
  a.q = static_cast<const __nv_bfloat16*>(q);
  a.out = static_cast<__nv_bfloat16*>(out);
  a.len = cache->len;
  a.part = nullptr;
  a.cnt = nullptr;
  a.R = R;
  a.Hq = Hq;
  a.Hkv = Hkv;
  a.G = Hq / Hkv;
  a.M = a.G * R;
  a.cap = cap;
  a.n_sp = 1;
  a.block = block;
  a.scale_log2 = scale_log2;
  return D == 64 ? run_rows<64>(tk, tv, a, B, p, workspace, st)
                 : run_rows<128>(tk, tv, a, B, p, workspace, st);
}
