// K3 on the 5th-generation tensor cores (tcgen05 + TMEM): verify attention
// of the K + 1 new rows against the cached prefix (Eq. verify, Sec. 2.2),
// for head_dim 128 and up to 32 packed query rows per KV head.
//
// The packed query tile is small (G*R = 32 rows for 32 q / 8 KV heads and
// K = 7), so both products run TRANSPOSED, with the 128-wide dimension on the
// MMA's M side and no padding waste:
//     S^T[128 keys][32 rows] = K_tile[128 keys][128 d] . Q^T      (K-major A, B)
//     O^T[128 d][32 rows]   += V_tile^T[128 d][128 keys] . P^T     (MN-major A, K-major B)
// Both accumulators live in tensor memory (S double-buffered): 96 columns.
//
// Warp roles in a CTA (192 threads):
//   warp 0      TMA producer: 128-key stages of K and V (128B-swizzled boxes)
//   warp 1      allocates tensor memory; one lane issues every tcgen05.mma
//   warps 2..5  softmax: thread t owns key lane t of S^T (all 32 rows of it):
//               masks, row maxima by a warp butterfly + one shared exchange,
//               P = exp2(S - m) in bf16 into shared memory, lazy O rescale
//               (only when a row maximum grows) through tcgen05.ld/st.
// Work split: one thread-block cluster per (scene, KV head); its CTAs take
// contiguous 32-key-aligned ranges of the valid keys, and their (m, l, O)
// partials merge through distributed shared memory at the end. Every wait
// is bounded (SD_DEVERR_TIMEOUT instead of a hang).
#include "common.cuh"

#include <cuda.h>

#include <math.h>
#include <stdlib.h>
#include <mutex>

SD_DEFINE_ERROR_ACCESSOR(sd_take_error_attention_tc)

namespace {

constexpr int kD = 128;         // head dim
constexpr int kRows = 32;       // packed query rows per CTA (N of both MMAs)
constexpr int kStageKeys = 128; // M of S^T
constexpr int kStages = 3;
constexpr int kHalf = kStageKeys * 128;     // one 64-column half of a 128-key tile (16 KB)
constexpr int kKV = 2 * kHalf;              // K (or V) tile of a stage (32 KB)
constexpr int kStage = 2 * kKV;             // 64 KB
constexpr int kRing = kStages * kStage;     // 192 KB
constexpr int kQHalf = kRows * 128;         // 4 KB
constexpr int kQ = 2 * kQHalf;              // 8 KB
constexpr int kP = 2 * kQHalf;              // one P buffer [32 rows][128 keys] bf16, 8 KB
constexpr int kThreads = 192;
constexpr int kTmemCols = 128;              // S0 | S1 | O  (32 columns each)
constexpr uint32_t kSpinLimit = 1u << 20;

// shared memory layout (offsets from the 1024-aligned base)
constexpr int kOffQ = kRing;
constexpr int kOffP = kOffQ + kQ;
constexpr int kOffBar = kOffP + 2 * kP;
// barriers: full[3] empty[3] s_full[2] s_free[2] p_full[2] o_done[2] q_full recv append
constexpr int kNumBars = 3 + 3 + 2 + 2 + 2 + 2 + 1 + 1 + 1;
constexpr int kOffMisc = kOffBar + kNumBars * 8;
// misc: tmem slot (4), grow flag (4), red[4][32] + 2 x 4 warp flags, mnew[32], corr[32]
constexpr int kOffRed = kOffMisc + 16;
constexpr int kOffMnew = kOffRed + 4 * 32 * 4 + 32;
constexpr int kOffCorr = kOffMnew + 32 * 4;
constexpr int kSmemBytes = kOffCorr + 32 * 4 + 1024;
static_assert(kSmemBytes <= 227 * 1024, "shared memory budget");

// cluster merge buffers (in the ring, free once this CTA's last MMA is done):
// a partial row is [O(128) | m | l | 2 pad] fp32 = 528 bytes
constexpr int kRowF = kD + 4;
constexpr int kRowBytes = kRowF * 4;
constexpr int kSend = 0;                            // this CTA's 32 rows
constexpr int kRecv = 20 * 1024;                    // 32 slots received from the peers
static_assert(kRecv >= kRows * kRowBytes && kRecv + kRows * kRowBytes <= kRing, "merge buffers");

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
__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
__device__ __forceinline__ void named_bar_sync(int id, int threads) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(threads) : "memory");
}
__device__ __forceinline__ void cluster_arrive() {
  asm volatile("barrier.cluster.arrive.release.aligned;" ::: "memory");
}
__device__ __forceinline__ void cluster_wait() {
  asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory");
}
// shared::cta -> shared::cluster bulk copy, completing on the destination's mbarrier
__device__ __forceinline__ void bulk_copy_s2s(uint32_t dst_cluster, uint32_t src_cta, uint32_t bytes,
                                              uint32_t bar_cluster) {
  asm volatile(
      "cp.async.bulk.shared::cluster.shared::cta.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
          dst_cluster),
      "r"(src_cta), "r"(bytes), "r"(bar_cluster)
      : "memory");
}
__device__ __forceinline__ uint32_t cluster_map(uint32_t addr, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(addr), "r"(rank));
  return r;
}
// ---------------------------------------------------------------- tcgen05
// Shared-memory matrix descriptor, 128-byte swizzle (sm_100 family format):
// start address, leading / stride byte offsets (>> 4), version 1, layout 2.
__device__ __forceinline__ uint64_t umma_desc(uint32_t addr, uint32_t lbo, uint32_t sbo) {
  return static_cast<uint64_t>((addr >> 4) & 0x3FFF) |
         (static_cast<uint64_t>((lbo >> 4) & 0x3FFF) << 16) |
         (static_cast<uint64_t>((sbo >> 4) & 0x3FFF) << 32) | (1ull << 46) | (2ull << 61);
}
// Instruction descriptor, kind::f16: fp32 accumulate, bf16 A and B.
constexpr uint32_t umma_idesc(int M, int N, int a_mn_major, int b_mn_major) {
  return (1u << 4) | (1u << 7) | (1u << 10) | (static_cast<uint32_t>(a_mn_major) << 15) |
         (static_cast<uint32_t>(b_mn_major) << 16) | (static_cast<uint32_t>(N >> 3) << 17) |
         (static_cast<uint32_t>(M >> 4) << 24);
}
constexpr uint32_t kIdescS = umma_idesc(128, kRows, 0, 0);
constexpr uint32_t kIdescO = umma_idesc(128, kRows, 1, 0);

__device__ __forceinline__ void umma(uint32_t d_tmem, uint64_t a, uint64_t b, uint32_t idesc,
                                     int accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(a), "l"(b), "r"(idesc), "r"(accumulate)
      : "memory");
}
__device__ __forceinline__ void umma_commit(uint32_t bar) {
  asm volatile(
      "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
      : "memory");
}
__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

#define SD_R32(r)                                                                              \
  "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),          \
      "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),  \
      "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]),            \
      "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]),            \
      "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
#define SD_W32(r)                                                                              \
  "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]),      \
      "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]),        \
      "r"(r[15]), "r"(r[16]), "r"(r[17]), "r"(r[18]), "r"(r[19]), "r"(r[20]), "r"(r[21]),      \
      "r"(r[22]), "r"(r[23]), "r"(r[24]), "r"(r[25]), "r"(r[26]), "r"(r[27]), "r"(r[28]),      \
      "r"(r[29]), "r"(r[30]), "r"(r[31])

// 32 consecutive fp32 columns of this warp's 32 TMEM lanes -> 32 registers
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,"
      "%14,%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
      : SD_R32(r)
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_st32(uint32_t taddr, const uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,"
      "%13,%14,%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};" ::"r"(
          taddr),
      SD_W32(r)
      : "memory");
  asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}

struct TcArgs {
  const __nv_bfloat16* q;   // rotated q rows (standalone attention)
  __nv_bfloat16* out;
  int32_t* len;
  // fused verify layer only
  __nv_bfloat16* qw;        // raw q rows, rotated in place
  __nv_bfloat16* k_new;     // raw new key rows [B][R][Hkv][D], rotated in place
  const __nv_bfloat16* v_new;
  __nv_bfloat16* kc;        // cache K / V [B][Hkv][cap][D] (append target)
  __nv_bfloat16* vc;
  const int32_t* pos;       // [B][R][3]
  uint32_t* ticket;         // [B] per-scene CTA tickets (zeroed, re-armed)
  int early;                // the prefix may be streamed before the dependency wait
  int R, Hq, Hkv, G, M, cap, n_mblocks;
  float scale_log2;
};

__device__ __forceinline__ void griddep_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void griddep_launch() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// ------------------------------------------------------------------ kernel
// kFused = false: attention over a cache that already holds the R new rows,
// with the rotated query rows loaded by TMA.
// kFused = true: the whole verify layer -- M-RoPE of the raw query and key
// rows, the KV append and the attention -- with len[b] the prefix length.
// Prefix tiles are independent of the kernel that precedes this one in the
// stream (for every layer but the first of a step), so when a.early is set
// they stream before the programmatic-dependency wait.
template <bool kFused>
__global__ void __launch_bounds__(kThreads, 1)
    verify_attn_tc_kernel(const __grid_constant__ CUtensorMap tm_k128,
                          const __grid_constant__ CUtensorMap tm_v128,
                          const __grid_constant__ CUtensorMap tm_k32,
                          const __grid_constant__ CUtensorMap tm_v32,
                          const __grid_constant__ CUtensorMap tm_q, const TcArgs a,
                          const RopeTable tab) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  const uint32_t base = smem_addr(smem);
  const uint32_t qs = base + kOffQ;
  auto bar = [&](int i) { return base + kOffBar + 8u * i; };
  // barrier indices
  auto FULL = [&](int s) { return bar(s); };
  auto EMPTY = [&](int s) { return bar(3 + s); };
  auto SFULL = [&](int b) { return bar(6 + b); };
  auto SFREE = [&](int b) { return bar(8 + b); };
  auto PFULL = [&](int b) { return bar(10 + b); };
  auto ODONE = [&](int b) { return bar(12 + b); };
  const uint32_t QFULL = bar(14);
  const uint32_t RECV = bar(15);  // the cluster merge's incoming partial rows
  const uint32_t APPEND = bar(16);  // fused: the new K/V rows are in the cache
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + kOffMisc);
  int* grow_flag = reinterpret_cast<int*>(smem + kOffMisc + 4);
  float* red = reinterpret_cast<float*>(smem + kOffRed);    // [4][32]
  float* s_mnew = reinterpret_cast<float*>(smem + kOffMnew);
  float* s_corr = reinterpret_cast<float*>(smem + kOffCorr);

  const int rank = blockIdx.x;
  const int csize = gridDim.x;
  const int kvh = blockIdx.y % a.Hkv;
  const int mblock = blockIdx.y / a.Hkv;
  const int b = blockIdx.z;
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(FULL(s), 1);
      mbar_init(EMPTY(s), 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(SFULL(i), 1);
      mbar_init(SFREE(i), 4);
      mbar_init(PFULL(i), 4);
      mbar_init(ODONE(i), 1);
    }
    mbar_init(QFULL, kFused ? 128 : 129);  // (producer's expect_tx +) 128 softmax threads
    mbar_init(RECV, 1);
    mbar_init(APPEND, 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_addr(tmem_slot)),
                 "r"(kTmemCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const uint32_t tmem_s = tmem;          // S buffer b at column 32 * b
  const uint32_t tmem_o = tmem + 64;     // O^T

  if (kFused && !a.early) griddep_wait();  // len and the prefix may come from the previous kernel
  int n_keys, L_pre;
  bool valid;
  if (kFused) {
    L_pre = a.len[b];
    n_keys = L_pre + a.R;
    valid = L_pre >= 0 && n_keys <= a.cap;
    if (!valid && rank == 0 && threadIdx.x == 0 && blockIdx.y == 0)
      sd_set_error(L_pre < 0 ? SD_DEVERR_LENGTH : SD_DEVERR_KV_OVERFLOW);
  } else {
    n_keys = a.len[b];
    valid = n_keys >= a.R && n_keys <= a.cap;
    L_pre = n_keys - a.R;
    if (!valid && rank == 0 && threadIdx.x == 0 && blockIdx.y == 0) sd_set_error(SD_DEVERR_LENGTH);
  }
  const int nblk = valid ? (n_keys + 31) / 32 : 0;
  int blk_begin, blk_end;
  if (kFused) {
    // blocks wholly inside the prefix split evenly; the last CTA also takes
    // the block(s) holding the new rows, which it appends itself
    const int blk_new0 = valid ? L_pre / 32 : 0;
    blk_begin = static_cast<int>((static_cast<long long>(rank) * blk_new0) / csize);
    blk_end = rank == csize - 1 ? nblk
                                : static_cast<int>((static_cast<long long>(rank + 1) * blk_new0) / csize);
  } else {
    blk_begin = static_cast<int>((static_cast<long long>(rank) * nblk) / csize);
    blk_end = static_cast<int>((static_cast<long long>(rank + 1) * nblk) / csize);
  }
  const int key_begin = blk_begin * 32;
  const int key_end = min(blk_end * 32, n_keys);
  const int n_tiles = (blk_end - blk_begin + 3) / 4;
  const bool owns_new = kFused && valid && rank == csize - 1;
  const int t_new = owns_new ? (L_pre / 32 - blk_begin) / 4 : n_tiles;  // first tile with new rows

  if (warp == 0) {
    // -------------------------------------------------------------- producer
    if (lane == 0 && n_tiles > 0) {
      if (!kFused) {
        // the packed query tile first: box (64 d, G heads, R rows) lands as
        // rows p = i * G + g of 128 bytes, the B operand's K-major layout
        mbar_expect_tx(QFULL, static_cast<uint32_t>(2 * a.M * 128));
        for (int h = 0; h < 2; ++h)
          tma_load_3d(qs + h * kQHalf, &tm_q, QFULL, h * 64, kvh * a.G, b * a.R);
      }
      asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tm_k128)) : "memory");
      asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tm_v128)) : "memory");
      const int z = b * a.Hkv + kvh;
      for (int t = 0; t < n_tiles; ++t) {
        const int s = t % kStages;
        if (t >= kStages) mbar_wait(EMPTY(s), ((t / kStages) - 1) & 1);
        if (kFused && t == t_new) mbar_wait(APPEND, 0);  // the new rows are in the cache
        const int nb = min(4, blk_end - blk_begin - 4 * t);
        const int y0 = key_begin + t * kStageKeys;
        const uint32_t kst = base + s * kStage, vst = kst + kKV;
        mbar_expect_tx(FULL(s), static_cast<uint32_t>(nb * 32 * 128 * 2 * 2));
        if (nb == 4) {
          for (int h = 0; h < 2; ++h) {
            tma_load_3d(kst + h * kHalf, &tm_k128, FULL(s), h * 64, y0, z);
            tma_load_3d(vst + h * kHalf, &tm_v128, FULL(s), h * 64, y0, z);
          }
        } else {
          for (int j = 0; j < nb; ++j)
            for (int h = 0; h < 2; ++h) {
              tma_load_3d(kst + h * kHalf + j * 4096, &tm_k32, FULL(s), h * 64, y0 + 32 * j, z);
              tma_load_3d(vst + h * kHalf + j * 4096, &tm_v32, FULL(s), h * 64, y0 + 32 * j, z);
            }
        }
      }
    }
    __syncwarp();
    cluster_arrive();  // the cluster's rings are free (see the softmax branch)
    cluster_wait();
  } else if (warp == 1) {
    // -------------------------------------------------------------- MMA issue
    if (lane == 0 && n_tiles > 0) {
      mbar_wait(QFULL, 0);
      auto issue_pv = [&](int u) {
        const int bb = u & 1, s = u % kStages;
        mbar_wait(PFULL(bb), (u >> 1) & 1);
        tc_fence_after();
        const uint32_t vst = base + s * kStage + kKV;
        const uint32_t pb = base + kOffP + bb * kP;
#pragma unroll
        for (int kk = 0; kk < 8; ++kk) {
          const uint64_t ad = umma_desc(vst + kk * 2048, kHalf, 1024);      // V^T: MN-major
          const uint64_t bd = umma_desc(pb + (kk >> 2) * kQHalf + (kk & 3) * 32, 16, 1024);
          umma(tmem_o, ad, bd, kIdescO, (u > 0 || kk > 0) ? 1 : 0);
        }
        umma_commit(ODONE(bb));
        umma_commit(EMPTY(s));
      };
      for (int t = 0; t < n_tiles; ++t) {
        const int s = t % kStages, bb = t & 1;
        mbar_wait(FULL(s), (t / kStages) & 1);
        if (t >= 2) mbar_wait(SFREE(bb), ((t >> 1) - 1) & 1);
        tc_fence_after();
        const uint32_t kst = base + s * kStage;
#pragma unroll
        for (int kk = 0; kk < 8; ++kk) {
          const uint64_t ad = umma_desc(kst + (kk >> 2) * kHalf + (kk & 3) * 32, 16, 1024);
          const uint64_t bd = umma_desc(qs + (kk >> 2) * kQHalf + (kk & 3) * 32, 16, 1024);
          umma(tmem_s + 32 * bb, ad, bd, kIdescS, kk > 0 ? 1 : 0);
        }
        umma_commit(SFULL(bb));
        if (t >= 1) issue_pv(t - 1);
      }
      issue_pv(n_tiles - 1);
    }
    __syncwarp();
    cluster_arrive();
    cluster_wait();
  } else {
    // -------------------------------------------------------------- softmax
    const int st = threadIdx.x - 64;       // 0..127
    const int quarter = warp & 3;          // TMEM lane quarter of this warp
    const int kl = quarter * 32 + lane;    // key lane of S^T / d lane of O^T
    const uint32_t lane_off = static_cast<uint32_t>(quarter * 32) << 16;
    if (!kFused) {
      // query rows past M stay zero (the TMA box covers rows 0..M-1 only)
      for (int idx = st; idx < (kRows - a.M) * 16; idx += 128) {
        const int row = a.M + idx / 16, c = idx % 16;
        asm volatile("st.shared.v4.u32 [%0], {%1,%1,%1,%1};" ::"r"(qs + (c >> 3) * kQHalf + row * 128 + (c & 7) * 16),
                     "r"(0)
                     : "memory");
      }
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
      mbar_arrive(QFULL);
    } else {
      // the raw rows come from earlier kernels; once they are visible every
      // older kernel has finished, so the next layer may launch
      griddep_wait();
      if (st == 0) griddep_launch();
      // M-RoPE of the packed query rows, straight into the swizzled tile
      for (int idx = st; idx < kRows * 16; idx += 128) {
        const int row = idx / 16, c = idx % 16;
        const int p = mblock * kRows + row;
        uint32_t w[4] = {0u, 0u, 0u, 0u};
        if (valid && p < a.M) {
          const int i = p / a.G, gq = p % a.G;
          const uint4 v = *reinterpret_cast<const uint4*>(
              a.qw + ((static_cast<long long>(b) * a.R + i) * a.Hq + kvh * a.G + gq) * kD + c * 8);
          w[0] = v.x; w[1] = v.y; w[2] = v.z; w[3] = v.w;
          const int32_t* pp = a.pos + (static_cast<long long>(b) * a.R + i) * 3;
          const int p3[3] = {pp[0], pp[1], pp[2]};
          sd_rope_rotate8(w, c, p3, tab);
        }
        asm volatile("st.shared.v4.u32 [%0], {%1,%2,%3,%4};" ::"r"(
                         qs + (c >> 3) * kQHalf + row * 128 + (((c & 7) ^ (row & 7)) << 4)),
                     "r"(w[0]), "r"(w[1]), "r"(w[2]), "r"(w[3])
                     : "memory");
      }
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
      mbar_arrive(QFULL);
      if (owns_new) {
        // M-RoPE of this head's new key rows and the append of K and V; the
        // rotated keys also go back to k_new, like the standalone rotation
        for (int idx = st; idx < a.R * 16; idx += 128) {
          const int i = idx / 16, c = idx % 16;
          const long long src = ((static_cast<long long>(b) * a.R + i) * a.Hkv + kvh) * kD + c * 8;
          const long long dst = ((static_cast<long long>(b) * a.Hkv + kvh) * a.cap + L_pre + i) * kD + c * 8;
          const uint4 kv = *reinterpret_cast<const uint4*>(a.k_new + src);
          uint32_t w[4] = {kv.x, kv.y, kv.z, kv.w};
          const int32_t* pp = a.pos + (static_cast<long long>(b) * a.R + i) * 3;
          const int p3[3] = {pp[0], pp[1], pp[2]};
          sd_rope_rotate8(w, c, p3, tab);
          const uint4 kr = make_uint4(w[0], w[1], w[2], w[3]);
          *reinterpret_cast<uint4*>(a.kc + dst) = kr;
          *reinterpret_cast<uint4*>(a.k_new + src) = kr;
          *reinterpret_cast<uint4*>(a.vc + dst) = *reinterpret_cast<const uint4*>(a.v_new + src);
        }
        asm volatile("fence.proxy.async.global;" ::: "memory");  // visible to the TMA loads
        named_bar_sync(2, 128);
        if (st == 0) mbar_arrive(APPEND);
      }
    }

    const int L_prefix = n_keys - a.R;
    const float sl = a.scale_log2;
    // Reference maximum per query row (log2 units), identical in every
    // softmax thread. It is set exactly on the first tile; later tiles keep it
    // unless some score exceeds it by more than kSlack, so exp2(s - ref) <= 2^8
    // stays exact in bf16 / fp32 and the common tile needs no cross-warp work.
    constexpr float kSlack = 8.f;
    float mref[32];
    float lp[32];  // per-row partial sums of this thread's key lane
#pragma unroll
    for (int j = 0; j < 32; ++j) {
      mref[j] = -INFINITY;
      lp[j] = 0.f;
    }

    for (int t = 0; t < n_tiles; ++t) {
      const int bb = t & 1, s = t % kStages;
      const int key0 = key_begin + t * kStageKeys;
      const int key = key0 + kl;
      mbar_wait(SFULL(bb), (t >> 1) & 1);
      tc_fence_after();
      uint32_t r[32];
      tmem_ld32(tmem_s + 32 * bb + lane_off, r);
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(SFREE(bb));
      // scale, range / causal mask
      float sv[32];
      const bool key_ok = key < key_end;
      const bool tail = key0 + kStageKeys - 1 > L_prefix;
      bool over = false;
#pragma unroll
      for (int j = 0; j < 32; ++j) {
        float x = key_ok ? __uint_as_float(r[j]) * sl : -INFINITY;
        if (tail) {
          const int p = mblock * kRows + j;
          const int lim = min(L_prefix + p / a.G, n_keys - 1);
          if (key > lim) x = -INFINITY;
        }
        sv[j] = x;
        over |= x > mref[j] + kSlack;
      }
      // do the four warps agree to keep the references? (one barrier)
      const bool warp_over = __any_sync(0xffffffffu, over);
      // flags are double-buffered by tile parity: a warp that runs ahead to
      // the next tile cannot overwrite a slot another warp has yet to read
      volatile int* flags = reinterpret_cast<volatile int*>(red) + 128 + 4 * bb;
      if (lane == 0) flags[quarter] = warp_over ? 1 : 0;
      named_bar_sync(2, 128);
      const bool slow = (flags[0] | flags[1] | flags[2] | flags[3]) != 0;
      bool rescale = false;
      if (slow) {
        // exact row maxima of this tile: warp butterfly (lane ends with row
        // `lane`), then across the four warps through shared memory
        float v[32];
#pragma unroll
        for (int j = 0; j < 32; ++j) v[j] = sv[j];
#pragma unroll
        for (int w = 16; w >= 1; w >>= 1) {
          const bool upper = (lane & w) != 0;
#pragma unroll
          for (int i = 0; i < w; ++i) {
            const float send = upper ? v[i] : v[i + w];
            const float keep = upper ? v[i + w] : v[i];
            v[i] = fmaxf(keep, __shfl_xor_sync(0xffffffffu, send, w));
          }
        }
        red[quarter * 32 + lane] = v[0];
        named_bar_sync(2, 128);
        if (quarter == 0) {
          const float smax = fmaxf(fmaxf(red[lane], red[32 + lane]), fmaxf(red[64 + lane], red[96 + lane]));
          const float old = s_mnew[lane];
          const float nw = t == 0 ? smax : fmaxf(old, smax);
          s_corr[lane] = (t == 0 || old == -INFINITY || nw == old) ? 1.f : ex2(old - nw);
          s_mnew[lane] = nw;
          const bool grow = t > 0 && old != -INFINITY && nw > old;
          const bool any_grow = __any_sync(0xffffffffu, grow);
          if (lane == 0) *grow_flag = any_grow ? 1 : 0;
        }
        named_bar_sync(2, 128);
        rescale = *grow_flag != 0;
#pragma unroll
        for (int j = 0; j < 32; ++j) mref[j] = s_mnew[j];
        if (rescale) {
#pragma unroll
          for (int j = 0; j < 32; ++j) lp[j] *= s_corr[j];
        }
      }
      // P = exp2(S - ref) in bf16; l partials from the same rounded weights
      uint16_t pb[32];
#pragma unroll
      for (int j = 0; j < 32; ++j) {
        const float mb = mref[j] == -INFINITY ? 0.f : mref[j];
        const __nv_bfloat16 h = __float2bfloat16_rn(ex2(sv[j] - mb));
        pb[j] = *reinterpret_cast<const uint16_t*>(&h);
        lp[j] += __bfloat162float(h);
      }
      // P buffer bb is free once PV of tile t-2 is done
      if (t >= 2) mbar_wait(ODONE(bb), ((t >> 1) - 1) & 1);
      if (rescale) {
        // O^T holds PV of tiles < t at the old references: wait for PV t-1,
        // then scale column j (query row j) of this thread's d lane
        mbar_wait(ODONE((t - 1) & 1), ((t - 1) >> 1) & 1);
        tc_fence_after();
        uint32_t o[32];
        tmem_ld32(tmem_o + lane_off, o);
#pragma unroll
        for (int j = 0; j < 32; ++j) o[j] = __float_as_uint(__uint_as_float(o[j]) * s_corr[j]);
        tmem_st32(tmem_o + lane_off, o);
      }
      const uint32_t pbuf = base + kOffP + bb * kP + (kl >> 6) * kQHalf;
      const int kc = (kl & 63) >> 3, kw = (kl & 7) * 2;
#pragma unroll
      for (int j = 0; j < 32; ++j) {
        const uint32_t addr = pbuf + j * 128 + ((kc ^ (j & 7)) << 4) + kw;
        asm volatile("st.shared.u16 [%0], %1;" ::"r"(addr), "h"(pb[j]) : "memory");
      }
      if (!key_ok) {
        // stale or foreign key row: zero its V row so 0 * NaN cannot reach O
        const uint32_t vrow = base + s * kStage + kKV + kl * 128;
#pragma unroll
        for (int h = 0; h < 2; ++h)
#pragma unroll
          for (int c = 0; c < 8; ++c)
            asm volatile("st.shared.v4.u32 [%0], {%1,%1,%1,%1};" ::"r"(vrow + h * kHalf + c * 16),
                         "r"(0)
                         : "memory");
      }
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(PFULL(bb));
    }

    // ---- CTA partial: O^T (tensor memory) of this thread's d lane, and the
    //      per-row m (reference) and l (sum over all 128 key lanes)
    float o_f[32];
    if (n_tiles > 0) {
      mbar_wait(ODONE((n_tiles - 1) & 1), ((n_tiles - 1) >> 1) & 1);
      tc_fence_after();
      uint32_t o[32];
      tmem_ld32(tmem_o + lane_off, o);
#pragma unroll
      for (int j = 0; j < 32; ++j) o_f[j] = __uint_as_float(o[j]);
    } else {
#pragma unroll
      for (int j = 0; j < 32; ++j) o_f[j] = 0.f;
    }
    // every MMA of this CTA is done: its ring may now receive peers' partials
    cluster_arrive();
#pragma unroll
    for (int w = 16; w >= 1; w >>= 1) {
      const bool upper = (lane & w) != 0;
#pragma unroll
      for (int i = 0; i < w; ++i) {
        const float send = upper ? lp[i] : lp[i + w];
        const float keep = upper ? lp[i + w] : lp[i];
        lp[i] = keep + __shfl_xor_sync(0xffffffffu, send, w);
      }
    }
    named_bar_sync(2, 128);
    red[quarter * 32 + lane] = lp[0];
    named_bar_sync(2, 128);
    const float l_row = (red[lane] + red[32 + lane]) + (red[64 + lane] + red[96 + lane]);
    const float m_row = n_tiles > 0 ? s_mnew[lane] : -INFINITY;
    // stage the partial row-major: row j = [O(128) | m | l | pad], 528 bytes
    float* send = reinterpret_cast<float*>(smem + kSend);
#pragma unroll
    for (int j = 0; j < 32; ++j) send[j * kRowF + kl] = o_f[j];
    if (quarter == 0) {
      send[lane * kRowF + kD] = m_row;
      send[lane * kRowF + kD + 1] = l_row;
    }
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    named_bar_sync(2, 128);
    const int rpc = kRows / csize;
    if (st == 0) mbar_expect_tx(RECV, static_cast<uint32_t>(csize * rpc * kRowBytes));
    cluster_wait();  // every peer's ring is free to receive
    if (st == 0) {
      // rows [c * rpc, (c + 1) * rpc) go to rank c, into its slots [rank * rpc, ...)
      for (int c = 0; c < csize; ++c)
        bulk_copy_s2s(cluster_map(base + kRecv + rank * rpc * kRowBytes, c),
                      base + kSend + c * rpc * kRowBytes, static_cast<uint32_t>(rpc * kRowBytes),
                      cluster_map(RECV, c));
      asm volatile("cp.async.bulk.commit_group;" ::: "memory");
      asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory");
    }
    // ---- local merge of the rows this CTA owns; slot c * rpc + rr came from rank c
    mbar_wait(RECV, 0);
    const float* recv = reinterpret_cast<const float*>(smem + kRecv);
    for (int rr = 0; rr < rpc; ++rr) {
      const int row = rank * rpc + rr;
      const int p = mblock * kRows + row;
      float mmax = -INFINITY;
      for (int c = 0; c < csize; ++c) mmax = fmaxf(mmax, recv[(c * rpc + rr) * kRowF + kD]);
      float acc = 0.f, lsum = 0.f;
      for (int c = 0; c < csize; ++c) {
        const float* slot = recv + (c * rpc + rr) * kRowF;
        const float mc = slot[kD];
        const float f = mc == -INFINITY ? 0.f : ex2(mc - mmax);
        acc = fmaf(f, slot[kl], acc);
        lsum = fmaf(f, slot[kD + 1], lsum);
      }
      if (valid && p < a.M && lsum > 0.f) {
        const int i = p / a.G, gq = p % a.G;
        a.out[((static_cast<long long>(b) * a.R + i) * a.Hq + kvh * a.G + gq) * kD + kl] =
            __float2bfloat16_rn(acc / lsum);
      }
    }
  }
  if (kFused && rank == 0 && warp >= 2) {
    // every CTA of the cluster read the raw query rows before its main loop
    // (the cluster barrier above is behind all of them): store the rotated rows
    for (int idx = threadIdx.x - 64; idx < a.M * 16 && valid; idx += 128) {
      const int row = idx / 16, c = idx % 16;
      const int p = mblock * kRows + row;
      if (p >= a.M) continue;
      const int i = p / a.G, gq = p % a.G;
      const uint4 v = *reinterpret_cast<const uint4*>(smem + kOffQ + (c >> 3) * kQHalf + row * 128 +
                                                      (((c & 7) ^ (row & 7)) << 4));
      *reinterpret_cast<uint4*>(a.qw + ((static_cast<long long>(b) * a.R + i) * a.Hq + kvh * a.G + gq) * kD +
                                c * 8) = v;
    }
  }
  tc_fence_before();
  __syncthreads();  // every tensor-memory read is done
  if (kFused && threadIdx.x == 0) {
    // the last CTA of the scene to finish advances its length: every CTA of
    // the scene read len[b] before it got here
    const uint32_t total = gridDim.x * gridDim.y;
    if (atomicAdd(&a.ticket[b], 1u) == total - 1) {
      if (valid) a.len[b] = L_pre + a.R;
      a.ticket[b] = 0;
    }
  }
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem),
                 "r"(kTmemCols)
                 : "memory");
  }
}

// ------------------------------------------------------------------ host
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

// q [B][R][Hq][D] as (D, Hq, B*R); box (64, G, R): one KV group's packed rows
bool make_q_map(CUtensorMap* map, const void* q, int B, int R, int Hq, int G) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[3] = {static_cast<cuuint64_t>(kD), static_cast<cuuint64_t>(Hq),
                        static_cast<cuuint64_t>(B) * R};
  cuuint64_t strides[2] = {static_cast<cuuint64_t>(kD) * 2, static_cast<cuuint64_t>(Hq) * kD * 2};
  cuuint32_t box[3] = {64, static_cast<cuuint32_t>(G), static_cast<cuuint32_t>(R)};
  cuuint32_t estr[3] = {1, 1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(q), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool make_map(CUtensorMap* map, void* base, int cap, int planes, int box_rows) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[3] = {static_cast<cuuint64_t>(kD), static_cast<cuuint64_t>(cap),
                        static_cast<cuuint64_t>(planes)};
  cuuint64_t strides[2] = {static_cast<cuuint64_t>(kD) * 2,
                           static_cast<cuuint64_t>(cap) * static_cast<cuuint64_t>(kD) * 2};
  cuuint32_t box[3] = {64, static_cast<cuuint32_t>(box_rows), 1};
  cuuint32_t estr[3] = {1, 1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, base, dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

constexpr int kClusterSizes[5] = {1, 2, 4, 8, 16};

struct DevState {
  bool ready = false;
  bool ok = false;
  int active[5] = {0, 0, 0, 0, 0};
};

DevState* state() {
  static DevState st[16];
  static std::mutex mu;
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev < 0 || dev >= 16) return nullptr;
  std::lock_guard<std::mutex> lock(mu);
  DevState& s = st[dev];
  if (!s.ready) {
    s.ready = true;
    auto kern = verify_attn_tc_kernel<false>;
    auto kern_f = verify_attn_tc_kernel<true>;
    if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes) !=
            cudaSuccess ||
        cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) !=
            cudaSuccess ||
        cudaFuncSetAttribute(kern_f, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes) !=
            cudaSuccess ||
        cudaFuncSetAttribute(kern_f, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) !=
            cudaSuccess) {
      (void)cudaGetLastError();
      return &s;
    }
    for (int i = 0; i < 5; ++i) {
      cudaLaunchConfig_t cfg = {};
      cudaLaunchAttribute attr[1];
      attr[0].id = cudaLaunchAttributeClusterDimension;
      attr[0].val.clusterDim.x = kClusterSizes[i];
      attr[0].val.clusterDim.y = 1;
      attr[0].val.clusterDim.z = 1;
      cfg.gridDim = dim3(kClusterSizes[i], 1, 1);
      cfg.blockDim = dim3(kThreads, 1, 1);
      cfg.dynamicSmemBytes = kSmemBytes;
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
    s.ok = true;
  }
  return &s;
}

// Cluster size: minimise waves x (32-key blocks per CTA + a fixed per-CTA cost)
int pick_cluster(const DevState& s, long long units, int cap) {
  const long long nblk = (cap + 31) / 32;
  long long best_cost = -1;
  int best = 0;
  for (int i = 0; i < 5; ++i) {
    const int cs = kClusterSizes[i];
    if (s.active[i] <= 0) continue;
    if (cs > 1 && nblk < 2LL * cs) continue;
    const long long waves = (units + s.active[i] - 1) / s.active[i];
    const long long cost = waves * ((nblk + cs - 1) / cs + 6);
    if (best_cost < 0 || cost < best_cost) {
      best_cost = cost;
      best = cs;
    }
  }
  return best;
}

}  // namespace

static bool tc_enabled() {
  // SD_ATTENTION_KERNEL=mma selects the mma.sync kernel for every shape
  // (comparison and testing); anything else keeps the tcgen05 path.
  static const bool on = [] {
    const char* e = getenv("SD_ATTENTION_KERNEL");
    return !(e && e[0] == 'm');
  }();
  return on;
}

static int serving_cluster(int B, int R, int Hq, int Hkv, int D, int cap);

bool sd_internal_tc_serves(int B, int R, int Hq, int Hkv, int D, int cap) {
  return serving_cluster(B, R, Hq, Hkv, D, cap) > 0;
}

template <bool kFused>
static sd_status launch_tc(const sd_kv_cache* cache, const void* q_for_map, const TcArgs& a,
                    const RopeTable& tab, int cs, bool pdl, cudaStream_t stream) {
  const int B = cache->batch, Hkv = cache->n_kv_heads, cap = cache->capacity;
  CUtensorMap k128, v128, k32, v32, qm;
  if (!make_map(&k128, cache->k, cap, B * Hkv, 128) || !make_map(&v128, cache->v, cap, B * Hkv, 128) ||
      !make_map(&k32, cache->k, cap, B * Hkv, 32) || !make_map(&v32, cache->v, cap, B * Hkv, 32) ||
      !make_q_map(&qm, q_for_map, B, a.R, a.Hq, a.G))
    return SD_ERR_CUDA;
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = cs;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.gridDim = dim3(cs, Hkv, B);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = kSmemBytes;
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 2 : 1;
  if (cudaLaunchKernelEx(&cfg, verify_attn_tc_kernel<kFused>, k128, v128, k32, v32, qm, a, tab) !=
      cudaSuccess) {
    (void)cudaGetLastError();
    return SD_ERR_CUDA;
  }
  return SD_OK;
}

static int serving_cluster(int B, int R, int Hq, int Hkv, int D, int cap) {
  if (!tc_enabled() || D != kD || Hkv <= 0 || Hq % Hkv) return 0;
  if ((Hq / Hkv) * R > kRows) return 0;
  DevState* s = state();
  if (!s || !s->ok) return 0;
  return pick_cluster(*s, static_cast<long long>(B) * Hkv, cap);
}

// Routed here by sd_verify_attention for head_dim 128 and G * R <= 32.
sd_status sd_internal_verify_attention_tc(const void* q, const sd_kv_cache* cache, void* out,
                                          int R, int Hq, float scale_log2, cudaStream_t stream,
                                          bool* handled) {
  *handled = false;
  const int B = cache->batch, Hkv = cache->n_kv_heads;
  const int cs = serving_cluster(B, R, Hq, Hkv, cache->head_dim, cache->capacity);
  if (cs <= 0) return SD_OK;
  TcArgs a = {};
  a.q = static_cast<const __nv_bfloat16*>(q);
  a.out = static_cast<__nv_bfloat16*>(out);
  a.len = cache->len;
  a.R = R;
  a.Hq = Hq;
  a.Hkv = Hkv;
  a.G = Hq / Hkv;
  a.M = a.G * R;
  a.cap = cache->capacity;
  a.n_mblocks = 1;
  a.scale_log2 = scale_log2;
  RopeTable tab = {};
  *handled = true;
  return launch_tc<false>(cache, q, a, tab, cs, false, stream);
}

// The fused verify layer (rope + append + attention) on the tcgen05 path.
sd_status sd_internal_verify_layer_tc(void* q, void* k_new, const void* v_new, const int32_t* pos,
                                      const RopeTable& tab, const sd_kv_cache* cache, void* out,
                                      int R, int Hq, float scale_log2, uint32_t* ticket, int early,
                                      cudaStream_t stream, bool* handled) {
  *handled = false;
  const int B = cache->batch, Hkv = cache->n_kv_heads;
  const int cs = serving_cluster(B, R, Hq, Hkv, cache->head_dim, cache->capacity);
  if (cs <= 0) return SD_OK;
  TcArgs a = {};
  a.q = static_cast<const __nv_bfloat16*>(q);
  a.out = static_cast<__nv_bfloat16*>(out);
  a.len = cache->len;
  a.qw = static_cast<__nv_bfloat16*>(q);
  a.k_new = static_cast<__nv_bfloat16*>(k_new);
  a.v_new = static_cast<const __nv_bfloat16*>(v_new);
  a.kc = static_cast<__nv_bfloat16*>(cache->k);
  a.vc = static_cast<__nv_bfloat16*>(cache->v);
  a.pos = pos;
  a.ticket = ticket;
  a.early = early ? 1 : 0;
  a.R = R;
  a.Hq = Hq;
  a.Hkv = Hkv;
  a.G = Hq / Hkv;
  a.M = a.G * R;
  a.cap = cache->capacity;
  a.n_mblocks = 1;
  a.scale_log2 = scale_log2;
  *handled = true;
  return launch_tc<true>(cache, q, a, tab, cs, early != 0, stream);
}
