// K3 on the 5th-generation tensor cores (tcgen05 + TMEM): verify attention
// of the K + 1 new rows against the cached prefix (Eq. verify, Sec. 3.2),
// for head_dim 128 and up to 128 packed query rows per KV head, and the fused
// verify layer (M-RoPE of Sec. 3.3 / Sec. 4.2 + the KV append of Eq. commit +
// the attention) on the same machinery.
//
// The packed query tile is small (G*R = 32 rows for 32 q / 8 KV heads and
// K = 7), so both products run TRANSPOSED, with the 128-wide dimension on the
// MMA's M side and no padding waste:
//     S^T[128 keys][kR rows] = K_tile[128 keys][128 d] . Q^T      (K-major A, B)
//     O^T[128 d][kR rows]   += V_tile^T[128 d][128 keys] . P^T     (MN-major A, B)
// kR = 32 (G*R <= 32) or 64 (G*R <= 64, and m-blocks of 64 rows up to 128);
// an N = 64 product costs about what an N = 32 one does. Both accumulators
// live in tensor memory, S triple-buffered: 4 kR columns.
//
// Warp roles in a CTA (352 threads). The issuing warps run converged: every
// lane waits on the barriers and one elected lane issues (issued from a
// one-lane branch instead, a batch of 8 MMAs took ~270 ns).
//   warp 0      TMA producer: 128-key tiles of K and V (128B-swizzled boxes)
//               into a K ring and a V ring of kS slots each (32 rows: 3, 64
//               rows: 2), with a barrier each: a K slot refills once its S
//               product is done, a V slot once its PV product is.
//   warp 1      allocates tensor memory; issues S(t) once the softmax has read
//               the buffer's previous S, S(t - 3), and commits "S(t) ready".
//   warps 2..9  softmax: thread (t, h) owns key lane t of S^T and query rows
//               h kR/2 .. h kR/2 + kR/2 - 1; P = exp2(S - ref) goes to shared
//               memory as P^T (MN-major; 64-byte swizzle for 32 rows, 128-byte
//               for 64), 16-byte stores, once PV(t - 2) has read that buffer.
//   warp 10     issues PV(t) once P(t) is stored and commits "PV(t) done";
//               one batch is issued while the other executes.
//
// Softmax with a fixed reference. The reference of a row is, in the
// standalone kernel, the exact maximum of the CTA's first tile and, in the
// fused layer, the row's larger score against its own new key and new key 0
// (keys the row sees, so its largest weight is about 1 or more), taken while
// the first S products run; every tile uses it unchanged, so the loop has no
// cross-warp step and O is never rescaled. The result is exact as long as
// no score exceeds its reference by more than kSlack (log2 units), which keeps
// every weight below 2^kSlack and every sum far inside fp32 range; each thread
// tracks the largest excess it saw, and a CTA where some excess is larger runs
// the whole range a second time with the exact maxima as references.
//
// Work split: one thread-block cluster per (scene, KV head); its CTAs take
// contiguous 32-key-aligned ranges of the keys, and their (m, l, O) partials
// merge through distributed shared memory at the end. In the fused layer the
// tensor-core loop covers the cached prefix only; the R new keys (rotated in
// shared memory, never re-read from the cache) enter as one more partial that
// each CTA forms on the CUDA cores for the rows it merges. Every wait is
// bounded (SD_DEVERR_TIMEOUT instead of a hang).
#include "common.cuh"

#include <cuda.h>

#include <math.h>
#include <stdlib.h>
#include <atomic>
#include <mutex>

SD_DEFINE_ERROR_ACCESSOR(sd_take_error_attention_tc)

namespace {

constexpr int kD = 128;         // head dim
constexpr int kStageKeys = 128; // M of S^T
constexpr int kHalf = kStageKeys * 128;     // one 64-column half of a 128-key tile (16 KB)
constexpr int kKV = 2 * kHalf;              // one K (or V) tile of 128 keys (32 KB)
constexpr int kNewRow = kD * 2;             // one new key / value row (256 B)
constexpr int kSoftWarps = 8;
constexpr int kSoftThreads = 32 * kSoftWarps;
constexpr int kPvWarp = 2 + kSoftWarps;        // the warp after the softmax warps issues PV
constexpr int kThreads = 96 + kSoftThreads;
constexpr uint32_t kSpinLimit = 1u << 20;
constexpr float kSlack = 64.f;              // log2 units a score may exceed its reference by
// a partial row sent to its owner is [O(128) | l by TMEM lane quarter (4) | m |
// 3 pad] fp32 = 544 bytes (16-byte multiple: one bulk copy per peer)
constexpr int kRowF = kD + 8;
constexpr int kRowL = kD;       // the four l terms (float4)
constexpr int kRowM = kD + 4;   // the row's reference m
constexpr int kRowBytes = kRowF * 4;
constexpr int round_up(int x, int m) { return (x + m - 1) / m * m; }

// Everything that depends on the packed query rows per CTA (kR = 32 or 64:
// the N of both MMAs). A softmax thread owns kR / 2 rows of one key lane.
template <int kR>
struct Cfg {
  static_assert(kR == 32 || kR == 64, "row tile");
  static constexpr int kRpt = kR / 2;                       // rows per softmax thread
  static constexpr int kMaxNew = kR == 32 ? 16 : 32;        // new rows the fused kernel takes
  // K and V rings of kStages tiles each: a K slot is free once its S product
  // is done, a V slot once its PV product is
  static constexpr int kStages = kR == 32 ? 3 : 2;
  static constexpr int kRingV = kStages * kKV;              // V slots follow the K slots
  static constexpr int kRing = 2 * kStages * kKV;
  static constexpr int kQHalf = kR * 128;
  static constexpr int kQ = 2 * kQHalf;
  static constexpr int kPRow = kR * 2;                      // one key of P^T in bf16
  static constexpr int kP = kStageKeys * kPRow;             // one P^T buffer
  // P^T is MN-major: 64-byte swizzle for 32 rows (a 64-byte key row), 128-byte
  // swizzle for 64 rows; 8-key groups are kPRow * 8 bytes apart
  static constexpr uint64_t kPLayout = kR == 32 ? 4 : 2;
  static constexpr int kTmemCols = kR == 32 ? 128 : 256;    // S0 | S1 | S2 | O, kR columns each
  // shared memory layout (offsets from the 1024-aligned base)
  static constexpr int kOffQ = kRing;
  // P^T buffers; before the tiles the second one holds the fused layer's
  // rotation table
  static constexpr int kOffP = kOffQ + kQ;
  static constexpr int kOffTab = kOffP + kP;
  static constexpr int kOffNewK = kOffP + 2 * kP;
  static constexpr int kOffNewV = kOffNewK + kMaxNew * kNewRow;
  static constexpr int kOffBar = kOffNewV + kMaxNew * kNewRow;
  // three S buffers in tensor memory (S0 | S1 | S2 | O fill the 128 or 256
  // columns)
  static constexpr int kSBuf = 3;
  // barriers: full_k[S] full_v[S] p_full[2] s_ready[3] pv_done[S] q_full recv
  // decide s_free[3] tmem_done
  static constexpr int kNumBars = 3 * kStages + 12;
  // tmem slot, (unused), decision, len (and, 64 rows, the last reader of the new key rows)
  static constexpr int kOffMisc = round_up(kOffBar + kNumBars * 8, 16);
  static constexpr int kOffRowA = kOffMisc + (kR == 32 ? 16 : 32);  // [kR] per-row results (reductions)
  static constexpr int kOffRef = kOffRowA + kR * 4;         // [kR] per-row references
  static constexpr int kOffLim = kOffRef + kR * 4;          // [kR] per-row causal key limits
  static constexpr int kSmemBytes = kOffLim + kR * 4 + 1024;
  static_assert(kSmemBytes <= 227 * 1024, "shared memory budget");
  static_assert(kOffQ % 1024 == 0 && kOffP % 1024 == 0 && kP % 1024 == 0 && kOffNewK % 16 == 0 &&
                    kOffNewV % 16 == 0 && kOffBar % 8 == 0 && kOffRowA % 16 == 0 && kOffRef % 16 == 0,
                "alignment of the shared-memory regions (swizzle atoms, vector accesses, mbarriers)");
  static_assert(kMaxNew * 64 * 8 <= kP, "rotation table fits the second P buffer");
  static_assert(kR * 128 * 4 <= 2 * kP, "row reductions fit the P buffers");
  // cluster merge buffers (in the rings, free once this CTA's last MMA is done)
  static constexpr int kSend = 0;                           // this CTA's kR rows
  static constexpr int kRecv = round_up(kR * kRowBytes, 1024);
  // slots for ceil(kR / c) rows from each of c ranks, c in {1, 2, 4, 6, 8, 16}
  static constexpr int kRecvSlots = kR == 32 ? 36 : 66;
  static constexpr int kNewS = round_up(kRecv + kRecvSlots * kRowBytes, 1024);  // new-key scores [rows][R]
  static_assert(kNewS + kR * kMaxNew * 4 <= kRing, "merge buffers");
};

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
__device__ __noinline__ void mbar_timed_out() { sd_set_error(SD_DEVERR_TIMEOUT); }
// One small loop per call site (the timeout report is out of line): the code
// that the warps run at the same time must stay inside the instruction cache.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity) {
#pragma unroll 1
  for (uint32_t i = 0; i < kSpinLimit; ++i)
    if (mbar_try_wait(bar, parity)) return true;
  mbar_timed_out();
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
// The same load with an L2 eviction policy (createpolicy): the cached prefix is
// read once per step, so its lines go first and the code and the per-step rows
// stay in L2 (an instruction fetch that misses L2 waits behind the stream).
__device__ __forceinline__ void tma_load_3d_hint(uint32_t dst, const CUtensorMap* map, uint32_t bar, int x, int y,
                                                 int z, uint64_t policy) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes.L2::cache_hint"
      " [%0], [%1, {%3, %4, %5}], [%2], %6;" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(bar), "r"(x), "r"(y), "r"(z), "l"(policy)
      : "memory");
}
__device__ __forceinline__ uint64_t l2_evict_first_policy() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
  return p;
}
__device__ __forceinline__ void tma_prefetch_3d(const CUtensorMap* map, int x, int y, int z) {
  asm volatile("cp.async.bulk.prefetch.tensor.3d.L2.global.tile [%0, {%1, %2, %3}];" ::"l"(
                   reinterpret_cast<uint64_t>(map)),
               "r"(x), "r"(y), "r"(z)
               : "memory");
}
__device__ __forceinline__ void bulk_prefetch_l2(const void* p, uint32_t bytes) {
  asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(reinterpret_cast<uint64_t>(p)), "r"(bytes)
               : "memory");
}
__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
// two floats -> bf16x2 (round to nearest even), lo in the low half
__device__ __forceinline__ uint32_t cvt_bf16x2(float lo, float hi) {
  uint32_t r;
  asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(hi), "f"(lo));
  return r;
}
__device__ __forceinline__ void named_bar_sync(int id, int threads) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(threads) : "memory");
}
// bar.sync over `threads` threads that also ORs a predicate across them
__device__ __forceinline__ bool named_bar_or(int id, int threads, bool p) {
  uint32_t r;
  asm volatile(
      "{\n\t.reg .pred pi, po;\n\tsetp.ne.u32 pi, %1, 0;\n\t"
      "bar.red.or.pred po, %2, %3, pi;\n\tselp.u32 %0, 1, 0, po;\n\t}"
      : "=r"(r)
      : "r"(static_cast<uint32_t>(p)), "r"(id), "r"(threads)
      : "memory");
  return r != 0;
}
// Sum over the 32 lanes of a warp of each of kN per-lane values (kN = 16 or
// 32), by a butterfly reduce-scatter: at the step of stride s a lane keeps the
// half of its values selected by its bit s and adds its partner's copy of that
// half. Lane L ends with the sum of value `row` (kN = 16: lanes L and L ^ 1
// hold the same value).
template <int kN>
__device__ __forceinline__ float warp_rows_sum(const float (&v0)[kN], int lane, int& row) {
  static_assert(kN == 16 || kN == 32, "rows per thread");
  float v[kN];
#pragma unroll
  for (int i = 0; i < kN; ++i) v[i] = v0[i];
  int r = 0;
#pragma unroll
  for (int n = kN, s = 16; n > 1; n >>= 1, s >>= 1) {
    const bool hi = (lane & s) != 0;
#pragma unroll
    for (int i = 0; i < n / 2; ++i) {
      const float keep = hi ? v[i + n / 2] : v[i];
      const float give = hi ? v[i] : v[i + n / 2];
      v[i] = keep + __shfl_xor_sync(0xffffffffu, give, s);
    }
    if (hi) r += n / 2;
  }
  float x = v[0];
  if (kN == 16) x += __shfl_xor_sync(0xffffffffu, x, 1);
  row = r;
  return x;
}
// an arrival that orders nothing: no data passes through the barrier
__device__ __forceinline__ void cluster_arrive_relaxed() {
  asm volatile("barrier.cluster.arrive.relaxed.aligned;" ::: "memory");
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
__device__ __forceinline__ void st_shared_v4(uint32_t addr, uint32_t x, uint32_t y, uint32_t z,
                                             uint32_t w) {
  asm volatile("st.shared.v4.u32 [%0], {%1,%2,%3,%4};" ::"r"(addr), "r"(x), "r"(y), "r"(z), "r"(w)
               : "memory");
}
// ---------------------------------------------------------------- tcgen05
// Shared-memory matrix descriptor (sm_100 family format): start address,
// leading / stride byte offsets (>> 4), version 1, layout type (2 = 128-byte
// swizzle, 4 = 64-byte swizzle).
__device__ __forceinline__ uint64_t umma_desc(uint32_t addr, uint32_t lbo, uint32_t sbo,
                                              uint64_t layout = 2) {
  return static_cast<uint64_t>((addr >> 4) & 0x3FFF) |
         (static_cast<uint64_t>((lbo >> 4) & 0x3FFF) << 16) |
         (static_cast<uint64_t>((sbo >> 4) & 0x3FFF) << 32) | (1ull << 46) | (layout << 61);
}
// Instruction descriptor, kind::f16: fp32 accumulate, bf16 A and B.
constexpr uint32_t umma_idesc(int M, int N, int a_mn_major, int b_mn_major) {
  return (1u << 4) | (1u << 7) | (1u << 10) | (static_cast<uint32_t>(a_mn_major) << 15) |
         (static_cast<uint32_t>(b_mn_major) << 16) | (static_cast<uint32_t>(N >> 3) << 17) |
         (static_cast<uint32_t>(M >> 4) << 24);
}

__device__ __forceinline__ void umma(uint32_t d_tmem, uint64_t a, uint64_t b, uint32_t idesc,
                                     int accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(a), "l"(b), "r"(idesc), "r"(accumulate)
      : "memory");
}
__device__ __forceinline__ __nv_bfloat162 as_bf162(uint32_t w) {
  __nv_bfloat162 v;
  memcpy(&v, &w, 4);
  return v;
}
// one lane of the (converged) warp
__device__ __forceinline__ bool elect_one() {
  uint32_t pred = 0;
  asm volatile(
      "{\n\t.reg .pred p;\n\telect.sync _|p, 0xffffffff;\n\tselp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(pred));
  return pred != 0;
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

// 16 consecutive fp32 columns of this warp's 32 TMEM lanes -> 16 registers
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,"
      "%14,%15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
        "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

// Per-row reduction (max or sum) over the 128 key lanes of a CTA, for the 256
// softmax threads: thread (key lane kl, rows row0 .. row0 + kN - 1) contributes
// v[j] to row row0 + j. The values pass through buf ([2 kN rows][128] fp32,
// free while this runs); the 2 kN results land in out[]. Called by all
// softmax threads; compact on purpose (it runs once or twice a launch).
template <bool kMax, int kN>
__device__ __forceinline__ void rows_reduce(const float (&v)[kN], int kl, int row0, int st, float* buf,
                                            float* out) {
  constexpr int kRowsAll = 2 * kN;
  constexpr int kPer = kSoftThreads / kRowsAll;  // threads per row (8 or 4)
  constexpr int kVals = 128 / kPer;              // values each of them reads (16 or 32)
#pragma unroll
  for (int j = 0; j < kN; ++j) buf[(row0 + j) * 128 + kl] = v[j];
  asm volatile("bar.sync 2, 256;" ::: "memory");
  const int r = st / kPer, part = st % kPer;
  // part p reads float4 q * kPer + p of its row: per load, the kPer threads of
  // a row cover kPer * 16 contiguous bytes (no bank conflicts beyond the rows)
  const float4* src = reinterpret_cast<const float4*>(buf + r * 128) + part;
  float acc = kMax ? -INFINITY : 0.f;
#pragma unroll
  for (int q = 0; q < kVals / 4; ++q) {
    const float4 x = src[q * kPer];
    acc = kMax ? fmaxf(acc, fmaxf(fmaxf(x.x, x.y), fmaxf(x.z, x.w))) : acc + ((x.x + x.y) + (x.z + x.w));
  }
#pragma unroll
  for (int w = 1; w < kPer; w <<= 1) {
    const float o = __shfl_xor_sync(0xffffffffu, acc, w);
    acc = kMax ? fmaxf(acc, o) : acc + o;
  }
  if (part == 0) out[r] = acc;
  asm volatile("bar.sync 2, 256;" ::: "memory");
}

// Second pass (fixed references exceeded): row r's reference moves to
// ref + max over the range of (score - ref); buf holds every thread's 16 or 32
// per-row maxima at [row][key lane]. Out of line: it runs only when a score
// exceeded its reference by more than the slack.
template <int kN>
__device__ __noinline__ void redo_references(int kl, int row0, int st, int quarter, int lane, float* buf,
                                             float* row_a, float* row_ref) {
  constexpr int kRowsAll = 2 * kN;
  constexpr int kPer = kSoftThreads / kRowsAll;
  constexpr int kVals = 128 / kPer;
  asm volatile("bar.sync 2, 256;" ::: "memory");
  const int r = st / kPer, part = st % kPer;
  const float4* src = reinterpret_cast<const float4*>(buf + r * 128) + part;
  float acc = -INFINITY;
#pragma unroll 1
  for (int q = 0; q < kVals / 4; ++q) {
    const float4 x = src[q * kPer];
    acc = fmaxf(acc, fmaxf(fmaxf(x.x, x.y), fmaxf(x.z, x.w)));
  }
  for (int w = 1; w < kPer; w <<= 1) acc = fmaxf(acc, __shfl_xor_sync(0xffffffffu, acc, w));
  if (part == 0) row_a[r] = acc;
  asm volatile("bar.sync 2, 256;" ::: "memory");
  if (quarter == 0 && lane < kN) {
    const float e = row_a[row0 + lane];
    const float m0 = row_ref[row0 + lane] == -INFINITY ? 0.f : row_ref[row0 + lane];
    row_ref[row0 + lane] = e == -INFINITY ? -INFINITY : m0 + e;
  }
  asm volatile("bar.sync 2, 256;" ::: "memory");
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
  uint32_t* kv_ticket;      // [B][Hkv] read-before-write-back tickets (several m-blocks)
  // kernels whose new keys enter as S_new: bit 0 = prefix, len (and pos) may
  // be read before the dependency wait, bit 1 = the block mask (every new row
  // sees all R new rows); the all-keys kernel: nonzero = the block mask
  int early;
  int R, Hq, Hkv, G, M, cap, n_mblocks;
  float inv_g;              // 1 / G: p / G == int((p + 0.5) / G) exactly for the p < 128 used here
  float scale_log2;
};

__device__ __forceinline__ void griddep_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void griddep_launch() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// ------------------------------------------------------------------ kernel
// kMode 0: attention over a cache that already holds the R new rows, every
// key in the tensor-core loop, the rotated query rows read from a.q.
// kMode 2: the same attention with the loop over the prefix keys only; the R
// new rows (read from the cache) enter as one more product S_new.
// kMode 1: the whole verify layer -- M-RoPE of the raw query and key rows, the
// KV append and the attention -- with len[b] the prefix length; the rotated
// new keys enter as S_new. Prefix tiles, len and pos are independent of the
// kernel that precedes this one in the stream (for every layer but the first
// of a step), so they are read before the programmatic-dependency wait.
// kMode 3: the same layer as a plain launch (everything after the wait).
// kMode 2 reads its prefix before the wait when bit 0 of a.early is set.
// Grid: (cluster size, Hkv * n_mblocks, B); m-block mb takes packed query rows
// mb * kR .. mb * kR + kR - 1.
template <int kR, int kMode>
__global__ void __launch_bounds__(kThreads, 1)
    verify_attn_tc_kernel(const __grid_constant__ CUtensorMap tm_k128,
                          const __grid_constant__ CUtensorMap tm_v128, const TcArgs a,
                          const RopeTable tab) {
  using C = Cfg<kR>;
  constexpr bool kFused = kMode == 1 || kMode == 3;
  constexpr bool kNew = kMode != 0;  // the R new keys enter as S_new, not as tiles
  // prefix (and len) before the dependency wait; the block mask
  const bool early = kMode == 1 || (kMode == 2 && (a.early & 1) != 0);
  // (the fused layer's 32-row tile takes no block mask: its callers are the
  // target's causal verify steps; the host sends block-masked layers of up to
  // 32 packed rows to the 64-row tile)
  const bool block = kMode == 0 ? a.early != 0 : ((kMode == 2 || kR == 64) && (a.early & 2) != 0);
  constexpr int kS = C::kStages;
  constexpr int kRpt = C::kRpt;
  constexpr uint32_t kIdescS = umma_idesc(128, kR, 0, 0);
  constexpr uint32_t kIdescO = umma_idesc(128, kR, 1, 1);
  constexpr int kTmemAlloc = C::kTmemCols;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  const uint32_t base = smem_addr(smem);
  const uint32_t qs = base + C::kOffQ;
  auto bar = [&](int i) { return base + C::kOffBar + 8u * i; };
  // barrier indices; T counts tiles over both passes. SREADY(T) and PVDONE(T)
  // (one slot per ring stage) are tcgen05.commit arrivals. A slot's next
  // phase cannot complete before each of its waiters has seen the current
  // one: S(T + kS) needs the K tile loaded after the producer's wait for
  // SREADY(T); PV(T + kS) needs the V tile loaded after the producer's wait
  // for PVDONE(T); the softmax's tile T + 1 follows its wait for SREADY(T),
  // and its wait for PVDONE(T) comes before P(T + 2), which PV(T + kS) needs.
  // K and V of a tile have their own barriers: a K slot refills once its S
  // product is done, a V slot once its PV product is.
  auto FULLK = [&](int s) { return bar(s); };
  auto FULLV = [&](int s) { return bar(kS + s); };
  auto PFULL = [&](int b) { return bar(2 * kS + b); };
  auto SREADY = [&](int T) { return bar(2 * kS + 2 + T % 3); };  // one per S buffer
  auto PVDONE = [&](int T) { return bar(2 * kS + 5 + T % kS); };
  auto ring_parity = [](int T) { return static_cast<uint32_t>((T / kS) & 1); };
  const uint32_t QFULL = bar(3 * kS + 5);
  const uint32_t RECV = bar(3 * kS + 6);    // the cluster merge's incoming partial rows
  const uint32_t DECIDE = bar(3 * kS + 7);  // whether the range runs a second time
  // 32 rows: the softmax has read S(T) (its tensor-memory buffer takes S(T + 3))
  auto SFREE = [&](int T) { return bar(3 * kS + 8 + T % 3); };
  auto s_parity = [](int T) { return static_cast<uint32_t>((T / 3) & 1); };  // SREADY, SFREE phases
  const uint32_t TMEMDONE = bar(3 * kS + 11);  // every softmax warp has read its last column
  constexpr int kSB = C::kSBuf;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + C::kOffMisc);
  int* s_redo = reinterpret_cast<int*>(smem + C::kOffMisc + 8);
  int* s_kvlast = reinterpret_cast<int*>(smem + C::kOffMisc + 16);  // 64 rows only
  float* row_a = reinterpret_cast<float*>(smem + C::kOffRowA);  // [kR] reduction results
  float* row_ref = reinterpret_cast<float*>(smem + C::kOffRef); // [kR] references
  int* row_lim = reinterpret_cast<int*>(smem + C::kOffLim);      // [kR] last key a row sees

  auto gdiv = [&](int p) { return __float2int_rz((static_cast<float>(p) + 0.5f) * a.inv_g); };
  const int rank = blockIdx.x;
  const int csize = gridDim.x;
  const int kvh = blockIdx.y % a.Hkv;
  const int mblock = blockIdx.y / a.Hkv;
  const int b = blockIdx.z;
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kS; ++s) {
      mbar_init(FULLK(s), 1);
      mbar_init(FULLV(s), 1);
      mbar_init(PVDONE(s), 1);
    }
    for (int i = 0; i < 3; ++i) mbar_init(SREADY(i), 1);
    for (int i = 0; i < 2; ++i) mbar_init(PFULL(i), kSoftWarps);
    mbar_init(QFULL, 1);  // one softmax thread, once the query tile is stored
    mbar_init(RECV, 1);
    mbar_init(DECIDE, 1);
    for (int i = 0; i < 3; ++i) mbar_init(SFREE(i), kSoftWarps);
    mbar_init(TMEMDONE, kSoftWarps);
    *s_redo = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_addr(tmem_slot)),
                 "r"(kTmemAlloc)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  // len, pos, the rows and the prefix may come from the previous kernel: a
  // launch without the early prefix waits here, before any global access
  if (kNew && !early) griddep_wait();
  int* s_len = reinterpret_cast<int*>(smem + C::kOffMisc + 12);
  if (threadIdx.x == 0) {
    *s_len = a.len[b];  // the scene's length advances at the producer's end
  }
  // The fused layer's raw q / k / v rows do not depend on len or pos. In a
  // plain launch (the dependency wait above comes before everything) the
  // softmax threads issue their row loads together with the pos loads of the
  // rotation table: one global round trip before the tiles instead of two.
  constexpr int kQc = kR * 16 / kSoftThreads;        // 16-byte query chunks a thread
  constexpr int kKvc = C::kMaxNew * 16 / kSoftThreads;  // 16-byte new key / value chunks a thread
  constexpr bool rows_first = kMode == 3;
  uint4 pre_q[kQc], pre_k[kKvc], pre_v[kKvc];
  auto preload_rows = [&](int st) {
#pragma unroll
    for (int u = 0; u < kQc; ++u) {
      const int idx = st + u * kSoftThreads, p = mblock * kR + (idx >> 4), c = idx & 15;
      const int i = gdiv(p);
      pre_q[u] = p < a.M ? __ldcg(reinterpret_cast<const uint4*>(
                               a.qw + ((static_cast<long long>(b) * a.R + i) * a.Hq + kvh * a.G + (p - i * a.G)) * kD +
                               c * 8))
                         : make_uint4(0, 0, 0, 0);
    }
#pragma unroll
    for (int u = 0; u < kKvc; ++u) {
      const int idx = st + u * kSoftThreads;
      const long long src = ((static_cast<long long>(b) * a.R + (idx >> 4)) * a.Hkv + kvh) * kD + (idx & 15) * 8;
      const bool ok = idx < a.R * 16;
      pre_k[u] = ok ? __ldcg(reinterpret_cast<const uint4*>(a.k_new + src)) : make_uint4(0, 0, 0, 0);
      pre_v[u] = ok ? __ldcg(reinterpret_cast<const uint4*>(a.v_new + src)) : make_uint4(0, 0, 0, 0);
    }
  };
  if (kFused && threadIdx.x >= 64 && threadIdx.x < 64 + kSoftThreads) {
    if (rows_first) preload_rows(threadIdx.x - 64);
    // rotation table of the R new positions: (cos, sin) per (row, pair),
    // built while thread 0 takes the scene's length
    float2* tabw = reinterpret_cast<float2*>(smem + C::kOffTab);
#pragma unroll 1
    for (int idx = threadIdx.x - 64; idx < a.R * 64; idx += kSoftThreads) {
      const int i = idx >> 6, d = idx & 63;
      const int32_t pc = a.pos[(static_cast<long long>(blockIdx.z) * a.R + i) * 3 + tab.axis[d]];
      tabw[idx] = sd_rope_cs(static_cast<float>(pc), d, tab);
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const uint32_t tmem_s = tmem;            // S buffer b at column kR * b
  const uint32_t tmem_o = tmem + kSB * kR; // O^T

  int n_keys, L_pre;
  bool valid;
  if (kFused) {
    L_pre = *s_len;
    n_keys = L_pre + a.R;
    valid = L_pre >= 0 && n_keys <= a.cap;
    if (!valid && rank == 0 && threadIdx.x == 0 && blockIdx.y == 0)
      sd_set_error(L_pre < 0 ? SD_DEVERR_LENGTH : SD_DEVERR_KV_OVERFLOW);
  } else {
    n_keys = *s_len;
    valid = n_keys >= a.R && n_keys <= a.cap;
    L_pre = n_keys - a.R;
    if (!valid && rank == 0 && threadIdx.x == 0 && blockIdx.y == 0) sd_set_error(SD_DEVERR_LENGTH);
  }
  // the tensor-core loop covers the prefix (fused) or every key (standalone)
  const int loop_keys = valid ? (kNew ? L_pre : n_keys) : 0;
  const int nblk = (loop_keys + 31) / 32;
  // rank * nblk < 2^31 (16 ranks, nblk <= cap / 32): 32-bit division
  const int blk_begin = static_cast<int>((static_cast<uint32_t>(rank) * nblk) / static_cast<uint32_t>(csize));
  const int blk_end = static_cast<int>((static_cast<uint32_t>(rank + 1) * nblk) / static_cast<uint32_t>(csize));
  const int key_begin = blk_begin * 32;
  const int key_end = min(blk_end * 32, loop_keys);
  const int n_tiles = (blk_end - blk_begin + 3) / 4;
  // rank c merges packed rows [c * rpc, c * rpc + rows_of(c)) of the m-block's
  // rows_in rows that exist (the tile's rows past M are never exchanged: a
  // single-row draft step with G = 4 moves 4 rows, not 32), rpc = ceil(rows_in / csize)
  const int rows_in = max(1, min(kR, a.M - mblock * kR));
  const int rpc = (rows_in + csize - 1) / csize;
  auto rows_of = [&](int c) { return max(0, min(rpc, rows_in - c * rpc)); };
  const int my_rows = rows_of(rank);
  const int mrow0 = rank * rpc;
  if (warp == 0) {
    // -------------------------------------------------------------- producer
    // the whole warp waits, one elected lane issues the copies
    const int z = b * a.Hkv + kvh;
    const uint64_t evict_first = l2_evict_first_policy();
    auto issue_tiles = [&](int pass) {
      for (int t = 0; t < n_tiles; ++t) {
        const int T = pass * n_tiles + t;
        const int s = T % kS;
        // a whole 128-row box even for a short last tile: keys past the
        // range are masked, rows past the capacity arrive zero-filled
        const int y0 = key_begin + t * kStageKeys;
        // slot s last held tile T - kS (all of pass 0 is done before pass 1)
        const uint32_t kst = base + s * kKV, vst = base + C::kRingV + s * kKV;
        if (t >= kS) mbar_wait(SREADY(T - kS), s_parity(T - kS));
        if (elect_one()) {
          mbar_expect_tx(FULLK(s), static_cast<uint32_t>(kKV));
#pragma unroll
          for (int h = 0; h < 2; ++h) tma_load_3d_hint(kst + h * kHalf, &tm_k128, FULLK(s), h * 64, y0, z, evict_first);
        }
        __syncwarp();
        if (t >= kS) mbar_wait(PVDONE(T - kS), ring_parity(T - kS));
        if (elect_one()) {
          mbar_expect_tx(FULLV(s), static_cast<uint32_t>(kKV));
#pragma unroll
          for (int h = 0; h < 2; ++h) tma_load_3d_hint(vst + h * kHalf, &tm_v128, FULLV(s), h * 64, y0, z, evict_first);
        }
        __syncwarp();
      }
    };
    if (n_tiles > 0) {
      if (elect_one()) {
        asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tm_k128)) : "memory");
        asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tm_v128)) : "memory");
        // chained layers: the cluster launched last (the last KV head of the
        // last scene) starts only when the previous layer frees its SMs; the
        // first head's CTAs bring that head's tiles of their own key range
        // into L2 meanwhile
        if (kNew && early && kvh == 0 && b == static_cast<int>(gridDim.z) - 1 && a.Hkv > 1) {
          const int zl = b * a.Hkv + a.Hkv - 1;
          for (int t = 0; t < n_tiles; ++t)
#pragma unroll
            for (int h = 0; h < 2; ++h) {
              tma_prefetch_3d(&tm_k128, h * 64, key_begin + t * kStageKeys, zl);
              tma_prefetch_3d(&tm_v128, h * 64, key_begin + t * kStageKeys, zl);
            }
          // and that head's query and new key / value rows
          if (rank == 0)
            for (int i = 0; i < a.R; ++i) {
              const long long row = static_cast<long long>(b) * a.R + i;
              bulk_prefetch_l2((kFused ? a.qw : a.q) + (row * a.Hq + (a.Hkv - 1) * a.G) * kD, a.G * kD * 2);
              if (kFused) {
                bulk_prefetch_l2(a.k_new + (row * a.Hkv + a.Hkv - 1) * kD, kD * 2);
                bulk_prefetch_l2(a.v_new + (row * a.Hkv + a.Hkv - 1) * kD, kD * 2);
              }
            }
        }
      }
      __syncwarp();
      issue_tiles(0);
    }
    __syncwarp();
    // The cluster barrier lets peers write partials into this CTA's rings: the
    // softmax threads arrive only after the last MMA of the last pass, so this
    // warp (as the issuing warps) arrives before the second-pass decision.
    cluster_arrive_relaxed();
    if (kFused && elect_one()) {
      // advance the scene's length once every CTA of the scene has read it:
      // the last CTA to take a ticket writes it. This lane (thread 0) read
      // the length in the prologue; the fence orders that read before the
      // ticket. Taken after the cluster arrival, so no barrier waits for it.
      __threadfence();
      const uint32_t total = gridDim.x * gridDim.y;
      if (atomicAdd(&a.ticket[b], 1u) == total - 1) {
        const int len0 = *s_len;
        if (len0 >= 0 && len0 + a.R <= a.cap) a.len[b] = len0 + a.R;
        a.ticket[b] = 0;
      }
    }
    __syncwarp();
    if (n_tiles > 0) {
      // every MMA of pass 0 is done when the decision is out
      mbar_wait(DECIDE, 0);
      if (*reinterpret_cast<volatile int*>(s_redo)) issue_tiles(1);
    }
    __syncwarp();
    cluster_wait();
  } else if (warp == 1) {
    // -------------------------------------------------------------- S issue
    // S(T) and PV(T) come from two warps (this one and the PV warp), so that
    // one batch is issued while the other executes; the whole warp waits and
    // one elected lane issues.
    bool arrived = false;
    if (n_tiles > 0) {
      mbar_wait(QFULL, 0);
      // base descriptors; a K step only moves the start address (low field, no carry)
      const uint64_t dK0 = umma_desc(base, 16, 1024);  // K tile: K-major
      const uint64_t dQ = umma_desc(qs, 16, 1024);     // Q: K-major
      for (int pass = 0; pass < 2; ++pass) {
        if (pass == 1) {
          cluster_arrive_relaxed();  // before the decision (see the producer)
          arrived = true;
          mbar_wait(DECIDE, 0);
          if (!*reinterpret_cast<volatile int*>(s_redo)) break;
        }
        const int T0 = pass * n_tiles;
        for (int t = 0; t < n_tiles; ++t) {
          // S(T) reuses the S buffer of tile T - 3: the softmax has read it
          // once SFREE(T - 3) is out; pass 1 starts after all of pass 0
          const int T = T0 + t, st_ = T % kS;
          if (t >= 3) mbar_wait(SFREE(T), s_parity(T - 3));
          mbar_wait(FULLK(st_), ring_parity(T));
          tc_fence_after();
          const uint64_t dk = dK0 + static_cast<uint64_t>((st_ * kKV) >> 4);
          const uint32_t ts = tmem_s + kR * (T % kSB);
          if (elect_one()) {
#pragma unroll
            for (int kk = 0; kk < 8; ++kk)
              umma(ts, dk + (((kk >> 2) * kHalf + (kk & 3) * 32) >> 4),
                   dQ + (((kk >> 2) * C::kQHalf + (kk & 3) * 32) >> 4), kIdescS, kk > 0 ? 1 : 0);
            umma_commit(SREADY(T));
          }
          __syncwarp();
        }
      }
    }
    __syncwarp();
    if (!arrived) cluster_arrive_relaxed();
    // the allocating warp frees the tensor memory once every softmax warp has
    // read its last column (every MMA is done by then)
    mbar_wait(TMEMDONE, 0);
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTmemAlloc) : "memory");
    cluster_wait();
  } else if (warp == kPvWarp) {
    // -------------------------------------------------------------- PV issue
    bool arrived = false;
    if (n_tiles > 0) {
      const uint64_t dV0 = umma_desc(base + C::kRingV, kHalf, 1024);  // V^T: MN-major
      // P^T: MN-major, one swizzle atom wide (kR rows), 8-key groups 8 * kPRow apart
      const uint64_t dP0 = umma_desc(base + C::kOffP, 0, 8 * C::kPRow, C::kPLayout);
      for (int pass = 0; pass < 2; ++pass) {
        if (pass == 1) {
          cluster_arrive_relaxed();  // before the decision (see the producer)
          arrived = true;
          mbar_wait(DECIDE, 0);
          if (!*reinterpret_cast<volatile int*>(s_redo)) break;
        }
        const int T0 = pass * n_tiles;
        for (int t = 0; t < n_tiles; ++t) {
          const int T = T0 + t;
          mbar_wait(PFULL(T & 1), (T >> 1) & 1);
          mbar_wait(FULLV(T % kS), ring_parity(T));  // the V tile has landed
          tc_fence_after();
          const uint64_t dv = dV0 + static_cast<uint64_t>(((T % kS) * kKV) >> 4);
          const uint64_t dp = dP0 + static_cast<uint64_t>(((T & 1) * C::kP) >> 4);
          if (elect_one()) {
#pragma unroll
            for (int kk = 0; kk < 8; ++kk)
              umma(tmem_o, dv + (kk * 2048 >> 4), dp + (kk * 16 * C::kPRow >> 4), kIdescO,
                   (t > 0 || kk > 0) ? 1 : 0);
            umma_commit(PVDONE(T));
          }
          __syncwarp();
        }
      }
    }
    __syncwarp();
    if (!arrived) cluster_arrive_relaxed();
    cluster_wait();
  } else {
    // -------------------------------------------------------------- softmax
    const int st = threadIdx.x - 64;       // 0..255
    const int half = (warp - 2) >> 2;      // query rows kRpt*half .. kRpt*half + kRpt - 1
    const int quarter = warp & 3;          // TMEM lane quarter of this warp
    const int kl = quarter * 32 + lane;    // key lane of S^T / d lane of O^T
    const uint32_t lane_off = static_cast<uint32_t>(quarter * 32) << 16;
    const int row0 = kRpt * half;          // first query row of this thread
    const float2* cs_tab = reinterpret_cast<const float2*>(smem + C::kOffTab);  // [R][64] (cos, sin)
    {
      // the packed query tile: this thread's 16-byte chunks (row, chunk c),
      // rows past M zero; in the fused layer also one chunk of a new key and
      // value row
      const __nv_bfloat16* q_src[kQc];
      int q_cs[kQc];
      bool q_ok[kQc];
#pragma unroll
      for (int u = 0; u < kQc; ++u) {
        const int idx = st + u * kSoftThreads, p = mblock * kR + (idx >> 4), c = idx & 15;
        const int i = gdiv(p);
        q_ok[u] = valid && p < a.M;
        q_src[u] = (kFused ? a.qw : a.q) +
                   ((static_cast<long long>(b) * a.R + i) * a.Hq + kvh * a.G + (p - i * a.G)) * kD + c * 8;
        q_cs[u] = i * 64 + c * 4;
      }
      // new key / value rows: chunk st + u * 256 (row >> 4, 16-byte chunk & 15);
      // one chunk a thread with 32 rows (16 new rows), two with 64 (32)
      const bool append = kFused && valid && rank == csize - 1 && mblock == 0;
      bool has_kv[kKvc];
      long long kv_src[kKvc];
#pragma unroll
      for (int u = 0; u < kKvc; ++u) {
        const int idx = st + u * kSoftThreads;
        has_kv[u] = kNew && valid && idx < a.R * 16;
        // fused: the raw rows [B][R][Hkv][D]; attention-only: cache rows L_pre + i
        kv_src[u] = kFused ? ((static_cast<long long>(b) * a.R + (idx >> 4)) * a.Hkv + kvh) * kD + (idx & 15) * 8
                           : ((static_cast<long long>(b) * a.Hkv + kvh) * a.cap + L_pre + (idx >> 4)) * kD + (idx & 15) * 8;
      }
      // Fused: iteration 0 runs BEFORE the dependency wait on whatever the
      // rows hold: it brings this code into the instruction cache and the rows
      // into L2, and iteration 1 overwrites everything it stored. The loads
      // bypass L1 (.cg) so that iteration 1 cannot hit a line read before the wait.
      // the cluster launched last starts when the previous kernel is done or
      // nearly so: no warm-up pass, its rows are read once, after the wait
      const bool last_cluster = blockIdx.y == gridDim.y - 1 && blockIdx.z == gridDim.z - 1;
#pragma unroll 1
      for (int it = (kNew && !rows_first && !(early && last_cluster)) ? 0 : 1; it < 2; ++it) {
        if (kNew && it == 1 && early && !rows_first) griddep_wait();  // the rows come from earlier kernels
        uint4 qv[kQc], kv[kKvc], vv[kKvc];
        if (rows_first) {
#pragma unroll
          for (int u = 0; u < kQc; ++u) qv[u] = q_ok[u] ? pre_q[u] : make_uint4(0, 0, 0, 0);
#pragma unroll
          for (int u = 0; u < kKvc; ++u) {
            kv[u] = has_kv[u] ? pre_k[u] : make_uint4(0, 0, 0, 0);
            vv[u] = has_kv[u] ? pre_v[u] : make_uint4(0, 0, 0, 0);
          }
        } else {
#pragma unroll
          for (int u = 0; u < kQc; ++u)
            qv[u] = q_ok[u] ? __ldcg(reinterpret_cast<const uint4*>(q_src[u])) : make_uint4(0, 0, 0, 0);
#pragma unroll
          for (int u = 0; u < kKvc; ++u) {
            kv[u] = has_kv[u] ? __ldcg(reinterpret_cast<const uint4*>((kFused ? a.k_new : a.kc) + kv_src[u]))
                              : make_uint4(0, 0, 0, 0);
            vv[u] = has_kv[u] ? __ldcg(reinterpret_cast<const uint4*>((kFused ? a.v_new : a.vc) + kv_src[u]))
                              : make_uint4(0, 0, 0, 0);
          }
        }
        // (fused: M-RoPE of) the packed query rows, straight into the swizzled tile
#pragma unroll
        for (int u = 0; u < kQc; ++u) {
          const int idx = st + u * kSoftThreads, row = idx >> 4, c = idx & 15;
          uint32_t w[4] = {qv[u].x, qv[u].y, qv[u].z, qv[u].w};
          if (kFused && q_ok[u]) {
            const float2* cs = cs_tab + q_cs[u];
#pragma unroll
            for (int j = 0; j < 4; ++j) w[j] = sd_rope_pair(w[j], cs[j].x, cs[j].y);
          }
          st_shared_v4(qs + (c >> 3) * C::kQHalf + row * 128 + (((c & 7) ^ (row & 7)) << 4), w[0], w[1],
                       w[2], w[3]);
        }
        // the new key rows (rotated) and value rows of this head; value rows
        // past R stay zero (the merge reads all kMaxNew rows)
#pragma unroll
        for (int u = 0; u < kKvc; ++u) {
          if (!kNew) break;
          const int idx = st + u * kSoftThreads, i = idx >> 4, c = idx & 15;
          if (has_kv[u]) {
            uint32_t w[4] = {kv[u].x, kv[u].y, kv[u].z, kv[u].w};
            if (kFused) {
              const float2* cs = cs_tab + i * 64 + c * 4;
#pragma unroll
              for (int j = 0; j < 4; ++j) w[j] = sd_rope_pair(w[j], cs[j].x, cs[j].y);
            }
            st_shared_v4(base + C::kOffNewK + i * kNewRow + c * 16, w[0], w[1], w[2], w[3]);
            st_shared_v4(base + C::kOffNewV + i * kNewRow + c * 16, vv[u].x, vv[u].y, vv[u].z, vv[u].w);
            if (append && it == 1) {
              // the append (the head's last rank of m-block 0): cache rows
              // L_pre .. L_pre + R - 1, which no CTA of this launch reads
              const long long dst = ((static_cast<long long>(b) * a.Hkv + kvh) * a.cap + L_pre + i) * kD + c * 8;
              *reinterpret_cast<uint4*>(a.kc + dst) = make_uint4(w[0], w[1], w[2], w[3]);
              *reinterpret_cast<uint4*>(a.vc + dst) = vv[u];
            }
          } else {
            st_shared_v4(base + C::kOffNewV + i * kNewRow + c * 16, 0u, 0u, 0u, 0u);
          }
        }
      }
      // causal limit of each packed row: row p = i * G + g is new row i and
      // sees keys 0 .. L_prefix + i (Eq. verify's mask)
      if (!kNew && st < kR)
        row_lim[st] = block ? n_keys - 1 : min(n_keys - a.R + gdiv(mblock * kR + st), n_keys - 1);
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
      named_bar_sync(2, kSoftThreads);  // Q is complete; the rotation table is no longer read
      if (st == 0) {
        mbar_arrive(QFULL);
        // every older kernel has finished: the next layer may launch
        if (kNew) griddep_launch();
        // with several m-blocks the head's raw key rows are read by several
        // clusters: the last of the head's CTAs to have read them writes the
        // rotated rows back (the fence orders this CTA's reads before its ticket)
        if constexpr (kR == 64) {
          if (kFused && valid) {
            if (a.n_mblocks > 1) {
              __threadfence();
              *s_kvlast = atomicAdd(&a.kv_ticket[b * a.Hkv + kvh], 1u) ==
                          static_cast<uint32_t>(csize * a.n_mblocks - 1);
            } else {
              *s_kvlast = rank == csize - 1;
            }
          }
        }
      }
    }

    const float sl = a.scale_log2;
    // The reference of a row (log2 units, -inf: no key yet) lives in row_ref;
    // with 32 rows a thread also keeps its 16 in registers, with 64 rows it
    // reloads them every tile (broadcast loads) to stay within the registers
    // that 11 warps leave a thread.
    constexpr bool kRefRegs = kR == 32;
    float ref[kRefRegs ? kRpt : 1];
    float lp[kRpt];   // per-row partial sums of this thread's key lane
    float ex[kRpt];   // largest score - reference seen
#pragma unroll
    for (int j = 0; j < kRpt; ++j) {
      lp[j] = 0.f;
      ex[j] = -INFINITY;
    }
    ref[0] = -INFINITY;
    const int L_prefix = n_keys - a.R;
    // per-key-lane mask of rows row0 + j0 .. row0 + j0 + 15 for a tile: the
    // key range, and the causal limit of the new rows that the standalone
    // kernel's range contains
    auto tile_mask = [&](int key0, int j0, bool (&ok)[16]) {
      const int key = key0 + kl;
      const bool key_ok = key < key_end;
      const bool tail = !kNew && key0 + kStageKeys - 1 > L_prefix;
#pragma unroll
      for (int j = 0; j < 16; ++j) {
        ok[j] = key_ok;
        if (tail) ok[j] = ok[j] && key <= row_lim[row0 + j0 + j];
      }
    };
    if (kNew) {
      // references: the larger score of each row against its own new key and
      // new key 0 (keys the row sees, so its largest weight is at least about
      // 1 and its sum cannot vanish), taken while S(0) and S(1) run; bf16 dot
      // products suffice for a reference. 8 threads a row, 16 d each.
      const int sub = lane & 7;
#pragma unroll 1
      for (int r = st >> 3; r < kR; r += kSoftThreads / 8) {  // warp-uniform trip count
        const int p = mblock * kR + r;
        const bool row_ok = valid && p < a.M;
        const int n = row_ok ? gdiv(p) : 0;  // the row's own new key
        __nv_bfloat162 acc0 = __float2bfloat162_rn(0.f), acc1 = acc0, acc2 = acc0, acc3 = acc0;
#pragma unroll
        for (int u = 0; u < 2; ++u) {
          const int c = sub + 8 * u;
          const uint4 qw = *reinterpret_cast<const uint4*>(smem + C::kOffQ + (c >> 3) * C::kQHalf + r * 128 +
                                                           (((c & 7) ^ (r & 7)) << 4));
          const uint4 kw = *reinterpret_cast<const uint4*>(smem + C::kOffNewK + n * kNewRow + c * 16);
          const uint4 k0 = *reinterpret_cast<const uint4*>(smem + C::kOffNewK + c * 16);
          acc0 = __hfma2(as_bf162(qw.x), as_bf162(kw.x), acc0);
          acc1 = __hfma2(as_bf162(qw.y), as_bf162(kw.y), acc1);
          acc2 = __hfma2(as_bf162(qw.x), as_bf162(k0.x), acc2);
          acc3 = __hfma2(as_bf162(qw.y), as_bf162(k0.y), acc3);
          acc0 = __hfma2(as_bf162(qw.z), as_bf162(kw.z), acc0);
          acc1 = __hfma2(as_bf162(qw.w), as_bf162(kw.w), acc1);
          acc2 = __hfma2(as_bf162(qw.z), as_bf162(k0.z), acc2);
          acc3 = __hfma2(as_bf162(qw.w), as_bf162(k0.w), acc3);
        }
        float sd = (__low2float(acc0) + __high2float(acc0)) + (__low2float(acc1) + __high2float(acc1));
        float s0 = (__low2float(acc2) + __high2float(acc2)) + (__low2float(acc3) + __high2float(acc3));
#pragma unroll
        for (int sh = 1; sh < 8; sh <<= 1) {
          sd += __shfl_xor_sync(0xffffffffu, sd, sh);
          s0 += __shfl_xor_sync(0xffffffffu, s0, sh);
        }
        const float best = row_ok ? fmaxf(sd, s0) : -INFINITY;
        if (sub == 0) row_ref[r] = best == -INFINITY ? -INFINITY : best * sl;
      }
      named_bar_sync(2, kSoftThreads);
      if (kRefRegs) {
        const float4* rr4 = reinterpret_cast<const float4*>(row_ref + row0);
#pragma unroll
        for (int j4 = 0; j4 < (kRefRegs ? kRpt / 4 : 0); ++j4) {
          const float4 x = rr4[j4];
          ref[(4 * j4 + 0) % (kRefRegs ? kRpt : 1)] = x.x;
          ref[(4 * j4 + 1) % (kRefRegs ? kRpt : 1)] = x.y;
          ref[(4 * j4 + 2) % (kRefRegs ? kRpt : 1)] = x.z;
          ref[(4 * j4 + 3) % (kRefRegs ? kRpt : 1)] = x.w;
        }
      }
    } else if (n_tiles > 0) {
      // references: exact row maxima of the first tile (through the P buffers,
      // which no P has used yet)
      mbar_wait(SREADY(0), 0);
      tc_fence_after();
      float v[kRpt];
#pragma unroll
      for (int j0 = 0; j0 < kRpt; j0 += 16) {
        uint32_t r[16];
        tmem_ld16(tmem_s + row0 + j0 + lane_off, r);
        bool ok[16];
        tile_mask(key_begin, j0, ok);
#pragma unroll
        for (int j = 0; j < 16; ++j) v[j0 + j] = ok[j] ? __uint_as_float(r[j]) * sl : -INFINITY;
      }
      rows_reduce<true>(v, kl, row0, st, reinterpret_cast<float*>(smem + C::kOffP), row_ref);
      if (kRefRegs) {
        const float4* rr4 = reinterpret_cast<const float4*>(row_ref + row0);
#pragma unroll
        for (int j4 = 0; j4 < (kRefRegs ? kRpt / 4 : 0); ++j4) {
          const float4 x = rr4[j4];
          ref[4 * j4 + 0] = x.x;
          ref[4 * j4 + 1] = x.y;
          ref[4 * j4 + 2] = x.z;
          ref[4 * j4 + 3] = x.w;
        }
      }
    }
    bool redo = false;
    for (int pass = 0; pass < 2; ++pass) {
      if (pass == 1 && !redo) break;
      for (int t = 0; t < n_tiles; ++t) {
        const int T = pass * n_tiles + t;
        const int bb = T & 1, s = T % kS;
        const int key0 = key_begin + t * kStageKeys;
        const int key = key0 + kl;
        mbar_wait(SREADY(T), s_parity(T));  // S(T) is ready
        tc_fence_after();
        const bool key_ok = key < key_end;
        // P^T key row kl, once PV(T - 2) has read the buffer: kRpt rows =
        // kRpt / 8 16-byte chunks of 8 query rows, swizzled
        const uint32_t prow = base + C::kOffP + bb * C::kP + kl * C::kPRow;
        const int sw = kR == 32 ? (kl >> 1) & 3 : kl & 7;
#pragma unroll
        for (int j0 = 0; j0 < kRpt; j0 += 16) {
          // 16 rows past the tile's existing rows (warp-uniform): no scores to
          // read and no P to write; their P columns stay stale and reach only
          // O columns that are never read. The buffer release and the PV wait
          // stay, so every barrier phase still completes in order.
          if (row0 + j0 >= rows_in) {
            if (j0 + 16 >= kRpt) {
              tc_fence_before();
              __syncwarp();
              if (lane == 0) mbar_arrive(SFREE(T));
            }
            if (T >= 2 && j0 == 0) mbar_wait(PVDONE(T - 2), ring_parity(T - 2));
            continue;
          }
          uint32_t r[16];
          tmem_ld16(tmem_s + kR * (T % kSB) + row0 + j0 + lane_off, r);
          if (j0 + 16 >= kRpt) {
            // S(T) is in registers (its last 16 rows): its buffer may take S(T + 3)
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(SFREE(T));
          }
          bool ok[16];
          tile_mask(key0, j0, ok);
          float rc[16];
#pragma unroll
          for (int j = 0; j < 16; ++j) rc[j] = kRefRegs ? ref[(j0 + j) % (kRefRegs ? kRpt : 1)] : 0.f;
          if (!kRefRegs) {
            const float4* rr4 = reinterpret_cast<const float4*>(row_ref + row0 + j0);
#pragma unroll
            for (int j4 = 0; j4 < 4; ++j4) {
              const float4 x = rr4[j4];
              rc[4 * j4 + 0] = x.x;
              rc[4 * j4 + 1] = x.y;
              rc[4 * j4 + 2] = x.z;
              rc[4 * j4 + 3] = x.w;
            }
          }
          // P = exp2(S * scale - ref) in bf16; l partials from the same rounded weights
          uint32_t pw[8];
#pragma unroll
          for (int j = 0; j < 16; j += 2) {
            const float m0 = rc[j] == -INFINITY ? 0.f : rc[j];
            const float m1 = rc[j + 1] == -INFINITY ? 0.f : rc[j + 1];
            const float y0 = ok[j] ? fmaf(__uint_as_float(r[j]), sl, -m0) : -INFINITY;
            const float y1 = ok[j + 1] ? fmaf(__uint_as_float(r[j + 1]), sl, -m1) : -INFINITY;
            ex[j0 + j] = fmaxf(ex[j0 + j], y0);
            ex[j0 + j + 1] = fmaxf(ex[j0 + j + 1], y1);
            const uint32_t w = cvt_bf16x2(ex2(y0), ex2(y1));
            pw[j >> 1] = w;
            lp[j0 + j] += sd_bf16_lo(w);
            lp[j0 + j + 1] += sd_bf16_hi(w);
          }
          if (T >= 2 && j0 == 0) mbar_wait(PVDONE(T - 2), ring_parity(T - 2));  // PV(T - 2) has read P buffer bb
          const int ch = (row0 + j0) >> 3;
          st_shared_v4(prow + ((ch ^ sw) << 4), pw[0], pw[1], pw[2], pw[3]);
          st_shared_v4(prow + (((ch + 1) ^ sw) << 4), pw[4], pw[5], pw[6], pw[7]);
        }
        if (!key_ok) {
          // stale or foreign key row: zero its V row (this thread's 64-column
          // half) so 0 * NaN cannot reach O, once the tile has landed
          mbar_wait(FULLV(s), ring_parity(T));
          const uint32_t vrow = base + C::kRingV + s * kKV + half * kHalf + kl * 128;
#pragma unroll
          for (int c = 0; c < 8; ++c) st_shared_v4(vrow + c * 16, 0u, 0u, 0u, 0u);
        }
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(PFULL(bb));
      }
      if (pass == 0) {
        // did any score exceed its reference by more than kSlack? (one
        // OR-reducing barrier over the softmax threads, while the last PV
        // product runs)
        bool over = false;
#pragma unroll
        for (int j = 0; j < kRpt; ++j) over |= ex[j] > kSlack;
        redo = named_bar_or(2, kSoftThreads, over);
        // before a second pass every MMA of the first is done (the producer
        // refills the rings once the decision is out)
        if (redo && n_tiles > 0) mbar_wait(PVDONE(n_tiles - 1), ring_parity(n_tiles - 1));
        if (st == 0) {
          *s_redo = redo ? 1 : 0;
          mbar_arrive(DECIDE);
        }
        if (redo) {
          // second pass with the exact row maxima of the whole range (every
          // MMA is done: the P buffers are free)
          float* rb = reinterpret_cast<float*>(smem + C::kOffP);
#pragma unroll
          for (int j = 0; j < kRpt; ++j) {
            rb[(row0 + j) * 128 + kl] = ex[j];
            lp[j] = 0.f;
          }
          redo_references<kRpt>(kl, row0, st, quarter, lane, rb, row_a, row_ref);
          if (kRefRegs) {
            const float4* rr4 = reinterpret_cast<const float4*>(row_ref + row0);
#pragma unroll
            for (int j4 = 0; j4 < (kRefRegs ? kRpt / 4 : 0); ++j4) {
              const float4 x = rr4[j4];
              ref[(4 * j4 + 0) % (kRefRegs ? kRpt : 1)] = x.x;
              ref[(4 * j4 + 1) % (kRefRegs ? kRpt : 1)] = x.y;
              ref[(4 * j4 + 2) % (kRefRegs ? kRpt : 1)] = x.z;
              ref[(4 * j4 + 3) % (kRefRegs ? kRpt : 1)] = x.w;
            }
          }
        }
      }
    }

    // ---- this CTA's partial, staged row-major for the rows' owners: row r =
    //      [O(128) | l per TMEM lane quarter (4) | m | pad]. The send, receive
    //      and score buffers sit in the K ring (32-row tile), free once the
    //      last S product was read: the l terms, the new keys' scores and the
    //      cluster arrival (relaxed: no data passes, it only orders execution)
    //      go ahead of the last PV product; the 64-row tile's buffers reach
    //      into the V ring, so it arrives after it.
    constexpr bool kEarlyArrive = C::kNewS + kR * C::kMaxNew * 4 <= C::kRingV;
    float* send = reinterpret_cast<float*>(smem + C::kSend);
    if (kEarlyArrive) asm volatile("barrier.cluster.arrive.relaxed.aligned;" ::: "memory");
    {
      // l of each row over this warp's 32 key lanes; the owner adds the four
      // quarters
      int lrow;
      const float lw = warp_rows_sum<kRpt>(lp, lane, lrow);
      if (kRpt == 32 || (lane & 1) == 0) send[(row0 + lrow) * kRowF + kRowL + quarter] = lw;
      if (quarter == 0 && lane < kRpt)
        send[(row0 + lane) * kRowF + kRowM] = n_tiles > 0 ? row_ref[row0 + lane] : -INFINITY;
    }
    float* s_new = reinterpret_cast<float*>(smem + C::kNewS);  // [my_rows][R] new-key scores
    if (n_tiles > 0) {
      // every MMA is done once the last PV is (PVDONE's phases complete in order)
      const int Tl = (redo ? 2 : 1) * n_tiles - 1;
      mbar_wait(PVDONE(Tl), ring_parity(Tl));
      tc_fence_after();
    }
    if (!kEarlyArrive) asm volatile("barrier.cluster.arrive.relaxed.aligned;" ::: "memory");
#pragma unroll
    for (int j0 = 0; j0 < kRpt; j0 += 16) {
      uint32_t o[16];
      if (n_tiles > 0) {
        tmem_ld16(tmem_o + row0 + j0 + lane_off, o);
      } else {
#pragma unroll
        for (int j = 0; j < 16; ++j) o[j] = 0u;
      }
#pragma unroll
      for (int j = 0; j < 16; ++j) send[(row0 + j0 + j) * kRowF + kl] = __uint_as_float(o[j]);
    }
    // this warp's last tensor-memory read is done: the allocating warp frees the
    // columns while the partials merge (the kernel's end is not held by it)
    tc_fence_before();
    __syncwarp();
    if (lane == 0) mbar_arrive(TMEMDONE);
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    named_bar_sync(2, kSoftThreads);
    if (st == 0) mbar_expect_tx(RECV, static_cast<uint32_t>(csize * my_rows * kRowBytes));
    cluster_wait();  // every peer's ring is free to receive
    // softmax warp w sends rank c's rows to rank c (c = w, w + 8), into its
    // slots [rank * rpc, ...); one elected lane of the converged warp issues
    if (elect_one()) {
#pragma unroll 1
      for (int c = warp - 2; c < csize; c += kSoftWarps)
        if (rows_of(c) > 0)
          bulk_copy_s2s(cluster_map(base + C::kRecv + rank * rpc * kRowBytes, c),
                        base + C::kSend + c * rpc * kRowBytes, static_cast<uint32_t>(rows_of(c) * kRowBytes),
                        cluster_map(RECV, c));
      asm volatile("cp.async.bulk.commit_group;" ::: "memory");
    }
    __syncwarp();
    // While the partials travel: the scores of the R new keys against the
    // rows this CTA merges, on the CUDA cores from the rotated rows in shared
    // memory (query tile, new key rows): 8 lanes a dot product, 16 d each,
    // fp32 sums of the bf16 products. Scaled to log2 units; causal: row p =
    // i * G + g sees new keys 0..i; the block mask: all R. Every lane of a warp
    // runs the loop and the shuffles (the warp's 4 dot products of an
    // iteration may run past the last one).
    const int n_new = (kNew && valid) ? a.R : 0;
    const int n_dots = my_rows * n_new;
#pragma unroll 1
    for (int base0 = (st >> 5) * 4; kNew && base0 < n_dots; base0 += kSoftThreads / 8) {  // warp-uniform
      const int dot = base0 + (lane >> 3), sub = lane & 7;
      const bool act = dot < n_dots;
      const int rr = act ? dot / n_new : 0, n = act ? dot - rr * n_new : 0, row = mrow0 + rr;
      float acc = 0.f;
#pragma unroll
      for (int u = 0; u < 2; ++u) {
        const int c = sub + 8 * u;
        const uint4 qw = *reinterpret_cast<const uint4*>(smem + C::kOffQ + (c >> 3) * C::kQHalf + row * 128 +
                                                         (((c & 7) ^ (row & 7)) << 4));
        const uint4 kw = *reinterpret_cast<const uint4*>(smem + C::kOffNewK + n * kNewRow + c * 16);
        acc = fmaf(sd_bf16_lo(qw.x), sd_bf16_lo(kw.x), acc);
        acc = fmaf(sd_bf16_hi(qw.x), sd_bf16_hi(kw.x), acc);
        acc = fmaf(sd_bf16_lo(qw.y), sd_bf16_lo(kw.y), acc);
        acc = fmaf(sd_bf16_hi(qw.y), sd_bf16_hi(kw.y), acc);
        acc = fmaf(sd_bf16_lo(qw.z), sd_bf16_lo(kw.z), acc);
        acc = fmaf(sd_bf16_hi(qw.z), sd_bf16_hi(kw.z), acc);
        acc = fmaf(sd_bf16_lo(qw.w), sd_bf16_lo(kw.w), acc);
        acc = fmaf(sd_bf16_hi(qw.w), sd_bf16_hi(kw.w), acc);
      }
#pragma unroll
      for (int sh = 1; sh < 8; sh <<= 1) acc += __shfl_xor_sync(0xffffffffu, acc, sh);
      const int p = mblock * kR + row;
      if (act && sub == 0)
        s_new[rr * n_new + n] = (p < a.M && (block || n <= gdiv(p))) ? acc * a.scale_log2 : -INFINITY;
    }
    if (kFused && valid) {
      // while the partials travel: every CTA of the cluster read the raw rows
      // before its tiles (the cluster barrier above is behind all of them), so
      // the rotated query rows this CTA merges go back to q, and the head's
      // last reader of the raw key rows writes the rotated ones back to k_new
#pragma unroll 1
      for (int idx = st; idx < my_rows * 16; idx += kSoftThreads) {
        const int row = mrow0 + idx / 16, c = idx % 16;
        const int p = mblock * kR + row;
        if (p >= a.M) continue;
        const uint4 v = *reinterpret_cast<const uint4*>(smem + C::kOffQ + (c >> 3) * C::kQHalf + row * 128 +
                                                        (((c & 7) ^ (row & 7)) << 4));
        *reinterpret_cast<uint4*>(a.qw + ((static_cast<long long>(b) * a.R + gdiv(p)) * a.Hq + kvh * a.G +
                                          (p - gdiv(p) * a.G)) * kD + c * 8) = v;
      }
      // 32 rows: one m-block, one cluster, so its last rank
      bool write_k = rank == csize - 1 && mblock == 0;
      if constexpr (kR == 64) write_k = *s_kvlast != 0;
      if (write_k) {
#pragma unroll 1
        for (int idx = st; idx < a.R * 16; idx += kSoftThreads) {
          const int i = idx / 16, c = idx % 16;
          const long long src = ((static_cast<long long>(b) * a.R + i) * a.Hkv + kvh) * kD + c * 8;
          *reinterpret_cast<uint4*>(a.k_new + src) =
              *reinterpret_cast<const uint4*>(smem + C::kOffNewK + i * kNewRow + c * 16);
        }
        if (kR == 64 && a.n_mblocks > 1 && st == 0) a.kv_ticket[b * a.Hkv + kvh] = 0;  // re-armed
      }
    }
    // ---- merge of the rows this CTA owns; slot c * rpc + rr came from rank c.
    // 64 threads a row, two adjacent d a thread. While the partials travel,
    // the new keys' part: with M = max(the row's reference, its new-key
    // scores), sum_n w_n v_n and sum_n w_n, w_n = 2^(s_n - M). When every rank
    // used the row's reference (the common case: the second pass is rare), the
    // partials then add with the one weight 2^(ref - M); otherwise every
    // partial takes its own weight.
    named_bar_sync(2, kSoftThreads);  // every new-key score is in s_new
    const int rr = st >> 6, d = 2 * (st & 63);  // my_rows <= 4 here; more rows loop below
    float nx = 0.f, ny = 0.f, nl = 0.f, mloc = -INFINITY, rref = -INFINITY;
    if (rr < my_rows) {
      rref = n_tiles > 0 ? row_ref[mrow0 + rr] : -INFINITY;
      mloc = rref;
      const float* sn = s_new + rr * a.R;
#pragma unroll 1
      for (int n = 0; n < n_new; ++n) mloc = fmaxf(mloc, sn[n]);
      const float msub = mloc == -INFINITY ? 0.f : mloc;
#pragma unroll 4
      for (int n = 0; n < n_new; ++n) {
        const float w = ex2(sn[n] - msub);
        const uint32_t v2 = *reinterpret_cast<const uint32_t*>(smem + C::kOffNewV + n * kNewRow + d * 2);
        nl += w;
        nx = fmaf(w, sd_bf16_lo(v2), nx);
        ny = fmaf(w, sd_bf16_hi(v2), ny);
      }
    }
    mbar_wait(RECV, 0);
    const float* recv = reinterpret_cast<const float*>(smem + C::kRecv);
#pragma unroll 1
    for (int r = rr; r < my_rows; r += kSoftThreads / 64) {  // warp-uniform
      if (r != rr) {
        // rows beyond the first four (clusters of fewer than 8): their new keys here
        rref = n_tiles > 0 ? row_ref[mrow0 + r] : -INFINITY;
        mloc = rref;
        nx = ny = nl = 0.f;
        const float* sn = s_new + r * a.R;
        if constexpr (kR == 64) {
          // unrolled: the shared-memory loads of several keys issue together
          // (a rolled loop waits on each in turn, ~0.03 us a row and key: up
          // to 64 rows x 17 keys of a K = 16 block on one CTA)
#pragma unroll 4
          for (int n = 0; n < n_new; ++n) mloc = fmaxf(mloc, sn[n]);
          const float msub = mloc == -INFINITY ? 0.f : mloc;
#pragma unroll 4
          for (int n = 0; n < n_new; ++n) {
            const float w = ex2(sn[n] - msub);
            const uint32_t v2 = *reinterpret_cast<const uint32_t*>(smem + C::kOffNewV + n * kNewRow + d * 2);
            nl += w;
            nx = fmaf(w, sd_bf16_lo(v2), nx);
            ny = fmaf(w, sd_bf16_hi(v2), ny);
          }
        } else {
#pragma unroll 1
          for (int n = 0; n < n_new; ++n) mloc = fmaxf(mloc, sn[n]);
          const float msub = mloc == -INFINITY ? 0.f : mloc;
#pragma unroll 1
          for (int n = 0; n < n_new; ++n) {
            const float w = ex2(sn[n] - msub);
            const uint32_t v2 = *reinterpret_cast<const uint32_t*>(smem + C::kOffNewV + n * kNewRow + d * 2);
            nl += w;
            nx = fmaf(w, sd_bf16_lo(v2), nx);
            ny = fmaf(w, sd_bf16_hi(v2), ny);
          }
        }
      }
      const float* part = recv + r * kRowF;  // rank c's partial at part + c * rpc * kRowF
      float ox = 0.f, oy = 0.f, ls = 0.f;
      bool same = true;
#pragma unroll 4
      for (int c = 0; c < csize; ++c) {
        const float* pc = part + c * rpc * kRowF;
        const float2 o = *reinterpret_cast<const float2*>(pc + d);
        const float4 lq = *reinterpret_cast<const float4*>(pc + kRowL);
        same = same && pc[kRowM] == rref;
        ox += o.x;
        oy += o.y;
        ls += (lq.x + lq.y) + (lq.z + lq.w);
      }
      float wp = ex2(rref - (mloc == -INFINITY ? 0.f : mloc));  // ex2(-inf) = 0
      if (!same) {
        // some rank ran the second pass: weigh every partial by its own reference
        float mx = mloc;
#pragma unroll 1
        for (int c = 0; c < csize; ++c) mx = fmaxf(mx, part[c * rpc * kRowF + kRowM]);
        const float msub = mx == -INFINITY ? 0.f : mx;
        const float rescale = ex2((mloc == -INFINITY ? 0.f : mloc) - msub);  // the new keys' part was scaled by mloc
        nx *= rescale;
        ny *= rescale;
        nl *= rescale;
        ox = oy = ls = 0.f;
#pragma unroll 1
        for (int c = 0; c < csize; ++c) {
          const float* pc = part + c * rpc * kRowF;
          const float w = ex2(pc[kRowM] - msub);
          const float2 o = *reinterpret_cast<const float2*>(pc + d);
          const float4 lq = *reinterpret_cast<const float4*>(pc + kRowL);
          ox = fmaf(w, o.x, ox);
          oy = fmaf(w, o.y, oy);
          ls = fmaf(w, (lq.x + lq.y) + (lq.z + lq.w), ls);
        }
        wp = 1.f;
      }
      const float l = fmaf(wp, ls, nl);
      const int p = mblock * kR + mrow0 + r;
      if (valid && p < a.M && l > 0.f) {
        const float inv_l = 1.f / l;
        const int i = gdiv(p), gq = p - i * a.G;
        *reinterpret_cast<uint32_t*>(a.out + ((static_cast<long long>(b) * a.R + i) * a.Hq + kvh * a.G + gq) * kD +
                                     d) = cvt_bf16x2(fmaf(wp, ox, nx) * inv_l, fmaf(wp, oy, ny) * inv_l);
      }
    }
    if (elect_one()) asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory");
    __syncwarp();
  }
  // no CTA-wide barrier at the end: every warp leaves when its own work is
  // done (the softmax warps last: they wait for the partials coming in and for
  // their outgoing copies to have been read)
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

constexpr int kNumClusterSizes = 6;
constexpr int kClusterSizes[kNumClusterSizes] = {1, 2, 4, 6, 8, 16};

// per device: how many clusters of each size fit at once, for each row tile
// (index 0: 32 rows, 1: 64 rows)
struct DevState {
  bool ready = false;
  bool ok = false;
  int active[2][kNumClusterSizes] = {};
};

template <int kR>
bool set_attributes(int* active) {
  auto kern = verify_attn_tc_kernel<kR, 0>;
  auto kern_f = verify_attn_tc_kernel<kR, 1>;
  auto kern_n = verify_attn_tc_kernel<kR, 2>;
  auto kern_p = verify_attn_tc_kernel<kR, 3>;
  constexpr int smem = Cfg<kR>::kSmemBytes;
  if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) != cudaSuccess ||
      cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) != cudaSuccess ||
      cudaFuncSetAttribute(kern_f, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) != cudaSuccess ||
      cudaFuncSetAttribute(kern_f, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) != cudaSuccess ||
      cudaFuncSetAttribute(kern_n, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) != cudaSuccess ||
      cudaFuncSetAttribute(kern_n, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) != cudaSuccess ||
      cudaFuncSetAttribute(kern_p, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) != cudaSuccess ||
      cudaFuncSetAttribute(kern_p, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) != cudaSuccess) {
    (void)cudaGetLastError();
    return false;
  }
  for (int i = 0; i < kNumClusterSizes; ++i) {
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = kClusterSizes[i];
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.gridDim = dim3(kClusterSizes[i], 1, 1);
    cfg.blockDim = dim3(kThreads, 1, 1);
    cfg.dynamicSmemBytes = smem;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, reinterpret_cast<const void*>(kern), &cfg) != cudaSuccess) {
      (void)cudaGetLastError();
      n = 0;
    }
    active[i] = n;
  }
  return true;
}

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
    s.ok = set_attributes<32>(s.active[0]) && set_attributes<64>(s.active[1]);
  }
  return &s;
}

// Cluster size: minimise waves x (32-key blocks per CTA + a fixed per-CTA cost)
int pick_cluster(const int* active, long long units, int cap) {
  const long long nblk = (cap + 31) / 32;
  long long best_cost = -1;
  int best = 0;
  for (int i = 0; i < kNumClusterSizes; ++i) {
    const int cs = kClusterSizes[i];
    if (active[i] <= 0) continue;
    if (cs > 1 && nblk < 2LL * cs) continue;
    const long long waves = (units + active[i] - 1) / active[i];
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

// How the tcgen05 path runs a shape: row tile (32 or 64 packed query rows),
// m-blocks (row tiles per KV head) and cluster size; cs == 0: not served.
struct TcPlan {
  int rows = 0, mblocks = 0, cs = 0;
};

// Cluster size forced by sd_set_cluster_size (0: chosen per call).
static std::atomic<int> g_forced_cluster{0};

extern "C" sd_status sd_set_cluster_size(int cluster_size) {
  if (cluster_size == 0) {
    g_forced_cluster.store(0);
    return SD_OK;
  }
  for (int i = 0; i < kNumClusterSizes; ++i)
    if (kClusterSizes[i] == cluster_size) {
      g_forced_cluster.store(cluster_size);
      return SD_OK;
    }
  return SD_ERR_INVALID_ARG;
}

// rows64: the 64-row tile even for G * R <= 32 (the block-masked fused layer:
// the 32-row fused kernel is compiled causal only, and an N = 64 product
// costs about what an N = 32 one does)
static TcPlan tc_plan(int B, int R, int Hq, int Hkv, int D, int cap, int max_cs = 16, bool rows64 = false) {
  TcPlan p;
  if (!tc_enabled() || D != kD || Hkv <= 0 || Hq % Hkv || R <= 0) return p;
  const int M = (Hq / Hkv) * R;
  if (M > 2 * 64) return p;
  DevState* s = state();
  if (!s || !s->ok) return p;
  p.rows = M <= 32 && !rows64 ? 32 : 64;
  p.mblocks = (M + p.rows - 1) / p.rows;
  const int* active = s->active[p.rows == 32 ? 0 : 1];
  // sizes above max_cs are not used (the fused merge holds csize partials and
  // R new keys in the lanes of one warp)
  int capped[kNumClusterSizes];
  for (int i = 0; i < kNumClusterSizes; ++i) capped[i] = kClusterSizes[i] <= max_cs ? active[i] : 0;
  const int forced = g_forced_cluster.load();
  for (int i = 0; i < kNumClusterSizes && forced > 0; ++i)
    if (kClusterSizes[i] == forced && capped[i] > 0) p.cs = forced;
  if (p.cs == 0) p.cs = pick_cluster(capped, static_cast<long long>(B) * Hkv * p.mblocks, cap);
  return p;
}

bool sd_internal_tc_serves(int B, int R, int Hq, int Hkv, int D, int cap) {
  return tc_plan(B, R, Hq, Hkv, D, cap).cs > 0;
}

bool sd_internal_tc_serves_layer(int B, int R, int Hq, int Hkv, int D, int cap, bool block) {
  if (R > 32) return false;
  const TcPlan plan = tc_plan(B, R, Hq, Hkv, D, cap, 32 - R, block);
  return plan.cs > 0 && R <= (plan.rows == 32 ? Cfg<32>::kMaxNew : Cfg<64>::kMaxNew);
}

template <int kR, int kMode>
static sd_status launch_tc(const sd_kv_cache* cache, const TcArgs& a, const RopeTable& tab,
                           const TcPlan& plan, bool pdl, cudaStream_t stream) {
  const int B = cache->batch, Hkv = cache->n_kv_heads, cap = cache->capacity;
  CUtensorMap k128, v128;
  if (!make_map(&k128, cache->k, cap, B * Hkv, 128) || !make_map(&v128, cache->v, cap, B * Hkv, 128))
    return SD_ERR_CUDA;
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = plan.cs;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.gridDim = dim3(plan.cs, Hkv * plan.mblocks, B);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = Cfg<kR>::kSmemBytes;
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 2 : 1;
  if (cudaLaunchKernelEx(&cfg, verify_attn_tc_kernel<kR, kMode>, k128, v128, a, tab) != cudaSuccess) {
    (void)cudaGetLastError();
    return SD_ERR_CUDA;
  }
  return SD_OK;
}

template <int kMode>
static sd_status launch_plan(const sd_kv_cache* cache, const TcArgs& a, const RopeTable& tab,
                             const TcPlan& plan, bool pdl, cudaStream_t stream) {
  return plan.rows == 32 ? launch_tc<32, kMode>(cache, a, tab, plan, pdl, stream)
                         : launch_tc<64, kMode>(cache, a, tab, plan, pdl, stream);
}

// Routed here by sd_verify_attention for head_dim 128 and G * R <= 128. Up to
// kMaxNew new rows (and cluster sizes with csize + R <= 32) take the kernel
// whose tensor-core loop covers the prefix only and whose new rows enter as
// S_new (as in the fused layer), with the prefix optionally streamed before
// the dependency wait (SD_ATTN_PREFIX_EARLY); other shapes take the kernel
// whose loop covers every key (the flag is then a promise it does not need).
sd_status sd_internal_verify_attention_tc(const void* q, const sd_kv_cache* cache, void* out,
                                          int R, int Hq, float scale_log2, int flags, cudaStream_t stream,
                                          bool* handled) {
  *handled = false;
  const int B = cache->batch, Hkv = cache->n_kv_heads;
  const bool block = (flags & SD_ATTN_BLOCK_MASK) != 0, early = (flags & SD_ATTN_PREFIX_EARLY) != 0;
  TcPlan plan;
  int mode = 0;
  if (R <= 32) {
    plan = tc_plan(B, R, Hq, Hkv, cache->head_dim, cache->capacity, 32 - R);
    if (plan.cs > 0 && R <= (plan.rows == 32 ? Cfg<32>::kMaxNew : Cfg<64>::kMaxNew)) mode = 2;
  }
  if (mode == 0) plan = tc_plan(B, R, Hq, Hkv, cache->head_dim, cache->capacity);
  if (plan.cs <= 0) return SD_OK;
  TcArgs a = {};
  a.q = static_cast<const __nv_bfloat16*>(q);
  a.out = static_cast<__nv_bfloat16*>(out);
  a.len = cache->len;
  a.kc = static_cast<__nv_bfloat16*>(cache->k);
  a.vc = static_cast<__nv_bfloat16*>(cache->v);
  a.R = R;
  a.Hq = Hq;
  a.Hkv = Hkv;
  a.G = Hq / Hkv;
  a.M = a.G * R;
  a.inv_g = 1.0f / static_cast<float>(a.G);
  a.cap = cache->capacity;
  a.n_mblocks = plan.mblocks;
  a.scale_log2 = scale_log2;
  RopeTable tab = {};
  *handled = true;
  if (mode == 2) {
    a.early = (early ? 1 : 0) | (block ? 2 : 0);
    // a programmatic dependent launch either way: without the flag the kernel
    // waits before its first global access, so only its launch and set-up
    // (barriers, tensor memory) overlap the kernel before it
    return launch_plan<2>(cache, a, tab, plan, true, stream);
  }
  a.early = block ? 1 : 0;  // the all-keys kernel's block mask
  return launch_plan<0>(cache, a, tab, plan, false, stream);
}

// The fused verify layer (rope + append + attention) on the tcgen05 path.
sd_status sd_internal_verify_layer_tc(void* q, void* k_new, const void* v_new, const int32_t* pos,
                                      const RopeTable& tab, const sd_kv_cache* cache, void* out,
                                      int R, int Hq, float scale_log2, uint32_t* ticket, int early,
                                      int block, cudaStream_t stream, bool* handled) {
  *handled = false;
  const int B = cache->batch, Hkv = cache->n_kv_heads;
  // the new rows are held in shared memory (16 with the 32-row tile, 32 with
  // the 64-row tile) and merged in the lanes of one warp with the partials
  if (R > 32) return SD_OK;
  // block-masked layers take the 64-row tile (the 32-row fused kernel is causal only)
  const TcPlan plan = tc_plan(B, R, Hq, Hkv, cache->head_dim, cache->capacity, 32 - R, block != 0);
  if (plan.cs <= 0) return SD_OK;
  if (R > (plan.rows == 32 ? Cfg<32>::kMaxNew : Cfg<64>::kMaxNew)) return SD_OK;
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
  a.kv_ticket = ticket + B;
  a.early = (early ? 1 : 0) | (block ? 2 : 0);  // prefix before the wait; the block mask
  a.R = R;
  a.Hq = Hq;
  a.Hkv = Hkv;
  a.G = Hq / Hkv;
  a.M = a.G * R;
  a.inv_g = 1.0f / static_cast<float>(a.G);
  a.cap = cache->capacity;
  a.n_mblocks = plan.mblocks;
  a.scale_log2 = scale_log2;
  *handled = true;
  if (early) return launch_plan<1>(cache, a, tab, plan, true, stream);
  // dependent as well: the wait comes before any global access (the draft's
  // single-row steps, each reading the length the step before advanced)
  return launch_plan<3>(cache, a, tab, plan, true, stream);
}
