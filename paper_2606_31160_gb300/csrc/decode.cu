// The fused verify layer (M-RoPE of Sec. 3.3 / Sec. 4.2 + the KV append of
// Eq. commit + the verify attention of Eq. verify, Sec. 3.2) on small packed
// row tiles: the G * R query rows that share a KV head fit one 16-row tile,
// as in the draft's single-row decode steps (Eq. propose: R = 1, G = 4) and
// short verify blocks. The library sends it the block-masked short layers
// (the tcgen05 layer kernel's 32-row tile is causal only); the causal ones
// run faster on the tcgen05 kernel's 128-key tensor-memory products (see the
// routing note at layer_preferred below).
//
// Such a tile carries too few rows to pay for a 128-key tensor-memory product
// per key tile, and one (scene, KV head) holds too few keys to keep more than
// a few SMs busy. So every KV head gets a thread-block cluster of up to 16
// CTAs, sized so that the launch covers the GPU in one wave; each CTA takes a
// contiguous run of 32-key blocks of the head's keys and streams them through
// an 8-slot ring (TMA boxes of 32 rows x 64 columns, 128-byte swizzle, K and V
// of a block on one barrier); eight consumer warps each take every eighth
// block of the run:
//   S = Q K^T over the block's 32 keys     (mma.sync m16n8k16 bf16, fp32 sums)
//   online softmax per row, in registers   (P never leaves registers)
//   O += P V                               (mma.sync m16n8k16 bf16)
// The warps' (m, l, O) states merge in shared memory, then the CTAs' states
// merge through distributed shared memory: each rank finishes an equal slice
// of the head's output elements.
//
// In the fused layer every CTA rotates the query rows itself (a cos / sin
// table per (row, pair) in shared memory, the same arithmetic as the rotation
// kernel, so the bits match); the cluster's last CTA also rotates the R new
// keys, keeps them with the new values as one more block in shared memory
// (never re-read from the cache), writes both to the cache and the rotated
// keys back to k_new; rank 0 writes the rotated query rows back once every
// rank has read the raw ones; the last CTA of a scene to read len[b] advances
// it by R (a per-scene ticket in the caller's workspace).
//
// Launches are programmatic dependent launches. Without the early flag every
// thread waits for the preceding kernel before it touches memory; with it
// (the caller's promise that the preceding kernel writes neither this cache,
// nor its len, nor pos) len, pos and the prefix blocks are read before the
// wait and the query / new rows after it. Every mbarrier wait is bounded
// (SD_DEVERR_TIMEOUT instead of a hang).
#include "common.cuh"

#include <cuda.h>  // CUtensorMap and its enums (header only; no libcuda link)

#include <math.h>
#include <mutex>

SD_DEFINE_ERROR_ACCESSOR(sd_take_error_decode)

namespace {

constexpr int kD = 128;                    // head dim
constexpr int kBlk = 32;                   // keys per block (one TMA box height)
constexpr int kHalfBytes = kBlk * 128;     // one 64-column half of a block's K (or V): 4 KB
constexpr int kKVBytes = 2 * kHalfBytes;   // K (or V) of a block: 8 KB
constexpr int kSlotBytes = 2 * kKVBytes;   // K then V: 16 KB
constexpr int kSlots = 8;
constexpr int kRows = 16;                  // packed query rows (one m16 tile)
constexpr int kMaxNew = 16;                // new rows the fused layer takes
constexpr int kCW = 8;                     // consumer warps
constexpr int kCT = 32 * kCW;
constexpr int kThreads = kCT + 32;         // + the producer warp
constexpr int kMaxCluster = 16;
constexpr uint32_t kSpinLimit = 1u << 20;
constexpr int kLd = kD + 4;                     // padded fp32 row of a partial
constexpr int kPartFloats = kRows * kLd + 2 * kRows;  // (O, m, l) of 16 rows

// shared memory (offsets from a 1024-aligned base)
constexpr int kQHalf = kRows * 128;                         // 2 KB
constexpr int kOffQ = kSlots * kSlotBytes;                  // 128 KB of ring first
constexpr int kOffNew = kOffQ + 2 * kQHalf;                 // new K block, then new V block
constexpr int kOffPart = kOffNew + kSlotBytes;              // this CTA's (O, m, l)
constexpr int kOffCs = kOffPart + kPartFloats * 4;          // (cos, sin) [kMaxNew][64]
constexpr int kOffMm = kOffCs + kMaxNew * 64 * 8;           // peers' m [kMaxCluster][kRows]
constexpr int kOffLl = kOffMm + kMaxCluster * kRows * 4;    // peers' l
constexpr int kOffW = kOffLl + kMaxCluster * kRows * 4;     // merge weights
constexpr int kOffInvL = kOffW + kMaxCluster * kRows * 4;   // 1 / l per row
constexpr int kOffRed = kOffInvL + kRows * 4;               // [groups][slots] float4
constexpr int kRedBytes = kCT * 16;
constexpr int kOffBar = kOffRed + kRedBytes;                // full[kSlots], empty[kSlots]
constexpr int kSmemBytes = kOffBar + 2 * kSlots * 8 + 1024;  // + alignment slack
static_assert(kOffQ % 1024 == 0 && kOffNew % 1024 == 0, "swizzled regions are 1024-aligned");
static_assert(kCW * kPartFloats * 4 <= kOffQ, "warp partials overlay the ring");
static_assert(kSmemBytes <= 227 * 1024, "shared memory budget");

struct DecArgs {
  __nv_bfloat16* q;          // query rows: rotated (attention) or raw, rotated in place (layer)
  __nv_bfloat16* out;
  int32_t* len;
  __nv_bfloat16* k_new;      // layer: raw new key rows [B][R][Hkv][D], rotated in place
  const __nv_bfloat16* v_new;
  __nv_bfloat16* kc;         // layer: cache K / V [B][Hkv][cap][D] (append target)
  __nv_bfloat16* vc;
  const int32_t* pos;        // layer: [B][R][3]
  uint32_t* ticket;          // layer: [B] per-scene read tickets (zeroed, re-armed)
  int R, Hq, Hkv, G, M, cap;
  int early;                 // len, pos and the prefix may be read before the wait
  int block;                 // every new row sees all R new rows
  float scale_log2;          // softmax scale * log2(e)
};

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

__device__ __forceinline__ void mma_bf16(float (&c)[4], const uint32_t (&a)[4], uint32_t b0,
                                         uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
      "{%8,%9}, {%0,%1,%2,%3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
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

__device__ __forceinline__ void cluster_arrive_relaxed() {
  asm volatile("barrier.cluster.arrive.relaxed.aligned;" ::: "memory");
}

__device__ __forceinline__ void cluster_wait() {
  asm volatile("barrier.cluster.wait.aligned;" ::: "memory");
}

__device__ __forceinline__ uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}

// Address of the same shared-memory location in CTA `rank` of the cluster.
__device__ __forceinline__ uint32_t peer_addr(uint32_t local, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(local), "r"(rank));
  return r;
}

__device__ __forceinline__ float ld_peer_f32(uint32_t addr) {
  float v;
  asm volatile("ld.shared::cluster.f32 %0, [%1];" : "=f"(v) : "r"(addr) : "memory");
  return v;
}

__device__ __forceinline__ float4 ld_peer_f32x4(uint32_t addr) {
  float4 v;
  asm volatile("ld.shared::cluster.v4.f32 {%0,%1,%2,%3}, [%4];"
               : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
               : "r"(addr)
               : "memory");
  return v;
}

__device__ __forceinline__ uint32_t atom_add_acq_rel(uint32_t* p, uint32_t v) {
  uint32_t old;
  asm volatile("atom.acq_rel.gpu.global.add.u32 %0, [%1], %2;" : "=r"(old) : "l"(p), "r"(v) : "memory");
  return old;
}

__device__ __forceinline__ void griddep_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void griddep_launch() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

__device__ __forceinline__ void st_shared_zero16(uint32_t addr) {
  asm volatile("st.shared.v4.u32 [%0], {%1,%1,%1,%1};" ::"r"(addr), "r"(0) : "memory");
}

// 128-byte swizzle of a [rows][128 B] region whose base is 1024-byte aligned:
// 16-byte chunk c of row r sits at chunk c ^ (r & 7) (the layout TMA's
// SWIZZLE_128B writes and every ldmatrix below reads).
__device__ __forceinline__ uint32_t swz(int row, int chunk) {
  return static_cast<uint32_t>(row * 128 + ((chunk ^ (row & 7)) << 4));
}

// Rotate one 16-byte chunk (4 adjacent pairs) with the (cos, sin) of its pairs.
__device__ __forceinline__ uint4 rotate_chunk(uint4 w, const float2* cs) {
  w.x = sd_rope_pair(w.x, cs[0].x, cs[0].y);
  w.y = sd_rope_pair(w.y, cs[1].x, cs[1].y);
  w.z = sd_rope_pair(w.z, cs[2].x, cs[2].y);
  w.w = sd_rope_pair(w.w, cs[3].x, cs[3].y);
  return w;
}

// --------------------------------------------------------------------------
// Kernel body: len[b] is the prefix length, the new rows come from q /
// k_new / v_new. Grid: (cluster size, Hkv, B), one cluster per (scene, KV
// head).
//
// `issued`: prefix blocks the producer already issued before the dependency wait.
// --------------------------------------------------------------------------
__device__ __forceinline__ void decode_body(const CUtensorMap* tm_k, const CUtensorMap* tm_v,
                                            const DecArgs& a, const RopeTable& tab, uint8_t* smem,
                                            int issued) {
  const uint32_t base = smem_addr(smem);
  const uint32_t qs = base + kOffQ;
  const uint32_t new_k = base + kOffNew;
  const uint32_t new_v = new_k + kKVBytes;
  float* part = reinterpret_cast<float*>(smem + kOffPart);
  float2* cs_tab = reinterpret_cast<float2*>(smem + kOffCs);
  auto full_bar = [&](int s) { return base + kOffBar + 8u * s; };
  auto empty_bar = [&](int s) { return base + kOffBar + 8u * (kSlots + s); };

  const int C = static_cast<int>(gridDim.x);
  const int rank = static_cast<int>(cluster_rank());
  const int h = blockIdx.y;
  const int b = blockIdx.z;
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int tid = threadIdx.x;
  const bool early = a.early != 0;
  const int R = a.R, G = a.G, M = a.M;
  const bool last_rank = rank == C - 1;

  // ---- one global round trip before any arithmetic: len, and (consumer
  // threads) the positions, this thread's query-row chunk and, on the layer's
  // last rank, its new key / value chunk, all issued together. Consumer
  // thread t owns chunk t & 15 of packed query row t >> 4 and of new row
  // t >> 4 (16 rows x 16 chunks of 16 bytes each).
  const int len_in = a.len[b];
  const int my_p = tid >> 4, my_c = tid & 15;
  uint4 qraw = make_uint4(0u, 0u, 0u, 0u), kraw = qraw, vraw = qraw;
  // the (t, h, w) coordinates of the rows of this thread's rotation-table
  // entries, loaded whole (the axis is chosen once they are in)
  int pv[kMaxNew * 64 / kCT][3];
  if (warp < kCW) {
    {
#pragma unroll
      for (int e = 0; e < kMaxNew * 64 / kCT; ++e) {
        const int idx = tid + kCT * e;
        const int* src = a.pos + (static_cast<long long>(b) * R + (idx >> 6)) * 3;
#pragma unroll
        for (int x = 0; x < 3; ++x) pv[e][x] = idx < R * 64 ? src[x] : 0;
      }
    }
    {
      if (early) griddep_wait();
      if (my_p < M) {
        const int i = my_p / G, gq = my_p - i * G;
        qraw = *reinterpret_cast<const uint4*>(a.q + ((static_cast<long long>(b) * R + i) * a.Hq + h * G + gq) *
                                                         kD + my_c * 8);
      }
      if (last_rank && my_p < R) {
        const long long row = (static_cast<long long>(b) * R + my_p) * a.Hkv + h;
        kraw = *reinterpret_cast<const uint4*>(a.k_new + row * kD + my_c * 8);
        vraw = *reinterpret_cast<const uint4*>(a.v_new + row * kD + my_c * 8);
      }
    }
  }

  int L_b, n_keys;  // prefix length; keys the rows see at most
  bool valid;
  {
    L_b = len_in;
    n_keys = len_in + R;
    valid = len_in >= 0 && len_in + R <= a.cap;
    if (!valid && tid == 0 && rank == 0 && h == 0) sd_set_error(SD_DEVERR_KV_OVERFLOW);
  }
  if (!valid) return;  // the whole cluster agrees (same len[b]); nothing was written
  if (tid == 0) {
    // the last CTA of the scene to read len[b] advances it (after every read)
    const uint32_t n_ctas = static_cast<uint32_t>(a.Hkv) * static_cast<uint32_t>(C);
    if (atom_add_acq_rel(a.ticket + b, 1u) == n_ctas - 1) {
      a.ticket[b] = 0;
      a.len[b] = L_b + R;
    }
  }

  // ---- this CTA's run of 32-key blocks of the prefix
  const int loop_keys = L_b;
  const int nblk = (loop_keys + kBlk - 1) / kBlk;
  const int blk_begin = static_cast<int>((static_cast<long long>(rank) * nblk) / C);
  const int blk_end = static_cast<int>((static_cast<long long>(rank + 1) * nblk) / C);
  const int n_run = blk_end - blk_begin;
  const bool has_new = last_rank;
  const int n_items = n_run + (has_new ? 1 : 0);  // the new-key block is the last item

  if (warp == kCW) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      const int z = b * a.Hkv + h;
      for (int j = issued; j < n_run; ++j) {
        const int s = j % kSlots;
        if (j >= kSlots && !mbar_wait(empty_bar(s), ((j / kSlots) - 1) & 1)) break;
        mbar_expect_tx(full_bar(s), kSlotBytes);
        const int y = (blk_begin + j) * kBlk;
        const uint32_t dst = base + s * kSlotBytes;
        tma_load_3d(dst, tm_k, full_bar(s), 0, y, z);
        tma_load_3d(dst + kHalfBytes, tm_k, full_bar(s), 64, y, z);
        tma_load_3d(dst + kKVBytes, tm_v, full_bar(s), 0, y, z);
        tma_load_3d(dst + kKVBytes + kHalfBytes, tm_v, full_bar(s), 64, y, z);
      }
    }
    __syncwarp();
  } else {
    // ------------------------------------------------------------ consumers
    {
      // (cos, sin) of every (new row, pair): the rotation kernel's arithmetic
#pragma unroll
      for (int e = 0; e < kMaxNew * 64 / kCT; ++e) {
        const int idx = tid + kCT * e;
        if (idx >= R * 64) break;
        const int ax = tab.axis[idx & 63];
        const int p = ax == 0 ? pv[e][0] : (ax == 1 ? pv[e][1] : pv[e][2]);
        cs_tab[idx] = sd_rope_cs(static_cast<float>(p), idx & 63, tab);
      }
      named_bar_sync(1, kCT);
    }
    // the packed query row chunk -> shared memory (swizzled like the K boxes),
    // rotated; padding rows are zero
    if (my_p < M) qraw = rotate_chunk(qraw, cs_tab + (my_p / G) * 64 + my_c * 4);
    asm volatile("st.shared.v4.u32 [%0], {%1,%2,%3,%4};" ::"r"(qs + (my_c >> 3) * kQHalf + swz(my_p, my_c & 7)),
                 "r"(qraw.x), "r"(qraw.y), "r"(qraw.z), "r"(qraw.w)
                 : "memory");
    if (has_new) {
      // the R new keys (rotated) and values as one more 32-key block (rows
      // past R zero); both go to the cache, the rotated keys back to k_new
      if (my_p < R) {
        kraw = rotate_chunk(kraw, cs_tab + my_p * 64 + my_c * 4);
        const long long row = (static_cast<long long>(b) * R + my_p) * a.Hkv + h;
        const long long crow = (static_cast<long long>(b) * a.Hkv + h) * a.cap + L_b + my_p;
        *reinterpret_cast<uint4*>(a.k_new + row * kD + my_c * 8) = kraw;
        *reinterpret_cast<uint4*>(a.kc + crow * kD + my_c * 8) = kraw;
        *reinterpret_cast<uint4*>(a.vc + crow * kD + my_c * 8) = vraw;
      }
      const uint32_t off = (my_c >> 3) * kHalfBytes + swz(my_p, my_c & 7);
      asm volatile("st.shared.v4.u32 [%0], {%1,%2,%3,%4};" ::"r"(new_k + off), "r"(kraw.x), "r"(kraw.y),
                   "r"(kraw.z), "r"(kraw.w)
                   : "memory");
      asm volatile("st.shared.v4.u32 [%0], {%1,%2,%3,%4};" ::"r"(new_v + off), "r"(vraw.x), "r"(vraw.y),
                   "r"(vraw.z), "r"(vraw.w)
                   : "memory");
      const uint32_t off2 = (my_c >> 3) * kHalfBytes + swz(my_p + 16, my_c & 7);
      st_shared_zero16(new_k + off2);
      st_shared_zero16(new_v + off2);
    }
    named_bar_sync(1, kCT);

    const int g8 = lane >> 2;
    const int t4 = lane & 3;
    const float sl = a.scale_log2;
    // ldmatrix lane roles
    const int a_row = (lane & 7) + ((lane >> 3) & 1) * 8;  // A (Q) and trans-B (V): row in 16
    const int a_chk = lane >> 4;                             // A: +0 / +1 chunk
    const int b_row = (lane & 7) + (lane >> 4) * 8;          // B (K): key row in 16
    const int b_chk = (lane >> 3) & 1;                       // B: +0 / +1 chunk

    // Q fragments of the 8 k16 steps stay in registers
    uint32_t qa[8][4];
#pragma unroll
    for (int kk = 0; kk < 8; ++kk)
      ldsm_x4(qs + (kk >> 2) * kQHalf + swz(a_row, (kk & 3) * 2 + a_chk), qa[kk][0], qa[kk][1],
              qa[kk][2], qa[kk][3]);

    // last visible key of each of this thread's two rows (g8, g8 + 8): in the
    // cached blocks and, for the layer's new block, among the new keys
    int lim[2], lim_new[2];
#pragma unroll
    for (int hh = 0; hh < 2; ++hh) {
      const int p = g8 + 8 * hh;
      const int i = p < M ? p / G : R - 1;
      lim[hh] = L_b - 1;
      lim_new[hh] = a.block ? R - 1 : i;
    }
    // smallest limit over the rows; last key read (values past it are zeroed)
    const int mask_from = L_b - 1;
    const int last_key = L_b - 1;

    float o[16][4];
#pragma unroll
    for (int nd = 0; nd < 16; ++nd)
#pragma unroll
      for (int c = 0; c < 4; ++c) o[nd][c] = 0.f;
    float m_run[2] = {-INFINITY, -INFINITY}, l_run[2] = {0.f, 0.f};  // m in raw score units

    for (int j = warp; j < n_items; j += kCW) {
      const bool is_new = has_new && j == n_run;
      const int s = j % kSlots;
      uint32_t kb, vb;
      int key0;
      if (is_new) {
        kb = new_k;
        vb = new_v;
        key0 = 0;
      } else {
        if (!mbar_wait(full_bar(s), (j / kSlots) & 1)) break;
        kb = base + s * kSlotBytes;
        vb = kb + kKVBytes;
        key0 = (blk_begin + j) * kBlk;
        // stale rows past the last key (cache rows not yet written, possibly
        // NaN): zero their values so a zero weight gives zero
        if (key0 + kBlk - 1 > last_key) {
          const int first = max(last_key + 1 - key0, 0);
          for (int cidx = lane; cidx < (kBlk - first) * 16; cidx += 32) {
            const int r = first + (cidx >> 4), rem = cidx & 15;
            st_shared_zero16(vb + (rem >> 3) * kHalfBytes + r * 128 + (rem & 7) * 16);
          }
          __syncwarp();
        }
      }
      // ---- S = Q K^T over the block's 32 keys (4 n8 tiles); even and odd
      //      k16 steps accumulate apart (two dependent chains of 4, not 8)
      float sc[4][4], sc2[4][4];
#pragma unroll
      for (int nt = 0; nt < 4; ++nt)
#pragma unroll
        for (int c = 0; c < 4; ++c) sc[nt][c] = sc2[nt][c] = 0.f;
#pragma unroll
      for (int kk = 0; kk < 8; ++kk) {
        const uint32_t kh = kb + (kk >> 2) * kHalfBytes;
        const int chunk = (kk & 3) * 2;
        uint32_t kf[2][4];
#pragma unroll
        for (int np = 0; np < 2; ++np)
          ldsm_x4(kh + swz(np * 16 + b_row, chunk + b_chk), kf[np][0], kf[np][1], kf[np][2], kf[np][3]);
        float (&acc)[4][4] = (kk & 1) ? sc2 : sc;
#pragma unroll
        for (int np = 0; np < 2; ++np) {
          mma_bf16(acc[2 * np], qa[kk], kf[np][0], kf[np][1]);
          mma_bf16(acc[2 * np + 1], qa[kk], kf[np][2], kf[np][3]);
        }
      }
#pragma unroll
      for (int nt = 0; nt < 4; ++nt)
#pragma unroll
        for (int c = 0; c < 4; ++c) sc[nt][c] += sc2[nt][c];
      // ---- masks: the new block always, cached blocks only past the prefix
      if (is_new || key0 + kBlk - 1 > mask_from) {
#pragma unroll
        for (int nt = 0; nt < 4; ++nt)
#pragma unroll
          for (int c = 0; c < 4; ++c) {
            const int key = key0 + nt * 8 + 2 * t4 + (c & 1);
            const int lm = is_new ? lim_new[c >> 1] : lim[c >> 1];
            if (key > lm) sc[nt][c] = -INFINITY;
          }
      }
      // ---- online softmax (row maximum over the block; lazy O rescale)
      float m_new[2];
      bool grow = false;
#pragma unroll
      for (int hh = 0; hh < 2; ++hh) {
        float mx = -INFINITY;
#pragma unroll
        for (int nt = 0; nt < 4; ++nt) mx = fmaxf(mx, fmaxf(sc[nt][2 * hh], sc[nt][2 * hh + 1]));
        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 2));
        m_new[hh] = fmaxf(m_run[hh], mx);
        grow |= (m_run[hh] != -INFINITY) && (m_new[hh] > m_run[hh]);
      }
      if (__any_sync(0xffffffffu, grow)) {
#pragma unroll
        for (int hh = 0; hh < 2; ++hh) {
          const float corr = m_run[hh] == -INFINITY ? 1.f : ex2((m_run[hh] - m_new[hh]) * sl);
          l_run[hh] *= corr;
#pragma unroll
          for (int nd = 0; nd < 16; ++nd) {
            o[nd][2 * hh] *= corr;
            o[nd][2 * hh + 1] *= corr;
          }
        }
      }
      uint32_t pa[2][4];  // P as A fragments of the two k16 steps
#pragma unroll
      for (int hh = 0; hh < 2; ++hh) {
        m_run[hh] = m_new[hh];
        const float mb = m_new[hh] == -INFINITY ? 0.f : m_new[hh] * sl;
        float rs = 0.f;
#pragma unroll
        for (int nt = 0; nt < 4; ++nt) {
          const uint32_t w = sd_pack_bf16x2(ex2(fmaf(sc[nt][2 * hh], sl, -mb)),
                                            ex2(fmaf(sc[nt][2 * hh + 1], sl, -mb)));
          rs += sd_bf16_lo(w) + sd_bf16_hi(w);  // normaliser of the bf16 weights used
          pa[nt >> 1][(nt & 1) * 2 + hh] = w;
        }
        l_run[hh] += rs;
      }
      // ---- O += P V (two k16 steps)
#pragma unroll
      for (int k2 = 0; k2 < 2; ++k2) {
#pragma unroll
        for (int dp = 0; dp < 8; ++dp) {
          uint32_t v0, v1, v2, v3;
          ldsm_x4_t(vb + (dp >> 2) * kHalfBytes + swz(k2 * 16 + a_row, (dp & 3) * 2 + a_chk), v0, v1, v2,
                    v3);
          mma_bf16(o[2 * dp], pa[k2], v0, v1);
          mma_bf16(o[2 * dp + 1], pa[k2], v2, v3);
        }
      }
      if (!is_new) {
        __syncwarp();
        if (lane == 0) mbar_arrive(empty_bar(s));
      }
    }

    // ---- per-warp partials -> shared memory (over the ring: every block was
    //      consumed once all consumer warps pass this barrier)
    named_bar_sync(1, kCT);
    float* wp = reinterpret_cast<float*>(smem) + warp * kPartFloats;
#pragma unroll
    for (int hh = 0; hh < 2; ++hh) {
      float l = l_run[hh];
      l += __shfl_xor_sync(0xffffffffu, l, 1);
      l += __shfl_xor_sync(0xffffffffu, l, 2);
      const int r = g8 + 8 * hh;
#pragma unroll
      for (int nd = 0; nd < 16; ++nd)
        *reinterpret_cast<float2*>(wp + r * kLd + nd * 8 + 2 * t4) = make_float2(o[nd][2 * hh], o[nd][2 * hh + 1]);
      if (t4 == 0) {
        wp[kRows * kLd + r] = m_run[hh] == -INFINITY ? -INFINITY : m_run[hh] * sl;
        wp[kRows * kLd + kRows + r] = l;
      }
    }
    named_bar_sync(1, kCT);
    // ---- the eight warps' weights per row: thread (row, warp) = (tid >> 3,
    //      tid & 7) of the first four warps, maximum and sum over the row's
    //      eight lanes by shuffles; m in log2 units from here on
    const float* wpart = reinterpret_cast<const float*>(smem);
    float* wf = reinterpret_cast<float*>(smem + kOffW);  // [kRows][kCW]
    if (tid < kRows * kCW) {
      const int row = tid >> 3, w = tid & 7;
      const float mw = wpart[w * kPartFloats + kRows * kLd + row];
      const float lw = wpart[w * kPartFloats + kRows * kLd + kRows + row];
      float mx = mw;
#pragma unroll
      for (int o2 = 1; o2 < kCW; o2 <<= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o2));
      const float f = mw == -INFINITY ? 0.f : ex2(mw - mx);
      float ls = f * lw;
#pragma unroll
      for (int o2 = 1; o2 < kCW; o2 <<= 1) ls += __shfl_xor_sync(0xffffffffu, ls, o2);
      wf[tid] = f;
      if (w == 0) {
        part[kRows * kLd + row] = mx;
        part[kRows * kLd + kRows + row] = ls;
      }
    }
    named_bar_sync(1, kCT);
    // ---- this CTA's O: (row, 4 columns) per thread, the eight warps' loads
    //      issued together
    for (int idx = tid; idx < M * (kD / 4); idx += kCT) {
      const int row = idx >> 5;
      const int col = (idx & 31) * 4;
      float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
      for (int w4 = 0; w4 < kCW; w4 += 4) {
        float4 ov[4];
#pragma unroll
        for (int w = 0; w < 4; ++w)
          ov[w] = *reinterpret_cast<const float4*>(wpart + (w4 + w) * kPartFloats + row * kLd + col);
        const float4 fv = *reinterpret_cast<const float4*>(wf + row * kCW + w4);
        const float fw[4] = {fv.x, fv.y, fv.z, fv.w};
#pragma unroll
        for (int w = 0; w < 4; ++w) {
          acc.x = fmaf(fw[w], ov[w].x, acc.x);
          acc.y = fmaf(fw[w], ov[w].y, acc.y);
          acc.z = fmaf(fw[w], ov[w].z, acc.z);
          acc.w = fmaf(fw[w], ov[w].w, acc.w);
        }
      }
      *reinterpret_cast<float4*>(part + row * kLd + col) = acc;
    }
  }

  // every CTA's state is complete and visible to the cluster
  cluster_sync_all();

  // this rank's slice of the output elements (float4 slots of the M rows):
  // thread (group g, slot t) sums ranks g, g + ngrp, ...; with several
  // groups their sums meet in shared memory
  const int F = M * (kD / 4);
  const int f0 = (rank * F) / C, f1 = ((rank + 1) * F) / C;
  const int nf = f1 - f0;
  const int ngrp = nf > 0 ? max(1, min(C, kCT / nf)) : 1;
  float* wt = reinterpret_cast<float*>(smem + kOffMm);  // [kMaxCluster][kRows] rank weights
  float* inv_l = reinterpret_cast<float*>(smem + kOffInvL);
  float4* red = reinterpret_cast<float4*>(smem + kOffRed);
  const uint32_t part_a = base + kOffPart;
  auto store_out = [&](int f, float4 acc) {
    const int p = f >> 5, col = (f & 31) * 4;
    const float il = inv_l[p];
    const int i = p / G, gq = p - i * G;
    const long long off = ((static_cast<long long>(b) * R + i) * a.Hq + h * G + gq) * kD + col;
    *reinterpret_cast<uint2*>(a.out + off) =
        make_uint2(sd_pack_bf16x2(acc.x * il, acc.y * il), sd_pack_bf16x2(acc.z * il, acc.w * il));
  };
  if (warp < kCW) {
    // the layer's rotated query rows go back to q now that every rank has
    // read the raw ones (all ranks passed the cluster barrier above)
    if (rank == 0) {
      for (int idx = tid; idx < M * 16; idx += kCT) {
        const int p = idx >> 4, c = idx & 15;
        const int i = p / G, gq = p - i * G;
        uint4 w;
        asm volatile("ld.shared.v4.u32 {%0,%1,%2,%3}, [%4];"
                     : "=r"(w.x), "=r"(w.y), "=r"(w.z), "=r"(w.w)
                     : "r"(qs + (c >> 3) * kQHalf + swz(p, c & 7)));
        *reinterpret_cast<uint4*>(a.q + ((static_cast<long long>(b) * R + i) * a.Hq + h * G + gq) * kD + c * 8) = w;
      }
    }
    // the ranks' weights per row: thread (row p, rank c) = (tid / C, tid % C)
    // reads rank c's (m, l) of row p; maximum and sum over the row's C lanes
    // (C is a power of two <= 16) by shuffles
    if (tid < ((M * C + 31) & ~31)) {
      const int p = tid / C, c = tid - (tid / C) * C;
      float m = -INFINITY, l = 0.f;
      if (p < M) {
        const uint32_t src = peer_addr(part_a, static_cast<uint32_t>(c));
        m = ld_peer_f32(src + (kRows * kLd + p) * 4);
        l = ld_peer_f32(src + (kRows * kLd + kRows + p) * 4);
      }
      float mx = m;
      for (int o2 = 1; o2 < C; o2 <<= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o2));
      const float f = m == -INFINITY ? 0.f : ex2(m - mx);
      float ls = f * l;
      for (int o2 = 1; o2 < C; o2 <<= 1) ls += __shfl_xor_sync(0xffffffffu, ls, o2);
      if (p < M) {
        wt[c * kRows + p] = f;
        if (c == 0) inv_l[p] = ls > 0.f ? 1.f / ls : 0.f;
      }
    }
    named_bar_sync(1, kCT);
    for (int idx = tid; idx < nf * ngrp; idx += kCT) {
      const int t = idx % nf, g = idx / nf;
      const int f = f0 + t, p = f >> 5, col = (f & 31) * 4;
      float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
      for (int c = g; c < C; c += ngrp) {
        const float w = wt[c * kRows + p];
        const float4 v = ld_peer_f32x4(peer_addr(part_a, static_cast<uint32_t>(c)) + (p * kLd + col) * 4);
        acc.x = fmaf(w, v.x, acc.x);
        acc.y = fmaf(w, v.y, acc.y);
        acc.z = fmaf(w, v.z, acc.z);
        acc.w = fmaf(w, v.w, acc.w);
      }
      if (ngrp > 1)
        red[g * nf + t] = acc;
      else
        store_out(f, acc);
    }
  }
  // no more reads of peers' shared memory from here: arrive now, and wait
  // (so that no CTA leaves while a peer may still read it) after the stores
  cluster_arrive_relaxed();
  if (warp < kCW && ngrp > 1) {
    named_bar_sync(1, kCT);
    if (tid < nf) {
      float4 acc = red[tid];
      for (int g = 1; g < ngrp; ++g) {
        const float4 v = red[g * nf + tid];
        acc.x += v.x;
        acc.y += v.y;
        acc.z += v.z;
        acc.w += v.w;
      }
      store_out(f0 + tid, acc);
    }
  }
  cluster_wait();
}

__global__ void __launch_bounds__(kThreads, 1)
    verify_decode_kernel(const __grid_constant__ CUtensorMap tm_k,
                         const __grid_constant__ CUtensorMap tm_v, const DecArgs a,
                         const RopeTable tab) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  const uint32_t base = smem_addr(smem);
  const int tid = threadIdx.x;
  if (tid == 0) {
    for (int s = 0; s < kSlots; ++s) {
      mbar_init(base + kOffBar + 8u * s, 1);
      mbar_init(base + kOffBar + 8u * (kSlots + s), 1);
    }
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    griddep_launch();
  }
  if (tid == kCT) {
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tm_k)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tm_v)) : "memory");
  }
  __syncthreads();
  // with the early flag the producer starts the prefix stream now: the first
  // ring's worth of this CTA's blocks (len is not written by the preceding
  // kernel)
  int issued = 0;
  if (a.early && tid == kCT) {
    const int C = static_cast<int>(gridDim.x), rank = static_cast<int>(cluster_rank());
    const int h = blockIdx.y, b = blockIdx.z;
    const int len_in = a.len[b];
    const int L_b = len_in;
    const bool valid = len_in >= 0 && len_in + a.R <= a.cap;
    if (valid) {
      const int nblk = (L_b + kBlk - 1) / kBlk;
      const int blk_begin = static_cast<int>((static_cast<long long>(rank) * nblk) / C);
      const int blk_end = static_cast<int>((static_cast<long long>(rank + 1) * nblk) / C);
      issued = min(blk_end - blk_begin, kSlots);
      for (int j = 0; j < issued; ++j) {
        const uint32_t bar = base + kOffBar + 8u * j;
        mbar_expect_tx(bar, kSlotBytes);
        const int y = (blk_begin + j) * kBlk, z = b * a.Hkv + h;
        const uint32_t dst = base + j * kSlotBytes;
        tma_load_3d(dst, &tm_k, bar, 0, y, z);
        tma_load_3d(dst + kHalfBytes, &tm_k, bar, 64, y, z);
        tma_load_3d(dst + kKVBytes, &tm_v, bar, 0, y, z);
        tma_load_3d(dst + kKVBytes + kHalfBytes, &tm_v, bar, 64, y, z);
      }
    }
  }
  if (!a.early) griddep_wait();
  decode_body(&tm_k, &tm_v, a, tab, smem, issued);
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

// [B*Hkv][cap][128] bf16 viewed as a 3-D tensor; boxes of 64 columns x 32 rows.
bool make_map(CUtensorMap* map, void* ptr, int cap, int planes) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[3] = {static_cast<cuuint64_t>(kD), static_cast<cuuint64_t>(cap),
                        static_cast<cuuint64_t>(planes)};
  cuuint64_t strides[2] = {static_cast<cuuint64_t>(kD) * 2,
                           static_cast<cuuint64_t>(cap) * static_cast<cuuint64_t>(kD) * 2};
  cuuint32_t box[3] = {64, kBlk, 1};
  cuuint32_t estr[3] = {1, 1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, ptr, dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

constexpr int kSizes[] = {16, 8, 4, 2, 1};
constexpr int kNumSizes = 5;

// Per device: attributes set, and how many clusters of each size fit at once.
struct DevState {
  bool ok = false;
  int active[kNumSizes] = {};  // co-resident clusters of each size
};

bool setup_kernel(int* active) {
  auto kern = verify_decode_kernel;
  if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes) != cudaSuccess ||
      cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) != cudaSuccess) {
    (void)cudaGetLastError();
    return false;
  }
  for (int i = 0; i < kNumSizes; ++i) {
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = kSizes[i];
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.gridDim = dim3(kSizes[i], 1, 1);
    cfg.blockDim = dim3(kThreads, 1, 1);
    cfg.dynamicSmemBytes = kSmemBytes;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, kern, &cfg) != cudaSuccess) {
      (void)cudaGetLastError();
      n = 0;
    }
    active[i] = n;
  }
  return true;
}

DevState* state() {
  static DevState st[16];
  static bool done[16] = {};
  static std::mutex mu;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 16) {
    (void)cudaGetLastError();
    return nullptr;
  }
  std::lock_guard<std::mutex> lock(mu);
  if (!done[dev]) {
    done[dev] = true;
    st[dev].ok = setup_kernel(st[dev].active);
  }
  return &st[dev];
}

// Cluster size of a call: the size forced by sd_set_cluster_size when one is
// and fits, else the largest size whose clusters for every (scene, KV head)
// fit on the device in one wave and leave each CTA at least two 32-key blocks
// of the capacity; 0 when the kernel does not serve.
int pick_size(int B, int Hkv, int cap) {
  DevState* s = state();
  if (!s || !s->ok) return 0;
  const long long units = static_cast<long long>(B) * Hkv;
  const long long nblk = (cap + kBlk - 1) / kBlk;
  const int forced = sd_internal_forced_cluster();
  for (int i = 0; i < kNumSizes && forced > 0; ++i)
    if (kSizes[i] == forced && s->active[i] > 0) return forced;
  for (int i = 0; i < kNumSizes; ++i) {
    const int cs = kSizes[i];
    const int act = s->active[i];
    if (act <= 0) continue;
    if (cs > 1 && nblk < 2LL * cs) continue;
    if (units <= act || cs == 1) return cs;
  }
  return 0;
}

// The library sends this kernel the block-masked layers only (the tcgen05
// layer kernel's 32-row tile is causal only, so they would otherwise run as
// three kernels). Causal layers and every attention call run faster on the
// tcgen05 kernel, measured on one box: the draft step (one scene, 4 KV heads,
// one row) 8.0 against 9.0 us, and every K = 1 / K = 2 point of the batched
// sweep (e.g. B = 1, L = 8192: 0.38 against 0.31 of the measured copy; B = 8,
// L = 2048: 0.59 against 0.56), where 128-key tensor-memory products outrun
// 16-row mma.sync tiles (~1.7k cycles a 32-key block a warp).
bool layer_preferred(int block) { return block != 0; }

bool shape_served(int R, int Hq, int Hkv, int D) {
  if (D != kD || Hkv <= 0 || Hq % Hkv || R <= 0 || R > kMaxNew) return false;
  return (Hq / Hkv) * R <= kRows;
}

sd_status launch(const sd_kv_cache* cache, const DecArgs& a, const RopeTable& tab, int cs, cudaStream_t stream) {
  const int B = cache->batch, Hkv = cache->n_kv_heads, cap = cache->capacity;
  CUtensorMap tk, tv;
  if (!make_map(&tk, cache->k, cap, B * Hkv) || !make_map(&tv, cache->v, cap, B * Hkv)) return SD_ERR_CUDA;
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
  cfg.numAttrs = 2;
  if (cudaLaunchKernelEx(&cfg, verify_decode_kernel, tk, tv, a, tab) != cudaSuccess) {
    (void)cudaGetLastError();
    return SD_ERR_CUDA;
  }
  return SD_OK;
}

}  // namespace

bool sd_internal_decode_serves(int B, int R, int Hq, int Hkv, int D, int cap, bool block) {
  if (!layer_preferred(block) || !shape_served(R, Hq, Hkv, D) || B <= 0 || B > 65535 || Hkv > 65535) return false;
  return pick_size(B, Hkv, cap) > 0;
}

sd_status sd_internal_verify_layer_dec(void* q, void* k_new, const void* v_new, const int32_t* pos,
                                       const RopeTable& tab, const sd_kv_cache* cache, void* out, int R,
                                       int Hq, float scale_log2, uint32_t* ticket, int early, int block,
                                       cudaStream_t stream, bool* handled) {
  *handled = false;
  const int B = cache->batch, Hkv = cache->n_kv_heads;
  if (!layer_preferred(block) || !shape_served(R, Hq, Hkv, cache->head_dim) || B > 65535) return SD_OK;
  const int cs = pick_size(B, Hkv, cache->capacity);
  if (cs <= 0) return SD_OK;
  DecArgs a = {};
  a.q = static_cast<__nv_bfloat16*>(q);
  a.out = static_cast<__nv_bfloat16*>(out);
  a.len = cache->len;
  a.k_new = static_cast<__nv_bfloat16*>(k_new);
  a.v_new = static_cast<const __nv_bfloat16*>(v_new);
  a.kc = static_cast<__nv_bfloat16*>(cache->k);
  a.vc = static_cast<__nv_bfloat16*>(cache->v);
  a.pos = pos;
  a.ticket = ticket;
  a.R = R;
  a.Hq = Hq;
  a.Hkv = Hkv;
  a.G = Hq / Hkv;
  a.M = a.G * R;
  a.cap = cache->capacity;
  a.early = early ? 1 : 0;
  a.block = block ? 1 : 0;
  a.scale_log2 = scale_log2;
  *handled = true;
  return launch(cache, a, tab, cs, stream);
}
