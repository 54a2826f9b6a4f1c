/*
 * sd.h -- C ABI of libsd.so, the GB300 (sm_103a) verify step of two-reasoner
 * speculative decoding ("Reasoning-aware Speculative Decoding for Efficient
 * VLA Models in Autonomous Driving", arxiv 2606.31160).
 *
 * In the paper's propose / verify / commit loop (Sec. 3.2) a small draft
 * proposes K tokens and the unmodified multimodal target scores them in one
 * pass. This library is the data-parallel hot path of that pass: the rotary
 * position encoding of the new rows (Sec. 3.3, Sec. 4.2), the KV-cache append
 * and rollback (Eq. commit), the causally masked GQA attention of the K + 1
 * verify rows (Eq. verify), and the two acceptance rules (Eqs. accept,
 * commit; Leviathan/Chen rejection sampling, cited in Sec. 1-2).
 *
 * Conventions shared by every entry point:
 *   - All tensor pointers are DEVICE pointers owned by the caller, row-major
 *     with the innermost index last, 16-byte aligned. The library never
 *     allocates device memory and never synchronises, except
 *     sd_get_device_error(), which synchronises the stream it is given.
 *   - Every call is asynchronous on `stream` (NULL = legacy default stream).
 *     The rotation, append and rollback kernels (and the tcgen05 attention and
 *     layer kernels) are programmatic dependent launches: they may become
 *     resident while the kernel before them on the stream finishes, but touch
 *     no memory before it has completed (the early-prefix flags below are the
 *     one exception, and say what they promise). Stream order is kept.
 *   - Problems visible on the host (bad sizes, NULL pointers, unsupported
 *     shapes, short workspace) return a status before anything is launched.
 *     Problems only visible on the device (a length past the capacity, a
 *     rollback past the appended rows, a token id outside the vocabulary)
 *     set bits of a per-device error word, read with sd_get_device_error();
 *     the affected scene is skipped and no kernel traps.
 *   - bf16 is IEEE-754 binary32 truncated to its upper 16 bits (bfloat16),
 *     stored as uint16.
 *   - B = scenes, R = K + 1 verify rows, Hq / Hkv = query / KV heads with
 *     G = Hq / Hkv, D = head dim, V = vocabulary size.
 */
#ifndef SD_H_
#define SD_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* cudaStream_t without pulling in the CUDA headers. */
typedef struct CUstream_st* sd_stream_t;

typedef enum {
  SD_OK = 0,
  SD_ERR_INVALID_ARG = 1,  /* NULL pointer, non-positive size, misalignment   */
  SD_ERR_UNSUPPORTED = 2,  /* valid but not built: D not in {64,128}, ...      */
  SD_ERR_WORKSPACE = 3,    /* workspace NULL or smaller than the size query    */
  SD_ERR_CUDA = 4,         /* a CUDA runtime call failed (launch, attribute)   */
  SD_ERR_DEVICE = 5,       /* sd_get_device_error found device-side error bits */
  SD_ERR_TIMEOUT = 6       /* a bounded device wait gave up (see error bits)   */
} sd_status;

typedef enum { SD_BF16 = 0, SD_F32 = 1 } sd_dtype;

/* Device error bits (sd_get_device_error). */
#define SD_DEVERR_KV_OVERFLOW   0x1u  /* append would pass the capacity        */
#define SD_DEVERR_ROLLBACK      0x2u  /* committed outside [0, n_appended]     */
#define SD_DEVERR_TOKEN_RANGE   0x4u  /* a draft token outside [0, V)          */
#define SD_DEVERR_LENGTH        0x8u  /* len[b] < R or len[b] > capacity       */
#define SD_DEVERR_TIMEOUT       0x10u /* a bounded mbarrier wait ran out       */

/*
 * KV cache of one attention layer. k and v are [B][Hkv][capacity][D] bf16;
 * len is a device int32[B]: the number of valid rows of each scene. Rows at
 * or past len[b] are never read by the attention (their contents may be
 * anything, NaN included).
 */
typedef struct {
  void* k;
  void* v;
  int32_t* len;
  int32_t batch;
  int32_t n_kv_heads;
  int32_t capacity;
  int32_t head_dim;
} sd_kv_cache;

/* Name of a status code; a static string, never NULL. */
const char* sd_status_str(sd_status s);

/* Library version string, e.g. "sd 0.1 sm_103a". */
const char* sd_version(void);

/*
 * M-RoPE rotation of the new Q and K rows, in place (Sec. 3.3 Eq. rope-3d;
 * Sec. 4.2 Eqs. axis-assign, mrope-phase).
 *   q:   [B][R][Hq][D] bf16, k: [B][R][Hkv][D] bf16 (either may be NULL when
 *        its head count is 0).
 *   pos: [B][R][3] int32 (t, h, w) coordinates of each row, device memory.
 *   sections: HOST int32[3] = (s_T, s_H, s_W), summing to D / 2.
 *   interleaved: 0 = blocked axis assignment, 1 = a(d) = (T,H,W)[d mod 3].
 *   base: theta_d = base^(-2d/D).
 * Pair d is the adjacent dimensions (2d, 2d+1): x' = x cos(phi) - y sin(phi),
 * y' = x sin(phi) + y cos(phi), phi = theta_d * pos[a(d)]. Arithmetic is fp32
 * with an extended-precision angle; results round to bf16.
 * D must be 64 or 128 (SD_ERR_UNSUPPORTED otherwise).
 */
sd_status sd_rope_apply(void* q, void* k, int B, int R, int Hq, int Hkv, int D,
                        const int32_t* pos, const int32_t sections[3],
                        int interleaved, float base, sd_stream_t stream);

/*
 * FlatRoPE / plain 1D RoPE (Sec. 3.3 Eq. rope-1d; Sec. 4.2 Eq. flatrope-proj):
 * the same rotation with every axis at the sequence index pos1d[b][r]
 * (device int32[B][R]). Equal, bit for bit, to sd_rope_apply with
 * pos = (m, m, m) under any section layout.
 */
sd_status sd_rope_apply_1d(void* q, void* k, int B, int R, int Hq, int Hkv, int D,
                           const int32_t* pos1d, float base, sd_stream_t stream);

/*
 * Append R new rows per scene (Eq. commit: the verify pass writes the keys and
 * values of all K + 1 rows before the acceptance is known).
 *   k_new, v_new: [B][R][Hkv][D] bf16 (rotated keys; values).
 * Writes row i of scene b at cache position len[b] + i, then len[b] += R.
 * A scene with len[b] + R > capacity is left untouched and sets
 * SD_DEVERR_KV_OVERFLOW.
 */
sd_status sd_kv_append(const sd_kv_cache* cache, const void* k_new,
                       const void* v_new, int R, sd_stream_t stream);

/*
 * Roll the lengths back to the committed rows (Eq. commit: t <- t + l + 1).
 *   len:       device int32[count], count a multiple of B (one length array
 *              per layer, all layers' arrays contiguous: [n_layers][B]).
 *   committed: device int32[B], rows kept of the n_appended just appended
 *              (n_emit of sd_accept_greedy / sd_accept_sample).
 * len[l*B + b] <- len[l*B + b] - n_appended + committed[b]. A committed value
 * outside [0, n_appended] (or a length that would drop below 0) leaves that
 * entry untouched and sets SD_DEVERR_ROLLBACK.
 */
sd_status sd_kv_rollback(int32_t* len, int count, int B, const int32_t* committed,
                         int n_appended, sd_stream_t stream);

/*
 * Workspace bytes sd_verify_attention needs for this shape on the CURRENT
 * device (the split plan depends on its SM count): 0 when the batch alone
 * fills the GPU and no split merge is needed. capacity = cache capacity.
 */
size_t sd_verify_attention_workspace(int B, int R, int Hq, int Hkv, int D, int capacity);

/*
 * Verify attention (Eq. verify, Sec. 3.2): for scene b, query head h (KV head
 * g = h / G) and row i < R,
 *   o[b][i][h] = softmax_n( q[b][i][h] . k[b][g][n] * scale ) v[b][g][n],
 *   n = 0 .. len[b] - R + i
 * i.e. row i is the token at position L_b + i (L_b = len[b] - R, the prefix
 * before the append) and sees the prefix plus the new rows up to itself.
 *   q:   [B][R][Hq][D] bf16 (rotated), cache: keys/values already appended,
 *   out: [B][R][Hq][D] bf16.
 *   scale: 0 selects 1/sqrt(D).
 * The G*R query rows that share a KV head are packed into one tile, so each
 * K/V row is read from HBM once; when B*Hkv alone cannot fill the GPU each
 * head's keys are split over several CTAs whose partial softmax states merge
 * through `workspace` (sd_verify_attention_workspace bytes, zero-filled
 * before its first use and left zeroed by every completed call; calls that
 * share a workspace must not overlap on the device; after SD_ERR_TIMEOUT it
 * must be zero-filled again). Requires D in {64, 128}, Hq % Hkv == 0 and
 * G*R <= 128. A scene with len[b] < R or len[b] > capacity sets
 * SD_DEVERR_LENGTH and its output is left unwritten. The first call per
 * device and shape should come before any stream capture (it sets kernel
 * attributes and queries the occupancy).
 * Kernel choice is by shape: head_dim 128 with G*R <= 128 takes the tcgen05
 * kernel, every other shape the mma.sync kernel (sd_verify_kernel names it). A test-only override exists:
 * the environment variable SD_ATTENTION_KERNEL=mma, read once per process,
 * sends every shape to the mma.sync kernel so that tests can compare the two
 * kernels on the same inputs; production callers leave it unset.
 */
sd_status sd_verify_attention(const void* q, const sd_kv_cache* cache, void* out,
                              int R, int Hq, float scale, void* workspace, size_t ws_bytes,
                              sd_stream_t stream);

/* sd_verify_attention_ex flags: the block mask; the prefix read early. */
#define SD_ATTN_BLOCK_MASK 1
#define SD_ATTN_PREFIX_EARLY 2

/*
 * sd_verify_attention with flags. SD_ATTN_BLOCK_MASK selects the block mask of
 * the block-diffusion drafts (Sec. 5 "Targets and drafts": a block of K = 16
 * tokens proposed at once): every new row sees the prefix and all R new rows,
 * n = 0 .. len[b] - 1, instead of n <= len[b] - R + i.
 * SD_ATTN_PREFIX_EARLY declares that the kernel issued just before this call
 * on the stream writes neither this cache (its K / V rows, the new rows
 * included) nor its len (true when a step's layers are issued back to back
 * after their appends). For head_dim 128 and up to 16 new rows (32 when
 * G * R > 32) the call is then a programmatic dependent launch that reads len
 * and streams the whole cache while its predecessor still runs, and reads q
 * only after the predecessor has completed; other shapes ignore the flag.
 * Without the flag those shapes are programmatic dependent launches too, but
 * the kernel waits for its predecessor to complete before its first global
 * access, so only its launch and set-up overlap it.
 * Other bits: SD_ERR_INVALID_ARG. Everything else as sd_verify_attention
 * (which is this call with flags 0).
 */
sd_status sd_verify_attention_ex(const void* q, const sd_kv_cache* cache, void* out,
                                 int R, int Hq, float scale, int flags, void* workspace,
                                 size_t ws_bytes, sd_stream_t stream);

/*
 * Cluster size of the tcgen05 verify-attention kernels (sd_verify_attention
 * and sd_verify_layer, head_dim 128): one
 * thread-block cluster of `cluster_size` CTAs per (scene, KV head) splits that
 * head's keys evenly and merges the partial softmax states in distributed
 * shared memory (the split-L form of Eq. verify). 0 (the default) lets every
 * call choose from the occupancy of each size and the capacity; 1, 2, 4, 6, 8
 * or 16 forces that size for later calls on every device (a size of which no
 * cluster fits on the device falls back to the automatic choice). Process-wide, host-only, no
 * device work; results are the same for every size up to fp32 rounding order.
 * Returns SD_ERR_INVALID_ARG for any other value.
 */
sd_status sd_set_cluster_size(int cluster_size);

/*
 * Which kernel serves a shape on the CURRENT device: "tcgen05" or
 * "mma.sync" for sd_verify_attention (layer = 0), and for
 * sd_verify_layer (layer = 1, or 2 with SD_LAYER_BLOCK_MASK; "three kernels"
 * when the layer runs as the rotation, append and attention kernels in
 * sequence); "unsupported" for a shape neither call takes. Host-only, no
 * device work; a static string.
 */
const char* sd_verify_kernel(int B, int R, int Hq, int Hkv, int D, int capacity, int layer);

/*
 * Attention budget of the verify rows (Sec. 4.2 "Empirical confirmation",
 * Table tab:attn-budget), a diagnostic beside the verify path. For scene b,
 * query head h and row i, with p the softmax of q . k * scale over the keys
 * row i sees (0 .. len[b] - R + i, as in sd_verify_attention) and
 * L_b = len[b] - R:
 *   mass[b][i][h][0] = sum of p over the visual keys [0, n_visual[b])
 *   mass[b][i][h][1] = over the trajectory / prompt-text keys [n_visual[b], L_b)
 *   mass[b][i][h][2] = over the rows generated in this step [L_b, L_b + i]
 *   entropy[b][i][h] = entropy (nats) of p over the keys from n_visual[b] on,
 *                      renormalised, divided by the log of their number
 *                      (0 when there is at most one such key)
 *   q: [B][R][Hq][D] bf16 (rotated), cache: keys appended (len includes R),
 *   n_visual: int32 [B] device, mass: fp32 [B][R][Hq][3] device,
 *   entropy: fp32 [B][R][Hq] device; scale: 0 selects 1/sqrt(D).
 * One pass over the keys: bf16 tensor-core scores with fp32 accumulation,
 * fp32 sums with a running maximum per row (within 1e-4 of a float64 reference
 * on the target layer).
 * D in {64, 128}, Hq % Hkv == 0. A scene with len[b] < R or len[b] >
 * capacity sets SD_DEVERR_LENGTH and is left unwritten; n_visual[b] outside
 * [0, L_b] sets it too and is clamped.
 */
sd_status sd_attention_budget(const void* q, const sd_kv_cache* cache, int R, int Hq, float scale,
                              const int32_t* n_visual, float* mass, float* entropy,
                              sd_stream_t stream);

/* sd_verify_layer flags: see below. */
#define SD_LAYER_PREFIX_EARLY 1
#define SD_LAYER_BLOCK_MASK 2

/*
 * Workspace bytes sd_verify_layer needs on the CURRENT device for this shape.
 */
size_t sd_verify_layer_workspace(int B, int R, int Hq, int Hkv, int D, int capacity);

/*
 * One attention layer of the verify pass in one call (Eq. verify, Sec. 3.2):
 * the M-RoPE rotation of the R new query and key rows (Sec. 3.3 Eq. rope-3d,
 * Sec. 4.2 Eqs. axis-assign, mrope-phase), their append to the cache (Eq.
 * commit) and the verify attention over the prefix plus the new rows.
 * Equal to sd_rope_apply(q, k_new, ...) + sd_kv_append(cache, k_new, v_new)
 * + sd_verify_attention(q, cache, out): q and k_new are rotated in place,
 * rows len[b] .. len[b]+R-1 of the cache receive k_new / v_new, len[b] += R,
 * and out receives the attention. Here len[b] on entry is the PREFIX length.
 *   q [B][R][Hq][D], k_new / v_new [B][R][Hkv][D] bf16, pos [B][R][3] int32,
 *   sections (host), interleaved, base: as for sd_rope_apply; scale as for
 *   sd_verify_attention.
 *   workspace: sd_verify_layer_workspace() bytes, zero-filled before first
 *   use, left zeroed by every completed call; calls sharing it must not
 *   overlap on the device -- calls flagged SD_LAYER_PREFIX_EARLY overlap
 *   their predecessor, so give each layer its own workspace.
 *   flags: SD_LAYER_PREFIX_EARLY declares that the kernel issued just before
 *   this call on the stream writes neither this layer's cache, nor its len,
 *   nor pos (true for every layer but the first of a verify pass, when the
 *   layers are issued back to back and the positions were written before the
 *   pass). The call is then a programmatic dependent launch that reads len and
 *   pos and streams the cached prefix while its predecessor still runs; q,
 *   k_new and v_new are read only after the predecessor has completed.
 *   Without the flag the tcgen05 kernel is still a programmatic dependent
 *   launch, but it waits for its predecessor to complete before its first
 *   global access (only its launch and set-up overlap), so such calls may
 *   share a workspace.
 *   SD_LAYER_BLOCK_MASK: the attention uses the block mask (as
 *   SD_ATTN_BLOCK_MASK of sd_verify_attention_ex).
 * For head_dim 128 this is one kernel: the tcgen05 kernel for G * R <= 128
 * and R <= 31 (R <= 16 when a causal layer has G * R <= 32: its 32-row tile
 * is causal only, so block-masked layers always take the 64-row tile);
 * other shapes run the three kernels in sequence (sd_verify_kernel names the
 * choice). A scene whose append would pass the
 * capacity sets SD_DEVERR_KV_OVERFLOW and is left untouched.
 */
sd_status sd_verify_layer(void* q, void* k_new, const void* v_new, const int32_t* pos,
                          const int32_t sections[3], int interleaved, float base,
                          const sd_kv_cache* cache, void* out, int R, int Hq, float scale,
                          void* workspace, size_t ws_bytes, int flags, sd_stream_t stream);

/*
 * Workspace bytes sd_accept_greedy needs for (B, R = K + 1, V).
 */
size_t sd_accept_greedy_workspace(int B, int K, int V);

/*
 * Greedy acceptance (Eqs. verify, accept, commit; Sec. 4.3 Eq. accept-length).
 *   logits: [B][K+1][V] of `dtype` (SD_BF16 or SD_F32).
 *   draft:  [B][K] int32 draft tokens.
 * Outputs (device): argmax [B][K+1] int32, the lowest index among equal
 * maxima (values compare numerically, +0 == -0; NaN is outside the
 * contract); n_emit [B] int32 = l + 1, l = the number of leading drafts equal
 * to argmax; tokens [B][K+1] int32 = draft[0..l-1], argmax[l], then -1.
 * ws: caller-owned device scratch of sd_accept_greedy_workspace() bytes,
 * zero-filled before its first use; every call leaves it zero-filled again.
 * Calls that share a workspace must not overlap on the device.
 * argmax may be NULL. K = 0 is plain argmax.
 */
sd_status sd_accept_greedy(const void* logits, sd_dtype dtype, int B, int K, int V,
                           const int32_t* draft, int32_t* n_emit, int32_t* tokens,
                           int32_t* argmax, void* ws, size_t ws_bytes,
                           sd_stream_t stream);

/*
 * Greedy acceptance without a caller workspace (the paper has no counterpart:
 * this serves callers that cannot allocate device memory -- a serving loop
 * whose pool belongs to another runtime, a pre-planned graph that forbids
 * allocation while it runs, a host with no device allocator).
 * Same arguments, results and rules as sd_accept_greedy minus ws / ws_bytes.
 * Its scratch is a fixed array inside the library of
 * sd_accept_greedy_noalloc_max_bytes() bytes (1 MiB: per-scene tickets for up
 * to 4096 scenes, then B * (K + 1) * ceil(V / 4096) partials of 8 bytes), held
 * on every device that loads the library until the process exits. Larger
 * shapes return SD_ERR_WORKSPACE. Allocates nothing. The first call on a
 * device resolves the array's device address (make it before any stream
 * capture). All calls share the array: calls that overlap on the device race
 * and must not be issued; every completed call leaves it ready for the next.
 */
sd_status sd_accept_greedy_noalloc(const void* logits, sd_dtype dtype, int B, int K, int V,
                                   const int32_t* draft, int32_t* n_emit, int32_t* tokens,
                                   int32_t* argmax, sd_stream_t stream);

/* Bytes of the fixed scratch array behind sd_accept_greedy_noalloc. */
size_t sd_accept_greedy_noalloc_max_bytes(void);

/*
 * Workspace bytes sd_accept_sample needs for (B, K, V).
 */
size_t sd_accept_sample_workspace(int B, int K, int V);

/*
 * Rejection-sampling acceptance (Leviathan et al. / Chen et al., cited in
 * Sec. 1-2) at temperature T > 0, driven by caller-supplied uniforms.
 *   z_target: [B][K+1][V] fp32, z_draft: [B][K][V] fp32, draft: [B][K] int32,
 *   u: [B][K+1] fp32 uniforms in [0, 1).
 * With p_j = softmax(z_target[j] / T), q_j = softmax(z_draft[j] / T):
 * draft j is accepted iff u[j] * q_j(x) <= p_j(x); at the first rejection j
 * the token is drawn from (p_j - q_j)+ with u[K], and when all K are
 * accepted the bonus is drawn from p_K with u[K]; a draw from weights w takes
 * the smallest v with sum_{v' <= v} w(v') > u[K] * sum(w).
 * Outputs: n_emit [B] = l + 1 and tokens [B][K+1] (draft[0..l-1], the drawn
 * token, then -1). fp32 arithmetic with fixed-order reductions: the result is
 * a deterministic function of the inputs.
 * ws: as for sd_accept_greedy (zero-filled before first use, left zeroed).
 */
sd_status sd_accept_sample(const float* z_target, const float* z_draft, int B, int K,
                           int V, float temperature, const int32_t* draft,
                           const float* u, int32_t* n_emit, int32_t* tokens,
                           void* ws, size_t ws_bytes, sd_stream_t stream);

/*
 * Synchronise `stream`, return the device error bits accumulated on the
 * current device since the last call in *bits, and clear them.
 * Returns SD_OK when no bit is set, SD_ERR_DEVICE when some bit is set
 * (SD_ERR_TIMEOUT when SD_DEVERR_TIMEOUT is among them), SD_ERR_CUDA when the
 * synchronisation itself failed.
 */
sd_status sd_get_device_error(sd_stream_t stream, uint32_t* bits);

#ifdef __cplusplus
}
#endif

#endif /* SD_H_ */
