/*
 * wm.h -- C ABI of the WhiteMatter decode hot path on GB300 (sm_103a).
 *
 * WhiteMatter (Zhang & Ren, "All-to-All Cross-Layer Connections via KV
 * Mixing") replaces the L per-layer KV projections of a decoder with a
 * cross-layer KV pool (Sec. 3.1): for every token a router mixes the L layer
 * states into k <= L channels, each channel is projected to keys and values
 * and stored in a k-channel cache, and layer l attends over channel c(l).
 * One decode step (Sec. 3.2) is L calls of wm_decode_attn (one per layer,
 * each reading the existing cache) followed by one wm_kv_mix that appends
 * the new token's channels.
 *
 * Conventions for every entry point:
 *  - Memory: the caller owns and allocates everything (weights, states,
 *    queries, outputs, cache pools, page tables, workspaces, status word).
 *    Pointers marked "device" must be device (or managed) memory of the
 *    current CUDA device.  The library allocates no memory and keeps no state
 *    between calls other than per-device attribute and address caches, a
 *    process-wide counter that tags each attention call (its epoch), and the
 *    fixed scratch array of wm_decode_attn_noalloc.
 *  - Streams: `stream` is a cudaStream_t (NULL = legacy default stream).
 *    Compute calls only enqueue work and return; results are valid after the
 *    stream is synchronised.
 *  - Errors: argument errors detectable on the host return synchronously
 *    without launching anything.  A failed launch returns WM_ERR_CUDA.
 *    Errors found by a kernel (an out-of-range page id, slot or length; a
 *    pipeline wait that ran out) are written to the device word `dev_status`
 *    (if not NULL) as the largest wm_status code seen, and the offending
 *    access is skipped; no kernel traps.  The caller zeroes dev_status and
 *    reads it after synchronising.
 *  - dtype: WM_DT_BF16 tensors hold bf16 values (norms, router, mix and
 *    softmax run in fp32, projections take bf16 operands with fp32
 *    accumulation, cache and outputs are rounded to bf16); WM_DT_F32 tensors
 *    are fp32 and every step runs in fp32 FMA arithmetic.
 *  - Gains, router biases and weights have the dtype of the config.
 *
 * Cache layout (per pool, K and V alike), element (c, page, h, s, e) at
 *   (((c * num_pages + page) * Hkv + h) * page_size + s) * d + e
 * for channel c < k, physical page < num_pages, kv head h < Hkv, slot in page
 * s < page_size, element e < d.  Logical slot t of sequence b lives in page
 * page_table[b * max_pages + t / page_size] at in-page slot t % page_size.
 * Slot 0 of every sequence holds the learned dummy KV (Sec. 3.2); the token
 * at position i is stored at slot i + 1.  The page table is shared by all k
 * channels.
 */
#ifndef WM_H_
#define WM_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define WM_MAX_L 128

typedef enum {
  WM_OK = 0,
  WM_ERR_INVALID_ARG = 1, /* bad pointer, size or configuration value        */
  WM_ERR_UNSUPPORTED = 2, /* valid per the paper, not built here (e.g. d=80) */
  WM_ERR_CUDA = 3,        /* a CUDA runtime call or launch failed            */
  WM_ERR_BOUNDS = 4,      /* device: page id, slot or length out of range    */
  WM_ERR_TIMEOUT = 5      /* device: a bounded pipeline wait ran out         */
} wm_status;

typedef enum { WM_DT_F32 = 0, WM_DT_BF16 = 1 } wm_dtype;

/* Model shape of the pool (Sec. 3.1) and of the attention that reads it. */
typedef struct {
  int32_t L;          /* decoder layers = source states per token, 1..WM_MAX_L     */
  int32_t k;          /* KV channels, 1 <= k <= L                                  */
  int32_t D;          /* hidden width; multiple of 8, at most 4096                 */
  int32_t Hq;         /* query heads; multiple of Hkv, Hq/Hkv in {1,2,4,8}         */
  int32_t Hkv;        /* key/value heads per channel                               */
  int32_t d;          /* head dimension: 64, 96 or 128                             */
  int32_t p;          /* router reads every p-th layer from L-1 down, p >= 1       */
  int32_t page_size;  /* cache slots per page: a power of two, 1..4096             */
  int32_t dtype;      /* wm_dtype                                                  */
  float eps_rms;      /* epsilon of the pre-mix and per-channel RMSNorms           */
  float eps_qk;       /* epsilon of the per-channel key norm (QK-norm)             */
  double rope_theta;  /* RoPE base: inverse frequency theta^(-2i/d), i < d/2       */
  int32_t chan_of_layer[WM_MAX_L]; /* c(l) in [0, k): channel read by layer l     */
} wm_config;

/* Views of the two cache pools inside one caller buffer (see wm_cache_alloc). */
typedef struct {
  void* k_pool;       /* device: [k][num_pages][Hkv][page_size][d] rotated keys    */
  void* v_pool;       /* device: same layout, raw values                           */
  int32_t num_pages;  /* physical pages per channel                                */
  int32_t k, Hkv, page_size, d, dtype; /* copied from the config, checked per call */
} wm_cache;

/* Pool parameters (Sec. 3.1 Steps 1-2); index [X] is the branch, 0 = K, 1 = V.
 * All device pointers, dtype of the config, row-major:
 *   pre_g[X] [D]                pre-mix RMSNorm gain of branch X
 *   Wr[X]    [k*L][Lp*D]        router weights, Lp = ceil(L/p); input block m
 *                               holds the normed state of layer L-1-m*p
 *   br[X]    [k*L]              router bias; output j*L+l is alpha[j][l]
 *   ch_g[X]  [k][D]             per-channel RMSNorm gains
 *   Wkv[X]   [k][Hkv*d][D]      per-channel projections W^K_j / W^V_j
 *   qk_g     [k][d]             per-channel key-norm gains                    */
typedef struct {
  const void* pre_g[2];
  const void* Wr[2];
  const void* br[2];
  const void* ch_g[2];
  const void* Wkv[2];
  const void* qk_g;
} wm_mix_weights;

/* Human-readable name of a status code (static storage). */
const char* wm_status_string(wm_status s);

/* Validate a configuration without touching the GPU.  Returns WM_OK,
 * WM_ERR_INVALID_ARG (values outside the paper's definitions, e.g. k > L or
 * c(l) >= k) or WM_ERR_UNSUPPORTED (shapes this library does not build). */
wm_status wm_config_check(const wm_config* cfg);

/* Bytes of device memory wm_cache_alloc needs for `num_pages` pages per
 * channel: two pools of k*num_pages*Hkv*page_size*d elements (the k-channel
 * cache of Sec. 3.1 Step 2: k/L of a per-layer cache), each 256-byte aligned.
 * Returns 0 for an invalid config or num_pages < 1. */
size_t wm_cache_bytes(const wm_config* cfg, int32_t num_pages);

/* Lay the two pools out inside a caller buffer.  dev_buf must be 256-byte
 * aligned device memory of at least wm_cache_bytes(cfg, num_pages) bytes;
 * nothing is written to it.  Fills *out.  Errors: WM_ERR_INVALID_ARG for a
 * NULL pointer, a misaligned or too small buffer, or a bad config. */
wm_status wm_cache_alloc(const wm_config* cfg, void* dev_buf, size_t bytes, int32_t num_pages,
                         wm_cache* out);

/* Workspace bytes wm_kv_mix needs for a batch of B tokens. */
size_t wm_kv_mix_workspace(const wm_config* cfg, int32_t B);

/*
 * The cross-layer KV pool for B tokens (Sec. 3.1 Steps 1-2, appended as in
 * Sec. 3.2).  For each token b and branch X:
 *   hhat_l   = RMSNorm_pre^X(h[b][l])                     for l < L
 *   xi       = [hhat_{L-1}, hhat_{L-1-p}, ...]            (Lp states)
 *   alpha    = reshape_{k x L}(Wr[X] xi + br[X])          (signed, no softmax)
 *   htilde_j = sum_l alpha[j][l] hhat_l                   for j < k
 *   K_j = W^K_j RMSNorm^K_j(htilde^K_j),  V_j = W^V_j RMSNorm^V_j(htilde^V_j)
 *   Ktilde_j = RoPE(QKNorm_j(K_j) per head; pos = slot[b] - 1)
 * and writes Ktilde_j, V_j of every channel j and kv head to logical slot
 * slot[b] of sequence b.
 *   h          device [B][L][D]: states entering layers 0..L-1
 *   page_table device int32 [B][max_pages]
 *   slot       device int32 [B]: write slot, 1 <= slot[b] < max_pages*page_size
 *   workspace  device, >= wm_kv_mix_workspace(cfg, B) bytes, 256-byte aligned,
 *              no contents required
 * h, Wr, Wkv, pre_g and ch_g must be 16-byte aligned (WM_ERR_INVALID_ARG
 * otherwise): they are read as 16-byte vectors.
 * Only the B*k*2*Hkv*d cache elements addressed are written.  A bad slot or
 * page id skips that token's write and sets WM_ERR_BOUNDS.  B = 0 is a no-op.
 * The kernels are chained with programmatic dependent launch; the router and
 * projection kernels start streaming their weights (Wr, Wkv) before waiting
 * for the work before them, which is the library's own previous kernel.  So
 * the weights must not be written by a kernel that runs immediately before
 * the call and lets its dependents start early (ordinary kernels and copies
 * do not).
 */
wm_status wm_kv_mix(const wm_config* cfg, const wm_cache* cache, const wm_mix_weights* w,
                    const void* h, const int32_t* page_table, const int32_t* slot, int32_t B,
                    int32_t max_pages, void* workspace, size_t ws_bytes, int32_t* dev_status,
                    void* stream);

/* Kernels one wm_kv_mix call of B tokens enqueues (0 for B = 0), -1 for an
 * invalid config or B < 0; no GPU work: prenorm, router, mix and the
 * projection with its fused epilogue (4 for bf16), or a separate epilogue
 * after a SIMT projection (5: fp32, or no TMA encoder in the driver). */
int32_t wm_kv_mix_launches(const wm_config* cfg, int32_t B);

/* Workspace bytes wm_decode_attn needs for B sequences whose page tables
 * have max_pages entries. */
size_t wm_decode_attn_workspace(const wm_config* cfg, int32_t B, int32_t max_pages);

/*
 * Decode attention of one layer (Sec. 3.1 Step 3, with the dummy slot of
 * Sec. 3.2): query head hq of sequence b attends over logical slots
 * 0..seq_lens[b]-1 of channel c(layer) = cfg->chan_of_layer[layer], kv head
 * hq / (Hq/Hkv):  out = softmax(q K^T / sqrt(d)) V, fp32 softmax and
 * accumulation.  Slots at or beyond seq_lens[b] are never read into the
 * result (they may hold anything, NaN included).
 *   q          device [B][Hq][d], already normed and rotated by the caller
 *   seq_lens   device int32 [B], 1 <= seq_lens[b] <= max_pages*page_size
 *   out        device [B][Hq][d]
 *   workspace  device, >= wm_decode_attn_workspace(cfg, B, max_pages) bytes,
 *              256-byte aligned.  It must be zero-filled before its first
 *              use; every call leaves it ready for the next one (zero-fill it
 *              again after a call that reported WM_ERR_TIMEOUT).  One
 *              workspace serves calls of one configuration with any B and
 *              max_pages it is large enough for.  Calls that share a
 *              workspace must not overlap on the GPU.
 * A bad length or page id zero-fills that output row (length) or skips the
 * page, and sets WM_ERR_BOUNDS.  B = 0 is a no-op; B above 4096 or B * Hq
 * above 2^30 returns WM_ERR_UNSUPPORTED.
 */
wm_status wm_decode_attn(const wm_config* cfg, const wm_cache* cache, int32_t layer,
                         const void* q, const int32_t* page_table, const int32_t* seq_lens,
                         int32_t B, int32_t max_pages, void* out, void* workspace,
                         size_t ws_bytes, int32_t* dev_status, void* stream);

/* Flags of wm_decode_attn_flags. */
#define WM_ATTN_INPUTS_READY 1u
#define WM_ATTN_DYNAMIC_SPLIT 2u
#define WM_ATTN_UNIT_SPLIT 4u

/*
 * wm_decode_attn with flags; wm_decode_attn(...) is wm_decode_attn_flags(...,
 * flags = 0, ...).  Launches are chained with programmatic dependent launch:
 * a launch may start while the previous work on the stream finishes, and
 * waits for it before reading anything that work may have written.
 *   WM_ATTN_INPUTS_READY: the caller promises that the work immediately
 *     before this call on `stream` writes none of the cache pools, the page
 *     table and seq_lens (it may write q, out and this workspace: the kernel
 *     touches those only after the wait).  The kernel then starts fetching
 *     K/V while that work finishes and waits for it only before reading q.
 *     Within one decode step this holds for layers 1..L-1 (the previous
 *     layer's attention may share the workspace); it does NOT hold for the
 *     first layer after wm_kv_mix or after any update of seq_lens / the page
 *     table.
 *   WM_ATTN_DYNAMIC_SPLIT: hand the KV stream out in chunks from a device
 *     counter (about 8 chunks per warp, warps that stream faster take more)
 *     whatever the launch size.  Without it only launches reading at least
 *     2 GB of K/V do so; smaller ones give each warp one equal chunk.  The
 *     result is the same within rounding (the merge order of the pieces of
 *     a unit depends on where the chunks end, not on which warp takes them).
 *     wm_decode_attn_workspace covers either split.
 *   WM_ATTN_UNIT_SPLIT: give every (sequence, kv head) unit one cluster of
 *     C = min(8, max(1, SMs / units)) CTAs whose warps each stream an equal
 *     share of the unit and merge on chip (shared and distributed shared
 *     memory), whatever the launch size.  Without it the split is taken only
 *     for launches below 2 GB, or of a single sequence, where, at the
 *     largest C whose clusters are all resident at once, it runs at least
 *     60% of the warps of the static split above (the paper's model shape,
 *     48 units: C = 8; 192 units: C = 1; one sequence of 32 heads: C = 8);
 *     every other launch streams as above.  The unit split uses no
 *     workspace and gives the same result within rounding.
 * Unknown flag bits, or DYNAMIC_SPLIT together with UNIT_SPLIT, return
 * WM_ERR_INVALID_ARG.
 */
wm_status wm_decode_attn_flags(const wm_config* cfg, const wm_cache* cache, int32_t layer,
                               const void* q, const int32_t* page_table,
                               const int32_t* seq_lens, int32_t B, int32_t max_pages, void* out,
                               void* workspace, size_t ws_bytes, uint32_t flags,
                               int32_t* dev_status, void* stream);

/*
 * How wm_decode_attn_flags would split a launch (no GPU work; for tuning and
 * tests).  Fills plan[0..4] with: the grid (CTAs), warps in it, work
 * chunks a stream-K launch cuts the KV stream into at most, stages (8 KB of
 * K+V) per chunk (0: a static split, one chunk per warp, whose chunk count is
 * its warp count), and the CTAs per unit of the unit split (0: stream-K; then
 * the grid is persistent).  Returns WM_ERR_INVALID_ARG for a bad config,
 * B < 1, max_pages < 1, unknown or conflicting flags, or plan == NULL.
 */
wm_status wm_decode_attn_plan(const wm_config* cfg, int32_t B, int32_t max_pages, uint32_t flags,
                              int32_t plan[5]);

/*
 * Causal channel attention of one layer for many query positions at once:
 * prefill, and one pass of the token-parallel schedules (Sec. 3.1 Step 3
 * "standard causal SDPA"; dummy offset of Sec. 3.2; Jacobi and cyclic
 * Gauss-Seidel passes of Sec. 3.3, whose group q is the positions
 * {i : i mod g = q}).  The dummy sits at slot 0 and token t at slot t + 1, so
 * query row r of sequence b, the token at position i = pos[b*Tq + r],
 * attends over slots 0..i of channel c(layer) (the dummy and the tokens
 * before it, never its own slot i + 1), kv head hq / (Hq/Hkv):
 *   out = softmax(q K^T / sqrt(d)) V, fp32 softmax and accumulation, bf16
 *   probabilities into the P V product (tensor cores).
 *   q          device bf16 [B][Tq][Hq][d], already normed and rotated
 *   pos        device int32 [B][Tq], 0 <= pos < max_pages*page_size; any
 *              order; slots 0..pos must hold that sequence's cache entries
 *   page_table device int32 [B][max_pages]
 *   out        device bf16 [B][Tq][Hq][d]
 * No workspace.  Slots beyond the largest position of a 128-row tile may hold
 * anything (NaN included).  bf16 caches only, page_size >= 8, B and Hq at
 * most 65535 (else WM_ERR_UNSUPPORTED).  A bad position zero-fills that row
 * and sets WM_ERR_BOUNDS; a bad page id reads zeros for its slots and sets
 * WM_ERR_BOUNDS.  B = 0 or Tq = 0 is a no-op.  Launches chain with
 * programmatic dependent launch like wm_decode_attn.
 */
wm_status wm_prefill_attn(const wm_config* cfg, const wm_cache* cache, int32_t layer,
                          const void* q, const int32_t* pos, const int32_t* page_table,
                          int32_t B, int32_t Tq, int32_t max_pages, void* out,
                          int32_t* dev_status, void* stream);

/*
 * Self-test of the kernels' failure detection (no counterpart in the paper).
 * Every pipeline wait in this library is bounded; when a wait runs out the
 * kernel writes WM_ERR_TIMEOUT to the status word and returns instead of
 * hanging.  This launches one block that waits on a barrier that nothing
 * will complete, with a limit of limit_us microseconds (1 .. 2,000,000), so a
 * caller can check on its GPU that the status comes back and the context
 * stays usable.  dev_status: device int32, as for the other entry points.
 */
wm_status wm_selftest_bounded_wait(int32_t* dev_status, uint32_t limit_us, void* stream);

/*
 * Decode attention for callers that cannot allocate device memory.
 *
 * The paper has no counterpart: this is a deployment variant of
 * wm_decode_attn.  Some callers cannot provide the workspace that
 * wm_decode_attn asks for: for example a plugin running inside a host
 * program whose allocator owns all device memory and does not let it
 * allocate, or a caller working to a fixed memory plan with no room for
 * scratch.  This entry point computes exactly what wm_decode_attn computes,
 * with the same arguments minus the workspace, and allocates nothing: its
 * scratch is a fixed array of WM_NOALLOC_SCRATCH_BYTES bytes inside the
 * library's device image, which every GPU that loads the library keeps
 * until the process exits.
 *
 *  - The first call on a device looks up that array's device address
 *    (cudaGetSymbolAddress) with the device current; make that first call
 *    before any stream capture.
 *  - Each call checks every argument first; only then does it clear the
 *    span of the array its launch uses (arrival tickets and partial records,
 *    so that nothing a call that timed out left behind counts as published)
 *    with an asynchronous memset on `stream`, and launch.  A call refused on
 *    the host writes nothing to the array.
 *  - All calls in the process share the one array per device: calls that
 *    overlap on the GPU (different streams without ordering) race and give
 *    wrong results.  Serialise them, e.g. on one stream.
 *  - Returns WM_ERR_UNSUPPORTED when the launch would need more scratch than
 *    WM_NOALLOC_SCRATCH_BYTES (large batch x heads x group sizes); use
 *    wm_decode_attn with a workspace then.  Other errors as wm_decode_attn.
 */
#define WM_NOALLOC_SCRATCH_BYTES (8u << 20)

wm_status wm_decode_attn_noalloc(const wm_config* cfg, const wm_cache* cache, int32_t layer,
                                 const void* q, const int32_t* page_table,
                                 const int32_t* seq_lens, int32_t B, int32_t max_pages,
                                 void* out, int32_t* dev_status, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* WM_H_ */
