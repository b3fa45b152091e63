// C ABI of libwm (declared in include/wm.h): argument checks, workspace
// planning and kernel dispatch.  All device memory belongs to the caller.
#include <math.h>
#include <string.h>

#include <atomic>
#include <mutex>

#include "common.cuh"
#include "internal.h"
#include "wm.h"

namespace {

constexpr int kMaxDevices = 64;
int g_sm_count[kMaxDevices];  // per-device attribute cache (0 = not yet read)

int sm_count() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0) return 148;
  if (dev < kMaxDevices && g_sm_count[dev] > 0) return g_sm_count[dev];
  int n = 0;
  if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0)
    n = 148;
  if (dev < kMaxDevices) g_sm_count[dev] = n;
  return n;
}

bool is_pow2(int x) { return x > 0 && (x & (x - 1)) == 0; }
int ilog2(int x) {
  int r = 0;
  while ((1 << r) < x) ++r;
  return r;
}
size_t elem_size(int dtype) { return dtype == WM_DT_F32 ? 4 : 2; }
size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }
bool aligned(const void* p, size_t a) { return ((uintptr_t)p % a) == 0; }

// Persistent grid of one attention launch and its workspace layout.
struct AttnPlan {
  int stage_bytes, grid, nwarps, chunk_stages, max_chunks;
  int unit_ctas;  // > 0: unit split, one cluster of this many CTAs per unit
  size_t off_part, off_counters, total;
};

constexpr int kAttnMaxBatch = 4096;
constexpr uint32_t kAttnFlags = WM_ATTN_INPUTS_READY | WM_ATTN_DYNAMIC_SPLIT | WM_ATTN_UNIT_SPLIT;
// K + V bytes of one pipeline stage: 8 KB, 2 CTAs (8 warps) per SM.  A warp
// spends about as long on the bookkeeping of a stage (wait, copy issue,
// piece checks) as on its math, so 4 KB stages at 4 CTAs per SM were
// slower (24.0 vs 21.0 us on a 100 MB launch measured side by side).
constexpr int kAttnStageBytes = 8192;
// Launches reading at least this many KV bytes hand out work dynamically:
// chunks of the stage stream taken from an atomic counter, up to
// kAttnChunksPerWarp per warp, so warps that stream faster take more.
// Smaller launches split statically, one chunk per warp: their chunk ends
// (partial publish + ticket) would cost more than the balance gains.
constexpr double kAttnDynamicLaunchBytes = 2.0e9;
constexpr int kAttnChunksPerWarp = 16;
// ... but a unit (sequence, kv head) is cut into at most about this many
// pieces: the warp completing a unit merges one record per piece, so long
// units (few sequences of long context) take coarser chunks.  Measured on
// one GB300 (attention GB/s of measured peak, chunks per warp 2 / 8 / 16):
// 131072 slots x 1 sequence 88% / 75% / 61%, x 8 sequences 100% / 104% /
// 107%; 32 ragged sequences of 4096-8192 slots 86% / 100% / 102%.
constexpr int kAttnPiecesPerUnit = 64;
constexpr int kAttnMinChunkStages = 4;  // > the per-warp ring depth
// Fewest stages a warp is given when the work cannot fill the SMs (8 was
// measured as well: the same time on the paper's 38 MB layer).
constexpr int kAttnMinStagesPerWarp = 4;

// Most work chunks any launch on this device can cut: a full grid of warps
// (attn_ctas_per_sm CTAs per SM) times kAttnChunksPerWarp.
// A static split has at most one chunk per warp; a dynamic one chunks of
// ceil(NS / (warps * kAttnChunksPerWarp)) stages or more, so at most
// warps * kAttnChunksPerWarp of them.
// Unit split (one cluster of C CTAs per (sequence, kv head) unit, merged on
// chip) instead of a static stream-K split when, with the largest C at which
// every cluster is resident at once, it runs at least this share of the
// stream-K grid's warps.  Its merge costs a fraction of stream-K's cross-SM
// one, so it wins even with fewer warps: measured side by side, 10.5 vs 17.4
// us per launch on the paper's model shape (48 units, clusters of 8 CTAs of
// 4 warps) and 17.4 vs 20.2 us on 192 units of 2048 tokens (C = 1, 768
// warps against 1216).  It is static, so it suits units of similar length,
// which the small launches of one decode step have.  Launches of 2 GB or
// more take it only for a single sequence, whose units all have the same
// length (one sequence of 131072 slots, 32 units in clusters of 8: 317 vs
// 357 us per launch on stream-K); with more sequences the lengths may differ
// and stream-K balances them.
constexpr double kAttnUnitMinWarpShare = 0.6;

// Resident clusters of C unit-split CTAs for (dtype, d, G) on this device,
// cached (0: unknown or no device).
int unit_max_clusters(int dtype, int d, int G, int C) {
  static std::atomic<int> cache[kMaxDevices][2][3][4][wm::kAttnUnitMaxCluster + 1];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return 0;
  const int di = d == 64 ? 0 : d == 96 ? 1 : d == 128 ? 2 : -1;
  const int gi = G == 1 ? 0 : G == 2 ? 1 : G == 4 ? 2 : G == 8 ? 3 : -1;
  if (di < 0 || gi < 0 || C < 1 || C > wm::kAttnUnitMaxCluster) return 0;
  std::atomic<int>& slot = cache[dev][dtype == WM_DT_F32 ? 1 : 0][di][gi][C];
  int v = slot.load(std::memory_order_relaxed);
  if (v == 0) {
    v = 1 + wm::attn_unit_max_clusters(kAttnStageBytes, dtype, d, G, C);
    slot.store(v, std::memory_order_relaxed);
  }
  return v - 1;
}

int64_t attn_chunk_capacity() {
  return (int64_t)sm_count() * wm::attn_ctas_per_sm(kAttnStageBytes, 1) * wm::attn_warps_per_cta() *
         kAttnChunksPerWarp;
}

AttnPlan attn_plan(const wm_config& c, int32_t B, int32_t max_pages, uint32_t flags = 0) {
  const bool force_dynamic = (flags & WM_ATTN_DYNAMIC_SPLIT) != 0;
  const bool force_unit = (flags & WM_ATTN_UNIT_SPLIT) != 0;
  AttnPlan pl{};
  const int64_t max_slots = (int64_t)max_pages * c.page_size;
  const double kv_bytes = (double)B * c.Hkv * max_slots * 2.0 * c.d * elem_size(c.dtype);
  pl.stage_bytes = kAttnStageBytes;
  const int ctas_per_sm = wm::attn_ctas_per_sm(pl.stage_bytes, c.Hq / c.Hkv);
  const int stage = wm::attn_stage_slots(pl.stage_bytes, c.dtype, c.d);
  const int64_t ns_max = (int64_t)B * c.Hkv * ((max_slots + stage - 1) / stage);
  const int wpc = wm::attn_warps_per_cta();
  // fill the SMs, but keep at least kAttnMinStagesPerWarp stages per warp
  int64_t grid = (int64_t)sm_count() * ctas_per_sm;
  const int64_t by_work =
      (ns_max + (int64_t)kAttnMinStagesPerWarp * wpc - 1) / ((int64_t)kAttnMinStagesPerWarp * wpc);
  if (by_work < grid) grid = by_work;
  if (grid < 1) grid = 1;
  pl.grid = (int)grid;
  pl.nwarps = (int)grid * wpc;
  if (force_dynamic || kv_bytes >= kAttnDynamicLaunchBytes) {
    int64_t ch = (ns_max + (int64_t)pl.nwarps * kAttnChunksPerWarp - 1) /
                 ((int64_t)pl.nwarps * kAttnChunksPerWarp);
    const int64_t unit_stages = (max_slots + stage - 1) / stage;
    const int64_t by_pieces = (unit_stages + kAttnPiecesPerUnit - 1) / kAttnPiecesPerUnit;
    if (ch < by_pieces) ch = by_pieces;
    if (ch < kAttnMinChunkStages) ch = kAttnMinChunkStages;
    pl.chunk_stages = (int)ch;
    pl.max_chunks = (int)(ns_max / ch > 1 ? ns_max / ch : 1);  // the remainder joins the last chunk
  } else {
    pl.chunk_stages = 0;        // static: the kernel sizes one chunk per warp
    pl.max_chunks = pl.nwarps;  // at most one chunk per warp
  }
  // The counters sit first, at a size that depends only on the device, so a
  // workspace that served one call still has zeros where any later call (any
  // B, max_pages or shape) looks for its counters; the records after them
  // need no initial value (their flags carry the call's epoch).
  const int G = c.Hq / c.Hkv;
  size_t off = 0;
  pl.off_counters = off;
  off += align256(sizeof(int32_t) * (1 + (size_t)attn_chunk_capacity()));
  pl.off_part = off;
  off += align256(sizeof(float) * 2 * (size_t)pl.max_chunks * wm::attn_part_rec(G, c.d));
  pl.total = off;
  // the unit split (it needs no workspace; the stream-K layout above stays
  // the size the workspace query reports)
  const int64_t units = (int64_t)B * c.Hkv;
  const int nsm = sm_count();
  const int unit_warps = wm::attn_unit_warps_per_cta(pl.stage_bytes, c.dtype, c.d, G);
  if (force_unit) {
    int64_t C = nsm / units;
    pl.unit_ctas = (int)(C < 1 ? 1 : C > wm::kAttnUnitMaxCluster ? wm::kAttnUnitMaxCluster : C);
  } else if (!force_dynamic && (pl.chunk_stages == 0 || B == 1) && unit_warps > 0) {
    for (int C = wm::kAttnUnitMaxCluster; C >= 1; --C) {
      if (unit_max_clusters(c.dtype, c.d, G, C) < units) continue;
      if ((double)(units * C * unit_warps) >= kAttnUnitMinWarpShare * pl.nwarps) pl.unit_ctas = C;
      break;
    }
  }
  if (pl.unit_ctas > 0) {
    pl.grid = (int)(units * pl.unit_ctas);
    pl.nwarps = pl.grid * unit_warps;
    pl.chunk_stages = 0;
  }
  return pl;
}

// Shape fields of the pool's launch parameters.
void mix_shape(const wm_config& c, int32_t B, wm::MixParams& p) {
  p.B = B;
  p.L = c.L;
  p.k = c.k;
  p.D = c.D;
  p.Hkv = c.Hkv;
  p.d = c.d;
  p.p = c.p;
  p.Lp = (c.L + c.p - 1) / c.p;
  p.P = c.page_size;
  p.log2P = ilog2(c.page_size);
  p.eps_rms = c.eps_rms;
  p.eps_qk = c.eps_qk;
}

// Tag of one attention call (never 0): a partial record counts as published
// only when its flag holds the tag of the call reading it.
int32_t next_attn_epoch() {
  static std::atomic<uint32_t> counter{0};
  uint32_t e;
  do {
    e = counter.fetch_add(1, std::memory_order_relaxed) + 1;
  } while ((e & 0x7FFFFFFFu) == 0);
  return (int32_t)(e & 0x7FFFFFFFu);
}

wm_status check_cache(const wm_config& c, const wm_cache* cache) {
  if (!cache || !cache->k_pool || !cache->v_pool || cache->num_pages < 1) return WM_ERR_INVALID_ARG;
  if (cache->k != c.k || cache->Hkv != c.Hkv || cache->page_size != c.page_size ||
      cache->d != c.d || cache->dtype != c.dtype)
    return WM_ERR_INVALID_ARG;
  if (!aligned(cache->k_pool, 16) || !aligned(cache->v_pool, 16)) return WM_ERR_INVALID_ARG;
  return WM_OK;
}

// Checks, plans and launches one decode-attention call.  clear_workspace:
// zero the span of the workspace the launch uses (counters and records) on
// the stream just before the launch, after every argument check passed; the
// fixed scratch of wm_decode_attn_noalloc keeps whatever the last call left.
wm_status decode_attn_impl(const wm_config* c, const wm_cache* cache, int32_t layer, const void* q,
                           const int32_t* page_table, const int32_t* seq_lens, int32_t B,
                           int32_t max_pages, void* out, void* workspace, size_t ws_bytes,
                           uint32_t flags, bool clear_workspace, int32_t* dev_status,
                           void* stream) {
  wm_status st = wm_config_check(c);
  if (st != WM_OK) return st;
  if (flags & ~kAttnFlags) return WM_ERR_INVALID_ARG;
  if ((flags & WM_ATTN_DYNAMIC_SPLIT) && (flags & WM_ATTN_UNIT_SPLIT)) return WM_ERR_INVALID_ARG;
  if ((st = check_cache(*c, cache)) != WM_OK) return st;
  if (layer < 0 || layer >= c->L || B < 0 || max_pages < 1) return WM_ERR_INVALID_ARG;
  if ((int64_t)max_pages * c->page_size > INT32_MAX / 2) return WM_ERR_INVALID_ARG;
  if (B == 0) return WM_OK;
  if (B > kAttnMaxBatch) return WM_ERR_UNSUPPORTED;
  if ((int64_t)B * c->Hq > INT32_MAX / 2) return WM_ERR_UNSUPPORTED;  // 32-bit output rows
  if (!q || !page_table || !seq_lens || !out || !workspace) return WM_ERR_INVALID_ARG;
  if (!aligned(q, 16) || !aligned(out, 16) || !aligned(workspace, 256)) return WM_ERR_INVALID_ARG;
  const AttnPlan pl = attn_plan(*c, B, max_pages, flags);
  if (ws_bytes < pl.total) return WM_ERR_INVALID_ARG;
  if (pl.max_chunks > attn_chunk_capacity()) return WM_ERR_UNSUPPORTED;  // cannot happen

  const int chan = c->chan_of_layer[layer];
  const size_t esz = elem_size(c->dtype);
  const int64_t chan_elems = (int64_t)cache->num_pages * c->Hkv * c->page_size * c->d;
  wm::AttnParams p{};
  p.k_pool = (const char*)cache->k_pool + (size_t)chan * chan_elems * esz;
  p.v_pool = (const char*)cache->v_pool + (size_t)chan * chan_elems * esz;
  p.q = q;
  p.out = out;
  p.page_table = page_table;
  p.seq_lens = seq_lens;
  p.part = (float*)((char*)workspace + pl.off_part);
  p.counters = (int32_t*)((char*)workspace + pl.off_counters);
  p.status = dev_status;
  p.page_stride = (int64_t)c->Hkv * c->page_size * c->d;
  p.Hq = c->Hq;
  p.Hkv = c->Hkv;
  p.P = c->page_size;
  p.log2P = ilog2(c->page_size);
  p.num_pages = cache->num_pages;
  p.max_pages = max_pages;
  p.B = B;
  p.chunk_stages = pl.chunk_stages;
  p.max_chunks = pl.max_chunks;
  p.inputs_ready = (flags & WM_ATTN_INPUTS_READY) ? 1 : 0;
  p.epoch = next_attn_epoch();
  p.qscale = (float)(1.4426950408889634 / sqrt((double)c->d));
  // (the unit split touches no workspace)
  if (clear_workspace && pl.unit_ctas == 0 &&
      cudaMemsetAsync(workspace, 0, pl.total, (cudaStream_t)stream) != cudaSuccess)
    return WM_ERR_CUDA;
  cudaError_t e =
      pl.unit_ctas > 0
          ? wm::launch_decode_attn_unit(p, pl.stage_bytes, c->dtype, c->d, c->Hq / c->Hkv,
                                        B * c->Hkv, pl.unit_ctas, (cudaStream_t)stream)
          : wm::launch_decode_attn(p, pl.stage_bytes, c->dtype, c->d, c->Hq / c->Hkv, pl.grid,
                                   (cudaStream_t)stream);
  return e == cudaSuccess ? WM_OK : WM_ERR_CUDA;
}

}  // namespace

extern "C" {

const char* wm_status_string(wm_status s) {
  switch (s) {
    case WM_OK: return "ok";
    case WM_ERR_INVALID_ARG: return "invalid argument";
    case WM_ERR_UNSUPPORTED: return "unsupported configuration";
    case WM_ERR_CUDA: return "CUDA error";
    case WM_ERR_BOUNDS: return "index out of bounds (device)";
    case WM_ERR_TIMEOUT: return "pipeline wait timed out (device)";
  }
  return "unknown status";
}

wm_status wm_config_check(const wm_config* c) {
  if (!c) return WM_ERR_INVALID_ARG;
  if (c->L < 1 || c->L > WM_MAX_L || c->k < 1 || c->k > c->L || c->D < 1 || c->Hkv < 1 ||
      c->Hq < 1 || c->Hq % c->Hkv != 0 || c->d < 2 || c->p < 1 || c->page_size < 1 ||
      !(c->eps_rms >= 0.f) || !(c->eps_qk >= 0.f) || !(c->rope_theta > 0.0))
    return WM_ERR_INVALID_ARG;
  if (c->dtype != WM_DT_F32 && c->dtype != WM_DT_BF16) return WM_ERR_INVALID_ARG;
  for (int l = 0; l < c->L; ++l)
    if (c->chan_of_layer[l] < 0 || c->chan_of_layer[l] >= c->k) return WM_ERR_INVALID_ARG;
  // shapes this library builds
  if (c->d != 64 && c->d != 96 && c->d != 128) return WM_ERR_UNSUPPORTED;
  const int G = c->Hq / c->Hkv;
  if (G != 1 && G != 2 && G != 4 && G != 8) return WM_ERR_UNSUPPORTED;
  if (c->D % 8 != 0 || c->D > 4096) return WM_ERR_UNSUPPORTED;
  if (!is_pow2(c->page_size) || c->page_size > 4096) return WM_ERR_UNSUPPORTED;
  return WM_OK;
}

size_t wm_cache_bytes(const wm_config* c, int32_t num_pages) {
  if (wm_config_check(c) != WM_OK || num_pages < 1) return 0;
  const size_t pool = (size_t)c->k * num_pages * c->Hkv * c->page_size * c->d * elem_size(c->dtype);
  return 2 * align256(pool);
}

wm_status wm_cache_alloc(const wm_config* c, void* dev_buf, size_t bytes, int32_t num_pages,
                         wm_cache* out) {
  wm_status st = wm_config_check(c);
  if (st != WM_OK) return st;
  if (!dev_buf || !out || num_pages < 1 || !aligned(dev_buf, 256)) return WM_ERR_INVALID_ARG;
  const size_t need = wm_cache_bytes(c, num_pages);
  if (need == 0 || bytes < need) return WM_ERR_INVALID_ARG;
  memset(out, 0, sizeof *out);
  out->k_pool = dev_buf;
  out->v_pool = (char*)dev_buf + need / 2;
  out->num_pages = num_pages;
  out->k = c->k;
  out->Hkv = c->Hkv;
  out->page_size = c->page_size;
  out->d = c->d;
  out->dtype = c->dtype;
  return WM_OK;
}

size_t wm_decode_attn_workspace(const wm_config* c, int32_t B, int32_t max_pages) {
  if (wm_config_check(c) != WM_OK || B < 0 || max_pages < 1) return 0;
  if (B == 0) return 256;
  // enough for either split (WM_ATTN_DYNAMIC_SPLIT may cut more chunks)
  const size_t a = attn_plan(*c, B, max_pages, 0u).total;
  const size_t b = attn_plan(*c, B, max_pages, WM_ATTN_DYNAMIC_SPLIT).total;
  return a > b ? a : b;
}

wm_status wm_decode_attn_plan(const wm_config* c, int32_t B, int32_t max_pages, uint32_t flags,
                              int32_t plan[5]) {
  if (wm_config_check(c) != WM_OK || B < 1 || max_pages < 1 || !plan) return WM_ERR_INVALID_ARG;
  if (flags & ~kAttnFlags) return WM_ERR_INVALID_ARG;
  if ((flags & WM_ATTN_DYNAMIC_SPLIT) && (flags & WM_ATTN_UNIT_SPLIT)) return WM_ERR_INVALID_ARG;
  const AttnPlan pl = attn_plan(*c, B, max_pages, flags);
  plan[0] = pl.grid;
  plan[1] = pl.nwarps;
  plan[2] = pl.max_chunks;
  plan[3] = pl.chunk_stages;
  plan[4] = pl.unit_ctas;
  return WM_OK;
}

wm_status wm_decode_attn(const wm_config* c, const wm_cache* cache, int32_t layer, const void* q,
                         const int32_t* page_table, const int32_t* seq_lens, int32_t B,
                         int32_t max_pages, void* out, void* workspace, size_t ws_bytes,
                         int32_t* dev_status, void* stream) {
  return wm_decode_attn_flags(c, cache, layer, q, page_table, seq_lens, B, max_pages, out,
                              workspace, ws_bytes, 0u, dev_status, stream);
}

wm_status wm_decode_attn_flags(const wm_config* c, const wm_cache* cache, int32_t layer,
                               const void* q, const int32_t* page_table, const int32_t* seq_lens,
                               int32_t B, int32_t max_pages, void* out, void* workspace,
                               size_t ws_bytes, uint32_t flags, int32_t* dev_status, void* stream) {
  return decode_attn_impl(c, cache, layer, q, page_table, seq_lens, B, max_pages, out, workspace,
                          ws_bytes, flags, false, dev_status, stream);
}

wm_status wm_prefill_attn(const wm_config* c, const wm_cache* cache, int32_t layer,
                          const void* q, const int32_t* pos, const int32_t* page_table,
                          int32_t B, int32_t Tq, int32_t max_pages, void* out,
                          int32_t* dev_status, void* stream) {
  wm_status st = wm_config_check(c);
  if (st != WM_OK) return st;
  if ((st = check_cache(*c, cache)) != WM_OK) return st;
  if (layer < 0 || layer >= c->L || B < 0 || Tq < 0 || max_pages < 1) return WM_ERR_INVALID_ARG;
  if (c->dtype != WM_DT_BF16 || c->page_size < 8) return WM_ERR_UNSUPPORTED;
  if (B > 65535 || c->Hq > 65535) return WM_ERR_UNSUPPORTED;
  if ((int64_t)max_pages * c->page_size > INT32_MAX / 2) return WM_ERR_INVALID_ARG;
  if ((int64_t)B * Tq >= INT32_MAX) return WM_ERR_UNSUPPORTED;
  if ((int64_t)c->k * cache->num_pages * c->Hkv * c->page_size >= INT32_MAX)
    return WM_ERR_UNSUPPORTED;  // TMA row coordinates are 32-bit
  if (B == 0 || Tq == 0) return WM_OK;
  if (!q || !pos || !page_table || !out) return WM_ERR_INVALID_ARG;
  if (!aligned(q, 16) || !aligned(out, 16)) return WM_ERR_INVALID_ARG;
  if (!wm::tma_available()) return WM_ERR_CUDA;
  wm::PrefillLaunch L{};
  L.q = q;
  L.pos = pos;
  L.page_table = page_table;
  L.out = out;
  L.status = dev_status;
  L.k_pool = cache->k_pool;
  L.v_pool = cache->v_pool;
  L.B = B;
  L.Tq = Tq;
  L.Hq = c->Hq;
  L.Hkv = c->Hkv;
  L.d = c->d;
  L.k = c->k;
  L.chan = c->chan_of_layer[layer];
  L.num_pages = cache->num_pages;
  L.max_pages = max_pages;
  L.P = c->page_size;
  const cudaError_t e = wm::launch_prefill_attn(L, (cudaStream_t)stream);
  if (e == cudaErrorInvalidValue) return WM_ERR_INVALID_ARG;  // the tensor-map encoder refused
  return e == cudaSuccess ? WM_OK : WM_ERR_CUDA;
}

size_t wm_kv_mix_workspace(const wm_config* c, int32_t B) {
  if (wm_config_check(c) != WM_OK || B < 0) return 0;
  if (B == 0) return 256;
  return wm::mix_workspace_layout(*c, B, sm_count()).total;
}

int32_t wm_kv_mix_launches(const wm_config* c, int32_t B) {
  if (wm_config_check(c) != WM_OK || B < 0) return -1;
  wm::MixParams p{};
  mix_shape(*c, B, p);
  p.num_pages = 1;
  p.max_pages = 1;
  return wm::kv_mix_launches(p, c->dtype);
}

wm_status wm_kv_mix(const wm_config* c, const wm_cache* cache, const wm_mix_weights* w,
                    const void* h, const int32_t* page_table, const int32_t* slot, int32_t B,
                    int32_t max_pages, void* workspace, size_t ws_bytes, int32_t* dev_status,
                    void* stream) {
  wm_status st = wm_config_check(c);
  if (st != WM_OK) return st;
  if ((st = check_cache(*c, cache)) != WM_OK) return st;
  if (B < 0 || max_pages < 1 || !w) return WM_ERR_INVALID_ARG;
  if ((int64_t)max_pages * c->page_size > INT32_MAX / 2) return WM_ERR_INVALID_ARG;
  if (B == 0) return WM_OK;
  if (B > 65535) return WM_ERR_UNSUPPORTED;
  if (!h || !page_table || !slot || !workspace || !w->qk_g) return WM_ERR_INVALID_ARG;
  for (int X = 0; X < 2; ++X)
    if (!w->pre_g[X] || !w->Wr[X] || !w->br[X] || !w->ch_g[X] || !w->Wkv[X])
      return WM_ERR_INVALID_ARG;
  for (int X = 0; X < 2; ++X)
    if (!aligned(w->Wr[X], 16) || !aligned(w->Wkv[X], 16) || !aligned(w->pre_g[X], 16) ||
        !aligned(w->ch_g[X], 16))
      return WM_ERR_INVALID_ARG;
  if (!aligned(h, 16)) return WM_ERR_INVALID_ARG;
  if (!aligned(workspace, 256)) return WM_ERR_INVALID_ARG;
  const wm::MixWorkspace ws = wm::mix_workspace_layout(*c, B, sm_count());
  if (ws_bytes < ws.total) return WM_ERR_INVALID_ARG;

  wm::MixParams p{};
  mix_shape(*c, B, p);
  p.num_pages = cache->num_pages;
  p.max_pages = max_pages;
  p.h = h;
  for (int X = 0; X < 2; ++X) {
    p.pre_g[X] = w->pre_g[X];
    p.Wr[X] = w->Wr[X];
    p.br[X] = w->br[X];
    p.ch_g[X] = w->ch_g[X];
    p.Wkv[X] = w->Wkv[X];
  }
  p.qk_g = w->qk_g;
  p.page_table = page_table;
  p.slot = slot;
  p.k_pool = cache->k_pool;
  p.v_pool = cache->v_pool;
  char* base = (char*)workspace;
  p.inv_rms = (float*)(base + ws.inv_rms);
  p.xi = base + ws.xi;
  p.zpart = (float*)(base + ws.zpart);
  p.rope_cs = (float*)(base + ws.rope_cs);
  p.xop = base + ws.xop;
  p.proj = (float*)(base + ws.proj);
  p.nsplit_r = ws.nsplit_r;
  p.status = dev_status;
  for (int i = 0; i < c->d / 2 && i < wm::kMaxRopeHalf; ++i)
    p.inv_freq[i] = pow(c->rope_theta, -2.0 * i / c->d);
  cudaError_t e = wm::launch_kv_mix(p, c->dtype, (cudaStream_t)stream);
  return e == cudaSuccess ? WM_OK : WM_ERR_CUDA;
}

}  // extern "C"

// ------------------------------------------------------------------------
// Self-test of the bounded pipeline wait: one thread waits on an mbarrier
// that nothing arrives on, with the same helper the kernels use, gives up
// after limit_us microseconds and reports WM_ERR_TIMEOUT.
namespace {
__global__ void wait_selftest_kernel(int32_t* status, uint64_t limit_ns) {
  __shared__ uint64_t bar;
  if (threadIdx.x != 0) return;
  wm::mbar_init(&bar, 1);
  wm::fence_mbar_init();
  if (!wm::mbar_wait(&bar, 0, limit_ns)) wm::report(status, WM_ERR_TIMEOUT);
  // the barrier's pending arrival is never made; shared memory is released
  // with the block
}
}  // namespace

extern "C" wm_status wm_selftest_bounded_wait(int32_t* dev_status, uint32_t limit_us,
                                              void* stream) {
  if (!dev_status || limit_us == 0 || limit_us > 2000000u) return WM_ERR_INVALID_ARG;
  wait_selftest_kernel<<<1, 32, 0, (cudaStream_t)stream>>>(dev_status, (uint64_t)limit_us * 1000ull);
  return cudaGetLastError() == cudaSuccess ? WM_OK : WM_ERR_CUDA;
}

// ------------------------------------------------------------------------
// Decode attention without caller-provided scratch.
//
// Some callers cannot hand this library any device memory beyond the inputs
// and outputs of a call: a plugin inside a host program whose allocator owns
// the whole device and forbids other allocations, or a caller with a fixed
// memory plan that has no room for a workspace.  For them the attention's
// scratch (per-warp partial results and arrival tickets) lives in one
// fixed-size array that is part of this library's device image.  Every GPU
// that loads the library holds the array until the process exits.
namespace {

static __device__ __align__(256) unsigned char g_noalloc_scratch[WM_NOALLOC_SCRATCH_BYTES];

std::mutex g_noalloc_mu;
void* g_noalloc_ptr[kMaxDevices];  // device address of the array, per device

// Device address of the array on the current device.  Host code cannot use
// the symbol itself (it names a host-side stand-in), so the address is asked
// for once per device, with that device current.
wm_status noalloc_scratch(void** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return WM_ERR_CUDA;
  std::lock_guard<std::mutex> lock(g_noalloc_mu);
  if (!g_noalloc_ptr[dev]) {
    void* ptr = nullptr;
    if (cudaGetSymbolAddress(&ptr, g_noalloc_scratch) != cudaSuccess || !ptr) return WM_ERR_CUDA;
    g_noalloc_ptr[dev] = ptr;
  }
  *out = g_noalloc_ptr[dev];
  return WM_OK;
}

}  // namespace

extern "C" wm_status wm_decode_attn_noalloc(const wm_config* c, const wm_cache* cache,
                                            int32_t layer, const void* q,
                                            const int32_t* page_table, const int32_t* seq_lens,
                                            int32_t B, int32_t max_pages, void* out,
                                            int32_t* dev_status, void* stream) {
  wm_status st = wm_config_check(c);
  if (st != WM_OK) return st;
  if (B < 0 || max_pages < 1) return WM_ERR_INVALID_ARG;
  if (B == 0) return WM_OK;
  if (B > kAttnMaxBatch) return WM_ERR_UNSUPPORTED;
  const AttnPlan pl = attn_plan(*c, B, max_pages);
  if (pl.total > (size_t)WM_NOALLOC_SCRATCH_BYTES) return WM_ERR_UNSUPPORTED;
  void* scratch = nullptr;
  if ((st = noalloc_scratch(&scratch)) != WM_OK) return st;
  // The array keeps the last call's bytes.  Every argument is checked first;
  // then the span this launch uses (arrival tickets, and the partial records
  // whose flags a call that timed out may have left raised) is zeroed on the
  // stream just before the launch.
  return decode_attn_impl(c, cache, layer, q, page_table, seq_lens, B, max_pages, out, scratch,
                          (size_t)WM_NOALLOC_SCRATCH_BYTES, 0u, true, dev_status, stream);
}
