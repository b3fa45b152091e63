// Launch interfaces between the C-ABI layer (wm_api.cu) and the kernels.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "wm.h"

namespace wm {

// Opt kernel `kern` into `smem` bytes of dynamic shared memory on the current
// device (the limit is a per-device attribute of the function).  `done`
// holds, per device, the largest value set so far.
constexpr int kSmemOptDevices = 64;
template <typename Kern>
inline cudaError_t opt_in_smem(Kern kern, size_t smem, size_t (&done)[kSmemOptDevices]) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return cudaErrorInvalidDevice;
  const bool cached = dev >= 0 && dev < kSmemOptDevices;
  if (cached && smem <= done[dev]) return cudaSuccess;
  const cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e == cudaSuccess && cached) done[dev] = smem;
  return e;
}

// ------------------------------------------------------------ attention
struct AttnParams {
  const void* k_pool;     // channel c(layer) base of the K pool
  const void* v_pool;     // channel c(layer) base of the V pool
  const void* q;          // [B][Hq][d]
  void* out;              // [B][Hq][d]
  const int32_t* page_table;
  const int32_t* seq_lens;
  float* part;            // [2][max_chunks] records of attn_part_rec(G, d) floats: the
                          // partial of the first piece (side 0) / last piece (side 1) of
                          // each chunk that belongs to a unit crossing a chunk boundary
                          // ([G][d] unnormalised outputs, (max, sum) per query head in
                          // log2 units, then a published flag, zero between launches)
  int32_t* counters;      // [0]: chunk counter; [1 + g]: arrival tickets of the unit whose
                          // first piece ends chunk g; zero between launches
  int32_t* status;
  int64_t page_stride;    // elements between consecutive physical pages
  int32_t B, Hq, Hkv, P, log2P, num_pages, max_pages;
  int32_t chunk_stages;   // stages per work chunk (0: one chunk per warp)
  int32_t max_chunks;     // partial slots per side
  int32_t inputs_ready;   // the previous grid wrote no cache, table, length or workspace
  int32_t epoch;          // nonzero tag of this call: a record is published when its
                          // flag holds this value (a stale word from another call or
                          // layout never matches)
  float qscale;           // log2(e) / sqrt(d)
};

// Resident CTAs per SM the attention kernel is built for: 4 with 4 KB stages
// and one query head per kv head, else 2 (GQA keeps G query rows per lane).
// The planner uses 8 KB stages only.
constexpr int attn_ctas_per_sm(int stage_bytes, int G) { return stage_bytes == 4096 && G == 1 ? 4 : 2; }

// Floats per partial record: G*d outputs, (max, sum) per head, a "published"
// flag word, padded to 16 bytes so that consecutive records can be moved with
// one bulk copy.
constexpr int attn_part_rec(int G, int d) { return G * d + (2 * G + 1 + 3) / 4 * 4; }

int attn_stage_slots(int stage_bytes, int dtype, int d);
int attn_warps_per_cta();
size_t attn_smem_bytes(int stage_bytes, int dtype, int d, int G, int B);
cudaError_t launch_decode_attn(const AttnParams& p, int stage_bytes, int dtype, int d, int G,
                               int grid, cudaStream_t s);
// Unit split (attn_unit.cuh): one cluster of `cluster` CTAs (<= 8) per
// (sequence, kv head) unit, `units` = B * Hkv clusters.
constexpr int kAttnUnitMaxCluster = 8;
int attn_unit_warps_per_cta(int stage_bytes, int dtype, int d, int G);  // 0: unsupported
size_t attn_unit_smem_bytes(int stage_bytes, int dtype, int d, int G);
int attn_unit_max_clusters(int stage_bytes, int dtype, int d, int G, int cluster);
cudaError_t launch_decode_attn_unit(const AttnParams& p, int stage_bytes, int dtype, int d, int G,
                                    int units, int cluster, cudaStream_t s);

// ------------------------------------------------------------ prefill attention
struct PrefillLaunch {
  const void* q;              // [B][Tq][Hq][d] bf16
  const int32_t* pos;         // [B][Tq] token position of each query row
  const int32_t* page_table;  // [B][max_pages]
  void* out;                  // [B][Tq][Hq][d] bf16
  int32_t* status;
  const void* k_pool;         // whole pools, all channels: [k][num_pages][Hkv][P][d]
  const void* v_pool;
  int32_t B, Tq, Hq, Hkv, d, k, chan, num_pages, max_pages, P;
};
cudaError_t launch_prefill_attn(const PrefillLaunch& L, cudaStream_t s);

// ------------------------------------------------------------ TMA tensor maps
// 2-D map of a row-major bf16 matrix [rows][cols] with a row pitch of
// pitch_elems elements (a multiple of 8), a box of 64 columns x box_rows
// rows and 128-byte swizzle; elements outside the matrix read as zero.
// `tm` points at a CUtensorMap.  False if the encoder is missing or refuses.
bool tma_available();
bool tma_map_bf16_2d(void* tm, const void* ptr, uint64_t rows, uint64_t cols, uint64_t pitch_elems,
                     uint32_t box_rows);

// ------------------------------------------------------------ KV pool (mix)
constexpr int kMaxRopeHalf = 64;  // d/2 for d <= 128

struct MixParams {
  // shape
  int32_t B, L, k, D, Hkv, d, p, Lp, P, log2P, num_pages, max_pages;
  float eps_rms, eps_qk;
  // inputs
  const void* h;                  // [B][L][D]
  const void* pre_g[2];
  const void* Wr[2];
  const void* br[2];
  const void* ch_g[2];
  const void* Wkv[2];
  const void* qk_g;
  const int32_t* page_table;
  const int32_t* slot;
  // cache
  void* k_pool;
  void* v_pool;
  // workspace
  float* inv_rms;                 // [B][L]
  void* xi;                       // [2][B][Lp*D] router inputs (dtype of the config)
  float* zpart;                   // [2][nsplit_r][B][k*L] router partial sums
  float* rope_cs;                 // [B][d/2][2] cos, sin at pos = slot - 1
  void* xop;                      // [2][k][B][D] normed channels, dtype
  float* proj;                    // [2][k][B][Hkv*d] projection outputs
  int32_t nsplit_r;
  int32_t* status;
  double inv_freq[kMaxRopeHalf];  // theta^(-2i/d), computed on the host in fp64
};

struct MixWorkspace {
  size_t inv_rms, xi, zpart, rope_cs, xop, proj, total;
  int32_t nsplit_r;
};

MixWorkspace mix_workspace_layout(const wm_config& cfg, int32_t B, int sm_count);
cudaError_t launch_kv_mix(MixParams& p, int dtype, cudaStream_t s);
int kv_mix_launches(const MixParams& p, int dtype);  // kernels launch_kv_mix enqueues

// tcgen05 projection with the fused key/value epilogue, and the tcgen05
// router with split-K fp32 partials (bf16 only)
bool proj_tc_supported(const MixParams& p);
cudaError_t launch_proj_tc(const MixParams& p, cudaStream_t s);
bool router_tc_supported(int B);
int router_tc_splits(int k, int L, int Lp, int D, int B, int sms);
cudaError_t launch_router_tc(const MixParams& p, cudaStream_t s);

}  // namespace wm
