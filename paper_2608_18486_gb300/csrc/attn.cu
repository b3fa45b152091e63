// Host side of the decode attention (kernel in attn_kernel.cuh): stage
// geometry shared with the planner, shared-memory size and dtype dispatch.
#include "attn_unit.cuh"

namespace wm {

int attn_stage_slots(int stage_bytes, int dtype, int d) {
  const int row = 2 * d * (dtype == WM_DT_F32 ? 4 : 2);  // K + V bytes of one slot
  int slots = 1;
  while (slots * 2 * row <= stage_bytes && slots < 32) slots *= 2;
  return slots;
}

int attn_warps_per_cta() { return attn_detail::kWarps; }
int attn_unit_warps_per_cta(int stage_bytes, int dtype, int d, int G) {
  using namespace attn_unit_detail;
  if (stage_bytes != 8192) return 0;
  if (dtype == WM_DT_F32) {
    if (d == 64) return unit_warps_g<float, 64, 8192>(G);
    if (d == 96) return unit_warps_g<float, 96, 8192>(G);
    if (d == 128) return unit_warps_g<float, 128, 8192>(G);
    return 0;
  }
  if (d == 64) return unit_warps_g<__nv_bfloat16, 64, 8192>(G);
  if (d == 96) return unit_warps_g<__nv_bfloat16, 96, 8192>(G);
  if (d == 128) return unit_warps_g<__nv_bfloat16, 128, 8192>(G);
  return 0;
}

size_t attn_smem_bytes(int stage_bytes, int dtype, int d, int G, int B) {
  const size_t esz = dtype == WM_DT_F32 ? 4 : 2;
  const size_t stage = (size_t)attn_stage_slots(stage_bytes, dtype, d) * 2 * d * esz;
  return (size_t)attn_detail::kWarps * attn_detail::kWStages * stage +
         (size_t)attn_detail::kWarps * attn_detail::kWStages * G * d * esz +
         sizeof(int) * (2 * (size_t)B + 1);
}

cudaError_t launch_decode_attn(const AttnParams& p, int stage_bytes, int dtype, int d, int G,
                               int grid, cudaStream_t s) {
  const size_t smem = attn_smem_bytes(stage_bytes, dtype, d, G, p.B);
  if (dtype == WM_DT_F32) return launch_attn_f32(p, stage_bytes, d, G, grid, smem, s);
  return launch_attn_bf16(p, stage_bytes, d, G, grid, smem, s);
}

size_t attn_unit_smem_bytes(int stage_bytes, int dtype, int d, int G) {
  const size_t esz = dtype == WM_DT_F32 ? 4 : 2;
  const size_t stage = (size_t)attn_stage_slots(stage_bytes, dtype, d) * 2 * d * esz;
  return (size_t)attn_unit_warps_per_cta(stage_bytes, dtype, d, G) * attn_unit_detail::kUStages * stage +
         (size_t)(attn_unit_detail::unit_rec(G, d) + 3) / 4 * 4 * sizeof(float);
}

int attn_unit_max_clusters(int stage_bytes, int dtype, int d, int G, int cluster) {
  const size_t smem = attn_unit_smem_bytes(stage_bytes, dtype, d, G);
  if (dtype == WM_DT_F32) return attn_unit_max_clusters_f32(stage_bytes, d, G, cluster, smem);
  return attn_unit_max_clusters_bf16(stage_bytes, d, G, cluster, smem);
}

cudaError_t launch_decode_attn_unit(const AttnParams& p, int stage_bytes, int dtype, int d, int G,
                                    int units, int cluster, cudaStream_t s) {
  const size_t smem = attn_unit_smem_bytes(stage_bytes, dtype, d, G);
  if (dtype == WM_DT_F32) return launch_attn_unit_f32(p, stage_bytes, d, G, units, cluster, smem, s);
  return launch_attn_unit_bf16(p, stage_bytes, d, G, units, cluster, smem, s);
}

}  // namespace wm
