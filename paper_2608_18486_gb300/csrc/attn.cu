// Host side of the decode attention (kernel in attn_kernel.cuh): stage
// geometry shared with the planner, shared-memory size and dtype dispatch.
#include "attn_kernel.cuh"

namespace wm {

int attn_stage_slots(int stage_bytes, int dtype, int d) {
  const int row = 2 * d * (dtype == WM_DT_F32 ? 4 : 2);  // K + V bytes of one slot
  int slots = 1;
  while (slots * 2 * row <= stage_bytes && slots < 32) slots *= 2;
  return slots;
}

int attn_warps_per_cta() { return attn_detail::kWarps; }

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

}  // namespace wm
