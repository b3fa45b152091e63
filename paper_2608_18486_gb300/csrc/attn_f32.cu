// Instantiations of the decode attention kernel for fp32 caches.
#include "attn_kernel.cuh"

namespace wm {

cudaError_t launch_attn_f32(const AttnParams& p, int stage_bytes, int d, int G, int grid, size_t smem,
                             cudaStream_t s) {
  using namespace attn_detail;
  if (stage_bytes == 8192) {
    if (d == 64) return launch_g<float, 64, 8192>(p, G, grid, smem, s);
    if (d == 96) return launch_g<float, 96, 8192>(p, G, grid, smem, s);
    if (d == 128) return launch_g<float, 128, 8192>(p, G, grid, smem, s);
  }
  return cudaErrorInvalidValue;
}

}  // namespace wm
