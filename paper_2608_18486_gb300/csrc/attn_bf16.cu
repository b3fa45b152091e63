// Instantiations of the decode attention kernel for bf16 caches.
#include "attn_kernel.cuh"

namespace wm {

cudaError_t launch_attn_bf16(const AttnParams& p, int stage_bytes, int d, int G, int grid, size_t smem,
                             cudaStream_t s) {
  using namespace attn_detail;
  if (stage_bytes == 8192) {
    if (d == 64) return launch_g<__nv_bfloat16, 64, 8192>(p, G, grid, smem, s);
    if (d == 96) return launch_g<__nv_bfloat16, 96, 8192>(p, G, grid, smem, s);
    if (d == 128) return launch_g<__nv_bfloat16, 128, 8192>(p, G, grid, smem, s);
  }
  return cudaErrorInvalidValue;
}

}  // namespace wm
