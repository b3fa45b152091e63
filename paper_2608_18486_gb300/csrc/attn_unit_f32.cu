// Instantiations of the unit-split decode attention kernel for f32 caches.
#include "attn_unit.cuh"

namespace wm {

cudaError_t launch_attn_unit_f32(const AttnParams& p, int stage_bytes, int d, int G, int units,
                                int cluster, size_t smem, cudaStream_t s) {
  using namespace attn_unit_detail;
  if (stage_bytes == 8192) {
    if (d == 64) return launch_unit_g<float, 64, 8192>(p, G, units, cluster, smem, s);
    if (d == 96) return launch_unit_g<float, 96, 8192>(p, G, units, cluster, smem, s);
    if (d == 128) return launch_unit_g<float, 128, 8192>(p, G, units, cluster, smem, s);
  }
  return cudaErrorInvalidValue;
}

int attn_unit_max_clusters_f32(int stage_bytes, int d, int G, int cluster, size_t smem) {
  using namespace attn_unit_detail;
  if (stage_bytes == 8192) {
    if (d == 64) return max_clusters_g<float, 64, 8192>(G, cluster, smem);
    if (d == 96) return max_clusters_g<float, 96, 8192>(G, cluster, smem);
    if (d == 128) return max_clusters_g<float, 128, 8192>(G, cluster, smem);
  }
  return 0;
}

}  // namespace wm
