// Device side of the counter-based synthetic value generator.
//
// Same definition as gen.py in this folder: the i-th value of stream
// (seed, stream) is the i-th SplitMix64 output (Steele, Lea & Flood,
// OOPSLA 2014) from state key(seed, stream), turned into an approximately
// normal fp32 value by summing its four 16-bit fields, then scaled by std and
// shifted by mean with separately rounded fp32 operations, and stored as fp32
// or as round-to-nearest-even bf16.  No arithmetic of the decode method lives
// here: this only fills input buffers.
#include <cstdint>
#include <cuda_runtime.h>

namespace {

constexpr uint64_t kGamma = 0x9E3779B97F4A7C15ull;

__host__ __device__ inline uint64_t mix64(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

// 1 / sqrt(4 * (65536^2 - 1) / 12), rounded to fp32 on the host at launch.
__device__ inline float normal_value(uint64_t key, uint64_t i, float scale, float stdv,
                                     float mean) {
  uint64_t z = mix64(key + (i + 1ull) * kGamma);
  int64_t s = (int64_t)(z & 0xFFFFull) + (int64_t)((z >> 16) & 0xFFFFull) +
              (int64_t)((z >> 32) & 0xFFFFull) + (int64_t)(z >> 48);
  float c = (float)(s - 131070);
  float n = __fmul_rn(c, scale);
  float v = __fmul_rn(n, stdv);
  return __fadd_rn(v, mean);
}

__device__ inline uint16_t bf16_rne_bits(float f) {
  uint32_t u = __float_as_uint(f);
  if ((u & 0x7FFFFFFFu) > 0x7F800000u) return (uint16_t)((u >> 16) | 0x40u);
  u = u + 0x7FFFu + ((u >> 16) & 1u);
  return (uint16_t)(u >> 16);
}

__global__ void fill_kernel(void* dst, int dtype, uint64_t count, uint64_t key, uint64_t start,
                            float scale, float stdv, float mean) {
  uint64_t tid = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x;
  uint64_t nthr = (uint64_t)gridDim.x * blockDim.x;
  for (uint64_t i = tid; i < count; i += nthr) {
    float v = normal_value(key, start + i, scale, stdv, mean);
    if (dtype == 0)
      reinterpret_cast<float*>(dst)[i] = v;
    else
      reinterpret_cast<uint16_t*>(dst)[i] = bf16_rne_bits(v);
  }
}

}  // namespace

extern "C" {

// Fill dst[0..count) with values start..start+count-1 of stream (seed, stream).
// dtype 0 = fp32, 1 = bf16.  scale must be the fp32 unit-variance factor.
// Returns 0, or the cudaError_t of the launch.
int wms_fill(void* dst, int dtype, uint64_t count, uint64_t seed, uint64_t stream,
             uint64_t start, float scale, float stdv, float mean, void* cuda_stream) {
  if (count == 0) return 0;
  uint64_t key = mix64((seed << 32) + stream + kGamma);
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  uint64_t blocks = (count + 255) / 256;
  uint64_t cap = (uint64_t)(sms > 0 ? sms : 1) * 32;
  if (blocks > cap) blocks = cap;
  fill_kernel<<<(unsigned)blocks, 256, 0, (cudaStream_t)cuda_stream>>>(dst, dtype, count, key,
                                                                       start, scale, stdv, mean);
  return (int)cudaGetLastError();
}

}  // extern "C"
