/*
 * Host fill of the seeded synthetic values, compiled for speed: the same
 * definition as gen.py (which states it and remains the reference) and as
 * synth.cu on the device.  This file holds no arithmetic of the method; it
 * only turns (stream key, flat index) into a value.
 *
 *   raw(i)  = mix64(key + (i + 1) * GAMMA)             (SplitMix64 output i)
 *   n       = (sum of the four 16-bit fields of raw(i) - 131070) * scale
 *   value   = n * std + mean                           (each fp32 operation
 *                                                       rounded separately)
 *   bf16    = round-to-nearest-even of the fp32 value
 *
 * Build with -ffp-contract=off so that no multiply-add is fused.
 */
#include <stdint.h>
#include <string.h>

#ifdef _OPENMP
#include <omp.h>
#endif

static const uint64_t kGamma = 0x9E3779B97F4A7C15ull;

static inline uint64_t mix64(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

static inline float value_of(uint64_t key, uint64_t i, float scale, float std, float mean) {
  const uint64_t z = mix64(key + (i + 1u) * kGamma);
  const int64_t s = (int64_t)((z & 0xFFFFu) + ((z >> 16) & 0xFFFFu) + ((z >> 32) & 0xFFFFu) + (z >> 48));
  const float c = (float)(s - 131070);
  const float n = c * scale;
  const float v = n * std;
  return v + mean;
}

static inline uint16_t bf16_rne(float x) {
  uint32_t u;
  memcpy(&u, &x, sizeof u);
  if ((u & 0x7FFFFFFFu) > 0x7F800000u) return (uint16_t)((u >> 16) | 0x40u);
  return (uint16_t)(((uint64_t)u + 0x7FFFu + ((u >> 16) & 1u)) >> 16);
}

/* out[i] = value at flat index (index ? index[i] : start + i), i < count;
 * dtype 0: float32 out, 1: bf16 bit patterns (uint16) out. */
void wmg_fill(int dtype, uint64_t key, uint64_t start, int64_t count, const uint64_t* index,
              float scale, float std, float mean, void* out, int nthreads) {
#ifdef _OPENMP
  if (nthreads < 1) nthreads = omp_get_max_threads();
#pragma omp parallel for schedule(static) num_threads(nthreads) if (count > (1 << 16))
#endif
  for (int64_t i = 0; i < count; ++i) {
    const uint64_t idx = index ? index[i] : start + (uint64_t)i;
    const float v = value_of(key, idx, scale, std, mean);
    if (dtype == 0)
      ((float*)out)[i] = v;
    else
      ((uint16_t*)out)[i] = bf16_rne(v);
  }
  (void)nthreads;
}

/* out[r * run_len + i] = value at flat index starts[r] + i, for r < nruns and
 * i < run_len: the gather of many contiguous runs (e.g. the pages of one
 * sequence) in one call. */
void wmg_fill_runs(int dtype, uint64_t key, const uint64_t* starts, int64_t nruns, int64_t run_len,
                   float scale, float std, float mean, void* out, int nthreads) {
#ifdef _OPENMP
  if (nthreads < 1) nthreads = omp_get_max_threads();
#pragma omp parallel for schedule(static) num_threads(nthreads) if (nruns * run_len > (1 << 16))
#endif
  for (int64_t r = 0; r < nruns; ++r) {
    for (int64_t i = 0; i < run_len; ++i) {
      const float v = value_of(key, starts[r] + (uint64_t)i, scale, std, mean);
      if (dtype == 0)
        ((float*)out)[r * run_len + i] = v;
      else
        ((uint16_t*)out)[r * run_len + i] = bf16_rne(v);
    }
  }
  (void)nthreads;
}
