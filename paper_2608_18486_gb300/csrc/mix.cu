// The cross-layer KV pool for a decode batch (Sec. 3.1 Steps 1-2), appended
// to the paged cache (Sec. 3.2).
//
// Kernels, in launch order:
//   1. prenorm   : per (token, layer) inverse RMS of h_l; writes the router
//                  input xi = [hhat_{L-1}, hhat_{L-1-p}, ...] for both branches;
//                  per token the RoPE cos/sin at pos = slot - 1.
//   2. router    : z = Wr[X] xi (split over the L'D reduction), fp32 partials;
//                  tcgen05 for bf16 (proj_tc.cu), SIMT FMA for fp32.
//   3. mix       : alpha = reshape(z + br), htilde_j = sum_l alpha[j][l] hhat_l,
//                  RMSNorm_j, rounded to the projection operand dtype.
//   4. projection: W^X_j x^X_j for every branch and channel; for bf16 on
//                  tcgen05 with the epilogue fused (proj_tc.cu).
//   5. epilogue  : (fp32) keys: per-head QK-norm then RoPE; keys and values
//                  are written to the token's cache slot.
// Every kernel is launched with programmatic dependent launch and waits for
// its predecessor with griddepcontrol.wait before reading anything.
#include <math.h>

#include <utility>

#include "common.cuh"
#include "internal.h"

namespace wm {

namespace {

constexpr int kMixThreads = 256;
constexpr int kChanGroup = 4; // channels mixed per CTA
constexpr int kVecPerThread = 2;  // 8-element vectors per thread: D <= 256*8*2
// Token counts from which the pool runs its batched forms of prenorm and mix
// (prefill groups): several tokens per CTA, whole warps on every row.  Below
// it (decode steps) one token per CTA spreads the few tokens over more SMs.
constexpr int kBatchedTokens = 64;
constexpr int kMixCG = 8;     // channels per CTA in the batched mix
constexpr int kMixLC = 8;     // most layers per staged chunk of h in the batched mix
constexpr size_t kMixStageBudget = 160 * 1024;  // shared memory for the staged chunks

// 16-byte asynchronous global -> shared copies (no registers held while in flight)
__device__ __forceinline__ void cp_async16(void* dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_u32(dst)), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory"); }

__device__ __forceinline__ void pdl_wait() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  asm volatile("griddepcontrol.wait;" ::: "memory");
}

template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                       Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, std::forward<Args>(args)...);
}

// 8 consecutive elements as fp32 (one 16-byte load for bf16, two for fp32)
template <typename T>
__device__ __forceinline__ void load8f(const T* src, float* f);
template <>
__device__ __forceinline__ void load8f<float>(const float* src, float* f) {
  const float4 a = *reinterpret_cast<const float4*>(src);
  const float4 c = *reinterpret_cast<const float4*>(src + 4);
  f[0] = a.x; f[1] = a.y; f[2] = a.z; f[3] = a.w;
  f[4] = c.x; f[5] = c.y; f[6] = c.z; f[7] = c.w;
}
template <>
__device__ __forceinline__ void load8f<__nv_bfloat16>(const __nv_bfloat16* src, float* f) {
  Elem<__nv_bfloat16>::unpack(*reinterpret_cast<const uint4*>(src), f);
}
template <typename T>
__device__ __forceinline__ void store8f(T* dst, const float* f);
template <>
__device__ __forceinline__ void store8f<float>(float* dst, const float* f) {
  *reinterpret_cast<float4*>(dst) = make_float4(f[0], f[1], f[2], f[3]);
  *reinterpret_cast<float4*>(dst + 4) = make_float4(f[4], f[5], f[6], f[7]);
}
template <>
__device__ __forceinline__ void store8f<__nv_bfloat16>(__nv_bfloat16* dst, const float* f) {
  uint4 u;
  __nv_bfloat162 t;
  t = __floats2bfloat162_rn(f[0], f[1]); u.x = *reinterpret_cast<uint32_t*>(&t);
  t = __floats2bfloat162_rn(f[2], f[3]); u.y = *reinterpret_cast<uint32_t*>(&t);
  t = __floats2bfloat162_rn(f[4], f[5]); u.z = *reinterpret_cast<uint32_t*>(&t);
  t = __floats2bfloat162_rn(f[6], f[7]); u.w = *reinterpret_cast<uint32_t*>(&t);
  *reinterpret_cast<uint4*>(dst) = u;
}

// ---------------------------------------------------------------- prenorm
template <typename T>
__global__ void __launch_bounds__(kMixThreads) prenorm_kernel(const MixParams p) {
  __shared__ float red[32];
  __shared__ float s_r;
  const int l = blockIdx.x, b = blockIdx.y, tid = threadIdx.x;
  pdl_wait();
  const T* hp = reinterpret_cast<const T*>(p.h) + ((int64_t)b * p.L + l) * p.D;
  float ss = 0.f;
  for (int e = tid; e < p.D; e += kMixThreads) {
    const float v = ldf(hp + e);
    ss = fmaf(v, v, ss);
  }
  ss = block_sum(ss, red);
  if (tid == 0) {
    s_r = rsqrtf(ss / (float)p.D + p.eps_rms);
    p.inv_rms[b * p.L + l] = s_r;
  }
  __syncthreads();
  const float r = s_r;
  // router input block m holds layer L-1-m*p
  const int from_top = p.L - 1 - l;
  if (from_top % p.p == 0) {
    const int m = from_top / p.p;
    for (int X = 0; X < 2; ++X) {
      const T* g = reinterpret_cast<const T*>(p.pre_g[X]);
      T* xo = reinterpret_cast<T*>(p.xi) + ((int64_t)X * p.B + b) * ((int64_t)p.Lp * p.D) +
              (int64_t)m * p.D;
      for (int e = tid; e < p.D; e += kMixThreads)
        xo[e] = Elem<T>::from_f(ldf(hp + e) * r * ldf(g + e));
    }
  }
  if (l == 0) {
    // RoPE angle pos * theta^(-2i/d) in fp64, reduced to [-pi, pi] before sincosf
    const int s = p.slot[b];
    const double pos = (double)(s - 1);
    for (int i = tid; i < p.d / 2; i += kMixThreads) {
      const double a = pos * p.inv_freq[i];
      const double two_pi = 6.283185307179586476925286766559;
      const float ar = (float)(a - two_pi * rint(a / two_pi));
      float sn, cs;
      sincosf(ar, &sn, &cs);
      p.rope_cs[((int64_t)b * (p.d / 2) + i) * 2] = cs;
      p.rope_cs[((int64_t)b * (p.d / 2) + i) * 2 + 1] = sn;
    }
  }
}

// Batched form: one warp per (token, layer) row, 8 rows per CTA, 16-byte
// vectors.  Same outputs as prenorm_kernel.
template <typename T>
__global__ void __launch_bounds__(kMixThreads) prenorm_rows_kernel(const MixParams p) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int row = blockIdx.x * (kMixThreads / 32) + warp;  // b * L + l
  pdl_wait();
  if (row >= p.B * p.L) return;  // warp-level from here on
  const int b = row / p.L, l = row % p.L;
  const int nvec = p.D / 8;
  const T* hp = reinterpret_cast<const T*>(p.h) + (int64_t)row * p.D;
  float ss = 0.f;
  for (int v = lane; v < nvec; v += 32) {
    float f[8];
    load8f<T>(hp + v * 8, f);
#pragma unroll
    for (int i = 0; i < 8; ++i) ss = fmaf(f[i], f[i], ss);
  }
  const float r = rsqrtf(warp_sum(ss) / (float)p.D + p.eps_rms);
  if (lane == 0) p.inv_rms[row] = r;
  const int from_top = p.L - 1 - l;
  if (from_top % p.p == 0) {  // router input block m holds layer L-1-m*p
    const int m = from_top / p.p;
    for (int X = 0; X < 2; ++X) {
      const T* g = reinterpret_cast<const T*>(p.pre_g[X]);
      T* xo = reinterpret_cast<T*>(p.xi) + ((int64_t)X * p.B + b) * ((int64_t)p.Lp * p.D) +
              (int64_t)m * p.D;
      for (int v = lane; v < nvec; v += 32) {
        float f[8], gv[8];
        load8f<T>(hp + v * 8, f);
        load8f<T>(g + v * 8, gv);
#pragma unroll
        for (int i = 0; i < 8; ++i) f[i] *= r * gv[i];
        store8f<T>(xo + v * 8, f);
      }
    }
  }
  if (l == 0) {
    // RoPE angle pos * theta^(-2i/d) in fp64, reduced to [-pi, pi] before sincosf
    const double pos = (double)(p.slot[b] - 1);
    for (int i = lane; i < p.d / 2; i += 32) {
      const double a = pos * p.inv_freq[i];
      const double two_pi = 6.283185307179586476925286766559;
      const float ar = (float)(a - two_pi * rint(a / two_pi));
      float sn, cs;
      sincosf(ar, &sn, &cs);
      p.rope_cs[((int64_t)b * (p.d / 2) + i) * 2] = cs;
      p.rope_cs[((int64_t)b * (p.d / 2) + i) * 2 + 1] = sn;
    }
  }
}

// ---------------------------------------------------------------- W x^T (SIMT)
// out[z][n][m] = sum_{k in split} W[m][k] * X[n][k], z = batch * nsplit + split.
// Weights of batch item `bi` start at W[bi / per_branch] + (bi % per_branch) * w_stride.
constexpr int BM = 64, BN = 32, BK = 32;

struct GemmArgs {
  const void* W[2];
  int64_t w_stride;      // elements between consecutive items of one branch
  int per_branch;        // batch items per branch
  const void* X;         // [batch][N][K]
  int64_t x_stride;      // elements between batch items of X
  float* out;            // [batch][nsplit][N][M]
  int M, N, K, nsplit, k_per_split;
};

template <typename T>
__device__ __forceinline__ void load8(const T* src, float* f);
template <>
__device__ __forceinline__ void load8<float>(const float* src, float* f) {
  const float4 a = *reinterpret_cast<const float4*>(src);
  const float4 c = *reinterpret_cast<const float4*>(src + 4);
  f[0] = a.x; f[1] = a.y; f[2] = a.z; f[3] = a.w;
  f[4] = c.x; f[5] = c.y; f[6] = c.z; f[7] = c.w;
}
template <>
__device__ __forceinline__ void load8<__nv_bfloat16>(const __nv_bfloat16* src, float* f) {
  Elem<__nv_bfloat16>::unpack(*reinterpret_cast<const uint4*>(src), f);
}

template <typename TW, typename TX>
__global__ void __launch_bounds__(256) gemm_wxT_simt(const GemmArgs a) {
  __shared__ float Ws[BK][BM + 4];
  __shared__ float Xs[BK][BN + 4];
  const int split = blockIdx.z % a.nsplit, bi = blockIdx.z / a.nsplit;
  const int m0 = blockIdx.x * BM, n0 = blockIdx.y * BN;
  const int kbeg = split * a.k_per_split;
  const int kend = min(a.K, kbeg + a.k_per_split);
  const TW* W = reinterpret_cast<const TW*>(a.W[bi / a.per_branch]) +
                (int64_t)(bi % a.per_branch) * a.w_stride;
  const TX* X = reinterpret_cast<const TX*>(a.X) + (int64_t)bi * a.x_stride;
  const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
  pdl_wait();
  float acc[4][2] = {};
  for (int k0 = kbeg; k0 < kend; k0 += BK) {
    {  // W tile: row tid/4, 8 consecutive k
      const int r = tid >> 2, kk = (tid & 3) * 8;
      const int m = m0 + r, k = k0 + kk;
      float f[8];
      if (m < a.M && k + 8 <= kend) {
        load8<TW>(W + (int64_t)m * a.K + k, f);
      } else {
#pragma unroll
        for (int i = 0; i < 8; ++i)
          f[i] = (m < a.M && k + i < kend) ? ldf(W + (int64_t)m * a.K + k + i) : 0.f;
      }
#pragma unroll
      for (int i = 0; i < 8; ++i) Ws[kk + i][r] = f[i];
    }
    {  // X tile: token tid/8, 4 consecutive k
      const int n = tid >> 3, kk = (tid & 7) * 4;
      const int nn = n0 + n, k = k0 + kk;
#pragma unroll
      for (int i = 0; i < 4; ++i)
        Xs[kk + i][n] = (nn < a.N && k + i < kend) ? ldf(X + (int64_t)nn * a.K + k + i) : 0.f;
    }
    __syncthreads();
#pragma unroll 8
    for (int kk = 0; kk < BK; ++kk) {
      const float4 w = *reinterpret_cast<const float4*>(&Ws[kk][tx * 4]);
      const float2 x = *reinterpret_cast<const float2*>(&Xs[kk][ty * 2]);
      acc[0][0] = fmaf(w.x, x.x, acc[0][0]);
      acc[1][0] = fmaf(w.y, x.x, acc[1][0]);
      acc[2][0] = fmaf(w.z, x.x, acc[2][0]);
      acc[3][0] = fmaf(w.w, x.x, acc[3][0]);
      acc[0][1] = fmaf(w.x, x.y, acc[0][1]);
      acc[1][1] = fmaf(w.y, x.y, acc[1][1]);
      acc[2][1] = fmaf(w.z, x.y, acc[2][1]);
      acc[3][1] = fmaf(w.w, x.y, acc[3][1]);
    }
    __syncthreads();
  }
  float* out = a.out + (int64_t)blockIdx.z * a.N * a.M;
#pragma unroll
  for (int j = 0; j < 2; ++j) {
    const int n = n0 + ty * 2 + j;
    if (n >= a.N) continue;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int m = m0 + tx * 4 + i;
      if (m < a.M) out[(int64_t)n * a.M + m] = acc[i][j];
    }
  }
}

// ---------------------------------------------------------------- mix
// One CTA per (token, branch, group of kChanGroup channels).  Thread t owns
// the 8-element vectors t, t + 256 of D, so h, gains and the output move as
// 16-byte vectors.  PRE (decode shapes: L <= kMixPreL, D <= 8 * 256): the
// thread's h vectors of every layer and its gains are loaded before the
// router partials are summed, so the kernel waits for one round of loads.
constexpr int kMixPreL = 16;

template <typename T, bool PRE>
__global__ void __launch_bounds__(kMixThreads) mix_kernel(const MixParams p) {
  extern __shared__ float sm[];  // alpha[kChanGroup][L], r[L]
  __shared__ float red[kMixThreads / 32][kChanGroup];
  float* alpha = sm;
  float* rl = sm + kChanGroup * p.L;
  const int b = blockIdx.x, X = blockIdx.y, j0 = blockIdx.z * kChanGroup;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int nj = min(kChanGroup, p.k - j0);
  const int kL = p.k * p.L;
  const int nvec = p.D / 8;
  const T* hp = reinterpret_cast<const T*>(p.h) + (int64_t)b * p.L * p.D;
  const T* g = reinterpret_cast<const T*>(p.pre_g[X]);
  pdl_wait();
  // PRE: this thread's vector of every layer, of the pre-mix gain and of the
  // channel gains, all in flight before the router partials are read
  uint4 hpre[PRE ? kMixPreL : 1], gpre, cpre[kChanGroup];
  if (PRE && tid < nvec) {
#pragma unroll
    for (int l = 0; l < (PRE ? kMixPreL : 1); ++l)
      if (l < p.L) hpre[l] = __ldg(reinterpret_cast<const uint4*>(hp + (int64_t)l * p.D + tid * 8));
    gpre = __ldg(reinterpret_cast<const uint4*>(g + tid * 8));
#pragma unroll
    for (int jj = 0; jj < kChanGroup; ++jj)
      if (jj < nj)
        cpre[jj] = __ldg(reinterpret_cast<const uint4*>(reinterpret_cast<const T*>(p.ch_g[X]) +
                                                        (int64_t)(j0 + jj) * p.D + tid * 8));
  }
  const T* br = reinterpret_cast<const T*>(p.br[X]);
  // alpha[j][l] = z[j*L + l] = bias + sum of the router's split partials
  for (int i = tid; i < nj * p.L; i += kMixThreads) {
    const int o = j0 * p.L + i;
    const float* zp = p.zpart + ((int64_t)X * p.nsplit_r * p.B + b) * kL + o;
    float z = ldf(br + o);
#pragma unroll 8
    for (int s2 = 0; s2 < p.nsplit_r; ++s2) z += zp[(int64_t)s2 * p.B * kL];
    alpha[i] = z;
  }
  for (int i = tid; i < p.L; i += kMixThreads) rl[i] = p.inv_rms[b * p.L + i];
  __syncthreads();

  float gv[kVecPerThread][8];
  float acc[kChanGroup][kVecPerThread][8];
#pragma unroll
  for (int v = 0; v < kVecPerThread; ++v) {
    const int vi = tid + v * kMixThreads;
    if (PRE) {
      if (v == 0 && vi < nvec) Elem<T>::unpack(gpre, gv[0]);
    } else if (vi < nvec) {
      load8f<T>(g + vi * 8, gv[v]);
    }
#pragma unroll
    for (int jj = 0; jj < kChanGroup; ++jj)
#pragma unroll
      for (int i = 0; i < 8; ++i) acc[jj][v][i] = 0.f;
  }
  if (PRE) {
    if (tid < nvec) {
#pragma unroll
      for (int l = 0; l < (PRE ? kMixPreL : 1); ++l) {
        if (l >= p.L) break;
        const float r = rl[l];
        float a[kChanGroup];
#pragma unroll
        for (int jj = 0; jj < kChanGroup; ++jj) a[jj] = jj < nj ? alpha[jj * p.L + l] : 0.f;
        float hv[8];
        Elem<T>::unpack(hpre[l], hv);
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          const float hh = hv[i] * r * gv[0][i];  // pre-mix RMSNorm with gain
#pragma unroll
          for (int jj = 0; jj < kChanGroup; ++jj) acc[jj][0][i] = fmaf(a[jj], hh, acc[jj][0][i]);
        }
      }
    }
  } else {
#pragma unroll 4
    for (int l = 0; l < p.L; ++l) {
      const float r = rl[l];
      float a[kChanGroup];
#pragma unroll
      for (int jj = 0; jj < kChanGroup; ++jj) a[jj] = jj < nj ? alpha[jj * p.L + l] : 0.f;
#pragma unroll
      for (int v = 0; v < kVecPerThread; ++v) {
        const int vi = tid + v * kMixThreads;
        if (vi < nvec) {
          float hv[8];
          load8f<T>(hp + (int64_t)l * p.D + vi * 8, hv);
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            const float hh = hv[i] * r * gv[v][i];  // pre-mix RMSNorm with gain
#pragma unroll
            for (int jj = 0; jj < kChanGroup; ++jj) acc[jj][v][i] = fmaf(a[jj], hh, acc[jj][v][i]);
          }
        }
      }
    }
  }
  // per-channel sums of squares, reduced over the block for all channels at once
  float ss[kChanGroup];
#pragma unroll
  for (int jj = 0; jj < kChanGroup; ++jj) {
    float t = 0.f;
#pragma unroll
    for (int v = 0; v < kVecPerThread; ++v)
#pragma unroll
      for (int i = 0; i < 8; ++i) t = fmaf(acc[jj][v][i], acc[jj][v][i], t);
    t = warp_sum(t);
    if (lane == 0) red[warp][jj] = t;
  }
  __syncthreads();
#pragma unroll
  for (int jj = 0; jj < kChanGroup; ++jj) {
    float t = 0.f;
#pragma unroll
    for (int w = 0; w < kMixThreads / 32; ++w) t += red[w][jj];
    ss[jj] = rsqrtf(t / (float)p.D + p.eps_rms);
  }
  T* xop = reinterpret_cast<T*>(p.xop);
#pragma unroll
  for (int jj = 0; jj < kChanGroup; ++jj) {
    if (jj >= nj) break;
    const int j = j0 + jj;
    const T* cg = reinterpret_cast<const T*>(p.ch_g[X]) + (int64_t)j * p.D;
    T* xo = xop + (((int64_t)X * p.k + j) * p.B + b) * p.D;
#pragma unroll
    for (int v = 0; v < kVecPerThread; ++v) {
      const int vi = tid + v * kMixThreads;
      if (vi < nvec) {
        float cv[8], o[8];
        if (PRE)
          Elem<T>::unpack(cpre[jj], cv);
        else
          load8f<T>(cg + vi * 8, cv);
#pragma unroll
        for (int i = 0; i < 8; ++i) o[i] = acc[jj][v][i] * ss[jj] * cv[i];
        store8f<T>(xo + vi * 8, o);
      }
    }
  }
}

// Batched form: one CTA per (tb tokens, branch, kMixCG channels); tpt
// threads (whole warps) per token, thread u of a token owning the 8-element
// vectors u, u + tpt, ... of D.  alpha of the CTA's tokens is summed from the
// router's split partials once, into shared memory.  Each thread streams its
// own vectors of h through a private 2 x kMixLC-layer buffer in shared memory
// with asynchronous copies, so many loads are in flight without holding
// registers.
template <typename T, int VPT>
__global__ void __launch_bounds__(kMixThreads) mix_tokens_kernel(const MixParams p, int tpt, int tb,
                                                                  int lc) {
  // alpha[tb][kMixCG][L], rl[tb][L], red[warps][kMixCG], then (16-byte
  // aligned) the h staging buffers [2][lc][VPT][threads] of one vector
  // (8 elements: VB 16-byte units) each; lc <= kMixLC layers per chunk
  extern __shared__ float sm[];
  constexpr int VB = 8 * (int)sizeof(T) / 16;
  const int X = blockIdx.y, j0 = blockIdx.z * kMixCG;
  const int nj = min(kMixCG, p.k - j0);
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int t = tid / tpt, u = tid % tpt;
  const int b0 = blockIdx.x * tb, b = b0 + t;
  const bool live = t < tb && b < p.B;
  const int L = p.L, kL = p.k * p.L, nvec = p.D / 8;
  float* alpha = sm;
  float* rl = alpha + tb * kMixCG * L;
  float* red = rl + tb * L;
  uint4* hbuf = reinterpret_cast<uint4*>(
      (reinterpret_cast<uintptr_t>(red + (blockDim.x / 32) * kMixCG) + 15) & ~static_cast<uintptr_t>(15));
  const int nth = blockDim.x;
  auto hslot = [&](int stage, int l, int v) -> uint4* {
    return hbuf + (((stage * lc + l) * VPT + v) * nth + tid) * VB;
  };
  const T* hp = reinterpret_cast<const T*>(p.h) + (int64_t)b * L * p.D;
  // copies of layers [l0, l0 + lc) of this thread's vectors into `stage`
  auto stage_chunk = [&](int stage, int l0) {
    if (live)
      for (int l = l0; l < min(L, l0 + lc); ++l)
#pragma unroll
        for (int v = 0; v < VPT; ++v) {
          const int vi = u + v * tpt;
          if (vi < nvec)
#pragma unroll
            for (int q = 0; q < VB; ++q)
              cp_async16(hslot(stage, l - l0, v) + q,
                         reinterpret_cast<const uint4*>(hp + (int64_t)l * p.D + vi * 8) + q);
        }
    cp_async_commit();
  };
  pdl_wait();
  stage_chunk(0, 0);
  stage_chunk(1, lc);
  const T* br = reinterpret_cast<const T*>(p.br[X]);
  for (int i = tid; i < tb * nj * L; i += blockDim.x) {
    const int tt = i / (nj * L), rem = i % (nj * L);
    const int bb = b0 + tt, o = j0 * L + rem;
    float z = 0.f;
    if (bb < p.B) {
      z = ldf(br + o);
      const float* zp = p.zpart + ((int64_t)X * p.nsplit_r * p.B + bb) * kL + o;
#pragma unroll 8
      for (int s2 = 0; s2 < p.nsplit_r; ++s2) z += zp[(int64_t)s2 * p.B * kL];
    }
    alpha[tt * kMixCG * L + rem] = z;  // [tt][jj][l] with jj = rem / L, l = rem % L
  }
  for (int i = tid; i < tb * L; i += blockDim.x) {
    const int bb = b0 + i / L;
    rl[i] = bb < p.B ? p.inv_rms[(int64_t)bb * L + i % L] : 0.f;
  }
  __syncthreads();

  const T* g = reinterpret_cast<const T*>(p.pre_g[X]);
  float gv[VPT][8];
  float acc[kMixCG][VPT][8];
#pragma unroll
  for (int v = 0; v < VPT; ++v) {
    const int vi = u + v * tpt;
    if (live && vi < nvec) load8f<T>(g + vi * 8, gv[v]);
#pragma unroll
    for (int jj = 0; jj < kMixCG; ++jj)
#pragma unroll
      for (int i = 0; i < 8; ++i) acc[jj][v][i] = 0.f;
  }
  {
    const float* al = alpha + t * kMixCG * L;
    for (int l0 = 0, c = 0; l0 < L; l0 += lc, ++c) {
      cp_async_wait<1>();  // this thread's copies of chunk c have landed
      for (int l = l0; l < min(L, l0 + lc); ++l) {
      if (!live) break;
      const float r = rl[t * L + l];
      float a[kMixCG];
#pragma unroll
      for (int jj = 0; jj < kMixCG; ++jj) a[jj] = jj < nj ? al[jj * L + l] : 0.f;
#pragma unroll
      for (int v = 0; v < VPT; ++v) {
        const int vi = u + v * tpt;
        if (vi < nvec) {
          float hv[8];
          load8f<T>(reinterpret_cast<const T*>(hslot(c & 1, l - l0, v)), hv);
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            const float hh = hv[i] * r * gv[v][i];  // pre-mix RMSNorm with gain
#pragma unroll
            for (int jj = 0; jj < kMixCG; ++jj) acc[jj][v][i] = fmaf(a[jj], hh, acc[jj][v][i]);
          }
        }
      }
      }
      stage_chunk(c & 1, l0 + 2 * lc);  // refill the buffer just consumed
    }
    cp_async_wait<0>();
  }
  // per-channel sums of squares over the token's warps
#pragma unroll
  for (int jj = 0; jj < kMixCG; ++jj) {
    float q = 0.f;
#pragma unroll
    for (int v = 0; v < VPT; ++v)
#pragma unroll
      for (int i = 0; i < 8; ++i) q = fmaf(acc[jj][v][i], acc[jj][v][i], q);
    q = warp_sum(q);
    if (lane == 0) red[warp * kMixCG + jj] = q;
  }
  __syncthreads();
  if (!live) return;
  const int w0 = t * (tpt / 32), nw = tpt / 32;
  T* xop = reinterpret_cast<T*>(p.xop);
#pragma unroll
  for (int jj = 0; jj < kMixCG; ++jj) {
    if (jj >= nj) break;
    float q = 0.f;
    for (int w = 0; w < nw; ++w) q += red[(w0 + w) * kMixCG + jj];
    const float sc = rsqrtf(q / (float)p.D + p.eps_rms);
    const int j = j0 + jj;
    const T* cg = reinterpret_cast<const T*>(p.ch_g[X]) + (int64_t)j * p.D;
    T* xo = xop + (((int64_t)X * p.k + j) * p.B + b) * p.D;
#pragma unroll
    for (int v = 0; v < VPT; ++v) {
      const int vi = u + v * tpt;
      if (vi < nvec) {
        float cv[8], o[8];
        load8f<T>(cg + vi * 8, cv);
#pragma unroll
        for (int i = 0; i < 8; ++i) o[i] = acc[jj][v][i] * sc * cv[i];
        store8f<T>(xo + vi * 8, o);
      }
    }
  }
}

// ---------------------------------------------------------------- epilogue
// fp32 path: one CTA per (token, channel, branch), a warp per kv head; lane t
// handles the RoPE pairs (i, i + HD/2) for i = t, t + 32, ...
template <typename T, int HD>
__global__ void __launch_bounds__(128) kv_epilogue_kernel(const MixParams p) {
  constexpr int HALF = HD / 2;
  constexpr int NP = (HALF + 31) / 32;
  const int b = blockIdx.x, j = blockIdx.y, X = blockIdx.z;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  pdl_wait();
  const int s = p.slot[b];
  if (s < 1 || s >= p.max_pages * p.P) {
    if (threadIdx.x == 0 && j == 0 && X == 0) report(p.status, WM_ERR_BOUNDS);
    return;
  }
  const int pg = p.page_table[(int64_t)b * p.max_pages + (s >> p.log2P)];
  if (pg < 0 || pg >= p.num_pages) {
    if (threadIdx.x == 0 && j == 0 && X == 0) report(p.status, WM_ERR_BOUNDS);
    return;
  }
  const int nout = p.Hkv * HD;
  const float* src = p.proj + (((int64_t)X * p.k + j) * p.B + b) * nout;
  T* pool = reinterpret_cast<T*>(X == 0 ? p.k_pool : p.v_pool);
  const int64_t base = (((int64_t)j * p.num_pages + pg) * p.Hkv) * p.P + (s & (p.P - 1));
  const T* qg = reinterpret_cast<const T*>(p.qk_g) + (int64_t)j * HD;
  for (int hh = warp; hh < p.Hkv; hh += 4) {
    float y0[NP], y1[NP];
#pragma unroll
    for (int t = 0; t < NP; ++t) {
      const int i = lane + 32 * t;
      y0[t] = i < HALF ? src[hh * HD + i] : 0.f;
      y1[t] = i < HALF ? src[hh * HD + i + HALF] : 0.f;
    }
    if (X == 0) {
      float ss = 0.f;
#pragma unroll
      for (int t = 0; t < NP; ++t) ss = fmaf(y0[t], y0[t], fmaf(y1[t], y1[t], ss));
      ss = warp_sum(ss);
      const float rr = rsqrtf(ss / (float)HD + p.eps_qk);
#pragma unroll
      for (int t = 0; t < NP; ++t) {
        const int i = lane + 32 * t;
        if (i < HALF) {
          const float x0 = y0[t] * rr * ldf(qg + i), x1 = y1[t] * rr * ldf(qg + i + HALF);
          const float cs = p.rope_cs[((int64_t)b * HALF + i) * 2];
          const float sn = p.rope_cs[((int64_t)b * HALF + i) * 2 + 1];
          y0[t] = x0 * cs - x1 * sn;  // rotate-half RoPE
          y1[t] = x1 * cs + x0 * sn;
        }
      }
    }
    T* dst = pool + (base + (int64_t)hh * p.P) * HD;
#pragma unroll
    for (int t = 0; t < NP; ++t) {
      const int i = lane + 32 * t;
      if (i < HALF) {
        dst[i] = Elem<T>::from_f(y0[t]);
        dst[i + HALF] = Elem<T>::from_f(y1[t]);
      }
    }
  }
}

template <typename T>
cudaError_t launch_all(MixParams& p, cudaStream_t s) {
  const int kL = p.k * p.L;
  const bool bf16 = sizeof(T) == 2;
  const bool batched = p.B >= kBatchedTokens;
  cudaError_t e;
  if (batched) {
    const int rows = p.B * p.L, per = kMixThreads / 32;
    e = launch_pdl(prenorm_rows_kernel<T>, dim3((rows + per - 1) / per), dim3(kMixThreads), 0, s,
                   p);
  } else {
    e = launch_pdl(prenorm_kernel<T>, dim3(p.L, p.B), dim3(kMixThreads), 0, s, p);
  }
  if (e != cudaSuccess) return e;
  if (bf16 && router_tc_supported(p.B)) {
    e = launch_router_tc(p, s);
  } else {
    GemmArgs a{};
    a.W[0] = p.Wr[0];
    a.W[1] = p.Wr[1];
    a.w_stride = 0;
    a.per_branch = 1;
    a.X = p.xi;
    a.x_stride = (int64_t)p.B * p.Lp * p.D;
    a.out = p.zpart;
    a.M = kL;
    a.N = p.B;
    a.K = p.Lp * p.D;
    a.nsplit = p.nsplit_r;
    a.k_per_split = ((a.K + p.nsplit_r - 1) / p.nsplit_r + BK - 1) / BK * BK;
    dim3 grid((a.M + BM - 1) / BM, (a.N + BN - 1) / BN, 2 * a.nsplit);
    e = launch_pdl(gemm_wxT_simt<T, T>, grid, dim3(256), 0, s, a);
  }
  if (e != cudaSuccess) return e;
  if (batched) {
    const int nvec = p.D / 8;
    const bool two = nvec > kMixThreads;  // D > 2048: two vectors per thread
    const int per = two ? (nvec + 1) / 2 : nvec;
    const int tpt = (per + 31) / 32 * 32;
    const int tb = tpt >= kMixThreads ? 1 : kMixThreads / tpt;
    const size_t per_layer = (size_t)2 * (two ? 2 : 1) * tb * tpt * 8 * sizeof(T);  // both stages
    int lc = kMixLC;
    while (lc > 1 && (size_t)lc * per_layer > kMixStageBudget) lc /= 2;
    const size_t smem = sizeof(float) * ((size_t)tb * kMixCG * p.L + (size_t)tb * p.L +
                                         (size_t)(tb * tpt / 32) * kMixCG) +
                        16 + (size_t)lc * per_layer;
    dim3 grid((p.B + tb - 1) / tb, 2, (p.k + kMixCG - 1) / kMixCG);
    auto kern = two ? mix_tokens_kernel<T, 2> : mix_tokens_kernel<T, 1>;
    static size_t smem_set[2][kSmemOptDevices] = {};  // per variant and device
    e = opt_in_smem(kern, smem, smem_set[two]);
    if (e != cudaSuccess) return e;
    e = launch_pdl(kern, grid, dim3(tb * tpt), smem, s, p, tpt, tb, lc);
    if (e != cudaSuccess) return e;
  } else {
    const size_t smem = sizeof(float) * (kChanGroup * p.L + p.L);
    dim3 grid(p.B, 2, (p.k + kChanGroup - 1) / kChanGroup);
    bool pre = false;  // bf16 decode shapes: every load issued up front
    if constexpr (sizeof(T) == 2) pre = p.L <= kMixPreL && p.D / 8 <= kMixThreads;
    if constexpr (sizeof(T) == 2) {
      e = pre ? launch_pdl(mix_kernel<T, true>, grid, dim3(kMixThreads), smem, s, p)
              : launch_pdl(mix_kernel<T, false>, grid, dim3(kMixThreads), smem, s, p);
    } else {
      e = launch_pdl(mix_kernel<T, false>, grid, dim3(kMixThreads), smem, s, p);
    }
    if (e != cudaSuccess) return e;
  }
  if (bf16 && proj_tc_supported(p)) {
    // bf16: tensor-core projection, QK-norm, RoPE and cache write in one kernel
    return launch_proj_tc(p, s);
  }
  {
    GemmArgs a{};
    a.W[0] = p.Wkv[0];
    a.W[1] = p.Wkv[1];
    a.w_stride = (int64_t)p.Hkv * p.d * p.D;
    a.per_branch = p.k;
    a.X = p.xop;
    a.x_stride = (int64_t)p.B * p.D;
    a.out = p.proj;
    a.M = p.Hkv * p.d;
    a.N = p.B;
    a.K = p.D;
    a.nsplit = 1;
    a.k_per_split = p.D;
    dim3 grid((a.M + BM - 1) / BM, (a.N + BN - 1) / BN, 2 * p.k);
    e = launch_pdl(gemm_wxT_simt<T, T>, grid, dim3(256), 0, s, a);
    if (e != cudaSuccess) return e;
  }
  {
    dim3 grid(p.B, p.k, 2);
    if (p.d == 64) return launch_pdl(kv_epilogue_kernel<T, 64>, grid, dim3(128), 0, s, p);
    if (p.d == 96) return launch_pdl(kv_epilogue_kernel<T, 96>, grid, dim3(128), 0, s, p);
    return launch_pdl(kv_epilogue_kernel<T, 128>, grid, dim3(128), 0, s, p);
  }
}

size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }

}  // namespace

MixWorkspace mix_workspace_layout(const wm_config& cfg, int32_t B, int sm_count) {
  MixWorkspace w{};
  const int Lp = (cfg.L + cfg.p - 1) / cfg.p;
  const int kL = cfg.k * cfg.L;
  const int64_t Kr = (int64_t)Lp * cfg.D;
  int ns;
  if (cfg.dtype == WM_DT_BF16 && router_tc_supported(B)) {
    ns = router_tc_splits(cfg.k, cfg.L, Lp, cfg.D, B, sm_count);
  } else {
    const int tiles = 2 * ((kL + BM - 1) / BM) * ((B + BN - 1) / BN);
    ns = (2 * sm_count + tiles - 1) / tiles;
    const int max_split = (int)((Kr + 255) / 256);
    ns = ns < 1 ? 1 : (ns > max_split ? max_split : ns);
    // same rounding as the launch: whole BK blocks per split
    const int64_t kps = ((Kr + ns - 1) / ns + BK - 1) / BK * BK;
    ns = (int)((Kr + kps - 1) / kps);
  }
  w.nsplit_r = ns;
  const size_t esz = cfg.dtype == WM_DT_F32 ? 4 : 2;
  size_t off = 0;
  w.inv_rms = off; off += align256(sizeof(float) * B * cfg.L);
  w.xi = off;      off += align256(esz * 2 * (size_t)B * Kr);
  w.zpart = off;   off += align256(sizeof(float) * 2 * (size_t)ns * B * kL);
  w.rope_cs = off; off += align256(sizeof(float) * (size_t)B * cfg.d);
  w.xop = off;     off += align256(esz * 2 * (size_t)cfg.k * B * cfg.D);
  w.proj = off;    off += align256(sizeof(float) * 2 * (size_t)cfg.k * B * cfg.Hkv * cfg.d);
  w.total = off;
  return w;
}

int kv_mix_launches(const MixParams& p, int dtype) {
  if (p.B == 0) return 0;
  // prenorm, router, mix, then the tensor-core projection with its epilogue
  // or a SIMT projection and a separate epilogue
  return dtype == WM_DT_BF16 && proj_tc_supported(p) ? 4 : 5;
}

cudaError_t launch_kv_mix(MixParams& p, int dtype, cudaStream_t s) {
  if (dtype == WM_DT_F32) return launch_all<float>(p, s);
  return launch_all<__nv_bfloat16>(p, s);
}

}  // namespace wm
