// Per-channel K/V projection on the tcgen05 tensor cores with a fused
// epilogue (Sec. 3.1 Step 2): K_j = W^K_j x^K_j, V_j = W^V_j x^V_j for the
// B tokens of a decode step, then per-head QK-norm and RoPE on keys, bf16
// rounding and the write to each token's cache slot.
//
// Shape: at decode the token count B is small (16..64) while the weights
// are large (Hkv*d x D per channel and branch), so the weights take the MMA's
// M side ("swap AB"): one CTA computes a 128-row tile of W^X_j against all
// B tokens, D[row][token] in TMEM (128 lanes x N fp32 columns).  The work is
// weight-streaming bound; TMA brings 128x64 weight tiles and Nx64 token
// tiles (128-byte swizzle) through a 4-stage mbarrier pipeline.  Warp 0 lane
// 0 issues TMA, warp 1 lane 0 issues tcgen05.mma; all four warps drain TMEM
// (each warp its 32-lane quadrant) into shared memory, then finish the
// per-(token, head) epilogue with a warp per item.
#include <cudaTypedefs.h>
#include <math.h>

#include "internal.h"
#include "tc.cuh"

namespace wm {

namespace {

constexpr int kTcM = 128;      // weight rows per tile (MMA M)
constexpr int kTcBK = 64;      // K elements per stage (128 bytes of bf16)
constexpr int kTcStages = 4;
constexpr int kTcThreads = 128;

struct ProjTcParams {
  int32_t k, B, Hkv, D, M_item, BN, nk;
  int32_t P, log2P, num_pages, max_pages;
  uint32_t tmem_cols;
  float eps_qk;
  const int32_t* page_table;
  const int32_t* slot;
  __nv_bfloat16* k_pool;
  __nv_bfloat16* v_pool;
  const __nv_bfloat16* qk_g;
  const float* rope_cs;
  int32_t* status;
};

template <int HD>
__global__ void __launch_bounds__(kTcThreads, 1)
    proj_tc_kernel(const __grid_constant__ CUtensorMap tmW0, const __grid_constant__ CUtensorMap tmW1,
                   const __grid_constant__ CUtensorMap tmX, const ProjTcParams p) {
  constexpr int EPL = HD / 32;
  extern __shared__ uint8_t smem_dyn[];
  __shared__ uint64_t full[kTcStages], empty[kTcStages], done;
  __shared__ uint32_t tmem_base;

  const int mt = blockIdx.x, j = blockIdx.y, X = blockIdx.z;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const CUtensorMap* tmW = X == 0 ? &tmW0 : &tmW1;
  uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_dyn) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  const uint32_t a_bytes = kTcM * 128;
  const uint32_t b_bytes = (uint32_t)p.BN * 128;
  uint8_t* As = base;
  uint8_t* Bs = base + kTcStages * a_bytes;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kTcStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    mbar_init(&done, 1);
    fence_mbar_init();
    tc::prefetch_tensormap(tmW);
    tc::prefetch_tensormap(&tmX);
  }
  if (warp == 0) {
    tc::tmem_alloc(&tmem_base, p.tmem_cols);
    tc::tmem_relinquish();
  }
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = tmem_base;
  const int wrow = j * p.M_item + mt * kTcM;
  const int xrow = (X * p.k + j) * p.B;

  if (warp == 0 && lane == 0) {
    // TMA producer
    for (int kb = 0; kb < p.nk; ++kb) {
      const int s = kb % kTcStages;
      if (kb >= kTcStages && !mbar_wait(&empty[s], ((kb / kTcStages) - 1) & 1)) {
        report(p.status, WM_ERR_TIMEOUT);
        break;
      }
      mbar_arrive_expect_tx(&full[s], a_bytes + b_bytes);
      tc::tma_load_2d(As + s * a_bytes, tmW, kb * kTcBK, wrow, &full[s]);
      tc::tma_load_2d(Bs + s * b_bytes, &tmX, kb * kTcBK, xrow, &full[s]);
    }
  } else if (warp == 1 && lane == 0) {
    // MMA issuer: 4 MMAs of K = 16 per stage
    const uint32_t idesc = tc::idesc_bf16_f32(kTcM, p.BN);
    for (int kb = 0; kb < p.nk; ++kb) {
      const int s = kb % kTcStages;
      if (!mbar_wait(&full[s], (kb / kTcStages) & 1)) {
        report(p.status, WM_ERR_TIMEOUT);
        break;
      }
      tc::fence_after_sync();
      const uint32_t a0 = smem_u32(As + s * a_bytes), b0 = smem_u32(Bs + s * b_bytes);
#pragma unroll
      for (int kk = 0; kk < kTcBK / 16; ++kk)
        tc::mma_bf16(tmem, tc::sdesc_kmajor_sw128(a0 + kk * 32), tc::sdesc_kmajor_sw128(b0 + kk * 32),
                     idesc, (kb | kk) != 0);
      tc::mma_commit(&empty[s]);  // the stage is free once these MMAs finish
    }
    tc::mma_commit(&done);  // always issued: fires when every MMA above is complete
  }
  const bool ok = mbar_wait(&done, 0);
  __syncwarp();
  tc::fence_after_sync();

  // TMEM -> shared tile T[token][row] (fp32); the stage buffers are free now
  float* T = reinterpret_cast<float*>(base);
  if (ok) {
    const uint32_t quad = (uint32_t)(warp * 32) << 16;
    const int row = warp * 32 + lane;
    for (int c0 = 0; c0 < p.BN; c0 += 16) {
      uint32_t r[16];
      tc::tmem_ld16(tmem + quad + (uint32_t)c0, r);
      tc::tmem_ld_wait();
#pragma unroll
      for (int i = 0; i < 16; ++i) T[(c0 + i) * kTcM + row] = __uint_as_float(r[i]);
    }
  } else if (threadIdx.x == 0) {
    report(p.status, WM_ERR_TIMEOUT);
  }
  tc::fence_before_sync();
  __syncthreads();
  if (warp == 0) {
    tc::fence_after_sync();
    tc::tmem_dealloc(tmem, p.tmem_cols);
  }
  if (!ok) return;

  // per (token, head) epilogue: keys QK-norm + RoPE, bf16 write to the cache slot
  const int hpt = kTcM / HD;
  const bool reporter = (mt == 0 && j == 0 && X == 0);
  __nv_bfloat16* pool = X == 0 ? p.k_pool : p.v_pool;
  const __nv_bfloat16* qg = p.qk_g + (int64_t)j * HD;
  for (int it = warp; it < p.B * hpt; it += kTcThreads / 32) {
    const int n = it / hpt, hl = it % hpt;
    const int hh = mt * hpt + hl;
    const int s = p.slot[n];
    if (s < 1 || s >= p.max_pages * p.P) {
      if (reporter && lane == 0) report(p.status, WM_ERR_BOUNDS);
      continue;
    }
    const int pg = p.page_table[(int64_t)n * p.max_pages + (s >> p.log2P)];
    if (pg < 0 || pg >= p.num_pages) {
      if (reporter && lane == 0) report(p.status, WM_ERR_BOUNDS);
      continue;
    }
    float y[EPL];
#pragma unroll
    for (int i = 0; i < EPL; ++i) y[i] = T[n * kTcM + hl * HD + lane + 32 * i];
    if (X == 0) {
      float ss = 0.f;
#pragma unroll
      for (int i = 0; i < EPL; ++i) ss = fmaf(y[i], y[i], ss);
      ss = warp_sum(ss);
      const float rr = rsqrtf(ss / (float)HD + p.eps_qk);
#pragma unroll
      for (int i = 0; i < EPL; ++i) y[i] = y[i] * rr * __bfloat162float(qg[lane + 32 * i]);
#pragma unroll
      for (int i = 0; i < EPL / 2; ++i) {
        const int e = lane + 32 * i;
        const float cs = p.rope_cs[((int64_t)n * (HD / 2) + e) * 2];
        const float sn = p.rope_cs[((int64_t)n * (HD / 2) + e) * 2 + 1];
        const float x0 = y[i], x1 = y[i + EPL / 2];
        y[i] = x0 * cs - x1 * sn;
        y[i + EPL / 2] = x1 * cs + x0 * sn;
      }
    }
    __nv_bfloat16* dst =
        pool + ((((int64_t)j * p.num_pages + pg) * p.Hkv + hh) * p.P + (s & (p.P - 1))) * HD;
#pragma unroll
    for (int i = 0; i < EPL; ++i) dst[lane + 32 * i] = __float2bfloat16_rn(y[i]);
  }
}

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (!fn) {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(ptr);
  }
  return fn;
}

// Row-major bf16 matrix [rows][cols] as a 2-D tensor map with a 64 x box_rows box.
bool encode_kmajor(CUtensorMap* tm, const void* ptr, uint64_t rows, uint64_t cols, uint32_t box_rows) {
  auto fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {cols * 2};
  cuuint32_t box[2] = {(cuuint32_t)kTcBK, box_rows};
  cuuint32_t estr[2] = {1, 1};
  return fn(tm, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(ptr), dims, strides, box,
            estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

uint32_t pow2_at_least(uint32_t x, uint32_t lo) {
  uint32_t r = lo;
  while (r < x) r <<= 1;
  return r;
}

}  // namespace

bool proj_tc_supported(const MixParams& mp) {
  return (mp.Hkv * mp.d) % kTcM == 0 && mp.B >= 1 && mp.B <= 256 && encode_fn() != nullptr;
}

cudaError_t launch_proj_tc(const MixParams& mp, cudaStream_t s) {
  ProjTcParams p{};
  p.k = mp.k;
  p.B = mp.B;
  p.Hkv = mp.Hkv;
  p.D = mp.D;
  p.M_item = mp.Hkv * mp.d;
  p.BN = (mp.B + 15) / 16 * 16;
  p.nk = (mp.D + kTcBK - 1) / kTcBK;
  p.P = mp.P;
  p.log2P = mp.log2P;
  p.num_pages = mp.num_pages;
  p.max_pages = mp.max_pages;
  p.tmem_cols = pow2_at_least((uint32_t)p.BN, 32);
  p.eps_qk = mp.eps_qk;
  p.page_table = mp.page_table;
  p.slot = mp.slot;
  p.k_pool = reinterpret_cast<__nv_bfloat16*>(mp.k_pool);
  p.v_pool = reinterpret_cast<__nv_bfloat16*>(mp.v_pool);
  p.qk_g = reinterpret_cast<const __nv_bfloat16*>(mp.qk_g);
  p.rope_cs = mp.rope_cs;
  p.status = mp.status;
  CUtensorMap tmW[2], tmX;
  for (int X = 0; X < 2; ++X)
    if (!encode_kmajor(&tmW[X], mp.Wkv[X], (uint64_t)mp.k * p.M_item, mp.D, kTcM))
      return cudaErrorInvalidValue;
  if (!encode_kmajor(&tmX, mp.xop, (uint64_t)2 * mp.k * mp.B, mp.D, (uint32_t)p.BN))
    return cudaErrorInvalidValue;
  const size_t smem = (size_t)kTcStages * (kTcM * 128 + p.BN * 128) + 1024;
  dim3 grid(p.M_item / kTcM, mp.k, 2);
  cudaError_t e;
  if (mp.d == 64) {
    e = cudaFuncSetAttribute(proj_tc_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    proj_tc_kernel<64><<<grid, kTcThreads, smem, s>>>(tmW[0], tmW[1], tmX, p);
  } else {
    e = cudaFuncSetAttribute(proj_tc_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    proj_tc_kernel<128><<<grid, kTcThreads, smem, s>>>(tmW[0], tmW[1], tmX, p);
  }
  return cudaGetLastError();
}

}  // namespace wm
