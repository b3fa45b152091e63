// The two dense contractions of the cross-layer KV pool on the tcgen05
// tensor cores (bf16 operands, fp32 accumulation in TMEM):
//  * the per-channel K/V projection with a fused epilogue (Sec. 3.1 Step 2):
//    K_j = W^K_j x^K_j, V_j = W^V_j x^V_j for the B tokens of a decode step,
//    then per-head QK-norm and RoPE on keys, bf16 rounding and the write to
//    each token's cache slot;
//  * the router logits W^alpha xi (Sec. 3.1 Step 1), split over the long L'D
//    reduction, each split storing fp32 partial sums.
//
// Shape: at decode the token count B is small (16..64) while the weights
// are large (Hkv*d x D per channel and branch), so the weights take the MMA's
// M side ("swap AB"): one CTA computes a 128-row tile of W^X_j against all
// B tokens, D[row][token] in TMEM (128 lanes x N fp32 columns).  A projection
// tile covers whole heads (two of d=64, one of d=96 or 128; rows past the
// last head are computed and ignored).  The work is
// weight-streaming bound; TMA brings 128x64 weight tiles and Nx64 token
// tiles (128-byte swizzle) through a 4-stage mbarrier pipeline.  Warp 0 lane
// 0 issues TMA, warp 1 lane 0 issues tcgen05.mma, warps 2-7 fetch what the
// epilogue needs; all eight warps drain TMEM (warps w and w + 4 share the
// 32-lane quadrant w % 4) into shared memory, then finish the per-(token,
// head) epilogue, several items per warp at a time.
#include <cudaTypedefs.h>
#include <math.h>

#include "internal.h"
#include "kv_epi.cuh"
#include "tc.cuh"

namespace wm {

namespace {

constexpr int kTcM = 128;      // weight rows per tile (MMA M)
constexpr int kTcBK = 64;      // K elements per stage (128 bytes of bf16)
constexpr int kTcMaxStages = 12;
constexpr int kTcThreads = 256;
constexpr int kTcMaxTokens = 256;

enum { kEpiKV = 0, kEpiPartial = 1 };

struct ProjTcParams {
  int32_t k, B, Hkv, D, M_item, BN, nk, stages;
  int32_t kb_per_split, M_total;  // router: k-blocks per split, rows of W
  int32_t rope_smem_off;          // projection: byte offset of the RoPE table in smem, 0 = global
  float* zpart;                   // router: [2][nsplit][B][M_total]
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

// MODE kEpiKV: grid (ceil(Hkv/hpt), k, 2*ntiles) = (head tile, channel j, branch X + 2*token
// tile), hpt = 128/HD.
// MODE kEpiPartial: grid (ceil(kL/128), nsplit, 2*ntiles) = (row tile, split, branch X + 2*token
// tile).  A token tile is BN <= 256 tokens.
template <int HD, int MODE>
__global__ void __launch_bounds__(kTcThreads, 1)
    proj_tc_kernel(const __grid_constant__ CUtensorMap tmW0, const __grid_constant__ CUtensorMap tmW1,
                   const __grid_constant__ CUtensorMap tmX, const ProjTcParams p) {
  extern __shared__ uint8_t smem_dyn[];
  __shared__ uint64_t full[kTcMaxStages], empty[kTcMaxStages], done;
  __shared__ uint32_t tmem_base;
  __shared__ int s_slot[kTcMaxTokens], s_page[kTcMaxTokens];

  const int mt = blockIdx.x, j = blockIdx.y, X = blockIdx.z & 1;
  const int n0 = (blockIdx.z >> 1) * p.BN;      // first token of this tile
  const int nb = min(p.BN, p.B - n0);           // tokens in this tile
  const int NS = p.stages;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const CUtensorMap* tmW = X == 0 ? &tmW0 : &tmW1;
  uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_dyn) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  const uint32_t a_bytes = kTcM * 128;
  const uint32_t b_bytes = (uint32_t)p.BN * 128;
  uint8_t* As = base;
  uint8_t* Bs = base + NS * a_bytes;

  constexpr int HPT = kTcM / HD;  // whole heads per 128-row tile
  const int wrow = MODE == kEpiKV ? j * p.M_item + mt * HPT * HD : mt * kTcM;
  const int xrow = (MODE == kEpiKV ? (X * p.k + j) * p.B : X * p.B) + n0;
  const int kb0 = MODE == kEpiKV ? 0 : j * p.kb_per_split;
  const int kb1 = MODE == kEpiKV ? p.nk : min(p.nk, kb0 + p.kb_per_split);
  const int nkb = kb1 - kb0;
  if (threadIdx.x == 0) {
    for (int s = 0; s < NS; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    mbar_init(&done, 1);
    fence_mbar_init();
    tc::prefetch_tensormap(tmW);
    tc::prefetch_tensormap(&tmX);
    // The weights are inputs no earlier kernel writes: the first ring's worth
    // streams in while the previous grid finishes.  Each stage's barrier
    // expects these bytes now and completes only after the arrival that
    // comes with the activation tile, after the dependency wait.
    for (int kb = 0; kb < NS && kb < nkb; ++kb) {
      mbar_expect_tx(&full[kb], a_bytes);
      tc::tma_load_2d(As + kb * a_bytes, tmW, (kb0 + kb) * kTcBK, wrow, &full[kb]);
    }
  }
  // programmatic dependent launch: the activations come from the previous grid
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  asm volatile("griddepcontrol.wait;" ::: "memory");
  float* rope_s = reinterpret_cast<float*>(base + p.rope_smem_off);  // [B][HD/2][2] or unused
  if (warp == 0) {
    tc::tmem_alloc(&tmem_base, p.tmem_cols);
    tc::tmem_relinquish();
  }
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = tmem_base;

  if (warp == 0 && lane == 0) {
    // TMA producer: activation tiles for the prefetched stages, then whole
    // stages as the ring frees up
    for (int kb = 0; kb < nkb; ++kb) {
      const int s = kb % NS;
      if (kb < NS) {
        mbar_arrive_expect_tx(&full[s], b_bytes);
        tc::tma_load_2d(Bs + s * b_bytes, &tmX, (kb0 + kb) * kTcBK, xrow, &full[s]);
        continue;
      }
      if (!mbar_wait(&empty[s], ((kb / NS) - 1) & 1)) {
        report(p.status, WM_ERR_TIMEOUT);
        break;
      }
      mbar_arrive_expect_tx(&full[s], a_bytes + b_bytes);
      tc::tma_load_2d(As + s * a_bytes, tmW, (kb0 + kb) * kTcBK, wrow, &full[s]);
      tc::tma_load_2d(Bs + s * b_bytes, &tmX, (kb0 + kb) * kTcBK, xrow, &full[s]);
    }
  } else if (MODE == kEpiKV && warp >= 2) {
    // meanwhile warps 2-3 fetch what the epilogue needs: the RoPE table of the
    // tile's tokens and each token's destination slot and page
    const int t2 = threadIdx.x - 64, n2 = kTcThreads - 64;
    if (p.rope_smem_off > 0)
      for (int i = t2; i < nb * HD; i += n2) rope_s[i] = p.rope_cs[(int64_t)n0 * HD + i];
    for (int n = t2; n < nb; n += n2) {
      const int s = p.slot[n0 + n];
      int pg = -1;
      if (s >= 1 && s < p.max_pages * p.P)
        pg = p.page_table[(int64_t)(n0 + n) * p.max_pages + (s >> p.log2P)];
      s_slot[n] = s;
      s_page[n] = (pg >= 0 && pg < p.num_pages) ? pg : -1;
    }
  } else if (warp == 1 && lane == 0) {
    // MMA issuer: 4 MMAs of K = 16 per stage
    const uint32_t idesc = tc::idesc_bf16_f32(kTcM, p.BN);
    for (int kb = 0; kb < nkb; ++kb) {
      const int s = kb % NS;
      if (!mbar_wait(&full[s], (kb / NS) & 1)) {
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
  // warp-uniform: the TMEM loads below are warp-collective
  const bool ok = __all_sync(0xFFFFFFFFu, mbar_wait(&done, 0));
  tc::fence_after_sync();

  // TMEM -> shared tile T[token][row] (fp32); the stage buffers are free now.
  // Warps w and w + 4 share lane quadrant w % 4 and split its columns.
  float* T = reinterpret_cast<float*>(base);
  if (ok) {
    const uint32_t quad = (uint32_t)((warp & 3) * 32) << 16;
    const int row = (warp & 3) * 32 + lane;
    for (int c0 = (warp >> 2) * 16; c0 < p.BN; c0 += 32) {
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

  if (MODE == kEpiPartial) {
    // fp32 partial logits of this split: zpart[X][split][n][row]
    float* z = p.zpart + (((int64_t)X * gridDim.y + j) * p.B + n0) * p.M_total;
    const int m0 = mt * kTcM;
    for (int i = threadIdx.x; i < nb * kTcM; i += kTcThreads) {
      const int n = i / kTcM, r = i % kTcM;
      if (m0 + r < p.M_total) z[(int64_t)n * p.M_total + m0 + r] = T[n * kTcM + r];
    }
    return;
  }
  // per (token, head) epilogue: keys QK-norm + RoPE, bf16 write to the cache slot
  KvEpiArgs ea;
  ea.Hkv = p.Hkv;
  ea.P = p.P;
  ea.num_pages = p.num_pages;
  ea.eps_qk = p.eps_qk;
  ea.qk_g = p.qk_g;
  ea.k_pool = p.k_pool;
  ea.v_pool = p.v_pool;
  ea.status = p.status;
  const bool local_tab = p.rope_smem_off > 0;
  kv_epilogue_tile<HD, kTcThreads / 32>(T, nb, mt, j, X, nullptr, s_slot, s_page,
                                        local_tab ? rope_s : p.rope_cs, local_tab ? 0 : n0,
                                        mt == 0 && j == 0 && X == 0, ea);
}

// Row-major bf16 matrix [rows][cols] as a 2-D tensor map with a 64 x box_rows box.
bool encode_kmajor(CUtensorMap* tm, const void* ptr, uint64_t rows, uint64_t cols, uint32_t box_rows) {
  return tma_map_bf16_2d(tm, ptr, rows, cols, cols, box_rows);
}

uint32_t pow2_at_least(uint32_t x, uint32_t lo) {
  uint32_t r = lo;
  while (r < x) r <<= 1;
  return r;
}

int sm_count_cur() {
  int dev = 0, n = 0;
  if (cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0)
    n = 148;
  return n;
}

// Pipeline depth: deep enough to keep one round trip of weights in flight;
// shallow enough for two CTAs per SM when the grid has more than one wave.
int pick_stages(int nkb, int BN, int64_t grid, int sms) {
  const int stage_bytes = kTcM * 128 + BN * 128;
  const int budget = grid > sms ? 100 * 1024 : 200 * 1024;
  int ns = budget / stage_bytes;
  ns = ns < 2 ? 2 : (ns > kTcMaxStages ? kTcMaxStages : ns);
  return ns > nkb ? (nkb < 2 ? 2 : nkb) : ns;
}

size_t tc_smem(int stages, int BN) {
  const size_t pipe = (size_t)stages * (kTcM * 128 + BN * 128);
  const size_t tile = (size_t)BN * kTcM * sizeof(float);  // epilogue reuses the stages
  return (pipe > tile ? pipe : tile) + 1024;
}

template <int HD, int MODE>
cudaError_t launch_mode(dim3 grid, size_t smem, const CUtensorMap& w0, const CUtensorMap& w1,
                        const CUtensorMap& x, const ProjTcParams& p, cudaStream_t s) {
  static size_t smem_set[kSmemOptDevices] = {};
  auto kern = proj_tc_kernel<HD, MODE>;
  if (cudaError_t e = opt_in_smem(kern, smem, smem_set); e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = dim3(kTcThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, w0, w1, x, p);
}

}  // namespace

int token_tile(int B) {  // tokens per MMA N tile: a multiple of 16, at most 256
  const int t = B < kTcMaxTokens ? B : kTcMaxTokens;
  return (t + 15) / 16 * 16;
}

bool proj_tc_supported(const MixParams& mp) {
  return (mp.d == 64 || mp.d == 96 || mp.d == 128) && mp.B >= 1 && tma_available();
}

bool router_tc_supported(int B) { return B >= 1; }

int router_tc_splits(int k, int L, int Lp, int D, int B, int sms) {
  const int nk = (Lp * D + kTcBK - 1) / kTcBK;
  const int ntiles = (B + token_tile(B) - 1) / token_tile(B);
  const int tiles = 2 * ((k * L + kTcM - 1) / kTcM) * ntiles;
  int ns = (sms + tiles - 1) / tiles;
  const int max_ns = nk / 8 > 1 ? nk / 8 : 1;  // at least 8 k-blocks per split
  ns = ns < 1 ? 1 : (ns > max_ns ? max_ns : ns);
  const int per = (nk + ns - 1) / ns;
  (void)B;
  return (nk + per - 1) / per;
}

cudaError_t launch_proj_tc(const MixParams& mp, cudaStream_t s) {
  ProjTcParams p{};
  p.k = mp.k;
  p.B = mp.B;
  p.Hkv = mp.Hkv;
  p.D = mp.D;
  p.M_item = mp.Hkv * mp.d;
  p.BN = token_tile(mp.B);
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
  const int hpt = kTcM / mp.d;
  const int ntiles = (mp.B + p.BN - 1) / p.BN;
  dim3 grid((mp.Hkv + hpt - 1) / hpt, mp.k, 2 * ntiles);
  p.stages = pick_stages(p.nk, p.BN, (int64_t)grid.x * grid.y * grid.z, sm_count_cur());
  size_t smem = tc_smem(p.stages, p.BN);
  const size_t rope_bytes = (size_t)p.BN * mp.d * sizeof(float);
  if (smem + rope_bytes <= 200 * 1024) {
    p.rope_smem_off = (int32_t)(smem - 1024);  // offset from the 1 KB-aligned base
    smem += rope_bytes;
  }
  if (mp.d == 64) return launch_mode<64, kEpiKV>(grid, smem, tmW[0], tmW[1], tmX, p, s);
  if (mp.d == 96) return launch_mode<96, kEpiKV>(grid, smem, tmW[0], tmW[1], tmX, p, s);
  return launch_mode<128, kEpiKV>(grid, smem, tmW[0], tmW[1], tmX, p, s);
}

cudaError_t launch_router_tc(const MixParams& mp, cudaStream_t s) {
  ProjTcParams p{};
  const int kL = mp.k * mp.L;
  const int K = mp.Lp * mp.D;
  p.k = mp.k;
  p.B = mp.B;
  p.D = K;
  p.BN = token_tile(mp.B);
  p.nk = (K + kTcBK - 1) / kTcBK;
  p.kb_per_split = (p.nk + mp.nsplit_r - 1) / mp.nsplit_r;
  p.M_total = kL;
  p.zpart = mp.zpart;
  p.tmem_cols = pow2_at_least((uint32_t)p.BN, 32);
  p.status = mp.status;
  CUtensorMap tmW[2], tmX;
  for (int X = 0; X < 2; ++X)
    if (!encode_kmajor(&tmW[X], mp.Wr[X], (uint64_t)kL, K, kTcM)) return cudaErrorInvalidValue;
  if (!encode_kmajor(&tmX, mp.xi, (uint64_t)2 * mp.B, K, (uint32_t)p.BN))
    return cudaErrorInvalidValue;
  dim3 grid((kL + kTcM - 1) / kTcM, mp.nsplit_r, 2 * ((mp.B + p.BN - 1) / p.BN));
  p.stages = pick_stages(p.kb_per_split, p.BN, (int64_t)grid.x * grid.y * grid.z, sm_count_cur());
  const size_t smem = tc_smem(p.stages, p.BN);
  return launch_mode<64, kEpiPartial>(grid, smem, tmW[0], tmW[1], tmX, p, s);
}

}  // namespace wm
