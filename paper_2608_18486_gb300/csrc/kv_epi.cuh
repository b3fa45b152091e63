#pragma once
// Epilogue of the per-channel K/V projection (Sec. 3.1 Step 2), shared by
// the tensor-core projection kernel and the fused decode pool: for every
// (token, kv head) of a 128-row output tile, keys get the per-head QK-norm
// (RMSNorm over d with the channel's gain) and rotate-half RoPE at the
// token's position; keys and values are rounded to bf16 and written to the
// token's cache slot (Sec. 3.2: the token at position i goes to slot i + 1).
#include "common.cuh"

namespace wm {

struct KvEpiArgs {
  int32_t Hkv, P, num_pages;
  float eps_qk;
  const __nv_bfloat16* qk_g;  // [k][d]
  __nv_bfloat16* k_pool;      // [k][num_pages][Hkv][P][d]
  __nv_bfloat16* v_pool;
  int32_t* status;
};

// T: shared [token][128] fp32 projection outputs of rows mt*HPT*HD.. of
// channel j, branch X (0 = K, 1 = V), for the nb tokens of the tile.
// row_scale (optional, per tile token): multiplies the projection output
// first (the 1/RMS of the channel state when the operand was not normed).
// s_slot / s_page: each tile token's cache slot and physical page (-1: bad,
// skipped and reported).  cs_tab: RoPE (cos, sin) pairs [row][HD/2], row =
// cs_row0 + tile token.  Executed by all NW warps of the block.
template <int HD, int NW>
__device__ __forceinline__ void kv_epilogue_tile(const float* T, int nb, int mt, int j, int X,
                                                 const float* row_scale, const int* s_slot,
                                                 const int* s_page, const float* cs_tab,
                                                 int cs_row0, bool reporter, const KvEpiArgs& a) {
  constexpr int kM = 128;
  constexpr int HPT = kM / HD;          // whole heads per 128-row tile
  constexpr int HALF = HD / 2;
  constexpr int NP = (HALF + 31) / 32;  // pairs per lane
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  __nv_bfloat16* pool = X == 0 ? a.k_pool : a.v_pool;
  float qg0[NP], qg1[NP];  // QK-norm gain of channel j, the same for every item
#pragma unroll
  for (int t = 0; t < NP; ++t) {
    const int i = lane + 32 * t;
    qg0[t] = i < HALF ? __bfloat162float(a.qk_g[(int64_t)j * HD + i]) : 0.f;
    qg1[t] = i < HALF ? __bfloat162float(a.qk_g[(int64_t)j * HD + i + HALF]) : 0.f;
  }
  // Each warp takes IPW items per round, their loads, reductions and stores
  // interleaved so that the latencies overlap.
  constexpr int IPW = 4;
  const int nitems = nb * HPT;
  for (int it0 = warp * IPW; it0 < nitems; it0 += NW * IPW) {
    float y0[IPW][NP], y1[IPW][NP];
    int n_[IPW], hh_[IPW], pg_[IPW];
    bool on[IPW];
#pragma unroll
    for (int q = 0; q < IPW; ++q) {
      const int it = it0 + q;
      const int n = it / HPT, hl = it % HPT;  // n: token within the tile
      n_[q] = n;
      hh_[q] = mt * HPT + hl;
      pg_[q] = it < nitems ? s_page[n] : -1;
      on[q] = it < nitems && hh_[q] < a.Hkv && pg_[q] >= 0;
      if (it < nitems && hh_[q] < a.Hkv && pg_[q] < 0 && reporter && hl == 0 && lane == 0)
        report(a.status, WM_ERR_BOUNDS);
      const float* src = T + n * kM + hl * HD;
      const float sc = (row_scale != nullptr && it < nitems) ? row_scale[n] : 1.f;
#pragma unroll
      for (int t = 0; t < NP; ++t) {
        const int i = lane + 32 * t;
        y0[q][t] = on[q] && i < HALF ? src[i] : 0.f;
        y1[q][t] = on[q] && i < HALF ? src[i + HALF] : 0.f;
        if (row_scale != nullptr) {
          y0[q][t] *= sc;
          y1[q][t] *= sc;
        }
      }
    }
    if (X == 0) {
      float ss[IPW];
#pragma unroll
      for (int q = 0; q < IPW; ++q) {
        ss[q] = 0.f;
#pragma unroll
        for (int t = 0; t < NP; ++t) ss[q] = fmaf(y0[q][t], y0[q][t], fmaf(y1[q][t], y1[q][t], ss[q]));
      }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1)
#pragma unroll
        for (int q = 0; q < IPW; ++q) ss[q] += __shfl_xor_sync(0xFFFFFFFFu, ss[q], o);
#pragma unroll
      for (int q = 0; q < IPW; ++q) {
        const float rr = rsqrtf(ss[q] / (float)HD + a.eps_qk);
        const int row = cs_row0 + n_[q];
#pragma unroll
        for (int t = 0; t < NP; ++t) {
          const int i = lane + 32 * t;
          if (on[q] && i < HALF) {
            const float x0 = y0[q][t] * rr * qg0[t], x1 = y1[q][t] * rr * qg1[t];
            const float2 csn = reinterpret_cast<const float2*>(cs_tab)[row * HALF + i];
            y0[q][t] = x0 * csn.x - x1 * csn.y;  // rotate-half RoPE
            y1[q][t] = x1 * csn.x + x0 * csn.y;
          }
        }
      }
    }
#pragma unroll
    for (int q = 0; q < IPW; ++q) {
      if (!on[q]) continue;
      const int s = s_slot[n_[q]];
      __nv_bfloat16* dst =
          pool + ((((int64_t)j * a.num_pages + pg_[q]) * a.Hkv + hh_[q]) * a.P + (s & (a.P - 1))) * HD;
#pragma unroll
      for (int t = 0; t < NP; ++t) {
        const int i = lane + 32 * t;
        if (i < HALF) {
          dst[i] = __float2bfloat16_rn(y0[q][t]);
          dst[i + HALF] = __float2bfloat16_rn(y1[q][t]);
        }
      }
    }
  }
}

}  // namespace wm
