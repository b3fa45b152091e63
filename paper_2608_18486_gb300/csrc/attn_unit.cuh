#pragma once
// Decode attention over one channel of the paged k-channel cache, unit split
// (Sec. 3.1 Step 3; dummy slot of Sec. 3.2), for launches with few
// (sequence b, kv head h) units: the paper's own model shape (16 sequences x
// 3 kv heads) has 48 of them for 152 SMs.
//
// Design.  Each unit gets one thread-block cluster of C CTAs (at most 8, all
// clusters resident at once), and each of its C x NW warps streams a contiguous,
// near-equal share of the unit's stages through a private 3-deep ring of bulk
// async copies, with the same stage math as the stream-K kernel
// (attn_kernel.cuh).  The partial softmax states then merge on chip: the
// warps of a CTA through shared memory, the CTAs of the cluster through
// distributed shared memory, each CTA producing 1/C of the unit's G x d
// outputs.  No record goes through global memory and no flag or ticket is
// waited on; the stream-K kernel's cross-SM merge (flags raised on other SMs,
// records landed from L2) sits on the critical path of such short launches.
// The split is static, so it suits launches whose units have similar lengths;
// the planner takes it for launches below 2 GB, or of one sequence, when all
// its clusters are resident at once with enough warps (csrc/wm_api.cu).
#include <cooperative_groups.h>

#include "attn_kernel.cuh"

namespace wm {
namespace attn_unit_detail {

namespace cg = cooperative_groups;
using attn_detail::Shape;
using attn_detail::SoftState;

constexpr int kUStages = 3;  // ring depth per warp

// Warps per CTA: 4 where a kv head has at most two query heads (two or
// three CTAs per SM, by the stage size: smaller CTAs keep more clusters
// resident and more SMs busy), else 8 (one CTA per SM: the states of four or
// eight query heads take up to 255 registers).
template <typename T, int HD, int G, int SB>
constexpr int unit_warps() {
  return G <= 2 ? 4 : 8;
}
// CTAs per SM the register budget is sized for (at most 12 warps of 170
// registers per SM)
constexpr int unit_min_blocks(int nw) { return nw <= 4 ? 3 : nw <= 6 ? 2 : 1; }

// A row of global memory another grid may just have written, as the stage
// math reads it (lane part lp owns 16-byte vectors lp, lp + LPS, ...), through
// L2 (ld.global.cg): no stale L1 line can be read.
template <typename T, int HD, int SB>
__device__ __forceinline__ void load_row_l2(const T* row, int lp,
                                            float2 (&f)[Shape<T, HD, SB>::EPL / 2]) {
  using SH = Shape<T, HD, SB>;
#pragma unroll
  for (int v = 0; v < SH::NVL; ++v) {
    float t[SH::VEC];
    Elem<T>::unpack(__ldcg(reinterpret_cast<const uint4*>(row + (v * SH::LPS + lp) * SH::VEC)), t);
#pragma unroll
    for (int i = 0; i < SH::VEC / 2; ++i) f[v * SH::VEC / 2 + i] = make_float2(t[2 * i], t[2 * i + 1]);
  }
}

// floats of one partial state: G x HD unnormalised outputs, then (max, sum)
// per query head (log2 units)
constexpr int unit_rec(int G, int HD) { return G * HD + 2 * G; }

template <typename T, int HD, int G, int SB>
__global__ void __launch_bounds__(unit_warps<T, HD, G, SB>() * 32,
                                  unit_min_blocks(unit_warps<T, HD, G, SB>()))
    decode_attn_unit_kernel(const AttnParams p) {
  using SH = Shape<T, HD, SB>;
  constexpr int NW = unit_warps<T, HD, G, SB>();
  constexpr int VEC = SH::VEC, LPS = SH::LPS, E2 = SH::EPL / 2;
  constexpr int STAGE_SLOTS = SH::STAGE_SLOTS, STAGE_ELEMS = SH::STAGE_ELEMS;
  constexpr uint32_t KV_BYTES = STAGE_ELEMS * sizeof(T);
  constexpr int E = G * HD;  // output elements of a unit
  constexpr int REC = unit_rec(G, HD);
  constexpr unsigned FULLMASK = 0xFFFFFFFFu;
  // a warp's state goes into its own ring once the ring is idle
  static_assert((size_t)REC * sizeof(float) <= (size_t)kUStages * 2 * KV_BYTES, "record fits the ring");

  extern __shared__ __align__(128) unsigned char smem_raw[];
  T* ring = reinterpret_cast<T*>(smem_raw);  // [NW][S][2][STAGE_ELEMS]
  float* crec = reinterpret_cast<float*>(ring + NW * kUStages * 2 * STAGE_ELEMS);  // [REC]
  __shared__ uint64_t bars[NW][kUStages];
  __shared__ uint64_t masks[NW][kUStages];

  cg::cluster_group cluster = cg::this_cluster();
  const int C = (int)cluster.num_blocks();
  const int rank = (int)cluster.block_rank();
  const int unit = (int)(blockIdx.x / (unsigned)C);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int b = unit / p.Hkv, h = unit - b * p.Hkv;
  const int max_slots = p.max_pages * p.P;

  // Programmatic dependent launch, as in the stream-K kernel: with the
  // caller's inputs_ready promise the cache, table and lengths are read
  // before the dependency wait, and only the query after it.
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  const bool early = p.inputs_ready != 0;
  if (!early) asm volatile("griddepcontrol.wait;" ::: "memory");

  if (tid == 0) {
    for (int w = 0; w < NW; ++w)
      for (int s = 0; s < kUStages; ++s) mbar_init(&bars[w][s], 1);
  }
  fence_mbar_init();
  __syncthreads();

  const int S_in = __ldg(p.seq_lens + b);
  const bool len_ok = S_in >= 1 && S_in <= max_slots;
  const int S = len_ok ? S_in : 0;  // an invalid length reads nothing: zero rows
  if (!len_ok && h == 0 && rank == 0 && tid == 0) report(p.status, WM_ERR_BOUNDS);
  const int nst = (S + STAGE_SLOTS - 1) / STAGE_SLOTS;
  const int npieces = C * NW, piece = rank * NW + warp;
  const int s0 = (int)((int64_t)piece * nst / npieces);
  const int nmine = (int)((int64_t)(piece + 1) * nst / npieces) - s0;

  T* myring = ring + warp * kUStages * 2 * STAGE_ELEMS;
  const uint64_t policy = l2_evict_first_policy();
  const T* kbase = reinterpret_cast<const T*>(p.k_pool) + (int64_t)h * p.P * HD;
  const T* vbase = reinterpret_cast<const T*>(p.v_pool) + (int64_t)h * p.P * HD;

  // Page-table window: lane i holds the page id of logical page win0 + i
  // (cur) and win0 + 32 + i (nxt); all lanes call page_of together.
  const int32_t* ptab = p.page_table + (int64_t)b * p.max_pages;
  int win0 = -64, pg_cur = -1, pg_nxt = -1;
  auto load_pg = [&](int lp) -> int { return lp < p.max_pages ? __ldg(ptab + lp) : -1; };
  auto page_of = [&](int lp, int lane_off) -> int {
    if (lp < win0 || lp >= win0 + 64) {
      win0 = lp;
      pg_cur = load_pg(lp + lane);
      pg_nxt = load_pg(lp + 32 + lane);
    } else if (lp >= win0 + 32) {
      win0 += 32;
      pg_cur = pg_nxt;
      pg_nxt = load_pg(win0 + 32 + lane);
    }
    const int idx = lp + lane_off - win0;  // 0 .. 63
    const int a = __shfl_sync(FULLMASK, pg_cur, idx & 31);
    const int c = __shfl_sync(FULLMASK, pg_nxt, idx & 31);
    return idx < 32 ? a : c;
  };

  // Copy stage s of the unit (the i-th of this warp) into ring slot i % S.
  auto issue = [&](int s) {
    const int buf = (s - s0) % kUStages;
    T* kd = myring + buf * 2 * STAGE_ELEMS;
    T* vd = kd + STAGE_ELEMS;
    uint64_t* bar = &bars[warp][buf];
    const int s_begin = s * STAGE_SLOTS;
    if (p.P >= STAGE_SLOTS) {
      const int pg = page_of(s_begin >> p.log2P, 0);
      if (lane == 0) {
        const bool ok = pg >= 0 && pg < p.num_pages;
        masks[warp][buf] = ok ? 1ull : 0ull;
        if (!ok) report(p.status, WM_ERR_BOUNDS);
        mbar_arrive_expect_tx(bar, ok ? 2 * KV_BYTES : 0u);
        if (ok) {
          const int64_t off = (int64_t)pg * p.page_stride + (int64_t)(s_begin & (p.P - 1)) * HD;
          bulk_g2s(kd, kbase + off, KV_BYTES, bar, policy);
          bulk_g2s(vd, vbase + off, KV_BYTES, bar, policy);
        }
      }
    } else {
      const int npp = STAGE_SLOTS >> p.log2P;  // pages per stage (<= 32)
      const int lp0 = s_begin >> p.log2P;
      const int lpn = min(npp, ((S - 1) >> p.log2P) - lp0 + 1);
      const int pg = page_of(lp0, lane < lpn ? lane : 0);
      const bool ok = lane < lpn && pg >= 0 && pg < p.num_pages;
      const uint32_t mask = __ballot_sync(FULLMASK, ok);
      const uint32_t bytes = (uint32_t)p.P * HD * sizeof(T);
      if (lane == 0) {
        masks[warp][buf] = mask;
        if (__popc(mask) < lpn) report(p.status, WM_ERR_BOUNDS);
        mbar_arrive_expect_tx(bar, 2u * bytes * (uint32_t)__popc(mask));
      }
      __syncwarp();
      if (ok) {
        const int64_t off = (int64_t)pg * p.page_stride;
        bulk_g2s(kd + lane * p.P * HD, kbase + off, bytes, bar, policy);
        bulk_g2s(vd + lane * p.P * HD, vbase + off, bytes, bar, policy);
      }
    }
  };

  int issued = 0;
  for (; issued < nmine && issued < kUStages; ++issued) issue(s0 + issued);
  if (early) asm volatile("griddepcontrol.wait;" ::: "memory");

  // ---- stream this warp's stages
  const int lane_slot = lane / LPS, lane_part = lane % LPS;
  const int log2P_in_stage = p.P >= STAGE_SLOTS ? 30 : p.log2P;  // stage page index = slot >> this
  const uint64_t all_pages = p.P >= STAGE_SLOTS ? 1ull : ((1ull << (STAGE_SLOTS >> p.log2P)) - 1ull);
  SoftState<T, HD, G, SB> st;
  float2 q2[G][E2];
#pragma unroll
  for (int g = 0; g < G; ++g) {
    st.m[g] = -INFINITY;
    st.l[g] = 0.f;
#pragma unroll
    for (int i = 0; i < E2; ++i) st.acc[g][i] = make_float2(0.f, 0.f);
  }
  // the unit's G query rows, read through L2 after the dependency wait (the
  // previous grid may have written them)
  if (nmine > 0) {
    const T* qrow = reinterpret_cast<const T*>(p.q) + ((int64_t)b * p.Hq + h * G) * HD;
#pragma unroll
    for (int g = 0; g < G; ++g) load_row_l2<T, HD, SB>(qrow + g * HD, lane_part, q2[g]);
  }
  bool alive = true;
  int done = 0;  // stages consumed
  for (; done < nmine && alive; ++done) {
    const int buf = done % kUStages;
    if (!__all_sync(FULLMASK, mbar_wait(&bars[warp][buf], (done / kUStages) & 1))) {
      if (lane == 0) report(p.status, WM_ERR_TIMEOUT);
      alive = false;
      break;
    }
    const int s = s0 + done;
    const int valid_slots = S - s * STAGE_SLOTS;
    const uint64_t mask = masks[warp][buf];
    const T* Ks = myring + buf * 2 * STAGE_ELEMS;
    const T* Vs = Ks + STAGE_ELEMS;
    if (valid_slots >= STAGE_SLOTS && mask == all_pages)
      attn_detail::consume_stage<T, HD, G, SB, true>(Ks, Vs, lane_slot, lane_part, q2, p.qscale,
                                                     valid_slots, mask, log2P_in_stage, st);
    else
      attn_detail::consume_stage<T, HD, G, SB, false>(Ks, Vs, lane_slot, lane_part, q2, p.qscale,
                                                      valid_slots, mask, log2P_in_stage, st);
    __syncwarp();  // every lane is done with this ring slot
    if (issued < nmine) issue(s0 + issued++);
  }
  if (!alive) {
    // a copy never landed: wait (bounded) for what is still in flight and
    // contribute nothing
    if (lane == 0)
      for (int y = done; y < issued; ++y) mbar_wait(&bars[warp][y % kUStages], (y / kUStages) & 1);
    __syncwarp();
#pragma unroll
    for (int g = 0; g < G; ++g) {
      st.m[g] = -INFINITY;
      st.l[g] = 0.f;
#pragma unroll
      for (int i = 0; i < E2; ++i) st.acc[g][i] = make_float2(0.f, 0.f);
    }
  }

  // ---- merge the SPW lane groups of the warp, then store the warp's state
  // in its (idle) ring
  float* wrec = reinterpret_cast<float*>(myring);
#pragma unroll
  for (int g = 0; g < G; ++g) {
    float M = st.m[g];
#pragma unroll
    for (int o = LPS; o < 32; o <<= 1) M = fmaxf(M, __shfl_xor_sync(FULLMASK, M, o));
    const float w = (st.m[g] == -INFINITY) ? 0.f : exp2f(st.m[g] - M);
    float Ls = st.l[g] * w;
#pragma unroll
    for (int o = LPS; o < 32; o <<= 1) Ls += __shfl_xor_sync(FULLMASK, Ls, o);
#pragma unroll
    for (int i = 0; i < E2; ++i) {
      float2 a = __fmul2_rn(st.acc[g][i], make_float2(w, w));
#pragma unroll
      for (int o = LPS; o < 32; o <<= 1) {
        a.x += __shfl_xor_sync(FULLMASK, a.x, o);
        a.y += __shfl_xor_sync(FULLMASK, a.y, o);
      }
      st.acc[g][i] = a;
    }
    if (lane_slot == 0) {
#pragma unroll
      for (int v = 0; v < SH::NVL; ++v)
#pragma unroll
        for (int i = 0; i < VEC / 2; ++i)
          reinterpret_cast<float2*>(wrec + g * HD + (v * LPS + lane_part) * VEC)[i] =
              st.acc[g][v * VEC / 2 + i];
    }
    if (lane == 0) {
      wrec[E + 2 * g] = M;
      wrec[E + 2 * g + 1] = Ls;
    }
  }
  __syncthreads();

  // ---- merge the CTA's NW warp states, element by element
  T* outp = reinterpret_cast<T*>(p.out) + ((int64_t)b * p.Hq + h * G) * HD;
  auto warp_rec = [&](int w) -> const float* {
    return reinterpret_cast<const float*>(ring + w * kUStages * 2 * STAGE_ELEMS);
  };
  for (int e = tid; e < E; e += NW * 32) {
    const int g = e / HD;
    float mw[NW];
    float M = -INFINITY;
#pragma unroll
    for (int w = 0; w < NW; ++w) {
      mw[w] = warp_rec(w)[E + 2 * g];
      M = fmaxf(M, mw[w]);
    }
    float Ls = 0.f, O = 0.f;
#pragma unroll
    for (int w = 0; w < NW; ++w) {
      const float wt = mw[w] == -INFINITY ? 0.f : exp2f(mw[w] - M);
      Ls = fmaf(wt, warp_rec(w)[E + 2 * g + 1], Ls);
      O = fmaf(wt, warp_rec(w)[e], O);
    }
    if (C == 1) {
      outp[e] = Elem<T>::from_f(O * (Ls > 0.f ? 1.f / Ls : 0.f));
    } else {
      crec[e] = O;
      if (e == g * HD) {
        crec[E + 2 * g] = M;
        crec[E + 2 * g + 1] = Ls;
      }
    }
  }
  if (C == 1) return;

  // ---- merge the cluster's C CTA states: CTA `rank` finishes 1/C of the
  // unit's outputs, reading every CTA's state through distributed shared
  // memory; the second barrier keeps each CTA's shared memory alive until
  // every reader is done
  cluster.sync();
  const float* cr[kAttnUnitMaxCluster];
#pragma unroll
  for (int c = 0; c < kAttnUnitMaxCluster; ++c) cr[c] = c < C ? cluster.map_shared_rank(crec, c) : crec;
  const int e0 = rank * E / C, e1 = (rank + 1) * E / C;
  for (int e = e0 + tid; e < e1; e += NW * 32) {
    const int g = e / HD;
    float mq[kAttnUnitMaxCluster], lq[kAttnUnitMaxCluster], oq[kAttnUnitMaxCluster];
#pragma unroll
    for (int c = 0; c < kAttnUnitMaxCluster; ++c) {
      mq[c] = c < C ? cr[c][E + 2 * g] : -INFINITY;
      lq[c] = c < C ? cr[c][E + 2 * g + 1] : 0.f;
      oq[c] = c < C ? cr[c][e] : 0.f;
    }
    float M = -INFINITY;
#pragma unroll
    for (int c = 0; c < kAttnUnitMaxCluster; ++c) M = fmaxf(M, mq[c]);
    float Ls = 0.f, O = 0.f;
#pragma unroll
    for (int c = 0; c < kAttnUnitMaxCluster; ++c) {
      const float wt = mq[c] == -INFINITY ? 0.f : exp2f(mq[c] - M);
      Ls = fmaf(wt, lq[c], Ls);
      O = fmaf(wt, oq[c], O);
    }
    outp[e] = Elem<T>::from_f(O * (Ls > 0.f ? 1.f / Ls : 0.f));
  }
  cluster.sync();
}

template <typename T, int HD, int G, int SB>
inline cudaError_t launch_unit_t(const AttnParams& p, int units, int cluster, size_t smem,
                                 cudaStream_t stream) {
  static size_t smem_set[kSmemOptDevices] = {};
  auto kern = decode_attn_unit_kernel<T, HD, G, SB>;
  if (cudaError_t e = opt_in_smem(kern, smem, smem_set); e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)units * (unsigned)cluster);
  cfg.blockDim = dim3(unit_warps<T, HD, G, SB>() * 32);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeClusterDimension;
  attr[1].val.clusterDim.x = (unsigned)cluster;
  attr[1].val.clusterDim.y = 1;
  attr[1].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, kern, p);
}

// Clusters of `cluster` CTAs that can be resident at once (0: unknown).
template <typename T, int HD, int G, int SB>
inline int max_clusters_t(int cluster, size_t smem) {
  auto kern = decode_attn_unit_kernel<T, HD, G, SB>;
  if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) != cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)cluster * 64u);
  cfg.blockDim = dim3(unit_warps<T, HD, G, SB>() * 32);
  cfg.dynamicSmemBytes = smem;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = (unsigned)cluster;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, kern, &cfg) != cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  return n;
}

template <typename T, int HD, int SB>
inline int unit_warps_g(int G) {
  switch (G) {
    case 1: return unit_warps<T, HD, 1, SB>();
    case 2: return unit_warps<T, HD, 2, SB>();
    case 4: return unit_warps<T, HD, 4, SB>();
    case 8: return unit_warps<T, HD, 8, SB>();
    default: return 0;
  }
}

template <typename T, int HD, int SB>
inline int max_clusters_g(int G, int cluster, size_t smem) {
  switch (G) {
    case 1: return max_clusters_t<T, HD, 1, SB>(cluster, smem);
    case 2: return max_clusters_t<T, HD, 2, SB>(cluster, smem);
    case 4: return max_clusters_t<T, HD, 4, SB>(cluster, smem);
    case 8: return max_clusters_t<T, HD, 8, SB>(cluster, smem);
    default: return 0;
  }
}

template <typename T, int HD, int SB>
inline cudaError_t launch_unit_g(const AttnParams& p, int G, int units, int cluster, size_t smem,
                                 cudaStream_t s) {
  switch (G) {
    case 1: return launch_unit_t<T, HD, 1, SB>(p, units, cluster, smem, s);
    case 2: return launch_unit_t<T, HD, 2, SB>(p, units, cluster, smem, s);
    case 4: return launch_unit_t<T, HD, 4, SB>(p, units, cluster, smem, s);
    case 8: return launch_unit_t<T, HD, 8, SB>(p, units, cluster, smem, s);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace attn_unit_detail

// Per-dtype dispatch of the unit split (one translation unit each); the
// max_clusters entry points return 0 for an unsupported shape or no device.
cudaError_t launch_attn_unit_bf16(const AttnParams& p, int stage_bytes, int d, int G, int units,
                                  int cluster, size_t smem, cudaStream_t s);
cudaError_t launch_attn_unit_f32(const AttnParams& p, int stage_bytes, int d, int G, int units,
                                 int cluster, size_t smem, cudaStream_t s);
int attn_unit_max_clusters_bf16(int stage_bytes, int d, int G, int cluster, size_t smem);
int attn_unit_max_clusters_f32(int stage_bytes, int d, int G, int cluster, size_t smem);

}  // namespace wm
