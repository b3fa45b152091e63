// Decode attention over one channel of the paged k-channel cache
// (Sec. 3.1 Step 3; dummy slot of Sec. 3.2).
//
// Design (GB300).  The work is a stream over the KV blocks of every
// (sequence b, kv head h) unit of the chosen channel; it reads about one byte
// per FLOP, so it is HBM-bound and runs on the CUDA cores.
//
//  * Stream-K split.  Each unit is cut into pipeline stages of STAGE_SLOTS
//    slots (8 KB of K+V).  The stages of all units, concatenated, are divided
//    into equal contiguous ranges, one per warp of a persistent grid, so every
//    warp streams the same number of bytes whatever the sequence lengths.
//  * Private pipelines.  Each warp owns a 3-deep ring in shared memory and
//    fills it with 1-D bulk async copies (TMA engine, mbarrier completion,
//    L2 evict-first) of contiguous (page, kv-head) runs; it refills a slot as
//    soon as it has consumed it, so no block-wide barrier is ever taken.
//  * Compute.  d/VEC lanes own one slot (a 16-byte vector each), reduce q.k
//    with xor shuffles and keep an online softmax (running max m, sum l,
//    accumulator) per lane group; groups merge with shuffles at the end of a
//    piece.
//  * Merge.  A piece of a unit that lies inside one warp's range is written
//    straight to the output.  Only units that cross a warp boundary leave
//    partials (at most two per warp: its first and its last piece); the last
//    warp to finish such a unit (atomic ticket, no waiting) merges them.
#include <math.h>

#include "common.cuh"
#include "internal.h"

namespace wm {

namespace {

constexpr int kWarps = 4;
constexpr int kThreads = kWarps * 32;
constexpr int kWStages = 3;          // ring depth per warp
constexpr int kWStageBytes = 8192;   // K + V bytes per stage

template <typename T, int HD>
struct Shape {
  static constexpr int VEC = Elem<T>::kVec;                       // elements per lane load
  static constexpr int LPS = HD / VEC;                            // lanes per slot
  static constexpr int SPW = 32 / LPS;                            // slots per warp step
  static constexpr int STAGE_SLOTS = kWStageBytes / (2 * HD * (int)sizeof(T));
  static constexpr int STAGE_ELEMS = STAGE_SLOTS * HD;
  static constexpr int ITERS = STAGE_SLOTS / SPW;
  static_assert(LPS >= 1 && LPS <= 32 && (32 % LPS) == 0, "lane split");
  static_assert(ITERS >= 1 && STAGE_SLOTS % SPW == 0 && STAGE_SLOTS <= 32, "stage split");
};

template <typename T>
__device__ __forceinline__ void store_vec(T* dst, const float* v);
template <>
__device__ __forceinline__ void store_vec<float>(float* dst, const float* v) {
  *reinterpret_cast<float4*>(dst) = make_float4(v[0], v[1], v[2], v[3]);
}
template <>
__device__ __forceinline__ void store_vec<__nv_bfloat16>(__nv_bfloat16* dst, const float* v) {
  uint4 u;
  __nv_bfloat162 t;
  t = __floats2bfloat162_rn(v[0], v[1]); u.x = *reinterpret_cast<uint32_t*>(&t);
  t = __floats2bfloat162_rn(v[2], v[3]); u.y = *reinterpret_cast<uint32_t*>(&t);
  t = __floats2bfloat162_rn(v[4], v[5]); u.z = *reinterpret_cast<uint32_t*>(&t);
  t = __floats2bfloat162_rn(v[6], v[7]); u.w = *reinterpret_cast<uint32_t*>(&t);
  *reinterpret_cast<uint4*>(dst) = u;
}

// Position in the stage stream: sequence b, kv head h, stage st of nst.
struct Cursor {
  int b, h, st, nst;
};

__device__ __forceinline__ Cursor locate(int64_t x, const int* pre, int B, int Hkv) {
  int lo = 0, hi = B;  // largest b with Hkv * pre[b] <= x
  while (hi - lo > 1) {
    const int mid = (lo + hi) >> 1;
    if ((int64_t)Hkv * pre[mid] <= x) lo = mid; else hi = mid;
  }
  Cursor c;
  c.b = lo;
  c.nst = pre[lo + 1] - pre[lo];
  const int64_t r = x - (int64_t)Hkv * pre[lo];
  c.h = (int)(r / c.nst);
  c.st = (int)(r % c.nst);
  return c;
}

__device__ __forceinline__ void advance(Cursor& c, const int* pre, int B, int Hkv) {
  if (++c.st < c.nst) return;
  c.st = 0;
  if (++c.h < Hkv) return;
  c.h = 0;
  do { ++c.b; } while (c.b < B && pre[c.b + 1] == pre[c.b]);
  if (c.b < B) c.nst = pre[c.b + 1] - pre[c.b];
}

// Warp owning global stage x: the largest g with floor(g * NS / GW) <= x.
__device__ __forceinline__ int64_t warp_of(int64_t x, int64_t NS, int64_t GW) {
  return ((x + 1) * GW - 1) / NS;
}

template <typename T, int HD, int G>
__global__ void __launch_bounds__(kThreads) decode_attn_kernel(const AttnParams p) {
  using SH = Shape<T, HD>;
  constexpr int VEC = SH::VEC, LPS = SH::LPS, SPW = SH::SPW;
  constexpr int STAGE_SLOTS = SH::STAGE_SLOTS, STAGE_ELEMS = SH::STAGE_ELEMS, ITERS = SH::ITERS;
  constexpr uint32_t KV_BYTES = STAGE_ELEMS * sizeof(T);
  constexpr uint32_t Q_BYTES = G * HD * sizeof(T);

  extern __shared__ __align__(128) unsigned char smem_raw[];
  T* ring = reinterpret_cast<T*>(smem_raw);                       // [W][S][2][STAGE_ELEMS]
  T* qring = ring + kWarps * kWStages * 2 * STAGE_ELEMS;          // [W][S][G*HD]
  int* pre = reinterpret_cast<int*>(qring + kWarps * kWStages * G * HD);  // [B+1]
  int* lens = pre + p.B + 1;                                      // [B]
  __shared__ uint64_t bars[kWarps][kWStages];
  __shared__ uint64_t masks[kWarps][kWStages];
  __shared__ int scan[kThreads];

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int B = p.B, Hkv = p.Hkv;
  const int max_slots = p.max_pages * p.P;

  // ---- stages per sequence and their prefix sums (every CTA, all threads)
  {
    const int per = (B + kThreads - 1) / kThreads;
    const int i0 = min(B, tid * per), i1 = min(B, i0 + per);
    int sum = 0;
    for (int i = i0; i < i1; ++i) {
      const int S = p.seq_lens[i];
      const bool ok = S >= 1 && S <= max_slots;
      lens[i] = ok ? S : 0;
      sum += ok ? (S + STAGE_SLOTS - 1) / STAGE_SLOTS : 0;
    }
    scan[tid] = sum;
    __syncthreads();
    for (int o = 1; o < kThreads; o <<= 1) {  // inclusive Hillis-Steele scan
      const int v = tid >= o ? scan[tid - o] : 0;
      __syncthreads();
      scan[tid] += v;
      __syncthreads();
    }
    int run = scan[tid] - sum;
    for (int i = i0; i < i1; ++i) {
      pre[i] = run;
      run += lens[i] ? (lens[i] + STAGE_SLOTS - 1) / STAGE_SLOTS : 0;
    }
    if (tid == kThreads - 1) pre[B] = scan[tid];
    if (lane == 0)
      for (int s = 0; s < kWStages; ++s) mbar_init(&bars[warp][s], 1);
    fence_mbar_init();
    __syncthreads();
  }
  // ---- sequences with an invalid length: zero output rows, report once
  if (blockIdx.x == 0) {
    for (int b = 0; b < B; ++b) {
      if (lens[b] != 0) continue;
      T* o = reinterpret_cast<T*>(p.out) + (int64_t)b * p.Hq * HD;
      for (int i = tid; i < p.Hq * HD; i += kThreads) o[i] = Elem<T>::from_f(0.f);
      if (tid == 0) report(p.status, WM_ERR_BOUNDS);
    }
  }

  // Equal stage ranges over the first GW warps; with fewer stages than warps
  // only NS warps take one stage each, so every warp in a unit's span has work.
  const int64_t NS = (int64_t)Hkv * pre[B];
  const int64_t GW = min((int64_t)gridDim.x * kWarps, NS);
  const int64_t gw = (int64_t)blockIdx.x * kWarps + warp;
  if (gw >= GW) return;  // warp-level from here on: no block barriers below
  const int64_t x0 = gw * NS / GW, x1 = (gw + 1) * NS / GW;

  T* myring = ring + warp * kWStages * 2 * STAGE_ELEMS;
  T* myq = qring + warp * kWStages * G * HD;
  const uint64_t policy = l2_evict_first_policy();
  const int lane_slot = lane / LPS, lane_part = lane % LPS;

  // ---- producer: stage xp at cursor pc into ring slot buf
  Cursor pc = locate(x0, pre, B, Hkv);
  int64_t xp = x0;
  auto issue = [&](int buf) {
    const bool first = (xp == x0) || pc.st == 0;
    const int S = lens[pc.b];
    const int s_begin = pc.st * STAGE_SLOTS;
    const int32_t* pt = p.page_table + (int64_t)pc.b * p.max_pages;
    const T* kb = reinterpret_cast<const T*>(p.k_pool) + (int64_t)pc.h * p.P * HD;
    const T* vb = reinterpret_cast<const T*>(p.v_pool) + (int64_t)pc.h * p.P * HD;
    T* kd = myring + buf * 2 * STAGE_ELEMS;
    T* vd = kd + STAGE_ELEMS;
    uint64_t* bar = &bars[warp][buf];
    const uint32_t qb = first ? Q_BYTES : 0u;
    const T* qsrc = reinterpret_cast<const T*>(p.q) + ((int64_t)pc.b * p.Hq + pc.h * G) * HD;
    if (p.P >= STAGE_SLOTS) {
      if (lane == 0) {
        const int pg = pt[s_begin >> p.log2P];
        const bool ok = pg >= 0 && pg < p.num_pages;
        masks[warp][buf] = ok ? 1ull : 0ull;
        if (!ok) report(p.status, WM_ERR_BOUNDS);
        mbar_arrive_expect_tx(bar, (ok ? 2 * KV_BYTES : 0u) + qb);
        if (ok) {
          const int64_t off = (int64_t)pg * p.page_stride + (int64_t)(s_begin & (p.P - 1)) * HD;
          bulk_g2s(kd, kb + off, KV_BYTES, bar, policy);
          bulk_g2s(vd, vb + off, KV_BYTES, bar, policy);
        }
        if (first) bulk_g2s(myq + buf * G * HD, qsrc, Q_BYTES, bar, policy);
      }
    } else {
      const int npp = STAGE_SLOTS >> p.log2P;           // pages per stage (<= 32)
      const int lp0 = s_begin >> p.log2P;
      const int lpn = min(npp, ((S - 1) >> p.log2P) - lp0 + 1);
      int pg = -1;
      if (lane < lpn) pg = pt[lp0 + lane];
      const bool ok = lane < lpn && pg >= 0 && pg < p.num_pages;
      const uint32_t mask = __ballot_sync(0xFFFFFFFFu, ok);
      const uint32_t bytes = (uint32_t)p.P * HD * sizeof(T);
      if (lane == 0) {
        masks[warp][buf] = mask;
        if (__popc(mask) < lpn) report(p.status, WM_ERR_BOUNDS);
        mbar_arrive_expect_tx(bar, 2u * bytes * (uint32_t)__popc(mask) + qb);
        if (first) bulk_g2s(myq + buf * G * HD, qsrc, Q_BYTES, bar, policy);
      }
      __syncwarp();
      if (ok) {
        const int64_t off = (int64_t)pg * p.page_stride;
        bulk_g2s(kd + lane * p.P * HD, kb + off, bytes, bar, policy);
        bulk_g2s(vd + lane * p.P * HD, vb + off, bytes, bar, policy);
      }
    }
    ++xp;
    advance(pc, pre, B, Hkv);
  };

  for (int s = 0; s < kWStages && xp < x1; ++s) issue(s);

  // ---- consumer
  Cursor cc = locate(x0, pre, B, Hkv);
  bool piece_first = true;  // the piece that starts at x0 is this warp's first
  float qv[G][VEC];
  float m[G], l[G], acc[G][VEC];
  for (int64_t x = x0; x < x1; ++x) {
    const int buf = (int)((x - x0) % kWStages);
    const uint32_t parity = (uint32_t)(((x - x0) / kWStages) & 1);
    const bool ok = mbar_wait(&bars[warp][buf], parity);
    if (__any_sync(0xFFFFFFFFu, !ok)) {
      // a copy never landed: report, drain what is in flight (bounded) and stop
      if (lane == 0) {
        report(p.status, WM_ERR_TIMEOUT);
        for (int64_t y = x; y < xp; ++y)
          mbar_wait(&bars[warp][(y - x0) % kWStages], (uint32_t)(((y - x0) / kWStages) & 1));
      }
      __syncwarp();
      return;
    }
    const bool start = (x == x0) || cc.st == 0;
    if (start) {
      const T* qs = myq + buf * G * HD + lane_part * VEC;
#pragma unroll
      for (int g = 0; g < G; ++g) {
        float f[VEC];
        Elem<T>::unpack(*reinterpret_cast<const uint4*>(qs + g * HD), f);
#pragma unroll
        for (int v = 0; v < VEC; ++v) qv[g][v] = f[v] * p.qscale;
        m[g] = -INFINITY;
        l[g] = 0.f;
#pragma unroll
        for (int v = 0; v < VEC; ++v) acc[g][v] = 0.f;
      }
    }
    const int S = lens[cc.b];
    const int s_begin = cc.st * STAGE_SLOTS;
    const uint64_t mask = masks[warp][buf];
    const T* Ks = myring + buf * 2 * STAGE_ELEMS;
    const T* Vs = Ks + STAGE_ELEMS;
    float sc[G][ITERS];
#pragma unroll
    for (int it = 0; it < ITERS; ++it) {
      const int ls = it * SPW + lane_slot;
      float kf[VEC];
      Elem<T>::unpack(*reinterpret_cast<const uint4*>(Ks + ls * HD + lane_part * VEC), kf);
      const int pidx = (p.P >= STAGE_SLOTS) ? 0 : (ls >> p.log2P);
      const bool valid = (s_begin + ls < S) && ((mask >> pidx) & 1ull);
#pragma unroll
      for (int g = 0; g < G; ++g) {
        float s = 0.f;
#pragma unroll
        for (int v = 0; v < VEC; ++v) s = fmaf(qv[g][v], kf[v], s);
        s = group_sum<LPS>(s);
        sc[g][it] = valid ? s : -INFINITY;
      }
    }
#pragma unroll
    for (int g = 0; g < G; ++g) {
      float mx = sc[g][0];
#pragma unroll
      for (int it = 1; it < ITERS; ++it) mx = fmaxf(mx, sc[g][it]);
      const float mnew = fmaxf(m[g], mx);
      if (mnew != -INFINITY) {
        const float corr = exp2f(m[g] - mnew);  // 0 while m is still -inf
        l[g] *= corr;
#pragma unroll
        for (int v = 0; v < VEC; ++v) acc[g][v] *= corr;
        m[g] = mnew;
      }
    }
#pragma unroll
    for (int it = 0; it < ITERS; ++it) {
      const int ls = it * SPW + lane_slot;
      float vf[VEC];
      Elem<T>::unpack(*reinterpret_cast<const uint4*>(Vs + ls * HD + lane_part * VEC), vf);
#pragma unroll
      for (int g = 0; g < G; ++g) {
        if (sc[g][it] != -INFINITY) {  // masked slots never touch the sums (NaN-safe)
          const float pr = exp2f(sc[g][it] - m[g]);
          l[g] += pr;
#pragma unroll
          for (int v = 0; v < VEC; ++v) acc[g][v] = fmaf(pr, vf[v], acc[g][v]);
        }
      }
    }
    __syncwarp();  // every lane is done with this ring slot
    if (xp < x1) issue(buf);

    const bool end = (x == x1 - 1) || cc.st == cc.nst - 1;
    if (end) {
      // merge the lane groups of the warp
#pragma unroll
      for (int g = 0; g < G; ++g) {
        float M = m[g];
#pragma unroll
        for (int o = LPS; o < 32; o <<= 1) M = fmaxf(M, __shfl_xor_sync(0xFFFFFFFFu, M, o));
        const float w = (m[g] == -INFINITY) ? 0.f : exp2f(m[g] - M);
        float Ls = l[g] * w;
#pragma unroll
        for (int o = LPS; o < 32; o <<= 1) Ls += __shfl_xor_sync(0xFFFFFFFFu, Ls, o);
#pragma unroll
        for (int v = 0; v < VEC; ++v) {
          float a = acc[g][v] * w;
#pragma unroll
          for (int o = LPS; o < 32; o <<= 1) a += __shfl_xor_sync(0xFFFFFFFFu, a, o);
          acc[g][v] = a;
        }
        m[g] = M;
        l[g] = Ls;
      }
      const int64_t rowbase = (int64_t)cc.b * p.Hq + cc.h * G;
      const int64_t U = (int64_t)Hkv * pre[cc.b] + (int64_t)cc.h * cc.nst;
      const int64_t g_first = warp_of(U, NS, GW), g_last = warp_of(U + cc.nst - 1, NS, GW);
      T* outp = reinterpret_cast<T*>(p.out);
      if (g_first == g_last) {
        if (lane_slot == 0) {
#pragma unroll
          for (int g = 0; g < G; ++g) {
            float o[VEC];
            const float inv = l[g] > 0.f ? 1.f / l[g] : 0.f;
#pragma unroll
            for (int v = 0; v < VEC; ++v) o[v] = acc[g][v] * inv;
            store_vec<T>(outp + (rowbase + g) * HD + lane_part * VEC, o);
          }
        }
      } else {
        // partial of this piece: its warp's first piece -> A[gw], last piece -> Z[gw]
        const bool is_last_piece = (x == x1 - 1);
        for (int side = 0; side < 2; ++side) {
          if ((side == 0 && !piece_first) || (side == 1 && !is_last_piece)) continue;
          float* po = p.part_o + ((int64_t)side * p.nwarps + gw) * G * HD;
          float* pm = p.part_ml + ((int64_t)side * p.nwarps + gw) * G * 2;
          if (lane_slot == 0) {
#pragma unroll
            for (int g = 0; g < G; ++g)
#pragma unroll
              for (int v = 0; v < VEC; ++v) po[g * HD + lane_part * VEC + v] = acc[g][v];
          }
          if (lane == 0) {
#pragma unroll
            for (int g = 0; g < G; ++g) {
              pm[2 * g] = m[g];
              pm[2 * g + 1] = l[g];
            }
          }
        }
        __threadfence();
        __syncwarp();
        int last = 0;
        if (lane == 0) {
          const int t = atomicAdd(&p.counters[cc.b * Hkv + cc.h], 1);
          last = (t == (int)(g_last - g_first));
        }
        last = __shfl_sync(0xFFFFFFFFu, last, 0);
        if (last) {
          __threadfence();
          // merge pieces of warps g_first .. g_last (Z of the first, A of the rest)
          for (int g = 0; g < G; ++g) {
            float M = -INFINITY;
            for (int64_t q = g_first; q <= g_last; ++q) {
              const int side = q == g_first ? 1 : 0;
              M = fmaxf(M, __ldcg(p.part_ml + ((int64_t)side * p.nwarps + q) * G * 2 + 2 * g));
            }
            float o[HD / 32];
#pragma unroll
            for (int i = 0; i < HD / 32; ++i) o[i] = 0.f;
            float Ls = 0.f;
            for (int64_t q = g_first; q <= g_last; ++q) {
              const int side = q == g_first ? 1 : 0;
              const float* pm = p.part_ml + ((int64_t)side * p.nwarps + q) * G * 2 + 2 * g;
              const float mq = __ldcg(pm);
              if (mq == -INFINITY) continue;
              const float w = exp2f(mq - M);
              Ls = fmaf(w, __ldcg(pm + 1), Ls);
              const float* po = p.part_o + (((int64_t)side * p.nwarps + q) * G + g) * HD;
#pragma unroll
              for (int i = 0; i < HD / 32; ++i) o[i] = fmaf(w, __ldcg(po + lane + 32 * i), o[i]);
            }
            const float inv = Ls > 0.f ? 1.f / Ls : 0.f;
#pragma unroll
            for (int i = 0; i < HD / 32; ++i)
              outp[(rowbase + g) * HD + lane + 32 * i] = Elem<T>::from_f(o[i] * inv);
          }
          if (lane == 0) p.counters[cc.b * Hkv + cc.h] = 0;
        }
      }
      piece_first = false;
    }
    advance(cc, pre, B, Hkv);
  }
}

template <typename T, int HD>
constexpr int stage_slots() {
  return Shape<T, HD>::STAGE_SLOTS;
}

template <typename T, int HD, int G>
cudaError_t launch_t(const AttnParams& p, int grid, size_t smem, cudaStream_t stream) {
  static size_t smem_set = 0;  // largest dynamic smem opted into so far
  auto kern = decode_attn_kernel<T, HD, G>;
  if (smem > smem_set) {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    smem_set = smem;
  }
  kern<<<grid, kThreads, smem, stream>>>(p);
  return cudaGetLastError();
}

template <typename T, int HD>
cudaError_t launch_g(const AttnParams& p, int G, int grid, size_t smem, cudaStream_t s) {
  switch (G) {
    case 1: return launch_t<T, HD, 1>(p, grid, smem, s);
    case 2: return launch_t<T, HD, 2>(p, grid, smem, s);
    case 4: return launch_t<T, HD, 4>(p, grid, smem, s);
    case 8: return launch_t<T, HD, 8>(p, grid, smem, s);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace

int attn_stage_slots(int dtype, int d) {
  if (dtype == WM_DT_F32) return d == 64 ? stage_slots<float, 64>() : stage_slots<float, 128>();
  return d == 64 ? stage_slots<__nv_bfloat16, 64>() : stage_slots<__nv_bfloat16, 128>();
}

int attn_warps_per_cta() { return kWarps; }

size_t attn_smem_bytes(int dtype, int d, int G, int B) {
  const size_t esz = dtype == WM_DT_F32 ? 4 : 2;
  return (size_t)kWarps * kWStages * kWStageBytes + (size_t)kWarps * kWStages * G * d * esz +
         sizeof(int) * (2 * (size_t)B + 1);
}

cudaError_t launch_decode_attn(const AttnParams& p, int dtype, int d, int G, int grid,
                               cudaStream_t s) {
  const size_t smem = attn_smem_bytes(dtype, d, G, p.B);
  if (dtype == WM_DT_F32) {
    return d == 64 ? launch_g<float, 64>(p, G, grid, smem, s)
                   : launch_g<float, 128>(p, G, grid, smem, s);
  }
  return d == 64 ? launch_g<__nv_bfloat16, 64>(p, G, grid, smem, s)
                 : launch_g<__nv_bfloat16, 128>(p, G, grid, smem, s);
}

}  // namespace wm
