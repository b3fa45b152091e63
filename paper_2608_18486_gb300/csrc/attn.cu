// Decode attention over one channel of the paged k-channel cache
// (Sec. 3.1 Step 3; dummy slot of Sec. 3.2).
//
// Design (GB300): one CTA per (chunk of slots, kv head, sequence).  The
// (page, kv-head) blocks of the cache are contiguous [page_size][d] runs, so a
// single thread streams them into shared memory with 1-D bulk async copies
// (TMA engine, mbarrier completion, L2 evict-first), NST stages deep.  Four
// warps consume each stage on the CUDA cores: a group of d/VEC lanes owns
// one slot (one 16-byte vector per lane), reduces q.k with xor shuffles, and
// keeps an online-softmax state (running max m, sum l, output accumulator).
// This work reads about one byte per FLOP, so it is HBM-bound and stays off
// the tensor cores.  Group states merge in shared memory; when a sequence
// spans several chunks, each CTA writes a partial (m, l, o) and the last CTA
// to arrive (atomic ticket, no waiting) merges them and resets its ticket.
#include <math.h>

#include "common.cuh"
#include "internal.h"

namespace wm {

namespace {

constexpr int kAttnWarps = 4;
constexpr int kAttnThreads = kAttnWarps * 32;
constexpr int kAttnStages = 4;
constexpr int kStageBytes = 16384;  // K + V bytes per pipeline stage

template <typename T, int HD>
struct AttnShape {
  static constexpr int VEC = Elem<T>::kVec;                 // elements per lane load
  static constexpr int LPS = HD / VEC;                      // lanes per slot
  static constexpr int SPW = 32 / LPS;                      // slots per warp step
  static constexpr int STAGE_SLOTS = kStageBytes / (2 * HD * (int)sizeof(T));
  static constexpr int STAGE_ELEMS = STAGE_SLOTS * HD;
  static constexpr int SLOTS_PER_WARP = STAGE_SLOTS / kAttnWarps;
  static constexpr int ITERS = SLOTS_PER_WARP / SPW;
  static_assert(LPS >= 1 && LPS <= 32 && (32 % LPS) == 0, "lane split");
  static_assert(ITERS >= 1 && SLOTS_PER_WARP % SPW == 0, "stage split");
};

template <typename T, int HD, int G>
__global__ void __launch_bounds__(kAttnThreads)
    decode_attn_kernel(const AttnParams p) {
  using S_ = AttnShape<T, HD>;
  constexpr int VEC = S_::VEC, LPS = S_::LPS, SPW = S_::SPW;
  constexpr int STAGE_SLOTS = S_::STAGE_SLOTS, STAGE_ELEMS = S_::STAGE_ELEMS;
  constexpr int ITERS = S_::ITERS, NST = kAttnStages;
  constexpr int NGRP = kAttnWarps * SPW;  // independent softmax states per CTA

  extern __shared__ __align__(128) unsigned char smem_raw[];
  T* kbuf = reinterpret_cast<T*>(smem_raw);
  T* vbuf = kbuf + NST * STAGE_ELEMS;
  __shared__ uint64_t bars[NST];
  __shared__ uint64_t page_ok[NST];  // bit i: page i of the stage was fetched
  __shared__ int s_last;

  const int c = blockIdx.x, hkv = blockIdx.y, b = blockIdx.z;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int lane_slot = lane / LPS, lane_part = lane % LPS;
  const int max_slots = p.max_pages * p.P;
  const int S = p.seq_lens[b];
  const int row0 = b * p.Hq + hkv * G;  // first query row of this kv group

  if (S < 1 || S > max_slots) {
    if (c == 0) {
      T* o = reinterpret_cast<T*>(p.out) + (int64_t)row0 * HD;
      for (int i = tid; i < G * HD; i += kAttnThreads) o[i] = Elem<T>::from_f(0.f);
      if (tid == 0) report(p.status, WM_ERR_BOUNDS);
    }
    return;
  }
  const int nchunks = (S + p.chunk_slots - 1) / p.chunk_slots;
  if (c >= nchunks) return;
  const int slot0 = c * p.chunk_slots;
  const int slot_end = min(S, slot0 + p.chunk_slots);
  const int nstages = (slot_end - slot0 + STAGE_SLOTS - 1) / STAGE_SLOTS;
  const int32_t* pt = p.page_table + (int64_t)b * p.max_pages;
  const T* kb = reinterpret_cast<const T*>(p.k_pool) + (int64_t)hkv * p.P * HD;
  const T* vb = reinterpret_cast<const T*>(p.v_pool) + (int64_t)hkv * p.P * HD;
  const int last_page = (S - 1) >> p.log2P;  // last logical page holding a slot < S

  if (tid == 0) {
    for (int i = 0; i < NST; ++i) mbar_init(&bars[i], 1);
    fence_mbar_init();
  }
  __syncthreads();

  const uint64_t policy = l2_evict_first_policy();
  // Thread 0 only: fetch stage st (slots slot0 + st*STAGE_SLOTS ...) into its buffer.
  auto issue = [&](int st) {
    const int buf = st % NST;
    const int s_begin = slot0 + st * STAGE_SLOTS;
    T* kd = kbuf + buf * STAGE_ELEMS;
    T* vd = vbuf + buf * STAGE_ELEMS;
    if (p.P >= STAGE_SLOTS) {
      const int pg = pt[s_begin >> p.log2P];
      const bool ok = pg >= 0 && pg < p.num_pages;
      page_ok[buf] = ok ? 1ull : 0ull;
      if (ok) {
        constexpr uint32_t bytes = STAGE_ELEMS * sizeof(T);
        const int64_t off = (int64_t)pg * p.page_stride + (int64_t)(s_begin & (p.P - 1)) * HD;
        mbar_arrive_expect_tx(&bars[buf], 2 * bytes);
        bulk_g2s(kd, kb + off, bytes, &bars[buf], policy);
        bulk_g2s(vd, vb + off, bytes, &bars[buf], policy);
      } else {
        report(p.status, WM_ERR_BOUNDS);
        mbar_arrive_expect_tx(&bars[buf], 0);
      }
    } else {
      const int npp = STAGE_SLOTS >> p.log2P;
      const int lp0 = s_begin >> p.log2P;
      const int lpn = min(npp, last_page - lp0 + 1);
      const uint32_t bytes = (uint32_t)p.P * HD * sizeof(T);
      uint64_t mask = 0;
      int nvalid = 0;
      for (int i = 0; i < lpn; ++i) {
        const int pg = pt[lp0 + i];
        if (pg >= 0 && pg < p.num_pages) {
          mask |= 1ull << i;
          ++nvalid;
        }
      }
      if (nvalid < lpn) report(p.status, WM_ERR_BOUNDS);
      page_ok[buf] = mask;
      mbar_arrive_expect_tx(&bars[buf], 2u * bytes * (uint32_t)nvalid);
      for (int i = 0; i < lpn; ++i) {
        if (!((mask >> i) & 1ull)) continue;
        const int64_t off = (int64_t)pt[lp0 + i] * p.page_stride;
        bulk_g2s(kd + i * p.P * HD, kb + off, bytes, &bars[buf], policy);
        bulk_g2s(vd + i * p.P * HD, vb + off, bytes, &bars[buf], policy);
      }
    }
  };

  if (tid == 0)
    for (int st = 0; st < min(NST, nstages); ++st) issue(st);

  // query of the G heads of this kv group, pre-scaled to log2 units
  float qv[G][VEC];
  {
    const T* qp = reinterpret_cast<const T*>(p.q) + (int64_t)row0 * HD + lane_part * VEC;
#pragma unroll
    for (int g = 0; g < G; ++g) {
      float f[VEC];
      Elem<T>::unpack(*reinterpret_cast<const uint4*>(qp + g * HD), f);
#pragma unroll
      for (int v = 0; v < VEC; ++v) qv[g][v] = f[v] * p.qscale;
    }
  }
  float m[G], l[G], acc[G][VEC];
#pragma unroll
  for (int g = 0; g < G; ++g) {
    m[g] = -INFINITY;
    l[g] = 0.f;
#pragma unroll
    for (int v = 0; v < VEC; ++v) acc[g][v] = 0.f;
  }

  const int log2pp = p.log2P;  // page index inside a stage = local slot >> log2P
  bool timed_out = false;
  int st = 0;
  for (; st < nstages; ++st) {
    const int buf = st % NST;
    const bool ok = mbar_wait(&bars[buf], (st / NST) & 1);
    if (__syncthreads_or(!ok)) {
      timed_out = true;
      break;
    }
    const T* Ks = kbuf + buf * STAGE_ELEMS;
    const T* Vs = vbuf + buf * STAGE_ELEMS;
    const uint64_t mask = page_ok[buf];
    const int s_begin = slot0 + st * STAGE_SLOTS;
    float sc[G][ITERS];
#pragma unroll
    for (int it = 0; it < ITERS; ++it) {
      const int ls = warp * S_::SLOTS_PER_WARP + it * SPW + lane_slot;
      float kf[VEC];
      Elem<T>::unpack(*reinterpret_cast<const uint4*>(Ks + ls * HD + lane_part * VEC), kf);
      const int pidx = (p.P >= STAGE_SLOTS) ? 0 : (ls >> log2pp);
      const bool valid = (s_begin + ls < slot_end) && ((mask >> pidx) & 1ull);
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
      const int ls = warp * S_::SLOTS_PER_WARP + it * SPW + lane_slot;
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
    __syncthreads();  // every warp is done with this buffer
    if (tid == 0 && st + NST < nstages) issue(st + NST);
  }

  if (timed_out) {
    // drain the copies still in flight (bounded), then contribute nothing
    if (tid == 0) {
      report(p.status, WM_ERR_TIMEOUT);
      for (int s2 = st; s2 < min(nstages, st + NST); ++s2) mbar_wait(&bars[s2 % NST], (s2 / NST) & 1);
    }
    __syncthreads();
#pragma unroll
    for (int g = 0; g < G; ++g) {
      m[g] = -INFINITY;
      l[g] = 0.f;
    }
  }

  // ---- merge the NGRP group states of this CTA (stage buffers are free now)
  float* red = reinterpret_cast<float*>(smem_raw);  // [NGRP][G][HD]
  float* redml = red + NGRP * G * HD;               // [NGRP][G][2]
  {
    const int grp = warp * SPW + lane_slot;
#pragma unroll
    for (int g = 0; g < G; ++g) {
#pragma unroll
      for (int v = 0; v < VEC; ++v) red[(grp * G + g) * HD + lane_part * VEC + v] = acc[g][v];
      if (lane_part == 0) {
        redml[(grp * G + g) * 2] = m[g];
        redml[(grp * G + g) * 2 + 1] = l[g];
      }
    }
  }
  __syncthreads();
  T* outp = reinterpret_cast<T*>(p.out);
  for (int i = tid; i < G * HD; i += kAttnThreads) {
    const int g = i / HD, e = i % HD;
    float M = -INFINITY;
    for (int q = 0; q < NGRP; ++q) M = fmaxf(M, redml[(q * G + g) * 2]);
    float o = 0.f, Ls = 0.f;
    if (M != -INFINITY) {
      for (int q = 0; q < NGRP; ++q) {
        const float mq = redml[(q * G + g) * 2];
        if (mq != -INFINITY) {
          const float w = exp2f(mq - M);
          o = fmaf(w, red[(q * G + g) * HD + e], o);
          Ls = fmaf(w, redml[(q * G + g) * 2 + 1], Ls);
        }
      }
    }
    const int64_t row = row0 + g;
    if (nchunks == 1) {
      outp[row * HD + e] = Elem<T>::from_f(Ls > 0.f ? o / Ls : 0.f);
    } else {
      const int64_t pr = row * p.max_chunks + c;
      p.part_o[pr * HD + e] = o;
      if (e == 0) {
        p.part_ml[pr * 2] = M;
        p.part_ml[pr * 2 + 1] = Ls;
      }
    }
  }
  if (nchunks == 1) return;

  // ---- the last chunk CTA of this (sequence, kv head) merges all partials
  __threadfence();
  __syncthreads();
  if (tid == 0) {
    const int t = atomicAdd(&p.counters[b * p.Hkv + hkv], 1);
    s_last = (t == nchunks - 1);
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  for (int i = tid; i < G * HD; i += kAttnThreads) {
    const int g = i / HD, e = i % HD;
    const int64_t row = row0 + g;
    const float* ml = p.part_ml + row * p.max_chunks * 2;
    const float* po = p.part_o + row * p.max_chunks * HD + e;
    float M = -INFINITY;
    for (int cc = 0; cc < nchunks; ++cc) M = fmaxf(M, __ldcg(ml + 2 * cc));
    float o = 0.f, Ls = 0.f;
    if (M != -INFINITY) {
      for (int cc = 0; cc < nchunks; ++cc) {
        const float mc = __ldcg(ml + 2 * cc);
        if (mc != -INFINITY) {
          const float w = exp2f(mc - M);
          o = fmaf(w, __ldcg(po + (int64_t)cc * HD), o);
          Ls = fmaf(w, __ldcg(ml + 2 * cc + 1), Ls);
        }
      }
    }
    outp[row * HD + e] = Elem<T>::from_f(Ls > 0.f ? o / Ls : 0.f);
  }
  if (tid == 0) p.counters[b * p.Hkv + hkv] = 0;
}

template <typename T, int HD>
int stage_slots() {
  return AttnShape<T, HD>::STAGE_SLOTS;
}

template <typename T, int HD, int G>
cudaError_t launch_t(const AttnParams& p, int B, int Hkv, cudaStream_t stream) {
  const size_t smem = (size_t)kAttnStages * kStageBytes;  // K and V stage buffers
  auto kern = decode_attn_kernel<T, HD, G>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  dim3 grid(p.max_chunks, Hkv, B);
  kern<<<grid, kAttnThreads, smem, stream>>>(p);
  return cudaGetLastError();
}

template <typename T, int HD>
cudaError_t launch_g(const AttnParams& p, int G, int B, int Hkv, cudaStream_t s) {
  switch (G) {
    case 1: return launch_t<T, HD, 1>(p, B, Hkv, s);
    case 2: return launch_t<T, HD, 2>(p, B, Hkv, s);
    case 4: return launch_t<T, HD, 4>(p, B, Hkv, s);
    case 8: return launch_t<T, HD, 8>(p, B, Hkv, s);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace

int attn_stage_slots(int dtype, int d) {
  if (dtype == WM_DT_F32) return d == 64 ? stage_slots<float, 64>() : stage_slots<float, 128>();
  return d == 64 ? stage_slots<__nv_bfloat16, 64>() : stage_slots<__nv_bfloat16, 128>();
}

cudaError_t launch_decode_attn(const AttnParams& p, int dtype, int d, int G, int B, int Hkv,
                               cudaStream_t s) {
  if (dtype == WM_DT_F32) {
    return d == 64 ? launch_g<float, 64>(p, G, B, Hkv, s) : launch_g<float, 128>(p, G, B, Hkv, s);
  }
  return d == 64 ? launch_g<__nv_bfloat16, 64>(p, G, B, Hkv, s)
                 : launch_g<__nv_bfloat16, 128>(p, G, B, Hkv, s);
}

}  // namespace wm
