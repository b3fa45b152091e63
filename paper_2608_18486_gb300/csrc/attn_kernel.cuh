#pragma once
// Decode attention over one channel of the paged k-channel cache
// (Sec. 3.1 Step 3; dummy slot of Sec. 3.2).
//
// Design (GB300).  The work is a stream over the KV blocks of every
// (sequence b, kv head h) unit of the chosen channel; it reads about one byte
// per FLOP, so it is HBM-bound and runs on the CUDA cores.
//
//  * Stream-K split.  Each unit is cut into pipeline stages of STAGE_SLOTS
//    slots (4 or 8 KB of K+V).  The stages of all units, concatenated, are
//    cut into equal chunks of CH stages.  Warp w of the persistent grid
//    starts on chunk w and then takes further chunks from an atomic counter
//    (requested one chunk ahead), so warps that stream faster take more
//    chunks and all finish together whatever the sequence lengths.
//  * Private pipelines.  Each warp owns a 3-deep ring in shared memory and
//    fills it with 1-D bulk async copies (TMA engine, mbarrier completion,
//    L2 evict-first) of contiguous (page, kv-head) runs; it refills a slot as
//    soon as it has consumed it, so no block-wide barrier is ever taken.
//  * Compute.  8 lanes own one slot (16-byte vectors, conflict-free shared
//    loads), reduce q.k with xor shuffles and keep an online softmax
//    (running max m, sum l, accumulator) per lane group; groups merge with
//    shuffles at the end of a piece.
//  * Merge.  A piece of a unit that lies inside one chunk is written straight
//    to the output.  Only units that cross a chunk boundary leave partials
//    (at most two per chunk: its first and its last piece).  A warp takes
//    its ticket on the unit first: the warp that completes the unit merges,
//    every other one publishes its partial and then flags it (a release
//    store), so the merger never publishes its own piece and waits (bounded)
//    only for flags that are in flight.  A piece that ends in the middle of
//    its warp's chunk stores its record and takes its ticket without
//    waiting for either, and raises its flag (or merges, if it was last) at
//    the chunk's end: a release or fence issued while the warp's bulk copies
//    are in flight waits for them, which stalled the stream at every unit
//    boundary.  Tickets are taken before the math of a piece's last stage.
//    When the merger has no stage left in flight, its idle ring receives the
//    unit's partial records with bulk copies (one round trip for up to a
//    ring's worth), and the merge reads them from shared memory.
#include <math.h>

#include "common.cuh"
#include "internal.h"

namespace wm {
namespace attn_detail {

constexpr int kWarps = 4;
constexpr int kThreads = kWarps * 32;
constexpr int kWStages = 3;          // ring depth per warp

// Largest power of two <= x (x >= 1).
constexpr int pow2_floor(int x) { return x >= 2 ? 2 * pow2_floor(x / 2) : 1; }

// SB: K + V byte budget of one pipeline stage (4 KB or 8 KB).
template <typename T, int HD, int SB>
struct Shape {
  // A slot row is ROW_VECS 16-byte vectors.  LPS lanes own one slot, lane
  // part p holding vectors p, p + LPS, ...; with 8 lanes a quarter warp reads
  // one contiguous 128-byte run, with 4 lanes (rows of 12 vectors, d = 96
  // bf16) it reads 64 bytes from each of two rows 192 bytes apart, which
  // fall on disjoint banks.  Either way every 16-byte shared load of the
  // warp is bank-conflict free.
  static constexpr int VEC = Elem<T>::kVec;                       // elements per 16 bytes
  static constexpr int ROW_VECS = HD * (int)sizeof(T) / 16;
  static constexpr int LPS = ROW_VECS % 8 == 0 ? 8 : 4;           // lanes per slot
  static constexpr int SPW = 32 / LPS;                            // slots per warp step
  static constexpr int NVL = ROW_VECS / LPS;                      // 16-byte vectors per lane
  static constexpr int EPL = NVL * VEC;                           // elements per lane
  static constexpr int STAGE_SLOTS = pow2_floor(SB / (2 * HD * (int)sizeof(T)));
  static constexpr int STAGE_ELEMS = STAGE_SLOTS * HD;
  static constexpr int ITERS = STAGE_SLOTS / SPW;
  static_assert(ROW_VECS % LPS == 0 && NVL >= 1, "lane split");
  static_assert(ITERS >= 1 && STAGE_SLOTS % SPW == 0 && STAGE_SLOTS <= 32, "stage split");
};

// Lane part `lp` owns the 16-byte vectors lp, lp + 8, ... of a slot row.
template <typename T, int HD, int SB>
__device__ __forceinline__ void load_row(const T* row, int lp, float2 (&f)[Shape<T, HD, SB>::EPL / 2]) {
  using SH = Shape<T, HD, SB>;
#pragma unroll
  for (int v = 0; v < SH::NVL; ++v) {
    float t[SH::VEC];
    Elem<T>::unpack(*reinterpret_cast<const uint4*>(row + (v * SH::LPS + lp) * SH::VEC), t);
#pragma unroll
    for (int i = 0; i < SH::VEC / 2; ++i) f[v * SH::VEC / 2 + i] = make_float2(t[2 * i], t[2 * i + 1]);
  }
}

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
  const int64_t r = x - (int64_t)Hkv * pre[lo];  // < Hkv * nst
  if (r <= INT32_MAX) {
    c.h = (int)((uint32_t)r / (uint32_t)c.nst);
    c.st = (int)((uint32_t)r - (uint32_t)c.h * (uint32_t)c.nst);
  } else {
    c.h = (int)(r / c.nst);
    c.st = (int)(r % c.nst);
  }
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


// Online-softmax state of one lane: G query heads, EPL output elements each.
template <typename T, int HD, int G, int SB>
struct SoftState {
  float m[G], l[G];
  float2 acc[G][Shape<T, HD, SB>::EPL / 2];
};

// One pipeline stage of K/V rows for this warp's current piece.  FULL: every
// slot of the stage is inside the sequence and on a fetched page, so no
// masking is needed; otherwise masked slots never touch the sums (NaN-safe).
template <typename T, int HD, int G, int SB, bool FULL>
__device__ __forceinline__ void consume_stage(const T* Ks, const T* Vs, int lane_slot, int lane_part,
                                              const float2 (&q2)[G][Shape<T, HD, SB>::EPL / 2],
                                              float qscale, int valid_slots, uint64_t mask,
                                              int log2P_in_stage, SoftState<T, HD, G, SB>& st) {
  using SH = Shape<T, HD, SB>;
  constexpr int SPW = SH::SPW, ITERS = SH::ITERS, E2 = SH::EPL / 2;
  float sc[G][ITERS];
#pragma unroll
  for (int it = 0; it < ITERS; ++it) {
    const int ls = it * SPW + lane_slot;
    float2 kf[E2];
    load_row<T, HD, SB>(Ks + ls * HD, lane_part, kf);
    bool valid = true;
    if (!FULL) valid = (ls < valid_slots) && ((mask >> (ls >> log2P_in_stage)) & 1ull);
#pragma unroll
    for (int g = 0; g < G; ++g) {
      float2 a = make_float2(0.f, 0.f);
#pragma unroll
      for (int i = 0; i < E2; ++i) a = __ffma2_rn(q2[g][i], kf[i], a);
      float s = group_sum<SH::LPS>(a.x + a.y) * qscale;
      sc[g][it] = valid ? s : -INFINITY;
    }
  }
#pragma unroll
  for (int g = 0; g < G; ++g) {
    float mx = sc[g][0];
#pragma unroll
    for (int it = 1; it < ITERS; ++it) mx = fmaxf(mx, sc[g][it]);
    const float mnew = fmaxf(st.m[g], mx);
    if (FULL || mnew != -INFINITY) {
      const float corr = exp2f(st.m[g] - mnew);  // 0 while m is still -inf
      st.l[g] *= corr;
      const float2 c2 = make_float2(corr, corr);
#pragma unroll
      for (int i = 0; i < E2; ++i) st.acc[g][i] = __fmul2_rn(st.acc[g][i], c2);
      st.m[g] = mnew;
    }
  }
#pragma unroll
  for (int it = 0; it < ITERS; ++it) {
    const int ls = it * SPW + lane_slot;
    float2 vf[E2];
    load_row<T, HD, SB>(Vs + ls * HD, lane_part, vf);
#pragma unroll
    for (int g = 0; g < G; ++g) {
      if (FULL || sc[g][it] != -INFINITY) {
        const float pr = exp2f(sc[g][it] - st.m[g]);
        st.l[g] += pr;
        const float2 p2 = make_float2(pr, pr);
#pragma unroll
        for (int i = 0; i < E2; ++i) st.acc[g][i] = __ffma2_rn(p2, vf[i], st.acc[g][i]);
      }
    }
  }
}

// Write G rows of d outputs (lanes of slot group 0 own vectors lane, lane+8, ...).
template <typename T, int HD, int G, int SB>
__device__ __forceinline__ void write_rows(T* out_rows, int lane_part, const SoftState<T, HD, G, SB>& st) {
  using SH = Shape<T, HD, SB>;
#pragma unroll
  for (int g = 0; g < G; ++g) {
    const float inv = st.l[g] > 0.f ? 1.f / st.l[g] : 0.f;
#pragma unroll
    for (int v = 0; v < SH::NVL; ++v) {
      float o[SH::VEC];
#pragma unroll
      for (int i = 0; i < SH::VEC / 2; ++i) {
        o[2 * i] = st.acc[g][v * SH::VEC / 2 + i].x * inv;
        o[2 * i + 1] = st.acc[g][v * SH::VEC / 2 + i].y * inv;
      }
      store_vec<T>(out_rows + g * HD + (v * SH::LPS + lane_part) * SH::VEC, o);
    }
  }
}

template <typename T, int HD, int G, int SB>
__global__ void __launch_bounds__(kThreads, attn_ctas_per_sm(SB, G)) decode_attn_kernel(const AttnParams p) {
  using SH = Shape<T, HD, SB>;
  constexpr int VEC = SH::VEC, LPS = SH::LPS, E2 = SH::EPL / 2;
  constexpr int STAGE_SLOTS = SH::STAGE_SLOTS, STAGE_ELEMS = SH::STAGE_ELEMS;
  constexpr uint32_t KV_BYTES = STAGE_ELEMS * sizeof(T);
  constexpr uint32_t Q_BYTES = G * HD * sizeof(T);
  constexpr int REC = attn_part_rec(G, HD);                        // floats per partial record
  constexpr int FLAG = G * HD + 2 * G;                             // the record's "published" word
  constexpr int RING_RECS = (int)(kWStages * 2 * KV_BYTES / (REC * sizeof(float)));
  static_assert(RING_RECS >= 1 && (REC * sizeof(float)) % 16 == 0, "partial records");
  // Partial merges take pieces in batches of MB (every load of a batch issued
  // before any is used); both merge paths run the same batches in the same
  // order, so the result does not depend on which path a warp takes.
  constexpr int MB = (HD >= 96 ? 4 : 8) < RING_RECS ? (HD >= 96 ? 4 : 8) : RING_RECS;
  constexpr int ROUND = RING_RECS / MB * MB;  // records per bulk round: whole batches
  constexpr unsigned FULLMASK = 0xFFFFFFFFu;

  extern __shared__ __align__(128) unsigned char smem_raw[];
  T* ring = reinterpret_cast<T*>(smem_raw);                       // [W][S][2][STAGE_ELEMS]
  T* qring = ring + kWarps * kWStages * 2 * STAGE_ELEMS;          // [W][S][G*HD]
  int* pre = reinterpret_cast<int*>(qring + kWarps * kWStages * G * HD);  // [B+1]
  int* lens = pre + p.B + 1;                                      // [B]
  __shared__ uint64_t bars[kWarps][kWStages];
  __shared__ uint64_t qbars[kWarps];  // query of the warp's first piece
  __shared__ uint64_t masks[kWarps][kWStages];
  __shared__ int scan[kThreads];

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int B = p.B, Hkv = p.Hkv;
  const int max_slots = p.max_pages * p.P;

  // Programmatic dependent launch: the next grid on the stream may be
  // scheduled now.  This grid waits for the previous one (finished and
  // flushed) before reading anything it may have written.  With the caller's
  // promise that the previous grid wrote neither the cache, the page table,
  // the lengths nor the workspace (inputs_ready), the wait moves down to just
  // before the query is read, and the first K/V copies overlap its tail.
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  const bool early = p.inputs_ready != 0;
  if (!early) asm volatile("griddepcontrol.wait;" ::: "memory");

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
    // exclusive prefix sum over the block: shuffles within each warp, then
    // the warp totals (one barrier instead of one per doubling step)
    int incl = sum;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int v = __shfl_up_sync(0xFFFFFFFFu, incl, o);
      if (lane >= o) incl += v;
    }
    if (lane == 31) scan[warp] = incl;
    __syncthreads();
    int before = 0, total = 0;
#pragma unroll
    for (int w = 0; w < kWarps; ++w) {
      before += w < warp ? scan[w] : 0;
      total += scan[w];
    }
    int run = before + incl - sum;
    for (int i = i0; i < i1; ++i) {
      pre[i] = run;
      run += lens[i] ? (lens[i] + STAGE_SLOTS - 1) / STAGE_SLOTS : 0;
    }
    if (tid == kThreads - 1) pre[B] = total;
    if (lane == 0) {
      for (int s = 0; s < kWStages; ++s) mbar_init(&bars[warp][s], 1);
      mbar_init(&qbars[warp], 1);
    }
    fence_mbar_init();
    __syncthreads();
  }
  // ---- sequences with an invalid length: zero output rows, report once
  if (blockIdx.x == 0) {
    if (early) asm volatile("griddepcontrol.wait;" ::: "memory");
    for (int b = 0; b < B; ++b) {
      if (lens[b] != 0) continue;
      T* o = reinterpret_cast<T*>(p.out) + (int64_t)b * p.Hq * HD;
      for (int i = tid; i < p.Hq * HD; i += kThreads) o[i] = Elem<T>::from_f(0.f);
      if (tid == 0) report(p.status, WM_ERR_BOUNDS);
    }
  }

  // The NS stages split into nchunks near-equal chunks [c*NS/n, (c+1)*NS/n).
  // Every chunk has at least CH > kWStages stages, so the producer, at most
  // kWStages stages ahead, is never more than one chunk ahead of the consumer.
  // chunk_stages == 0: static split, one chunk per warp and no chunk counter.
  const int64_t NS = (int64_t)Hkv * pre[B];  // stages of all units, concatenated
  const int64_t GW = (int64_t)gridDim.x * kWarps;
  const bool dynamic = p.chunk_stages > 0;
  const int64_t CH = dynamic ? p.chunk_stages : (int64_t)kWStages + 1;
  int64_t nchunks = NS / CH > 1 ? NS / CH : 1;
  if (!dynamic && nchunks > GW) nchunks = GW;
  // (32-bit division whenever the products fit: most launches)
  const bool narrow = (NS + 1) * nchunks < (int64_t)UINT32_MAX;
  auto chunk_begin = [&](int64_t c) -> int64_t {
    return narrow ? (int64_t)((uint32_t)(c * NS) / (uint32_t)nchunks) : c * NS / nchunks;
  };
  auto chunk_end_x = [&](int64_t c) -> int64_t { return chunk_begin(c + 1); };
  auto chunk_of = [&](int64_t x) -> int64_t {
    const int64_t t = (x + 1) * nchunks - 1;
    return narrow ? (int64_t)((uint32_t)t / (uint32_t)NS) : t / NS;
  };
  const int64_t gw = (int64_t)blockIdx.x * kWarps + warp;
  int32_t* grab_ctr = p.counters;
  // Every warp ends with exactly one request that finds no chunk; the request
  // that is last of all resets the counter for the next launch.  A request is
  // issued one chunk ahead and its result read only when the chunk is needed.
  const int64_t total_grabs = (nchunks > GW ? nchunks - GW : 0) + GW;
  int grab_t = 0;  // lane 0: counter value of the outstanding request
  auto grab_issue = [&]() {
    if (dynamic && lane == 0) grab_t = atomicAdd(grab_ctr, 1);
  };
  auto grab_take = [&]() -> int64_t {
    if (!dynamic) return nchunks;  // static split: no further chunk
    if (lane == 0 && grab_t == total_grabs - 1) atomicExch(grab_ctr, 0);
    return GW + __shfl_sync(FULLMASK, grab_t, 0);
  };
  if (gw >= nchunks || NS == 0) {
    if (early) asm volatile("griddepcontrol.wait;" ::: "memory");
    grab_issue();
    grab_take();
    return;  // warp-level from here on: no block barriers below
  }

  T* myring = ring + warp * kWStages * 2 * STAGE_ELEMS;
  T* myq = qring + warp * kWStages * G * HD;
  const uint64_t policy = l2_evict_first_policy();
  const int lane_slot = lane / LPS, lane_part = lane % LPS;

  // ---- page-table window of the producer: lane i holds the page id of
  // logical page win0 + i (cur) and win0 + 32 + i (nxt) of sequence win_b.
  // The first 64 page ids of the unit after the current one are fetched one
  // stage before its first copy (pf_*), and nxt is read only when a stage
  // needs it, so no page-table load sits between two copies of the stream.
  int win_b = -1, win0 = 0, pg_cur = -1, pg_nxt = -1;
  int pf_b = -1, pf_cur = -1, pf_nxt = -1;
  auto load_pg = [&](int b, int lp) -> int {
    return lp < p.max_pages ? __ldg(p.page_table + (int64_t)b * p.max_pages + lp) : -1;
  };
  // page id of logical page lp + (this lane's offset) -- all lanes call it together
  auto page_of = [&](int b, int lp, int lane_off) -> int {
    if (b != win_b || lp < win0 || lp >= win0 + 64) {
      win_b = b;
      win0 = lp;
      if (lp == 0 && b == pf_b) {
        pg_cur = pf_cur;
        pg_nxt = pf_nxt;
      } else {
        pg_cur = load_pg(b, lp + lane);
        pg_nxt = load_pg(b, lp + 32 + lane);
      }
    } else if (lp >= win0 + 32) {
      win0 += 32;
      pg_cur = pg_nxt;
      pg_nxt = load_pg(b, win0 + 32 + lane);
    }
    const int idx = lp + lane_off - win0;  // 0 .. 63
    const int a = __shfl_sync(FULLMASK, pg_cur, idx & 31);
    if (__all_sync(FULLMASK, idx < 32)) return a;
    const int c = __shfl_sync(FULLMASK, pg_nxt, idx & 31);
    return idx < 32 ? a : c;
  };

  // ---- producer: walks its chunks stage by stage, kWStages ahead of the consumer
  int64_t p_chunk = gw;
  int64_t px = chunk_begin(p_chunk), pend = chunk_end_x(p_chunk), pbeg = px;
  int64_t chunk_for_consumer = -1;              // the producer's chunk after a switch
  bool p_done = false;
  Cursor pc = locate(px, pre, B, Hkv);
  uint32_t pseq = 0;                            // stages issued
  auto issue = [&]() {
    const int buf = (int)(pseq % kWStages);
    const bool first = (px == pbeg) || pc.st == 0;
    const int S = lens[pc.b];
    const int s_begin = pc.st * STAGE_SLOTS;
    const T* kb = reinterpret_cast<const T*>(p.k_pool) + (int64_t)pc.h * p.P * HD;
    const T* vb = reinterpret_cast<const T*>(p.v_pool) + (int64_t)pc.h * p.P * HD;
    T* kd = myring + buf * 2 * STAGE_ELEMS;
    T* vd = kd + STAGE_ELEMS;
    uint64_t* bar = &bars[warp][buf];
    // the first piece's query arrives on qbars (issued after the dependency wait)
    const bool with_q = first && pseq > 0;
    const uint32_t qb = with_q ? Q_BYTES : 0u;
    const T* qsrc = reinterpret_cast<const T*>(p.q) + ((int64_t)pc.b * p.Hq + pc.h * G) * HD;
    if (p.P >= STAGE_SLOTS) {
      const int pg = page_of(pc.b, s_begin >> p.log2P, 0);
      if (lane == 0) {
        const bool ok = pg >= 0 && pg < p.num_pages;
        masks[warp][buf] = ok ? 1ull : 0ull;
        if (!ok) report(p.status, WM_ERR_BOUNDS);
        mbar_arrive_expect_tx(bar, (ok ? 2 * KV_BYTES : 0u) + qb);
        if (ok) {
          const int64_t off = (int64_t)pg * p.page_stride + (int64_t)(s_begin & (p.P - 1)) * HD;
          bulk_g2s(kd, kb + off, KV_BYTES, bar, policy);
          bulk_g2s(vd, vb + off, KV_BYTES, bar, policy);
        }
        if (with_q) bulk_g2s(myq + buf * G * HD, qsrc, Q_BYTES, bar, policy);
      }
    } else {
      const int npp = STAGE_SLOTS >> p.log2P;  // pages per stage (<= 32)
      const int lp0 = s_begin >> p.log2P;
      const int lpn = min(npp, ((S - 1) >> p.log2P) - lp0 + 1);
      const int pg = page_of(pc.b, lp0, lane < lpn ? lane : 0);
      const bool ok = lane < lpn && pg >= 0 && pg < p.num_pages;
      const uint32_t mask = __ballot_sync(FULLMASK, ok);
      const uint32_t bytes = (uint32_t)p.P * HD * sizeof(T);
      if (lane == 0) {
        masks[warp][buf] = mask;
        if (__popc(mask) < lpn) report(p.status, WM_ERR_BOUNDS);
        mbar_arrive_expect_tx(bar, 2u * bytes * (uint32_t)__popc(mask) + qb);
        if (with_q) bulk_g2s(myq + buf * G * HD, qsrc, Q_BYTES, bar, policy);
      }
      __syncwarp();
      if (ok) {
        const int64_t off = (int64_t)pg * p.page_stride;
        bulk_g2s(kd + lane * p.P * HD, kb + off, bytes, bar, policy);
        bulk_g2s(vd + lane * p.P * HD, vb + off, bytes, bar, policy);
      }
    }
    ++pseq;
    ++px;
    advance(pc, pre, B, Hkv);
    if (pc.st == 0 && px < pend && pc.b < B && pc.b != pf_b) {  // the next copy opens a unit
      pf_b = pc.b;
      pf_cur = load_pg(pc.b, lane);
      pf_nxt = load_pg(pc.b, 32 + lane);
    }
  };
  // Issue the next stage; when the current chunk is used up, first move on
  // to the chunk requested ahead (the consumer follows through
  // chunk_for_consumer: the switch always happens before the consumer has
  // finished the previous chunk, because that chunk's stages were all issued
  // at least one consumer step earlier).
  auto producer_step = [&]() {
    if (p_done) return;
    if (px == pend) {
      p_chunk = grab_take();
      chunk_for_consumer = p_chunk;
      if (p_chunk >= nchunks) {
        p_done = true;
        return;
      }
      px = chunk_begin(p_chunk);
      pend = chunk_end_x(p_chunk);
      pbeg = px;
      pc = locate(px, pre, B, Hkv);
      grab_issue();
    }
    issue();
  };

  const Cursor pc0 = pc;  // first piece of this warp
  for (int s = 0; s < kWStages && !p_done && px < pend; ++s) issue();
  if (early) asm volatile("griddepcontrol.wait;" ::: "memory");
  if (lane == 0) {
    mbar_arrive_expect_tx(&qbars[warp], Q_BYTES);
    bulk_g2s(myq, reinterpret_cast<const T*>(p.q) + ((int64_t)pc0.b * p.Hq + pc0.h * G) * HD,
             Q_BYTES, &qbars[warp], policy);
  }
  grab_issue();  // the next chunk, requested one ahead

  // ---- consumer
  const int log2P_in_stage = p.P >= STAGE_SLOTS ? 30 : p.log2P;  // stage page index = slot >> this
  const uint64_t all_pages = p.P >= STAGE_SLOTS ? 1ull : ((1ull << (STAGE_SLOTS >> p.log2P)) - 1ull);
  int64_t c_chunk = gw;
  int64_t cx = chunk_begin(c_chunk), cend = chunk_end_x(c_chunk), cbeg = cx;
  Cursor cc = locate(cx, pre, B, Hkv);
  float2 q2[G][E2];
  SoftState<T, HD, G, SB> st;
  T* outp = reinterpret_cast<T*>(p.out);

  // ---- partial records of units that cross chunk boundaries.  The records
  // of a unit whose first piece ends chunk gf: side 1 of chunk gf, then
  // side 0 of chunks gf + 1, gf + 2, ... (consecutive).  Each piece takes its
  // ticket (counter 1 + gf: no other crossing unit starts in chunk gf) before
  // its flag goes up; the piece completing the unit merges, every other one
  // publishes its record and then sets the record's flag (the word after the
  // (m, l) pairs) to this call's epoch, so the merging warp never publishes
  // its own piece.  The merger clears every flag the unit raised and the
  // ticket (a CUDA graph replays a call with the same epoch, possibly over
  // other lengths).
  auto rec_at = [&](int gf, int j) -> float* {
    return p.part + (j == 0 ? (int64_t)(p.max_chunks + gf) : (int64_t)(gf + j)) * REC;
  };
  auto flag_at = [&](float* r) -> int* { return reinterpret_cast<int*>(r + FLAG); };
  // this warp's merged piece (registers) as a record
  auto store_record = [&](float* po) {
    float* pm = po + G * HD;
    if (lane_slot == 0) {
#pragma unroll
      for (int g = 0; g < G; ++g)
#pragma unroll
        for (int v = 0; v < SH::NVL; ++v)
#pragma unroll
          for (int i = 0; i < VEC / 2; ++i)
            reinterpret_cast<float2*>(po + g * HD + (v * LPS + lane_part) * VEC)[i] =
                st.acc[g][v * VEC / 2 + i];
    }
    if (lane == 0) {
#pragma unroll
      for (int g = 0; g < G; ++g) {
        pm[2 * g] = st.m[g];
        pm[2 * g + 1] = st.l[g];
      }
    }
  };
  // every other piece has its ticket and at most its stores left: wait
  // (bounded) for their flags; false (and WM_ERR_TIMEOUT) if one never came
  auto wait_flags = [&](int gf, int np, int j_own) -> bool {
    bool ready = false;
    const uint64_t t0 = globaltimer_ns();
    for (uint32_t it = 0;; ++it) {
      bool mine = true;
      for (int j = lane; j < np; j += 32)
        if (j != j_own) mine = mine && (ld_acquire_gpu(flag_at(rec_at(gf, j))) == p.epoch);
      ready = __all_sync(FULLMASK, mine);
      if (ready || ((it & 63u) == 63u && globaltimer_ns() - t0 > kWaitLimitNs)) break;
    }
    if (!ready && lane == 0) report(p.status, WM_ERR_TIMEOUT);
    __syncwarp();  // every lane's acquire precedes the whole warp's reads
    return ready;
  };
  // merge all np records of the unit from global memory into its output rows
  auto merge_global = [&](int gf, int np, int rowbase) {
    for (int g = 0; g < G; ++g) {
      float M = -INFINITY, Ls = 0.f;
      float o[HD / 32];
#pragma unroll
      for (int i = 0; i < HD / 32; ++i) o[i] = 0.f;
      for (int r0 = 0; r0 < np; r0 += MB) {
        float mq[MB], lq[MB], ov[MB][HD / 32];
#pragma unroll
        for (int jb = 0; jb < MB; ++jb) {
          const int j = r0 + jb;
          const bool in = j < np;
          const float* rj = rec_at(gf, j);
          mq[jb] = in ? __ldcg(rj + G * HD + 2 * g) : -INFINITY;
          lq[jb] = in ? __ldcg(rj + G * HD + 2 * g + 1) : 0.f;
#pragma unroll
          for (int i = 0; i < HD / 32; ++i)
            ov[jb][i] = in ? __ldcg(rj + g * HD + lane + 32 * i) : 0.f;
        }
        float Mn = M;
#pragma unroll
        for (int jb = 0; jb < MB; ++jb) Mn = fmaxf(Mn, mq[jb]);
        if (Mn == -INFINITY) continue;
        const float rescale = exp2f(M - Mn);  // 0 on the first batch
        Ls *= rescale;
#pragma unroll
        for (int i = 0; i < HD / 32; ++i) o[i] *= rescale;
#pragma unroll
        for (int jb = 0; jb < MB; ++jb) {
          if (mq[jb] == -INFINITY) continue;
          const float w = exp2f(mq[jb] - Mn);
          Ls = fmaf(w, lq[jb], Ls);
#pragma unroll
          for (int i = 0; i < HD / 32; ++i) o[i] = fmaf(w, ov[jb][i], o[i]);
        }
        M = Mn;
      }
      const float inv = Ls > 0.f ? 1.f / Ls : 0.f;
#pragma unroll
      for (int i = 0; i < HD / 32; ++i)
        outp[((int64_t)rowbase + g) * HD + lane + 32 * i] = Elem<T>::from_f(o[i] * inv);
    }
  };
  // ready for the next launch: flags down, ticket counter zero
  auto release_unit = [&](int gf, int np, int j_own) {
    for (int j = lane; j < np; j += 32)
      if (j != j_own) *reinterpret_cast<volatile int*>(flag_at(rec_at(gf, j))) = 0;
    if (lane == 0) p.counters[1 + gf] = 0;
  };
  int pend_np = 0, pend_tk = 0, pend_g = 0, pend_row = 0;  // a piece awaiting its flag
  for (uint32_t seq = 0;; ++seq) {
    const int buf = (int)(seq % kWStages);
    bool ok = mbar_wait(&bars[warp][buf], (seq / kWStages) & 1);
    if (seq == 0) ok = mbar_wait(&qbars[warp], 0) && ok;  // the first piece's query
    if (__any_sync(FULLMASK, !ok)) {
      // a copy never landed: report, drain what is in flight (bounded) and stop
      if (lane == 0) {
        report(p.status, WM_ERR_TIMEOUT);
        for (uint32_t y = seq; y < pseq; ++y) mbar_wait(&bars[warp][y % kWStages], (y / kWStages) & 1);
        if (seq == 0) mbar_wait(&qbars[warp], 0);
      }
      __syncwarp();
      return;
    }
    if (cx == cbeg || cc.st == 0) {
      const T* qs = myq + buf * G * HD;
#pragma unroll
      for (int g = 0; g < G; ++g) {
        load_row<T, HD, SB>(qs + g * HD, lane_part, q2[g]);
        st.m[g] = -INFINITY;
        st.l[g] = 0.f;
#pragma unroll
        for (int i = 0; i < E2; ++i) st.acc[g][i] = make_float2(0.f, 0.f);
      }
    }
    // A stage that ends a piece of a unit crossing chunk boundaries takes the
    // piece's ticket before its math, so the atomic's round trip overlaps it.
    const bool chunk_end = (cx == cend - 1);
    const bool piece_end = chunk_end || cc.st == cc.nst - 1;
    int64_t g_first = 0, g_last = 0;
    int tk = 0;
    if (piece_end) {
      const int64_t U = (int64_t)Hkv * pre[cc.b] + (int64_t)cc.h * cc.nst;
      g_first = chunk_of(U);
      g_last = chunk_of(U + cc.nst - 1);
      if (g_first != g_last && lane == 0) tk = atomicAdd(p.counters + 1 + g_first, 1);
    }
    const int valid_slots = lens[cc.b] - cc.st * STAGE_SLOTS;
    const uint64_t mask = masks[warp][buf];
    const T* Ks = myring + buf * 2 * STAGE_ELEMS;
    const T* Vs = Ks + STAGE_ELEMS;
    if (valid_slots >= STAGE_SLOTS && mask == all_pages)
      consume_stage<T, HD, G, SB, true>(Ks, Vs, lane_slot, lane_part, q2, p.qscale, valid_slots,
                                        mask, log2P_in_stage, st);
    else
      consume_stage<T, HD, G, SB, false>(Ks, Vs, lane_slot, lane_part, q2, p.qscale, valid_slots,
                                         mask, log2P_in_stage, st);
    __syncwarp();  // every lane is done with this ring slot
    producer_step();

    if (pend_np > 0 && chunk_end) {
      // the piece that ended in the middle of this chunk: its record and
      // ticket went out then; its flag goes up now, where (in a static split)
      // no copy of this warp is in flight any more -- a release issued
      // while bulk copies are in flight waited for them
      const bool last = __shfl_sync(FULLMASK, pend_tk, 0) == pend_np - 1;
      if (!last) {
        __syncwarp();
        if (lane == 0) st_release_gpu(flag_at(rec_at(pend_g, pend_np - 1)), p.epoch);
      } else if (wait_flags(pend_g, pend_np, pend_np - 1)) {
        merge_global(pend_g, pend_np, pend_row);
        release_unit(pend_g, pend_np, pend_np - 1);
      }
      pend_np = 0;
    }
    if (piece_end) {
      // merge the SPW lane groups of the warp
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
        st.m[g] = M;
        st.l[g] = Ls;
      }
      const int rowbase = cc.b * p.Hq + cc.h * G;
      if (g_first == g_last) {
        if (lane_slot == 0) write_rows<T, HD, G, SB>(outp + (int64_t)rowbase * HD, lane_part, st);
      } else {
        const int gf = (int)g_first;
        const int np = (int)(g_last - g_first + 1);
        const int j_own = (int)(c_chunk - g_first);  // this piece's record in the merge
        if (!chunk_end) {
          // The unit ends here and the chunk goes on (so this is the unit's
          // last piece, j_own = np - 1; a chunk holds at most one such
          // piece, its first): store the record now, read the ticket and
          // raise the flag (or merge) at the chunk's end instead of stalling
          // the stream in its middle.
          store_record(rec_at(gf, j_own));
          pend_tk = tk;
          pend_np = np;
          pend_g = gf;
          pend_row = rowbase;
        } else {
          const bool last = __shfl_sync(FULLMASK, tk, 0) == np - 1;
          if (!last) {
            store_record(rec_at(gf, j_own));
            __syncwarp();
            if (lane == 0) st_release_gpu(flag_at(rec_at(gf, j_own)), p.epoch);
          } else if (wait_flags(gf, np, j_own)) {
            if (p_done && seq + 1 == pseq) {
              // no stage in flight: the ring takes ROUND records per round
              float* rs = reinterpret_cast<float*>(myring);
              float M[G], Ls[G], o[G][HD / 32];
#pragma unroll
              for (int g = 0; g < G; ++g) {
                M[g] = -INFINITY;
                Ls[g] = 0.f;
#pragma unroll
                for (int i = 0; i < HD / 32; ++i) o[g][i] = 0.f;
              }
              fence_proxy_async_global();
              fence_proxy_async_shared();
              bool landed = true;
              for (int r0 = 0; r0 < np; r0 += ROUND) {
                const int n = min(ROUND, np - r0);
                constexpr uint32_t RB = REC * sizeof(float);
                if (lane == 0) {
                  mbar_arrive_expect_tx(&qbars[warp], (uint32_t)n * RB);
                  if (r0 == 0) {
                    bulk_g2s(rs, rec_at(gf, 0), RB, &qbars[warp], policy);
                    if (n > 1) bulk_g2s(rs + REC, rec_at(gf, 1), (uint32_t)(n - 1) * RB, &qbars[warp], policy);
                  } else {
                    bulk_g2s(rs, rec_at(gf, r0), (uint32_t)n * RB, &qbars[warp], policy);
                  }
                }
                // qbars completed phase 0 with the first query; round r is phase r + 1
                const uint32_t parity = (uint32_t)(r0 / ROUND + 1) & 1u;
                landed = mbar_wait(&qbars[warp], parity);
                if (__any_sync(FULLMASK, !landed)) {
                  if (lane == 0) {
                    report(p.status, WM_ERR_TIMEOUT);
                    mbar_wait(&qbars[warp], parity);
                  }
                  landed = false;
                  break;
                }
                if (j_own >= r0 && j_own < r0 + n) {
                  // this warp's own piece was never published: take it from registers
                  float* ro = rs + (j_own - r0) * REC;
                  if (lane_slot == 0) {
#pragma unroll
                    for (int g = 0; g < G; ++g)
#pragma unroll
                      for (int v = 0; v < SH::NVL; ++v)
#pragma unroll
                        for (int i = 0; i < VEC / 2; ++i)
                          reinterpret_cast<float2*>(ro + g * HD + (v * LPS + lane_part) * VEC)[i] =
                              st.acc[g][v * VEC / 2 + i];
                  }
                  if (lane == 0) {
#pragma unroll
                    for (int g = 0; g < G; ++g) {
                      ro[G * HD + 2 * g] = st.m[g];
                      ro[G * HD + 2 * g + 1] = st.l[g];
                    }
                  }
                  __syncwarp();
                }
#pragma unroll
                for (int g = 0; g < G; ++g) {
                  for (int b0 = 0; b0 < n; b0 += MB) {
                    float mq[MB], lq[MB];
#pragma unroll
                    for (int jb = 0; jb < MB; ++jb) {
                      const bool in = b0 + jb < n;
                      mq[jb] = in ? rs[(b0 + jb) * REC + G * HD + 2 * g] : -INFINITY;
                      lq[jb] = in ? rs[(b0 + jb) * REC + G * HD + 2 * g + 1] : 0.f;
                    }
                    float Mn = M[g];
#pragma unroll
                    for (int jb = 0; jb < MB; ++jb) Mn = fmaxf(Mn, mq[jb]);
                    if (Mn == -INFINITY) continue;
                    const float rescale = exp2f(M[g] - Mn);  // 0 on the first batch
                    Ls[g] *= rescale;
#pragma unroll
                    for (int i = 0; i < HD / 32; ++i) o[g][i] *= rescale;
#pragma unroll
                    for (int jb = 0; jb < MB; ++jb) {
                      if (mq[jb] == -INFINITY) continue;
                      const float w = exp2f(mq[jb] - Mn);
                      Ls[g] = fmaf(w, lq[jb], Ls[g]);
                      const float* rj = rs + (b0 + jb) * REC + g * HD + lane;
#pragma unroll
                      for (int i = 0; i < HD / 32; ++i) o[g][i] = fmaf(w, rj[32 * i], o[g][i]);
                    }
                    M[g] = Mn;
                  }
                }
                __syncwarp();  // every lane is done with the ring before the next round
              }
              if (landed) {
#pragma unroll
                for (int g = 0; g < G; ++g) {
                  const float inv = Ls[g] > 0.f ? 1.f / Ls[g] : 0.f;
#pragma unroll
                  for (int i = 0; i < HD / 32; ++i)
                    outp[((int64_t)rowbase + g) * HD + lane + 32 * i] = Elem<T>::from_f(o[g][i] * inv);
                }
              }
            } else {
              // stages in flight: the same batches, straight from global
              // memory (this warp's own record first, for its other lanes)
              store_record(rec_at(gf, j_own));
              __threadfence();
              __syncwarp();
              merge_global(gf, np, rowbase);
            }
            release_unit(gf, np, j_own);
          }
        }
      }
    }
    if (chunk_end) {  // continue with the chunk the producer moved on to
      if (chunk_for_consumer < 0) producer_step();  // a chunk shorter than the ring
      c_chunk = chunk_for_consumer;
      if (c_chunk < 0 || c_chunk >= nchunks) break;
      cx = chunk_begin(c_chunk);
      cend = chunk_end_x(c_chunk);
      cbeg = cx;
      cc = locate(cx, pre, B, Hkv);
    } else {
      ++cx;
      advance(cc, pre, B, Hkv);
    }
  }
}

template <typename T, int HD, int G, int SB>
inline cudaError_t launch_t(const AttnParams& p, int grid, size_t smem, cudaStream_t stream) {
  static size_t smem_set[kSmemOptDevices] = {};
  auto kern = decode_attn_kernel<T, HD, G, SB>;
  if (cudaError_t e = opt_in_smem(kern, smem, smem_set); e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, p);
}

template <typename T, int HD, int SB>
inline cudaError_t launch_g(const AttnParams& p, int G, int grid, size_t smem, cudaStream_t s) {
  switch (G) {
    case 1: return launch_t<T, HD, 1, SB>(p, grid, smem, s);
    case 2: return launch_t<T, HD, 2, SB>(p, grid, smem, s);
    case 4: return launch_t<T, HD, 4, SB>(p, grid, smem, s);
    case 8: return launch_t<T, HD, 8, SB>(p, grid, smem, s);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace attn_detail

// Per-dtype dispatch (one translation unit each, compiled in parallel).
cudaError_t launch_attn_bf16(const AttnParams& p, int stage_bytes, int d, int G, int grid,
                             size_t smem, cudaStream_t s);
cudaError_t launch_attn_f32(const AttnParams& p, int stage_bytes, int d, int G, int grid,
                            size_t smem, cudaStream_t s);

}  // namespace wm
