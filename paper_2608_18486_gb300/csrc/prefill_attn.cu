// Causal channel attention for prefill and for the token-parallel passes
// (Sec. 3.1 Step 3 "standard causal SDPA", with the dummy offset of Sec. 3.2
// and the Jacobi / cyclic Gauss-Seidel schedules of Sec. 3.3).  Query row r
// of sequence b is the query of the token at position pos[b][r]; it reads
// slots 0 .. pos of its layer's channel: the dummy and the tokens before it.
//
// Design (GB300).  A prefill pass is a dense contraction on both sides of the
// softmax, so it runs on the tcgen05 tensor cores (bf16 operands, fp32
// accumulation in TMEM), warp-specialised in the manner of flash attention on
// this architecture.  One CTA (10 warps, one per SM) owns two 128-row query
// tiles of one query head and walks the 128-slot KV tiles of the sequence's
// channel up to each tile's largest position:
//    With grouped-query attention (an even number G of query heads per kv
//    head) the two tiles are the same 128 rows of two query heads that share
//    a kv head: equal causal ranges, and one K/V stream serves both.
//    Otherwise they are two consecutive 128-row tiles of one head.
//  * warp 8 (TMA): the two Q tiles once, then K and V of every KV tile
//    through separate rings (128-byte swizzle, 64-column boxes; paged: one
//    box per page, or per 128 slots of a longer page);
//  * warp 9 (MMA): S_i = Q_i K^T into TMEM, and O_i += P_i V with P_i read
//    from TMEM and V as an MN-major operand straight from its [slot][d] tile;
//    issue order PV_0(j), S_0(j+1), PV_1(j), S_1(j+1) keeps one tile's
//    matrix products running while the other tile's softmax works;
//  * warps 0-3 and 4-7 (softmax of tile 0 / 1): one thread per query row
//    reads its S row from TMEM, applies the causal mask slot <= pos (on
//    tiles the diagonal crosses), and writes the bf16 probabilities back over
//    the S columns it has read, where P V takes them as its A operand.  The
//    running max is raised only when it grows by more than 2^8: only then is
//    the row of O in TMEM rescaled; in between the probabilities stay below
//    2^8, and the final O / l is exact either way.
// Slots beyond the CTA's largest position may hold anything (unwritten
// cache); their V rows are zeroed in shared memory before P V, and masked
// scores are replaced, never multiplied, so no NaN there reaches the output.
#include <math.h>

#include "internal.h"
#include "tc.cuh"

namespace wm {
namespace {

constexpr int kPM = 128;                    // query rows per tile (MMA M)
constexpr int kPN = 128;                    // slots per KV tile
constexpr int kQT = 2;                      // query tiles per CTA
constexpr int kSoftWarps = 4 * kQT;         // one 4-warp group per query tile
constexpr int kLoadWarp = kSoftWarps;       // TMA producer
constexpr int kMmaWarp = kSoftWarps + 1;    // MMA issuer
constexpr int kPThreads = (kSoftWarps + 2) * 32;
constexpr uint32_t kBlock = 128u * 128u;    // one 64-column block of a 128-row tile
constexpr uint32_t kTmemCols = 512;         // S_i at 128 i (P_i over its first 64), O_i at 256 + 128 i
constexpr float kStaleMax = 8.f;            // log2 headroom before O is rescaled

template <int HD>
struct PShape {
  static constexpr int CB = (HD + 63) / 64;          // 64-column blocks of a head row
  // Ring depths: the next K tile is waited for first (S of the next KV tile
  // is issued behind P V of this one), so K gets the deeper ring.
  static constexpr int NSK = HD <= 64 ? 4 : 3;
  static constexpr int NSV = HD <= 64 ? 4 : 2;
  static constexpr uint32_t Q_BYTES = CB * kBlock;   // one Q tile
  static constexpr uint32_t KV_BYTES = CB * kBlock;  // one K or V tile
  static constexpr uint32_t SMEM = kQT * Q_BYTES + (NSK + NSV) * KV_BYTES + 1024;  // + alignment
  static_assert(SMEM <= 227 * 1024, "shared memory");
};

struct PrefillParams {
  const int32_t* pos;         // [B][Tq]
  const int32_t* page_table;  // [B][max_pages]
  void* out;                  // [B][Tq][Hq][d] bf16
  int32_t* status;
  int32_t B, Tq, Hq, G, Hkv, chan, num_pages, max_pages, P, log2P;
  int32_t pair;               // 1: the two tiles are query heads 2y, 2y+1 over the same rows
  float qscale;               // log2(e) / sqrt(d)
};

__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

template <int HD>
__global__ void __launch_bounds__(kPThreads, 1)
    prefill_attn_kernel(const __grid_constant__ CUtensorMap tmQ,
                        const __grid_constant__ CUtensorMap tmK,
                        const __grid_constant__ CUtensorMap tmV, const PrefillParams p) {
  using SH = PShape<HD>;
  constexpr int CB = SH::CB, NSK = SH::NSK, NSV = SH::NSV;
  extern __shared__ uint8_t smem_dyn[];
  __shared__ uint64_t qbar, kfull[NSK], kempty[NSK], vfull[NSV], vempty[NSV];
  __shared__ uint64_t sfull[kQT], pfull[kQT], odone[kQT];
  __shared__ uint32_t tmem_base;
  __shared__ int wmax[kSoftWarps];

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  // query tile i: rows rb[i] .. rb[i] + 127 of query head hh[i]
  const int b = blockIdx.z;
  const int rows_cta = p.pair ? kPM : kQT * kPM;
  const int nblk = (p.Tq + rows_cta - 1) / rows_cta;
  const int r0 = (nblk - 1 - (int)blockIdx.x) * rows_cta;  // later rows (more work) first
  int rb[kQT], hh[kQT];
#pragma unroll
  for (int i = 0; i < kQT; ++i) {
    rb[i] = p.pair ? r0 : r0 + i * kPM;
    hh[i] = p.pair ? kQT * (int)blockIdx.y + i : (int)blockIdx.y;
  }
  const int hkv = hh[0] / p.G;  // the same kv head for both tiles
  uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_dyn) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* Qs = base;                         // [kQT] Q tiles
  uint8_t* Ks = Qs + kQT * SH::Q_BYTES;       // [NSK] K tiles
  uint8_t* Vs = Ks + NSK * SH::KV_BYTES;      // [NSV] V tiles

  if (tid == 0) {
    mbar_init(&qbar, 1);
    for (int s = 0; s < NSK; ++s) {
      mbar_init(&kfull[s], 1);
      mbar_init(&kempty[s], 1);
    }
    for (int s = 0; s < NSV; ++s) {
      mbar_init(&vfull[s], 1);
      mbar_init(&vempty[s], 1);
    }
    for (int i = 0; i < kQT; ++i) {
      mbar_init(&sfull[i], 1);
      mbar_init(&pfull[i], kPM);
      mbar_init(&odone[i], 1);
    }
    fence_mbar_init();
    tc::prefetch_tensormap(&tmQ);
    tc::prefetch_tensormap(&tmK);
    tc::prefetch_tensormap(&tmV);
  }
  if (warp == 0) {
    tc::tmem_alloc(&tmem_base, kTmemCols);
    tc::tmem_relinquish();
  }
  // programmatic dependent launch: positions, table, queries and cache may
  // come from the previous grid
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  asm volatile("griddepcontrol.wait;" ::: "memory");

  // ---- positions of the softmax threads' rows; the largest of each tile
  const int max_slots = p.max_pages * p.P;
  int mypos = -1;  // -1: row absent or invalid, fully masked
  const int my_tile = warp < kSoftWarps ? warp >> 2 : 0;
  const int r = rb[my_tile] + (tid - my_tile * kPM);
  if (warp < kSoftWarps && r < p.Tq) {
    const int v = p.pos[(int64_t)b * p.Tq + r];
    if (v >= 0 && v < max_slots) mypos = v;
    else report(p.status, WM_ERR_BOUNDS);
  }
  if (warp < kSoftWarps) {
    int mx = mypos;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      mx = max(mx, __shfl_xor_sync(0xFFFFFFFFu, mx, o));
    }
    if (lane == 0) {
      wmax[warp] = mx;
    }
  }
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = tmem_base;
  int ntile[kQT], tmaxpos = -1;
#pragma unroll
  for (int i = 0; i < kQT; ++i) {
    const int mx = max(max(wmax[4 * i], wmax[4 * i + 1]), max(wmax[4 * i + 2], wmax[4 * i + 3]));
    ntile[i] = mx >= 0 ? mx / kPN + 1 : 0;  // KV tiles of query tile i
    tmaxpos = max(tmaxpos, mx);
  }
  const int nmax = tmaxpos >= 0 ? tmaxpos / kPN + 1 : 0;

  if (warp == kLoadWarp) {
    // ================================================================ TMA
    // Lane t owns box t of every KV tile (one box per page, or one per 128
    // slots of a longer page): its page id for the next tile is fetched
    // while the current tile is issued, so no page-table load sits on the
    // issue path.  Lane 0 posts the expected bytes before the lanes copy.
    if (nmax > 0) {
      bool ok = true;
      if (lane == 0) {
        mbar_arrive_expect_tx(&qbar, kQT * SH::Q_BYTES);
        for (int i = 0; i < kQT; ++i)
#pragma unroll
          for (int cb = 0; cb < CB; ++cb)
            tc::tma_load_2d(Qs + i * SH::Q_BYTES + cb * kBlock, &tmQ, hh[i] * HD + cb * 64,
                            b * p.Tq + rb[i], &qbar);
      }
      const int boxes = p.P >= kPN ? 1 : kPN >> p.log2P;  // <= 16 for pages of >= 8 slots
      const int brows = p.P >= kPN ? kPN : p.P;
      // tensor-map row of this lane's box of KV tile j (-brows: read zeros)
      auto box_row = [&](int j) -> int {
        const int s = j * kPN + lane * brows;  // first slot of the box
        const int lp = s >> p.log2P;           // logical page
        int row = -brows;
        if (lane < boxes && s <= tmaxpos && lp < p.max_pages) {
          const int pg = p.page_table[(int64_t)b * p.max_pages + lp];
          if (pg >= 0 && pg < p.num_pages)
            row = (int)((((int64_t)p.chan * p.num_pages + pg) * p.Hkv + hkv) * p.P + (s & (p.P - 1)));
          else
            report(p.status, WM_ERR_BOUNDS);
        }
        return row;
      };
      auto load_tile = [&](const CUtensorMap* tm, uint8_t* dst, int row, uint64_t* bar) {
        if (lane == 0) mbar_arrive_expect_tx(bar, SH::KV_BYTES);
        __syncwarp();
        if (lane < boxes)
#pragma unroll
          for (int cb = 0; cb < CB; ++cb)
            tc::tma_load_2d(dst + cb * kBlock + lane * brows * 128, tm, cb * 64, row, bar);
      };
      int row_next = box_row(0);
      for (int j = 0; j < nmax && ok; ++j) {
        const int row = row_next;
        if (j + 1 < nmax) row_next = box_row(j + 1);
        const int sk = j % NSK, sv = j % NSV;
        if (j >= NSK) ok = __all_sync(0xFFFFFFFFu, mbar_wait(&kempty[sk], (j / NSK - 1) & 1));
        if (!ok) break;
        load_tile(&tmK, Ks + sk * SH::KV_BYTES, row, &kfull[sk]);
        if (j >= NSV) ok = __all_sync(0xFFFFFFFFu, mbar_wait(&vempty[sv], (j / NSV - 1) & 1));
        if (!ok) break;
        load_tile(&tmV, Vs + sv * SH::KV_BYTES, row, &vfull[sv]);
      }
      if (!ok && lane == 0) report(p.status, WM_ERR_TIMEOUT);
    }
  } else if (warp == kMmaWarp) {
    // ================================================================ MMA
    // every lane runs the schedule (all wait, all zero the last V tile's
    // unwritten rows, wait outcomes made warp-uniform); lane 0 issues
    const uint32_t idesc_s = tc::idesc_bf16_f32(kPM, kPN);
    const uint32_t idesc_o = tc::idesc_bf16_f32(kPM, HD) | tc::kIdescBMajorMN;
    auto wait_all = [&](uint64_t* bar, uint32_t parity) {
      return __all_sync(0xFFFFFFFFu, mbar_wait(bar, parity));
    };
    bool ok = nmax == 0 || wait_all(&qbar, 0);
    auto issue_s = [&](int i, int j) {  // S_i = Q_i K_j^T
      if (lane == 0) {
        const uint32_t q0 = smem_u32(Qs + i * SH::Q_BYTES);
        const uint32_t k0 = smem_u32(Ks + (j % NSK) * SH::KV_BYTES);
#pragma unroll
        for (int kk = 0; kk < HD / 16; ++kk) {
          const uint32_t off = (kk >> 2) * kBlock + (kk & 3) * 32;
          tc::mma_bf16(tmem + 128 * i, tc::sdesc_kmajor_sw128(q0 + off),
                       tc::sdesc_kmajor_sw128(k0 + off), idesc_s, kk > 0);
        }
        tc::mma_commit(&sfull[i]);
      }
    };
    auto issue_pv = [&](int i, int j) {  // O_i += P_i V_j
      if (lane == 0) {
        const uint32_t v0 = smem_u32(Vs + (j % NSV) * SH::KV_BYTES);
#pragma unroll
        for (int kk = 0; kk < kPN / 16; ++kk)
          tc::mma_bf16_ts(tmem + 256 + 128 * i, tmem + 128 * i + 8 * kk,
                          tc::sdesc_mnmajor_sw128(v0 + kk * 16 * 128, kBlock, 1024), idesc_o,
                          (j | kk) != 0);
        tc::mma_commit(&odone[i]);
      }
    };
    if (ok && nmax > 0) {
      ok = wait_all(&kfull[0], 0);
      tc::fence_after_sync();
      if (ok) {
        for (int i = 0; i < kQT; ++i)
          if (ntile[i] > 0) issue_s(i, 0);
        if (lane == 0) tc::mma_commit(&kempty[0]);
      }
    }
    for (int j = 0; j < nmax && ok; ++j) {
      const int st = j % NSV;
      ok = wait_all(&vfull[st], (j / NSV) & 1);
      if (!ok) break;
      const int s0 = j * kPN;
      if (j == nmax - 1 && s0 + kPN - 1 > tmaxpos) {
        // slots past the largest position may be unwritten: zero their V rows
        uint8_t* vt = Vs + st * SH::KV_BYTES;
        for (int row = tmaxpos - s0 + 1 + lane; row < kPN; row += 32)
#pragma unroll
          for (int cb = 0; cb < CB; ++cb)
#pragma unroll
            for (int u = 0; u < 8; ++u)
              *reinterpret_cast<uint4*>(vt + cb * kBlock + row * 128 + u * 16) =
                  make_uint4(0, 0, 0, 0);
        fence_proxy_async_shared();
        __syncwarp();
      }
      const bool more = j + 1 < nmax;
      if (more) {
        ok = wait_all(&kfull[(j + 1) % NSK], ((j + 1) / NSK) & 1);
        if (!ok) break;
      }
      for (int i = 0; i < kQT && ok; ++i) {
        if (j >= ntile[i]) continue;
        ok = wait_all(&pfull[i], j & 1);
        if (!ok) break;
        tc::fence_after_sync();
        issue_pv(i, j);
        if (j + 1 < ntile[i]) issue_s(i, j + 1);
      }
      if (lane == 0) {
        tc::mma_commit(&vempty[st]);
        if (more) tc::mma_commit(&kempty[(j + 1) % NSK]);
      }
      __syncwarp();
    }
    if (!ok && lane == 0) report(p.status, WM_ERR_TIMEOUT);
  } else {
    // ================================================================ softmax
    const int i = warp >> 2;  // query tile
    const int n = ntile[i];
    const uint32_t lane_base = tmem + ((uint32_t)((warp & 3) * 32) << 16);
    const uint32_t scol = 128 * i, ocol = 256 + 128 * i;
    float m = -INFINITY, l = 0.f;  // max used for P (log2 units) and running sum
    bool ok = true;
    // tcgen05.ld / st are warp-collective: every lane of the warp issues each
    // one, and the wait outcomes are made warp-uniform before any branch
    for (int j = 0; j < n && ok; ++j) {
      ok = __all_sync(0xFFFFFFFFu, mbar_wait(&sfull[i], j & 1));
      if (!ok) break;
      tc::fence_after_sync();
      const int s0 = j * kPN;
      // Visible slots of this row in the tile: e < vis (all 128 unless the
      // diagonal crosses the tile).  The masked path only runs there.
      const int vis = min(max(mypos - s0 + 1, 0), kPN);
      // the whole S row in one TMEM read
      uint32_t v[kPN / 32][32];
#pragma unroll
      for (int c = 0; c < kPN / 32; ++c) tc::tmem_ld32(lane_base + scol + 32 * c, v[c]);
      tc::tmem_ld_wait();
      float mx = -INFINITY;
      if (vis == kPN) {
#pragma unroll
        for (int c = 0; c < kPN / 32; ++c)
#pragma unroll
          for (int e = 0; e < 32; ++e) mx = fmaxf(mx, __uint_as_float(v[c][e]));
      } else {
#pragma unroll
        for (int c = 0; c < kPN / 32; ++c)
#pragma unroll
          for (int e = 0; e < 32; ++e)
            if (32 * c + e < vis) mx = fmaxf(mx, __uint_as_float(v[c][e]));
      }
      const float mt = mx * p.qscale;  // qscale > 0: the max commutes with the scale
      float scale = 1.f;
      const bool raise = (m == -INFINITY) ? (mt != -INFINITY) : (mt > m + kStaleMax);
      if (raise) {
        scale = (m == -INFINITY) ? 0.f : ex2(m - mt);
        m = mt;
      }
      // p = 2^(s * qscale - m) in pairs; masked slots (and rows with nothing
      // visible yet) give 0
      const float2 qs2 = make_float2(p.qscale, p.qscale), nm2 = make_float2(-m, -m);
      const bool live = m != -INFINITY;
      float2 sum2 = make_float2(0.f, 0.f);
#pragma unroll
      for (int c = 0; c < kPN / 32; ++c) {
        uint32_t w[16];
        const int lim = live ? vis - 32 * c : 0;
        if (lim >= 32) {
#pragma unroll
          for (int e = 0; e < 32; e += 2) {
            const float2 x = __ffma2_rn(
                make_float2(__uint_as_float(v[c][e]), __uint_as_float(v[c][e + 1])), qs2, nm2);
            const float2 pr = make_float2(ex2(x.x), ex2(x.y));
            sum2 = __fadd2_rn(sum2, pr);
            const __nv_bfloat162 h = __floats2bfloat162_rn(pr.x, pr.y);
            w[e / 2] = *reinterpret_cast<const uint32_t*>(&h);
          }
        } else {
#pragma unroll
          for (int e = 0; e < 32; e += 2) {
            const float2 x = __ffma2_rn(
                make_float2(__uint_as_float(v[c][e]), __uint_as_float(v[c][e + 1])), qs2, nm2);
            const float2 pr = make_float2(e < lim ? ex2(x.x) : 0.f, e + 1 < lim ? ex2(x.y) : 0.f);
            sum2 = __fadd2_rn(sum2, pr);
            const __nv_bfloat162 h = __floats2bfloat162_rn(pr.x, pr.y);
            w[e / 2] = *reinterpret_cast<const uint32_t*>(&h);
          }
        }
        // P over the S columns (all read above): packed pairs, columns 16c .. 16c+15
        tc::tmem_st16(lane_base + scol + 16 * c, w);
      }
      const float sum = sum2.x + sum2.y;
      l = l * scale + sum;
      if (__any_sync(0xFFFFFFFFu, raise && j > 0)) {
        // a row's max grew past the headroom: rescale O (every lane of the
        // warp takes part; rows that did not raise their max scale by 1)
        // once P V of the previous tile has landed in it
        if (!(raise && j > 0)) scale = 1.f;
        ok = __all_sync(0xFFFFFFFFu, mbar_wait(&odone[i], (j - 1) & 1));
        if (!ok) break;
        tc::fence_after_sync();
#pragma unroll
        for (int c = 0; c < HD / 32; ++c) {
          uint32_t v[32];
          tc::tmem_ld32(lane_base + ocol + 32 * c, v);
          tc::tmem_ld_wait();
          uint32_t w0[16], w1[16];
#pragma unroll
          for (int e = 0; e < 16; ++e) {
            w0[e] = __float_as_uint(__uint_as_float(v[e]) * scale);
            w1[e] = __float_as_uint(__uint_as_float(v[16 + e]) * scale);
          }
          tc::tmem_st16(lane_base + ocol + 32 * c, w0);
          tc::tmem_st16(lane_base + ocol + 32 * c + 16, w1);
        }
      }
      tc::tmem_st_wait();
      tc::fence_before_sync();
      mbar_arrive(&pfull[i]);
    }
    if (ok && n > 0) ok = __all_sync(0xFFFFFFFFu, mbar_wait(&odone[i], (n - 1) & 1));
    if (!ok) {
      report(p.status, WM_ERR_TIMEOUT);
    } else {
      __nv_bfloat16* dst =
          reinterpret_cast<__nv_bfloat16*>(p.out) + (((int64_t)b * p.Tq + r) * p.Hq + hh[i]) * HD;
      const float inv = (n > 0 && l > 0.f) ? 1.f / l : 0.f;
      tc::fence_after_sync();
#pragma unroll
      for (int c = 0; c < HD / 32; ++c) {
        uint32_t v[32];
        if (n > 0) {  // n is the same for the whole warp group
          tc::tmem_ld32(lane_base + ocol + 32 * c, v);
          tc::tmem_ld_wait();
        }
        if (r >= p.Tq) continue;
#pragma unroll
        for (int e = 0; e < 32; e += 8) {
          float f[8];
#pragma unroll
          for (int t = 0; t < 8; ++t) f[t] = n > 0 ? __uint_as_float(v[e + t]) * inv : 0.f;
          uint4 u;
          __nv_bfloat162 t0 = __floats2bfloat162_rn(f[0], f[1]);
          __nv_bfloat162 t1 = __floats2bfloat162_rn(f[2], f[3]);
          __nv_bfloat162 t2 = __floats2bfloat162_rn(f[4], f[5]);
          __nv_bfloat162 t3 = __floats2bfloat162_rn(f[6], f[7]);
          u.x = *reinterpret_cast<uint32_t*>(&t0);
          u.y = *reinterpret_cast<uint32_t*>(&t1);
          u.z = *reinterpret_cast<uint32_t*>(&t2);
          u.w = *reinterpret_cast<uint32_t*>(&t3);
          *reinterpret_cast<uint4*>(dst + 32 * c + e) = u;
        }
      }
    }
  }
  // Every MMA this CTA issued has completed (each was waited on through its
  // commit barrier, or the CTA gave up after a bounded wait); release TMEM.
  tc::fence_before_sync();
  __syncthreads();
  if (warp == 0) {
    tc::fence_after_sync();
    tc::tmem_dealloc(tmem, kTmemCols);
  }
}

template <int HD>
cudaError_t launch_hd(const CUtensorMap& q, const CUtensorMap& k, const CUtensorMap& v,
                      const PrefillParams& p, cudaStream_t s) {
  static size_t smem_set[kSmemOptDevices] = {};
  auto kern = prefill_attn_kernel<HD>;
  if (cudaError_t e = opt_in_smem(kern, (size_t)PShape<HD>::SMEM, smem_set); e != cudaSuccess)
    return e;
  cudaLaunchConfig_t cfg = {};
  const int rows_cta = p.pair ? kPM : kQT * kPM;
  cfg.gridDim = dim3((p.Tq + rows_cta - 1) / rows_cta, p.pair ? p.Hq / kQT : p.Hq, p.B);
  cfg.blockDim = dim3(kPThreads);
  cfg.dynamicSmemBytes = PShape<HD>::SMEM;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, q, k, v, p);
}

}  // namespace

cudaError_t launch_prefill_attn(const PrefillLaunch& L, cudaStream_t s) {
  CUtensorMap tq, tk, tv;
  const uint64_t pool_rows = (uint64_t)L.k * L.num_pages * L.Hkv * L.P;
  const uint32_t box_rows = L.P >= kPN ? (uint32_t)kPN : (uint32_t)L.P;
  if (!tma_map_bf16_2d(&tq, L.q, (uint64_t)L.B * L.Tq, (uint64_t)L.Hq * L.d,
                       (uint64_t)L.Hq * L.d, (uint32_t)kPM) ||
      !tma_map_bf16_2d(&tk, L.k_pool, pool_rows, L.d, L.d, box_rows) ||
      !tma_map_bf16_2d(&tv, L.v_pool, pool_rows, L.d, L.d, box_rows))
    return cudaErrorInvalidValue;
  PrefillParams p{};
  p.pos = L.pos;
  p.page_table = L.page_table;
  p.out = L.out;
  p.status = L.status;
  p.B = L.B;
  p.Tq = L.Tq;
  p.Hq = L.Hq;
  p.G = L.Hq / L.Hkv;
  p.pair = (p.G % kQT == 0) ? 1 : 0;
  p.Hkv = L.Hkv;
  p.chan = L.chan;
  p.num_pages = L.num_pages;
  p.max_pages = L.max_pages;
  p.P = L.P;
  int lg = 0;
  while ((1 << lg) < L.P) ++lg;
  p.log2P = lg;
  p.qscale = (float)(1.4426950408889634 / sqrt((double)L.d));
  switch (L.d) {
    case 64: return launch_hd<64>(tq, tk, tv, p, s);
    case 96: return launch_hd<96>(tq, tk, tv, p, s);
    case 128: return launch_hd<128>(tq, tk, tv, p, s);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace wm
