// Causal channel attention for prefill and for the token-parallel passes
// (Sec. 3.1 Step 3 "standard causal SDPA", with the dummy offset of Sec. 3.2
// and the Jacobi / cyclic Gauss-Seidel schedules of Sec. 3.3).  Query row r
// of sequence b is the query of the token at position pos[b][r]; it reads
// slots 0 .. pos of its layer's channel: the dummy and the tokens before it.
//
// Design (GB300).  A prefill pass is a dense contraction on both sides of the
// softmax, so it runs on the tcgen05 tensor cores (bf16 operands, fp32
// accumulation in TMEM).  One CTA (4 warps) owns 128 query rows of one query
// head and walks the 128-slot KV tiles of the sequence's channel up to the
// tile's largest position:
//  * TMA brings the Q tile once and the K and V tiles of each KV tile
//    (128-byte swizzle, 64-column boxes; paged: one box per page or per 128
//    slots of a page) through a 2-deep stage ring;
//  * S = Q K^T lands in TMEM columns [0, 128); each thread owns one query row
//    (its TMEM lane), applies the causal mask slot <= pos, keeps the running
//    max and sum, and writes the bf16 probabilities P into shared memory in
//    the layout of an MMA A operand;
//  * O_tile = P V lands in TMEM columns [128, 128 + d) (V is read as an
//    MN-major B operand straight from its [slot][d] tile); each thread folds
//    its row into registers with the softmax correction;
//  * S of the next KV tile is issued right behind P V, so the tensor core
//    works on it while the threads drain O_tile.
// Slots beyond the tile's largest position may hold anything (unwritten
// cache); their V rows are zeroed in shared memory before P V, and masked
// scores are replaced, never multiplied, so no NaN there reaches the output.
#include <math.h>

#include "internal.h"
#include "tc.cuh"

namespace wm {
namespace {

constexpr int kPM = 128;         // query rows per CTA (MMA M)
constexpr int kPN = 128;         // slots per KV tile
constexpr int kPThreads = 128;   // one thread per query row
constexpr uint32_t kBlock = 128u * 128u;  // one 64-column block of a 128-row tile

template <int HD>
struct PShape {
  static constexpr int CB = (HD + 63) / 64;                   // 64-column blocks of a head row
  static constexpr uint32_t Q_BYTES = CB * kBlock;
  static constexpr uint32_t KV_BYTES = CB * kBlock;           // one K or V tile
  static constexpr uint32_t STAGE = 2 * KV_BYTES;             // K then V
  static constexpr uint32_t P_BYTES = 2 * kBlock;             // 128 x 128 bf16
  static constexpr uint32_t SMEM = Q_BYTES + 2 * STAGE + P_BYTES + 1024;  // + alignment
};
constexpr uint32_t kPTmemCols = 256;  // S in [0, 128), O_tile in [128, 128 + d)

struct PrefillParams {
  const int32_t* pos;         // [B][Tq]
  const int32_t* page_table;  // [B][max_pages]
  void* out;                  // [B][Tq][Hq][d] bf16
  int32_t* status;
  int32_t B, Tq, Hq, G, Hkv, chan, num_pages, max_pages, P, log2P;
  float qscale;               // log2(e) / sqrt(d)
};

__device__ __forceinline__ int block_max(int v, int* red) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = max(v, __shfl_xor_sync(0xFFFFFFFFu, v, o));
  __syncthreads();
  if (lane == 0) red[warp] = v;
  __syncthreads();
  return max(max(red[0], red[1]), max(red[2], red[3]));
}

template <int HD>
__global__ void __launch_bounds__(kPThreads, 1)
    prefill_attn_kernel(const __grid_constant__ CUtensorMap tmQ,
                        const __grid_constant__ CUtensorMap tmK,
                        const __grid_constant__ CUtensorMap tmV, const PrefillParams p) {
  using SH = PShape<HD>;
  constexpr int CB = SH::CB;
  extern __shared__ uint8_t smem_dyn[];
  __shared__ uint64_t qbar, full[2], sbar, obar;
  __shared__ uint32_t tmem_base;
  __shared__ int red[4];

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int b = blockIdx.z, hq = blockIdx.y, hkv = hq / p.G;
  const int ntiles = (p.Tq + kPM - 1) / kPM;
  const int r0 = (ntiles - 1 - (int)blockIdx.x) * kPM;  // later rows (more work) start first
  const int r = r0 + tid;
  uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_dyn) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* Qs = base;
  uint8_t* KVs = Qs + SH::Q_BYTES;  // [2 stages][K | V]
  uint8_t* Ps = KVs + 2 * SH::STAGE;

  if (tid == 0) {
    mbar_init(&qbar, 1);
    mbar_init(&full[0], 1);
    mbar_init(&full[1], 1);
    mbar_init(&sbar, 1);
    mbar_init(&obar, 1);
    fence_mbar_init();
    tc::prefetch_tensormap(&tmQ);
    tc::prefetch_tensormap(&tmK);
    tc::prefetch_tensormap(&tmV);
  }
  if (warp == 0) {
    tc::tmem_alloc(&tmem_base, kPTmemCols);
    tc::tmem_relinquish();
  }
  // programmatic dependent launch: positions, table, queries and cache may
  // come from the previous grid
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  asm volatile("griddepcontrol.wait;" ::: "memory");

  const int max_slots = p.max_pages * p.P;
  int mypos = -1;  // -1: row absent or invalid, fully masked
  if (r < p.Tq) {
    const int v = p.pos[(int64_t)b * p.Tq + r];
    if (v >= 0 && v < max_slots) mypos = v;
    else report(p.status, WM_ERR_BOUNDS);
  }
  tc::fence_before_sync();
  const int maxpos = block_max(mypos, red);  // also publishes the barrier inits and TMEM base
  tc::fence_after_sync();
  const uint32_t tmem = tmem_base;
  const int nkv = maxpos >= 0 ? maxpos / kPN + 1 : 0;  // KV tiles 0 .. nkv-1

  // ---- producer (thread 0): K and V of KV tile j into stage j & 1
  auto issue_kv = [&](int j) {
    const int st = j & 1;
    uint8_t* Kd = KVs + st * SH::STAGE;
    uint8_t* Vd = Kd + SH::KV_BYTES;
    mbar_arrive_expect_tx(&full[st], SH::STAGE);
    const int s0 = j * kPN;
    const int boxes = p.P >= kPN ? 1 : kPN >> p.log2P;
    const int brows = p.P >= kPN ? kPN : p.P;
    for (int t = 0; t < boxes; ++t) {
      const int s = s0 + t * brows;        // first slot of the box
      const int lp = s >> p.log2P;         // logical page
      int row = -brows;                    // fully outside the map: reads zeros
      if (s <= maxpos && lp < p.max_pages) {
        const int pg = p.page_table[(int64_t)b * p.max_pages + lp];
        if (pg >= 0 && pg < p.num_pages)
          row = (int)((((int64_t)p.chan * p.num_pages + pg) * p.Hkv + hkv) * p.P + (s & (p.P - 1)));
        else
          report(p.status, WM_ERR_BOUNDS);
      }
#pragma unroll
      for (int cb = 0; cb < CB; ++cb) {
        tc::tma_load_2d(Kd + cb * kBlock + t * brows * 128, &tmK, cb * 64, row, &full[st]);
        tc::tma_load_2d(Vd + cb * kBlock + t * brows * 128, &tmV, cb * 64, row, &full[st]);
      }
    }
  };
  const uint32_t idesc_s = tc::idesc_bf16_f32(kPM, kPN);
  const uint32_t idesc_o = tc::idesc_bf16_f32(kPM, HD) | tc::kIdescBMajorMN;
  auto issue_s = [&](int j) {  // S = Q K_j^T into TMEM columns [0, 128)
    const uint32_t q0 = smem_u32(Qs), k0 = smem_u32(KVs + (j & 1) * SH::STAGE);
#pragma unroll
    for (int kk = 0; kk < HD / 16; ++kk) {
      const uint32_t off = (kk >> 2) * kBlock + (kk & 3) * 32;
      tc::mma_bf16(tmem, tc::sdesc_kmajor_sw128(q0 + off), tc::sdesc_kmajor_sw128(k0 + off),
                   idesc_s, kk > 0);
    }
    tc::mma_commit(&sbar);
  };
  auto issue_o = [&](int j) {  // O_tile = P V_j into TMEM columns [128, 128 + HD)
    const uint32_t p0 = smem_u32(Ps), v0 = smem_u32(KVs + (j & 1) * SH::STAGE + SH::KV_BYTES);
#pragma unroll
    for (int kk = 0; kk < kPN / 16; ++kk) {
      const uint64_t adesc = tc::sdesc_kmajor_sw128(p0 + (kk >> 2) * kBlock + (kk & 3) * 32);
      const uint64_t bdesc = tc::sdesc_mnmajor_sw128(v0 + kk * 16 * 128, kBlock, 1024);
      tc::mma_bf16(tmem + kPM, adesc, bdesc, idesc_o, kk > 0);
    }
    tc::mma_commit(&obar);
  };

  bool ok = true;
  if (tid == 0 && nkv > 0) {
    mbar_arrive_expect_tx(&qbar, SH::Q_BYTES);
#pragma unroll
    for (int cb = 0; cb < CB; ++cb)
      tc::tma_load_2d(Qs + cb * kBlock, &tmQ, hq * HD + cb * 64, b * p.Tq + r0, &qbar);
    issue_kv(0);
    if (nkv > 1) issue_kv(1);
    ok = mbar_wait(&qbar, 0) && mbar_wait(&full[0], 0);
    if (ok) {
      tc::fence_after_sync();
      issue_s(0);
    }
  }

  float m = -INFINITY, l = 0.f;  // running max (log2 units) and sum of this row
  float o[HD];
#pragma unroll
  for (int i = 0; i < HD; ++i) o[i] = 0.f;
  const uint32_t lane_base = tmem + ((uint32_t)(warp * 32) << 16);
  uint8_t* prow = Ps + tid * 128;
  const int sw = tid & 7;  // 128-byte swizzle: 16-byte unit u of row t sits at u ^ (t & 7)

  for (int j = 0; j < nkv; ++j) {
    ok = __syncthreads_and(ok);
    if (!ok) break;
    ok = mbar_wait(&sbar, j & 1);
    tc::fence_after_sync();
    const int s0 = j * kPN;
    // pass 1: row max of the masked, scaled scores
    float mx = -INFINITY;
#pragma unroll
    for (int c = 0; c < kPN / 16; ++c) {
      uint32_t v[16];
      tc::tmem_ld16(lane_base + c * 16, v);
      tc::tmem_ld_wait();
#pragma unroll
      for (int i = 0; i < 16; ++i)
        if (s0 + c * 16 + i <= mypos) mx = fmaxf(mx, __uint_as_float(v[i]) * p.qscale);
    }
    const float mn = fmaxf(m, mx);
    const float corr = (m == -INFINITY) ? 0.f : exp2f(m - mn);
    // pass 2: probabilities (bf16) into the P tile, and their sum
    float sum = 0.f;
#pragma unroll
    for (int c = 0; c < kPN / 16; ++c) {
      uint32_t v[16];
      tc::tmem_ld16(lane_base + c * 16, v);
      tc::tmem_ld_wait();
      uint32_t packed[8];
#pragma unroll
      for (int i = 0; i < 16; i += 2) {
        const bool in0 = s0 + c * 16 + i <= mypos, in1 = s0 + c * 16 + i + 1 <= mypos;
        const float p0 = in0 ? exp2f(__uint_as_float(v[i]) * p.qscale - mn) : 0.f;
        const float p1 = in1 ? exp2f(__uint_as_float(v[i + 1]) * p.qscale - mn) : 0.f;
        const __nv_bfloat162 h = __floats2bfloat162_rn(p0, p1);
        sum += __low2float(h) + __high2float(h);
        packed[i / 2] = *reinterpret_cast<const uint32_t*>(&h);
      }
      // columns 16c .. 16c+15: K block c/4, 16-byte units 2(c%4) and 2(c%4)+1
      uint8_t* blk = prow + (c >> 2) * kBlock;
      const int u = (c & 3) * 2;
      *reinterpret_cast<uint4*>(blk + (((u) ^ sw) << 4)) =
          make_uint4(packed[0], packed[1], packed[2], packed[3]);
      *reinterpret_cast<uint4*>(blk + (((u + 1) ^ sw) << 4)) =
          make_uint4(packed[4], packed[5], packed[6], packed[7]);
    }
    l = l * corr + sum;
    m = mn;
    if (j == nkv - 1 && s0 + kPN - 1 > maxpos) {
      // slots past the largest position may be unwritten: zero their V rows
      ok = mbar_wait(&full[j & 1], (j >> 1) & 1) && ok;
      if (tid > maxpos - s0) {
        uint8_t* vrow = KVs + (j & 1) * SH::STAGE + SH::KV_BYTES + tid * 128;
#pragma unroll
        for (int cb = 0; cb < CB; ++cb)
#pragma unroll
          for (int u = 0; u < 8; ++u)
            *reinterpret_cast<uint4*>(vrow + cb * kBlock + u * 16) = make_uint4(0, 0, 0, 0);
      }
    }
    fence_proxy_async_shared();  // P (and zeroed V rows) visible to the tensor core
    tc::fence_before_sync();
    ok = __syncthreads_and(ok);
    if (!ok) break;
    if (tid == 0) {
      tc::fence_after_sync();
      issue_o(j);
      if (j + 1 < nkv) {
        ok = mbar_wait(&full[(j + 1) & 1], ((j + 1) >> 1) & 1);
        tc::fence_after_sync();
        if (ok) issue_s(j + 1);
      }
    }
    ok = mbar_wait(&obar, j & 1) && ok;
    tc::fence_after_sync();
#pragma unroll
    for (int c = 0; c < HD / 16; ++c) {
      uint32_t v[16];
      tc::tmem_ld16(lane_base + kPM + c * 16, v);
      tc::tmem_ld_wait();
#pragma unroll
      for (int i = 0; i < 16; ++i) o[c * 16 + i] = fmaf(o[c * 16 + i], corr, __uint_as_float(v[i]));
    }
    tc::fence_before_sync();
    // stage j & 1 is free (S_j and P V_j are done): bring KV tile j + 2
    if (tid == 0 && j + 2 < nkv && ok) issue_kv(j + 2);
  }
  if (!ok) {
    report(p.status, WM_ERR_TIMEOUT);
  } else if (r < p.Tq) {
    const float inv = l > 0.f ? 1.f / l : 0.f;
    __nv_bfloat16* dst =
        reinterpret_cast<__nv_bfloat16*>(p.out) + (((int64_t)b * p.Tq + r) * p.Hq + hq) * HD;
#pragma unroll
    for (int i = 0; i < HD; i += 8) {
      uint4 w;
      __nv_bfloat162 t0 = __floats2bfloat162_rn(o[i] * inv, o[i + 1] * inv);
      __nv_bfloat162 t1 = __floats2bfloat162_rn(o[i + 2] * inv, o[i + 3] * inv);
      __nv_bfloat162 t2 = __floats2bfloat162_rn(o[i + 4] * inv, o[i + 5] * inv);
      __nv_bfloat162 t3 = __floats2bfloat162_rn(o[i + 6] * inv, o[i + 7] * inv);
      w.x = *reinterpret_cast<uint32_t*>(&t0);
      w.y = *reinterpret_cast<uint32_t*>(&t1);
      w.z = *reinterpret_cast<uint32_t*>(&t2);
      w.w = *reinterpret_cast<uint32_t*>(&t3);
      *reinterpret_cast<uint4*>(dst + i) = w;
    }
  }
  // Every MMA this CTA issued has completed (each was waited on through its
  // commit barrier, or the CTA gave up after a bounded wait); release TMEM.
  tc::fence_before_sync();
  __syncthreads();
  if (warp == 0) {
    tc::fence_after_sync();
    tc::tmem_dealloc(tmem, kPTmemCols);
  }
}

template <int HD>
cudaError_t launch_hd(const CUtensorMap& q, const CUtensorMap& k, const CUtensorMap& v,
                      const PrefillParams& p, cudaStream_t s) {
  static bool attr_set = false;
  auto kern = prefill_attn_kernel<HD>;
  if (!attr_set) {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)PShape<HD>::SMEM);
    if (e != cudaSuccess) return e;
    attr_set = true;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((p.Tq + kPM - 1) / kPM, p.Hq, p.B);
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
