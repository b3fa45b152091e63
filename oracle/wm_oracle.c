/*
 * WhiteMatter decode hot path -- fp64 CPU oracle.
 *
 * TEST INFRASTRUCTURE ONLY.  Only tests/, __graft_entry__.smoke() and the
 * CPU-baseline leg of bench.py load this library.  The product library
 * (paper_2608_18486_gb300) never calls it, and the two share no code,
 * headers, tables or helpers.
 *
 * What it computes, in plain loops and in double precision, for each token:
 *   Sec. 3.1 Step 1: pre-mix RMSNorm of the L states entering the layers,
 *                    a linear router over every p-th normed state counting
 *                    down from layer L-1, reshape of its kL outputs to k x L,
 *                    and the signed L-way mix into k channels (per branch).
 *   Sec. 3.1 Step 2: per-channel RMSNorm, per-channel K/V projection,
 *                    per-channel key normalisation (QK-norm) and RoPE on keys.
 *   Sec. 3.1 Step 3: layer l attends over the cache of its channel c(l) with
 *                    standard softmax attention.
 *   Sec. 3.2:        a dummy KV entry occupies cache slot 0, so the token at
 *                    position i is stored at slot i + 1.
 *   Sec. 3.2-3.3:    causal attention for prefill and the token-parallel
 *                    (Jacobi / cyclic Gauss-Seidel) passes: the query of the
 *                    token at position i reads slots 0 .. i of its layer's
 *                    channel, i.e. the dummy and the tokens before it.
 * Inputs are the same fp32 values, or bf16 bit patterns, the GPU receives;
 * they are widened to double on every read.
 *
 * Readings of points the paper leaves open (each documented with the tests):
 *   - RMSNorm(x) = x / sqrt(mean(x^2) + eps) * gain, with learned gains; the
 *     pre-mix gain is one D-vector per branch shared by all layers.
 *   - The router input stacks the selected layers in the order they are
 *     enumerated (L-1, L-1-p, ...); the kL router outputs are reshaped
 *     row-major, alpha[j][l] = z[j*L + l].  No activation, no normalisation.
 *   - QK-norm is an RMSNorm over each head's d key elements with a
 *     per-channel d-vector gain; RoPE is the rotate-half form pairing element
 *     i with i + d/2 at inverse frequency theta^(-2i/d).
 *   - Attention scale 1/sqrt(d); no softcap, window or mask other than the
 *     sequence length; query head hq reads kv head hq / (Hq/Hkv).
 *
 * Cache layout read by orc_decode_attn (the library's documented layout):
 *   pool[c][page][hkv][slot_in_page][e], page = page_table[b][s / P].
 */
#include <math.h>
#include <stddef.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

enum { ORC_F32 = 0, ORC_BF16 = 1 };
enum { ORC_OK = 0, ORC_ERR_ARG = 1, ORC_ERR_BOUNDS = 4 };

/* Read element i of an fp32 array or of an array of bf16 bit patterns. */
static double rd(const void* p, int64_t i, int dt) {
  if (dt == ORC_F32) return (double)((const float*)p)[i];
  uint32_t u = ((uint32_t)((const uint16_t*)p)[i]) << 16;
  float f;
  memcpy(&f, &u, sizeof f);
  return (double)f;
}

static const void* adv(const void* p, int64_t n, int dt) {
  return (const char*)p + n * (dt == ORC_F32 ? 4 : 2);
}

int orc_max_threads(void) {
#ifdef _OPENMP
  return omp_get_max_threads();
#else
  return 1;
#endif
}

/* RMSNorm: y = x / sqrt(mean(x^2) + eps) * g.  g == NULL means unit gain. */
void orc_rmsnorm(const double* x, int n, double eps, const double* g, double* y) {
  double ss = 0.0;
  for (int i = 0; i < n; ++i) ss += x[i] * x[i];
  double r = 1.0 / sqrt(ss / n + eps);
  for (int i = 0; i < n; ++i) y[i] = x[i] * r * (g ? g[i] : 1.0);
}

/* Rotate-half RoPE of one head vector at position pos, in place:
 * for i < d/2, with a = pos * theta^(-2i/d):
 *   y[i]       <- y[i] cos a - y[i+d/2] sin a
 *   y[i+d/2]   <- y[i+d/2] cos a + y[i] sin a                               */
void orc_rope(double* y, int d, double pos, double theta) {
  int h = d / 2;
  for (int i = 0; i < h; ++i) {
    double a = pos * pow(theta, -2.0 * i / d);
    double c = cos(a), s = sin(a);
    double x0 = y[i], x1 = y[i + h];
    y[i] = x0 * c - x1 * s;
    y[i + h] = x1 * c + x0 * s;
  }
}

/*
 * Sec. 3.1 Step 1 for one token, both branches (X = 0 keys, X = 1 values).
 *   h      [L][D]              hidden states entering layers 0..L-1
 *   pre_g  [2][D]              pre-mix RMSNorm gains
 *   Wr     [2][k*L][Lp*D]      router weights, Lp = ceil(L / p)
 *   br     [2][k*L]            router biases
 * Outputs:
 *   hhat   [2][L][D]           pre-mix normed states
 *   alpha  [2][k][L]           mixing weights (signed, unnormalised)
 *   macs[0] += router multiply-accumulates
 */
void orc_pool_route(int L, int k, int D, int p, double eps, int dt, const void* h,
                    const void* pre_g, const void* Wr, const void* br, double* hhat,
                    double* alpha, int64_t* macs) {
  int Lp = (L + p - 1) / p;
  int64_t in_dim = (int64_t)Lp * D;
  double* x = (double*)malloc(sizeof(double) * D);
  double* g = (double*)malloc(sizeof(double) * D);
  double* xi = (double*)malloc(sizeof(double) * in_dim);
  for (int X = 0; X < 2; ++X) {
    for (int e = 0; e < D; ++e) g[e] = rd(pre_g, (int64_t)X * D + e, dt);
    /* pre-mix RMSNorm of each source state */
    for (int l = 0; l < L; ++l) {
      for (int e = 0; e < D; ++e) x[e] = rd(h, (int64_t)l * D + e, dt);
      orc_rmsnorm(x, D, eps, g, hhat + ((int64_t)X * L + l) * D);
    }
    /* router input: every p-th normed state, counting down from layer L-1 */
    for (int m = 0; m < Lp; ++m) {
      int l = L - 1 - m * p;
      memcpy(xi + (int64_t)m * D, hhat + ((int64_t)X * L + l) * D, sizeof(double) * D);
    }
    /* linear router, then reshape of the kL outputs to k x L (row-major) */
    const void* W = adv(Wr, (int64_t)X * k * L * in_dim, dt);
    for (int o = 0; o < k * L; ++o) {
      double z = rd(br, (int64_t)X * k * L + o, dt);
      for (int64_t c = 0; c < in_dim; ++c) z += rd(W, (int64_t)o * in_dim + c, dt) * xi[c];
      macs[0] += in_dim;
      int j = o / L, l = o % L;
      alpha[((int64_t)X * k + j) * L + l] = z;
    }
  }
  free(x);
  free(g);
  free(xi);
}

/*
 * Sec. 3.1 Step 1 (mix) and Step 2 for one token, one branch, one channel j.
 *   hhat_X   [L][D]          pre-mix normed states of this branch
 *   alpha_Xj [L]             mixing weights of channel j
 *   ch_g_Xj  [D]             gain of RMSNorm^X_j
 *   W_Xj     [Hkv*d][D]      projection W^K_j or W^V_j
 *   qk_g_j   [d]             QK-norm gain of channel j (keys only)
 *   is_key   1: apply QK-norm and RoPE at position pos to each head
 * Outputs: htilde [D] (may be NULL), out [Hkv*d];
 *   macs[0] += mix MACs, macs[1] += projection MACs.
 */
void orc_pool_channel(int L, int D, int Hkv, int d, double eps, double eps_qk, double theta,
                      int is_key, double pos, int dt, const double* hhat_X,
                      const double* alpha_Xj, const void* ch_g_Xj, const void* W_Xj,
                      const void* qk_g_j, double* htilde, double* out, int64_t* macs) {
  double* ht = (double*)malloc(sizeof(double) * D);
  double* xn = (double*)malloc(sizeof(double) * D);
  double* g = (double*)malloc(sizeof(double) * D);
  /* h~_j = sum_l alpha[j, l] hhat_l */
  for (int e = 0; e < D; ++e) ht[e] = 0.0;
  for (int l = 0; l < L; ++l)
    for (int e = 0; e < D; ++e) ht[e] += alpha_Xj[l] * hhat_X[(int64_t)l * D + e];
  macs[0] += (int64_t)L * D;
  if (htilde) memcpy(htilde, ht, sizeof(double) * D);
  /* RMSNorm_j, then the channel's projection */
  for (int e = 0; e < D; ++e) g[e] = rd(ch_g_Xj, e, dt);
  orc_rmsnorm(ht, D, eps, g, xn);
  int64_t n_out = (int64_t)Hkv * d;
  for (int64_t n = 0; n < n_out; ++n) {
    double acc = 0.0;
    for (int e = 0; e < D; ++e) acc += rd(W_Xj, n * D + e, dt) * xn[e];
    out[n] = acc;
  }
  macs[1] += n_out * D;
  /* keys: per-head QK-norm, then RoPE at pos; values stay raw */
  if (is_key) {
    double* gq = (double*)malloc(sizeof(double) * d);
    double* y = (double*)malloc(sizeof(double) * d);
    for (int e = 0; e < d; ++e) gq[e] = rd(qk_g_j, e, dt);
    for (int hh = 0; hh < Hkv; ++hh) {
      orc_rmsnorm(out + (int64_t)hh * d, d, eps_qk, gq, y);
      orc_rope(y, d, pos, theta);
      memcpy(out + (int64_t)hh * d, y, sizeof(double) * d);
    }
    free(gq);
    free(y);
  }
  free(ht);
  free(xn);
  free(g);
}

/*
 * The whole pool for B tokens (Sec. 3.1 Steps 1-2; Sec. 3.2 decode order).
 *   h    [B][L][D];  pos [B]: rotary position of each token
 *   ch_g [2][k][D];  Wkv [2][k][Hkv*d][D];  qk_g [k][d]
 * Outputs: K_out, V_out [B][k][Hkv*d]; alpha_out [B][2][k][L] (may be NULL);
 *   macs[3] += router, mix, projection MACs.
 * Tokens are independent; nthreads > 1 runs them on OpenMP threads.
 */
void orc_kv_mix(int B, int L, int k, int D, int Hkv, int d, int p, double eps, double eps_qk,
                double theta, int dt, const void* h, const double* pos, const void* pre_g,
                const void* Wr, const void* br, const void* ch_g, const void* Wkv,
                const void* qk_g, double* K_out, double* V_out, double* alpha_out, int64_t* macs,
                int nthreads) {
  int64_t n_out = (int64_t)Hkv * d;
  int64_t m_router = 0, m_mix = 0, m_proj = 0;
#ifdef _OPENMP
#pragma omp parallel for schedule(dynamic, 1) num_threads(nthreads > 0 ? nthreads : 1) \
    reduction(+ : m_router, m_mix, m_proj)
#endif
  for (int b = 0; b < B; ++b) {
    double* hhat = (double*)malloc(sizeof(double) * 2 * L * D);
    double* alpha = (double*)malloc(sizeof(double) * 2 * k * L);
    int64_t mr[1] = {0}, mc[2] = {0, 0};
    orc_pool_route(L, k, D, p, eps, dt, adv(h, (int64_t)b * L * D, dt), pre_g, Wr, br, hhat,
                   alpha, mr);
    for (int X = 0; X < 2; ++X)
      for (int j = 0; j < k; ++j) {
        double* dst = (X == 0 ? K_out : V_out) + ((int64_t)b * k + j) * n_out;
        orc_pool_channel(L, D, Hkv, d, eps, eps_qk, theta, X == 0, pos[b], dt,
                         hhat + (int64_t)X * L * D, alpha + ((int64_t)X * k + j) * L,
                         adv(ch_g, ((int64_t)X * k + j) * D, dt),
                         adv(Wkv, ((int64_t)X * k + j) * n_out * D, dt),
                         adv(qk_g, (int64_t)j * d, dt), NULL, dst, mc);
      }
    if (alpha_out) memcpy(alpha_out + (int64_t)b * 2 * k * L, alpha, sizeof(double) * 2 * k * L);
    m_router += mr[0];
    m_mix += mc[0];
    m_proj += mc[1];
    free(hhat);
    free(alpha);
  }
  macs[0] += m_router;
  macs[1] += m_mix;
  macs[2] += m_proj;
}

/*
 * Sec. 3.1 Step 3 with the dummy slot of Sec. 3.2: decode attention of
 * query head hq of sequence b over slots 0 .. seq_lens[b]-1 of channel chan.
 *   k_pool, v_pool [kch][num_pages][Hkv][P][d]
 *   page_table [B][max_pages];  seq_lens [B] (slots incl. the dummy)
 *   q [B][Hq][d]
 *   units [nunits][2] = (b, hq) pairs to evaluate; out [nunits][d]
 * Two-pass softmax: s_t = q . K[t] / sqrt(d); w_t = exp(s_t - max s);
 * o = sum_t w_t V[t] / sum_t w_t.  Returns ORC_ERR_BOUNDS if a page id used
 * is outside [0, num_pages) or a length exceeds the page table.
 */
int orc_decode_attn(int Hq, int Hkv, int d, int P, int num_pages, int max_pages, int chan,
                    int dt, const void* k_pool, const void* v_pool, const int32_t* page_table,
                    const int32_t* seq_lens, const void* q, int nunits, const int32_t* units,
                    double* out, int64_t* macs, int nthreads) {
  if (Hkv <= 0 || Hq % Hkv != 0) return ORC_ERR_ARG;
  int group = Hq / Hkv;
  int err = ORC_OK;
  int64_t m_attn = 0;
#ifdef _OPENMP
#pragma omp parallel for schedule(dynamic, 1) num_threads(nthreads > 0 ? nthreads : 1) \
    reduction(+ : m_attn) reduction(max : err)
#endif
  for (int u = 0; u < nunits; ++u) {
    int b = units[2 * u], hq = units[2 * u + 1];
    int hkv = hq / group;
    int S = seq_lens[b];
    double* o = out + (int64_t)u * d;
    for (int e = 0; e < d; ++e) o[e] = 0.0;
    if (S <= 0 || (S + P - 1) / P > max_pages) {
      err = ORC_ERR_BOUNDS;
      continue;
    }
    double* s = (double*)malloc(sizeof(double) * S);
    int64_t* base = (int64_t*)malloc(sizeof(int64_t) * S);
    double inv_sqrt_d = 1.0 / sqrt((double)d);
    int bad = 0;
    for (int t = 0; t < S; ++t) {
      int32_t pg = page_table[(int64_t)b * max_pages + t / P];
      if (pg < 0 || pg >= num_pages) {
        bad = 1;
        break;
      }
      base[t] = ((((int64_t)chan * num_pages + pg) * Hkv + hkv) * P + (t % P)) * d;
    }
    if (bad) {
      err = ORC_ERR_BOUNDS;
      free(s);
      free(base);
      continue;
    }
    int64_t qoff = ((int64_t)b * Hq + hq) * d;
    double smax = -INFINITY;
    for (int t = 0; t < S; ++t) {
      double acc = 0.0;
      for (int e = 0; e < d; ++e) acc += rd(q, qoff + e, dt) * rd(k_pool, base[t] + e, dt);
      s[t] = acc * inv_sqrt_d;
      if (s[t] > smax) smax = s[t];
    }
    double wsum = 0.0;
    for (int t = 0; t < S; ++t) {
      double wt = exp(s[t] - smax);
      wsum += wt;
      for (int e = 0; e < d; ++e) o[e] += wt * rd(v_pool, base[t] + e, dt);
    }
    for (int e = 0; e < d; ++e) o[e] /= wsum;
    m_attn += 2 * (int64_t)S * d;
    free(s);
    free(base);
  }
  if (macs) macs[0] += m_attn;
  return err;
}

/*
 * Sec. 3.1 Step 3 ("standard causal SDPA") with the dummy offset of Sec. 3.2,
 * for many query positions at once: prefill, and one pass of the parallel
 * schedules of Sec. 3.3 (Jacobi: every position; cyclic Gauss-Seidel: the
 * strided group {i : i mod g = q}).  The dummy sits at slot 0 and token t at
 * slot t + 1, so the query of the token at position i may read slots 0 .. i
 * and never the channels at slot i + 1 that its own states produce.
 *
 * q is [B][Tq][Hq][d]: row r of sequence b is the query of the token at
 * position pos[b][r].  For each listed unit (b, r, hq), with hkv = hq / (Hq/Hkv):
 *   s_t = q . K[t] / sqrt(d) for t = 0 .. pos,  w_t = exp(s_t - max s),
 *   o = sum_t w_t V[t] / sum_t w_t.
 * Returns ORC_ERR_BOUNDS if a position is negative or beyond the page table,
 * or a page id used is outside [0, num_pages).
 */
int orc_prefill_attn(int Hq, int Hkv, int d, int P, int num_pages, int max_pages, int chan,
                     int dt, const void* k_pool, const void* v_pool, const int32_t* page_table,
                     const int32_t* pos, int Tq, const void* q, int nunits, const int32_t* units,
                     double* out, int64_t* macs, int nthreads) {
  if (Hkv <= 0 || Hq % Hkv != 0 || Tq <= 0) return ORC_ERR_ARG;
  int group = Hq / Hkv;
  int err = ORC_OK;
  int64_t m_attn = 0;
#ifdef _OPENMP
#pragma omp parallel for schedule(dynamic, 1) num_threads(nthreads > 0 ? nthreads : 1) \
    reduction(+ : m_attn) reduction(max : err)
#endif
  for (int u = 0; u < nunits; ++u) {
    int b = units[3 * u], r = units[3 * u + 1], hq = units[3 * u + 2];
    int hkv = hq / group;
    int i = pos[(int64_t)b * Tq + r];
    double* o = out + (int64_t)u * d;
    for (int e = 0; e < d; ++e) o[e] = 0.0;
    int nslots = i + 1; /* slots 0 .. i */
    if (i < 0 || (nslots + P - 1) / P > max_pages) {
      err = ORC_ERR_BOUNDS;
      continue;
    }
    double* s = (double*)malloc(sizeof(double) * nslots);
    int64_t* base = (int64_t*)malloc(sizeof(int64_t) * nslots);
    int bad = 0;
    for (int t = 0; t < nslots; ++t) {
      int32_t pg = page_table[(int64_t)b * max_pages + t / P];
      if (pg < 0 || pg >= num_pages) {
        bad = 1;
        break;
      }
      base[t] = ((((int64_t)chan * num_pages + pg) * Hkv + hkv) * P + (t % P)) * d;
    }
    if (bad) {
      err = ORC_ERR_BOUNDS;
      free(s);
      free(base);
      continue;
    }
    int64_t qoff = (((int64_t)b * Tq + r) * Hq + hq) * d;
    double scale = 1.0 / sqrt((double)d), smax = -INFINITY;
    for (int t = 0; t < nslots; ++t) {
      double acc = 0.0;
      for (int e = 0; e < d; ++e) acc += rd(q, qoff + e, dt) * rd(k_pool, base[t] + e, dt);
      s[t] = acc * scale;
      if (s[t] > smax) smax = s[t];
    }
    double wsum = 0.0;
    for (int t = 0; t < nslots; ++t) {
      double wt = exp(s[t] - smax);
      wsum += wt;
      for (int e = 0; e < d; ++e) o[e] += wt * rd(v_pool, base[t] + e, dt);
    }
    for (int e = 0; e < d; ++e) o[e] /= wsum;
    m_attn += 2 * (int64_t)nslots * d;
    free(s);
    free(base);
  }
  if (macs) macs[0] += m_attn;
  return err;
}
