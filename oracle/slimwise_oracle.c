/*
 * slimwise_oracle.c -- plain, slow CPU oracle for the pruned-pool batched-decode
 * MoE layer of SlimWise (arXiv 2609.34117).
 *
 * TEST INFRASTRUCTURE ONLY.  Only the test suite, the smoke check and the
 * benchmark's CPU-baseline leg may load this library.  The CUDA product path
 * never calls, links or includes it, and it includes nothing from the product.
 *
 * What it computes, in the paper's order:
 *   1. router logits z[t,e] = sum_h x[t,h] * Wr[e,h]             (Sec. 3.1, "router logits z")
 *   2. masked logits  z~_e = z_e on the retained set K', tau off  (Sec. 3.1, Eq. 2)
 *   3. top-k of z~ (k unchanged by pruning)                         (Sec. 2.3, Sec. 3.1)
 *   4. gates renormalised over the k selected experts alone         (Sec. 3.1, after Eq. 2)
 *   5. grouping of the (token, slot) pairs by expert and the union
 *      of selected experts, whose weights a decode step reads      (Sec. 2.1, Eq. 1)
 *   6. per (token, expert) SwiGLU expert FFN
 *   7. gate-weighted sum of the k expert outputs
 *
 * Readings where the paper is silent (each one is listed in the design notes):
 *   - tau = -infinity; since k <= m' it is never selected.
 *   - ties in top-k go to the lowest original expert id; the comparison is
 *     IEEE ">" on fp32 logits, so -0 and +0 tie.
 *   - selection compares logits (monotone-equivalent to probabilities).
 *   - logit summation order is fixed (the "canonical order" below) because the
 *     top-k decision is an integer result that must match the kernel bit for
 *     bit; both sides make that decision in fp32, the kernel's precision.
 *   - the expert FFN is SwiGLU with a fused [gate; up] weight (gate rows first),
 *     W_gu [E, 2I, H] and W_down [E, H, I] (out x in).
 *   - everything after the routing decision (gates, FFN, combine) is evaluated
 *     in fp64 from the bf16/fp32 inputs; the activation between the two GEMMs
 *     is not rounded.
 *   - the grouping of slots is the stable order (expert asc, token asc).
 *
 * Build: gcc -O2 -ffp-contract=off -fPIC -shared (no fast-math).  A second
 * build with -fopenmp spreads the tokens of oracle_experts_combine over the
 * host's cores; it is used only to time the oracle on all cores.  Each token
 * is computed by one thread with the same arithmetic in the same order, so
 * both builds give identical results.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

/* Threads the token loop uses: 1 unless built with OpenMP. */
int oracle_num_threads(void) {
#ifdef _OPENMP
  return omp_get_max_threads();
#else
  return 1;
#endif
}

/* bf16 is the upper half of an fp32 bit pattern. */
static float bf16_to_float(uint16_t v) {
  uint32_t u = ((uint32_t)v) << 16;
  float f;
  memcpy(&f, &u, sizeof f);
  return f;
}

/*
 * Router logits in the canonical fp32 order (Sec. 3.1: "router logits z").
 * 32 partial sums p[l]; for each 128-wide chunk c and q = 0..3 the element
 * h = 128c + 4l + q is accumulated into p[l] by one fused multiply-add, chunks
 * and q ascending.  The 32 partials are then combined by five rounds of
 * p[l] <- p[l] + p[l xor off] for off = 16, 8, 4, 2, 1 (all l at once), and
 * z = p[0].  H must be a multiple of 128.
 *
 * x: bf16 [B, H] row-major, wr: fp32 [E, H] row-major, z: fp32 [B, E].
 */
void oracle_router_logits(const uint16_t *x, const float *wr, int B, int H,
                          int E, float *z) {
  for (int t = 0; t < B; ++t) {
    for (int e = 0; e < E; ++e) {
      float p[32], tmp[32];
      for (int l = 0; l < 32; ++l) p[l] = 0.0f;
      for (int c = 0; c < H / 128; ++c)
        for (int l = 0; l < 32; ++l)
          for (int q = 0; q < 4; ++q) {
            int h = 128 * c + 4 * l + q;
            p[l] = fmaf(bf16_to_float(x[(size_t)t * H + h]),
                        wr[(size_t)e * H + h], p[l]);
          }
      for (int off = 16; off >= 1; off >>= 1) {
        for (int l = 0; l < 32; ++l) tmp[l] = p[l] + p[l ^ off];
        for (int l = 0; l < 32; ++l) p[l] = tmp[l];
      }
      z[(size_t)t * E + e] = p[0];
    }
  }
}

/*
 * Eq. 2 masking, top-k and renormalised gates for each token.
 *
 * retained: n_retained expert ids (any order) forming K'; pass NULL for the
 * full pool (K' = all E experts).  idx: int32 [B, k] in selection order
 * (logit descending, id ascending on ties).  gates: fp64 [B, k],
 * g_j = exp(z_j - z_1) / sum_j' exp(z_j' - z_1) over the k selected only.
 * Returns 0, or -1 if k is not in [1, |K'|] or an id is out of range.
 */
int oracle_route(const float *z, int B, int E, const int32_t *retained,
                 int n_retained, int k, int32_t *idx, double *gates) {
  int m_prime = retained ? n_retained : E;
  if (k < 1 || k > m_prime) return -1;
  unsigned char *in_set = (unsigned char *)calloc((size_t)E, 1);
  unsigned char *taken = (unsigned char *)calloc((size_t)E, 1);
  float *zm = (float *)malloc(sizeof(float) * (size_t)E);
  if (!in_set || !taken || !zm) {
    free(in_set); free(taken); free(zm);
    return -1;
  }
  if (retained) {
    for (int r = 0; r < n_retained; ++r) {
      if (retained[r] < 0 || retained[r] >= E) {
        free(in_set); free(taken); free(zm);
        return -1;
      }
      in_set[retained[r]] = 1;
    }
  } else {
    memset(in_set, 1, (size_t)E);
  }
  for (int t = 0; t < B; ++t) {
    /* Eq. 2: keep the logit on K', tau = -inf elsewhere. */
    for (int e = 0; e < E; ++e)
      zm[e] = in_set[e] ? z[(size_t)t * E + e] : -INFINITY;
    memset(taken, 0, (size_t)E);
    for (int j = 0; j < k; ++j) {
      int best = -1;
      for (int e = 0; e < E; ++e) {
        if (taken[e]) continue;
        if (best < 0 || zm[e] > zm[best]) best = e;
      }
      taken[best] = 1;
      idx[(size_t)t * k + j] = best;
    }
    /* Renormalisation over the selected k alone (Sec. 3.1). */
    double z1 = (double)zm[idx[(size_t)t * k]];
    double denom = 0.0;
    for (int j = 0; j < k; ++j)
      denom += exp((double)zm[idx[(size_t)t * k + j]] - z1);
    for (int j = 0; j < k; ++j)
      gates[(size_t)t * k + j] =
          exp((double)zm[idx[(size_t)t * k + j]] - z1) / denom;
  }
  free(in_set); free(taken); free(zm);
  return 0;
}

/*
 * Grouping of the B*k (token, slot) pairs by expert (Sec. 2.1: a decode step
 * reads the union of the experts selected across the batch, Eq. 1).
 *   counts[e]   number of slots routed to e                      [E]
 *   offsets[e]  exclusive prefix sum of counts, offsets[E]=B*k   [E+1]
 *   union_ids   experts with counts > 0, ascending               [E]
 *   *union_size number of such experts (the measured E_distinct)
 *   perm[p]     flat slot t*k+j at grouped position p, ordered by
 *               (expert asc, token asc)                          [B*k]
 *   pos[t*k+j]  grouped position of slot (t, j), the inverse     [B*k]
 */
void oracle_group_by_expert(const int32_t *idx, int B, int k, int E,
                            int32_t *counts, int32_t *offsets,
                            int32_t *union_ids, int32_t *union_size,
                            int32_t *perm, int32_t *pos) {
  for (int e = 0; e < E; ++e) counts[e] = 0;
  for (int s = 0; s < B * k; ++s) counts[idx[s]] += 1;
  offsets[0] = 0;
  for (int e = 0; e < E; ++e) offsets[e + 1] = offsets[e] + counts[e];
  int u = 0;
  for (int e = 0; e < E; ++e)
    if (counts[e] > 0) union_ids[u++] = e;
  for (int e = u; e < E; ++e) union_ids[e] = -1;
  *union_size = u;
  int32_t *fill = (int32_t *)malloc(sizeof(int32_t) * (size_t)(E > 0 ? E : 1));
  for (int e = 0; e < E; ++e) fill[e] = offsets[e];
  for (int t = 0; t < B; ++t)
    for (int j = 0; j < k; ++j) {
      int s = t * k + j;
      int p = fill[idx[s]]++;
      perm[p] = s;
      pos[s] = p;
    }
  free(fill);
}

/*
 * One expert applied to one token: SwiGLU FFN in fp64.
 *   g_i = sum_h Wgu[i, h] x_h,   u_i = sum_h Wgu[I + i, h] x_h
 *   a_i = SiLU(g_i) * u_i,       SiLU(v) = v / (1 + exp(-v))
 *   y_h = sum_i Wd[h, i] a_i
 * x: bf16 [H]; wgu: bf16 [2I, H] of this expert; wd: bf16 [H, I] of this
 * expert; a: fp64 scratch [I]; y: fp64 [H].
 */
void oracle_expert_swiglu(const uint16_t *x, const uint16_t *wgu,
                          const uint16_t *wd, int H, int I, double *a,
                          double *y) {
  for (int i = 0; i < I; ++i) {
    double g = 0.0, u = 0.0;
    for (int h = 0; h < H; ++h) {
      double xh = (double)bf16_to_float(x[h]);
      g += (double)bf16_to_float(wgu[(size_t)i * H + h]) * xh;
      u += (double)bf16_to_float(wgu[(size_t)(I + i) * H + h]) * xh;
    }
    a[i] = g / (1.0 + exp(-g)) * u;
  }
  for (int h = 0; h < H; ++h) {
    double acc = 0.0;
    for (int i = 0; i < I; ++i)
      acc += (double)bf16_to_float(wd[(size_t)h * I + i]) * a[i];
    y[h] = acc;
  }
}

/*
 * Expert FFNs and gate-weighted combine for the tokens in `tokens`
 * (n_tokens entries, any subset of [0, B)), given their routing.
 * out: fp64 [n_tokens, H], row r belongs to token tokens[r]:
 *   out[t, h] = sum_{j=0..k-1} gates[t, j] * y^{(idx[t, j])}_h(x_t),  j ascending.
 * Returns 0, or -1 on allocation failure.
 */
int oracle_experts_combine(const uint16_t *x, const int32_t *idx,
                           const double *gates, const uint16_t *w_gate_up,
                           const uint16_t *w_down, int H, int I, int k,
                           const int32_t *tokens, int n_tokens, double *out) {
  int failed = 0;
#pragma omp parallel for schedule(dynamic, 1) reduction(| : failed)
  for (int r = 0; r < n_tokens; ++r) {
    double *a = (double *)malloc(sizeof(double) * (size_t)I);
    double *y = (double *)malloc(sizeof(double) * (size_t)H);
    if (!a || !y) {
      free(a); free(y);
      failed = 1;
      continue;
    }
    int t = tokens[r];
    double *o = out + (size_t)r * H;
    for (int h = 0; h < H; ++h) o[h] = 0.0;
    for (int j = 0; j < k; ++j) {
      int e = idx[(size_t)t * k + j];
      double g = gates[(size_t)t * k + j];
      oracle_expert_swiglu(x + (size_t)t * H,
                           w_gate_up + (size_t)e * 2 * I * H,
                           w_down + (size_t)e * H * I, H, I, a, y);
      for (int h = 0; h < H; ++h) o[h] += g * y[h];
    }
    free(a); free(y);
  }
  return failed ? -1 : 0;
}

/*
 * Shared expert (Sec. 3.3): an always-on SwiGLU expert of intermediate width
 * I_s, scaled per token by a sigmoid gate.  The distilled layer keeps the
 * original shared expert and adds a second of the same width under the same
 * gate, so the deployed form is one expert of twice the width; the oracle
 * takes whatever width it is given.
 *   z_t = w_sg . x_t            (canonical fp32 order, as a router logit)
 *   s_t = 1 / (1 + exp(-z_t))   (fp64)
 *   out[r, h] += s_t * y^{SE}_h(x_t)        for t = tokens[r]
 * The shared term is added after the k routed terms.
 * w_sg: fp32 [H]; w_gu_s: bf16 [2 I_s, H] (gate rows first); w_d_s: bf16
 * [H, I_s]; out: fp64 [n_tokens, H]; gate_out: fp64 [n_tokens] or NULL.
 * Returns 0, or -1 on allocation failure.
 */
int oracle_shared_expert_add(const uint16_t *x, const float *w_sg,
                             const uint16_t *w_gu_s, const uint16_t *w_d_s,
                             int H, int I_s, const int32_t *tokens,
                             int n_tokens, double *out, double *gate_out) {
  double *a = (double *)malloc(sizeof(double) * (size_t)(I_s > 0 ? I_s : 1));
  double *y = (double *)malloc(sizeof(double) * (size_t)H);
  if (!a || !y) {
    free(a); free(y);
    return -1;
  }
  for (int r = 0; r < n_tokens; ++r) {
    int t = tokens[r];
    float z;
    oracle_router_logits(x + (size_t)t * H, w_sg, 1, H, 1, &z);
    double s = 1.0 / (1.0 + exp(-(double)z));
    if (gate_out) gate_out[r] = s;
    oracle_expert_swiglu(x + (size_t)t * H, w_gu_s, w_d_s, H, I_s, a, y);
    double *o = out + (size_t)r * H;
    for (int h = 0; h < H; ++h) o[h] += s * y[h];
  }
  free(a); free(y);
  return 0;
}

/*
 * The whole decode MoE layer over the retained pool for every token:
 * logits -> Eq. 2 mask -> top-k -> renormalised gates -> expert FFNs ->
 * gate-weighted combine.  retained = NULL means the full pool.
 * idx: int32 [B, k]; gates: fp64 [B, k]; out: fp64 [B, H].
 * Returns 0, or -1 on bad arguments / allocation failure.
 */
int oracle_moe_decode(const uint16_t *x, const float *router_w,
                      const int32_t *retained, int n_retained,
                      const uint16_t *w_gate_up, const uint16_t *w_down, int B,
                      int H, int E, int I, int k, int32_t *idx, double *gates,
                      double *out) {
  if (B == 0) return 0;
  float *z = (float *)malloc(sizeof(float) * (size_t)B * E);
  int32_t *tokens = (int32_t *)malloc(sizeof(int32_t) * (size_t)B);
  if (!z || !tokens) {
    free(z); free(tokens);
    return -1;
  }
  oracle_router_logits(x, router_w, B, H, E, z);
  int rc = oracle_route(z, B, E, retained, n_retained, k, idx, gates);
  if (rc == 0) {
    for (int t = 0; t < B; ++t) tokens[t] = t;
    rc = oracle_experts_combine(x, idx, gates, w_gate_up, w_down, H, I, k,
                                tokens, B, out);
  }
  free(z); free(tokens);
  return rc;
}

/*
 * Expert-importance statistics over calibration tokens (Sec. 2.3: routing
 * mass aggregates gate probabilities, EAN measures expert output norms, REAP
 * weights those norms by the gates; App. A: one pass over the calibration
 * data with the full pool).  Routing over the full pool as in
 * oracle_moe_decode; for each token t and each of its k selections e with
 * gate g and expert output y = y^{(e)}(x_t), tokens in order:
 *   stats[e*4 + 0] += 1                 tokens routed to e
 *   stats[e*4 + 1] += g                 routing mass
 *   stats[e*4 + 2] += ||y||_2           expert activation norm (EAN)
 *   stats[e*4 + 3] += g * ||y||_2       REAP numerator (score: / count)
 * stats: fp64 [E, 4], accumulated into.  Returns 0, or -1 on failure.
 */
int oracle_expert_stats(const uint16_t *x, const float *router_w,
                        const uint16_t *w_gate_up, const uint16_t *w_down,
                        int B, int H, int E, int I, int k, double *stats) {
  if (B == 0) return 0;
  float *z = (float *)malloc(sizeof(float) * (size_t)B * E);
  int32_t *idx = (int32_t *)malloc(sizeof(int32_t) * (size_t)B * k);
  double *gates = (double *)malloc(sizeof(double) * (size_t)B * k);
  double *a = (double *)malloc(sizeof(double) * (size_t)I);
  double *y = (double *)malloc(sizeof(double) * (size_t)H);
  int rc = -1;
  if (z && idx && gates && a && y) {
    oracle_router_logits(x, router_w, B, H, E, z);
    rc = oracle_route(z, B, E, NULL, 0, k, idx, gates);
    for (int t = 0; rc == 0 && t < B; ++t)
      for (int j = 0; j < k; ++j) {
        const int e = idx[(size_t)t * k + j];
        const double g = gates[(size_t)t * k + j];
        oracle_expert_swiglu(x + (size_t)t * H, w_gate_up + (size_t)e * 2 * I * H,
                             w_down + (size_t)e * H * I, H, I, a, y);
        double n2 = 0.0;
        for (int h = 0; h < H; ++h) n2 += y[h] * y[h];
        const double nrm = sqrt(n2);
        stats[(size_t)e * 4 + 0] += 1.0;
        stats[(size_t)e * 4 + 1] += g;
        stats[(size_t)e * 4 + 2] += nrm;
        stats[(size_t)e * 4 + 3] += g * nrm;
      }
  }
  free(z); free(idx); free(gates); free(a); free(y);
  return rc;
}

/*
 * Retained set K' from the statistics (Sec. 3.1: rank the layer's experts by
 * an importance criterion and keep the top m').  Score of expert e:
 *   criterion 0  routing mass   stats[e*4 + 1]
 *   criterion 1  EAN            stats[e*4 + 2]
 *   criterion 2  REAP           stats[e*4 + 3] / stats[e*4 + 0]  (0 if unrouted)
 * The m' highest scores are kept, ties to the lowest id; ids ascending.
 * Returns 0, or -1 on bad arguments.
 */
int oracle_select_retained(const double *stats, int E, int m_prime,
                           int criterion, int32_t *ids) {
  if (m_prime < 0 || m_prime > E || criterion < 0 || criterion > 2) return -1;
  double *score = (double *)malloc(sizeof(double) * (size_t)(E > 0 ? E : 1));
  char *taken = (char *)calloc((size_t)(E > 0 ? E : 1), 1);
  if (!score || !taken) {
    free(score); free(taken);
    return -1;
  }
  for (int e = 0; e < E; ++e) {
    const double *st = stats + (size_t)e * 4;
    if (criterion == 0) score[e] = st[1];
    else if (criterion == 1) score[e] = st[2];
    else score[e] = st[0] > 0.0 ? st[3] / st[0] : 0.0;
  }
  /* m' rounds of arg-max over the remaining experts */
  for (int r = 0; r < m_prime; ++r) {
    int best = -1;
    for (int e = 0; e < E; ++e)
      if (!taken[e] && (best < 0 || score[e] > score[best])) best = e;
    taken[best] = 1;
  }
  int n = 0;
  for (int e = 0; e < E; ++e)
    if (taken[e]) ids[n++] = e;
  free(score); free(taken);
  return 0;
}
