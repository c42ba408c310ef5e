/*
 * body_oracle.c -- fp64 CPU oracle for the paper's two-block expert body.
 *
 * TEST INFRASTRUCTURE ONLY, like soma_oracle.c (whose Philox probe stream it
 * calls).  Nothing in the product path may call, link or load it.  It shares
 * no code with the CUDA library.
 *
 * The model (Sec. "Model size", the width-32 ensembles; App. E for the loss):
 *   - V = 256 bytes; one frozen matrix E [V][d] embeds and decodes.  It is
 *     shared by every expert and is not perturbed.
 *   - The residual stream starts at x = E[byte_t] (d_E = d_t = d: no
 *     projection).
 *   - D pre-norm residual blocks.  Block k:
 *       u  = LN(x) * ga_k                   gain-only LayerNorm
 *       a  = W_ih^k u + W_hh^k h_k          bias-free LSTM, gates i, f, g, o
 *       c_k = f c_k + i g,  h_k = o tanh(c_k)      (state reset per sequence)
 *       x  = x + h_k
 *       v  = LN(x) * gb_k
 *       x  = x + W_2^k GELU(W_1^k v)        bias-free MLP of width 4d,
 *                                           exact (erf) GELU
 *   - y = LN(x) * gf; logits = E y (logit_v = e_v . y); the loss is the
 *     mean next-byte cross entropy in nats/byte (App. E, L_CE).
 *   LN(x) = (x - mean(x)) / sqrt(var(x) + 1e-5), var the mean squared
 *   deviation over the d features.
 *
 * Body parameters of one expert, M_body = 16 D d^2 + (2D + 1) d, flat:
 *   for k = 0..D-1: W_ih^k [4d][d], W_hh^k [4d][d], W_1^k [4d][d], W_2^k [d][4d]
 *   then for k = 0..D-1: ga_k [d], gb_k [d]; then gf [d].
 * The weights come first, so every coordinate p >= 16 D d^2 is a
 * normalisation gain.
 *
 * Probes (App. E): kind 0 is dense Rademacher on every coordinate.  Kind 1
 * is the paper's training law.  Gain coordinates take the dense sign (never
 * zero).  Every other coordinate is the sparse probe of soma_oracle.c (0
 * with probability 1/2).  Both draw on the same Philox stream and bit map,
 * keyed by the expert index and the flat coordinate.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#ifdef _OPENMP
#include <omp.h>
#endif

#define BODY_V 256
#define BODY_LN_EPS 1e-5

/* from soma_oracle.c (the same library) */
int oracle_probe(uint64_t seed, uint64_t step, uint32_t expert, uint32_t probe, int kind,
                 int64_t p0, int64_t count, int8_t* z);

int64_t oracle_body_param_count(int d, int D) {
  if (d <= 0 || D <= 0) return -1;
  return 16LL * D * d * d + (2LL * D + 1) * d;
}

/* First normalisation-gain coordinate. */
int64_t oracle_body_gain_offset(int d, int D) { return 16LL * D * d * d; }

/* Probe entries [p0, p0 + count) of the body's coordinates (file header). */
int oracle_body_probe(uint64_t seed, uint64_t step, uint32_t expert, uint32_t probe, int kind,
                      int d, int D, int64_t p0, int64_t count, int8_t* z) {
  if (kind != 0 && kind != 1) return 1;
  if (oracle_probe(seed, step, expert, probe, kind, p0, count, z)) return 2;
  if (kind == 1) {
    int64_t g0 = oracle_body_gain_offset(d, D);
    int64_t from = p0 > g0 ? p0 : g0;
    if (from < p0 + count) /* gains: the dense sign */
      if (oracle_probe(seed, step, expert, probe, 0, from, p0 + count - from, z + (from - p0)))
        return 2;
  }
  return 0;
}

typedef struct {
  const double *w_ih, *w_hh, *w1, *w2; /* block k: add k * 16 d^2 */
  const double *ga, *gb, *gf;          /* block k: add k * 2d to ga, gb */
} body_view;

static body_view view_body(const double* theta, int d, int D) {
  body_view v;
  int64_t q = (int64_t)d * d;
  v.w_ih = theta;
  v.w_hh = theta + 4 * q;
  v.w1 = theta + 8 * q;
  v.w2 = theta + 12 * q;
  v.ga = theta + 16LL * D * q;
  v.gb = v.ga + d;
  v.gf = v.ga + 2LL * D * d;
  return v;
}

static double sigm(double a) { return 1.0 / (1.0 + exp(-a)); }

/* out = (x - mean) / sqrt(var + eps) * g over d features */
static void layer_norm(const double* x, const double* g, int d, double* out) {
  double mu = 0.0;
  for (int k = 0; k < d; ++k) mu += x[k];
  mu /= d;
  double var = 0.0;
  for (int k = 0; k < d; ++k) var += (x[k] - mu) * (x[k] - mu);
  var /= d;
  double r = 1.0 / sqrt(var + BODY_LN_EPS);
  for (int k = 0; k < d; ++k) out[k] = (x[k] - mu) * r * g[k];
}

static double gelu(double a) { return 0.5 * a * (1.0 + erf(a / sqrt(2.0))); }

/* Sum of the next-byte NLLs of one sequence of T+1 bytes.
 * Scratch: d (x) + d (u) + 2 D d (h, c) + 4d (a or MLP hidden) + d (h new) + V. */
static double body_sequence_nll(const body_view* m, int d, int D, const double* head,
                                const uint8_t* seq, int T, double* scratch, double* nll_out) {
  double* x = scratch;
  double* u = x + d;
  double* h = u + d;             /* [D][d] */
  double* c = h + (int64_t)D * d; /* [D][d] */
  double* a = c + (int64_t)D * d; /* 4d */
  double* hn = a + 4 * d;        /* d */
  double* logit = hn + d;        /* V */
  int64_t blk = 16LL * d * d;
  for (int q = 0; q < 2 * D * d; ++q) h[q] = 0.0; /* h and c, every block */
  double total = 0.0;
  for (int t = 0; t < T; ++t) {
    for (int k = 0; k < d; ++k) x[k] = head[(int64_t)seq[t] * d + k];
    for (int b = 0; b < D; ++b) {
      const double* w_ih = m->w_ih + b * blk;
      const double* w_hh = m->w_hh + b * blk;
      const double* w1 = m->w1 + b * blk;
      const double* w2 = m->w2 + b * blk;
      double* hb = h + (int64_t)b * d;
      double* cb = c + (int64_t)b * d;
      /* LSTM sublayer on the normalised stream */
      layer_norm(x, m->ga + 2LL * b * d, d, u);
      for (int r = 0; r < 4 * d; ++r) {
        double s = 0.0;
        for (int k = 0; k < d; ++k) s += w_ih[(int64_t)r * d + k] * u[k];
        for (int k = 0; k < d; ++k) s += w_hh[(int64_t)r * d + k] * hb[k];
        a[r] = s;
      }
      for (int j = 0; j < d; ++j) {
        double ig = sigm(a[j]), fg = sigm(a[d + j]);
        double gg = tanh(a[2 * d + j]), og = sigm(a[3 * d + j]);
        cb[j] = fg * cb[j] + ig * gg;
        hn[j] = og * tanh(cb[j]);
      }
      for (int j = 0; j < d; ++j) { hb[j] = hn[j]; x[j] += hn[j]; }
      /* MLP sublayer */
      layer_norm(x, m->gb + 2LL * b * d, d, u);
      for (int r = 0; r < 4 * d; ++r) {
        double s = 0.0;
        for (int k = 0; k < d; ++k) s += w1[(int64_t)r * d + k] * u[k];
        a[r] = gelu(s);
      }
      for (int j = 0; j < d; ++j) {
        double s = 0.0;
        for (int k = 0; k < 4 * d; ++k) s += w2[(int64_t)j * 4 * d + k] * a[k];
        x[j] += s;
      }
    }
    /* final norm, tied decode and cross entropy */
    layer_norm(x, m->gf, d, u);
    double mx = -INFINITY;
    for (int v = 0; v < BODY_V; ++v) {
      double s = 0.0;
      for (int k = 0; k < d; ++k) s += head[(int64_t)v * d + k] * u[k];
      logit[v] = s;
      if (s > mx) mx = s;
    }
    double se = 0.0;
    for (int v = 0; v < BODY_V; ++v) se += exp(logit[v] - mx);
    double nll = mx + log(se) - logit[seq[t + 1]];
    if (nll_out) nll_out[t] = nll;
    total += nll;
  }
  return total;
}

static int body_threads(int requested) {
#ifdef _OPENMP
  if (requested > 0) return requested;
  return omp_get_max_threads();
#else
  (void)requested;
  return 1;
#endif
}

/* Mean cross entropy (nats/byte) of one expert body over B sequences of
 * T+1 bytes; head is E [V][d].  nll_out, if not NULL, receives [B][T]. */
double oracle_body_loss(const double* theta, int d, int D, const double* head,
                        const uint8_t* bytes, int B, int T, double* nll_out, int n_threads) {
  if (d <= 0 || D <= 0 || B <= 0 || T <= 0) return NAN;
  body_view m = view_body(theta, d, D);
  double* per_seq = (double*)calloc((size_t)B, sizeof(double));
  int nt = body_threads(n_threads);
#pragma omp parallel for schedule(dynamic, 1) num_threads(nt)
  for (int b = 0; b < B; ++b) {
    double* scratch = (double*)malloc(sizeof(double) * (size_t)(8 * d + 2 * D * d + BODY_V));
    per_seq[b] = body_sequence_nll(&m, d, D, head, bytes + (int64_t)b * (T + 1), T, scratch,
                                   nll_out ? nll_out + (int64_t)b * T : NULL);
    free(scratch);
  }
  double total = 0.0;
  for (int b = 0; b < B; ++b) total += per_seq[b];
  free(per_seq);
  return total / ((double)B * (double)T);
}

/* Antithetic losses of the selected probes (Eq. localspsa's estimator with
 * the frozen head E).  theta [N][P_body], bytes [N][B][T+1] shared by every
 * probe and both signs, head [V][d].  Row e is expert e0 + e.
 *   out_L [N][n_sel][2] = L(theta_e + eps z), L(theta_e - eps z)
 *   out_coef [N][n_sel] = (L+ - L-) / (2 eps); 0 when eps == 0. */
int oracle_body_spsa_losses(const double* theta, int N, int e0, int d, int D,
                            const double* head, double eps, int kind, uint64_t seed,
                            uint64_t step, const uint8_t* bytes, int B, int T,
                            const int32_t* sel, int n_sel, double* out_L, double* out_coef,
                            int n_threads) {
  int64_t P = oracle_body_param_count(d, D);
  if (P <= 0 || N <= 0 || B <= 0 || T <= 0 || n_sel < 0 || (kind != 0 && kind != 1)) return 1;
  double* theta_s = (double*)malloc(sizeof(double) * (size_t)P);
  int8_t* z = (int8_t*)malloc((size_t)P);
  if (!theta_s || !z) { free(theta_s); free(z); return 2; }
  for (int e = 0; e < N; ++e) {
    const double* th = theta + (int64_t)e * P;
    const uint8_t* bx = bytes + (int64_t)e * B * (T + 1);
    for (int q = 0; q < n_sel; ++q) {
      oracle_body_probe(seed, step, (uint32_t)(e0 + e), (uint32_t)sel[q], kind, d, D, 0, P, z);
      double L[2];
      for (int s = 0; s < 2; ++s) {
        double sign = (s == 0) ? 1.0 : -1.0;
        for (int64_t p = 0; p < P; ++p) theta_s[p] = th[p] + sign * eps * (double)z[p];
        L[s] = oracle_body_loss(theta_s, d, D, head, bx, B, T, NULL, n_threads);
      }
      out_L[((int64_t)e * n_sel + q) * 2 + 0] = L[0];
      out_L[((int64_t)e * n_sel + q) * 2 + 1] = L[1];
      out_coef[(int64_t)e * n_sel + q] = (eps == 0.0) ? 0.0 : (L[0] - L[1]) / (2.0 * eps);
    }
  }
  free(theta_s);
  free(z);
  return 0;
}

/* theta_out = theta - lr * (1/n_pert) sum_i coef[e][i] z_{e,i}, fp64, with
 * probes of the given kind.  coef [N][n_pert]. */
int oracle_body_spsa_update(const double* theta, int N, int d, int D, int n_pert, int kind,
                            double lr, uint64_t seed, uint64_t step, const double* coef,
                            double* theta_out) {
  int64_t P = oracle_body_param_count(d, D);
  if (P <= 0 || N <= 0 || n_pert <= 0 || (kind != 0 && kind != 1)) return 1;
  double* g = (double*)malloc(sizeof(double) * (size_t)P);
  int8_t* z = (int8_t*)malloc((size_t)P);
  if (!g || !z) { free(g); free(z); return 2; }
  for (int e = 0; e < N; ++e) {
    for (int64_t p = 0; p < P; ++p) g[p] = 0.0;
    for (int i = 0; i < n_pert; ++i) {
      double ci = coef[(int64_t)e * n_pert + i];
      oracle_body_probe(seed, step, (uint32_t)e, (uint32_t)i, kind, d, D, 0, P, z);
      for (int64_t p = 0; p < P; ++p) g[p] += ci * (double)z[p];
    }
    const double* th = theta + (int64_t)e * P;
    double* to = theta_out + (int64_t)e * P;
    for (int64_t p = 0; p < P; ++p) to[p] = th[p] - lr * (g[p] / (double)n_pert);
  }
  free(g);
  free(z);
  return 0;
}

/* The paper's optimizer step (Eq. localspsa, coupled weight decay before the
 * moments, bias-corrected Adam) on the body coordinates, in fp64.
 * theta, m, v [N][P]; coef [A][N][n_pert]; steps[A] the probe step counters. */
int oracle_body_adam_update(const double* theta, const double* m, const double* v, int N, int d,
                            int D, int n_pert, int kind, uint64_t seed, const uint64_t* steps,
                            int A, const double* coef, double lr, double beta1, double beta2,
                            double delta, double wd, int t, double* theta_out, double* m_out,
                            double* v_out) {
  int64_t P = oracle_body_param_count(d, D);
  if (P <= 0 || N <= 0 || n_pert <= 0 || A <= 0 || t < 1 || (kind != 0 && kind != 1)) return 1;
  double* g = (double*)malloc(sizeof(double) * (size_t)P);
  int8_t* z = (int8_t*)malloc((size_t)P);
  if (!g || !z) { free(g); free(z); return 2; }
  double bc1 = 1.0 - pow(beta1, (double)t), bc2 = 1.0 - pow(beta2, (double)t);
  for (int e = 0; e < N; ++e) {
    for (int64_t p = 0; p < P; ++p) g[p] = 0.0;
    for (int a = 0; a < A; ++a)
      for (int i = 0; i < n_pert; ++i) {
        double ci = coef[((int64_t)a * N + e) * n_pert + i];
        oracle_body_probe(seed, steps[a], (uint32_t)e, (uint32_t)i, kind, d, D, 0, P, z);
        for (int64_t p = 0; p < P; ++p) g[p] += ci * (double)z[p];
      }
    const double* th = theta + (int64_t)e * P;
    const double* me = m + (int64_t)e * P;
    const double* ve = v + (int64_t)e * P;
    double* to = theta_out + (int64_t)e * P;
    double* mo = m_out + (int64_t)e * P;
    double* vo = v_out + (int64_t)e * P;
    for (int64_t p = 0; p < P; ++p) {
      double gp = g[p] / ((double)A * (double)n_pert) + wd * th[p];
      double mp = beta1 * me[p] + (1.0 - beta1) * gp;
      double vp = beta2 * ve[p] + (1.0 - beta2) * gp * gp;
      mo[p] = mp;
      vo[p] = vp;
      to[p] = th[p] - lr * (mp / bc1) / (sqrt(vp / bc2) + delta);
    }
  }
  free(g);
  free(z);
  return 0;
}
