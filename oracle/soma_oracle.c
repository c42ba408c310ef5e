/*
 * soma_oracle.c -- fp64 CPU oracle for the SOMA SPSA training step.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing in the product path may call, link or
 * load this file; only the tests, the smoke check and the timed CPU baseline
 * of bench.py do.  It shares no code, header, table or helper with the CUDA
 * library: its Philox generator, its LSTM and its update are written here,
 * independently, in the plainest form that can be checked against the paper
 * by eye.  Every loop follows the definition in the order the paper states it;
 * there is no blocking, fusion or reordering.
 *
 * What it computes (paper: "Scaling Zero-Order Pretraining through Model
 * Sharding"):
 *   - the perturbation probes z_j in {-1,+1}^d (Sec. 4, Eq. main-spsa: dense
 *     Rademacher probes), drawn from Philox4x32-10 (Salmon et al., SC'11) so
 *     that they can be regenerated from (seed, step, expert, probe);
 *   - the expert model: byte embedding -> one LSTM layer -> linear head to the
 *     256-byte vocabulary, hidden state reset to zero for every sequence
 *     (Sec. 3, App. C; state reset per window, Sec. 6 "Evaluation");
 *   - the loss: mean next-byte cross entropy in nats/byte over all scored
 *     targets (Table experimental-setup, "Evaluation protocol"; App. E, the
 *     L_CE form log-sum-exp minus the target logit);
 *   - the antithetic losses L(theta + eps z_j), L(theta - eps z_j) on one
 *     shared batch, their coefficients (L+ - L-)/(2 eps) and the update
 *     theta <- theta - lr * (1/n_pert) sum_j coef_j z_j (Eq. main-spsa; the
 *     plain-SGD form of Eq. localspsa without moments);
 *   - the exact batch gradient by back-propagation through time (used only
 *     to pin the epsilon -> 0 limit of the estimator, App. F, Prop. 1 proof);
 *   - the paper's own optimizer step (App. E, Eq. localspsa): sparse
 *     Rademacher probes (a coordinate is 0 with probability 1/2 and -1 or +1
 *     with probability 1/4 each), the estimate averaged over A accumulation
 *     batches, coupled weight decay added before the moments, and Adam with
 *     bias-corrected moments;
 *   - routed inference: the average of the routed experts' next-byte
 *     probabilities (Sec. 3, Eq. main-mixture).
 *
 * Parameter layout of one expert (flat, row-major, gate blocks i,f,g,o):
 *   Emb[V][E], W_ih[4H][E], W_hh[4H][H], b[4H], W_out[V][H], b_out[V].
 *
 * Probe stream: z for flat parameter index p of expert e, probe i, at update
 * `step`, under `seed`:
 *   key     = (seed & 0xffffffff, seed >> 32)
 *   counter = (p >> 7, i, step & 0xffffffff, e)
 *   w[0..3] = Philox4x32-10(counter, key)
 *   o       = p & 31  (position inside the 32-parameter run of one word)
 *   bit     = (w[(p & 127) >> 5] >> ((o >> 1) + 16 * (o & 1))) & 1
 *   z       = 1 - 2 * bit.
 * Within each word, parameters 2j and 2j+1 of the run read bits j and
 * j + 16: an even/odd interleave of the two 16-bit halves.
 *
 * Sparse probes (App. E) use two bits per coordinate from the same key,
 * step and expert: the sign bit above, and an activity bit taken at the same
 * position of the block whose counter word 1 is probe | 0x80000000.
 *   z = (activity bit set) ? 1 - 2 * bit : 0.
 * A coordinate is therefore nonzero with probability 1/2, and a nonzero
 * sparse coordinate equals the dense probe's coordinate.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

#define SOMA_V 256

/* ------------------------------------------------------------------ */
/* Philox4x32-10, from its published definition (Salmon, Moraes, Dror, */
/* Shaw, "Parallel random numbers: as easy as 1, 2, 3", SC'11, Sec. 4). */
/* ------------------------------------------------------------------ */

/* Round multipliers and Weyl key increments of Philox4x32 (SC'11, Table 2
 * and the key schedule "add the golden ratio and sqrt(3)-1" constants). */
static const uint32_t PHILOX_M0 = 0xD2511F53u;
static const uint32_t PHILOX_M1 = 0xCD9E8D57u;
static const uint32_t PHILOX_W0 = 0x9E3779B9u;
static const uint32_t PHILOX_W1 = 0xBB67AE85u;

void oracle_philox4x32_10(const uint32_t ctr_in[4], const uint32_t key_in[2],
                          uint32_t out[4]) {
  uint32_t x0 = ctr_in[0], x1 = ctr_in[1], x2 = ctr_in[2], x3 = ctr_in[3];
  uint32_t k0 = key_in[0], k1 = key_in[1];
  for (int round = 0; round < 10; ++round) {
    /* One Philox S-box round: two 32x32->64 products, the high halves
     * xor-ed with the other two words and the round key. */
    uint64_t p0 = (uint64_t)PHILOX_M0 * (uint64_t)x0;
    uint64_t p1 = (uint64_t)PHILOX_M1 * (uint64_t)x2;
    uint32_t hi0 = (uint32_t)(p0 >> 32), lo0 = (uint32_t)p0;
    uint32_t hi1 = (uint32_t)(p1 >> 32), lo1 = (uint32_t)p1;
    uint32_t y0 = hi1 ^ x1 ^ k0;
    uint32_t y1 = lo1;
    uint32_t y2 = hi0 ^ x3 ^ k1;
    uint32_t y3 = lo0;
    x0 = y0; x1 = y1; x2 = y2; x3 = y3;
    /* Key schedule: bump the key by the Weyl constants between rounds. */
    k0 += PHILOX_W0;
    k1 += PHILOX_W1;
  }
  out[0] = x0; out[1] = x1; out[2] = x2; out[3] = x3;
}

/* z_{e,i}[p] for p in [p0, p0 + count): one Philox call per parameter,
 * exactly as the mapping in the file header states (no caching). */
void oracle_rademacher(uint64_t seed, uint64_t step, uint32_t expert,
                       uint32_t probe, int64_t p0, int64_t count, int8_t* z) {
  uint32_t key[2] = {(uint32_t)(seed & 0xffffffffu), (uint32_t)(seed >> 32)};
  for (int64_t q = 0; q < count; ++q) {
    int64_t p = p0 + q;
    uint32_t ctr[4] = {(uint32_t)(p >> 7), probe,
                       (uint32_t)(step & 0xffffffffu), expert};
    uint32_t w[4];
    oracle_philox4x32_10(ctr, key, w);
    int k = (int)(p & 127);
    int o = k & 31;
    uint32_t bit = (w[k >> 5] >> ((o >> 1) + 16 * (o & 1))) & 1u;
    z[q] = (int8_t)(1 - 2 * (int)bit);
  }
}

/* z_{e,i}[p] for p in [p0, p0 + count) of the given kind: 0 = dense
 * Rademacher (as above), 1 = sparse (file header).  One Philox call per
 * parameter and stream, no caching. */
int oracle_probe(uint64_t seed, uint64_t step, uint32_t expert, uint32_t probe, int kind,
                 int64_t p0, int64_t count, int8_t* z) {
  if (kind != 0 && kind != 1) return 1;
  oracle_rademacher(seed, step, expert, probe, p0, count, z);
  if (kind == 0) return 0;
  int8_t* act = (int8_t*)malloc((size_t)(count > 0 ? count : 1));
  if (!act) return 2;
  /* the activity stream: same bit map, counter word 1 with its top bit set */
  oracle_rademacher(seed, step, expert, probe | 0x80000000u, p0, count, act);
  for (int64_t q = 0; q < count; ++q)
    if (act[q] == 1) z[q] = 0; /* bit 0 (z would be +1): inactive */
  free(act);
  return 0;
}

/* ------------------------------------------------------------------ */
/* Model                                                               */
/* ------------------------------------------------------------------ */

int64_t oracle_param_count(int E, int H) {
  if (E <= 0 || H <= 0) return -1;
  int64_t V = SOMA_V;
  return V * E + 4LL * H * E + 4LL * H * H + 4LL * H + V * H + V;
}

typedef struct {
  const double *emb, *w_ih, *w_hh, *b, *w_out, *b_out;
} lstm_view;

static lstm_view view_params(const double* theta, int E, int H) {
  lstm_view v;
  int64_t V = SOMA_V;
  v.emb = theta;
  v.w_ih = v.emb + V * E;
  v.w_hh = v.w_ih + 4LL * H * E;
  v.b = v.w_hh + 4LL * H * H;
  v.w_out = v.b + 4LL * H;
  v.b_out = v.w_out + V * H;
  return v;
}

static double sigmoid(double a) { return 1.0 / (1.0 + exp(-a)); }

/* Sum of the next-byte negative log-likelihoods of one sequence of T+1
 * bytes, hidden and cell state starting at zero.  Scratch: 4H + 3H + V. */
static double sequence_nll_sum(const lstm_view* m, int E, int H,
                               const uint8_t* seq, int T, double* scratch,
                               double* nll_out) {
  double* a = scratch;           /* 4H gate pre-activations */
  double* h = a + 4 * H;         /* H */
  double* c = h + H;             /* H */
  double* hn = c + H;            /* H: h_t while h_{t-1} is still read */
  double* logit = hn + H;        /* V */
  for (int j = 0; j < H; ++j) { h[j] = 0.0; c[j] = 0.0; }
  double total = 0.0;
  for (int t = 0; t < T; ++t) {
    const double* x = m->emb + (int64_t)seq[t] * E;
    /* a = W_ih x + W_hh h_{t-1} + b */
    for (int r = 0; r < 4 * H; ++r) {
      double s = m->b[r];
      const double* wi = m->w_ih + (int64_t)r * E;
      for (int k = 0; k < E; ++k) s += wi[k] * x[k];
      const double* wh = m->w_hh + (int64_t)r * H;
      for (int k = 0; k < H; ++k) s += wh[k] * h[k];
      a[r] = s;
    }
    /* gates in the order i, f, g, o; cell and hidden update */
    for (int j = 0; j < H; ++j) {
      double ig = sigmoid(a[j]);
      double fg = sigmoid(a[H + j]);
      double gg = tanh(a[2 * H + j]);
      double og = sigmoid(a[3 * H + j]);
      c[j] = fg * c[j] + ig * gg;
      hn[j] = og * tanh(c[j]);
    }
    for (int j = 0; j < H; ++j) h[j] = hn[j];
    /* logits = W_out h_t + b_out; nll = logsumexp(logits) - logits[y] */
    double mx = -INFINITY;
    for (int v = 0; v < SOMA_V; ++v) {
      double s = m->b_out[v];
      const double* wo = m->w_out + (int64_t)v * H;
      for (int k = 0; k < H; ++k) s += wo[k] * h[k];
      logit[v] = s;
      if (s > mx) mx = s;
    }
    double se = 0.0;
    for (int v = 0; v < SOMA_V; ++v) se += exp(logit[v] - mx);
    double nll = mx + log(se) - logit[seq[t + 1]];
    if (nll_out) nll_out[t] = nll;
    total += nll;
  }
  return total;
}

static int num_threads(int requested) {
#ifdef _OPENMP
  if (requested > 0) return requested;
  return omp_get_max_threads();
#else
  (void)requested;
  return 1;
#endif
}

/* Mean cross entropy (nats/byte) of one expert over B sequences of T+1
 * bytes.  nll_out, if not NULL, receives the B*T per-target values. */
double oracle_loss(const double* theta, int E, int H, const uint8_t* bytes,
                   int B, int T, double* nll_out, int n_threads) {
  if (B <= 0 || T <= 0) return NAN;
  lstm_view m = view_params(theta, E, H);
  double* per_seq = (double*)calloc((size_t)B, sizeof(double));
  int nt = num_threads(n_threads);
#pragma omp parallel for schedule(dynamic, 1) num_threads(nt)
  for (int b = 0; b < B; ++b) {
    double* scratch = (double*)malloc(sizeof(double) * (size_t)(7 * H + SOMA_V));
    per_seq[b] = sequence_nll_sum(&m, E, H, bytes + (int64_t)b * (T + 1), T,
                                  scratch, nll_out ? nll_out + (int64_t)b * T : NULL);
    free(scratch);
  }
  /* fixed summation order: sequence by sequence */
  double total = 0.0;
  for (int b = 0; b < B; ++b) total += per_seq[b];
  free(per_seq);
  return total / ((double)B * (double)T);
}

/* ------------------------------------------------------------------ */
/* SPSA (Eq. main-spsa)                                                */
/* ------------------------------------------------------------------ */

/* Antithetic losses of the selected probes.
 *   theta [N][P] (fp64), bytes [N][B][T+1] (one batch per expert, shared by
 *   every probe and both signs) or, with batch_per_probe, [N][n_pert][B][T+1]
 *   (one batch per probe, App. D), sel[n_sel] probe indices in [0, n_pert).
 *   summed_loss: the control arm of App. D, whose coefficient for probe sel[q]
 *   is (sum_e L+_e - sum_e L-_e) / (2 eps) for every expert.
 *   Row e of theta is expert e0 + e (its index in the probe counter).
 *   out_L  [N][n_sel][2] = L(theta_e + eps z), L(theta_e - eps z)
 *   out_coef [N][n_sel]  = (L+ - L-) / (2 eps); 0 when eps == 0.
 * Returns 0 on success. */
int oracle_spsa_losses_opts(const double* theta, int N, int e0, int E, int H, double eps,
                            int kind, int batch_per_probe, int summed_loss, int n_pert,
                            uint64_t seed, uint64_t step, const uint8_t* bytes, int B, int T,
                            const int32_t* sel, int n_sel, double* out_L, double* out_coef,
                            int n_threads) {
  int64_t P = oracle_param_count(E, H);
  if (P <= 0 || N <= 0 || B <= 0 || T <= 0 || n_sel < 0 || (kind != 0 && kind != 1)) return 1;
  if (batch_per_probe && n_pert <= 0) return 1;
  double* theta_s = (double*)malloc(sizeof(double) * (size_t)P);
  int8_t* z = (int8_t*)malloc((size_t)P);
  if (!theta_s || !z) { free(theta_s); free(z); return 2; }
  int64_t seq_block = (int64_t)B * (T + 1);
  for (int e = 0; e < N; ++e) {
    const double* th = theta + (int64_t)e * P;
    for (int q = 0; q < n_sel; ++q) {
      int i = sel[q];
      /* one batch per expert (Sec. 4), or one per (expert, probe) */
      const uint8_t* bx = bytes + (batch_per_probe ? ((int64_t)e * n_pert + i) * seq_block
                                                   : (int64_t)e * seq_block);
      oracle_probe(seed, step, (uint32_t)(e0 + e), (uint32_t)i, kind, 0, P, z);
      double L[2];
      for (int s = 0; s < 2; ++s) {
        double sign = (s == 0) ? 1.0 : -1.0;
        for (int64_t p = 0; p < P; ++p) theta_s[p] = th[p] + sign * eps * (double)z[p];
        L[s] = oracle_loss(theta_s, E, H, bx, B, T, NULL, n_threads);
      }
      out_L[((int64_t)e * n_sel + q) * 2 + 0] = L[0];
      out_L[((int64_t)e * n_sel + q) * 2 + 1] = L[1];
      out_coef[(int64_t)e * n_sel + q] = (eps == 0.0) ? 0.0 : (L[0] - L[1]) / (2.0 * eps);
    }
  }
  if (summed_loss) {
    /* the control arm (App. D): the experts' losses are summed, then the
     * finite difference of the sums is every expert's coefficient */
    for (int q = 0; q < n_sel; ++q) {
      double Lp = 0.0, Lm = 0.0;
      for (int e = 0; e < N; ++e) {
        Lp += out_L[((int64_t)e * n_sel + q) * 2 + 0];
        Lm += out_L[((int64_t)e * n_sel + q) * 2 + 1];
      }
      double c = (eps == 0.0) ? 0.0 : (Lp - Lm) / (2.0 * eps);
      for (int e = 0; e < N; ++e) out_coef[(int64_t)e * n_sel + q] = c;
    }
  }
  free(theta_s);
  free(z);
  return 0;
}

/* Antithetic losses of the selected probes with probe kind `kind`, one batch
 * per expert shared by every probe, each expert's own loss. */
int oracle_spsa_losses_kind(const double* theta, int N, int e0, int E, int H, double eps,
                            int kind, uint64_t seed, uint64_t step, const uint8_t* bytes,
                            int B, int T, const int32_t* sel, int n_sel,
                            double* out_L, double* out_coef, int n_threads) {
  return oracle_spsa_losses_opts(theta, N, e0, E, H, eps, kind, 0, 0, 0, seed, step, bytes, B, T,
                                 sel, n_sel, out_L, out_coef, n_threads);
}

/* The same with dense probes (Eq. main-spsa). */
int oracle_spsa_losses(const double* theta, int N, int e0, int E, int H, double eps,
                       uint64_t seed, uint64_t step, const uint8_t* bytes,
                       int B, int T, const int32_t* sel, int n_sel,
                       double* out_L, double* out_coef, int n_threads) {
  return oracle_spsa_losses_kind(theta, N, e0, E, H, eps, 0, seed, step, bytes, B, T, sel,
                                 n_sel, out_L, out_coef, n_threads);
}

/* theta_out = theta - lr * (1/n_pert) * sum_i coef[e][i] z_{e,i}, in fp64.
 * coef [N][n_pert]; theta, theta_out [N][P]. */
int oracle_spsa_update(const double* theta, int N, int E, int H, int n_pert,
                       double lr, uint64_t seed, uint64_t step,
                       const double* coef, double* theta_out) {
  int64_t P = oracle_param_count(E, H);
  if (P <= 0 || N <= 0 || n_pert <= 0) return 1;
  double* g = (double*)malloc(sizeof(double) * (size_t)P);
  int8_t* z = (int8_t*)malloc((size_t)P);
  if (!g || !z) { free(g); free(z); return 2; }
  for (int e = 0; e < N; ++e) {
    for (int64_t p = 0; p < P; ++p) g[p] = 0.0;
    for (int i = 0; i < n_pert; ++i) {
      double ci = coef[(int64_t)e * n_pert + i];
      oracle_rademacher(seed, step, (uint32_t)e, (uint32_t)i, 0, P, z);
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

/* The paper's optimizer step (App. E, Eq. localspsa), in fp64, for every
 * expert e:
 *   ghat[p]  = (1/A) sum_a (1/n_pert) sum_i coef[a][e][i] z_{e,i}^{(a)}[p],
 *              z^{(a)} drawn with step counter steps[a] (kind 0 dense, 1 sparse)
 *   g        = ghat + wd * theta            (coupled weight decay, before the moments)
 *   m        = beta1 m + (1 - beta1) g,     v = beta2 v + (1 - beta2) g^2
 *   mhat     = m / (1 - beta1^t),           vhat = v / (1 - beta2^t)
 *   theta'   = theta - lr * mhat / (sqrt(vhat) + delta)
 * t >= 1 is the update count (m = v = 0 before the first update).
 * theta, m, v and the outputs are [N][P]; coef is [A][N][n_pert]. */
int oracle_adam_update(const double* theta, const double* m, const double* v, int N, int E,
                       int H, int n_pert, int kind, uint64_t seed, const uint64_t* steps, int A,
                       const double* coef, double lr, double beta1, double beta2, double delta,
                       double wd, int t, double* theta_out, double* m_out, double* v_out) {
  int64_t P = oracle_param_count(E, H);
  if (P <= 0 || N <= 0 || n_pert <= 0 || A <= 0 || t < 1 || (kind != 0 && kind != 1)) return 1;
  double* g = (double*)malloc(sizeof(double) * (size_t)P);
  int8_t* z = (int8_t*)malloc((size_t)P);
  if (!g || !z) { free(g); free(z); return 2; }
  double bc1 = 1.0 - pow(beta1, (double)t), bc2 = 1.0 - pow(beta2, (double)t);
  for (int e = 0; e < N; ++e) {
    for (int64_t p = 0; p < P; ++p) g[p] = 0.0;
    for (int a = 0; a < A; ++a) {
      for (int i = 0; i < n_pert; ++i) {
        double ci = coef[((int64_t)a * N + e) * n_pert + i];
        oracle_probe(seed, steps[a], (uint32_t)e, (uint32_t)i, kind, 0, P, z);
        for (int64_t p = 0; p < P; ++p) g[p] += ci * (double)z[p];
      }
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

/* Routed inference (Sec. 3, Eq. main-mixture), in fp64: request r is read by
 * its k routed experts routes[r][j] (state reset to zero), and
 *   out[r][t - t0] = -log( (1/k) sum_j p_{routes[r][j]}(byte_{t+1} | bytes_<=t) )
 * for t0 <= t < T.  theta [N][P], requests [R][T+1]. */
int oracle_mixture_nll(const double* theta, int N, int E, int H, const uint8_t* requests, int R,
                       int T, const int32_t* routes, int k, int t0, double* out, int n_threads) {
  int64_t P = oracle_param_count(E, H);
  if (P <= 0 || N <= 0 || R <= 0 || T <= 0 || k <= 0 || t0 < 0 || t0 >= T) return 1;
  double* nll = (double*)malloc(sizeof(double) * (size_t)k * T);
  if (!nll) return 2;
  for (int r = 0; r < R; ++r) {
    const uint8_t* seq = requests + (int64_t)r * (T + 1);
    for (int j = 0; j < k; ++j) {
      int e = routes[(int64_t)r * k + j];
      if (e < 0 || e >= N) { free(nll); return 1; }
      oracle_loss(theta + (int64_t)e * P, E, H, seq, 1, T, nll + (int64_t)j * T, n_threads);
    }
    for (int t = t0; t < T; ++t) {
      double p = 0.0;
      for (int j = 0; j < k; ++j) p += exp(-nll[(int64_t)j * T + t]);
      out[(int64_t)r * (T - t0) + (t - t0)] = -log(p / (double)k);
    }
  }
  free(nll);
  return 0;
}

/* ------------------------------------------------------------------ */
/* Exact batch gradient by back-propagation through time (fp64).       */
/* Used only to pin the eps -> 0 limit: (L+ - L-)/(2 eps) -> g . z.    */
/* ------------------------------------------------------------------ */

double oracle_bptt_grad(const double* theta, int E, int H, const uint8_t* bytes,
                        int B, int T, double* grad) {
  int64_t P = oracle_param_count(E, H);
  int64_t V = SOMA_V;
  lstm_view m = view_params(theta, E, H);
  for (int64_t p = 0; p < P; ++p) grad[p] = 0.0;
  double* g_emb = grad;
  double* g_wih = g_emb + V * E;
  double* g_whh = g_wih + 4LL * H * E;
  double* g_b = g_whh + 4LL * H * H;
  double* g_wout = g_b + 4LL * H;
  double* g_bout = g_wout + V * H;

  /* per-step storage of one sequence: gates i,f,g,o, c_t, h_t (t = 0..T,
   * index 0 holding the zero initial state for c and h) */
  double* gi = (double*)malloc(sizeof(double) * (size_t)T * H);
  double* gf = (double*)malloc(sizeof(double) * (size_t)T * H);
  double* gg = (double*)malloc(sizeof(double) * (size_t)T * H);
  double* go = (double*)malloc(sizeof(double) * (size_t)T * H);
  double* cs = (double*)malloc(sizeof(double) * (size_t)(T + 1) * H);
  double* hs = (double*)malloc(sizeof(double) * (size_t)(T + 1) * H);
  double* prob = (double*)malloc(sizeof(double) * (size_t)T * V);
  double* a = (double*)malloc(sizeof(double) * (size_t)4 * H);
  double* da = (double*)malloc(sizeof(double) * (size_t)4 * H);
  double* dh = (double*)malloc(sizeof(double) * (size_t)H);
  double* dh_rec = (double*)malloc(sizeof(double) * (size_t)H);
  double* dc_next = (double*)malloc(sizeof(double) * (size_t)H);
  double* dlogit = (double*)malloc(sizeof(double) * (size_t)V);
  double total = 0.0;
  double scale = 1.0 / ((double)B * (double)T);

  for (int b = 0; b < B; ++b) {
    const uint8_t* seq = bytes + (int64_t)b * (T + 1);
    for (int j = 0; j < H; ++j) { cs[j] = 0.0; hs[j] = 0.0; }
    /* forward, keeping every intermediate */
    for (int t = 0; t < T; ++t) {
      const double* x = m.emb + (int64_t)seq[t] * E;
      const double* hp = hs + (int64_t)t * H;
      for (int r = 0; r < 4 * H; ++r) {
        double s = m.b[r];
        for (int k = 0; k < E; ++k) s += m.w_ih[(int64_t)r * E + k] * x[k];
        for (int k = 0; k < H; ++k) s += m.w_hh[(int64_t)r * H + k] * hp[k];
        a[r] = s;
      }
      double* cp = cs + (int64_t)t * H;
      double* cn = cs + (int64_t)(t + 1) * H;
      double* hn = hs + (int64_t)(t + 1) * H;
      for (int j = 0; j < H; ++j) {
        gi[(int64_t)t * H + j] = sigmoid(a[j]);
        gf[(int64_t)t * H + j] = sigmoid(a[H + j]);
        gg[(int64_t)t * H + j] = tanh(a[2 * H + j]);
        go[(int64_t)t * H + j] = sigmoid(a[3 * H + j]);
        cn[j] = gf[(int64_t)t * H + j] * cp[j] + gi[(int64_t)t * H + j] * gg[(int64_t)t * H + j];
        hn[j] = go[(int64_t)t * H + j] * tanh(cn[j]);
      }
      double* pr = prob + (int64_t)t * V;
      double mx = -INFINITY;
      for (int v = 0; v < V; ++v) {
        double s = m.b_out[v];
        for (int k = 0; k < H; ++k) s += m.w_out[(int64_t)v * H + k] * hn[k];
        pr[v] = s;
        if (s > mx) mx = s;
      }
      double se = 0.0;
      for (int v = 0; v < V; ++v) se += exp(pr[v] - mx);
      double lse = mx + log(se);
      total += lse - pr[seq[t + 1]];
      for (int v = 0; v < V; ++v) pr[v] = exp(pr[v] - lse); /* softmax */
    }
    /* backward through time */
    for (int j = 0; j < H; ++j) { dh_rec[j] = 0.0; dc_next[j] = 0.0; }
    for (int t = T - 1; t >= 0; --t) {
      const double* hn = hs + (int64_t)(t + 1) * H;
      const double* hp = hs + (int64_t)t * H;
      const double* cn = cs + (int64_t)(t + 1) * H;
      const double* cp = cs + (int64_t)t * H;
      const double* pr = prob + (int64_t)t * V;
      /* d loss / d logits = (softmax - onehot(y_{t+1})) / (B T) */
      for (int v = 0; v < V; ++v) dlogit[v] = pr[v] * scale;
      dlogit[seq[t + 1]] -= scale;
      for (int j = 0; j < H; ++j) dh[j] = dh_rec[j];
      for (int v = 0; v < V; ++v) {
        g_bout[v] += dlogit[v];
        for (int k = 0; k < H; ++k) {
          g_wout[(int64_t)v * H + k] += dlogit[v] * hn[k];
          dh[k] += m.w_out[(int64_t)v * H + k] * dlogit[v];
        }
      }
      for (int j = 0; j < H; ++j) {
        double ig = gi[(int64_t)t * H + j], fg = gf[(int64_t)t * H + j];
        double ggv = gg[(int64_t)t * H + j], og = go[(int64_t)t * H + j];
        double tc = tanh(cn[j]);
        double d_o = dh[j] * tc;
        double dc = dh[j] * og * (1.0 - tc * tc) + dc_next[j];
        double d_i = dc * ggv;
        double d_g = dc * ig;
        double d_f = dc * cp[j];
        da[j] = d_i * ig * (1.0 - ig);
        da[H + j] = d_f * fg * (1.0 - fg);
        da[2 * H + j] = d_g * (1.0 - ggv * ggv);
        da[3 * H + j] = d_o * og * (1.0 - og);
        dc_next[j] = dc * fg;
      }
      const double* x = m.emb + (int64_t)seq[t] * E;
      double* gx = g_emb + (int64_t)seq[t] * E;
      for (int j = 0; j < H; ++j) dh_rec[j] = 0.0;
      for (int r = 0; r < 4 * H; ++r) {
        g_b[r] += da[r];
        for (int k = 0; k < E; ++k) {
          g_wih[(int64_t)r * E + k] += da[r] * x[k];
          gx[k] += m.w_ih[(int64_t)r * E + k] * da[r];
        }
        for (int k = 0; k < H; ++k) {
          g_whh[(int64_t)r * H + k] += da[r] * hp[k];
          dh_rec[k] += m.w_hh[(int64_t)r * H + k] * da[r];
        }
      }
    }
  }
  free(gi); free(gf); free(gg); free(go); free(cs); free(hs); free(prob);
  free(a); free(da); free(dh); free(dh_rec); free(dc_next); free(dlogit);
  return total * scale;
}
