/*
 * GBLA layer-core forward: plain fp64 CPU oracle.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing on the product path may include, link or
 * call this file: only the tests, the smoke check and the bench's CPU-baseline
 * leg use it.  It shares no code, header, constant or helper with the CUDA
 * library; the two are written independently from the paper.
 *
 * Paper: "Gated Bidirectional Linear Attention for Generative Retrieval",
 * Sec. 2 (bidirectional linear attention, Eq. bla) and Sec. 2.1 (GBLA:
 * Conv1D, key gating, gated RMSNorm; multi-head paragraph).
 *
 * Everything is computed in double precision with straightforward loops in
 * the order the paper states the layer:
 *   1. Conv1D          x~ = Conv1D(x)       (Sec. 2.1 item 1)
 *   2. feature map     phi(x) = elu(x) + 1  (Sec. 2, BLA paragraph)
 *   3. key gate        g = softmax over the sequence of the gate logits
 *                                           (Sec. 2.1 item 2)
 *   4. state           S = K^T V,  z = K^T 1 with K^ = g * phi(K~)
 *                                           (Sec. 2.1 item 2, matrix form)
 *   5. readout         O_i = phi(q~_i)^T S / phi(q~_i)^T z
 *   6. gated RMSNorm   y = RmsNorm(O) * SiLU(out_gate)   (Sec. 2.1 item 3)
 *
 * Readings of the paper that the text leaves open (each one is a choice, not
 * something the paper fixes):
 *   - phi is elu(x)+1 with alpha = 1, applied to q~ and k~ (the paper gives it
 *     as the example feature map of BLA and does not restate it for GBLA).
 *   - The conv is depthwise and causal over the sequence, width W, left zero
 *     padding, no bias, no activation.  Tap i multiplies x[t-(W-1)+i], so tap
 *     W-1 multiplies the current token (cross-correlation order).  The core
 *     takes projected q, k, v, so each of their channels is convolved with its
 *     own taps; with one kernel shared by all channels this equals convolving
 *     X before the projections, because both are linear maps on different axes.
 *   - The gate and the output-gate input arrive already derived from X~; the
 *     core does not convolve them.
 *   - The gate softmax runs over the valid positions j < L of one (batch, head).
 *   - RmsNorm(O)_d = O_d / sqrt(mean_d O_d^2 + eps) * w_d, weight per head.
 *   - SiLU(x) = x * sigmoid(x).
 *
 * The layer front end (oracle_gbla_project, at the end of this file) takes
 * the embedded sequence X instead: it runs the Conv1D on X, as Sec. 2.1 item 1
 * states it, and then the per-head projections Q, K, V, W_R and w_g.
 *
 * Ablation switches follow the paper's ablation table (W/o Conv1D, W/o key
 * gating, W/o gated RMSNorm; all three off gives plain BLA, Eq. bla).
 */
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define ORACLE_NO_CONV 1 /* identity Conv1D:   x~ = x                   */
#define ORACLE_NO_GATE 2 /* uniform key gate:  g_j = 1/L                */
#define ORACLE_NO_NORM 4 /* no gated RMSNorm:  y = O                    */

/* Feature map, Sec. 2: phi(x) = elu(x) + 1, strictly positive. */
double oracle_phi(double x) { return x > 0.0 ? x + 1.0 : exp(x); }

/* SiLU(x) = x * sigmoid(x), Sec. 2.1 item 3. */
double oracle_silu(double x) { return x / (1.0 + exp(-x)); }

/*
 * Conv1D, Sec. 2.1 item 1: causal depthwise convolution along the sequence.
 *   y[t][c] = sum_{i=0}^{W-1} w[c][i] * x[t-(W-1)+i][c],  x[s] = 0 for s < 0.
 * x: L rows of C channels, row stride ldx (elements).  w: [C][W].  y: [L][C].
 */
void oracle_conv1d(const double *x, long L, int C, long ldx, const double *w,
                   int W, double *y) {
  for (long t = 0; t < L; ++t)
    for (int c = 0; c < C; ++c) {
      double acc = 0.0;
      for (int i = 0; i < W; ++i) {
        long s = t - (W - 1) + i;
        if (s >= 0) acc += w[(long)c * W + i] * x[s * ldx + c];
      }
      y[t * C + c] = acc;
    }
}

/*
 * Key gate, Sec. 2.1 item 2: g = softmax(a) over the L positions of one
 * sequence, with the maximum subtracted before exponentiating.
 * a: L logits at stride lda.  g: L outputs.
 */
void oracle_softmax(const double *a, long L, long lda, double *g) {
  if (L <= 0) return;
  double m = a[0];
  for (long j = 1; j < L; ++j)
    if (a[j * lda] > m) m = a[j * lda];
  double s = 0.0;
  for (long j = 0; j < L; ++j) {
    g[j] = exp(a[j * lda] - m);
    s += g[j];
  }
  for (long j = 0; j < L; ++j) g[j] /= s;
}

/*
 * Gated RMSNorm of one row, Sec. 2.1 item 3:
 *   y_d = O_d / sqrt(mean_d O_d^2 + eps) * w_d * SiLU(og_d).
 */
void oracle_gated_rmsnorm_row(const double *O, const double *og,
                              const double *w, int D, double eps, double *y) {
  double ms = 0.0;
  for (int d = 0; d < D; ++d) ms += O[d] * O[d];
  ms /= (double)D;
  double r = 1.0 / sqrt(ms + eps);
  for (int d = 0; d < D; ++d) y[d] = O[d] * r * w[d] * oracle_silu(og[d]);
}

/* Steps 1-3 shared by the linear-time and the quadratic form. */
static void gbla_prepare(const double *q, const double *k, const double *v,
                         const double *a, long ld, long lda, long L, int D,
                         const double *wq, const double *wk, const double *wv,
                         int W, int flags, double *qt, double *kt, double *vt,
                         double *g) {
  if (flags & ORACLE_NO_CONV) {
    for (long t = 0; t < L; ++t)
      for (int d = 0; d < D; ++d) {
        qt[t * D + d] = q[t * ld + d];
        kt[t * D + d] = k[t * ld + d];
        vt[t * D + d] = v[t * ld + d];
      }
  } else {
    oracle_conv1d(q, L, D, ld, wq, W, qt);
    oracle_conv1d(k, L, D, ld, wk, W, kt);
    oracle_conv1d(v, L, D, ld, wv, W, vt);
  }
  if (flags & ORACLE_NO_GATE) {
    for (long j = 0; j < L; ++j) g[j] = 1.0 / (double)L;
  } else {
    oracle_softmax(a, L, lda, g);
  }
}

static void gbla_finish(const double *O, const double *og, long ld, long L,
                        int D, const double *norm_w, double eps, int flags,
                        double *y) {
  for (long i = 0; i < L; ++i) {
    if (flags & ORACLE_NO_NORM) {
      for (int d = 0; d < D; ++d) y[i * D + d] = O[i * D + d];
    } else {
      oracle_gated_rmsnorm_row(O + i * D, og + i * ld, norm_w, D, eps,
                               y + i * D);
    }
  }
}

static void *xmalloc(size_t n) { return malloc(n ? n : 1); }

/*
 * One (batch, head) of the GBLA core in the linear-time matrix form of
 * Sec. 2.1 item 2:  S = K^T V,  z = K^T 1,  O_i = phi(q~_i)^T S / phi(q~_i)^T z,
 * with K^ = g * phi(K~) and the sums over j taken in sequence order.
 *
 * q, k, v, og: L rows of D values at row stride ld.  a: L gate logits at
 * stride lda.  wq, wk, wv: conv taps [D][W].  norm_w: [D].  y: [L][D].
 * Optional intermediates (NULL to skip): qt, kt, vt [L][D] (after Conv1D),
 * g [L], S [D][D] (S[d][e] = sum_j g_j phi(k~_j)_d v~_j,e), z [D], O [L][D].
 * Returns 0, or -1 on a bad argument.
 */
int oracle_gbla_head(const double *q, const double *k, const double *v,
                     const double *a, const double *og, long ld, long lda,
                     long L, int D, const double *wq, const double *wk,
                     const double *wv, int W, const double *norm_w, double eps,
                     int flags, double *y, double *qt_out, double *kt_out,
                     double *vt_out, double *g_out, double *S_out,
                     double *z_out, double *O_out) {
  if (L < 0 || D <= 0 || W <= 0) return -1;
  if (L == 0) return 0;
  double *qt = xmalloc(sizeof(double) * L * D);
  double *kt = xmalloc(sizeof(double) * L * D);
  double *vt = xmalloc(sizeof(double) * L * D);
  double *g = xmalloc(sizeof(double) * L);
  double *S = xmalloc(sizeof(double) * D * D);
  double *z = xmalloc(sizeof(double) * D);
  double *O = xmalloc(sizeof(double) * L * D);
  double *pk = xmalloc(sizeof(double) * D);
  double *pq = xmalloc(sizeof(double) * D);

  gbla_prepare(q, k, v, a, ld, lda, L, D, wq, wk, wv, W, flags, qt, kt, vt, g);

  /* State: S = sum_j g_j phi(k~_j) v~_j^T and z = sum_j g_j phi(k~_j). */
  memset(S, 0, sizeof(double) * D * D);
  memset(z, 0, sizeof(double) * D);
  for (long j = 0; j < L; ++j) {
    for (int d = 0; d < D; ++d) pk[d] = g[j] * oracle_phi(kt[j * D + d]);
    for (int d = 0; d < D; ++d) {
      z[d] += pk[d];
      for (int e = 0; e < D; ++e) S[d * D + e] += pk[d] * vt[j * D + e];
    }
  }

  /* Readout: O_i = phi(q~_i)^T S / phi(q~_i)^T z. */
  for (long i = 0; i < L; ++i) {
    for (int d = 0; d < D; ++d) pq[d] = oracle_phi(qt[i * D + d]);
    double den = 0.0;
    for (int d = 0; d < D; ++d) den += pq[d] * z[d];
    for (int e = 0; e < D; ++e) {
      double num = 0.0;
      for (int d = 0; d < D; ++d) num += pq[d] * S[d * D + e];
      O[i * D + e] = num / den;
    }
  }

  gbla_finish(O, og, ld, L, D, norm_w, eps, flags, y);

  if (qt_out) memcpy(qt_out, qt, sizeof(double) * L * D);
  if (kt_out) memcpy(kt_out, kt, sizeof(double) * L * D);
  if (vt_out) memcpy(vt_out, vt, sizeof(double) * L * D);
  if (g_out) memcpy(g_out, g, sizeof(double) * L);
  if (S_out) memcpy(S_out, S, sizeof(double) * D * D);
  if (z_out) memcpy(z_out, z, sizeof(double) * D);
  if (O_out) memcpy(O_out, O, sizeof(double) * L * D);
  free(qt); free(kt); free(vt); free(g); free(S); free(z); free(O);
  free(pk); free(pq);
  return 0;
}

/*
 * The same (batch, head) in the scalar form of Sec. 2.1 item 2 written out as
 * an explicit L x L matrix:  A_ij = g_j phi(q~_i)^T phi(k~_j),
 * O_i = sum_j A_ij v~_j / sum_j A_ij.  Quadratic; for small L only.
 * Arguments as oracle_gbla_head; O_out optional.
 */
int oracle_gbla_head_quadratic(const double *q, const double *k,
                               const double *v, const double *a,
                               const double *og, long ld, long lda, long L,
                               int D, const double *wq, const double *wk,
                               const double *wv, int W, const double *norm_w,
                               double eps, int flags, double *y,
                               double *O_out) {
  if (L < 0 || D <= 0 || W <= 0) return -1;
  if (L == 0) return 0;
  double *qt = xmalloc(sizeof(double) * L * D);
  double *kt = xmalloc(sizeof(double) * L * D);
  double *vt = xmalloc(sizeof(double) * L * D);
  double *g = xmalloc(sizeof(double) * L);
  double *A = xmalloc(sizeof(double) * L * L);
  double *O = xmalloc(sizeof(double) * L * D);

  gbla_prepare(q, k, v, a, ld, lda, L, D, wq, wk, wv, W, flags, qt, kt, vt, g);

  for (long i = 0; i < L; ++i)
    for (long j = 0; j < L; ++j) {
      double s = 0.0;
      for (int d = 0; d < D; ++d)
        s += oracle_phi(qt[i * D + d]) * oracle_phi(kt[j * D + d]);
      A[i * L + j] = g[j] * s;
    }
  for (long i = 0; i < L; ++i) {
    double rs = 0.0;
    for (long j = 0; j < L; ++j) rs += A[i * L + j];
    for (int e = 0; e < D; ++e) {
      double acc = 0.0;
      for (long j = 0; j < L; ++j) acc += A[i * L + j] * vt[j * D + e];
      O[i * D + e] = acc / rs;
    }
  }

  gbla_finish(O, og, ld, L, D, norm_w, eps, flags, y);
  if (O_out) memcpy(O_out, O, sizeof(double) * L * D);
  free(qt); free(kt); free(vt); free(g); free(A); free(O);
  return 0;
}

/*
 * Whole layer core over [B, N, H, D] tensors (multi-head paragraph of
 * Sec. 2.1: heads are independent, each with its own taps, gate and norm
 * weight).  q, k, v, og: [B][N][H][D]; gate: [B][N][H]; conv_w: [3][H][D][W]
 * for q, k, v; norm_w: [H][D]; seq_lens: [B] or NULL (= N).  Row t of batch b
 * is computed for t < seq_lens[b] only; other rows of y are not written.
 * (batch, head) pairs are spread over n_threads POSIX threads.
 */
typedef struct {
  const double *q, *k, *v, *gate, *og, *conv_w, *norm_w;
  const int32_t *seq_lens;
  long B, H, N;
  int D, W, flags;
  double eps;
  double *y;
  long next;
  int status;
  pthread_mutex_t mu;
} oracle_job;

static void run_pair(oracle_job *J, long p) {
  long b = p / J->H, h = p % J->H;
  long L = J->seq_lens ? J->seq_lens[b] : J->N;
  if (L < 0) L = 0;
  if (L > J->N) L = J->N;
  long D = J->D, W = J->W, ld = J->H * D;
  long base = (b * J->N * J->H + h) * D;
  double *yh = xmalloc(sizeof(double) * (L > 0 ? L : 1) * D);
  int rc = oracle_gbla_head(
      J->q + base, J->k + base, J->v + base,
      J->gate + b * J->N * J->H + h, J->og + base, ld, J->H, L, J->D,
      J->conv_w + ((0 * J->H + h) * D) * W, J->conv_w + ((1 * J->H + h) * D) * W,
      J->conv_w + ((2 * J->H + h) * D) * W, J->W, J->norm_w + h * D, J->eps,
      J->flags, yh, NULL, NULL, NULL, NULL, NULL, NULL, NULL);
  if (rc != 0) J->status = rc;
  for (long t = 0; t < L; ++t)
    memcpy(J->y + base + t * ld, yh + t * D, sizeof(double) * D);
  free(yh);
}

static void *worker(void *arg) {
  oracle_job *J = (oracle_job *)arg;
  for (;;) {
    pthread_mutex_lock(&J->mu);
    long p = J->next++;
    pthread_mutex_unlock(&J->mu);
    if (p >= J->B * J->H) break;
    run_pair(J, p);
  }
  return NULL;
}

int oracle_gbla_forward(const double *q, const double *k, const double *v,
                        const double *gate, const double *og,
                        const double *conv_w, const double *norm_w,
                        const int32_t *seq_lens, long B, long H, long N, int D,
                        int W, double eps, int flags, int n_threads,
                        double *y) {
  if (B < 0 || H < 0 || N < 0 || D <= 0 || W <= 0) return -1;
  oracle_job J = {q, k, v, gate, og, conv_w, norm_w, seq_lens, B, H, N,
                  D, W, flags, eps, y, 0, 0};
  pthread_mutex_init(&J.mu, NULL);
  if (n_threads < 1) n_threads = 1;
  if (n_threads == 1) {
    worker(&J);
  } else {
    pthread_t *th = xmalloc(sizeof(pthread_t) * n_threads);
    for (int i = 0; i < n_threads; ++i) pthread_create(&th[i], NULL, worker, &J);
    for (int i = 0; i < n_threads; ++i) pthread_join(th[i], NULL);
    free(th);
  }
  pthread_mutex_destroy(&J.mu);
  return J.status;
}

/* ------------------------------------------------------------------------
 * Backward of the layer core (training; the paper trains the model end to
 * end, Sec. 3's training-speed table).  The paper states only the forward;
 * the gradients below are the chain rule through the six forward steps,
 * taken in reverse order, written out term by term:
 *
 *   6'. gated RMSNorm   y = O r w silu(og),  r = (mean_e O_e^2 + eps)^(-1/2)
 *         dog_e = dy_e O_e r w_e silu'(og_e),  silu'(x) = s(x) (1 + x (1 - s(x)))
 *         dw_e += dy_e O_e r silu(og_e)
 *         u_e = dy_e w_e silu(og_e);  dO_e = r u_e - (r^3 / D) O_e sum_f u_f O_f
 *   5'. readout         O = num / den,  num = S^T P,  den = P . z,  P = phi(q~)
 *         dnum = dO / den;  dden = -(dO . O) / den
 *         dP = S dnum + z dden;  dS += P dnum^T;  dz += P dden
 *   4'. state           S = sum_j K^_j v~_j^T,  z = sum_j K^_j,  K^_j = g_j phi(k~_j)
 *         dK^_j = dS v~_j + dz;  dv~_j = dS^T K^_j
 *         dphi(k~_j) = g_j dK^_j;  dg_j = phi(k~_j) . dK^_j
 *   3'. key gate        g = softmax(a):  da_j = g_j (dg_j - sum_i g_i dg_i)
 *   2'. feature map     phi'(x) = 1 (x > 0), e^x (x <= 0)
 *   1'. Conv1D          x~_t = sum_i w_i x_{t-(W-1)+i}:
 *         dx_s = sum_i w_i dx~_{s+(W-1)-i} (terms with s+(W-1)-i < L),
 *         dw_i += sum_t dx~_t x_{t-(W-1)+i}
 * Ablation switches: identity conv (dx = dx~, no tap gradient), uniform gate
 * (no logit gradient), no norm (dO = dy, no out_gate / weight gradient).
 * ------------------------------------------------------------------------ */

static double oracle_sigmoid(double x) { return 1.0 / (1.0 + exp(-x)); }

/* Conv1D backward for one channel block: dx (stride ldx) from dxt [L][C]. */
static void conv1d_backward(const double *x, const double *dxt, long L, int C,
                            long ldx, const double *w, int W, double *dx,
                            double *dw) {
  for (long s = 0; s < L; ++s)
    for (int c = 0; c < C; ++c) {
      double acc = 0.0;
      for (int i = 0; i < W; ++i) {
        long t = s + (W - 1) - i;
        if (t < L) acc += w[(long)c * W + i] * dxt[t * C + c];
      }
      dx[s * ldx + c] = acc;
    }
  for (int c = 0; c < C; ++c)
    for (int i = 0; i < W; ++i) {
      double acc = 0.0;
      for (long t = 0; t < L; ++t) {
        long s = t - (W - 1) + i;
        if (s >= 0) acc += dxt[t * C + c] * x[s * ldx + c];
      }
      dw[(long)c * W + i] += acc;
    }
}

static double phi_prime(double x) { return x > 0.0 ? 1.0 : exp(x); }

/* Error scales of the gradients (see oracle_gbla_head_backward): the
 * backward steps 6' to 1' on magnitudes, from the inputs q, k, v, the forward
 * intermediates qt, kt, vt, g, O, den and the exact dO.  Per-token scales are
 * written; tap and norm-weight scales are ADDED (sums over the batch). */
static void backward_scales(const double *q, const double *k, const double *v, long L, int D,
                            long ld, long lda, int W, const double *wq, const double *wk,
                            const double *wv, const double *norm_w, double eps, int flags,
                            const double *dy, const double *og, const double *qt,
                            const double *kt, const double *vt, const double *g,
                            const double *O, const double *dO, const double *den,
                            double *mdq, double *mdk, double *mdv, double *mda,
                            double *mdog, double *mdwq, double *mdwk, double *mdwv,
                            double *mdnw) {
  double *Sa = xmalloc(sizeof(double) * D * D);
  double *Oa = xmalloc(sizeof(double) * L * D);
  double *dOa = xmalloc(sizeof(double) * L * D);
  double *dSa = xmalloc(sizeof(double) * D * D);
  double *dza = xmalloc(sizeof(double) * D);
  double *dqta = xmalloc(sizeof(double) * L * D);
  double *dkta = xmalloc(sizeof(double) * L * D);
  double *dvta = xmalloc(sizeof(double) * L * D);
  double *dga = xmalloc(sizeof(double) * L);
  double *dKa = xmalloc(sizeof(double) * D);
  double *za = xmalloc(sizeof(double) * D);  /* z = sum_j K^_j > 0: its own magnitude */

  /* forward on magnitudes: Sa = sum_j K^_j |v~_j|^T, Oa_i = P_i^T Sa / den_i */
  memset(Sa, 0, sizeof(double) * D * D);
  memset(za, 0, sizeof(double) * D);
  for (long j = 0; j < L; ++j)
    for (int d = 0; d < D; ++d) {
      const double kh = g[j] * oracle_phi(kt[j * D + d]);
      za[d] += kh;
      for (int e = 0; e < D; ++e) Sa[d * D + e] += kh * fabs(vt[j * D + e]);
    }
  for (long i = 0; i < L; ++i)
    for (int e = 0; e < D; ++e) {
      double s = 0.0;
      for (int d = 0; d < D; ++d) s += oracle_phi(qt[i * D + d]) * Sa[d * D + e];
      Oa[i * D + e] = s / den[i];
    }

  /* 6'. gated RMSNorm: dO = r u - (r^3 / D) O (u . O) */
  for (long i = 0; i < L; ++i) {
    const double *Oi = O + i * D, *Oai = Oa + i * D, *dyi = dy + i * ld, *ogi = og + i * ld;
    double *dOai = dOa + i * D, *mdogi = mdog + i * ld;
    if (flags & ORACLE_NO_NORM) {
      for (int e = 0; e < D; ++e) {
        dOai[e] = fabs(dyi[e]);
        mdogi[e] = 0.0;
      }
      continue;
    }
    double ms = 0.0;
    for (int e = 0; e < D; ++e) ms += Oi[e] * Oi[e];
    ms /= (double)D;
    const double r = 1.0 / sqrt(ms + eps);
    double uo = 0.0, uoa = 0.0;
    for (int e = 0; e < D; ++e) {
      const double u = dyi[e] * norm_w[e] * oracle_silu(ogi[e]);
      uo += u * Oi[e];
      uoa += fabs(u) * Oai[e];
    }
    for (int e = 0; e < D; ++e) {
      const double sg = oracle_sigmoid(ogi[e]);
      const double u = dyi[e] * norm_w[e] * oracle_silu(ogi[e]);
      dOai[e] = r * fabs(u) + (r * r * r / (double)D) * (Oai[e] * fabs(uo) + fabs(Oi[e]) * uoa);
      mdogi[e] = fabs(dyi[e]) * Oai[e] * r * fabs(norm_w[e]) *
                 fabs(sg * (1.0 + ogi[e] * (1.0 - sg)));
      mdnw[e] += fabs(dyi[e]) * Oai[e] * r * fabs(oracle_silu(ogi[e]));
    }
  }

  /* 5'. readout: dnum = dO / den, dden = -(dO . O) / den, dP = S dnum + z dden */
  memset(dSa, 0, sizeof(double) * D * D);
  memset(dza, 0, sizeof(double) * D);
  for (long i = 0; i < L; ++i) {
    const double *Oi = O + i * D, *Oai = Oa + i * D, *dOi = dO + i * D, *dOai = dOa + i * D;
    double ddena = 0.0;
    for (int e = 0; e < D; ++e) ddena += dOai[e] * fabs(Oi[e]) + fabs(dOi[e]) * Oai[e];
    ddena /= den[i];
    for (int d = 0; d < D; ++d) {
      const double P = oracle_phi(qt[i * D + d]);
      double s = za[d] * ddena;
      for (int e = 0; e < D; ++e) s += Sa[d * D + e] * dOai[e] / den[i];
      dqta[i * D + d] = phi_prime(qt[i * D + d]) * s;
      dza[d] += P * ddena;
      for (int e = 0; e < D; ++e) dSa[d * D + e] += P * dOai[e] / den[i];
    }
  }

  /* 4'. state: dK^_j = dS v~_j + dz, dv~_j = dS^T K^_j, dg_j = phi(k~_j) . dK^_j */
  double gdga = 0.0;
  for (long j = 0; j < L; ++j) {
    double dg = 0.0;
    for (int d = 0; d < D; ++d) {
      double s = dza[d];
      for (int e = 0; e < D; ++e) s += dSa[d * D + e] * fabs(vt[j * D + e]);
      dKa[d] = s;
      dkta[j * D + d] = g[j] * phi_prime(kt[j * D + d]) * s;
      dg += oracle_phi(kt[j * D + d]) * s;
    }
    dga[j] = dg;
    gdga += g[j] * dg;
    for (int e = 0; e < D; ++e) {
      double s = 0.0;
      for (int d = 0; d < D; ++d) s += g[j] * oracle_phi(kt[j * D + d]) * dSa[d * D + e];
      dvta[j * D + e] = s;
    }
  }

  /* 3'. key gate: da_j = g_j (dg_j - sum_i g_i dg_i) */
  for (long j = 0; j < L; ++j)
    mda[j * lda] = (flags & ORACLE_NO_GATE) ? 0.0 : g[j] * (dga[j] + gdga);

  /* 1'. Conv1D: dx_s = sum_i w_i dx~_{s+(W-1)-i} on magnitudes */
  const double *taps[3] = {wq, wk, wv};
  const double *src[3] = {dqta, dkta, dvta};
  const double *xin[3] = {q, k, v};
  double *dst[3] = {mdq, mdk, mdv};
  double *dwa[3] = {mdwq, mdwk, mdwv};
  for (int m = 0; m < 3; ++m)
    for (long s0 = 0; s0 < L; ++s0)
      for (int c = 0; c < D; ++c) {
        double acc = 0.0;
        if (flags & ORACLE_NO_CONV) {
          acc = src[m][s0 * D + c];
        } else {
          for (int i = 0; i < W; ++i) {
            const long t = s0 + (W - 1) - i;
            if (t < L) acc += fabs(taps[m][(long)c * W + i]) * src[m][t * D + c];
          }
        }
        dst[m][s0 * ld + c] = acc;
      }
  /*     dw_i += sum_t dx~_t x_{t-(W-1)+i} on magnitudes */
  if (!(flags & ORACLE_NO_CONV))
    for (int m = 0; m < 3; ++m)
      for (int c = 0; c < D; ++c)
        for (int i = 0; i < W; ++i) {
          double acc = 0.0;
          for (long t = 0; t < L; ++t) {
            const long s0 = t - (W - 1) + i;
            if (s0 >= 0) acc += src[m][t * D + c] * fabs(xin[m][s0 * ld + c]);
          }
          dwa[m][(long)c * W + i] += acc;
        }

  free(Sa); free(Oa); free(dOa); free(dSa); free(dza); free(dqta); free(dkta);
  free(dvta); free(dga); free(dKa); free(za);
}

/*
 * One (batch, head): gradients of sum(dy * y) with respect to every input.
 * Inputs as oracle_gbla_head plus dy (L rows at stride ld).  Outputs: dq, dk,
 * dv, dog (L rows at stride ld), da (stride lda), and tap / norm-weight
 * gradients ADDED to dwq, dwk, dwv [D][W] and dnw [D].
 *
 * Optional error scales (all NULL, or all given; same layouts as dq, dk, dv,
 * da, dog, dwq, dwk, dwv, dnw, the last four ADDED to): for every gradient,
 * the first-order magnitude of what a relative perturbation of size 1 in each
 * rounded intermediate can move it by.
 * They are the same chain rule evaluated on magnitudes: every product and sum
 * on absolute values, and in place of the state and its gradient (both sums
 * over the whole sequence, which cancel) their absolute sums
 *   Sa = sum_j K^_j |v~_j|^T,  dSa = sum_i P_i dnuma_i^T,  dza = sum_i P_i ddena_i,
 * so a computation whose every rounded quantity x carries an error of at most
 * eps |x| (or eps times its own scale) stays within a small multiple of
 * eps times these scales.  Each scale is at least |gradient|.
 * Returns 0 or -1.
 */
int oracle_gbla_head_backward(const double *q, const double *k, const double *v,
                              const double *a, const double *og, long ld, long lda,
                              long L, int D, const double *wq, const double *wk,
                              const double *wv, int W, const double *norm_w,
                              double eps, int flags, const double *dy, double *dq,
                              double *dk, double *dv, double *da, double *dog,
                              double *dwq, double *dwk, double *dwv, double *dnw,
                              double *mdq, double *mdk, double *mdv, double *mda,
                              double *mdog, double *mdwq, double *mdwk, double *mdwv,
                              double *mdnw) {
  if (L < 0 || D <= 0 || W <= 0) return -1;
  if (L == 0) return 0;
  double *qt = xmalloc(sizeof(double) * L * D);
  double *kt = xmalloc(sizeof(double) * L * D);
  double *vt = xmalloc(sizeof(double) * L * D);
  double *g = xmalloc(sizeof(double) * L);
  double *S = xmalloc(sizeof(double) * D * D);
  double *z = xmalloc(sizeof(double) * D);
  double *O = xmalloc(sizeof(double) * L * D);
  double *dO = xmalloc(sizeof(double) * L * D);
  double *dS = xmalloc(sizeof(double) * D * D);
  double *dz = xmalloc(sizeof(double) * D);
  double *dqt = xmalloc(sizeof(double) * L * D);
  double *dkt = xmalloc(sizeof(double) * L * D);
  double *dvt = xmalloc(sizeof(double) * L * D);
  double *dg = xmalloc(sizeof(double) * L);
  double *P = xmalloc(sizeof(double) * D);
  double *dnum = xmalloc(sizeof(double) * D);
  double *Kh = xmalloc(sizeof(double) * D);
  double *dKh = xmalloc(sizeof(double) * D);
  double *den = xmalloc(sizeof(double) * L);

  /* forward, steps 1-5 (Sec. 2.1 items 1 and 2) */
  int rc = oracle_gbla_head(q, k, v, a, og, ld, lda, L, D, wq, wk, wv, W, norm_w,
                            eps, flags, dO /* y, unused */, qt, kt, vt, g, S, z, O);
  if (rc != 0) goto done;
  for (long i = 0; i < L; ++i) {
    double s = 0.0;
    for (int d = 0; d < D; ++d) s += oracle_phi(qt[i * D + d]) * z[d];
    den[i] = s;
  }

  /* 6'. gated RMSNorm */
  for (long i = 0; i < L; ++i) {
    const double *Oi = O + i * D, *dyi = dy + i * ld, *ogi = og + i * ld;
    double *dOi = dO + i * D, *dogi = dog + i * ld;
    if (flags & ORACLE_NO_NORM) {
      for (int e = 0; e < D; ++e) {
        dOi[e] = dyi[e];
        dogi[e] = 0.0;
      }
      continue;
    }
    double ms = 0.0;
    for (int e = 0; e < D; ++e) ms += Oi[e] * Oi[e];
    ms /= (double)D;
    const double r = 1.0 / sqrt(ms + eps);
    double uo = 0.0;
    for (int e = 0; e < D; ++e) {
      const double sg = oracle_sigmoid(ogi[e]), si = ogi[e] * sg;
      dogi[e] = dyi[e] * Oi[e] * r * norm_w[e] * sg * (1.0 + ogi[e] * (1.0 - sg));
      dnw[e] += dyi[e] * Oi[e] * r * si;
      uo += dyi[e] * norm_w[e] * si * Oi[e];
    }
    for (int e = 0; e < D; ++e) {
      const double u = dyi[e] * norm_w[e] * oracle_silu(ogi[e]);
      dOi[e] = r * u - (r * r * r / (double)D) * Oi[e] * uo;
    }
  }

  /* 5'. readout */
  memset(dS, 0, sizeof(double) * D * D);
  memset(dz, 0, sizeof(double) * D);
  for (long i = 0; i < L; ++i) {
    const double *Oi = O + i * D, *dOi = dO + i * D;
    for (int d = 0; d < D; ++d) P[d] = oracle_phi(qt[i * D + d]);
    double dOO = 0.0;
    for (int e = 0; e < D; ++e) {
      dnum[e] = dOi[e] / den[i];
      dOO += dOi[e] * Oi[e];
    }
    const double dden = -dOO / den[i];
    for (int d = 0; d < D; ++d) {
      double dP = z[d] * dden;
      for (int e = 0; e < D; ++e) dP += S[d * D + e] * dnum[e];
      dqt[i * D + d] = dP * phi_prime(qt[i * D + d]);
      dz[d] += P[d] * dden;
      for (int e = 0; e < D; ++e) dS[d * D + e] += P[d] * dnum[e];
    }
  }

  /* 4'. state */
  for (long j = 0; j < L; ++j) {
    for (int d = 0; d < D; ++d) Kh[d] = g[j] * oracle_phi(kt[j * D + d]);
    double dgj = 0.0;
    for (int d = 0; d < D; ++d) {
      double s = dz[d];
      for (int e = 0; e < D; ++e) s += dS[d * D + e] * vt[j * D + e];
      dKh[d] = s;
      dkt[j * D + d] = g[j] * s * phi_prime(kt[j * D + d]);
      dgj += oracle_phi(kt[j * D + d]) * s;
    }
    dg[j] = dgj;
    for (int e = 0; e < D; ++e) {
      double s = 0.0;
      for (int d = 0; d < D; ++d) s += Kh[d] * dS[d * D + e];
      dvt[j * D + e] = s;
    }
  }

  /* 3'. key gate */
  if (flags & ORACLE_NO_GATE) {
    for (long j = 0; j < L; ++j) da[j * lda] = 0.0;
  } else {
    double gdg = 0.0;
    for (long j = 0; j < L; ++j) gdg += g[j] * dg[j];
    for (long j = 0; j < L; ++j) da[j * lda] = g[j] * (dg[j] - gdg);
  }

  /* 1'. Conv1D (step 2' was applied with dqt / dkt above) */
  if (flags & ORACLE_NO_CONV) {
    for (long t = 0; t < L; ++t)
      for (int d = 0; d < D; ++d) {
        dq[t * ld + d] = dqt[t * D + d];
        dk[t * ld + d] = dkt[t * D + d];
        dv[t * ld + d] = dvt[t * D + d];
      }
  } else {
    conv1d_backward(q, dqt, L, D, ld, wq, W, dq, dwq);
    conv1d_backward(k, dkt, L, D, ld, wk, W, dk, dwk);
    conv1d_backward(v, dvt, L, D, ld, wv, W, dv, dwv);
  }

  if (mdq) backward_scales(q, k, v, L, D, ld, lda, W, wq, wk, wv, norm_w, eps, flags, dy, og,
                           qt, kt, vt, g, O, dO, den, mdq, mdk, mdv, mda, mdog, mdwq, mdwk,
                           mdwv, mdnw);

done:
  free(qt); free(kt); free(vt); free(g); free(S); free(z); free(O); free(dO);
  free(dS); free(dz); free(dqt); free(dkt); free(dvt); free(dg); free(P);
  free(dnum); free(Kh); free(dKh); free(den);
  return rc;
}

/*
 * Whole-layer backward over [B, N, H, D] tensors (layout of
 * oracle_gbla_forward).  Rows t >= seq_lens[b] of dq, dk, dv, dog and dgate
 * are set to 0 (padding does not reach the outputs).  dconv_w [3][H][D][W]
 * and dnorm_w [H][D] are overwritten with sums over the batch in batch order.
 * (batch, head) pairs run one after another.
 */
int oracle_gbla_backward(const double *q, const double *k, const double *v,
                         const double *gate, const double *og, const double *conv_w,
                         const double *norm_w, const int32_t *seq_lens, long B, long H,
                         long N, int D, int W, double eps, int flags, const double *dy,
                         double *dq, double *dk, double *dv, double *dgate,
                         double *dog, double *dconv_w, double *dnorm_w) {
  if (B < 0 || H < 0 || N < 0 || D <= 0 || W <= 0) return -1;
  const long ld = H * D;
  memset(dq, 0, sizeof(double) * B * N * ld);
  memset(dk, 0, sizeof(double) * B * N * ld);
  memset(dv, 0, sizeof(double) * B * N * ld);
  memset(dog, 0, sizeof(double) * B * N * ld);
  memset(dgate, 0, sizeof(double) * B * N * H);
  memset(dconv_w, 0, sizeof(double) * 3 * H * D * W);
  memset(dnorm_w, 0, sizeof(double) * H * D);
  for (long b = 0; b < B; ++b)
    for (long h = 0; h < H; ++h) {
      long L = seq_lens ? seq_lens[b] : N;
      if (L < 0) L = 0;
      if (L > N) L = N;
      const long base = (b * N * H + h) * D, gbase = b * N * H + h;
      int rc = oracle_gbla_head_backward(
          q + base, k + base, v + base, gate + gbase, og + base, ld, H, L, D,
          conv_w + ((0 * H + h) * D) * W, conv_w + ((1 * H + h) * D) * W,
          conv_w + ((2 * H + h) * D) * W, W, norm_w + h * D, eps, flags, dy + base,
          dq + base, dk + base, dv + base, dgate + gbase, dog + base,
          dconv_w + ((0 * H + h) * D) * W, dconv_w + ((1 * H + h) * D) * W,
          dconv_w + ((2 * H + h) * D) * W, dnorm_w + h * D, NULL, NULL, NULL, NULL, NULL,
          NULL, NULL, NULL, NULL);
      if (rc != 0) return rc;
    }
  return 0;
}

/* ------------------------------------------------------------------------
 * Layer front end: the X-space Conv1D and the per-head projections.
 *
 *   X~ = Conv1D(X)                            (Sec. 2.1 item 1)
 *   Q = X~ W_Q,  K = X~ W_K,  V = X~ W_V      (Sec. 2.1 item 1)
 *   gate logits = X~ w_g                      (Sec. 2.1 item 2)
 *   out-gate input = X~ W_R                   (Sec. 2.1 item 3)
 * with one set of matrices per head (the multi-head paragraph of Sec. 2.1).
 *
 * Readings: the Conv1D on X is depthwise over the d channels, causal, with
 * the tap order of oracle_conv1d (tap W-1 multiplies the current token), no
 * bias and no activation.  The weights of all heads and projections are
 * stacked into one matrix w [F][d], F = 4 H D + H, one row per output feature
 * over the d input channels (row f gives output f = sum_c x~[c] w[f][c]):
 * rows s*H*D + h*D + e for stream s = Q, K, V, R (W_R) and head h, dim e, then
 * rows 4 H D + h for w_g of head h.
 *
 * x [B][N][d]; conv_x [d][W]; q, k, v, og [B][N][H][D]; gate [B][N][H].
 * Rows t >= seq_lens[b] are not written (they are padding, and no valid row
 * reads them: the Conv1D is causal).  absdot, when given, is [B][N][F] and
 * receives sum_c |x~[c] w[f][c]| per output: the scale of any rounding error
 * in computing the output (the error bound of a dot product is proportional
 * to it).
 * ------------------------------------------------------------------------ */
int oracle_gbla_project(const double *x, const double *conv_x, const double *w,
                        const int32_t *seq_lens, long B, long N, int d, int W, long H,
                        int D, double *q, double *k, double *v, double *og, double *gate,
                        double *absdot) {
  if (B < 0 || N < 0 || d <= 0 || W <= 0 || H <= 0 || D <= 0) return -1;
  const long HD = H * (long)D;
  const long F = 4 * HD + H;
  double *xt = (double *)xmalloc(sizeof(double) * (size_t)(N > 0 ? N : 1) * d);
  double *streams[4] = {q, k, v, og};
  for (long b = 0; b < B; ++b) {
    long L = seq_lens ? seq_lens[b] : N;
    if (L < 0) L = 0;
    if (L > N) L = N;
    oracle_conv1d(x + b * N * d, L, d, d, conv_x, W, xt);
    for (long t = 0; t < L; ++t) {
      const double *xr = xt + t * d;
      for (long f = 0; f < F; ++f) {
        const double *wr = w + f * d;
        double acc = 0.0, mag = 0.0;
        for (int c = 0; c < d; ++c) {
          acc += xr[c] * wr[c];
          mag += fabs(xr[c] * wr[c]);
        }
        if (f < 4 * HD) {
          const long s = f / HD, col = f % HD;
          streams[s][(b * N + t) * HD + col] = acc;
        } else {
          gate[(b * N + t) * H + (f - 4 * HD)] = acc;
        }
        if (absdot) absdot[(b * N + t) * F + f] = mag;
      }
    }
  }
  free(xt);
  return 0;
}

/* ------------------------------------------------------------------------
 * Bidirectional softmax attention (Sec. 2, "Bidirectional softmax
 * attention"), the SA layer of the hybrid [SA, LA, LA] encoder (Sec. 3):
 *   Attn(q_i, K, V) = sum_j exp(q_i . k_j / sqrt(d_h)) v_j / sum_j exp(q_i . k_j / sqrt(d_h)),
 * over the valid keys j < L of one (batch, head), for each valid query i < L.
 * Arrays are [B, N, H, D] (token-major, heads interleaved); rows t >= L of
 * out are left as they are.  The maximum score of each row is subtracted
 * before exponentiating (the quotient does not change; it keeps exp finite).
 * Rows are independent, so (batch, head) pairs run on n_threads threads.
 * ------------------------------------------------------------------------ */
typedef struct {
  const double *q, *k, *v;
  const int32_t *seq_lens;
  long B, N, H;
  int D;
  double *out, *absout;
  long next;
  pthread_mutex_t mu;
} oracle_sa_job;

/* One query row against the L keys and values of one (batch, head), strided
 * by ld between tokens: out[d] = the attention output, absout[d] (optional) =
 * sum_j p_j |v_j[d]| / sum_j p_j, the scale of the error a relative rounding
 * of the probabilities p_j makes.  s is scratch of L doubles. */
static void sa_row(const double *qi, const double *k, const double *v, long L, long ld, int D,
                   double *s, double *out, double *absout) {
  const double scale = 1.0 / sqrt((double)D);
  double m = -INFINITY;
  for (long j = 0; j < L; ++j) {
    const double *kj = k + j * ld;
    double dot = 0.0;
    for (int d = 0; d < D; ++d) dot += qi[d] * kj[d];
    s[j] = dot * scale;
    if (s[j] > m) m = s[j];
  }
  double den = 0.0;
  for (long j = 0; j < L; ++j) {
    s[j] = exp(s[j] - m);
    den += s[j];
  }
  for (int d = 0; d < D; ++d) {
    out[d] = 0.0;
    if (absout) absout[d] = 0.0;
  }
  for (long j = 0; j < L; ++j) {
    const double *vj = v + j * ld;
    for (int d = 0; d < D; ++d) {
      out[d] += s[j] * vj[d];
      if (absout) absout[d] += s[j] * fabs(vj[d]);
    }
  }
  for (int d = 0; d < D; ++d) {
    out[d] /= den;
    if (absout) absout[d] /= den;
  }
}

static void sa_pair(oracle_sa_job *J, long p) {
  const long b = p / J->H, h = p % J->H, N = J->N, H = J->H;
  const int D = J->D;
  long L = J->seq_lens ? J->seq_lens[b] : N;
  if (L < 0) L = 0;
  if (L > N) L = N;
  const long ld = H * D, base = (b * N * H + h) * D;
  double *s = (double *)xmalloc(sizeof(double) * (size_t)(L > 0 ? L : 1));
  for (long i = 0; i < L; ++i)
    sa_row(J->q + base + i * ld, J->k + base, J->v + base, L, ld, D, s, J->out + base + i * ld,
           J->absout ? J->absout + base + i * ld : NULL);
  free(s);
}

static void *sa_worker(void *arg) {
  oracle_sa_job *J = (oracle_sa_job *)arg;
  for (;;) {
    pthread_mutex_lock(&J->mu);
    const long p = J->next++;
    pthread_mutex_unlock(&J->mu);
    if (p >= J->B * J->H) break;
    sa_pair(J, p);
  }
  return NULL;
}

int oracle_softmax_attention(const double *q, const double *k, const double *v,
                             const int32_t *seq_lens, long B, long N, long H, int D,
                             int n_threads, double *out, double *absout) {
  if (B < 0 || N < 0 || H < 0 || D <= 0) return -1;
  oracle_sa_job J;
  J.q = q; J.k = k; J.v = v; J.seq_lens = seq_lens;
  J.B = B; J.N = N; J.H = H; J.D = D; J.out = out; J.absout = absout; J.next = 0;
  pthread_mutex_init(&J.mu, NULL);
  if (n_threads < 1) n_threads = 1;
  if (n_threads > 256) n_threads = 256;
  pthread_t th[256];
  int started = 0;
  for (int i = 1; i < n_threads; ++i)
    if (pthread_create(&th[started], NULL, sa_worker, &J) == 0) ++started;
  sa_worker(&J);
  for (int i = 0; i < started; ++i) pthread_join(th[i], NULL);
  pthread_mutex_destroy(&J.mu);
  return 0;
}

/* Selected query rows of one (batch, head): q_rows [R][D] against keys and
 * values k, v [L][D] (contiguous), giving out and absout [R][D] (see sa_row). */
int oracle_softmax_attention_rows(const double *q_rows, long R, const double *k,
                                  const double *v, long L, int D, double *out,
                                  double *absout) {
  if (R < 0 || L < 1 || D <= 0) return -1;
  double *s = (double *)xmalloc(sizeof(double) * (size_t)L);
  for (long r = 0; r < R; ++r)
    sa_row(q_rows + r * D, k, v, L, D, D, s, out + r * D, absout ? absout + r * D : NULL);
  free(s);
  return 0;
}
