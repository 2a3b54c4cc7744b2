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
