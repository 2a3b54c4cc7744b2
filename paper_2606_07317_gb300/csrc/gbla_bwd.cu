// Backward of the GBLA layer core (CUDA cores, fp32 arithmetic): gradients of
// sum(dy * y) with respect to q, k, v, the gate logits, out_gate, the Conv1D
// taps and the RMSNorm weight.  The paper states only the forward (Sec. 2.1);
// the gradients are the chain rule through its steps, in reverse:
//
//   6'. gated RMSNorm  y = O r w silu(og),  r = (mean O^2 + eps)^(-1/2)
//        dog = dy O r w silu'(og);  dw += dy O r silu(og)
//        u = dy w silu(og);  dO = r u - (r^3 / D) O (u . O)
//   5'. readout        O = num / den,  num = S^T P,  den = P . z,  P = phi(q~)
//        dnum = dO / den;  dden = -(dO . O) / den
//        dP = S dnum + z dden;  dS += P dnum^T;  dz += P dden
//   4'. state          S = sum_j K^_j v~_j^T,  z = sum_j K^_j,  K^_j = g_j phi(k~_j)
//        dK^_j = dS v~_j + dz;  dv~_j = dS^T K^_j;  dk~_j = g_j dK^_j phi'(k~_j)
//   3'. key gate       da_j = g_j (dg_j - c),  dg_j = phi(k~_j) . dK^_j,
//        c = sum_j g_j dg_j = <dS, S> + <dz, z>
//   1'. Conv1D         dx_s = sum_i w_i dx~_{s+3-i};  dw_i += sum_t dx~_t x_{t-3+i}
//
// Launches (all on the caller's stream, after the forward state S, z has been
// formed by the forward's own state path):
//   bwd_gate_split / bwd_gate_join  per (b, h): M = max a, Ltot = sum e^{a - M}
//                    (g_j = e^{a_j-M}/Ltot), over sequence splits, then combined;
//                    skipped when the tensor-core state path already wrote them
//   bwd_query        per (b, h, chunk): 5' and 6' per token; dq~ to scratch
//                    (the dq~, dk~, dv~ planes are stored in the I/O dtype);
//                    chunk partials of dS, dz and the norm-weight gradient
//   bwd_reduce_state per (b, h): fixed-order sums of the partials (and, for the
//                    tensor-core key pass, per-block partial sums of c)
//   bwd_key          per (b, h, chunk): c, then 4' and 3' per token; dk~, dv~ to
//                    scratch (tc_bwd_key_kernel and tc_bwd_query_kernel in
//                    gbla_bwd_tc.cu replace bwd_key and bwd_query for bf16, D = 64)
//   bwd_conv         per (stream, b, h, chunk): 1' (anti-causal taps) into dq,
//                    dk, dv; chunk partials of the tap gradients
//   bwd_reduce_w     fixed-order sums of the tap / norm-weight partials
// Every sum runs in a fixed order, so the results are deterministic.
#include <math.h>

#include "gbla_internal.cuh"
#include "gbla_sm100.cuh"

namespace gbla {
namespace {

constexpr int kNT = 256;      // threads per block of the token passes
constexpr int kChunk = 256;   // tokens per block

__device__ __forceinline__ float ldf(const float *p, size_t i) { return p[i]; }
__device__ __forceinline__ float ldf(const __nv_bfloat16 *p, size_t i) {
  return __bfloat162float(p[i]);
}
__device__ __forceinline__ void stf(float *p, size_t i, float x) { p[i] = x; }
__device__ __forceinline__ void stf(__nv_bfloat16 *p, size_t i, float x) {
  p[i] = __float2bfloat16_rn(x);
}
__device__ __forceinline__ float phi(float x) { return x > 0.f ? x + 1.f : expf(x); }
__device__ __forceinline__ float dphi(float x) { return x > 0.f ? 1.f : expf(x); }
__device__ __forceinline__ int clamp_len(const int32_t *seq_lens, int b, int N) {
  if (seq_lens == nullptr) return N;
  int L = seq_lens[b];
  return L < 0 ? 0 : (L > N ? N : L);
}
__device__ __forceinline__ float warp_sum(float x) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
  return x;
}
// Thread layout of a token pass: thread (tq, c), c = tid % D the channel and
// tokens tq * TPT .. tq * TPT + TPT - 1 of the batch.
template <int D>
struct Tok {
  static constexpr int TB = 16;                  // tokens per batch
  static constexpr int TQ = kNT / D;             // token quads per batch
  static constexpr int TPT = TB / TQ;            // tokens per thread
};

// Sums over the D channels of each of this thread's TPT tokens (every thread
// of the block calls it).  red: kNT / 32 * TPT floats of shared memory.
template <int D, int TPT>
__device__ __forceinline__ void chan_sum(float (&x)[TPT], float *red) {
  constexpr int WPT = D / 32;  // warps per token quad (D >= 32)
  const int w = threadIdx.x >> 5, tq = threadIdx.x / D;
#pragma unroll
  for (int u = 0; u < TPT; ++u) x[u] = warp_sum(x[u]);
  if (WPT == 1) return;
  __syncthreads();  // red free from the previous use
  if ((threadIdx.x & 31) == 0)
#pragma unroll
    for (int u = 0; u < TPT; ++u) red[w * TPT + u] = x[u];
  __syncthreads();
#pragma unroll
  for (int u = 0; u < TPT; ++u) {
    float s = 0.f;
#pragma unroll
    for (int i = 0; i < WPT; ++i) s += red[(tq * WPT + i) * TPT + u];
    x[u] = s;
  }
}

// Loads n consecutive floats of shared memory (n = 2, 4 or 8; p aligned to
// min(n, 4) floats) with 8- or 16-byte loads.
template <int n>
__device__ __forceinline__ void ld_vec(const float *p, float (&v)[n]) {
  if constexpr (n == 2) {
    const float2 a = *reinterpret_cast<const float2 *>(p);
    v[0] = a.x;
    v[1] = a.y;
  } else {
#pragma unroll
    for (int i = 0; i < n; i += 4) {
      const float4 a = *reinterpret_cast<const float4 *>(p + i);
      v[i] = a.x;
      v[i + 1] = a.y;
      v[i + 2] = a.z;
      v[i + 3] = a.w;
    }
  }
}

// y[u] = sum_k X[k][t_u] M[k][c] for this thread's tokens t_u = tq * TPT + u:
// X in shared memory as [D][TB] (k-major), M as [D][D] row-major.  The TPT
// tokens of a thread are one vector load per k and the products go through
// packed fp32 FMAs (two per instruction, each rounded as fmaf).
template <int D, int TPT>
__device__ __forceinline__ void xm(const float *X, const float *M, int tq, int c,
                                   float (&y)[TPT]) {
  static_assert(TPT % 2 == 0, "token pairs");
  float2 acc[TPT / 2];
#pragma unroll
  for (int i = 0; i < TPT / 2; ++i) acc[i] = make_float2(0.f, 0.f);
  const float *xr = X + tq * TPT;
#pragma unroll 8
  for (int k = 0; k < D; ++k) {
    const float m = M[k * D + c];
    float xv[TPT];
    ld_vec<TPT>(xr + k * Tok<D>::TB, xv);
#pragma unroll
    for (int i = 0; i < TPT / 2; ++i)
      acc[i] = __ffma2_rn(make_float2(xv[2 * i], xv[2 * i + 1]), make_float2(m, m), acc[i]);
  }
#pragma unroll
  for (int i = 0; i < TPT / 2; ++i) {
    y[2 * i] = acc[i].x;
    y[2 * i + 1] = acc[i].y;
  }
}

// Causal Conv1D of one channel at token t: sum_i w[i] x[t - 3 + i], x[<0] = 0.
template <typename T>
__device__ __forceinline__ float conv_at(const T *x, size_t rs, int t, const float (&w)[kConvW]) {
  float a = 0.f;
#pragma unroll
  for (int i = 0; i < kConvW; ++i) {
    const int s = t - (kConvW - 1) + i;
    if (s >= 0) a = fmaf(w[i], ldf(x, (size_t)s * rs), a);
  }
  return a;
}

// ---------------------------------------------------------------- gate stats
// Per (b, h): M = max_j a_j and Ltot = sum_j e^{a_j - M} over j < L_b, in two
// steps.  bwd_gate_split: block (bh, split) walks its kGateSplitLen tokens once,
// each thread keeping a running (max, sum) pair (the sum rescaled when the max
// grows), and combines the 256 pairs in a fixed tree order.  bwd_gate_join:
// the splits of one (b, h) in index order.
constexpr int kGateSplits = 16;
__device__ __forceinline__ float2 ms_join(float2 x, float2 y) {  // (max, sum) pairs
  const float m = fmaxf(x.x, y.x);
  if (m == -INFINITY) return make_float2(-INFINITY, 0.f);
  return make_float2(m, x.y * expf(x.x - m) + y.y * expf(y.x - m));
}
template <typename T>
__global__ void __launch_bounds__(256) bwd_gate_split(const T *__restrict__ gate,
                                                      const int32_t *__restrict__ seq_lens,
                                                      float2 *__restrict__ part, int H, int N) {
  const int bh = blockIdx.x, sp = blockIdx.y, b = bh / H, h = bh % H;
  const int L = clamp_len(seq_lens, b, N);
  const int len = (N + kGateSplits - 1) / kGateSplits;
  const int ta = sp * len, tb = min(ta + len, L);
  float2 acc = make_float2(-INFINITY, 0.f);
  for (int t = ta + threadIdx.x; t < tb; t += 256)
    acc = ms_join(acc, make_float2(ldf(gate, ((size_t)b * N + t) * H + h), 1.f));
  __shared__ float2 red[256];
  red[threadIdx.x] = acc;
  __syncthreads();
  for (int w = 128; w > 0; w >>= 1) {
    if (threadIdx.x < w) red[threadIdx.x] = ms_join(red[threadIdx.x], red[threadIdx.x + w]);
    __syncthreads();
  }
  if (threadIdx.x == 0) part[(size_t)bh * kGateSplits + sp] = red[0];
}
__global__ void __launch_bounds__(256) bwd_gate_join(const float2 *__restrict__ part,
                                                     float2 *__restrict__ stats, int BH) {
  const int bh = blockIdx.x * 256 + threadIdx.x;
  if (bh >= BH) return;
  float2 acc = make_float2(-INFINITY, 0.f);
  for (int sp = 0; sp < kGateSplits; ++sp) acc = ms_join(acc, part[(size_t)bh * kGateSplits + sp]);
  stats[bh] = acc;
}

// ---------------------------------------------------------------- query pass
// Partial record per (b, h, chunk): dS [D][D], dz [D], dnorm_w [D].
template <int D>
constexpr int qrec() { return D * D + 2 * D; }

template <typename T, int D>
__global__ void __launch_bounds__(kNT) bwd_query(
    const T *__restrict__ q, const T *__restrict__ og, const T *__restrict__ dy,
    const float *__restrict__ conv_w, const float *__restrict__ norm_w,
    const float *__restrict__ state, const int32_t *__restrict__ seq_lens, float eps,
    T *__restrict__ dog, T *__restrict__ dqt, float *__restrict__ part, int H, int N,
    int nck, int no_norm) {
  constexpr int F = D * D + D;
  constexpr int TPT = Tok<D>::TPT, kTB = Tok<D>::TB;
  constexpr int RB = D / 16;  // this thread's RB x RB block of dS (16 x 16 threads)
  extern __shared__ float sm[];
  float *S = sm, *St = S + D * D, *z = St + D * D;
  float *Pk = z + D, *Pt = Pk + D * kTB, *Nk = Pt + kTB * D, *Nt = Nk + D * kTB;
  float *sDd = Nt + kTB * D, *red = sDd + kTB;
  const int chunk = blockIdx.x, bh = blockIdx.y, b = bh / H, h = bh % H;
  const int tid = threadIdx.x, tq = tid / D, c = tid % D;
  const int L = clamp_len(seq_lens, b, N);
  const int t0 = chunk * kChunk, t1 = min(t0 + kChunk, N), tv = min(t1, L);
  const float *st = state + (size_t)bh * F;
  for (int i = tid; i < D * D; i += kNT) {
    const float x = st[i];
    S[i] = x;
    St[(i % D) * D + i / D] = x;
  }
  for (int i = tid; i < D; i += kNT) z[i] = st[D * D + i];
  float wq[kConvW];
#pragma unroll
  for (int i = 0; i < kConvW; ++i) wq[i] = conv_w[((size_t)h * D + c) * kConvW + i];
  const float nw = norm_w[(size_t)h * D + c];
  const size_t rs = (size_t)H * D;
  const T *qc = q + ((size_t)b * N * H + h) * D + c;
  const int bi = tid / 16, bj = tid % 16;  // dS block rows bi * RB.., columns bj * RB..
  float2 acc2[RB][RB / 2];
#pragma unroll
  for (int i = 0; i < RB; ++i)
#pragma unroll
    for (int j = 0; j < RB / 2; ++j) acc2[i][j] = make_float2(0.f, 0.f);
  float dz = 0.f, dnw = 0.f;
  __syncthreads();
  for (int base = t0; base < t1; base += kTB) {
    float qt[TPT], P[TPT], ogv[TPT], dyv[TPT], x[TPT];
#pragma unroll
    for (int u = 0; u < TPT; ++u) {
      const int tl = tq * TPT + u, t = base + tl;
      const bool valid = t < tv;
      const size_t row = (((size_t)b * N + t) * H + h) * D + c;
      qt[u] = valid ? conv_at(qc, rs, t, wq) : 0.f;
      P[u] = valid ? phi(qt[u]) : 0.f;
      ogv[u] = valid ? ldf(og, row) : 0.f;
      dyv[u] = valid ? ldf(dy, row) : 0.f;
      Pk[c * kTB + tl] = P[u];
      Pt[tl * D + c] = P[u];
      x[u] = P[u] * z[c];
    }
    chan_sum<D, TPT>(x, red);  // den
    float den[TPT];
#pragma unroll
    for (int u = 0; u < TPT; ++u) den[u] = x[u];
    __syncthreads();  // Pk complete
    float num[TPT];
    xm<D, TPT>(Pk, S, tq, c, num);
    float O[TPT];
#pragma unroll
    for (int u = 0; u < TPT; ++u) {
      O[u] = base + tq * TPT + u < tv ? num[u] / den[u] : 0.f;
      x[u] = O[u] * O[u];
    }
    chan_sum<D, TPT>(x, red);  // D * mean O^2
    float r[TPT], uu[TPT];
#pragma unroll
    for (int u = 0; u < TPT; ++u) {
      const int t = base + tq * TPT + u;
      r[u] = 1.f / sqrtf(x[u] / (float)D + eps);
      const float sg = 1.f / (1.f + expf(-ogv[u])), si = ogv[u] * sg;
      if (t < t1) {
        const size_t row = (((size_t)b * N + t) * H + h) * D + c;
        stf(dog, row, no_norm ? 0.f : dyv[u] * O[u] * r[u] * nw * sg * (1.f + ogv[u] * (1.f - sg)));
      }
      if (!no_norm) dnw = fmaf(dyv[u] * O[u], r[u] * si, dnw);
      uu[u] = dyv[u] * nw * si;
      x[u] = uu[u] * O[u];
    }
    chan_sum<D, TPT>(x, red);  // u . O
    float dO[TPT];
#pragma unroll
    for (int u = 0; u < TPT; ++u) {
      // without the gated RMSNorm (ablation) o = O, so dO = dy
      dO[u] = no_norm ? dyv[u] : r[u] * uu[u] - (r[u] * r[u] * r[u] / (float)D) * O[u] * x[u];
      x[u] = dO[u] * O[u];
    }
    chan_sum<D, TPT>(x, red);  // dO . O
#pragma unroll
    for (int u = 0; u < TPT; ++u) {
      const int tl = tq * TPT + u;
      const bool valid = base + tl < tv;
      const float dn = valid ? dO[u] / den[u] : 0.f;
      Nk[c * kTB + tl] = dn;
      Nt[tl * D + c] = dn;
      if (c == 0) sDd[tl] = valid ? -x[u] / den[u] : 0.f;
    }
    __syncthreads();  // Nk, Nt, sDd complete
    float dP[TPT];
    xm<D, TPT>(Nk, St, tq, c, dP);  // dP_t[d] = sum_e dnum_t[e] S[d][e]
#pragma unroll
    for (int u = 0; u < TPT; ++u) {
      const int tl = tq * TPT + u, t = base + tl;
      const float dd = sDd[tl];
      if (t < t1) {
        const size_t row = (((size_t)b * N + t) * H + h) * D + c;
        stf(dqt, row, (dP[u] + z[c] * dd) * dphi(qt[u]) * (t < tv ? 1.f : 0.f));
      }
      dz = fmaf(P[u], dd, dz);
    }
    // dS += P^T dnum over the batch's tokens (RB values of P and of dnum per
    // token as vector loads; packed FMAs over pairs of columns)
#pragma unroll 2
    for (int tl = 0; tl < kTB; ++tl) {
      float pv[RB], nv[RB];
      ld_vec<RB>(Pt + tl * D + bi * RB, pv);
      ld_vec<RB>(Nt + tl * D + bj * RB, nv);
#pragma unroll
      for (int i = 0; i < RB; ++i)
#pragma unroll
        for (int j = 0; j < RB / 2; ++j)
          acc2[i][j] = __ffma2_rn(make_float2(pv[i], pv[i]),
                                  make_float2(nv[2 * j], nv[2 * j + 1]), acc2[i][j]);
    }
    __syncthreads();  // the batch's shared arrays are rewritten next
  }
  float *rec = part + ((size_t)bh * nck + chunk) * qrec<D>();
#pragma unroll
  for (int i = 0; i < RB; ++i)
#pragma unroll
    for (int j = 0; j < RB / 2; ++j)
      *reinterpret_cast<float2 *>(rec + (bi * RB + i) * D + bj * RB + 2 * j) = acc2[i][j];
  // dz and dnw: sum over the token quads in order
  Pk[tq * D + c] = dz;
  Nk[tq * D + c] = dnw;
  __syncthreads();
  if (tid < D) {
    float a = 0.f, w = 0.f;
    for (int i = 0; i < Tok<D>::TQ; ++i) {
      a += Pk[i * D + tid];
      w += Nk[i * D + tid];
    }
    rec[D * D + tid] = a;
    rec[D * D + D + tid] = w;
  }
}

// ---------------------------------------------------------------- state reduction
// red record per (b, h): dS [D][D], dz [D] (chunk partials summed in chunk order).
template <int D>
// With state and dotpart given, block x of (b, h) also writes the partial dot
// product of its slice of [dS | dz] with [S | z] (lanes, then warps in order):
// c = <dS, S> + <dz, z> is the sum of the gridDim.x partials in order.
__global__ void __launch_bounds__(256) bwd_reduce_state(const float *__restrict__ part,
                                                        float *__restrict__ red,
                                                        const float *__restrict__ state,
                                                        float *__restrict__ dotpart, int nck) {
  constexpr int F = D * D + D;
  const int bh = blockIdx.y, i = blockIdx.x * 256 + threadIdx.x;
  sm100::grid_dep_wait();  // the partials come from the query pass
  sm100::grid_dep_launch();
  float a = 0.f;
  if (i < F) {
    for (int ch = 0; ch < nck; ++ch) a += part[((size_t)bh * nck + ch) * qrec<D>() + i];
    red[(size_t)bh * F + i] = a;
  }
  if (dotpart == nullptr) return;
  const float d = warp_sum(i < F ? a * state[(size_t)bh * F + i] : 0.f);
  __shared__ float wsum[8];
  if ((threadIdx.x & 31) == 0) wsum[threadIdx.x >> 5] = d;
  __syncthreads();
  if (threadIdx.x == 0) {
    float c = 0.f;
    for (int w = 0; w < 8; ++w) c += wsum[w];
    dotpart[(size_t)bh * gridDim.x + blockIdx.x] = c;
  }
}

// ---------------------------------------------------------------- key pass
template <typename T, int D>
__global__ void __launch_bounds__(kNT) bwd_key(
    const T *__restrict__ k, const T *__restrict__ v, const T *__restrict__ gate,
    const float *__restrict__ conv_w, const float2 *__restrict__ stats,
    const float *__restrict__ state, const float *__restrict__ red,
    const int32_t *__restrict__ seq_lens, T *__restrict__ dgate, T *__restrict__ dkt,
    T *__restrict__ dvt, int H, int N) {
  constexpr int F = D * D + D;
  constexpr int TPT = Tok<D>::TPT, kTB = Tok<D>::TB;
  extern __shared__ float sm[];
  float *dS = sm, *dSt = dS + D * D, *dz = dSt + D * D;
  float *Kk = dz + D, *Vk = Kk + D * kTB, *rd = Vk + D * kTB;
  const int chunk = blockIdx.x, bh = blockIdx.y, b = bh / H, h = bh % H;
  const int tid = threadIdx.x, tq = tid / D, c = tid % D;
  const int L = clamp_len(seq_lens, b, N);
  const int t0 = chunk * kChunk, t1 = min(t0 + kChunk, N), tv = min(t1, L);
  const float *rr = red + (size_t)bh * F;
  const float *st = state + (size_t)bh * F;
  float cs = 0.f;  // c = <dS, S> + <dz, z>, this thread's part
  for (int i = tid; i < F; i += kNT) {
    const float x = rr[i];
    if (i < D * D) {
      dS[i] = x;
      dSt[(i % D) * D + i / D] = x;
    } else {
      dz[i - D * D] = x;
    }
    cs = fmaf(x, st[i], cs);
  }
  cs = warp_sum(cs);
  if ((tid & 31) == 0) rd[tid >> 5] = cs;
  __syncthreads();
  float cval = 0.f;
  for (int i = 0; i < kNT / 32; ++i) cval += rd[i];
  const float2 gs = stats[bh];
  float wk[kConvW], wv[kConvW];
#pragma unroll
  for (int i = 0; i < kConvW; ++i) {
    wk[i] = conv_w[((size_t)(H + h) * D + c) * kConvW + i];
    wv[i] = conv_w[((size_t)(2 * H + h) * D + c) * kConvW + i];
  }
  const size_t rs = (size_t)H * D;
  const T *kc = k + ((size_t)b * N * H + h) * D + c;
  const T *vc = v + ((size_t)b * N * H + h) * D + c;
  __syncthreads();  // rd read before chan_sum reuses it
  for (int base = t0; base < t1; base += kTB) {
    float kt[TPT], pk[TPT], g[TPT];
#pragma unroll
    for (int u = 0; u < TPT; ++u) {
      const int tl = tq * TPT + u, t = base + tl;
      const bool valid = t < tv;
      kt[u] = valid ? conv_at(kc, rs, t, wk) : 0.f;
      const float vt = valid ? conv_at(vc, rs, t, wv) : 0.f;
      g[u] = valid ? expf(ldf(gate, ((size_t)b * N + t) * H + h) - gs.x) / gs.y : 0.f;
      pk[u] = valid ? phi(kt[u]) : 0.f;
      Kk[c * kTB + tl] = g[u] * pk[u];
      Vk[c * kTB + tl] = vt;
    }
    __syncthreads();  // Kk, Vk complete
    float dK[TPT], dvv[TPT];
    xm<D, TPT>(Vk, dSt, tq, c, dK);   // dK^_t[d] = sum_e dS[d][e] v~_t[e]
    xm<D, TPT>(Kk, dS, tq, c, dvv);   // dv~_t[e] = sum_d K^_t[d] dS[d][e]
    float x[TPT];
#pragma unroll
    for (int u = 0; u < TPT; ++u) {
      const int t = base + tq * TPT + u;
      dK[u] += dz[c];
      if (t < t1) {
        const size_t row = (((size_t)b * N + t) * H + h) * D + c;
        const bool valid = t < tv;
        stf(dkt, row, valid ? g[u] * dK[u] * dphi(kt[u]) : 0.f);
        stf(dvt, row, valid ? dvv[u] : 0.f);
      }
      x[u] = pk[u] * dK[u];
    }
    chan_sum<D, TPT>(x, rd);  // dg_t
#pragma unroll
    for (int u = 0; u < TPT; ++u) {
      const int t = base + tq * TPT + u;
      if (c == 0 && t < t1)
        stf(dgate, ((size_t)b * N + t) * H + h, t < tv ? g[u] * (x[u] - cval) : 0.f);
    }
    __syncthreads();  // Kk, Vk rewritten next
  }
}

// ---------------------------------------------------------------- Conv1D backward
// Stream s = 2 - blockIdx.z (0 q, 1 k, 2 v) over a block of RUNS x rl tokens of
// one (b, h): dx_t = sum_i w_i dx~_{t+3-i} (terms with t + 3 - i >= L dropped;
// dx_t = 0 for t >= L) and the block's partials of dw_i = sum_t dx~_t x_{t-3+i}.
// Thread (run, g) walks rl consecutive tokens of channels
// 4g .. 4g+3 with sliding windows (x of the 3 tokens before, dx~ of the 3
// after), every token's 4 channels one vector load; the runs' tap partials are
// then added in run order.
constexpr int kConvCh = 4;  // channels per thread
__device__ __forceinline__ void ld4(const float *p, float (&f)[4]) {
  const float4 a = __ldg((const float4 *)p);
  f[0] = a.x; f[1] = a.y; f[2] = a.z; f[3] = a.w;
}
__device__ __forceinline__ void ld4(const __nv_bfloat16 *p, float (&f)[4]) {
  const uint2 u = __ldg((const uint2 *)p);
  f[0] = __uint_as_float(u.x << 16); f[1] = __uint_as_float(u.x & 0xFFFF0000u);
  f[2] = __uint_as_float(u.y << 16); f[3] = __uint_as_float(u.y & 0xFFFF0000u);
}
// Four channels as loaded (raw), then widened to fp32: the Conv1D backward
// stages a batch of raw loads in shared memory before it converts any of them.
template <typename T> struct Raw4;
template <> struct Raw4<float> { using type = float4; };
template <> struct Raw4<__nv_bfloat16> { using type = uint2; };
__device__ __forceinline__ void cvt4raw(const float4 &a, float (&f)[4]) {
  f[0] = a.x; f[1] = a.y; f[2] = a.z; f[3] = a.w;
}
__device__ __forceinline__ void cvt4raw(const uint2 &u, float (&f)[4]) {
  f[0] = __uint_as_float(u.x << 16); f[1] = __uint_as_float(u.x & 0xFFFF0000u);
  f[2] = __uint_as_float(u.y << 16); f[3] = __uint_as_float(u.y & 0xFFFF0000u);
}
__device__ __forceinline__ void st4(float *p, const float (&f)[4]) {
  *(float4 *)p = make_float4(f[0], f[1], f[2], f[3]);
}
__device__ __forceinline__ void st4(__nv_bfloat16 *p, const float (&f)[4]) {
  const __nv_bfloat162 a = __floats2bfloat162_rn(f[0], f[1]), b = __floats2bfloat162_rn(f[2], f[3]);
  *(uint2 *)p = make_uint2(*reinterpret_cast<const uint32_t *>(&a),
                           *reinterpret_cast<const uint32_t *>(&b));
}

// Asynchronous copy of BYTES (8 or 16) global bytes into shared memory; the
// destination is zero-filled when src_bytes is 0 (src must still be a valid
// address, and is not read).
template <int BYTES>
__device__ __forceinline__ void cp_async_z(uint32_t dst, const void *src, uint32_t src_bytes) {
  if constexpr (BYTES == 16)
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src),
                 "r"(src_bytes)
                 : "memory");
  else
    asm volatile("cp.async.ca.shared.global [%0], [%1], %2, %3;" ::"r"(dst), "l"(src),
                 "n"(BYTES), "r"(src_bytes)
                 : "memory");
}
// Steps of the Conv1D backward whose loads are staged together, and the
// dynamic shared memory of the staging buffers (two batches in flight).
template <typename T>
constexpr int conv_batch() { return sizeof(T) == 2 ? 8 : 4; }
template <typename T>
constexpr size_t conv_stage_bytes() {
  return (size_t)2 * 2 * conv_batch<T>() * kNT * sizeof(typename Raw4<T>::type);
}

template <typename T, int D>
__global__ void __launch_bounds__(kNT, 2) bwd_conv(
    const T *__restrict__ q, const T *__restrict__ k, const T *__restrict__ v,
    const T *__restrict__ dxt, const float *__restrict__ conv_w,
    const int32_t *__restrict__ seq_lens, T *__restrict__ dq, T *__restrict__ dk,
    T *__restrict__ dv, float *__restrict__ wpart, int H, int N, int nck, int rl) {
  constexpr int G = D / kConvCh, RUNS = kNT / G;
  __shared__ float sw[RUNS][D * kConvW];
  // v first: its dv~ plane is the one most recently written (by the key pass)
  // and the most likely still to sit in L2 when the first blocks run
  const int chunk = blockIdx.x, bh = blockIdx.y, s = 2 - (int)blockIdx.z, b = bh / H, h = bh % H;
  const int tid = threadIdx.x, g = tid % G, run = tid / G;
  const T *x = s == 0 ? q : (s == 1 ? k : v);
  T *dx = s == 0 ? dq : (s == 1 ? dk : dv);
  const T *dxs = dxt + (size_t)s * ((size_t)gridDim.y / H) * N * H * D;
  const int L = clamp_len(seq_lens, b, N);
  const int ta = (chunk * RUNS + run) * rl, tb = min(ta + rl, N);
  float w[kConvCh][kConvW], dw[kConvCh][kConvW];
#pragma unroll
  for (int c = 0; c < kConvCh; ++c) {
    const float4 t4 =
        __ldg((const float4 *)(conv_w + ((size_t)(s * H + h) * D + kConvCh * g + c) * kConvW));
    w[c][0] = t4.x; w[c][1] = t4.y; w[c][2] = t4.z; w[c][3] = t4.w;
#pragma unroll
    for (int i = 0; i < kConvW; ++i) dw[c][i] = 0.f;
  }
  sm100::grid_dep_wait();  // the dx~ planes come from the token passes
  sm100::grid_dep_launch();
  const size_t rs = (size_t)H * D;
  const size_t col = ((size_t)b * N * H + h) * D + kConvCh * g;
  auto ldx = [&](int t, float (&f)[kConvCh]) {  // x_t, zero outside [0, L)
    if (t >= 0 && t < L) ld4(x + col + (size_t)t * rs, f);
    else
#pragma unroll
      for (int c = 0; c < kConvCh; ++c) f[c] = 0.f;
  };
  auto ldd = [&](int t, float (&f)[kConvCh]) {  // dx~_t, zero outside [0, L)
    if (t >= 0 && t < L) ld4(dxs + col + (size_t)t * rs, f);
    else
#pragma unroll
      for (int c = 0; c < kConvCh; ++c) f[c] = 0.f;
  };
  // xm[i] = x_{t-3+i} (i = 0..2), dm[i] = dx~_{t+i} (i = 0..2)
  float xm[3][kConvCh], dm[3][kConvCh];
#pragma unroll
  for (int i = 0; i < 3; ++i) {
    ldx(ta - 3 + i, xm[i]);
    ldd(ta + i, dm[i]);
  }
  // U steps at a time: their 2 U loads go to shared memory by cp.async (no
  // registers held while they are in flight), the next batch's copies are
  // issued before this batch is converted, and each thread reads back only
  // its own slots (no barrier).  Rows at or past L are zero-filled.
  using Raw = typename Raw4<T>::type;
  constexpr int U = conv_batch<T>();
  constexpr int RB = (int)sizeof(Raw);
  extern __shared__ __align__(16) uint8_t conv_stage[];
  // this thread's slot for x (arr 0) or dx~ (arr 1) of step u in batch buffer buf
  auto slot_off = [&](int buf, int arr, int u) {
    return (uint32_t)((((buf * 2 + arr) * U + u) * kNT + tid) * RB);
  };
  const uint32_t stg0 = (uint32_t)__cvta_generic_to_shared(conv_stage);
  const int nbat = (tb - ta + U - 1) / U;
  auto issue = [&](int bt) {
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int tx = ta + bt * U + u, td = tx + 3;
      const bool vx = tx < tb && tx < L, vd = tx < tb && td < L;
      cp_async_z<RB>(stg0 + slot_off(bt & 1, 0, u), x + col + (vx ? (size_t)tx * rs : 0),
                     vx ? RB : 0);
      cp_async_z<RB>(stg0 + slot_off(bt & 1, 1, u), dxs + col + (vd ? (size_t)td * rs : 0),
                     vd ? RB : 0);
    }
    asm volatile("cp.async.commit_group;" ::: "memory");
  };
  if (nbat > 0) issue(0);
  for (int bt = 0; bt < nbat; ++bt) {
    if (bt + 1 < nbat) {
      issue(bt + 1);
      asm volatile("cp.async.wait_group 1;" ::: "memory");
    } else {
      asm volatile("cp.async.wait_group 0;" ::: "memory");
    }
#pragma unroll
    for (int u = 0; u < U; ++u) {
    const int t = ta + bt * U + u;
    if (t >= tb) break;
    float xc[kConvCh], dn[kConvCh], o[kConvCh];
    cvt4raw(*(const Raw *)(conv_stage + slot_off(bt & 1, 0, u)), xc);  // x_t
    cvt4raw(*(const Raw *)(conv_stage + slot_off(bt & 1, 1, u)), dn);  // dx~_{t+3}
#pragma unroll
    for (int c = 0; c < kConvCh; ++c) {
      // dx_t = w0 dx~_{t+3} + w1 dx~_{t+2} + w2 dx~_{t+1} + w3 dx~_t
      float a = w[c][0] * dn[c];
      a = fmaf(w[c][1], dm[2][c], a);
      a = fmaf(w[c][2], dm[1][c], a);
      a = fmaf(w[c][3], dm[0][c], a);
      o[c] = t < L ? a : 0.f;
      // dw_i += dx~_t x_{t-3+i}  (dx~_t = 0 past L)
      dw[c][0] = fmaf(dm[0][c], xm[0][c], dw[c][0]);
      dw[c][1] = fmaf(dm[0][c], xm[1][c], dw[c][1]);
      dw[c][2] = fmaf(dm[0][c], xm[2][c], dw[c][2]);
      dw[c][3] = fmaf(dm[0][c], xc[c], dw[c][3]);
    }
    st4(dx + col + (size_t)t * rs, o);
#pragma unroll
    for (int c = 0; c < kConvCh; ++c) {
      xm[0][c] = xm[1][c]; xm[1][c] = xm[2][c]; xm[2][c] = xc[c];
      dm[0][c] = dm[1][c]; dm[1][c] = dm[2][c]; dm[2][c] = dn[c];
    }
    }
  }
#pragma unroll
  for (int c = 0; c < kConvCh; ++c)
#pragma unroll
    for (int i = 0; i < kConvW; ++i) sw[run][(kConvCh * g + c) * kConvW + i] = dw[c][i];
  __syncthreads();
  for (int j = tid; j < D * kConvW; j += kNT) {
    float a = 0.f;
    for (int r = 0; r < RUNS; ++r) a += sw[r][j];
    wpart[(((size_t)s * gridDim.y + bh) * nck + chunk) * D * kConvW + j] = a;
  }
}

// ---------------------------------------------------------------- weight reductions
// dconv_w[s][h][c][i] = sum_b sum_chunk wpart (nck chunks);  dnorm_w[h][c] = sum_b
// sum_chunk qpart.dnw (nckq query-pass records per (b, h)).  A block takes 32
// consecutive outputs (one per lane); its 8 warps take interleaved slices of
// the (b, chunk) partials, read coalesced across the lanes, and the 8 warp
// sums are added in warp order.
template <int D>
__global__ void __launch_bounds__(256) bwd_reduce_w(const float *__restrict__ wpart,
                                                    const float *__restrict__ qpart,
                                                    float *__restrict__ dconv_w,
                                                    float *__restrict__ dnorm_w, int B, int H,
                                                    int nck, int nckq) {
  const int total_w = 3 * H * D * kConvW;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int idx = blockIdx.x * 32 + lane;
  __shared__ float part[8][32];
  sm100::grid_dep_wait();  // the tap partials come from the Conv1D backward
  sm100::grid_dep_launch();
  float a = 0.f;
  if (idx < total_w) {
    const int s = idx / (H * D * kConvW), r = idx % (H * D * kConvW);
    const int h = r / (D * kConvW), ci = r % (D * kConvW);
    const int n = B * nck;
    for (int k = warp; k < n; k += 8) {
      const int b = k / nck, ch = k % nck;
      a += wpart[(((size_t)s * B * H + (size_t)b * H + h) * nck + ch) * D * kConvW + ci];
    }
  } else if (idx < total_w + H * D) {
    const int j = idx - total_w, h = j / D, cc = j % D;
    const int n = B * nckq;
    for (int k = warp; k < n; k += 8) {
      const int b = k / nckq, ch = k % nckq;
      a += qpart[(((size_t)b * H + h) * nckq + ch) * qrec<D>() + D * D + D + cc];
    }
  }
  part[warp][lane] = a;
  __syncthreads();
  if (warp == 0) {
    float t = 0.f;
    for (int w = 0; w < 8; ++w) t += part[w][lane];
    if (idx < total_w) dconv_w[idx] = t;
    else if (idx < total_w + H * D) dnorm_w[idx - total_w] = t;
  }
}

template <typename T, int D>
cudaError_t run_bwd(const Problem &p, const BwdArgs &a, float *scratch, bool stats_ready,
                    cudaStream_t st) {
  const int B = p.B, H = p.H, N = p.N, BH = B * H;
  const int nck = (N + kChunk - 1) / kChunk;
  const BwdLayout lay = bwd_layout(p);
  float2 *stats_w = (float2 *)(scratch + lay.stats);  // filled here unless stats_ready
  const float2 *stats = stats_ready ? a.stats : stats_w;
  float *qpart = scratch + lay.qpart, *red = scratch + lay.red;
  T *dxt = (T *)(scratch + lay.dxt);  // dq~, dk~, dv~ planes in the storage dtype
  float *wpart = scratch + lay.wpart;
  const float *state = a.state;
  const size_t plane = (size_t)B * N * H * D;
  cudaError_t e;
  float2 *gpart = (float2 *)(scratch + lay.gpart);
  if (!stats_ready) {
    bwd_gate_split<T><<<dim3(BH, kGateSplits), 256, 0, st>>>((const T *)a.gate, p.seq_lens,
                                                             gpart, H, N);
    bwd_gate_join<<<(BH + 255) / 256, 256, 0, st>>>(gpart, stats_w, BH);
    count_launch(2);
  }
  constexpr int TPT = Tok<D>::TPT, kTB = Tok<D>::TB;
  const size_t smq = sizeof(float) * (2 * D * D + D + 4 * D * kTB + kTB + kNT / 32 * TPT);
  const bool tc = bwd_tc_key_supported(p);  // bf16, D = 64, sm_103: both token passes on tcgen05
  int nckq = nck;                           // partial records of the query pass per (b, h)
  if (tc) {
    nckq = bwd_tc_query_chunks(p);
    if ((e = bwd_tc_query(p, a, state, qpart, dxt, st)) != cudaSuccess) return e;
  } else {
    auto kq = bwd_query<T, D>;
    if ((e = cudaFuncSetAttribute(kq, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smq)) !=
        cudaSuccess)
      return e;
    kq<<<dim3(nck, BH), kNT, smq, st>>>((const T *)a.q, (const T *)a.out_gate, (const T *)a.dy,
                                        a.conv_w, a.norm_w, state, p.seq_lens, kRmsEps,
                                        (T *)a.dout_gate, dxt, qpart, H, N, nck,
                                        (p.flags & GBLA_FLAG_NO_NORM) ? 1 : 0);
    count_launch();
  }
  constexpr int F = D * D + D;
  // on tensor cores the key pass forms c from the reduction's partial dot products
  if ((e = launch_pdl(bwd_reduce_state<D>, dim3((F + 255) / 256, BH), dim3(256), 0, st,
                      (const float *)qpart, red, tc ? state : nullptr,
                      tc ? scratch + lay.cpart : nullptr, nckq)) != cudaSuccess)
    return e;
  count_launch();
  if (tc) {
    if ((e = bwd_tc_key(p, a, stats, red, scratch + lay.cpart, (F + 255) / 256, dxt + plane,
                        dxt + 2 * plane, st)) != cudaSuccess)
      return e;
  } else {
  const size_t smk = sizeof(float) * (2 * D * D + D + 2 * D * kTB + kNT / 32 * TPT);
  auto kk = bwd_key<T, D>;
  if ((e = cudaFuncSetAttribute(kk, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smk)) !=
      cudaSuccess)
    return e;
  kk<<<dim3(nck, BH), kNT, smk, st>>>((const T *)a.k, (const T *)a.v, (const T *)a.gate,
                                      a.conv_w, stats, state, red, p.seq_lens, (T *)a.dgate,
                                      dxt + plane, dxt + 2 * plane, H, N);
  count_launch();
  }
  // Conv1D backward: 64 tokens a thread run (measured against 32..128-token
  // runs chosen to fill whole waves: those were slower)
  constexpr int kRuns = kNT / (D / kConvCh);
  const int rl = 64;
  const int nckc = (N + kRuns * rl - 1) / (kRuns * rl);  // Conv1D backward blocks per (b, h)
  // the staging buffers exceed the default 48 KB of dynamic shared memory
  if ((e = cudaFuncSetAttribute(bwd_conv<T, D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                (int)conv_stage_bytes<T>())) != cudaSuccess)
    return e;
  if ((e = launch_pdl(bwd_conv<T, D>, dim3(nckc, BH, 3), dim3(kNT), conv_stage_bytes<T>(), st,
                      (const T *)a.q, (const T *)a.k, (const T *)a.v, (const T *)dxt, a.conv_w,
                      p.seq_lens, (T *)a.dq, (T *)a.dk, (T *)a.dv, wpart, H, N, nckc, rl)) !=
      cudaSuccess)
    return e;
  count_launch();
  const int nw = 3 * H * D * kConvW + H * D;
  if ((e = launch_pdl(bwd_reduce_w<D>, dim3((nw + 31) / 32), dim3(256), 0, st,
                      (const float *)wpart, (const float *)qpart, a.dconv_w, a.dnorm_w, B, H,
                      nckc, nckq)) != cudaSuccess)
    return e;
  count_launch();
  return cudaGetLastError();
}

}  // namespace

BwdLayout bwd_layout(const Problem &p) {
  const size_t BH = (size_t)p.B * p.H, D = p.D;
  const size_t nck = ((size_t)p.N + kChunk - 1) / kChunk;
  const size_t F = D * D + D;
  auto up = [](size_t x) { return (x + 63) / 64 * 64; };  // 256-byte aligned (in floats)
  BwdLayout l;
  l.state = 0;
  l.stats = up(l.state + BH * F);
  l.gpart = up(l.stats + 2 * BH);
  l.qpart = up(l.gpart + 2 * BH * kGateSplits);
  l.red = up(l.qpart + BH * nck * (D * D + 2 * D));
  l.cpart = up(l.red + BH * (F + 1));
  l.dxt = up(l.cpart + BH * ((F + 255) / 256));
  l.wpart = up(l.dxt + 3 * BH * (size_t)p.N * D);
  l.total = up(l.wpart + 3 * BH * nck * D * kConvW);
  return l;
}

cudaError_t gate_stats(const Problem &p, const void *gate, float2 *part, float2 *stats,
                       cudaStream_t st) {
  const int BH = p.B * p.H;
  if (p.dtype == GBLA_BF16)
    bwd_gate_split<__nv_bfloat16><<<dim3(BH, kGateSplits), 256, 0, st>>>(
        (const __nv_bfloat16 *)gate, p.seq_lens, part, p.H, p.N);
  else
    bwd_gate_split<float><<<dim3(BH, kGateSplits), 256, 0, st>>>((const float *)gate, p.seq_lens,
                                                                 part, p.H, p.N);
  bwd_gate_join<<<(BH + 255) / 256, 256, 0, st>>>(part, stats, BH);
  count_launch(2);
  return cudaGetLastError();
}
size_t gate_stats_part_floats(const Problem &p) { return (size_t)2 * p.B * p.H * kGateSplits; }

namespace {
// Taps (0, 0, 0, 1) on n channels: the identity Conv1D (tap 3 on the current token).
__global__ void __launch_bounds__(256) identity_taps(float4 *__restrict__ taps, int n) {
  const int i = blockIdx.x * 256 + threadIdx.x;
  if (i < n) taps[i] = make_float4(0.f, 0.f, 0.f, 1.f);
}
}  // namespace

cudaError_t fill_identity_taps(float *taps, int n, cudaStream_t st) {
  if (n <= 0) return cudaSuccess;
  identity_taps<<<(n + 255) / 256, 256, 0, st>>>((float4 *)taps, n);
  count_launch();
  return cudaGetLastError();
}

cudaError_t bwd_run(const Problem &p, const BwdArgs &a, float *scratch, bool stats_ready,
                    cudaStream_t st) {
  if (p.dtype == GBLA_BF16) {
    switch (p.D) {
      case 32: return run_bwd<__nv_bfloat16, 32>(p, a, scratch, stats_ready, st);
      case 64: return run_bwd<__nv_bfloat16, 64>(p, a, scratch, stats_ready, st);
      case 128: return run_bwd<__nv_bfloat16, 128>(p, a, scratch, stats_ready, st);
    }
  } else {
    switch (p.D) {
      case 32: return run_bwd<float, 32>(p, a, scratch, stats_ready, st);
      case 64: return run_bwd<float, 64>(p, a, scratch, stats_ready, st);
      case 128: return run_bwd<float, 128>(p, a, scratch, stats_ready, st);
    }
  }
  return cudaErrorInvalidValue;
}

}  // namespace gbla
