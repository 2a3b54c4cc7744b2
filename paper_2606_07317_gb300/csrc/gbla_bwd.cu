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
//   bwd_gate_stats   per (b, h): M = max a, Ltot = sum e^{a - M} (g_j = e^{a_j-M}/Ltot)
//   bwd_query        per (b, h, chunk): 5' and 6' per token; dq~ to scratch;
//                    chunk partials of dS, dz and the norm-weight gradient
//   bwd_reduce_state per (b, h): fixed-order sums of the partials; c
//   bwd_key          per (b, h, chunk): 4' and 3' per token; dk~, dv~ to scratch
//   bwd_conv         per (stream, b, h, chunk): 1' (anti-causal taps) into dq,
//                    dk, dv; chunk partials of the tap gradients
//   bwd_reduce_w     fixed-order sums of the tap / norm-weight partials
// Every sum runs in a fixed order, so the results are deterministic.
#include <math.h>

#include "gbla_internal.cuh"

namespace gbla {
namespace {

constexpr int kBG = 4;        // tokens in flight per block (one thread group each)
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
__device__ __forceinline__ float warp_max(float x) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) x = fmaxf(x, __shfl_xor_sync(0xffffffffu, x, o));
  return x;
}

// Sum of x over the D threads of each token group (kBG groups side by side);
// every thread of the block calls it.  red: kBG * (D / 32) floats of shared memory.
template <int D>
__device__ __forceinline__ float group_sum(float x, float *red) {
  constexpr int WPG = D / 32;
  const int w = threadIdx.x >> 5, g = threadIdx.x / D;
  x = warp_sum(x);
  __syncthreads();  // red free from the previous use
  if ((threadIdx.x & 31) == 0) red[w] = x;
  __syncthreads();
  float s = 0.f;
#pragma unroll
  for (int i = 0; i < WPG; ++i) s += red[g * WPG + i];
  return s;
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
template <typename T>
__global__ void __launch_bounds__(256) bwd_gate_stats(const T *__restrict__ gate,
                                                      const int32_t *__restrict__ seq_lens,
                                                      float2 *__restrict__ stats, int H, int N) {
  const int bh = blockIdx.x, b = bh / H, h = bh % H;
  const int L = clamp_len(seq_lens, b, N);
  __shared__ float red[8];
  float m = -INFINITY;
  for (int t = threadIdx.x; t < L; t += 256) m = fmaxf(m, ldf(gate, ((size_t)b * N + t) * H + h));
  m = warp_max(m);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = m;
  __syncthreads();
  float M = red[0];
  for (int i = 1; i < 8; ++i) M = fmaxf(M, red[i]);
  __syncthreads();
  float l = 0.f;
  for (int t = threadIdx.x; t < L; t += 256) l += expf(ldf(gate, ((size_t)b * N + t) * H + h) - M);
  l = warp_sum(l);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = l;
  __syncthreads();
  if (threadIdx.x == 0) {
    float s = 0.f;
    for (int i = 0; i < 8; ++i) s += red[i];
    stats[bh] = make_float2(M, s);
  }
}

// ---------------------------------------------------------------- query pass
// Partial record per (b, h, chunk): dS [D][D], dz [D], dnorm_w [D].
template <int D>
constexpr int qrec() { return D * D + 2 * D; }

template <typename T, int D>
__global__ void __launch_bounds__(kBG * D) bwd_query(
    const T *__restrict__ q, const T *__restrict__ og, const T *__restrict__ dy,
    const float *__restrict__ conv_w, const float *__restrict__ norm_w,
    const float *__restrict__ state, const int32_t *__restrict__ seq_lens, float eps,
    T *__restrict__ dog, float *__restrict__ dqt, float *__restrict__ part, int H, int N,
    int nck) {
  constexpr int NT = kBG * D;
  constexpr int F = D * D + D;
  constexpr int PE = D * D / NT;  // dS entries per thread
  extern __shared__ float sm[];
  float *S = sm, *St = S + D * D, *z = St + D * D;
  float *sP = z + D, *sDn = sP + kBG * D, *sDd = sDn + kBG * D, *red = sDd + kBG;
  const int chunk = blockIdx.x, bh = blockIdx.y, b = bh / H, h = bh % H;
  const int tid = threadIdx.x, g = tid / D, c = tid % D;
  const int L = clamp_len(seq_lens, b, N);
  const int t0 = chunk * kChunk, t1 = min(t0 + kChunk, N);
  const float *st = state + (size_t)bh * F;
  for (int i = tid; i < D * D; i += NT) {
    const float x = st[i];
    S[i] = x;
    St[(i % D) * D + i / D] = x;
  }
  for (int i = tid; i < D; i += NT) z[i] = st[D * D + i];
  float wq[kConvW];
#pragma unroll
  for (int i = 0; i < kConvW; ++i) wq[i] = conv_w[((size_t)h * D + c) * kConvW + i];
  const float nw = norm_w[(size_t)h * D + c];
  const size_t rs = (size_t)H * D;
  const T *qc = q + ((size_t)b * N * H + h) * D + c;
  float dS[PE];
#pragma unroll
  for (int k = 0; k < PE; ++k) dS[k] = 0.f;
  float dz = 0.f, dnw = 0.f;
  __syncthreads();
  for (int base = t0; base < t1; base += kBG) {
    const int t = base + g;
    const bool valid = t < min(t1, L);
    const size_t row = (((size_t)b * N + t) * H + h) * D + c;
    const float qt = valid ? conv_at(qc, rs, t, wq) : 0.f;
    const float P = valid ? phi(qt) : 0.f;
    sP[g * D + c] = P;
    __syncthreads();
    float num = 0.f, den = 0.f;
#pragma unroll 8
    for (int d = 0; d < D; ++d) {
      const float pd = sP[g * D + d];
      num = fmaf(pd, S[d * D + c], num);
      den = fmaf(pd, z[d], den);
    }
    const float O = valid ? num / den : 0.f;
    const float ogv = valid ? ldf(og, row) : 0.f, dyv = valid ? ldf(dy, row) : 0.f;
    const float ms = group_sum<D>(O * O, red) / (float)D;
    const float r = 1.f / sqrtf(ms + eps);
    const float sg = 1.f / (1.f + expf(-ogv)), si = ogv * sg;
    if (t < t1) stf(dog, row, valid ? dyv * O * r * nw * sg * (1.f + ogv * (1.f - sg)) : 0.f);
    dnw = fmaf(dyv * O, r * si, dnw);
    const float u = dyv * nw * si;
    const float uo = group_sum<D>(u * O, red);
    const float dO = r * u - (r * r * r / (float)D) * O * uo;
    const float dnum = valid ? dO / den : 0.f;
    const float dOO = group_sum<D>(dO * O, red);
    const float dden = valid ? -dOO / den : 0.f;
    sDn[g * D + c] = dnum;
    if (c == 0) sDd[g] = dden;
    __syncthreads();
    float dP = z[c] * dden;
#pragma unroll 8
    for (int e = 0; e < D; ++e) dP = fmaf(St[e * D + c], sDn[g * D + e], dP);
    if (t < t1) dqt[row] = valid ? dP * dphi(qt) : 0.f;
    dz = fmaf(P, dden, dz);
#pragma unroll
    for (int k = 0; k < PE; ++k) {
      const int ent = tid + k * NT, d = ent / D, e = ent % D;
      float a = dS[k];
#pragma unroll
      for (int gg = 0; gg < kBG; ++gg) a = fmaf(sP[gg * D + d], sDn[gg * D + e], a);
      dS[k] = a;
    }
    __syncthreads();  // sP, sDn reused by the next tokens
  }
  // partial record: dS by entry; dz and dnw summed over the token groups in order
  float *rec = part + ((size_t)bh * nck + chunk) * qrec<D>();
#pragma unroll
  for (int k = 0; k < PE; ++k) rec[tid + k * NT] = dS[k];
  sP[g * D + c] = dz;
  sDn[g * D + c] = dnw;
  __syncthreads();
  if (tid < D) {
    float a = 0.f, w = 0.f;
    for (int gg = 0; gg < kBG; ++gg) {
      a += sP[gg * D + tid];
      w += sDn[gg * D + tid];
    }
    rec[D * D + tid] = a;
    rec[D * D + D + tid] = w;
  }
}

// ---------------------------------------------------------------- state reduction
// red record per (b, h): dS [D][D], dz [D], c.
template <int D>
__global__ void __launch_bounds__(256) bwd_reduce_state(const float *__restrict__ part,
                                                        const float *__restrict__ state,
                                                        float *__restrict__ red, int nck) {
  constexpr int F = D * D + D;
  const int bh = blockIdx.x;
  __shared__ float wred[8];
  float cs = 0.f;
  for (int i = threadIdx.x; i < F; i += 256) {
    float a = 0.f;
    for (int ch = 0; ch < nck; ++ch) a += part[((size_t)bh * nck + ch) * qrec<D>() + i];
    red[(size_t)bh * (F + 1) + i] = a;
    cs = fmaf(a, state[(size_t)bh * F + i], cs);
  }
  cs = warp_sum(cs);
  if ((threadIdx.x & 31) == 0) wred[threadIdx.x >> 5] = cs;
  __syncthreads();
  if (threadIdx.x == 0) {
    float s = 0.f;
    for (int i = 0; i < 8; ++i) s += wred[i];
    red[(size_t)bh * (F + 1) + F] = s;
  }
}

// ---------------------------------------------------------------- key pass
template <typename T, int D>
__global__ void __launch_bounds__(kBG * D) bwd_key(
    const T *__restrict__ k, const T *__restrict__ v, const T *__restrict__ gate,
    const float *__restrict__ conv_w, const float2 *__restrict__ stats,
    const float *__restrict__ red, const int32_t *__restrict__ seq_lens, T *__restrict__ dgate,
    float *__restrict__ dkt, float *__restrict__ dvt, int H, int N) {
  constexpr int NT = kBG * D;
  constexpr int F = D * D + D;
  extern __shared__ float sm[];
  float *dS = sm, *dSt = dS + D * D, *dz = dSt + D * D;
  float *sK = dz + D, *sV = sK + kBG * D, *rd = sV + kBG * D;
  const int chunk = blockIdx.x, bh = blockIdx.y, b = bh / H, h = bh % H;
  const int tid = threadIdx.x, g = tid / D, c = tid % D;
  const int L = clamp_len(seq_lens, b, N);
  const int t0 = chunk * kChunk, t1 = min(t0 + kChunk, N);
  const float *rr = red + (size_t)bh * (F + 1);
  for (int i = tid; i < D * D; i += NT) {
    const float x = rr[i];
    dS[i] = x;
    dSt[(i % D) * D + i / D] = x;
  }
  for (int i = tid; i < D; i += NT) dz[i] = rr[D * D + i];
  const float cval = rr[F];
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
  __syncthreads();
  for (int base = t0; base < t1; base += kBG) {
    const int t = base + g;
    const bool valid = t < min(t1, L);
    const size_t row = (((size_t)b * N + t) * H + h) * D + c;
    const float kt = valid ? conv_at(kc, rs, t, wk) : 0.f;
    const float vt = valid ? conv_at(vc, rs, t, wv) : 0.f;
    const float gj = valid ? expf(ldf(gate, ((size_t)b * N + t) * H + h) - gs.x) / gs.y : 0.f;
    const float pk = valid ? phi(kt) : 0.f;
    sK[g * D + c] = gj * pk;
    sV[g * D + c] = vt;
    __syncthreads();
    float dK = dz[c], dvv = 0.f;
#pragma unroll 8
    for (int e = 0; e < D; ++e) {
      dK = fmaf(dSt[e * D + c], sV[g * D + e], dK);
      dvv = fmaf(sK[g * D + e], dS[e * D + c], dvv);
    }
    if (t < t1) {
      dkt[row] = valid ? gj * dK * dphi(kt) : 0.f;
      dvt[row] = valid ? dvv : 0.f;
    }
    const float dg = group_sum<D>(pk * dK, rd);
    if (c == 0 && t < t1) stf(dgate, ((size_t)b * N + t) * H + h, valid ? gj * (dg - cval) : 0.f);
    __syncthreads();  // sK, sV reused by the next tokens
  }
}

// ---------------------------------------------------------------- Conv1D backward
// Stream s (0 q, 1 k, 2 v): dx_t = sum_i w_i dx~_{t+3-i} (t + 3 - i < L), and the
// chunk partials of dw_i = sum_t dx~_t x_{t-3+i} for the D channels of (b, h).
template <typename T, int D>
__global__ void __launch_bounds__(kBG * D) bwd_conv(
    const T *__restrict__ x, const float *__restrict__ dxt, const float *__restrict__ conv_w,
    const int32_t *__restrict__ seq_lens, T *__restrict__ dx, float *__restrict__ wpart, int s,
    int H, int N, int nck) {
  constexpr int NT = kBG * D;
  __shared__ float sw[kBG][D][kConvW];
  const int chunk = blockIdx.x, bh = blockIdx.y, b = bh / H, h = bh % H;
  const int tid = threadIdx.x, g = tid / D, c = tid % D;
  const int L = clamp_len(seq_lens, b, N);
  const int t0 = chunk * kChunk, t1 = min(t0 + kChunk, N);
  float w[kConvW], dw[kConvW];
#pragma unroll
  for (int i = 0; i < kConvW; ++i) {
    w[i] = conv_w[((size_t)(s * H + h) * D + c) * kConvW + i];
    dw[i] = 0.f;
  }
  const size_t rs = (size_t)H * D;
  const size_t col = ((size_t)b * N * H + h) * D + c;
  for (int t = t0 + g; t < t1; t += kBG) {
    float a = 0.f;
    if (t < L) {
#pragma unroll
      for (int i = 0; i < kConvW; ++i) {
        const int u = t + (kConvW - 1) - i;
        if (u < L) a = fmaf(w[i], dxt[col + (size_t)u * rs], a);
      }
      const float d = dxt[col + (size_t)t * rs];
#pragma unroll
      for (int i = 0; i < kConvW; ++i) {
        const int u = t - (kConvW - 1) + i;
        if (u >= 0) dw[i] = fmaf(d, ldf(x, col + (size_t)u * rs), dw[i]);
      }
    }
    stf(dx, col + (size_t)t * rs, a);
  }
#pragma unroll
  for (int i = 0; i < kConvW; ++i) sw[g][c][i] = dw[i];
  __syncthreads();
  if (tid < D * kConvW) {
    const int cc = tid / kConvW, i = tid % kConvW;
    float a = 0.f;
    for (int gg = 0; gg < kBG; ++gg) a += sw[gg][cc][i];
    wpart[(((size_t)s * gridDim.y + bh) * nck + chunk) * D * kConvW + tid] = a;
  }
  (void)NT;
}

// ---------------------------------------------------------------- weight reductions
// dconv_w[s][h][c][i] = sum_b sum_chunk wpart;  dnorm_w[h][c] = sum_b sum_chunk qpart.dnw
template <int D>
__global__ void __launch_bounds__(256) bwd_reduce_w(const float *__restrict__ wpart,
                                                    const float *__restrict__ qpart,
                                                    float *__restrict__ dconv_w,
                                                    float *__restrict__ dnorm_w, int B, int H,
                                                    int nck) {
  const int total_w = 3 * H * D * kConvW;
  for (int idx = blockIdx.x * 256 + threadIdx.x; idx < total_w + H * D;
       idx += gridDim.x * 256) {
    float a = 0.f;
    if (idx < total_w) {
      const int s = idx / (H * D * kConvW), r = idx % (H * D * kConvW);
      const int h = r / (D * kConvW), ci = r % (D * kConvW);
      for (int b = 0; b < B; ++b)
        for (int ch = 0; ch < nck; ++ch)
          a += wpart[(((size_t)s * B * H + (size_t)b * H + h) * nck + ch) * D * kConvW + ci];
      dconv_w[idx] = a;
    } else {
      const int j = idx - total_w, h = j / D, cc = j % D;
      for (int b = 0; b < B; ++b)
        for (int ch = 0; ch < nck; ++ch)
          a += qpart[(((size_t)b * H + h) * nck + ch) * qrec<D>() + D * D + D + cc];
      dnorm_w[j] = a;
    }
  }
}

template <typename T, int D>
cudaError_t run_bwd(const Problem &p, const BwdArgs &a, float *scratch, cudaStream_t st) {
  const int B = p.B, H = p.H, N = p.N, BH = B * H;
  const int nck = (N + kChunk - 1) / kChunk;
  const BwdLayout lay = bwd_layout(p);
  float2 *stats = (float2 *)(scratch + lay.stats);
  float *qpart = scratch + lay.qpart, *red = scratch + lay.red, *dxt = scratch + lay.dxt;
  float *wpart = scratch + lay.wpart;
  const float *state = scratch + lay.state;
  const size_t plane = (size_t)B * N * H * D;
  cudaError_t e;
  bwd_gate_stats<T><<<BH, 256, 0, st>>>((const T *)a.gate, p.seq_lens, stats, H, N);
  count_launch();
  const size_t smq = sizeof(float) * (2 * D * D + D + 2 * kBG * D + kBG + kBG * D / 32);
  auto kq = bwd_query<T, D>;
  if ((e = cudaFuncSetAttribute(kq, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smq)) !=
      cudaSuccess)
    return e;
  kq<<<dim3(nck, BH), kBG * D, smq, st>>>((const T *)a.q, (const T *)a.out_gate,
                                         (const T *)a.dy, a.conv_w, a.norm_w, state, p.seq_lens,
                                         kRmsEps, (T *)a.dout_gate, dxt, qpart, H, N, nck);
  count_launch();
  bwd_reduce_state<D><<<BH, 256, 0, st>>>(qpart, state, red, nck);
  count_launch();
  const size_t smk = sizeof(float) * (2 * D * D + D + 2 * kBG * D + kBG * D / 32);
  auto kk = bwd_key<T, D>;
  if ((e = cudaFuncSetAttribute(kk, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smk)) !=
      cudaSuccess)
    return e;
  kk<<<dim3(nck, BH), kBG * D, smk, st>>>((const T *)a.k, (const T *)a.v, (const T *)a.gate,
                                         a.conv_w, stats, red, p.seq_lens, (T *)a.dgate,
                                         dxt + plane, dxt + 2 * plane, H, N);
  count_launch();
  const void *xs[3] = {a.q, a.k, a.v};
  void *dxs[3] = {a.dq, a.dk, a.dv};
  for (int s = 0; s < 3; ++s) {
    bwd_conv<T, D><<<dim3(nck, BH), kBG * D, 0, st>>>((const T *)xs[s], dxt + s * plane,
                                                      a.conv_w, p.seq_lens, (T *)dxs[s], wpart,
                                                      s, H, N, nck);
    count_launch();
  }
  const int nw = 3 * H * D * kConvW + H * D;
  bwd_reduce_w<D><<<(nw + 255) / 256, 256, 0, st>>>(wpart, qpart, a.dconv_w, a.dnorm_w, B, H,
                                                     nck);
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
  l.qpart = up(l.stats + 2 * BH);
  l.red = up(l.qpart + BH * nck * (D * D + 2 * D));
  l.dxt = up(l.red + BH * (F + 1));
  l.wpart = up(l.dxt + 3 * BH * (size_t)p.N * D);
  l.total = up(l.wpart + 3 * BH * nck * D * kConvW);
  return l;
}

cudaError_t bwd_run(const Problem &p, const BwdArgs &a, float *scratch, cudaStream_t st) {
  if (p.dtype == GBLA_BF16) {
    switch (p.D) {
      case 32: return run_bwd<__nv_bfloat16, 32>(p, a, scratch, st);
      case 64: return run_bwd<__nv_bfloat16, 64>(p, a, scratch, st);
      case 128: return run_bwd<__nv_bfloat16, 128>(p, a, scratch, st);
    }
  } else {
    switch (p.D) {
      case 32: return run_bwd<float, 32>(p, a, scratch, st);
      case 64: return run_bwd<float, 64>(p, a, scratch, st);
      case 128: return run_bwd<float, 128>(p, a, scratch, st);
    }
  }
  return cudaErrorInvalidValue;
}

}  // namespace gbla
