// CUDA-core (SIMT) kernels of the GBLA core: every dtype and D in {32, 64, 128}.
//
// This family carries the exact-fp32 path (fp32 storage, fp32 FMA, accurate
// expf/division) and serves as the always-available kernel set.  The bf16
// tensor-core family lives in gbla_tc.cu.
//
// Steps (Sec. 2.1):
//   simt_partials_kernel  Conv1D of k, v; phi; key-gate weights exp(a - m_c)
//                         with a per-chunk max m_c; per-chunk partial sums
//                         S_c = sum_j w_j phi(k~_j) v~_j^T, z_c, l_c = sum_j w_j.
//   simt_reduce_kernel    fixed-order combination of the chunk partials into
//                         S = K^T V~ and z = K^T 1 with K^ = softmax(a) * phi(K~):
//                         M = max_c m_c, S = sum_c e^{m_c-M} S_c / sum_c e^{m_c-M} l_c.
//   simt_readout_kernel   Conv1D of q, phi, O = phi(q~)^T S / phi(q~)^T z,
//                         gated RMSNorm, one store of o.
#include <math.h>

#include "gbla_internal.cuh"

namespace gbla {
namespace {

constexpr int kThreads = 256;
constexpr int kTokTile = 32;  // tokens staged in shared memory per step

__device__ __forceinline__ float ldf(const float *p, size_t i) { return p[i]; }
__device__ __forceinline__ float ldf(const __nv_bfloat16 *p, size_t i) {
  return __bfloat162float(p[i]);
}
__device__ __forceinline__ void stf(float *p, size_t i, float x) { p[i] = x; }
__device__ __forceinline__ void stf(__nv_bfloat16 *p, size_t i, float x) {
  p[i] = __float2bfloat16_rn(x);
}

// phi(x) = elu(x) + 1 (Sec. 2).
__device__ __forceinline__ float phi(float x) { return x > 0.f ? x + 1.f : expf(x); }
// SiLU(x) = x * sigmoid(x) (Sec. 2.1 item 3).
__device__ __forceinline__ float silu(float x) { return x / (1.f + expf(-x)); }

__device__ __forceinline__ int clamp_len(const int32_t *seq_lens, int b, int N) {
  if (seq_lens == nullptr) return N;
  int L = seq_lens[b];
  return L < 0 ? 0 : (L > N ? N : L);
}

__device__ __forceinline__ float warp_max(float x) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) x = fmaxf(x, __shfl_xor_sync(0xffffffffu, x, o));
  return x;
}
__device__ __forceinline__ float warp_sum(float x) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
  return x;
}

template <typename T, int D>
__global__ void __launch_bounds__(kThreads)
simt_partials_kernel(const T *__restrict__ k, const T *__restrict__ v,
                     const T *__restrict__ gate, const float *__restrict__ conv_w,
                     const int32_t *__restrict__ seq_lens, float *__restrict__ part,
                     int H, int N, int chunk_len, int n_chunks, uint32_t flags) {
  constexpr int R = D / 16;  // each thread owns an R x R block of S_c
  constexpr int REC = 2 + D + D * D;
  const int c = blockIdx.x, h = blockIdx.y, b = blockIdx.z;
  const int tid = threadIdx.x;
  const int L = clamp_len(seq_lens, b, N);
  const int t0 = c * chunk_len;
  const int t1 = min(t0 + chunk_len, L);
  float *rec = part + (((size_t)b * H + h) * n_chunks + c) * REC;
  if (t0 >= t1) {  // chunk entirely past the sequence end: empty partial
    for (int i = tid; i < REC; i += kThreads) rec[i] = (i == 0) ? -INFINITY : 0.f;
    return;
  }

  __shared__ float s_k[kTokTile][D];
  __shared__ float s_v[kTokTile][D];
  __shared__ float s_w[kTokTile];
  __shared__ float s_wk[D][kConvW], s_wv[D][kConvW];
  __shared__ float s_red[kThreads / 32];

  const bool no_conv = flags & GBLA_FLAG_NO_CONV, no_gate = flags & GBLA_FLAG_NO_GATE;
  for (int i = tid; i < D * kConvW; i += kThreads) {
    const float id = (i % kConvW) == kConvW - 1 ? 1.f : 0.f;  // identity taps
    s_wk[i / kConvW][i % kConvW] = no_conv ? id : conv_w[((size_t)(1 * H + h) * D) * kConvW + i];
    s_wv[i / kConvW][i % kConvW] = no_conv ? id : conv_w[((size_t)(2 * H + h) * D) * kConvW + i];
  }
  // uniform key gate: every logit 0
  auto logit = [&](size_t i) { return no_gate ? 0.f : ldf(gate, i); };

  // Chunk maximum of the gate logits: exp(a - m_c) <= 1 never overflows.
  const size_t gbase = (size_t)b * N * H + h;
  float m = -INFINITY;
  for (int t = t0 + tid; t < t1; t += kThreads) m = fmaxf(m, logit(gbase + (size_t)t * H));
  m = warp_max(m);
  if ((tid & 31) == 0) s_red[tid >> 5] = m;
  __syncthreads();
  m = s_red[0];
#pragma unroll
  for (int i = 1; i < kThreads / 32; ++i) m = fmaxf(m, s_red[i]);

  const size_t rs = (size_t)H * D;  // token stride of [B, N, H, D]
  const T *kb = k + ((size_t)b * N * H + h) * D;
  const T *vb = v + ((size_t)b * N * H + h) * D;
  const int i0 = (tid / 16) * R, j0 = (tid % 16) * R;
  float acc[R][R];
#pragma unroll
  for (int r = 0; r < R; ++r)
#pragma unroll
    for (int s = 0; s < R; ++s) acc[r][s] = 0.f;
  float zacc = 0.f, lacc = 0.f;

  for (int ts = t0; ts < t1; ts += kTokTile) {
    for (int idx = tid; idx < kTokTile * D; idx += kThreads) {
      const int tt = idx / D, d = idx % D, t = ts + tt;
      float kh = 0.f, vv = 0.f;
      if (t < t1) {
        float xk = 0.f, xv = 0.f;
#pragma unroll
        for (int i = 0; i < kConvW; ++i) {
          const int s = t - (kConvW - 1) + i;
          if (s >= 0) {
            xk = fmaf(s_wk[d][i], ldf(kb, (size_t)s * rs + d), xk);
            xv = fmaf(s_wv[d][i], ldf(vb, (size_t)s * rs + d), xv);
          }
        }
        const float w = expf(logit(gbase + (size_t)t * H) - m);
        kh = w * phi(xk);
        vv = xv;
      }
      s_k[tt][d] = kh;
      s_v[tt][d] = vv;
    }
    if (tid < kTokTile) {
      const int t = ts + tid;
      s_w[tid] = t < t1 ? expf(logit(gbase + (size_t)t * H) - m) : 0.f;
    }
    __syncthreads();
#pragma unroll 4
    for (int tt = 0; tt < kTokTile; ++tt) {
      float a[R], bv[R];
#pragma unroll
      for (int r = 0; r < R; ++r) a[r] = s_k[tt][i0 + r];
#pragma unroll
      for (int s = 0; s < R; ++s) bv[s] = s_v[tt][j0 + s];
#pragma unroll
      for (int r = 0; r < R; ++r)
#pragma unroll
        for (int s = 0; s < R; ++s) acc[r][s] = fmaf(a[r], bv[s], acc[r][s]);
    }
    if (tid < D)
      for (int tt = 0; tt < kTokTile; ++tt) zacc += s_k[tt][tid];
    if (tid == kThreads - 1)
      for (int tt = 0; tt < kTokTile; ++tt) lacc += s_w[tt];
    __syncthreads();
  }

  if (tid == 0) rec[0] = m;
  if (tid == kThreads - 1) rec[1] = lacc;
  if (tid < D) rec[2 + tid] = zacc;
#pragma unroll
  for (int r = 0; r < R; ++r)
#pragma unroll
    for (int s = 0; s < R; ++s) rec[2 + D + (size_t)(i0 + r) * D + j0 + s] = acc[r][s];
}

// One thread per state element; chunks are combined in index order.
template <int D>
__global__ void __launch_bounds__(kThreads)
simt_reduce_kernel(const float *__restrict__ part, float *__restrict__ state, int n_chunks) {
  constexpr int REC = 2 + D + D * D;
  constexpr int F = D * D + D;
  extern __shared__ float s_scale[];  // e^{m_c - M}, n_chunks entries
  __shared__ float s_M, s_l;
  const int bh = blockIdx.x;
  const float *base = part + (size_t)bh * n_chunks * REC;
  if (threadIdx.x < 32) {
    float M = -INFINITY;
    for (int c = threadIdx.x; c < n_chunks; c += 32) M = fmaxf(M, base[(size_t)c * REC]);
    M = warp_max(M);
    if (threadIdx.x == 0) s_M = M;
  }
  __syncthreads();
  const float M = s_M;
  for (int c = threadIdx.x; c < n_chunks; c += kThreads) {
    const float mc = base[(size_t)c * REC];
    s_scale[c] = (M == -INFINITY || mc == -INFINITY) ? 0.f : expf(mc - M);
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    float l = 0.f;
    for (int c = 0; c < n_chunks; ++c) l = fmaf(s_scale[c], base[(size_t)c * REC + 1], l);
    s_l = l;
  }
  __syncthreads();
  const int e = blockIdx.y * kThreads + threadIdx.x;
  if (e >= F) return;
  const int src = e < D * D ? 2 + D + e : 2 + (e - D * D);
  float acc = 0.f;
  for (int c = 0; c < n_chunks; ++c) acc = fmaf(s_scale[c], base[(size_t)c * REC + src], acc);
  state[(size_t)bh * F + e] = s_l > 0.f ? acc / s_l : 0.f;
}

// TO: type of the stored output; the product path stores the input type T, the
// fp32-output debug path (gbla_forward_f32out) float, from the same y.
template <typename T, typename TO, int D>
__global__ void __launch_bounds__(kThreads)
simt_readout_kernel(const T *__restrict__ q, const T *__restrict__ og,
                    const float *__restrict__ conv_w, const float *__restrict__ norm_w,
                    const int32_t *__restrict__ seq_lens, const float *__restrict__ state,
                    TO *__restrict__ o, int H, int N, float eps, uint32_t flags) {
  constexpr int J = D / 32;  // output columns per lane
  const int h = blockIdx.y, b = blockIdx.z;
  const int L = clamp_len(seq_lens, b, N);
  const int t0 = blockIdx.x * kTokTile;
  if (t0 >= L) return;
  extern __shared__ float smem[];
  float *sS = smem;                 // [D][D]
  float *sz = sS + D * D;           // [D]
  float *sq = sz + D;               // [kTokTile][D]  phi(q~)
  float *swq = sq + kTokTile * D;   // [D][kConvW]
  const int tid = threadIdx.x;
  const float *st = state + ((size_t)b * H + h) * (D * D + D);
  for (int i = tid; i < D * D + D; i += kThreads) sS[i] = st[i];
  for (int i = tid; i < D * kConvW; i += kThreads)
    swq[i] = (flags & GBLA_FLAG_NO_CONV) ? ((i % kConvW) == kConvW - 1 ? 1.f : 0.f)
                                          : conv_w[((size_t)(0 * H + h) * D) * kConvW + i];
  __syncthreads();

  const size_t rs = (size_t)H * D;
  const size_t hb = ((size_t)b * N * H + h) * D;
  for (int idx = tid; idx < kTokTile * D; idx += kThreads) {
    const int tt = idx / D, d = idx % D, t = t0 + tt;
    float val = 0.f;
    if (t < L) {
      float x = 0.f;
#pragma unroll
      for (int i = 0; i < kConvW; ++i) {
        const int s = t - (kConvW - 1) + i;
        if (s >= 0) x = fmaf(swq[d * kConvW + i], ldf(q, hb + (size_t)s * rs + d), x);
      }
      val = phi(x);
    }
    sq[idx] = val;
  }
  __syncthreads();

  const int warp = tid >> 5, lane = tid & 31;
  constexpr int kTokPerWarp = kTokTile / (kThreads / 32);
  for (int u = 0; u < kTokPerWarp; ++u) {
    const int tt = warp * kTokPerWarp + u, t = t0 + tt;
    if (t >= L) break;
    const float *pq = sq + tt * D;
    float den = 0.f, num[J];
#pragma unroll
    for (int j = 0; j < J; ++j) num[j] = 0.f;
    for (int d = 0; d < D; ++d) {
      const float a = pq[d];
      den = fmaf(a, sz[d], den);
#pragma unroll
      for (int j = 0; j < J; ++j) num[j] = fmaf(a, sS[d * D + lane + 32 * j], num[j]);
    }
    float O[J], ss = 0.f;
#pragma unroll
    for (int j = 0; j < J; ++j) {
      O[j] = num[j] / den;
      ss = fmaf(O[j], O[j], ss);
    }
    ss = warp_sum(ss);
    const float r = 1.f / sqrtf(ss / (float)D + eps);
    const size_t row = hb + (size_t)t * rs;
#pragma unroll
    for (int j = 0; j < J; ++j) {
      const int e = lane + 32 * j;
      const float y = (flags & GBLA_FLAG_NO_NORM)
                          ? O[j]
                          : O[j] * r * norm_w[(size_t)h * D + e] * silu(ldf(og, row + e));
      stf(o, row + e, y);
    }
  }
}

template <typename T, int D>
cudaError_t launch_state(const Problem &p, const SimtPlan &plan, const void *k,
                         const void *v, const void *gate, const float *conv_w,
                         float *partials, float *state, cudaStream_t st) {
  dim3 g1(plan.n_chunks, p.H, p.B);
  simt_partials_kernel<T, D><<<g1, kThreads, 0, st>>>(
      (const T *)k, (const T *)v, (const T *)gate, conv_w, p.seq_lens, partials,
      p.H, p.N, plan.chunk_len, plan.n_chunks, p.flags);
  count_launch();
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  constexpr int F = D * D + D;
  dim3 g2(p.B * p.H, (F + kThreads - 1) / kThreads);
  simt_reduce_kernel<D><<<g2, kThreads, plan.n_chunks * sizeof(float), st>>>(
      partials, state, plan.n_chunks);
  count_launch();
  return cudaGetLastError();
}

template <typename T, typename TO, int D>
cudaError_t launch_readout(const Problem &p, const void *q, const void *og,
                           const float *conv_w, const float *norm_w,
                           const float *state, void *o, cudaStream_t st) {
  const size_t smem = sizeof(float) * (D * D + D + kTokTile * D + D * kConvW);
  auto kern = simt_readout_kernel<T, TO, D>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)smem);
  if (e != cudaSuccess) return e;
  dim3 g((p.N + kTokTile - 1) / kTokTile, p.H, p.B);
  kern<<<g, kThreads, smem, st>>>((const T *)q, (const T *)og, conv_w, norm_w,
                                  p.seq_lens, state, (TO *)o, p.H, p.N, kRmsEps, p.flags);
  count_launch();
  return cudaGetLastError();
}

}  // namespace

SimtPlan simt_plan(const Problem &p) {
  // At most 2048 partials per (b, h); chunks of at least 256 tokens.
  int chunk = 256;
  while ((p.N + chunk - 1) / chunk > 2048) chunk *= 2;
  return SimtPlan{chunk, (p.N + chunk - 1) / chunk};
}

size_t simt_partials_bytes(const Problem &p, const SimtPlan &plan) {
  return sizeof(float) * partial_floats(p.D) * (size_t)p.B * p.H * plan.n_chunks;
}

cudaError_t simt_state(const Problem &p, const SimtPlan &plan, const void *k,
                       const void *v, const void *gate, const float *conv_w,
                       float *partials, float *state, cudaStream_t st) {
#define GBLA_SIMT_STATE(T, DD) \
  return launch_state<T, DD>(p, plan, k, v, gate, conv_w, partials, state, st)
  if (p.dtype == GBLA_FP32) {
    if (p.D == 32) GBLA_SIMT_STATE(float, 32);
    if (p.D == 64) GBLA_SIMT_STATE(float, 64);
    if (p.D == 128) GBLA_SIMT_STATE(float, 128);
  } else {
    if (p.D == 32) GBLA_SIMT_STATE(__nv_bfloat16, 32);
    if (p.D == 64) GBLA_SIMT_STATE(__nv_bfloat16, 64);
    if (p.D == 128) GBLA_SIMT_STATE(__nv_bfloat16, 128);
  }
#undef GBLA_SIMT_STATE
  return cudaErrorInvalidValue;
}

cudaError_t simt_readout(const Problem &p, const void *q, const void *og,
                         const float *conv_w, const float *norm_w,
                         const float *state, void *o, cudaStream_t st, bool f32_out) {
#define GBLA_SIMT_READ(T, DD)                                                      \
  return f32_out ? launch_readout<T, float, DD>(p, q, og, conv_w, norm_w, state, o, st) \
                 : launch_readout<T, T, DD>(p, q, og, conv_w, norm_w, state, o, st)
  if (p.dtype == GBLA_FP32) {
    if (p.D == 32) GBLA_SIMT_READ(float, 32);
    if (p.D == 64) GBLA_SIMT_READ(float, 64);
    if (p.D == 128) GBLA_SIMT_READ(float, 128);
  } else {
    if (p.D == 32) GBLA_SIMT_READ(__nv_bfloat16, 32);
    if (p.D == 64) GBLA_SIMT_READ(__nv_bfloat16, 64);
    if (p.D == 128) GBLA_SIMT_READ(__nv_bfloat16, 128);
  }
#undef GBLA_SIMT_READ
  return cudaErrorInvalidValue;
}

}  // namespace gbla
