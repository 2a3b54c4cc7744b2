// Combination of partial states of disjoint token segments of the same
// sequences (a sequence split across devices).  The state of Sec. 2.1 item 2
// is a softmax-weighted sum over the sequence; for segments p with their own
// softmax statistics (m_p = max logit, l_p = sum of exp(logit - m_p)) and
// their normalised partial states S_p, z_p, the whole sequence's state is
//   M = max_p m_p,  w_p = l_p e^{m_p - M},  S = sum_p w_p S_p / sum_p w_p
// (z likewise), the same max-rescaled combination the state reduction applies
// to its partial records.  Segments with l_p = 0 (no valid token) weigh 0.
// The sums run in segment order, so the result does not depend on timing.
#include <math.h>

#include "gbla_internal.cuh"

namespace gbla {
namespace {

constexpr int kCombThreads = 256;
constexpr int kMaxParts = 1024;

// Block (bh, slice): the weights of the P parts into shared memory, then each
// thread one state element of the slice.
__global__ void __launch_bounds__(kCombThreads) combine_kernel(
    const float *__restrict__ states, const float2 *__restrict__ stats, int P, int BH, int F,
    float *__restrict__ state, float2 *__restrict__ out_stats) {
  __shared__ float w[kMaxParts];
  __shared__ float s_inv;
  const int bh = blockIdx.x;
  if (threadIdx.x == 0) {
    float M = -INFINITY;
    for (int p = 0; p < P; ++p) {
      const float2 s = stats[(size_t)p * BH + bh];
      if (s.y > 0.f) M = fmaxf(M, s.x);
    }
    float wsum = 0.f;
    for (int p = 0; p < P; ++p) {
      const float2 s = stats[(size_t)p * BH + bh];
      w[p] = s.y > 0.f ? s.y * expf(s.x - M) : 0.f;
      wsum += w[p];
    }
    s_inv = wsum > 0.f ? 1.f / wsum : 0.f;
    if (blockIdx.y == 0) out_stats[bh] = make_float2(M, wsum);
  }
  __syncthreads();
  const float inv = s_inv;
  for (int e = blockIdx.y * kCombThreads + threadIdx.x; e < F; e += gridDim.y * kCombThreads) {
    float acc = 0.f;
    for (int p = 0; p < P; ++p)
      if (w[p] != 0.f) acc = fmaf(w[p], states[((size_t)p * BH + bh) * F + e], acc);
    state[(size_t)bh * F + e] = acc * inv;
  }
}

}  // namespace

cudaError_t combine_states(const float *states, const float2 *stats, int P, int BH, int D,
                           float *state, float2 *out_stats, cudaStream_t st) {
  if (P <= 0 || P > kMaxParts || BH <= 0) return cudaErrorInvalidValue;
  const int F = D * D + D;
  const int slices = (F + 4 * kCombThreads - 1) / (4 * kCombThreads);
  combine_kernel<<<dim3(BH, slices), kCombThreads, 0, st>>>(states, stats, P, BH, F, state,
                                                            out_stats);
  count_launch();
  return cudaGetLastError();
}

}  // namespace gbla
