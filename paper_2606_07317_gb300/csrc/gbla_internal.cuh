// Internal declarations shared by the C-ABI front end and the kernel files.
#pragma once

#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <stdint.h>

#include <initializer_list>

#include "gbla.h"

namespace gbla {

constexpr int kConvW = GBLA_CONV_WIDTH;
constexpr float kRmsEps = 1e-6f;

struct Problem {
  int B, H, N, D;
  gbla_dtype dtype;
  const int32_t *seq_lens;  // device [B] or nullptr
  uint32_t flags = 0;       // gbla_flags: ablations of Sec. 4, Table 4
};

// Floats in one partial-state record of a sequence chunk: m (chunk max of the
// gate logits), l (sum of exp(a - m) over the chunk), z[D], S[D*D].
inline size_t partial_floats(int D) { return 2 + (size_t)D + (size_t)D * D; }
inline size_t state_floats(int D) { return (size_t)D * D + D; }

// Counts every kernel this library enqueues (read by gbla_launch_count).
void count_launch(unsigned n = 1);

// Argument checks shared by every entry point (gbla_api.cu).
// check_dims: sizes and dtype; *empty is set when B, H or N is 0.
gbla_status check_dims(int B, int H, int N, int D, gbla_dtype dtype, bool *empty);
// check_ptrs: every pointer non-null and 16-byte aligned.
gbla_status check_ptrs(std::initializer_list<const void *> ptrs);
// check_seq_lens: NULL or 4-byte aligned.
gbla_status check_seq_lens(const int32_t *seq_lens);
// Maps a CUDA error to a status; a failure is recorded for gbla_last_cuda_error.
gbla_status from_cuda(cudaError_t e);

// ---- CUDA-core (SIMT) family: every dtype and D ---------------------------
struct SimtPlan {
  int chunk_len;  // tokens per partial
  int n_chunks;   // partials per (b, h)
};
SimtPlan simt_plan(const Problem &p);
size_t simt_partials_bytes(const Problem &p, const SimtPlan &plan);
cudaError_t simt_state(const Problem &p, const SimtPlan &plan, const void *k,
                       const void *v, const void *gate, const float *conv_w,
                       float *partials, float *state, cudaStream_t st);
// f32_out: store o in fp32 whatever the input dtype (gbla_forward_f32out).
cudaError_t simt_readout(const Problem &p, const void *q, const void *og,
                         const float *conv_w, const float *norm_w,
                         const float *state, void *o, cudaStream_t st,
                         bool f32_out = false);

// ---- tensor-core (tcgen05 + TMA) family: bf16, D in {64, 128} -------------
bool tc_supports(const Problem &p);
size_t tc_workspace_bytes(const Problem &p);
// gate_stats (optional, [B*H]): the key gate's softmax statistics (max of the
// logits, sum of exp(logit - max)) over each sequence, as the state used them.
cudaError_t tc_state(const Problem &p, const void *k, const void *v,
                     const void *gate, const float *conv_w, void *workspace,
                     float *state, cudaStream_t st, float2 *gate_stats = nullptr);
// after_state: launched right behind tc_state on the same stream; only the
// reads of `state` then wait for the preceding kernel (the other inputs were
// complete before tc_state started).
// f32_out: the debug instantiation that stores o in fp32 (full core only).
cudaError_t tc_readout(const Problem &p, const void *q, const void *og,
                       const float *conv_w, const float *norm_w,
                       const float *state, void *o, cudaStream_t st,
                       bool after_state = false, bool f32_out = false);
// Programmatic dependent launch: the grid may start while the kernel before it
// on the stream ends (once that kernel's blocks have all signalled, or
// exited); the kernel itself waits (griddepcontrol.wait) before it reads
// anything the kernel before may write, and before its first global write.
template <typename... KArgs, typename... Args>
inline cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                              cudaStream_t st, Args... args) {
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, args...);
}
// ---- backward (CUDA cores, fp32 arithmetic; gbla_bwd.cu) ------------------
struct BwdArgs {
  const void *q, *k, *v, *gate, *out_gate, *dy;
  const float *conv_w, *norm_w;
  void *dq, *dk, *dv, *dgate, *dout_gate;
  float *dconv_w, *dnorm_w;
  // the forward state S, z [B*H][D*D + D] and, when stats_ready, the key gate's
  // softmax statistics [B*H] (max, sum of exp): the scratch slots of the
  // layout below, or a forward's saved copies
  const float *state;
  const float2 *stats;
};
// Scratch of the backward, in floats from one base: the forward state (filled
// by the caller through the forward's state path, unless a saved state is
// given), gate statistics (filled by the caller too when stats_ready, else by
// the backward itself), chunk partials, reduced dS / dz, the per-token
// dq~ / dk~ / dv~ planes and the tap gradient partials.
struct BwdLayout {
  size_t state, stats, gpart, qpart, red, cpart, dxt, wpart, total;
};
BwdLayout bwd_layout(const Problem &p);
// The key gate's softmax statistics per (b, h) on CUDA cores: (max of the
// logits, sum of exp(logit - max)) over the valid positions, (-inf, 0) for an
// empty sequence.  `part` holds gate_stats_part_floats(p) floats of scratch.
cudaError_t gate_stats(const Problem &p, const void *gate, float2 *part, float2 *stats,
                       cudaStream_t st);
size_t gate_stats_part_floats(const Problem &p);
// Fixed-order max-rescaled combination of P partial states (gbla_seqsplit.cu).
cudaError_t combine_states(const float *states, const float2 *stats, int P, int BH, int D,
                           float *state, float2 *out_stats, cudaStream_t st);
// Taps (0, 0, 0, 1) for n channels (the identity Conv1D of the ablations), [n][4].
cudaError_t fill_identity_taps(float *taps, int n, cudaStream_t st);
// p.flags selects an ablation (the CUDA-core token passes; the caller
// substitutes identity taps and zero gate logits, see gbla_backward_variant).
cudaError_t bwd_run(const Problem &p, const BwdArgs &a, float *scratch, bool stats_ready,
                    cudaStream_t st);
// Key pass on tensor cores (gbla_bwd_tc.cu): bf16, D = 64, sm_103.  Writes the
// bf16 dk~ / dv~ planes and dgate (zero past seq_lens) from the reduced dS, dz
// and the ndot partial sums per (b, h) of c = <dS, S> + <dz, z>.
bool bwd_tc_key_supported(const Problem &p);
cudaError_t bwd_tc_key(const Problem &p, const BwdArgs &a, const float2 *stats,
                       const float *red, const float *dotpart, int ndot, void *dkt,
                       void *dvt, cudaStream_t st);
// Query pass on tensor cores (same conditions): dq~ plane, dout_gate, and one
// partial record [dS, dz, dnorm_w] per (b, h, chunk of bwd_tc_query_chunks).
int bwd_tc_query_chunks(const Problem &p);
cudaError_t bwd_tc_query(const Problem &p, const BwdArgs &a, const float *state, float *part,
                         void *dqt, cudaStream_t st);
unsigned bwd_device_error(bool reset);

// ---- layer front end (tcgen05; gbla_project.cu): bf16 ----------------------
struct ProjProblem {
  int B, N, d, H, D;
  const int32_t *seq_lens;  // device [B] or nullptr
};
// d a multiple of 64 in [64, 512], H * D a multiple of 64, H <= 256, sm_103.
bool project_supports(const ProjProblem &pp);
cudaError_t tc_project(const ProjProblem &pp, const void *x, const float *conv_x,
                       const void *w, void *q, void *k, void *v, void *og, void *gate,
                       cudaStream_t st);
unsigned project_device_error(bool reset);

// ---- bidirectional softmax attention (tcgen05; gbla_sa.cu): bf16, D = 64 --
bool sa_supports(int D, gbla_dtype dtype);
cudaError_t sa_forward(const void *q, const void *k, const void *v, const int32_t *seq_lens,
                       void *o, int B, int H, int N, cudaStream_t st);
unsigned sa_device_error(bool reset);

// Error bits set by tensor-core kernels whose bounded waits ran out (0 = none);
// synchronous read of the current device, optionally clearing it.
unsigned tc_device_error(bool reset);

}  // namespace gbla
