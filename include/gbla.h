/*
 * gbla.h -- C ABI of the GB300 (sm_103a) GBLA layer-core forward.
 *
 * The layer is Gated Bidirectional Linear Attention, Sec. 2.1 of "Gated
 * Bidirectional Linear Attention for Generative Retrieval".  For every batch
 * row b, head h and valid position i < L_b it computes
 *
 *   q~, k~, v~ = Conv1D(q), Conv1D(k), Conv1D(v)        (Sec. 2.1 item 1)
 *   g          = softmax_j(gate[b, j, h]), j < L_b     (Sec. 2.1 item 2)
 *   K^         = g * phi(K~),  phi(x) = elu(x) + 1     (Sec. 2 / 2.1 item 2)
 *   S = K^T V~ (D x D),  z = K^T 1 (D)                  (Sec. 2.1 item 2)
 *   O_i        = phi(q~_i)^T S / phi(q~_i)^T z
 *   o_i        = O_i / sqrt(mean(O_i^2) + eps) * norm_w[h] * SiLU(out_gate_i)
 *                                                       (Sec. 2.1 item 3)
 *
 * Conv1D is causal and depthwise over the sequence, width GBLA_CONV_WIDTH, left
 * zero padding, no bias: x~[t, c] = sum_i w[c, i] * x[t - (W-1) + i, c], so tap
 * W-1 multiplies the current token.  The gate logits and the output-gate
 * input are taken as given (already derived from the convolved sequence).
 * eps is gbla_rms_eps().
 *
 * Layouts (all contiguous, row-major, no padding between rows):
 *   q, k, v, out_gate, o : [B, N, H, D] of dtype
 *   gate                 : [B, N, H]    of dtype (softmax logits)
 *   conv_w               : [3, H, D, GBLA_CONV_WIDTH] fp32 (taps for q, k, v)
 *   norm_w               : [H, D] fp32 (RMSNorm weight per head)
 *   seq_lens             : [B] int32, or NULL meaning every row has length N;
 *                          values are clamped to [0, N] on the device
 *   state                : [B, H, D*D + D] fp32: S row-major (S[d][e]) then z
 *
 * Ownership: every pointer is a caller-owned DEVICE pointer on the current
 * device, 16-byte aligned.  The library keeps no pointer after a call returns.
 * Outputs must not overlap inputs.
 *
 * Asynchrony: every compute call only enqueues work on `stream` (NULL = the
 * legacy default stream) and returns; it never synchronises.  Scratch memory
 * is taken from the device's stream-ordered pool (cudaMallocAsync) and freed
 * on the same stream, so concurrent calls on different streams are safe.
 *
 * Errors: arguments are validated on the host before anything is enqueued.
 *   GBLA_ERR_INVALID_ARG  null pointer, negative size, misaligned pointer,
 *                         overlapping output, or a size beyond the limits
 *   GBLA_ERR_UNSUPPORTED  D not in {32, 64, 128}, unknown dtype or algo,
 *                         or an algo that does not cover (dtype, D)
 *   GBLA_ERR_ALLOC        the stream-ordered scratch allocation failed
 *   GBLA_ERR_CUDA         a CUDA call or kernel launch failed
 * A call with B, H or N equal to 0 has nothing to compute: it returns GBLA_OK
 * without touching any pointer.  Rows t >= L_b of o are never written, and a
 * sequence of length 0 writes nothing.
 */
#ifndef GBLA_H_
#define GBLA_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

struct CUstream_st; /* cudaStream_t is `struct CUstream_st *` */
typedef struct CUstream_st *gbla_stream_t;

#define GBLA_CONV_WIDTH 4

typedef enum gbla_status {
  GBLA_OK = 0,
  GBLA_ERR_INVALID_ARG = 1,
  GBLA_ERR_UNSUPPORTED = 2,
  GBLA_ERR_ALLOC = 3,
  GBLA_ERR_CUDA = 4
} gbla_status;

typedef enum gbla_dtype {
  GBLA_FP32 = 0, /* fp32 storage, exact fp32 arithmetic (CUDA-core FMA) */
  GBLA_BF16 = 1  /* bf16 storage, fp32 accumulation                      */
} gbla_dtype;

typedef enum gbla_algo {
  GBLA_ALGO_AUTO = 0, /* tensor-core kernels where they cover (dtype, D), else SIMT */
  GBLA_ALGO_SIMT = 1, /* CUDA-core kernels, every (dtype, D)                        */
  GBLA_ALGO_TC = 2    /* tcgen05/TMEM + TMA kernels: bf16 with D in {64, 128}      */
} gbla_algo;

/*
 * Ablations of the GBLA core (Sec. 4, Table 4): each flag turns one of the
 * three add-ons of Sec. 2.1 off; all three off is plain bidirectional linear
 * attention, Eq. bla.  Inputs an ablation ignores must still be valid pointers.
 */
typedef enum gbla_flags {
  GBLA_FLAG_NO_CONV = 1, /* identity Conv1D: q~ = q, k~ = k, v~ = v (conv_w unused)   */
  GBLA_FLAG_NO_GATE = 2, /* uniform key gate: g_j = 1 / L_b (gate logits unused)      */
  GBLA_FLAG_NO_NORM = 4, /* no gated RMSNorm: o = O (out_gate and norm_w unused)       */
  GBLA_FLAG_BLA = 7      /* all three off                                            */
} gbla_flags;

/*
 * gbla_forward -- the whole GBLA core, Sec. 2.1 (all three add-ons on).
 * Writes o[b, t, h, :] for every b, h and t < L_b.  Equivalent to
 * gbla_forward_ex(..., GBLA_ALGO_AUTO, stream).
 */
gbla_status gbla_forward(const void *q, const void *k, const void *v,
                         const void *gate, const void *out_gate,
                         const float *conv_w, const float *norm_w,
                         const int32_t *seq_lens, void *o, int B, int H, int N,
                         int D, gbla_dtype dtype, gbla_stream_t stream);

/* gbla_forward with an explicit kernel family (see gbla_algo). */
gbla_status gbla_forward_ex(const void *q, const void *k, const void *v,
                            const void *gate, const void *out_gate,
                            const float *conv_w, const float *norm_w,
                            const int32_t *seq_lens, void *o, int B, int H,
                            int N, int D, gbla_dtype dtype, gbla_algo algo,
                            gbla_stream_t stream);

/*
 * gbla_forward_variant -- gbla_forward_ex with ablation flags (gbla_flags,
 * OR-ed; 0 is gbla_forward_ex).  Flags outside GBLA_FLAG_BLA return
 * GBLA_ERR_INVALID_ARG before anything is enqueued.
 */
gbla_status gbla_forward_variant(const void *q, const void *k, const void *v,
                                 const void *gate, const void *out_gate,
                                 const float *conv_w, const float *norm_w,
                                 const int32_t *seq_lens, void *o, int B, int H, int N,
                                 int D, gbla_dtype dtype, gbla_algo algo, uint32_t flags,
                                 gbla_stream_t stream);

/*
 * gbla_forward_f32out -- debug variant of gbla_forward_ex (full core): the same
 * kernels run the same arithmetic, but the readout stores o32 [B, N, H, D] in
 * fp32 -- the value that gbla_forward would round to dtype -- so that the
 * computation error of the bf16 path (Sec. 2.1 item 3 output) can be measured
 * apart from the rounding of its stored result.  For bf16 inputs, rounding
 * o32 to bf16 (round to nearest even) gives gbla_forward's o bit for bit.
 * o32 must not overlap any input; rows t >= L_b are not written.  Arguments,
 * validation and errors otherwise as gbla_forward_ex.
 */
gbla_status gbla_forward_f32out(const void *q, const void *k, const void *v,
                                const void *gate, const void *out_gate,
                                const float *conv_w, const float *norm_w,
                                const int32_t *seq_lens, float *o32, int B, int H,
                                int N, int D, gbla_dtype dtype, gbla_algo algo,
                                gbla_stream_t stream);

/*
 * gbla_backward -- gradients of sum(dy * o) of the layer core (the full core;
 * gbla_backward_variant below takes the ablations) with respect to every input: the chain rule through the steps of
 * Sec. 2.1 in reverse (gated RMSNorm, readout, state, key-gate softmax, phi,
 * Conv1D).  Used to train the model end to end (the paper's training-speed
 * comparison, Sec. 3).
 *
 * Inputs as gbla_forward (same layouts, dtype and validation), plus
 *   dy        [B, N, H, D] dtype: gradient of the loss with respect to o.
 * Outputs (caller-owned device buffers, 16-byte aligned, no aliasing with any
 * input or with one another):
 *   dq, dk, dv, dout_gate  [B, N, H, D] dtype;  dgate [B, N, H] dtype;
 *   dconv_w [3, H, D, W] fp32 (q, k, v taps);   dnorm_w [H, D] fp32.
 * Rows t >= L_b of dq, dk, dv, dout_gate and dgate are written as 0; dconv_w
 * and dnorm_w are overwritten with sums over the batch.  The forward state is
 * recomputed inside (nothing is kept from a forward call; see
 * gbla_backward_from_state for a backward that takes it).  fp32 arithmetic
 * (for bf16 with D = 64 the token contractions run on tensor cores with bf16
 * operands, S and dS split into bf16 hi + lo, fp32 accumulation); every sum
 * runs in a fixed order (bitwise reproducible).  Asynchronous on
 * `stream`; scratch comes from the library's stream-ordered pool
 * (GBLA_ERR_ALLOC when it cannot).  Same error codes as gbla_forward.
 */
gbla_status gbla_backward(const void *q, const void *k, const void *v, const void *gate,
                          const void *out_gate, const float *conv_w, const float *norm_w,
                          const int32_t *seq_lens, const void *dy, void *dq, void *dk,
                          void *dv, void *dgate, void *dout_gate, float *dconv_w,
                          float *dnorm_w, int B, int H, int N, int D, gbla_dtype dtype,
                          gbla_stream_t stream);

/*
 * gbla_backward_variant -- gbla_backward of an ablation of Table 4 (`flags`:
 * gbla_flags OR-ed, as gbla_forward_variant; 0 is gbla_backward): the
 * gradients of sum(dy * o) with o the variant's output.  The parameters a
 * variant does not use get zero gradients: dconv_w under GBLA_FLAG_NO_CONV,
 * dgate (every row) under GBLA_FLAG_NO_GATE, dout_gate and dnorm_w under
 * GBLA_FLAG_NO_NORM.  Variants run the token passes on CUDA cores (fp32
 * arithmetic for every dtype and D); the identity Conv1D and the uniform gate
 * are computed as the full core on identity taps and all-zero gate logits
 * (scratch copies made by the call).  Flags outside GBLA_FLAG_BLA return
 * GBLA_ERR_INVALID_ARG; arguments, limits, errors and asynchrony otherwise
 * as gbla_backward.
 */
gbla_status gbla_backward_variant(const void *q, const void *k, const void *v,
                                  const void *gate, const void *out_gate,
                                  const float *conv_w, const float *norm_w,
                                  const int32_t *seq_lens, const void *dy, void *dq, void *dk,
                                  void *dv, void *dgate, void *dout_gate, float *dconv_w,
                                  float *dnorm_w, int B, int H, int N, int D,
                                  gbla_dtype dtype, uint32_t flags, gbla_stream_t stream);

/*
 * gbla_backward_from_state -- gbla_backward given the forward's state: for
 * training, where the forward ran as gbla_state_stats + gbla_readout and kept
 * what the backward needs instead of recomputing it (the key-gate softmax and
 * the state of Sec. 2.1 item 2 over the whole sequence):
 *   state [B, H, D*D + D] fp32  S and z of each sequence, and
 *   stats [B, H, 2] fp32        its (m, l),
 * exactly as gbla_state_stats returned them for the same k, v, gate, conv_w
 * and seq_lens (other values give gradients of another forward; nothing
 * checks them).  The call skips the state pass and reads nothing else of the
 * forward.  Both are inputs: device pointers, 16-byte aligned, not
 * overlapping any output (GBLA_ERR_INVALID_ARG otherwise).  Every other
 * argument, output, limit, error and the asynchrony as gbla_backward (the full
 * core).
 */
gbla_status gbla_backward_from_state(const void *q, const void *k, const void *v,
                                     const void *gate, const void *out_gate,
                                     const float *conv_w, const float *norm_w,
                                     const int32_t *seq_lens, const float *state,
                                     const float *stats, const void *dy, void *dq, void *dk,
                                     void *dv, void *dgate, void *dout_gate, float *dconv_w,
                                     float *dnorm_w, int B, int H, int N, int D,
                                     gbla_dtype dtype, gbla_stream_t stream);

/*
 * gbla_project -- the layer front end: Sec. 2.1 item 1 (X~ = Conv1D(X), then
 * Q = X~ W_Q, K = X~ W_K, V = X~ W_V), item 2 (gate logits X~ w_g) and item 3
 * (output-gate input X~ W_R), with one set of matrices per head (the
 * multi-head paragraph of Sec. 2.1), as one tensor-core contraction.
 *
 *   x        [B, N, d] dtype  the embedded sequence X (token-major).
 *   conv_x   [d, W] fp32      depthwise causal Conv1D taps on X; tap W-1
 *                             multiplies the current token, history before
 *                             t = 0 is zero; no bias, no activation.
 *   w_proj   [F, d] dtype     stacked projection weights, F = 4 H D + H, one
 *                             row per output feature over the d inputs (the
 *                             nn.Linear weight layout): rows s*H*D + h*D + e
 *                             give dim e of head h of stream s = Q, K, V, R
 *                             (W_R), rows 4*H*D + h give w_g of head h.
 *   seq_lens device [B] int32 or NULL, as gbla_forward.
 *   q, k, v, out_gate [B, N, H, D] dtype and gate [B, N, H] dtype: outputs,
 *                             laid out as gbla_forward's inputs.  Rows t >= L_b
 *                             are not written.
 * bf16 only (GBLA_FP32 returns GBLA_ERR_UNSUPPORTED): X~ is computed in fp32
 * and rounded once to bf16, the products are summed in fp32, each output is
 * rounded once to bf16.  Limits: d a multiple of 64 in [64, 512], H * D a
 * multiple of 64, H <= 256, D in {32, 64, 128}; otherwise
 * GBLA_ERR_UNSUPPORTED.  All pointers 16-byte aligned device pointers
 * (caller-owned); the outputs must not overlap any input or one another
 * (GBLA_ERR_INVALID_ARG).  Needs an sm_103 GPU (GBLA_ERR_UNSUPPORTED
 * otherwise).  Asynchronous on `stream`; allocates nothing.
 */
gbla_status gbla_project(const void *x, const float *conv_x, const void *w_proj,
                         const int32_t *seq_lens, void *q, void *k, void *v,
                         void *out_gate, void *gate, int B, int N, int d, int H,
                         int D, gbla_dtype dtype, gbla_stream_t stream);

/*
 * gbla_layer_forward -- the whole GBLA layer of Sec. 2.1 from X: gbla_project,
 * then the core (gbla_forward_variant with GBLA_FLAG_NO_CONV, since the
 * Conv1D already ran on X) with its Conv1D off.  Arguments as gbla_project
 * plus norm_w [H, D] fp32 and the output o [B, N, H, D] dtype (rows t < L_b
 * written).  q, k, v, out_gate and gate live in scratch from the library's
 * stream-ordered pool, stored in dtype between the two halves (GBLA_ERR_ALLOC
 * when the pool cannot provide 8 B N H D + 2 B N H bytes).  o must not overlap
 * an input.  Same limits and error codes as gbla_project.
 */
gbla_status gbla_layer_forward(const void *x, const float *conv_x, const void *w_proj,
                               const float *norm_w, const int32_t *seq_lens, void *o,
                               int B, int N, int d, int H, int D, gbla_dtype dtype,
                               gbla_stream_t stream);

/*
 * gbla_attention_forward -- bidirectional softmax attention, Sec. 2
 * ("Bidirectional softmax attention"): the SA layer of the hybrid [SA, LA, LA]
 * encoder of Sec. 3, whose latency the GBLA layer is compared with (Sec. 4,
 * Table 5).  For every batch row b, head h and valid query i < L_b,
 *   o_i = sum_j exp(q_i . k_j / sqrt(D)) v_j / sum_j exp(q_i . k_j / sqrt(D)),
 * over the valid keys j < L_b (no causal mask).
 *   q, k, v, o [B, N, H, D] dtype, token-major as gbla_forward's inputs;
 *   seq_lens   device [B] int32 or NULL (= all N), clamped to [0, N].
 * Rows t >= L_b of o are not written.  bf16 with D = 64 on an sm_103 GPU only
 * (tcgen05 tensor cores: bf16 operands, fp32 accumulation, probabilities
 * rounded to bf16 for the second product); anything else returns
 * GBLA_ERR_UNSUPPORTED.  o must not overlap an input.  Asynchronous on
 * `stream`; allocates nothing.
 */
gbla_status gbla_attention_forward(const void *q, const void *k, const void *v,
                                   const int32_t *seq_lens, void *o, int B, int H, int N,
                                   int D, gbla_dtype dtype, gbla_stream_t stream);

/*
 * gbla_state -- the sequence-global part of Sec. 2.1 item 2: Conv1D of k and
 * v, phi, the softmax key gate, and per (b, h) the state S = K^T V~ and the
 * normaliser z = K^T 1 with K^ = g * phi(K~), g the softmax over j < L_b.
 * Writes state[b, h, :] (layout above; zeros when L_b = 0).  The sum over the
 * sequence is split into chunks whose partial sums are combined in a fixed
 * order, so the result is bitwise reproducible for a given (N, seq_lens).
 */
gbla_status gbla_state(const void *k, const void *v, const void *gate,
                       const float *conv_w, const int32_t *seq_lens,
                       float *state, int B, int H, int N, int D,
                       gbla_dtype dtype, gbla_algo algo, gbla_stream_t stream);

/*
 * gbla_state_stats -- gbla_state plus the key gate's softmax statistics of
 * each sequence (Sec. 2.1 item 2): stats [B, H, 2] fp32 receives (m, l), m the
 * largest gate logit over the valid positions t < L_b and l = sum over them of
 * exp(logit - m); an empty sequence gives (-inf, 0) and a zero state.  These
 * are what combining the states of disjoint token segments of a sequence
 * needs (gbla_combine_states).  A logit of -inf gives its token weight 0, so a
 * segment may carry conv-history rows in front of its own tokens with -inf
 * logits.  Arguments, limits and errors as gbla_state; `stats` must not
 * overlap any input or `state`.
 */
gbla_status gbla_state_stats(const void *k, const void *v, const void *gate,
                             const float *conv_w, const int32_t *seq_lens, float *state,
                             float *stats, int B, int H, int N, int D, gbla_dtype dtype,
                             gbla_algo algo, gbla_stream_t stream);

/*
 * gbla_combine_states -- the state of whole sequences from the states of P
 * disjoint token segments of them (a sequence split across devices; Sec. 2.1
 * item 2, the softmax-weighted sums split over the segments):
 *   M = max_p m_p,  w_p = l_p exp(m_p - M),  S = sum_p w_p S_p / sum_p w_p,
 * z likewise, sums in segment order p = 0 .. P-1 (deterministic); segments
 * with l_p = 0 weigh 0.
 *   states    [P, B, H, D*D + D] fp32: gbla_state_stats of each segment.
 *   stats     [P, B, H, 2] fp32:       their (m, l).
 *   state     [B, H, D*D + D] fp32:    output, as gbla_state of the whole.
 *   out_stats [B, H, 2] fp32:          output (M, sum_p w_p).
 * 1 <= P <= 1024, D in {32, 64, 128} (GBLA_ERR_INVALID_ARG / _UNSUPPORTED);
 * device pointers, 16-byte aligned, outputs not overlapping the inputs or
 * each other.  Asynchronous on `stream`; allocates nothing.
 */
gbla_status gbla_combine_states(const float *states, const float *stats, int P, float *state,
                                float *out_stats, int B, int H, int D, gbla_stream_t stream);

/*
 * gbla_readout -- the per-token part: Conv1D of q, phi, O_i = phi(q~_i)^T S /
 * phi(q~_i)^T z (Sec. 2.1 item 2) and the gated RMSNorm (Sec. 2.1 item 3),
 * from a state laid out as gbla_state writes it.  Any positive common scale
 * of S and z gives the same o.  Writes o rows t < L_b only.
 */
gbla_status gbla_readout(const void *q, const void *out_gate,
                         const float *conv_w, const float *norm_w,
                         const int32_t *seq_lens, const float *state, void *o,
                         int B, int H, int N, int D, gbla_dtype dtype,
                         gbla_algo algo, gbla_stream_t stream);

/*
 * gbla_forward_host -- gbla_forward for callers whose tensors live in HOST
 * memory (pinned for full copy speed; pageable works).  Same layouts as
 * above, all pointers host pointers.  Copies the inputs to device scratch,
 * runs the forward and copies rows t < L_b of o back: k, v and the gate
 * first, then q and out_gate in chunks of 4096 tokens whose readouts start as
 * they land, o going back chunk by chunk (two streams of its own beside
 * `stream`, joined to it); o is gbla_forward's bit for bit.  The call waits
 * for `stream`, so o is ready on return.
 */
gbla_status gbla_forward_host(const void *q, const void *k, const void *v,
                              const void *gate, const void *out_gate,
                              const float *conv_w, const float *norm_w,
                              const int32_t *seq_lens, void *o, int B, int H,
                              int N, int D, gbla_dtype dtype,
                              gbla_stream_t stream);

/*
 * gbla_state_static_scratch -- gbla_state for callers that cannot allocate
 * GPU memory.  The paper has no counterpart: this is a deployment variant.
 *
 * Same arguments, layouts and result as gbla_state with the CUDA-core kernel
 * family, but the partial sums live in a fixed array of
 * GBLA_STATIC_SCRATCH_BYTES compiled into the library, so the call allocates
 * nothing (no cudaMalloc, no pool, no library allocator).  Meant for callers
 * whose device memory is entirely owned by another allocator, or who cannot
 * take the latency of an allocation call.
 *
 * Limits and rules:
 *   - B * H * (D*D + D + 2) * 4 bytes must fit in GBLA_STATIC_SCRATCH_BYTES
 *     (at most 2015 (batch, head) pairs at D = 64, 507 at D = 128); larger
 *     problems return GBLA_ERR_INVALID_ARG before anything is enqueued.  Long
 *     sequences are cut into fewer, longer chunks to fit.
 *   - Each GPU that loads the library holds the array until the process exits.
 *   - The first call on a device looks up the array's device address on that
 *     device (once); make that first call before any stream capture starts.
 *     The address is kept until the process exits, so after cudaDeviceReset
 *     (or another teardown of the primary context) do not call it again on
 *     that device.
 *   - Every call shares the one array.  Calls that overlap on the GPU (other
 *     streams or threads) race on it: serialise them.  Nothing carries over
 *     between calls; each call writes all the scratch it later reads.
 */
#define GBLA_STATIC_SCRATCH_BYTES (32u << 20)
gbla_status gbla_state_static_scratch(const void *k, const void *v,
                                      const void *gate, const float *conv_w,
                                      const int32_t *seq_lens, float *state,
                                      int B, int H, int N, int D,
                                      gbla_dtype dtype, gbla_stream_t stream);

/* Number of floats per (b, h) in a state buffer: D*D + D. */
size_t gbla_state_floats(int D);

/* RMSNorm epsilon used by the readout (1e-6; the paper leaves it unstated). */
float gbla_rms_eps(void);

/* Static description of a status code; never NULL. */
const char *gbla_status_string(gbla_status status);

/* Library version, e.g. "0.1.0". */
const char *gbla_version(void);

/* Returns the unused memory of the library's per-device scratch pools to the
 * driver.  Scratch freed at the end of a call otherwise stays mapped for the
 * next call (up to the largest amount one call has used).  Safe at any time;
 * allocations still in use are kept. */
void gbla_release(void);

/* Number of kernels this library has enqueued since it was loaded, over all
 * devices and threads (a counter for benchmarks and tests). */
uint64_t gbla_launch_count(void);

/* Error bits recorded on the current device by a tensor-core kernel whose
 * bounded wait (2 s per wait) ran out; 0 when none did.  Such a kernel stops
 * early, leaves its outputs undefined and keeps the CUDA context usable.  The
 * call synchronises with the device; reset != 0 clears the word afterwards.
 * Returns 0xFFFFFFFF if the word could not be read. */
uint32_t gbla_device_error(int reset);

/* Text of the CUDA error behind the calling thread's last GBLA_ERR_CUDA
 * ("no error" if there was none); static storage, never NULL. */
const char *gbla_last_cuda_error(void);

#ifdef __cplusplus
}
#endif

#endif /* GBLA_H_ */
