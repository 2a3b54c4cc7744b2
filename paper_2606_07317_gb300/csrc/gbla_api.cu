// C-ABI front end of the GBLA core: argument validation, scratch memory and
// kernel-family dispatch.  All arithmetic happens in the kernels of
// gbla_simt.cu and gbla_tc.cu.
#include <string.h>

#include <atomic>
#include <mutex>
#include <vector>

#include "gbla_internal.cuh"

using namespace gbla;

namespace gbla {
static std::atomic<unsigned long long> g_launches{0};
void count_launch(unsigned n) { g_launches.fetch_add(n, std::memory_order_relaxed); }
}  // namespace gbla

namespace {

constexpr size_t kAlign = 16;

bool aligned(const void *p) { return ((uintptr_t)p % kAlign) == 0; }

size_t elem_bytes(gbla_dtype dt) { return dt == GBLA_FP32 ? 4 : 2; }

struct Range {
  uintptr_t lo, hi;
};
bool overlap(Range a, Range b) { return a.lo < b.hi && b.lo < a.hi; }
Range range_of(const void *p, size_t bytes) {
  return Range{(uintptr_t)p, (uintptr_t)p + bytes};
}

// Size limits: grid dimensions and 64-bit element counts.
constexpr int kMaxBH = 65535;
constexpr int kMaxN = 1 << 28;

}  // namespace

namespace gbla {

gbla_status check_dims(int B, int H, int N, int D, gbla_dtype dtype, bool *empty) {
  if (B < 0 || H < 0 || N < 0 || D < 0) return GBLA_ERR_INVALID_ARG;
  if (dtype != GBLA_FP32 && dtype != GBLA_BF16) return GBLA_ERR_UNSUPPORTED;
  if (D != 32 && D != 64 && D != 128) return GBLA_ERR_UNSUPPORTED;
  if (B > kMaxBH || H > kMaxBH || N > kMaxN) return GBLA_ERR_INVALID_ARG;
  if ((unsigned long long)B * N * H * D > (1ull << 40)) return GBLA_ERR_INVALID_ARG;
  *empty = (B == 0 || H == 0 || N == 0);
  return GBLA_OK;
}

gbla_status check_ptrs(std::initializer_list<const void *> ptrs) {
  for (const void *p : ptrs)
    if (p == nullptr) return GBLA_ERR_INVALID_ARG;
  for (const void *p : ptrs)
    if (!aligned(p)) return GBLA_ERR_INVALID_ARG;
  return GBLA_OK;
}

gbla_status check_seq_lens(const int32_t *seq_lens) {
  if (seq_lens != nullptr && ((uintptr_t)seq_lens % 4) != 0) return GBLA_ERR_INVALID_ARG;
  return GBLA_OK;
}

static thread_local cudaError_t t_last_cuda_error = cudaSuccess;

gbla_status from_cuda(cudaError_t e) {
  if (e == cudaSuccess) return GBLA_OK;
  t_last_cuda_error = e;
  (void)cudaGetLastError();  // clear the non-sticky launch error
  return GBLA_ERR_CUDA;
}

static const char *last_cuda_error_string() { return cudaGetErrorString(t_last_cuda_error); }

}  // namespace gbla

namespace {

bool use_tc(const Problem &p, gbla_algo algo, gbla_status *st) {
  *st = GBLA_OK;
  switch (algo) {
    case GBLA_ALGO_AUTO: return tc_supports(p);
    case GBLA_ALGO_SIMT: return false;
    case GBLA_ALGO_TC:
      if (!tc_supports(p)) *st = GBLA_ERR_UNSUPPORTED;
      return true;
    default: *st = GBLA_ERR_UNSUPPORTED; return false;
  }
}

// Library-owned stream-ordered memory pool per device.  Its release threshold
// is unbounded, so memory freed at the end of a call stays mapped for the
// next one instead of being returned to the driver (and mapped again);
// gbla_release() trims it.
constexpr int kMaxDevices = 64;
std::mutex g_pool_mu;
cudaMemPool_t g_pools[kMaxDevices] = {};

cudaMemPool_t device_pool() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return nullptr;
  std::lock_guard<std::mutex> lock(g_pool_mu);
  if (!g_pools[dev]) {
    cudaMemPoolProps props = {};
    props.allocType = cudaMemAllocationTypePinned;
    props.location.type = cudaMemLocationTypeDevice;
    props.location.id = dev;
    cudaMemPool_t pool = nullptr;
    if (cudaMemPoolCreate(&pool, &props) != cudaSuccess) {
      (void)cudaGetLastError();
      return nullptr;
    }
    uint64_t thr = UINT64_MAX;
    cudaMemPoolSetAttribute(pool, cudaMemPoolAttrReleaseThreshold, &thr);
    g_pools[dev] = pool;
  }
  return g_pools[dev];
}

// Stream-ordered scratch from the library pool: freed on the same stream after
// the kernels using it.
struct Scratch {
  void *ptr = nullptr;
  cudaStream_t st = nullptr;
  ~Scratch() { release(); }
  void release() {
    if (ptr) cudaFreeAsync(ptr, st);
    ptr = nullptr;
  }
  gbla_status alloc(size_t bytes, cudaStream_t s) {
    st = s;
    if (bytes == 0) return GBLA_OK;
    cudaMemPool_t pool = device_pool();
    cudaError_t e = pool ? cudaMallocFromPoolAsync(&ptr, bytes, pool, s)
                         : cudaMallocAsync(&ptr, bytes, s);
    if (e != cudaSuccess) {
      (void)cudaGetLastError();
      ptr = nullptr;
      return GBLA_ERR_ALLOC;
    }
    return GBLA_OK;
  }
};

size_t round_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// State (Conv1D of k, v, phi, gate, S and z) into `state`; with the tensor-core
// family also the key gate's softmax statistics into gate_stats, if given.
gbla_status run_state(const Problem &p, bool tc, const void *k, const void *v,
                      const void *gate, const float *conv_w, float *state,
                      cudaStream_t st, float2 *gate_stats = nullptr) {
  Scratch ws;
  if (tc) {
    gbla_status s = ws.alloc(tc_workspace_bytes(p), st);
    if (s != GBLA_OK) return s;
    return from_cuda(tc_state(p, k, v, gate, conv_w, ws.ptr, state, st, gate_stats));
  }
  SimtPlan plan = simt_plan(p);
  gbla_status s = ws.alloc(simt_partials_bytes(p, plan), st);
  if (s != GBLA_OK) return s;
  return from_cuda(simt_state(p, plan, k, v, gate, conv_w, (float *)ws.ptr, state, st));
}

// after_state: the kernel just before on the stream is this library's state
// reduction, so only the readout's reads of `state` wait for it.
gbla_status run_readout(const Problem &p, bool tc, const void *q, const void *og,
                        const float *conv_w, const float *norm_w, const float *state,
                        void *o, cudaStream_t st, bool after_state = false,
                        bool f32_out = false) {
  if (tc)
    return from_cuda(tc_readout(p, q, og, conv_w, norm_w, state, o, st, after_state, f32_out));
  return from_cuda(simt_readout(p, q, og, conv_w, norm_w, state, o, st, f32_out));
}

}  // namespace

extern "C" {

size_t gbla_state_floats(int D) { return D > 0 ? state_floats(D) : 0; }

float gbla_rms_eps(void) { return kRmsEps; }

const char *gbla_version(void) { return "0.1.0"; }

const char *gbla_status_string(gbla_status s) {
  switch (s) {
    case GBLA_OK: return "ok";
    case GBLA_ERR_INVALID_ARG: return "invalid argument";
    case GBLA_ERR_UNSUPPORTED: return "unsupported configuration";
    case GBLA_ERR_ALLOC: return "scratch allocation failed";
    case GBLA_ERR_CUDA: return "CUDA error";
  }
  return "unknown status";
}

void gbla_release(void) {
  std::lock_guard<std::mutex> lock(g_pool_mu);
  for (int d = 0; d < kMaxDevices; ++d)
    if (g_pools[d]) cudaMemPoolTrimTo(g_pools[d], 0);
}

uint64_t gbla_launch_count(void) { return g_launches.load(std::memory_order_relaxed); }

uint32_t gbla_device_error(int reset) {
  const unsigned a = tc_device_error(reset != 0), b = project_device_error(reset != 0);
  const unsigned c = bwd_device_error(reset != 0), d = sa_device_error(reset != 0);
  return (a == 0xFFFFFFFFu || b == 0xFFFFFFFFu || c == 0xFFFFFFFFu || d == 0xFFFFFFFFu)
             ? 0xFFFFFFFFu
             : (a | b | c | d);
}

const char *gbla_last_cuda_error(void) { return last_cuda_error_string(); }

gbla_status gbla_state(const void *k, const void *v, const void *gate,
                       const float *conv_w, const int32_t *seq_lens, float *state,
                       int B, int H, int N, int D, gbla_dtype dtype, gbla_algo algo,
                       gbla_stream_t stream) {
  bool empty = false;
  gbla_status s = check_dims(B, H, N, D, dtype, &empty);
  if (s != GBLA_OK || empty) return s;
  if ((s = check_ptrs({k, v, gate, conv_w, state})) != GBLA_OK) return s;
  if ((s = check_seq_lens(seq_lens)) != GBLA_OK) return s;
  const size_t in_bytes = (size_t)B * N * H * D * elem_bytes(dtype);
  const Range out = range_of(state, sizeof(float) * state_floats(D) * B * H);
  if (overlap(out, range_of(k, in_bytes)) || overlap(out, range_of(v, in_bytes)) ||
      overlap(out, range_of(gate, (size_t)B * N * H * elem_bytes(dtype))) ||
      overlap(out, range_of(conv_w, sizeof(float) * 3 * H * D * kConvW)))
    return GBLA_ERR_INVALID_ARG;
  Problem p{B, H, N, D, dtype, seq_lens};
  bool tc = use_tc(p, algo, &s);
  if (s != GBLA_OK) return s;
  return run_state(p, tc, k, v, gate, conv_w, state, (cudaStream_t)stream);
}

gbla_status gbla_state_stats(const void *k, const void *v, const void *gate,
                             const float *conv_w, const int32_t *seq_lens, float *state,
                             float *stats, int B, int H, int N, int D, gbla_dtype dtype,
                             gbla_algo algo, gbla_stream_t stream) {
  bool empty = false;
  gbla_status s = check_dims(B, H, N, D, dtype, &empty);
  if (s != GBLA_OK || empty) return s;
  if ((s = check_ptrs({k, v, gate, conv_w, state, stats})) != GBLA_OK) return s;
  if ((s = check_seq_lens(seq_lens)) != GBLA_OK) return s;
  const size_t in_bytes = (size_t)B * N * H * D * elem_bytes(dtype);
  const Range out = range_of(state, sizeof(float) * state_floats(D) * B * H);
  const Range outs = range_of(stats, sizeof(float) * 2 * B * H);
  for (const Range &o : {out, outs})
    if (overlap(o, range_of(k, in_bytes)) || overlap(o, range_of(v, in_bytes)) ||
        overlap(o, range_of(gate, (size_t)B * N * H * elem_bytes(dtype))) ||
        overlap(o, range_of(conv_w, sizeof(float) * 3 * H * D * kConvW)) ||
        (seq_lens && overlap(o, range_of(seq_lens, sizeof(int32_t) * B))))
      return GBLA_ERR_INVALID_ARG;
  if (overlap(out, outs)) return GBLA_ERR_INVALID_ARG;
  Problem p{B, H, N, D, dtype, seq_lens};
  bool tc = use_tc(p, algo, &s);
  if (s != GBLA_OK) return s;
  cudaStream_t st = (cudaStream_t)stream;
  if (tc)  // the tensor-core reduction writes the statistics as it combines the records
    return run_state(p, tc, k, v, gate, conv_w, state, st, (float2 *)stats);
  if ((s = run_state(p, tc, k, v, gate, conv_w, state, st)) != GBLA_OK) return s;
  Scratch part;
  if ((s = part.alloc(sizeof(float) * gate_stats_part_floats(p), st)) != GBLA_OK) return s;
  return from_cuda(gate_stats(p, gate, (float2 *)part.ptr, (float2 *)stats, st));
}

gbla_status gbla_combine_states(const float *states, const float *stats, int P, float *state,
                                float *out_stats, int B, int H, int D, gbla_stream_t stream) {
  if (P <= 0 || P > 1024 || B < 0 || H < 0) return GBLA_ERR_INVALID_ARG;
  if (D != 32 && D != 64 && D != 128) return GBLA_ERR_UNSUPPORTED;
  if ((long long)B * H == 0) return GBLA_OK;
  gbla_status s = check_ptrs({states, stats, state, out_stats});
  if (s != GBLA_OK) return s;
  const size_t BH = (size_t)B * H;
  const Range ins[2] = {range_of(states, sizeof(float) * state_floats(D) * BH * P),
                        range_of(stats, sizeof(float) * 2 * BH * P)};
  const Range outs[2] = {range_of(state, sizeof(float) * state_floats(D) * BH),
                         range_of(out_stats, sizeof(float) * 2 * BH)};
  for (const Range &o : outs)
    for (const Range &i : ins)
      if (overlap(o, i)) return GBLA_ERR_INVALID_ARG;
  if (overlap(outs[0], outs[1])) return GBLA_ERR_INVALID_ARG;
  return from_cuda(combine_states(states, (const float2 *)stats, P, (int)BH, D, state,
                                  (float2 *)out_stats, (cudaStream_t)stream));
}

gbla_status gbla_readout(const void *q, const void *out_gate, const float *conv_w,
                         const float *norm_w, const int32_t *seq_lens,
                         const float *state, void *o, int B, int H, int N, int D,
                         gbla_dtype dtype, gbla_algo algo, gbla_stream_t stream) {
  bool empty = false;
  gbla_status s = check_dims(B, H, N, D, dtype, &empty);
  if (s != GBLA_OK || empty) return s;
  if ((s = check_ptrs({q, out_gate, conv_w, norm_w, state, o})) != GBLA_OK) return s;
  if ((s = check_seq_lens(seq_lens)) != GBLA_OK) return s;
  const size_t bytes = (size_t)B * N * H * D * elem_bytes(dtype);
  const Range out = range_of(o, bytes);
  if (overlap(out, range_of(q, bytes)) || overlap(out, range_of(out_gate, bytes)) ||
      overlap(out, range_of(state, sizeof(float) * state_floats(D) * B * H)) ||
      overlap(out, range_of(conv_w, sizeof(float) * 3 * H * D * kConvW)) ||
      overlap(out, range_of(norm_w, sizeof(float) * H * D)))
    return GBLA_ERR_INVALID_ARG;
  Problem p{B, H, N, D, dtype, seq_lens};
  bool tc = use_tc(p, algo, &s);
  if (s != GBLA_OK) return s;
  return run_readout(p, tc, q, out_gate, conv_w, norm_w, state, o, (cudaStream_t)stream);
}

gbla_status gbla_forward_ex(const void *q, const void *k, const void *v,
                            const void *gate, const void *out_gate,
                            const float *conv_w, const float *norm_w,
                            const int32_t *seq_lens, void *o, int B, int H, int N,
                            int D, gbla_dtype dtype, gbla_algo algo,
                            gbla_stream_t stream) {
  return gbla_forward_variant(q, k, v, gate, out_gate, conv_w, norm_w, seq_lens, o, B, H, N,
                              D, dtype, algo, 0u, stream);
}

// gbla_forward_variant, and with f32_out the debug path of gbla_forward_f32out
// (o is then fp32 whatever the input dtype).
static gbla_status forward_impl(const void *q, const void *k, const void *v, const void *gate,
                                const void *out_gate, const float *conv_w,
                                const float *norm_w, const int32_t *seq_lens, void *o, int B,
                                int H, int N, int D, gbla_dtype dtype, gbla_algo algo,
                                uint32_t flags, bool f32_out, gbla_stream_t stream) {
  if (flags & ~(uint32_t)GBLA_FLAG_BLA) return GBLA_ERR_INVALID_ARG;
  bool empty = false;
  gbla_status s = check_dims(B, H, N, D, dtype, &empty);
  if (s != GBLA_OK || empty) return s;
  if ((s = check_ptrs({q, k, v, gate, out_gate, conv_w, norm_w, o})) != GBLA_OK) return s;
  if ((s = check_seq_lens(seq_lens)) != GBLA_OK) return s;
  const size_t bytes = (size_t)B * N * H * D * elem_bytes(dtype);
  const Range out = range_of(o, f32_out ? (size_t)B * N * H * D * sizeof(float) : bytes);
  if (overlap(out, range_of(q, bytes)) || overlap(out, range_of(k, bytes)) ||
      overlap(out, range_of(v, bytes)) || overlap(out, range_of(out_gate, bytes)) ||
      overlap(out, range_of(gate, (size_t)B * N * H * elem_bytes(dtype))) ||
      overlap(out, range_of(conv_w, sizeof(float) * 3 * H * D * kConvW)) ||
      overlap(out, range_of(norm_w, sizeof(float) * H * D)) ||
      (seq_lens && overlap(out, range_of(seq_lens, sizeof(int32_t) * B))))
    return GBLA_ERR_INVALID_ARG;
  Problem p{B, H, N, D, dtype, seq_lens, flags};
  bool tc = use_tc(p, algo, &s);
  if (s != GBLA_OK) return s;
  cudaStream_t st = (cudaStream_t)stream;
  Scratch state;
  if ((s = state.alloc(sizeof(float) * state_floats(D) * B * H, st)) != GBLA_OK) return s;
  if ((s = run_state(p, tc, k, v, gate, conv_w, (float *)state.ptr, st)) != GBLA_OK) return s;
  return run_readout(p, tc, q, out_gate, conv_w, norm_w, (const float *)state.ptr, o, st,
                     true, f32_out);
}

gbla_status gbla_forward_variant(const void *q, const void *k, const void *v,
                                 const void *gate, const void *out_gate,
                                 const float *conv_w, const float *norm_w,
                                 const int32_t *seq_lens, void *o, int B, int H, int N,
                                 int D, gbla_dtype dtype, gbla_algo algo, uint32_t flags,
                                 gbla_stream_t stream) {
  return forward_impl(q, k, v, gate, out_gate, conv_w, norm_w, seq_lens, o, B, H, N, D, dtype,
                      algo, flags, false, stream);
}

gbla_status gbla_forward_f32out(const void *q, const void *k, const void *v,
                                const void *gate, const void *out_gate,
                                const float *conv_w, const float *norm_w,
                                const int32_t *seq_lens, float *o32, int B, int H, int N,
                                int D, gbla_dtype dtype, gbla_algo algo,
                                gbla_stream_t stream) {
  return forward_impl(q, k, v, gate, out_gate, conv_w, norm_w, seq_lens, o32, B, H, N, D,
                      dtype, algo, 0u, true, stream);
}

gbla_status gbla_forward(const void *q, const void *k, const void *v,
                         const void *gate, const void *out_gate,
                         const float *conv_w, const float *norm_w,
                         const int32_t *seq_lens, void *o, int B, int H, int N,
                         int D, gbla_dtype dtype, gbla_stream_t stream) {
  return gbla_forward_ex(q, k, v, gate, out_gate, conv_w, norm_w, seq_lens, o, B, H,
                         N, D, dtype, GBLA_ALGO_AUTO, stream);
}

gbla_status gbla_backward(const void *q, const void *k, const void *v, const void *gate,
                          const void *out_gate, const float *conv_w, const float *norm_w,
                          const int32_t *seq_lens, const void *dy, void *dq, void *dk,
                          void *dv, void *dgate, void *dout_gate, float *dconv_w,
                          float *dnorm_w, int B, int H, int N, int D, gbla_dtype dtype,
                          gbla_stream_t stream) {
  return gbla_backward_variant(q, k, v, gate, out_gate, conv_w, norm_w, seq_lens, dy, dq, dk,
                               dv, dgate, dout_gate, dconv_w, dnorm_w, B, H, N, D, dtype, 0u,
                               stream);
}

}  // extern "C"

// gbla_backward_variant, and gbla_backward_from_state when `saved` (state_in and
// stats_in are the forward's state and gate statistics; flags 0): the state
// pass is then skipped.
static gbla_status backward_impl(const void *q, const void *k, const void *v, const void *gate,
                                 const void *out_gate, const float *conv_w, const float *norm_w,
                                 const int32_t *seq_lens, const float *state_in,
                                 const float *stats_in, const void *dy, void *dq, void *dk,
                                 void *dv, void *dgate, void *dout_gate, float *dconv_w,
                                 float *dnorm_w, int B, int H, int N, int D, gbla_dtype dtype,
                                 uint32_t flags, bool saved, gbla_stream_t stream) {
  if (flags & ~(uint32_t)GBLA_FLAG_BLA) return GBLA_ERR_INVALID_ARG;
  bool empty = false;
  gbla_status s = check_dims(B, H, N, D, dtype, &empty);
  if (s != GBLA_OK) return s;
  if ((s = check_ptrs({q, k, v, gate, out_gate, conv_w, norm_w, dy, dq, dk, dv, dgate,
                       dout_gate, dconv_w, dnorm_w})) != GBLA_OK)
    return s;
  if ((s = check_seq_lens(seq_lens)) != GBLA_OK) return s;
  cudaStream_t st = (cudaStream_t)stream;
  const size_t wbytes = sizeof(float) * 3 * H * D * kConvW, nbytes = sizeof(float) * H * D;
  if (empty) {  // no tokens: the weight gradients are empty sums
    if (H > 0 && (cudaMemsetAsync(dconv_w, 0, wbytes, st) != cudaSuccess ||
                  cudaMemsetAsync(dnorm_w, 0, nbytes, st) != cudaSuccess))
      return GBLA_ERR_CUDA;
    return GBLA_OK;
  }
  if (saved && (state_in == nullptr || stats_in == nullptr || !aligned(state_in) ||
                !aligned(stats_in)))
    return GBLA_ERR_INVALID_ARG;
  const size_t bytes = (size_t)B * N * H * D * elem_bytes(dtype);
  const size_t gbytes = (size_t)B * N * H * elem_bytes(dtype);
  const Range outs[7] = {range_of(dq, bytes),     range_of(dk, bytes),
                         range_of(dv, bytes),     range_of(dgate, gbytes),
                         range_of(dout_gate, bytes), range_of(dconv_w, wbytes),
                         range_of(dnorm_w, nbytes)};
  const Range ins[9] = {range_of(q, bytes),      range_of(k, bytes),
                        range_of(v, bytes),      range_of(out_gate, bytes),
                        range_of(dy, bytes),     range_of(gate, gbytes),
                        range_of(conv_w, wbytes), range_of(norm_w, nbytes),
                        range_of(seq_lens, seq_lens ? sizeof(int32_t) * B : 0)};
  const Range kept[2] = {range_of(state_in, sizeof(float) * state_floats(D) * B * H),
                          range_of(stats_in, sizeof(float) * 2 * B * H)};
  for (int i = 0; i < 7; ++i) {
    for (int j = 0; j < 9; ++j)
      if (overlap(outs[i], ins[j])) return GBLA_ERR_INVALID_ARG;
    for (int j = 0; j < 2; ++j)
      if (saved && overlap(outs[i], kept[j])) return GBLA_ERR_INVALID_ARG;
    for (int j = i + 1; j < 7; ++j)
      if (overlap(outs[i], outs[j])) return GBLA_ERR_INVALID_ARG;
  }
  Problem p{B, H, N, D, dtype, seq_lens, 0u};
  bool tc = use_tc(p, GBLA_ALGO_AUTO, &s);
  if (s != GBLA_OK) return s;
  const BwdLayout lay = bwd_layout(p);
  // Ablations (Table 4): the identity Conv1D and the uniform key gate are the
  // full core on substituted inputs -- taps (0, 0, 0, 1) on every channel,
  // and all-zero gate logits, whose softmax over the valid positions is
  // 1 / L_b -- so every kernel runs as is on them; the gradients of the
  // parameters a variant does not use are zero.  Without the gated RMSNorm
  // the query pass takes dO = dy (its CUDA-core build; the tensor-core token
  // passes serve the full core only).
  const size_t tap_floats = (flags & GBLA_FLAG_NO_CONV) ? (size_t)3 * H * D * kConvW : 0;
  const size_t zgate_bytes = (flags & GBLA_FLAG_NO_GATE) ? gbytes : 0;
  const size_t sub_off = round_up(sizeof(float) * lay.total, 256);
  Scratch scr;
  if ((s = scr.alloc(sub_off + round_up(sizeof(float) * tap_floats, 256) + zgate_bytes, st)) !=
      GBLA_OK)
    return s;
  float *base = (float *)scr.ptr;
  const float *cw = conv_w;
  const void *gt = gate;
  if (tap_floats) {
    float *taps = (float *)((char *)scr.ptr + sub_off);
    if (fill_identity_taps(taps, 3 * H * D, st) != cudaSuccess) return GBLA_ERR_CUDA;
    cw = taps;
  }
  if (zgate_bytes) {
    void *zg = (char *)scr.ptr + sub_off + round_up(sizeof(float) * tap_floats, 256);
    if (cudaMemsetAsync(zg, 0, zgate_bytes, st) != cudaSuccess) return GBLA_ERR_CUDA;
    gt = zg;
  }
  BwdArgs a{q, k, v, gt, out_gate, dy, cw, norm_w, dq, dk, dv, dgate, dout_gate,
            dconv_w, dnorm_w, base + lay.state, (const float2 *)(base + lay.stats)};
  bool stats_ready = tc;
  if (saved) {  // the forward's own state and gate statistics
    a.state = state_in;
    a.stats = (const float2 *)stats_in;
    stats_ready = true;
  } else if ((s = run_state(p, tc, k, v, gt, cw, base + lay.state, st,
                            tc ? (float2 *)(base + lay.stats) : nullptr)) != GBLA_OK) {
    // the forward state S, z through the forward's own state path, which on
    // tensor cores also yields the gate statistics the backward needs
    return s;
  }
  Problem pb = p;
  pb.flags = flags;
  if ((s = from_cuda(bwd_run(pb, a, base, stats_ready, st))) != GBLA_OK) return s;
  if (((flags & GBLA_FLAG_NO_CONV) && cudaMemsetAsync(dconv_w, 0, wbytes, st) != cudaSuccess) ||
      ((flags & GBLA_FLAG_NO_GATE) && cudaMemsetAsync(dgate, 0, gbytes, st) != cudaSuccess))
    return from_cuda(cudaGetLastError());
  return GBLA_OK;
}

extern "C" {

gbla_status gbla_backward_variant(const void *q, const void *k, const void *v,
                                  const void *gate, const void *out_gate,
                                  const float *conv_w, const float *norm_w,
                                  const int32_t *seq_lens, const void *dy, void *dq, void *dk,
                                  void *dv, void *dgate, void *dout_gate, float *dconv_w,
                                  float *dnorm_w, int B, int H, int N, int D,
                                  gbla_dtype dtype, uint32_t flags, gbla_stream_t stream) {
  return backward_impl(q, k, v, gate, out_gate, conv_w, norm_w, seq_lens, nullptr, nullptr, dy,
                       dq, dk, dv, dgate, dout_gate, dconv_w, dnorm_w, B, H, N, D, dtype, flags,
                       false, stream);
}

gbla_status gbla_backward_from_state(const void *q, const void *k, const void *v,
                                     const void *gate, const void *out_gate,
                                     const float *conv_w, const float *norm_w,
                                     const int32_t *seq_lens, const float *state,
                                     const float *stats, const void *dy, void *dq, void *dk,
                                     void *dv, void *dgate, void *dout_gate, float *dconv_w,
                                     float *dnorm_w, int B, int H, int N, int D,
                                     gbla_dtype dtype, gbla_stream_t stream) {
  return backward_impl(q, k, v, gate, out_gate, conv_w, norm_w, seq_lens, state, stats, dy,
                       dq, dk, dv, dgate, dout_gate, dconv_w, dnorm_w, B, H, N, D, dtype, 0u,
                       true, stream);
}

// Validation shared by gbla_project and gbla_layer_forward.
static gbla_status check_project(const void *x, const float *conv_x, const void *w,
                                 const int32_t *seq_lens, int B, int N, int d, int H, int D,
                                 gbla_dtype dtype, bool *empty) {
  gbla_status s = check_dims(B, H, N, D, dtype, empty);
  if (s != GBLA_OK) return s;
  if (d < 0) return GBLA_ERR_INVALID_ARG;
  if (dtype != GBLA_BF16) return GBLA_ERR_UNSUPPORTED;
  if ((s = check_ptrs({x, conv_x, w})) != GBLA_OK) return s;
  if ((s = check_seq_lens(seq_lens)) != GBLA_OK) return s;
  if (*empty) return GBLA_OK;
  ProjProblem pp{B, N, d, H, D, seq_lens};
  if (!project_supports(pp)) return GBLA_ERR_UNSUPPORTED;
  return GBLA_OK;
}

gbla_status gbla_project(const void *x, const float *conv_x, const void *w_proj,
                         const int32_t *seq_lens, void *q, void *k, void *v,
                         void *out_gate, void *gate, int B, int N, int d, int H,
                         int D, gbla_dtype dtype, gbla_stream_t stream) {
  bool empty = false;
  gbla_status s = check_project(x, conv_x, w_proj, seq_lens, B, N, d, H, D, dtype, &empty);
  if (s != GBLA_OK) return s;
  if ((s = check_ptrs({q, k, v, out_gate, gate})) != GBLA_OK) return s;
  if (empty) return GBLA_OK;
  const size_t tok = (size_t)B * N;
  const size_t sb = tok * H * D * 2, gb = tok * H * 2;
  const Range outs[5] = {range_of(q, sb), range_of(k, sb), range_of(v, sb),
                         range_of(out_gate, sb), range_of(gate, gb)};
  const Range ins[4] = {range_of(x, tok * d * 2), range_of(conv_x, sizeof(float) * d * kConvW),
                        range_of(w_proj, ((size_t)4 * H * D + H) * d * 2),
                        range_of(seq_lens, seq_lens ? sizeof(int32_t) * B : 0)};
  for (int i = 0; i < 5; ++i) {
    for (int j = 0; j < 4; ++j)
      if (overlap(outs[i], ins[j])) return GBLA_ERR_INVALID_ARG;
    for (int j = i + 1; j < 5; ++j)
      if (overlap(outs[i], outs[j])) return GBLA_ERR_INVALID_ARG;
  }
  ProjProblem pp{B, N, d, H, D, seq_lens};
  return from_cuda(tc_project(pp, x, conv_x, w_proj, q, k, v, out_gate, gate,
                              (cudaStream_t)stream));
}

gbla_status gbla_layer_forward(const void *x, const float *conv_x, const void *w_proj,
                               const float *norm_w, const int32_t *seq_lens, void *o,
                               int B, int N, int d, int H, int D, gbla_dtype dtype,
                               gbla_stream_t stream) {
  bool empty = false;
  gbla_status s = check_project(x, conv_x, w_proj, seq_lens, B, N, d, H, D, dtype, &empty);
  if (s != GBLA_OK) return s;
  if ((s = check_ptrs({norm_w, o})) != GBLA_OK) return s;
  if (empty) return GBLA_OK;
  const size_t tok = (size_t)B * N;
  const size_t sb = tok * H * D * 2, gb = tok * H * 2;
  const Range out = range_of(o, sb);
  if (overlap(out, range_of(x, tok * d * 2)) ||
      overlap(out, range_of(conv_x, sizeof(float) * d * kConvW)) ||
      overlap(out, range_of(w_proj, ((size_t)4 * H * D + H) * d * 2)) ||
      overlap(out, range_of(norm_w, sizeof(float) * H * D)) ||
      (seq_lens && overlap(out, range_of(seq_lens, sizeof(int32_t) * B))))
    return GBLA_ERR_INVALID_ARG;
  cudaStream_t st = (cudaStream_t)stream;
  Problem p{B, H, N, D, dtype, seq_lens, (uint32_t)GBLA_FLAG_NO_CONV};
  bool tc = use_tc(p, GBLA_ALGO_AUTO, &s);
  if (s != GBLA_OK) return s;
  // q, k, v, out_gate, gate, then the state, in one scratch block
  const size_t off_g = 4 * sb, off_s = round_up(off_g + gb, 256);
  const size_t st_bytes = sizeof(float) * state_floats(D) * B * H;
  Scratch scr;
  if ((s = scr.alloc(off_s + st_bytes, st)) != GBLA_OK) return s;
  char *base = (char *)scr.ptr;
  void *q = base, *k = base + sb, *v = base + 2 * sb, *og = base + 3 * sb, *gate = base + off_g;
  float *state = (float *)(base + off_s);
  ProjProblem pp{B, N, d, H, D, seq_lens};
  if ((s = from_cuda(tc_project(pp, x, conv_x, w_proj, q, k, v, og, gate, st))) != GBLA_OK)
    return s;
  // the core with its Conv1D off (the taps are never read)
  if ((s = run_state(p, tc, k, v, gate, nullptr, state, st)) != GBLA_OK) return s;
  return run_readout(p, tc, q, og, nullptr, norm_w, state, o, st, true);
}

gbla_status gbla_attention_forward(const void *q, const void *k, const void *v,
                                   const int32_t *seq_lens, void *o, int B, int H, int N,
                                   int D, gbla_dtype dtype, gbla_stream_t stream) {
  bool empty = false;
  gbla_status s = check_dims(B, H, N, D, dtype, &empty);
  if (s != GBLA_OK || empty) return s;
  if ((s = check_ptrs({q, k, v, o})) != GBLA_OK) return s;
  if ((s = check_seq_lens(seq_lens)) != GBLA_OK) return s;
  if (!sa_supports(D, dtype)) return GBLA_ERR_UNSUPPORTED;
  const size_t bytes = (size_t)B * N * H * D * elem_bytes(dtype);
  const Range out = range_of(o, bytes);
  if (overlap(out, range_of(q, bytes)) || overlap(out, range_of(k, bytes)) ||
      overlap(out, range_of(v, bytes)) ||
      (seq_lens && overlap(out, range_of(seq_lens, sizeof(int32_t) * B))))
    return GBLA_ERR_INVALID_ARG;
  return from_cuda(sa_forward(q, k, v, seq_lens, o, B, H, N, (cudaStream_t)stream));
}

gbla_status gbla_forward_host(const void *q, const void *k, const void *v,
                              const void *gate, const void *out_gate,
                              const float *conv_w, const float *norm_w,
                              const int32_t *seq_lens, void *o, int B, int H, int N,
                              int D, gbla_dtype dtype, gbla_stream_t stream) {
  bool empty = false;
  gbla_status s = check_dims(B, H, N, D, dtype, &empty);
  if (s != GBLA_OK || empty) return s;
  if (!q || !k || !v || !gate || !out_gate || !conv_w || !norm_w || !o)
    return GBLA_ERR_INVALID_ARG;
  cudaStream_t st = (cudaStream_t)stream;
  const size_t es = elem_bytes(dtype);
  const size_t row = (size_t)H * D * es;        // one token of [N, H, D]
  const size_t grow = (size_t)H * es;           // one token of the gate
  const size_t tens = (size_t)B * N * row;      // one [B, N, H, D] tensor
  const size_t gbytes = (size_t)B * N * grow;
  const size_t cw = sizeof(float) * 3 * H * D * kConvW, nw = sizeof(float) * H * D;
  const size_t F = state_floats(D);
  auto valid_rows = [&](int b) -> size_t {
    long L = seq_lens ? seq_lens[b] : N;
    return (size_t)(L < 0 ? 0 : (L > N ? N : L));
  };
  // The readout goes in chunks of up to kHostChunk tokens of one batch row.  A
  // chunk's readout sees the h0 = min(3, t0) rows before it as Conv1D history:
  // its view of q and out_gate starts h0 rows early, and its output view, of
  // its own in the o region (obase: first row), holds those h0 rows' outputs
  // (not copied out) before the chunk's own.  Per token the readout does the
  // same arithmetic however the rows are cut, so o is that of gbla_forward.
  constexpr int kHostChunk = 4096;
  struct Chunk {
    int b, t0, t1;
    size_t obase;
  };
  std::vector<Chunk> chunks;
  size_t orows = 0;
  try {  // no exception may leave this C entry point
    for (int b = 0; b < B; ++b) {
      const int L = (int)valid_rows(b);
      for (int t0 = 0; t0 < L; t0 += kHostChunk) {
        const int t1 = t0 + kHostChunk < L ? t0 + kHostChunk : L;
        chunks.push_back({b, t0, t1, orows});
        orows += (size_t)(t1 - t0) + (size_t)(t0 < 3 ? t0 : 3);
      }
    }
  } catch (...) {
    return GBLA_ERR_ALLOC;
  }
  // Layout of the device scratch: q k v og | o chunks | gate | conv_w | norm_w |
  // seq_lens | state
  size_t off[10];
  size_t at = 0;
  for (int i = 0; i < 4; ++i) { off[i] = at; at = round_up(at + tens, 256); }
  off[4] = at; at = round_up(at + orows * row, 256);
  off[5] = at; at = round_up(at + gbytes, 256);
  off[6] = at; at = round_up(at + cw, 256);
  off[7] = at; at = round_up(at + nw, 256);
  off[8] = at; at = round_up(at + sizeof(int32_t) * B, 256);
  off[9] = at; at = round_up(at + sizeof(float) * F * B * H, 256);
  Problem p{B, H, N, D, dtype, nullptr};
  bool tc = use_tc(p, GBLA_ALGO_AUTO, &s);
  if (s != GBLA_OK) return s;
  Scratch dev;
  if ((s = dev.alloc(at, st)) != GBLA_OK) return s;
  char *base = (char *)dev.ptr;
  // rows [t0, t1) of batch row b of a [B, N, ...] host tensor into device slot i
  auto h2d = [&](int i, const void *src, size_t stride, int b, size_t t0, size_t t1,
                 cudaStream_t cs) {
    if (t1 <= t0) return cudaSuccess;
    const size_t o0 = ((size_t)b * N + t0) * stride;
    return cudaMemcpyAsync(base + off[i] + o0, (const char *)src + o0, (t1 - t0) * stride,
                           cudaMemcpyHostToDevice, cs);
  };
  // Streams: `stream` takes k, v, the gate and the weights, the state and the
  // readouts; `in_st` takes q and out_gate after k, v and the gate (the copies
  // share the host link, so they go in that order) while the state runs;
  // `out_st` takes o out chunk by chunk while later chunks come in.
  cudaStream_t in_st = nullptr, out_st = nullptr;
  cudaEvent_t ev_kvg = nullptr, ev_in = nullptr, ev_out = nullptr, ev_done = nullptr;
  auto cleanup = [&]() {
    if (ev_kvg) cudaEventDestroy(ev_kvg);
    if (ev_in) cudaEventDestroy(ev_in);
    if (ev_out) cudaEventDestroy(ev_out);
    if (ev_done) cudaEventDestroy(ev_done);
    if (in_st) cudaStreamDestroy(in_st);
    if (out_st) cudaStreamDestroy(out_st);
  };
  if (cudaStreamCreateWithFlags(&in_st, cudaStreamNonBlocking) != cudaSuccess ||
      cudaStreamCreateWithFlags(&out_st, cudaStreamNonBlocking) != cudaSuccess ||
      cudaEventCreateWithFlags(&ev_kvg, cudaEventDisableTiming) != cudaSuccess ||
      cudaEventCreateWithFlags(&ev_in, cudaEventDisableTiming) != cudaSuccess ||
      cudaEventCreateWithFlags(&ev_out, cudaEventDisableTiming) != cudaSuccess ||
      cudaEventCreateWithFlags(&ev_done, cudaEventDisableTiming) != cudaSuccess) {
    const cudaError_t e = cudaGetLastError();
    cleanup();
    dev.release();
    return from_cuda(e);
  }
  cudaError_t e = cudaSuccess;
  // 1. What the state needs (k, v, gate, weights, lengths), then the state.
  for (int b = 0; b < B && e == cudaSuccess; ++b) {
    const size_t L = valid_rows(b);
    if ((e = h2d(1, k, row, b, 0, L, st)) == cudaSuccess &&
        (e = h2d(2, v, row, b, 0, L, st)) == cudaSuccess)
      e = h2d(5, gate, grow, b, 0, L, st);
  }
  if (e == cudaSuccess &&
      (e = cudaMemcpyAsync(base + off[6], conv_w, cw, cudaMemcpyHostToDevice, st)) == cudaSuccess)
    e = cudaMemcpyAsync(base + off[7], norm_w, nw, cudaMemcpyHostToDevice, st);
  const int32_t *dsl = nullptr;
  if (e == cudaSuccess && seq_lens) {
    e = cudaMemcpyAsync(base + off[8], seq_lens, sizeof(int32_t) * B, cudaMemcpyHostToDevice, st);
    dsl = (const int32_t *)(base + off[8]);
  }
  if (e == cudaSuccess && (e = cudaEventRecord(ev_kvg, st)) == cudaSuccess)
    e = cudaStreamWaitEvent(in_st, ev_kvg, 0);
  p.seq_lens = dsl;
  float *state = (float *)(base + off[9]);
  const float *dcw = (const float *)(base + off[6]), *dnw = (const float *)(base + off[7]);
  if (e == cudaSuccess)
    s = run_state(p, tc, base + off[1], base + off[2], base + off[5], dcw, state, st);
  // 2. The readout chunk by chunk: its q and out_gate rows in on `in_st`, its
  // readout on `stream` (after the state), its o out on `out_st`.
  for (size_t c = 0; c < chunks.size() && e == cudaSuccess && s == GBLA_OK; ++c) {
    const Chunk &ch = chunks[c];
    const int h0 = ch.t0 < 3 ? ch.t0 : 3, n = ch.t1 - ch.t0 + h0;
    if ((e = h2d(0, q, row, ch.b, ch.t0, ch.t1, in_st)) != cudaSuccess ||
        (e = h2d(3, out_gate, row, ch.b, ch.t0, ch.t1, in_st)) != cudaSuccess ||
        (e = cudaEventRecord(ev_in, in_st)) != cudaSuccess ||
        (e = cudaStreamWaitEvent(st, ev_in, 0)) != cudaSuccess)
      break;
    const size_t v0 = ((size_t)ch.b * N + (ch.t0 - h0)) * row;  // first row of the view
    Problem pc{1, H, n, D, dtype, nullptr};  // every row of the view is valid
    char *ov = base + off[4] + ch.obase * row;
    if ((s = run_readout(pc, tc, base + off[0] + v0, base + off[3] + v0, dcw, dnw,
                         state + (size_t)ch.b * H * F, ov, st)) != GBLA_OK)
      break;
    if ((e = cudaEventRecord(ev_out, st)) != cudaSuccess ||
        (e = cudaStreamWaitEvent(out_st, ev_out, 0)) != cudaSuccess)
      break;
    e = cudaMemcpyAsync((char *)o + ((size_t)ch.b * N + ch.t0) * row, ov + (size_t)h0 * row,
                        (size_t)(ch.t1 - ch.t0) * row, cudaMemcpyDeviceToHost, out_st);
  }
  // the scratch is freed on `stream` only after both side streams are done with it
  const cudaError_t ej = [&]() {
    cudaError_t x;
    if ((x = cudaEventRecord(ev_done, in_st)) != cudaSuccess ||
        (x = cudaStreamWaitEvent(st, ev_done, 0)) != cudaSuccess ||
        (x = cudaEventRecord(ev_done, out_st)) != cudaSuccess)
      return x;
    return cudaStreamWaitEvent(st, ev_done, 0);
  }();
  if (e == cudaSuccess) e = ej;
  dev.release();
  const cudaError_t es2 = cudaStreamSynchronize(st);
  cleanup();
  if (s != GBLA_OK) return s;
  if (e != cudaSuccess) return from_cuda(e);
  return from_cuda(es2);
}

}  // extern "C"
