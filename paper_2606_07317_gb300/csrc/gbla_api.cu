// C-ABI front end of the GBLA core: argument validation, scratch memory and
// kernel-family dispatch.  All arithmetic happens in the kernels of
// gbla_simt.cu and gbla_tc.cu.
#include <string.h>

#include <atomic>

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

thread_local cudaError_t t_last_cuda_error = cudaSuccess;

gbla_status from_cuda(cudaError_t e) {
  if (e == cudaSuccess) return GBLA_OK;
  t_last_cuda_error = e;
  (void)cudaGetLastError();  // clear the non-sticky launch error
  return GBLA_ERR_CUDA;
}

// Stream-ordered scratch: freed on the same stream after the kernels using it.
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
    cudaError_t e = cudaMallocAsync(&ptr, bytes, s);
    if (e != cudaSuccess) {
      (void)cudaGetLastError();
      ptr = nullptr;
      return GBLA_ERR_ALLOC;
    }
    return GBLA_OK;
  }
};

size_t round_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// State (Conv1D of k, v, phi, gate, S and z) into `state`.
gbla_status run_state(const Problem &p, bool tc, const void *k, const void *v,
                      const void *gate, const float *conv_w, float *state,
                      cudaStream_t st) {
  Scratch ws;
  if (tc) {
    gbla_status s = ws.alloc(tc_workspace_bytes(p), st);
    if (s != GBLA_OK) return s;
    return from_cuda(tc_state(p, k, v, gate, conv_w, ws.ptr, state, st));
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
                        void *o, cudaStream_t st, bool after_state = false) {
  if (tc) return from_cuda(tc_readout(p, q, og, conv_w, norm_w, state, o, st, after_state));
  return from_cuda(simt_readout(p, q, og, conv_w, norm_w, state, o, st));
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

void gbla_release(void) {}

uint64_t gbla_launch_count(void) { return g_launches.load(std::memory_order_relaxed); }

uint32_t gbla_device_error(int reset) { return tc_device_error(reset != 0); }

const char *gbla_last_cuda_error(void) { return cudaGetErrorString(t_last_cuda_error); }

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
  bool empty = false;
  gbla_status s = check_dims(B, H, N, D, dtype, &empty);
  if (s != GBLA_OK || empty) return s;
  if ((s = check_ptrs({q, k, v, gate, out_gate, conv_w, norm_w, o})) != GBLA_OK) return s;
  if ((s = check_seq_lens(seq_lens)) != GBLA_OK) return s;
  const size_t bytes = (size_t)B * N * H * D * elem_bytes(dtype);
  const Range out = range_of(o, bytes);
  if (overlap(out, range_of(q, bytes)) || overlap(out, range_of(k, bytes)) ||
      overlap(out, range_of(v, bytes)) || overlap(out, range_of(out_gate, bytes)) ||
      overlap(out, range_of(gate, (size_t)B * N * H * elem_bytes(dtype))) ||
      overlap(out, range_of(conv_w, sizeof(float) * 3 * H * D * kConvW)) ||
      overlap(out, range_of(norm_w, sizeof(float) * H * D)) ||
      (seq_lens && overlap(out, range_of(seq_lens, sizeof(int32_t) * B))))
    return GBLA_ERR_INVALID_ARG;
  Problem p{B, H, N, D, dtype, seq_lens};
  bool tc = use_tc(p, algo, &s);
  if (s != GBLA_OK) return s;
  cudaStream_t st = (cudaStream_t)stream;
  Scratch state;
  if ((s = state.alloc(sizeof(float) * state_floats(D) * B * H, st)) != GBLA_OK) return s;
  if ((s = run_state(p, tc, k, v, gate, conv_w, (float *)state.ptr, st)) != GBLA_OK) return s;
  return run_readout(p, tc, q, out_gate, conv_w, norm_w, (const float *)state.ptr, o, st,
                     true);
}

gbla_status gbla_forward(const void *q, const void *k, const void *v,
                         const void *gate, const void *out_gate,
                         const float *conv_w, const float *norm_w,
                         const int32_t *seq_lens, void *o, int B, int H, int N,
                         int D, gbla_dtype dtype, gbla_stream_t stream) {
  return gbla_forward_ex(q, k, v, gate, out_gate, conv_w, norm_w, seq_lens, o, B, H,
                         N, D, dtype, GBLA_ALGO_AUTO, stream);
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
  // Layout of the device scratch: q k v og o | gate | conv_w | norm_w | seq_lens
  size_t off[10];
  size_t at = 0;
  for (int i = 0; i < 5; ++i) { off[i] = at; at = round_up(at + tens, 256); }
  off[5] = at; at = round_up(at + gbytes, 256);
  off[6] = at; at = round_up(at + cw, 256);
  off[7] = at; at = round_up(at + nw, 256);
  off[8] = at; at = round_up(at + sizeof(int32_t) * B, 256);
  Scratch dev;
  if ((s = dev.alloc(at, st)) != GBLA_OK) return s;
  char *base = (char *)dev.ptr;
  // Valid rows only: rows t >= L_b are never read by the kernels.
  const void *src[5] = {q, k, v, out_gate, nullptr};
  for (int b = 0; b < B; ++b) {
    long L = seq_lens ? seq_lens[b] : N;
    if (L < 0) L = 0;
    if (L > N) L = N;
    if (L == 0) continue;
    for (int i = 0; i < 4; ++i) {
      if (cudaMemcpyAsync(base + off[i] + (size_t)b * N * row, (const char *)src[i] + (size_t)b * N * row,
                          L * row, cudaMemcpyHostToDevice, st) != cudaSuccess)
        return GBLA_ERR_CUDA;
    }
    if (cudaMemcpyAsync(base + off[5] + (size_t)b * N * grow, (const char *)gate + (size_t)b * N * grow,
                        L * grow, cudaMemcpyHostToDevice, st) != cudaSuccess)
      return GBLA_ERR_CUDA;
  }
  if (cudaMemcpyAsync(base + off[6], conv_w, cw, cudaMemcpyHostToDevice, st) != cudaSuccess ||
      cudaMemcpyAsync(base + off[7], norm_w, nw, cudaMemcpyHostToDevice, st) != cudaSuccess)
    return GBLA_ERR_CUDA;
  const int32_t *dsl = nullptr;
  if (seq_lens) {
    if (cudaMemcpyAsync(base + off[8], seq_lens, sizeof(int32_t) * B, cudaMemcpyHostToDevice,
                        st) != cudaSuccess)
      return GBLA_ERR_CUDA;
    dsl = (const int32_t *)(base + off[8]);
  }
  s = gbla_forward(base + off[0], base + off[1], base + off[2], base + off[5], base + off[3],
                   (const float *)(base + off[6]), (const float *)(base + off[7]), dsl,
                   base + off[4], B, H, N, D, dtype, stream);
  if (s != GBLA_OK) return s;
  for (int b = 0; b < B; ++b) {
    long L = seq_lens ? seq_lens[b] : N;
    if (L < 0) L = 0;
    if (L > N) L = N;
    if (L == 0) continue;
    if (cudaMemcpyAsync((char *)o + (size_t)b * N * row, base + off[4] + (size_t)b * N * row, L * row,
                        cudaMemcpyDeviceToHost, st) != cudaSuccess)
      return GBLA_ERR_CUDA;
  }
  dev.release();
  return from_cuda(cudaStreamSynchronize(st));
}

}  // extern "C"
