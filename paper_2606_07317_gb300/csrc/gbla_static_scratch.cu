// gbla_state_static_scratch: the state step (Conv1D of k and v, phi, key gate,
// S and z) for callers that must not allocate GPU memory.
//
// Who needs it: a caller whose device memory is already entirely owned by
// another allocator (a serving process that reserved the whole GPU at start-up,
// a framework pool it cannot reach from C), or a latency-critical loop that
// cannot afford the implicit synchronisation and unpredictable latency of an
// allocation call.  gbla_state takes its partial-sum scratch from the stream
// pool; this entry point takes it from a fixed array compiled into the library
// instead, and performs no allocation of any kind.
//
// The scratch is a file-scope __device__ array of GBLA_STATIC_SCRATCH_BYTES.
// Every GPU on which this library's code is loaded holds that memory until the
// process exits.  Host code cannot use the array's name as a device address
// (on the host it names a host-side stand-in), so the device address is looked
// up once per device with cudaGetSymbolAddress, with that device current, the
// first time this entry point runs on it; that first call should therefore be
// made before any stream capture begins.  The address is kept for the life of
// the process: after cudaDeviceReset (or any other teardown of the device's
// primary context) the entry point must not be called again on that device.
//
// All calls share the one array and it keeps whatever the last call left in
// it.  Nothing has to start at zero: each call writes every partial record its
// own reduction reads (empty chunks included) before reading it.  Calls that
// overlap on the GPU (different streams, or different host threads) race on
// the array and produce garbage; serialise them.
#include <mutex>

#include "gbla_internal.cuh"

namespace gbla {
namespace {

constexpr size_t kScratchFloats = (size_t)GBLA_STATIC_SCRATCH_BYTES / sizeof(float);

static __device__ __align__(256) float g_static_scratch[kScratchFloats];

constexpr int kMaxDevices = 128;
std::mutex g_scratch_mu;
void *g_scratch_addr[kMaxDevices];  // device address per device ordinal, set once

// Device address of g_static_scratch on the current device (set up on first use).
cudaError_t static_scratch_address(void **out) {
  int dev = -1;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lock(g_scratch_mu);
  if (g_scratch_addr[dev] == nullptr) {
    void *p = nullptr;
    e = cudaGetSymbolAddress(&p, g_static_scratch);
    if (e != cudaSuccess) return e;
    g_scratch_addr[dev] = p;
  }
  *out = g_scratch_addr[dev];
  return cudaSuccess;
}

bool overlaps(const void *a, size_t na, const void *b, size_t nb) {
  const uintptr_t a0 = (uintptr_t)a, b0 = (uintptr_t)b;
  return a0 < b0 + nb && b0 < a0 + na;
}

}  // namespace
}  // namespace gbla

extern "C" gbla_status gbla_state_static_scratch(
    const void *k, const void *v, const void *gate, const float *conv_w,
    const int32_t *seq_lens, float *state, int B, int H, int N, int D,
    gbla_dtype dtype, gbla_stream_t stream) {
  using namespace gbla;
  // the same argument rules as gbla_state
  bool empty = false;
  gbla_status s = check_dims(B, H, N, D, dtype, &empty);
  if (s != GBLA_OK || empty) return s;
  if ((s = check_ptrs({k, v, gate, conv_w, state})) != GBLA_OK) return s;
  if ((s = check_seq_lens(seq_lens)) != GBLA_OK) return s;
  const size_t es = dtype == GBLA_FP32 ? 4 : 2;
  const size_t in_bytes = (size_t)B * N * H * D * es;
  const size_t st_bytes = sizeof(float) * state_floats(D) * B * H;
  if (overlaps(state, st_bytes, k, in_bytes) || overlaps(state, st_bytes, v, in_bytes) ||
      overlaps(state, st_bytes, gate, (size_t)B * N * H * es) ||
      overlaps(state, st_bytes, conv_w, sizeof(float) * 3 * H * D * kConvW))
    return GBLA_ERR_INVALID_ARG;

  // Fit the chunk plan into the fixed array: one partial record per
  // (b, h, chunk).  If even one chunk per (b, h) does not fit, refuse.
  Problem p{B, H, N, D, dtype, seq_lens};
  const size_t per_chunk = partial_floats(D) * (size_t)B * H;
  if (per_chunk > kScratchFloats) return GBLA_ERR_INVALID_ARG;
  SimtPlan plan = simt_plan(p);
  const size_t max_chunks = kScratchFloats / per_chunk;
  if ((size_t)plan.n_chunks > max_chunks) {
    int len = (int)((N + max_chunks - 1) / max_chunks);
    len = (len + 31) / 32 * 32;
    plan.chunk_len = len;
    plan.n_chunks = (N + len - 1) / len;
  }

  void *scratch = nullptr;
  if ((s = from_cuda(static_scratch_address(&scratch))) != GBLA_OK) return s;
  return from_cuda(simt_state(p, plan, k, v, gate, conv_w, (float *)scratch, state,
                              (cudaStream_t)stream));
}
