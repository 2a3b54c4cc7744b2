// Tensor-core (tcgen05 + TMA) kernels of the GBLA core for bf16.
#include "gbla_internal.cuh"

namespace gbla {

bool tc_supports(const Problem &) { return false; }
size_t tc_workspace_bytes(const Problem &) { return 0; }
cudaError_t tc_state(const Problem &, const void *, const void *, const void *,
                     const float *, void *, float *, cudaStream_t) {
  return cudaErrorNotSupported;
}
cudaError_t tc_readout(const Problem &, const void *, const void *, const float *,
                       const float *, const float *, void *, cudaStream_t) {
  return cudaErrorNotSupported;
}

}  // namespace gbla
