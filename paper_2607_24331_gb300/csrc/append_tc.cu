// Tensor-core (tcgen05) latent append: placeholder until the kernel lands.
#include "common.cuh"

namespace dck {
bool tc_append_supports(int, int, int, int) { return false; }
size_t tc_append_workspace(int, int, int) { return 0; }
cudaError_t launch_append_tc(const void*, int, int, const void*, const void*, int, int, const int64_t*, void*, void*,
                             int64_t, void*, size_t, int*, cudaStream_t) {
  return cudaErrorNotSupported;
}
}  // namespace dck
