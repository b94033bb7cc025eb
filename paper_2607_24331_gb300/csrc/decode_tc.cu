// Tensor-core (tcgen05) decode attention: placeholder until the kernel lands.
#include "common.cuh"

namespace dck {
bool tc_decode_supports(const LayerTable&, int) { return false; }
cudaError_t launch_decode_tc(const LayerTable&, const DecodeArgs&, cudaStream_t) { return cudaErrorNotSupported; }
}  // namespace dck
