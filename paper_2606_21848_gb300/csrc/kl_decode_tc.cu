// Tensor-core (tcgen05 + TMA) decode kernel -- placeholder until the kernel lands.
#include "kl_internal.cuh"

namespace kl {

bool tc_supported(const Geometry &, bool) { return false; }

cudaError_t launch_decode_tc(const DecodeArgs &, bool) { return cudaErrorNotSupported; }

}  // namespace kl
