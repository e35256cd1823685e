// Tensor-core (tcgen05 / TMEM) attention over [composed cache; suffix]: not built yet.
#include "internal.cuh"

namespace c2kv {

bool attn_tc_supported(int, int, int, int) { return false; }

cudaError_t launch_attn_tc(const AttnParams&, cudaStream_t) { return cudaErrorNotSupported; }

}  // namespace c2kv
