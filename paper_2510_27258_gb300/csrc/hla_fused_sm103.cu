// Fused tcgen05/TMA forward of masked second-order HLA for sm_103a.
// (The generic path serves every shape until this path is enabled.)
#include "hla_internal.h"

namespace hla {

size_t fused2_workspace_bytes(int, int, int, int, int, hla_dtype) { return 0; }

bool fused2_applicable(const Fwd2 &) { return false; }

cudaError_t fused2_forward(const Fwd2 &, cudaStream_t) { return cudaErrorNotSupported; }

}  // namespace hla
