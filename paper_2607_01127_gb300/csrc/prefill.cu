// Prefill GEMM (tcgen05) -- placeholder until the tensor-core kernel lands.
#include "internal.h"

namespace logq {
cudaError_t launch_prefill(const LinearArgs&, cudaStream_t) { return cudaErrorNotSupported; }
}  // namespace logq
