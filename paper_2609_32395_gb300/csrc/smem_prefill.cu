// smem_prefill.cu -- one-block reader pass (placeholder until the tensor-core
// kernel lands).
#include <cuda_runtime.h>

#include "smem_internal.h"

namespace smem {
cudaError_t launch_prefill(const PrefillArgs&, cudaStream_t) { return cudaErrorNotSupported; }
}  // namespace smem
