// gla_tc.cu -- tensor-core chunkwise schedule (placeholder until the tcgen05
// kernel lands) and the device status word.
#include "gla_internal.h"

namespace gtr {

__device__ unsigned int g_device_status;

bool tc_supported(const Problem &) { return false; }

cudaError_t launch_tc(const Problem &, cudaStream_t) { return cudaErrorNotSupported; }

cudaError_t read_and_clear_device_status(unsigned int *status) {
    cudaError_t e = cudaMemcpyFromSymbol(status, g_device_status, sizeof(unsigned int));
    if (e != cudaSuccess) return e;
    const unsigned int zero = 0;
    return cudaMemcpyToSymbol(g_device_status, &zero, sizeof(unsigned int));
}

}  // namespace gtr
