// rlm_prefill_tc.cu -- tcgen05 tensor-core prefill (bf16 I/O).
#include "rlm_device.cuh"
#include "rlm_internal.h"

namespace rlm {

// Device status word: RLM_OK, or RLM_ERR_TIMEOUT once a bounded wait expired.
__device__ int g_device_status = 0;

bool tc_prefill_supported(int64_t, int64_t, int, int, rlm_dtype) { return false; }

size_t tc_prefill_ws_bytes(int64_t, int64_t, int, int) { return 0; }

cudaError_t tc_prefill(const void *, void *, int64_t, int64_t, int, int, const float *,
                       const float *, const float *, const float *, float *, float *, void *,
                       cudaStream_t) {
    return cudaErrorNotSupported;
}

cudaError_t read_and_clear_device_status(int *status, cudaStream_t st) {
    cudaError_t e = cudaMemcpyFromSymbolAsync(status, g_device_status, sizeof(int), 0,
                                              cudaMemcpyDeviceToHost, st);
    if (e != cudaSuccess) return e;
    if ((e = cudaStreamSynchronize(st)) != cudaSuccess) return e;
    const int zero = 0;
    if ((e = cudaMemcpyToSymbolAsync(g_device_status, &zero, sizeof(int), 0,
                                     cudaMemcpyHostToDevice, st)) != cudaSuccess)
        return e;
    return cudaStreamSynchronize(st);
}

}  // namespace rlm
