// rlm_mixer.cuh -- device helpers of the mixer wrapper (Sec. 3.4) shared by its
// kernels.
#pragma once

#include <cuda_runtime.h>

namespace rlm {

// The gate sigma(v) = 1 / (1 + e^-v).
__device__ __forceinline__ float gatef(float v) { return __fdividef(1.0f, 1.0f + __expf(-v)); }

// Head coupling: C = I + (lambda_c / sqrt(H)) tanh(c_raw), H x H row-major, built
// by the calling block's threads (the caller synchronises before reading it).
__device__ __forceinline__ void build_coupling(float *C, const float *c_raw, float lam, int H) {
    const float k = lam * rsqrtf((float)H);
    for (int i = threadIdx.x; i < H * H; i += blockDim.x)
        C[i] = (i / H == i % H ? 1.0f : 0.0f) + k * tanhf(__ldg(c_raw + i));
}

}  // namespace rlm
