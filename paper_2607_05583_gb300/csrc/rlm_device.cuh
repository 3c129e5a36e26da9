// rlm_device.cuh -- small device helpers shared by the CUDA translation units.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace rlm {

template <typename T>
__device__ __forceinline__ float ld_elem(const T *p);
template <>
__device__ __forceinline__ float ld_elem<float>(const float *p) { return __ldg(p); }
template <>
__device__ __forceinline__ float ld_elem<__nv_bfloat16>(const __nv_bfloat16 *p) {
    return __bfloat162float(__ldg(p));
}

template <typename T>
__device__ __forceinline__ void st_elem(T *p, float v);
template <>
__device__ __forceinline__ void st_elem<float>(float *p, float v) { *p = v; }
template <>
__device__ __forceinline__ void st_elem<__nv_bfloat16>(__nv_bfloat16 *p, float v) {
    *p = __float2bfloat16_rn(v);
}

// Complex helpers on float2 (x = Re, y = Im).
__device__ __forceinline__ float2 cmul(float2 a, float2 b) {
    return make_float2(fmaf(a.x, b.x, -a.y * b.y), fmaf(a.x, b.y, a.y * b.x));
}
__device__ __forceinline__ float2 conj2(float2 a) { return make_float2(a.x, -a.y); }
// a*b + c
__device__ __forceinline__ float2 cfma(float2 a, float2 b, float2 c) {
    return make_float2(fmaf(a.x, b.x, fmaf(-a.y, b.y, c.x)), fmaf(a.x, b.y, fmaf(a.y, b.x, c.y)));
}

// lambda^n = exp(-gamma n) (cos(omega n) + i sin(omega n)) in fp32.  The
// products gamma*n and omega*n are formed with their exact FMA residuals, so
// the phase keeps full accuracy for large n (a plain fp32 omega*n is off by up
// to |omega n| * 2^-24 rad).  n must be an integer below 2^24.
__device__ __forceinline__ float2 lambda_pow(float gamma, float omega, float n) {
    float p = omega * n;
    float pe = fmaf(omega, n, -p);
    float sp, cp;
    sincosf(p, &sp, &cp);
    float q = gamma * n;
    float qe = fmaf(gamma, n, -q);
    float r = expf(-q) * (1.0f - qe);
    return make_float2(r * fmaf(-pe, sp, cp), r * fmaf(pe, cp, sp));
}

// c = A exp(i phi).
__device__ __forceinline__ float2 mode_coef(float amp, float phase) {
    float s, c;
    sincosf(phase, &s, &c);
    return make_float2(amp * c, amp * s);
}

}  // namespace rlm
