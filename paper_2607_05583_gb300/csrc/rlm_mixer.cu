// rlm_mixer.cu -- the mixer wrapper of Sec. 3.4 for the prefill paths that do not
// fuse it into their epilogue:
//   z_t[d] = sigma(g_t[d]) y_t[d] + s[d] sum_{k<K} w[d][k] u_{t-k}[d]
// applied in place to a field z that already holds the mixing y, plus the update
// of the local path's drive history (the last K-1 drives of history || x).
//
// k_mixer_epilogue: one thread per (b, run of kRun tokens, d), channel fastest so a
// warp reads consecutive channels of one token row.  The thread keeps the K most
// recent drives in registers, so x is read once (plus K-1 tokens of overlap per
// run).  The pass moves 8 (bf16) or 16 (fp32) bytes per token-channel: read x, g
// and y, write z.
#include "rlm_device.cuh"
#include "rlm_internal.h"

namespace rlm {
namespace {

constexpr int kRun = 32;
constexpr int kBlock = 256;
constexpr int kMaxK = RLM_MAX_LOCAL_K;

__device__ __forceinline__ float sigmoidf(float v) { return 1.0f / (1.0f + expf(-v)); }

// Plain (coherent) load of an element this kernel also writes.
__device__ __forceinline__ float ld_rw(const float *p) { return *p; }
__device__ __forceinline__ float ld_rw(const __nv_bfloat16 *p) { return __bfloat162float(*p); }

// u_{t}[d] of the sequence preceded by its history: t < 0 reads the history
// ([B][K-1][D], oldest first) or zero.
template <typename T>
__device__ __forceinline__ float drive_at(const T *x, const T *hist, int64_t b, int64_t t, int64_t L,
                                          int D, int K, int d) {
    if (t >= 0) return ld_elem(x + (b * L + t) * D + d);
    if (!hist) return 0.0f;
    return ld_elem(hist + (b * (K - 1) + (K - 1 + t)) * D + d);
}

template <typename T>
__global__ void __launch_bounds__(kBlock) k_mixer_epilogue(const T *__restrict__ x, const T *__restrict__ g,
                                                           T *__restrict__ z, const T *__restrict__ hist,
                                                           const float *__restrict__ conv_w,
                                                           const float *__restrict__ scale, int64_t B,
                                                           int64_t L, int D, int K) {
    const int64_t nruns = (L + kRun - 1) / kRun;
    const int64_t gid = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (gid >= B * nruns * D) return;
    const int d = (int)(gid % D);
    const int64_t br = gid / D;
    const int64_t b = br / nruns, t0 = (br % nruns) * kRun;
    const int64_t t1 = t0 + kRun < L ? t0 + kRun : L;
    float w[kMaxK], win[kMaxK];  // win[k] = u_{t-k}
    float s = 0.0f;
#pragma unroll
    for (int k = 0; k < kMaxK; ++k) {
        w[k] = k < K ? __ldg(conv_w + (int64_t)d * K + k) : 0.0f;
        win[k] = 0.0f;
    }
    if (K > 0) s = __ldg(scale + d);
#pragma unroll
    for (int k = 1; k < kMaxK; ++k)
        if (k < K) win[k] = drive_at(x, hist, b, t0 - k, L, D, K, d);
    for (int64_t t = t0; t < t1; ++t) {
        const int64_t i = (b * L + t) * D + d;
        win[0] = ld_elem(x + i);
        float l = 0.0f;
#pragma unroll
        for (int k = 0; k < kMaxK; ++k) l = fmaf(w[k], win[k], l);
        const float gate = g ? sigmoidf(ld_elem(g + i)) : 1.0f;
        st_elem(z + i, fmaf(gate, ld_rw(z + i), s * l));
#pragma unroll
        for (int k = kMaxK - 1; k > 0; --k) win[k] = win[k - 1];
    }
}

// The history after the last token: entry j is element L + j of history || x.
// One thread per (b, d) reads all K-1 values before writing, so out may alias in.
template <typename T>
__global__ void __launch_bounds__(kBlock) k_conv_tail(const T *__restrict__ x, const T *hist, T *out, int64_t B,
                                                      int64_t L, int D, int K) {
    const int64_t gid = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (gid >= B * D) return;
    const int64_t b = gid / D;
    const int d = (int)(gid % D);
    T v[kMaxK];
#pragma unroll
    for (int j = 0; j < kMaxK - 1; ++j) {
        if (j >= K - 1) break;
        const int64_t e = L + j;  // index into history || x
        if (e >= K - 1)
            v[j] = x[(b * L + (e - (K - 1))) * D + d];
        else
            v[j] = hist ? hist[(b * (K - 1) + e) * D + d] : T(0.0f);
    }
#pragma unroll
    for (int j = 0; j < kMaxK - 1; ++j) {
        if (j >= K - 1) break;
        out[(b * (K - 1) + j) * D + d] = v[j];
    }
}

template <typename T>
cudaError_t epilogue_t(const void *x, const void *g, void *z, const void *hist, const float *conv_w,
                       const float *scale, int64_t B, int64_t L, int D, int K, cudaStream_t st) {
    const int64_t n = B * ((L + kRun - 1) / kRun) * D;
    k_mixer_epilogue<T><<<(unsigned)((n + kBlock - 1) / kBlock), kBlock, 0, st>>>(
        static_cast<const T *>(x), static_cast<const T *>(g), static_cast<T *>(z), static_cast<const T *>(hist),
        conv_w, scale, B, L, D, K);
    count_launches(1);
    return cudaGetLastError();
}

template <typename T>
cudaError_t tail_t(const void *x, const void *hist, void *out, int64_t B, int64_t L, int D, int K,
                   cudaStream_t st) {
    const int64_t n = B * D;
    k_conv_tail<T><<<(unsigned)((n + kBlock - 1) / kBlock), kBlock, 0, st>>>(
        static_cast<const T *>(x), static_cast<const T *>(hist), static_cast<T *>(out), B, L, D, K);
    count_launches(1);
    return cudaGetLastError();
}

}  // namespace

cudaError_t mixer_epilogue(const void *x, const void *g, void *z, const void *hist, const float *conv_w,
                           const float *scale, rlm_dtype dt, int64_t B, int64_t L, int D, int K,
                           cudaStream_t st) {
    if (dt == RLM_BF16) return epilogue_t<__nv_bfloat16>(x, g, z, hist, conv_w, scale, B, L, D, K, st);
    return epilogue_t<float>(x, g, z, hist, conv_w, scale, B, L, D, K, st);
}

cudaError_t conv_tail(const void *x, const void *hist, void *out, rlm_dtype dt, int64_t B, int64_t L, int D,
                      int K, cudaStream_t st) {
    if (K < 2) return cudaSuccess;
    if (dt == RLM_BF16) return tail_t<__nv_bfloat16>(x, hist, out, B, L, D, K, st);
    return tail_t<float>(x, hist, out, B, L, D, K, st);
}

}  // namespace rlm
