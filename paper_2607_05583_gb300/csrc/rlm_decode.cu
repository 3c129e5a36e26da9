// rlm_decode.cu -- one autoregressive step of Sec. 3.3 (Eq. 4-5), fused:
//   s_bdm <- lambda_dm s_bdm + x_t[b,d];   y_t[b,d] = sum_m Re(c_dm s_bdm)
//
// The step is bound by moving the state (16 bytes per (b, d, m): read and
// write one complex fp32) plus the token and coefficient reads.  Each thread
// owns MPT consecutive modes of one (b, d) -- one 16-byte state load and
// store, and one 16-byte coefficient load per mode -- so a warp touches
// contiguous state.  The TPG threads of a (b, d) add their partial readouts
// with xor-shuffles.
//
// The mixer step (Sec. 3.4, kMix) runs in the same kernel: the thread that writes
// y_t[b,d] also applies the gate sigma(g_t), adds s * sum_k w[k] u_{t-k} over the
// cached drives, and shifts the drive history by one token.  Its loads are issued
// before the state update, so they add no round trip to the step.
//
// Launch: programmatic dependent launch.  The kernel waits on the previous
// grid (griddepcontrol.wait) before touching memory and lets the next step's
// grid be scheduled right after, which hides most of the per-step launch
// latency when decode steps are issued back to back or captured in a graph.
#include "rlm_device.cuh"
#include "rlm_internal.h"

namespace rlm {
namespace {

constexpr int kDecodeBlock = 256;
constexpr int kMaxK = RLM_MAX_LOCAL_K;

// The mixer's per-step inputs (null g: no gate; K = 0: no local path).
template <typename T>
struct MixStep {
    const T *g;          // [B][D]
    T *hist;             // [B][K-1][D], oldest first
    const float *conv_w; // [D][K]
    const float *scale;  // [D]
    int K;
};

// Plain (coherent) load of the drive history, which every step rewrites.
__device__ __forceinline__ float ld_hist(const float *p) { return *p; }
__device__ __forceinline__ float ld_hist(const __nv_bfloat16 *p) { return __bfloat162float(*p); }

// Loads of the mixer step, taken before the state update.
struct MixLoads {
    float gate, s, l;   // l: the local path without the current token
    float w0;
};

template <typename T>
__device__ __forceinline__ MixLoads mix_load(const MixStep<T> &m, int64_t bd, int D) {
    MixLoads r{1.0f, 0.0f, 0.0f, 0.0f};
    if (m.g) r.gate = ld_elem(m.g + bd);
    if (m.K > 0) {
        const int d = (int)(bd % D);
        const int64_t b = bd / D;
        r.s = __ldg(m.scale + d);
        r.w0 = __ldg(m.conv_w + (int64_t)d * m.K);
        const T *h = m.hist + b * (m.K - 1) * (int64_t)D + d;
#pragma unroll
        for (int k = 1; k < kMaxK; ++k)
            if (k < m.K) r.l = fmaf(__ldg(m.conv_w + (int64_t)d * m.K + k), ld_hist(h + (int64_t)(m.K - 1 - k) * D), r.l);
    }
    return r;
}

// z = sigma(g) y + s (w0 x + l); shifts the history and appends x.
template <typename T>
__device__ __forceinline__ float mix_finish(const MixStep<T> &m, const MixLoads &r, int64_t bd, int D, float y,
                                            const T *x_t) {
    const float gate = m.g ? 1.0f / (1.0f + expf(-r.gate)) : 1.0f;
    if (m.K == 0) return gate * y;
    const float xv = ld_elem(x_t + bd);
    if (m.K > 1) {
        const int64_t b = bd / D;
        T *h = m.hist + b * (m.K - 1) * (int64_t)D + (bd % D);
        T v[kMaxK];
#pragma unroll
        for (int j = 1; j < kMaxK - 1; ++j)
            if (j < m.K - 1) v[j] = h[(int64_t)j * D];
#pragma unroll
        for (int j = 1; j < kMaxK - 1; ++j)
            if (j < m.K - 1) h[(int64_t)(j - 1) * D] = v[j];
        h[(int64_t)(m.K - 2) * D] = x_t[bd];
    }
    return fmaf(gate, y, r.s * fmaf(r.w0, xv, r.l));
}

__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_launch_dependents() {
    asm volatile("griddepcontrol.launch_dependents;" :::);
}

// MPT = 2 with M even: state and coefficients move as 16-byte vectors.
template <typename T, bool kMix>
__global__ void __launch_bounds__(kDecodeBlock) k_decode_vec2(
    const T *__restrict__ x_t, T *__restrict__ y_t, int64_t BD, int D, int M, int log2_tpg,
    float4 *__restrict__ s, const float4 *__restrict__ coef, MixStep<T> mix) {
    pdl_wait();
    pdl_launch_dependents();
    const int64_t gid = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const int64_t bd = gid >> log2_tpg;
    const int g = (int)(gid & ((1 << log2_tpg) - 1));
    const int tpg = 1 << log2_tpg;
    const bool valid = bd < BD && 2 * g < M;
    MixLoads ml{};
    if (kMix && valid && g == 0) ml = mix_load(mix, bd, D);
    float acc = 0.0f;
    if (valid) {
        const int d = (int)(bd % D);
        const float xv = ld_elem(x_t + bd);
        const int64_t si = (bd * M) / 2 + g;  // pair index (M even)
        float4 st = s[si];
        const float4 c0 = __ldg(coef + d * M + 2 * g);
        const float4 c1 = __ldg(coef + d * M + 2 * g + 1);
        const float r0 = fmaf(c0.x, st.x, fmaf(-c0.y, st.y, xv));
        const float i0 = fmaf(c0.x, st.y, c0.y * st.x);
        const float r1 = fmaf(c1.x, st.z, fmaf(-c1.y, st.w, xv));
        const float i1 = fmaf(c1.x, st.w, c1.y * st.z);
        s[si] = make_float4(r0, i0, r1, i1);
        acc = fmaf(c0.z, r0, fmaf(-c0.w, i0, fmaf(c1.z, r1, -c1.w * i1)));
    }
    for (int o = tpg >> 1; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
    if (valid && g == 0) {
        if (kMix) acc = mix_finish(mix, ml, bd, D, acc, x_t);
        st_elem(y_t + bd, acc);
    }
}

// Any M: each thread owns up to MPT modes, accessed as float2.
template <typename T, bool kMix>
__global__ void __launch_bounds__(kDecodeBlock) k_decode_any(
    const T *__restrict__ x_t, T *__restrict__ y_t, int64_t BD, int D, int M, int log2_tpg,
    int mpt, float2 *__restrict__ s, const float4 *__restrict__ coef, MixStep<T> mix) {
    pdl_wait();
    pdl_launch_dependents();
    const int64_t gid = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const int64_t bd = gid >> log2_tpg;
    const int g = (int)(gid & ((1 << log2_tpg) - 1));
    const int tpg = 1 << log2_tpg;
    MixLoads ml{};
    if (kMix && bd < BD && g == 0) ml = mix_load(mix, bd, D);
    float acc = 0.0f;
    if (bd < BD) {
        const int d = (int)(bd % D);
        const float xv = ld_elem(x_t + bd);
        for (int j = 0; j < mpt; ++j) {
            const int m = g * mpt + j;
            if (m >= M) break;
            const float4 cf = __ldg(coef + d * M + m);
            const float2 st = s[bd * M + m];
            const float re = fmaf(cf.x, st.x, fmaf(-cf.y, st.y, xv));
            const float im = fmaf(cf.x, st.y, cf.y * st.x);
            s[bd * M + m] = make_float2(re, im);
            acc = fmaf(cf.z, re, fmaf(-cf.w, im, acc));
        }
    }
    for (int o = tpg >> 1; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
    if (bd < BD && g == 0) {
        if (kMix) acc = mix_finish(mix, ml, bd, D, acc, x_t);
        st_elem(y_t + bd, acc);
    }
}

__global__ void k_state_init(float2 *__restrict__ s, float4 *__restrict__ coef, int64_t BDM,
                             int DM, const float *__restrict__ decay,
                             const float *__restrict__ freq, const float *__restrict__ amp,
                             const float *__restrict__ phase) {
    const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (i < BDM) s[i] = make_float2(0.0f, 0.0f);
    if (i < DM) {
        const float2 lam = lambda_pow(decay[i], freq[i], 1.0f);
        const float2 c = mode_coef(amp[i], phase[i]);
        coef[i] = make_float4(lam.x, lam.y, c.x, c.y);
    }
}

template <typename Kern, typename... Args>
cudaError_t launch_pdl(Kern kern, unsigned grid, cudaStream_t st, Args... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(kDecodeBlock);
    cfg.dynamicSmemBytes = 0;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    count_launches(1);
    return cudaLaunchKernelEx(&cfg, kern, args...);
}

template <typename T, bool kMix>
cudaError_t decode_t(const T *x_t, T *y_t, int B, int D, int M, float *s, const float *coef,
                     MixStep<T> mix, cudaStream_t st) {
    int pairs = (M + 1) / 2;
    int log2_tpg = 0;
    while ((1 << log2_tpg) < pairs && log2_tpg < 5) ++log2_tpg;
    const int tpg = 1 << log2_tpg;
    const int64_t BD = (int64_t)B * D;
    const int64_t threads = BD * tpg;
    const unsigned grid = (unsigned)((threads + kDecodeBlock - 1) / kDecodeBlock);
    const float4 *cf = reinterpret_cast<const float4 *>(coef);
    if (M % 2 == 0 && 2 * tpg >= M)
        return launch_pdl(k_decode_vec2<T, kMix>, grid, st, x_t, y_t, BD, D, M, log2_tpg,
                          reinterpret_cast<float4 *>(s), cf, mix);
    const int mpt = (M + tpg - 1) / tpg;
    return launch_pdl(k_decode_any<T, kMix>, grid, st, x_t, y_t, BD, D, M, log2_tpg, mpt,
                      reinterpret_cast<float2 *>(s), cf, mix);
}

}  // namespace

cudaError_t decode_step(const void *x_t, void *y_t, rlm_dtype dt, int B, int D, int M, float *s,
                        const float *coef, cudaStream_t st) {
    if (dt == RLM_BF16)
        return decode_t<__nv_bfloat16, false>(static_cast<const __nv_bfloat16 *>(x_t),
                                              static_cast<__nv_bfloat16 *>(y_t), B, D, M, s, coef, {}, st);
    return decode_t<float, false>(static_cast<const float *>(x_t), static_cast<float *>(y_t), B, D, M, s, coef,
                                  {}, st);
}

cudaError_t mixer_decode_step(const void *x_t, const void *g_t, void *z_t, rlm_dtype dt, int B, int D, int M,
                              float *s, const float *coef, void *hist, const float *conv_w, const float *scale,
                              int K, cudaStream_t st) {
    if (dt == RLM_BF16) {
        using T = __nv_bfloat16;
        const MixStep<T> m{static_cast<const T *>(g_t), static_cast<T *>(hist), conv_w, scale, K};
        return decode_t<T, true>(static_cast<const T *>(x_t), static_cast<T *>(z_t), B, D, M, s, coef, m, st);
    }
    const MixStep<float> m{static_cast<const float *>(g_t), static_cast<float *>(hist), conv_w, scale, K};
    return decode_t<float, true>(static_cast<const float *>(x_t), static_cast<float *>(z_t), B, D, M, s, coef, m,
                                 st);
}

cudaError_t state_init(float *s, float *coef, int B, int D, int M, const float *decay,
                       const float *freq, const float *amp, const float *phase, cudaStream_t st) {
    const int64_t BDM = (int64_t)B * D * M;
    const int64_t n = BDM > (int64_t)D * M ? BDM : (int64_t)D * M;
    k_state_init<<<(unsigned)((n + 255) / 256), 256, 0, st>>>(
        reinterpret_cast<float2 *>(s), reinterpret_cast<float4 *>(coef), BDM, D * M, decay, freq,
        amp, phase);
    count_launches(1);
    return cudaGetLastError();
}

}  // namespace rlm
