// rlm_mixer.cu -- the mixer wrapper of Sec. 3.4 for the prefill paths that do not
// fuse it into their epilogue:
//   z_t[d] = sigma(g_t[d]) y_t[d] + s[d] sum_{k<K} w[d][k] u_{t-k}[d]
// applied in place to a field z that already holds the mixing y, plus the update
// of the local path's drive history (the last K-1 drives of history || x).
//
// k_mixer_epilogue: a block finishes a tile of kTT tokens x kTC channels.  It first
// stages the tile's drive rows, with the K - 1 rows before it (from x or the
// history), in shared memory with 16-byte loads; then each thread takes a channel
// pair for kTT / 4 tokens, reads its taps from shared memory (a warp reads 128
// contiguous bytes per row: no bank conflicts) and the gate and y from global
// memory, and writes z.  The kernel size K is a template parameter (2 K weights per
// thread in registers).  The pass moves 8 (bf16) or 16 (fp32) bytes per
// token-channel: read x, g and y, write z.
#include <algorithm>

#include "rlm_device.cuh"
#include "rlm_internal.h"
#include "rlm_mixer.cuh"

namespace rlm {
namespace {

constexpr int kBlock = 256;
constexpr int kMaxK = RLM_MAX_LOCAL_K;
constexpr int kTT = 64;    // tokens per tile
constexpr int kTC = 128;   // channels per tile (a multiple of 8 channels is staged)
constexpr int kEB = 256;   // threads per block of the mixer pass

// Two consecutive channels as floats, and back.
__device__ __forceinline__ float2 ld2(const float *p) { return *reinterpret_cast<const float2 *>(p); }
__device__ __forceinline__ float2 ld2(const __nv_bfloat16 *p) {
    const uint32_t v = *reinterpret_cast<const uint32_t *>(p);
    return make_float2(__uint_as_float(v << 16), __uint_as_float(v & 0xFFFF0000u));
}
__device__ __forceinline__ void st2(float *p, float2 v) { *reinterpret_cast<float2 *>(p) = v; }
__device__ __forceinline__ void st2(__nv_bfloat16 *p, float2 v) {
    uint32_t a;
    asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(a) : "f"(v.y), "f"(v.x));
    *reinterpret_cast<uint32_t *>(p) = a;
}

// Two consecutive channels as loaded (4 bytes of bf16 or 8 bytes of fp32).
template <typename T> struct Raw2;
template <> struct Raw2<float> { using type = float2; };
template <> struct Raw2<__nv_bfloat16> { using type = uint32_t; };
__device__ __forceinline__ float2 ld_raw2(const float *p) { return *reinterpret_cast<const float2 *>(p); }
__device__ __forceinline__ uint32_t ld_raw2(const __nv_bfloat16 *p) { return *reinterpret_cast<const uint32_t *>(p); }
__device__ __forceinline__ float2 raw_f2(float2 v) { return v; }
__device__ __forceinline__ float2 raw_f2(uint32_t v) {
    return make_float2(__uint_as_float(v << 16), __uint_as_float(v & 0xFFFF0000u));
}

template <typename T, int K>
__global__ void __launch_bounds__(kEB) k_mixer_epilogue(const T *__restrict__ x, const T *__restrict__ g,
                                                           T *__restrict__ z, const T *__restrict__ hist,
                                                           const float *__restrict__ conv_w,
                                                           const float *__restrict__ scale, int64_t L, int D) {
    constexpr int kRows = kTT + (K > 1 ? K - 1 : 0);
    constexpr int kVE = 16 / sizeof(T);                // elements per 16-byte vector
    constexpr int kPer = kTT / (kEB / (kTC / 2));      // tokens per thread
    __shared__ __align__(16) T xs[K > 0 ? kRows * kTC : 1];
    const int c0 = blockIdx.x * kTC;
    const int64_t t0 = (int64_t)blockIdx.y * kTT;
    const int64_t b = blockIdx.z;
    const int nc = min(kTC, D - c0);                   // a multiple of 8
    const int tid = threadIdx.x;
    const int cp = tid % (kTC / 2), tg = tid / (kTC / 2);
    const int c = 2 * cp;
    const bool active = c < nc;
    // This thread's y and gate for all its tokens, requested before the drive
    // tile is staged, so the block waits on memory once.
    typename Raw2<T>::type zr[kPer], gr[kPer];
#pragma unroll
    for (int tt = 0; tt < kPer; ++tt) {
        const int64_t t = t0 + tg * kPer + tt;
        if (active && t < L) {
            const int64_t i = (b * L + t) * D + c0 + c;
            zr[tt] = ld_raw2(z + i);
            if (g) gr[tt] = ld_raw2(g + i);
        }
    }
    if (K > 0) {
        const int vpr = nc / kVE;
        for (int i = tid; i < kRows * vpr; i += kEB) {
            const int r = i / vpr, v = i % vpr;
            const int64_t t = t0 - (K > 1 ? K - 1 : 0) + r;
            uint4 val = make_uint4(0u, 0u, 0u, 0u);
            if (t >= 0 && t < L)
                val = *reinterpret_cast<const uint4 *>(x + (b * L + t) * D + c0 + v * kVE);
            else if (t < 0 && hist)
                val = *reinterpret_cast<const uint4 *>(hist + (b * (K - 1) + (K - 1 + t)) * D + c0 + v * kVE);
            *reinterpret_cast<uint4 *>(xs + r * kTC + v * kVE) = val;
        }
        __syncthreads();
    }
    if (!active) return;
    float w0[K > 0 ? K : 1], w1[K > 0 ? K : 1];
    float s0 = 0.0f, s1 = 0.0f;
#pragma unroll
    for (int k = 0; k < K; ++k) {
        w0[k] = __ldg(conv_w + (int64_t)(c0 + c) * K + k);
        w1[k] = __ldg(conv_w + (int64_t)(c0 + c + 1) * K + k);
    }
    if (K > 0) {
        s0 = __ldg(scale + c0 + c);
        s1 = __ldg(scale + c0 + c + 1);
    }
#pragma unroll
    for (int tt = 0; tt < kPer; ++tt) {
        const int r = tg * kPer + tt;                   // token t0 + r
        const int64_t t = t0 + r;
        if (t >= L) break;
        float2 o = raw_f2(zr[tt]);
        if (g) {
            const float2 gv = raw_f2(gr[tt]);
            o = make_float2(o.x * gatef(gv.x), o.y * gatef(gv.y));
        }
        if (K > 0) {
            float l0 = 0.0f, l1 = 0.0f;
#pragma unroll
            for (int k = 0; k < K; ++k) {
                const float2 v = ld2(xs + (r + (K > 1 ? K - 1 : 0) - k) * kTC + c);
                l0 = fmaf(w0[k], v.x, l0);
                l1 = fmaf(w1[k], v.y, l1);
            }
            o = make_float2(fmaf(s0, l0, o.x), fmaf(s1, l1, o.y));
        }
        st2(z + (b * L + t) * D + c0 + c, o);
    }
}

__device__ __forceinline__ float as_f(float v) { return v; }
__device__ __forceinline__ float as_f(__nv_bfloat16 v) { return __bfloat162float(v); }

// k_couple: ybar = C y in place over z.  A block stages `rows` whole token rows of
// one batch row (16-byte loads) and writes them back coupled; a warp covers
// consecutive channels of one head, so its reads of each source head are
// contiguous in shared memory.
template <typename T>
__global__ void __launch_bounds__(kBlock) k_couple(T *z, const float *__restrict__ c_raw, float lam, int H,
                                                   int64_t L, int D, int rows) {
    extern __shared__ __align__(16) uint8_t sm[];
    float *C = reinterpret_cast<float *>(sm);
    T *ys = reinterpret_cast<T *>(sm + ((H * H * 4 + 15) & ~15));
    const int64_t b = blockIdx.y, t0 = (int64_t)blockIdx.x * rows;
    const int n = (int)(L - t0 < rows ? L - t0 : rows);
    T *zb = z + (b * L + t0) * D;
    build_coupling(C, c_raw, lam, H);
    constexpr int kVE = 16 / sizeof(T);
    for (int i = threadIdx.x; i < n * D / kVE; i += kBlock)
        reinterpret_cast<uint4 *>(ys)[i] = reinterpret_cast<const uint4 *>(zb)[i];
    __syncthreads();
    const int dh = D / H;
    for (int i = threadIdx.x; i < n * D; i += kBlock) {
        const int t = i / D, d = i % D, gh = d / dh, j = d % dh;
        const T *row = ys + (int64_t)t * D + j;
        const float *Cg = C + gh * H;
        float acc = 0.0f;
        for (int h = 0; h < H; ++h) acc = fmaf(Cg[h], as_f(row[h * dh]), acc);
        st_elem(zb + i, acc);
    }
}

// k_couple_small: the same for H <= 16 heads without staging: a thread owns kV
// consecutive in-head positions j of one token, loads its H head vectors (a warp
// reads consecutive j, so each head's load is contiguous), forms all H outputs
// with C from shared memory (broadcast reads) and writes them.
constexpr int kSmallH = 16;

template <typename T, int kV> struct VecIO;
template <typename T> struct VecIO<T, 1> {
    __device__ static void load(const T *p, float (&v)[1]) { v[0] = as_f(*p); }
    __device__ static void store(T *p, const float (&v)[1]) { st_elem(p, v[0]); }
};
template <> struct VecIO<__nv_bfloat16, 4> {
    __device__ static void load(const __nv_bfloat16 *p, float (&v)[4]) {
        const uint2 u = *reinterpret_cast<const uint2 *>(p);
        v[0] = __uint_as_float(u.x << 16); v[1] = __uint_as_float(u.x & 0xFFFF0000u);
        v[2] = __uint_as_float(u.y << 16); v[3] = __uint_as_float(u.y & 0xFFFF0000u);
    }
    __device__ static void store(__nv_bfloat16 *p, const float (&v)[4]) {
        uint32_t a, b;
        asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(a) : "f"(v[1]), "f"(v[0]));
        asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(b) : "f"(v[3]), "f"(v[2]));
        *reinterpret_cast<uint2 *>(p) = make_uint2(a, b);
    }
};
template <> struct VecIO<float, 4> {
    __device__ static void load(const float *p, float (&v)[4]) {
        const float4 u = *reinterpret_cast<const float4 *>(p);
        v[0] = u.x; v[1] = u.y; v[2] = u.z; v[3] = u.w;
    }
    __device__ static void store(float *p, const float (&v)[4]) {
        *reinterpret_cast<float4 *>(p) = make_float4(v[0], v[1], v[2], v[3]);
    }
};

// kHc = H when it is a compile-time 2, 4, 8 or 16 (loops unrolled, C rows read as
// 16-byte vectors); 0 for any other H <= 16.
template <typename T, int kV, int kHc>
__global__ void __launch_bounds__(kBlock) k_couple_small(T *z, const float *__restrict__ c_raw, float lam, int H_rt,
                                                         int64_t rows, int D) {
    __shared__ __align__(16) float C[kSmallH * kSmallH];
    const int H = kHc ? kHc : H_rt;
    build_coupling(C, c_raw, lam, H);
    __syncthreads();
    const int dh = D / H, nj = dh / kV;
    const int64_t i = (int64_t)blockIdx.x * kBlock + threadIdx.x;
    if (i >= rows * nj) return;
    const int64_t r = i / nj;
    const int j = (int)(i % nj) * kV;
    T *row = z + r * D + j;
    constexpr int kHm = kHc ? kHc : kSmallH;
    float y[kHm][kV];
#pragma unroll
    for (int h = 0; h < kHm; ++h) {
        if (kHc || h < H) {
            VecIO<T, kV>::load(row + h * dh, y[h]);
        } else {
#pragma unroll
            for (int e = 0; e < kV; ++e) y[h][e] = 0.0f;
        }
    }
#pragma unroll
    for (int gh = 0; gh < kHm; ++gh) {
        if (!kHc && gh >= H) break;
        float acc[kV];
#pragma unroll
        for (int e = 0; e < kV; ++e) acc[e] = 0.0f;
        if constexpr (kHc >= 4) {
#pragma unroll
            for (int h4 = 0; h4 < kHc; h4 += 4) {
                const float4 c4 = *reinterpret_cast<const float4 *>(C + gh * kHc + h4);
                const float cs[4] = {c4.x, c4.y, c4.z, c4.w};
#pragma unroll
                for (int q = 0; q < 4; ++q)
#pragma unroll
                    for (int e = 0; e < kV; ++e) acc[e] = fmaf(cs[q], y[h4 + q][e], acc[e]);
            }
        } else {
#pragma unroll
            for (int h = 0; h < kHm; ++h) {
                const float c = C[gh * H + (kHc || h < H ? h : 0)];
#pragma unroll
                for (int e = 0; e < kV; ++e) acc[e] = fmaf(c, y[h][e], acc[e]);
            }
        }
        VecIO<T, kV>::store(row + gh * dh, acc);
    }
}

// k_mixer_finish: one decode step's mixer for one batch row, after the recurrence
// step wrote y_t into z_t: coupling, gate, local path (the thread of channel d
// owns its history column, so it reads it all before shifting it).
template <typename T>
__global__ void __launch_bounds__(kBlock) k_mixer_finish(const T *__restrict__ x_t, const T *__restrict__ g_t,
                                                         T *__restrict__ z_t, T *hist,
                                                         const float *__restrict__ conv_w,
                                                         const float *__restrict__ scale, int K,
                                                         const float *__restrict__ c_raw, float lam, int H, int D) {
    asm volatile("griddepcontrol.wait;" ::: "memory");
    asm volatile("griddepcontrol.launch_dependents;" :::);
    extern __shared__ __align__(16) uint8_t sm[];
    float *C = reinterpret_cast<float *>(sm);
    float *ys = C + ((H * H + 3) & ~3);
    const int64_t b = blockIdx.x;
    build_coupling(C, c_raw, lam, H);
    for (int d = threadIdx.x; d < D; d += kBlock) ys[d] = as_f(z_t[b * D + d]);
    __syncthreads();
    const int dh = D / H;
    for (int d = threadIdx.x; d < D; d += kBlock) {
        const int gh = d / dh, j = d % dh;
        float v = 0.0f;
        for (int h = 0; h < H; ++h) v = fmaf(C[gh * H + h], ys[h * dh + j], v);
        if (g_t) v *= gatef(as_f(g_t[b * D + d]));
        if (K > 0) {
            const float xv = as_f(x_t[b * D + d]);
            float l = __ldg(conv_w + (int64_t)d * K) * xv;
            T *hc = hist + b * (K - 1) * (int64_t)D + d;    // entry j: u_{t-(K-1-j)}
            T hv[kMaxK];
            for (int j2 = 0; j2 < K - 1; ++j2) {
                hv[j2] = hc[(int64_t)j2 * D];
                l = fmaf(__ldg(conv_w + (int64_t)d * K + (K - 1 - j2)), as_f(hv[j2]), l);
            }
            for (int j2 = 1; j2 < K - 1; ++j2) hc[(int64_t)(j2 - 1) * D] = hv[j2];
            if (K > 1) hc[(int64_t)(K - 2) * D] = x_t[b * D + d];
            v = fmaf(__ldg(scale + d), l, v);
        }
        st_elem(z_t + b * D + d, v);
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

template <typename T, int K>
cudaError_t epilogue_k(const void *x, const void *g, void *z, const void *hist, const float *conv_w,
                       const float *scale, int64_t B, int64_t L, int D, cudaStream_t st) {
    const dim3 grid((unsigned)((D + kTC - 1) / kTC), (unsigned)((L + kTT - 1) / kTT), (unsigned)B);
    k_mixer_epilogue<T, K><<<grid, kEB, 0, st>>>(static_cast<const T *>(x), static_cast<const T *>(g),
                                                    static_cast<T *>(z), static_cast<const T *>(hist), conv_w,
                                                    scale, L, D);
    count_launches(1);
    return cudaGetLastError();
}

template <typename T>
cudaError_t epilogue_t(const void *x, const void *g, void *z, const void *hist, const float *conv_w,
                       const float *scale, int64_t B, int64_t L, int D, int K, cudaStream_t st) {
    switch (K) {
        case 0: return epilogue_k<T, 0>(x, g, z, hist, conv_w, scale, B, L, D, st);
        case 1: return epilogue_k<T, 1>(x, g, z, hist, conv_w, scale, B, L, D, st);
        case 2: return epilogue_k<T, 2>(x, g, z, hist, conv_w, scale, B, L, D, st);
        case 3: return epilogue_k<T, 3>(x, g, z, hist, conv_w, scale, B, L, D, st);
        case 4: return epilogue_k<T, 4>(x, g, z, hist, conv_w, scale, B, L, D, st);
        case 5: return epilogue_k<T, 5>(x, g, z, hist, conv_w, scale, B, L, D, st);
        case 6: return epilogue_k<T, 6>(x, g, z, hist, conv_w, scale, B, L, D, st);
        case 7: return epilogue_k<T, 7>(x, g, z, hist, conv_w, scale, B, L, D, st);
        default: return epilogue_k<T, 8>(x, g, z, hist, conv_w, scale, B, L, D, st);
    }
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

namespace {
template <typename T>
cudaError_t couple_t(void *z, const float *c_raw, float lam, int H, int64_t B, int64_t L, int D, cudaStream_t st) {
    if (H <= kSmallH) {
        const int dh = D / H;
        const int64_t n = B * L * (dh % 4 == 0 ? dh / 4 : dh);
        const unsigned grid = (unsigned)((n + kBlock - 1) / kBlock);
        T *zt = static_cast<T *>(z);
        if (dh % 4 == 0) {
            switch (H) {
                case 2: k_couple_small<T, 4, 2><<<grid, kBlock, 0, st>>>(zt, c_raw, lam, H, B * L, D); break;
                case 4: k_couple_small<T, 4, 4><<<grid, kBlock, 0, st>>>(zt, c_raw, lam, H, B * L, D); break;
                case 8: k_couple_small<T, 4, 8><<<grid, kBlock, 0, st>>>(zt, c_raw, lam, H, B * L, D); break;
                case 16: k_couple_small<T, 4, 16><<<grid, kBlock, 0, st>>>(zt, c_raw, lam, H, B * L, D); break;
                default: k_couple_small<T, 4, 0><<<grid, kBlock, 0, st>>>(zt, c_raw, lam, H, B * L, D); break;
            }
        } else {
            k_couple_small<T, 1, 0><<<grid, kBlock, 0, st>>>(zt, c_raw, lam, H, B * L, D);
        }
        count_launches(1);
        return cudaGetLastError();
    }
    // Whole rows of one batch row per block, up to 16 KB of them.
    const int rows = (int)std::max<int64_t>(1, std::min<int64_t>(64, 16384 / ((int64_t)D * sizeof(T))));
    const size_t smem = ((H * H * 4 + 15) & ~15) + (size_t)rows * D * sizeof(T);
    const dim3 grid((unsigned)((L + rows - 1) / rows), (unsigned)B);
    k_couple<T><<<grid, kBlock, smem, st>>>(static_cast<T *>(z), c_raw, lam, H, L, D, rows);
    count_launches(1);
    return cudaGetLastError();
}

template <typename T>
cudaError_t finish_t(const void *x_t, const void *g_t, void *z_t, void *hist, const float *conv_w, const float *scale,
                     int K, const float *c_raw, float lam, int H, int B, int D, cudaStream_t st) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)B);
    cfg.blockDim = dim3(kBlock);
    cfg.dynamicSmemBytes = ((H * H + 3) & ~3) * 4 + (size_t)D * 4;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    count_launches(1);
    return cudaLaunchKernelEx(&cfg, k_mixer_finish<T>, static_cast<const T *>(x_t), static_cast<const T *>(g_t),
                              static_cast<T *>(z_t), static_cast<T *>(hist), conv_w, scale, K, c_raw, lam, H, D);
}
}  // namespace

cudaError_t couple_heads(void *z, rlm_dtype dt, const float *c_raw, float lambda_c, int H, int64_t B, int64_t L,
                         int D, cudaStream_t st) {
    if (dt == RLM_BF16) return couple_t<__nv_bfloat16>(z, c_raw, lambda_c, H, B, L, D, st);
    return couple_t<float>(z, c_raw, lambda_c, H, B, L, D, st);
}

cudaError_t mixer_finish_coupled(const void *x_t, const void *g_t, void *z_t, void *hist, const float *conv_w,
                                 const float *scale, int K, const float *c_raw, float lambda_c, int H, rlm_dtype dt,
                                 int B, int D, cudaStream_t st) {
    if (dt == RLM_BF16)
        return finish_t<__nv_bfloat16>(x_t, g_t, z_t, hist, conv_w, scale, K, c_raw, lambda_c, H, B, D, st);
    return finish_t<float>(x_t, g_t, z_t, hist, conv_w, scale, K, c_raw, lambda_c, H, B, D, st);
}

cudaError_t conv_tail(const void *x, const void *hist, void *out, rlm_dtype dt, int64_t B, int64_t L, int D,
                      int K, cudaStream_t st) {
    if (K < 2) return cudaSuccess;
    if (dt == RLM_BF16) return tail_t<__nv_bfloat16>(x, hist, out, B, L, D, K, st);
    return tail_t<float>(x, hist, out, B, L, D, K, st);
}

}  // namespace rlm
