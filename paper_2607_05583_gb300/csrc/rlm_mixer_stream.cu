// rlm_mixer_stream.cu -- the mixer pass of Sec. 3.4 on whole-row tiles.
//
// After the mixing has written y into z, one pass forms, in place,
//   z_t = sigma(g_t) . (C y_t) + s . sum_{k<K} w_k . u_{t-k}
// with each part optional: the head coupling C = I + lambda_c / sqrt(H)
// tanh(c_raw) over head-major channels, the gate g, and the local path of
// kernel size K (drives before token 0 from the history, or zero).
//
// A tile is R consecutive tokens of one batch row with all D channels.  In the
// [B][L][D] layout that is one contiguous run of R * D elements, so each
// tensor's tile -- y, g, and the drive together with the K - 1 rows before it --
// is a single bulk copy (cp.async.bulk, global -> shared, completing on an
// mbarrier).  The kernel is persistent, one CTA per SM, walking the tiles
// blockIdx.x, blockIdx.x + gridDim.x, ... through a ring of shared-memory
// stages: warp 16 issues the copies of the next tiles while warps 0-15 compute
// the current one from shared memory and write z.  A compute thread owns 4
// consecutive channels at a fixed place in every row it handles, so its K x 4
// conv weights, 4 scales and (with coupling) its head's row of C stay in
// registers; it works on two rows at once, two independent chains.  With
// coupling, the thread's 4 channels lie in one head (d_h a multiple of 4) and
// C y needs the same 4 positions of every head, which are all in the staged
// rows.
//
// Every mbarrier wait is bounded: after kWaitLimitCycles the waiting thread sets
// a shared abort flag and the device status word (RLM_ERR_TIMEOUT); the roles
// leave their loops, the copy issuer waits (again bounded) for the copies it
// issued, and the CTA returns.
#include <algorithm>
#include <type_traits>

#include "rlm_device.cuh"
#include "rlm_internal.h"
#include "rlm_mixer.cuh"

namespace rlm {

// Device status word of this translation unit (RLM_OK or RLM_ERR_TIMEOUT).
__device__ int g_mixer_status = 0;

namespace {

constexpr int kCW = 16;                        // compute warps
constexpr int kCh = 4;                         // channels per compute thread
constexpr int kThreads = (kCW + 1) * 32;       // + the copy-issuing warp
constexpr int kMaxK = RLM_MAX_LOCAL_K;
constexpr int kMaxStages = 4;
constexpr int kMaxRowBytes = 2048;             // D * sizeof(T) covered
constexpr int kMaxH = 16;                      // coupling heads covered
constexpr int kHdr = 2048;                     // barriers, abort flag, C
constexpr int kSmemMax = 227 * 1024;
constexpr long long kWaitLimitCycles = 4000000000ll;  // about 2 s at 2 GHz

struct StreamArgs {
    const void *x, *g, *hist;
    void *z;
    const float *conv_w, *scale, *c_raw;
    float lam;
    int K, D, R, stages;
    int64_t L, ntb, ntiles;       // tiles per batch row, all tiles
    uint32_t stage_bytes, off_y, off_g;
};

// ------------------------------------------------------------ PTX wrappers
__device__ __forceinline__ uint32_t smem_u32(const void *p) {
    return (uint32_t)__cvta_generic_to_shared(p);
}
__device__ __forceinline__ void bar_init(uint32_t bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count));
}
__device__ __forceinline__ bool bar_try(uint32_t bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{ .reg .pred p; mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2; selp.u32 %0, 1, 0, p; }"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    return ok != 0;
}
__device__ __forceinline__ void bar_arrive(uint32_t bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}
__device__ __forceinline__ void bar_expect_tx(uint32_t bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
}
// Bulk copy of `bytes` (a multiple of 16, both addresses 16-byte aligned) from
// global to this CTA's shared memory, counted on the mbarrier.
__device__ __forceinline__ void bulk_load(uint32_t dst, const void *src, uint32_t bytes, uint32_t bar) {
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
                 ::"r"(dst), "l"(src), "r"(bytes), "r"(bar)
                 : "memory");
}

// Bounded wait on an mbarrier phase; false if this CTA aborted.  The clock is
// read every 256 failed polls.
__device__ __forceinline__ bool wait_bar(uint32_t bar, uint32_t parity, volatile int *abort_flag) {
    if (bar_try(bar, parity)) return true;
    long long t0 = 0;
    for (uint32_t it = 1;; ++it) {
        if (bar_try(bar, parity)) return true;
        if ((it & 255u) == 0) {
            if (*abort_flag) return false;
            const long long now = clock64();
            if (t0 == 0) {
                t0 = now;
            } else if (now - t0 > kWaitLimitCycles) {
                *abort_flag = 1;
                atomicExch(&g_mixer_status, (int)RLM_ERR_TIMEOUT);
                return false;
            }
        }
    }
}
// The copy issuer's last wait for its own copies: bounded, whatever the flag.
__device__ __forceinline__ void drain_bar(uint32_t bar, uint32_t parity) {
    const long long t0 = clock64();
    while (!bar_try(bar, parity)) {
        if (clock64() - t0 > kWaitLimitCycles) {
            atomicExch(&g_mixer_status, (int)RLM_ERR_TIMEOUT);
            return;
        }
    }
}

// kCh = 4 consecutive channels: shared memory -> floats, floats -> global.
template <typename T> struct V4;
template <> struct V4<__nv_bfloat16> {
    __device__ static void lds(const __nv_bfloat16 *p, float (&v)[4]) {
        const uint2 u = *reinterpret_cast<const uint2 *>(p);
        v[0] = __uint_as_float(u.x << 16);
        v[1] = __uint_as_float(u.x & 0xFFFF0000u);
        v[2] = __uint_as_float(u.y << 16);
        v[3] = __uint_as_float(u.y & 0xFFFF0000u);
    }
    __device__ static void stg(__nv_bfloat16 *p, const float (&v)[4]) {
        uint32_t lo, hi;
        asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(lo) : "f"(v[1]), "f"(v[0]));
        asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(hi) : "f"(v[3]), "f"(v[2]));
        *reinterpret_cast<uint2 *>(p) = make_uint2(lo, hi);
    }
};
template <> struct V4<float> {
    __device__ static void lds(const float *p, float (&v)[4]) {
        const float4 a = *reinterpret_cast<const float4 *>(p);
        v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w;
    }
    __device__ static void stg(float *p, const float (&v)[4]) {
        *reinterpret_cast<float4 *>(p) = make_float4(v[0], v[1], v[2], v[3]);
    }
};

// kHc: the number of coupled heads (1, 2, 4, 8 or 16), 0 without coupling; kKm:
// the largest local kernel size the instance takes (4 or 8: weight registers).
template <typename T, int kHc, int kKm>
__global__ void __launch_bounds__(kThreads, 1) k_mixer_stream(const StreamArgs a) {
    extern __shared__ __align__(128) uint8_t sm[];
    const uint32_t sb = smem_u32(sm);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(sm + 64);
    float *Cs = reinterpret_cast<float *>(sm + 128);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int S = a.stages;
    const uint32_t full0 = sb, empty0 = sb + 8u * kMaxStages;
    if (threadIdx.x == 0) {
        for (int s = 0; s < S; ++s) {
            bar_init(full0 + 8u * s, 1);
            bar_init(empty0 + 8u * s, kCW);
        }
        *abort_flag = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (kHc) build_coupling(Cs, a.c_raw, a.lam, kHc);
    __syncthreads();

    const int D = a.D, K = a.K;
    const int Kh = K > 1 ? K - 1 : 0;                  // history rows before a tile
    const int64_t rb = (int64_t)D * sizeof(T);         // bytes per token row
    const int64_t nmine = (a.ntiles - 1 - blockIdx.x) / gridDim.x + 1;   // blockIdx.x < ntiles
    // Tile blockIdx.x + i * gridDim.x is (batch row b, tile tt of that row); both
    // roles step (b, tt) and their ring slot without a division per tile.
    const int64_t gdiv = gridDim.x / a.ntb, gmod = gridDim.x % a.ntb;
    const int64_t b_first = blockIdx.x / a.ntb, tt_first = blockIdx.x % a.ntb;

    if (warp == kCW) {
        // ---- copy issuer
        if (lane != 0) return;
        const T *x = static_cast<const T *>(a.x);
        const T *g = static_cast<const T *>(a.g);
        const T *hist = static_cast<const T *>(a.hist);
        const T *y = static_cast<const T *>(a.z);
        int64_t i = 0, b = b_first, tt = tt_first;
        int s = 0;
        uint32_t ph = 0;
        for (; i < nmine; ++i) {
            if (i > 0) {
                b += gdiv;
                tt += gmod;
                if (tt >= a.ntb) { tt -= a.ntb; ++b; }
                if (++s == S) { s = 0; ph ^= 1u; }
            }
            if (!wait_bar(empty0 + 8u * s, ph ^ 1u, abort_flag)) break;
            const int64_t t0 = tt * a.R;
            const int n = (int)(a.L - t0 < a.R ? a.L - t0 : a.R);
            const uint32_t st = sb + kHdr + (uint32_t)s * a.stage_bytes;
            const int hx = K > 0 ? (int)(t0 < Kh ? t0 : Kh) : 0;         // rows before t0 from x
            const int hh = (K > 0 && hist) ? Kh - hx : 0;                  // rows before token 0
            const uint32_t xbytes = K > 0 ? (uint32_t)((n + hx + hh) * rb) : 0u;
            const uint32_t rbytes = (uint32_t)(n * rb);
            bar_expect_tx(full0 + 8u * s, xbytes + rbytes * (g ? 2u : 1u));
            // Stage row r of the drive is token t0 - Kh + r.
            if (hh) bulk_load(st, hist + (b * Kh + t0) * D, (uint32_t)(hh * rb), full0 + 8u * s);
            if (K > 0)
                bulk_load(st + (uint32_t)((Kh - hx) * rb), x + (b * a.L + t0 - hx) * D, (uint32_t)((n + hx) * rb),
                          full0 + 8u * s);
            bulk_load(st + a.off_y, y + (b * a.L + t0) * D, rbytes, full0 + 8u * s);
            if (g) bulk_load(st + a.off_g, g + (b * a.L + t0) * D, rbytes, full0 + 8u * s);
        }
        // The CTA may not leave while its copies are landing.
        for (int r = 0; r < S; ++r) {
            const int64_t fills = i > r ? (i - r + S - 1) / S : 0;
            if (fills) drain_bar(full0 + 8u * r, (uint32_t)((fills - 1) & 1));
        }
        return;
    }

    // ---- compute warps
    T *z = static_cast<T *>(a.z);
    const bool has_g = a.g != nullptr, has_hist = a.hist != nullptr;
    const int ngrp = D / kCh;                          // channel groups per row
    const int rpp = (kCW * 32) / ngrp;                 // row pairs per pass (>= 2)
    const int cgi = threadIdx.x % ngrp, r0 = threadIdx.x / ngrp;
    const bool active = r0 < rpp;
    const int c = kCh * cgi;
    float w[kKm][kCh], sc[kCh];
#pragma unroll
    for (int k = 0; k < kKm; ++k)
#pragma unroll
        for (int e = 0; e < kCh; ++e) w[k][e] = (k < K) ? __ldg(a.conv_w + (int64_t)(c + e) * K + k) : 0.0f;
#pragma unroll
    for (int e = 0; e < kCh; ++e) sc[e] = K > 0 ? __ldg(a.scale + c + e) : 0.0f;
    constexpr int kHr = kHc ? kHc : 1;
    float cr[kHr];
    int dh = D, jc = c;
    if (kHc) {
        dh = D / kHr;
        const int gh = c / dh;
        jc = c - gh * dh;                              // the same position in head 0
#pragma unroll
        for (int h = 0; h < kHr; ++h) cr[h] = Cs[gh * kHr + h];
    }
    const int pair = 2 * rpp * D;                      // elements from one pair of a thread to its next
    int64_t b = b_first, tt = tt_first;
    int s = 0;
    uint32_t ph = 0;
    for (int64_t i = 0; i < nmine; ++i) {
        if (i > 0) {
            b += gdiv;
            tt += gmod;
            if (tt >= a.ntb) { tt -= a.ntb; ++b; }
            if (++s == S) { s = 0; ph ^= 1u; }
        }
        if (!wait_bar(full0 + 8u * s, ph, abort_flag)) break;
        const int64_t t0 = tt * a.R;
        const int n = (int)(a.L - t0 < a.R ? a.L - t0 : a.R);
        const uint8_t *st = sm + kHdr + (size_t)s * a.stage_bytes;
        const T *xs = reinterpret_cast<const T *>(st);
        const T *ys = reinterpret_cast<const T *>(st + a.off_y);
        const T *gs = reinterpret_cast<const T *>(st + a.off_g);
        T *zt = z + (b * a.L + t0) * D + c;
        // Without a history, the stage rows before token 0 hold no drive: only a
        // sequence's first tile has taps that reach them, and only it masks them
        // (vmin = the first stage row that holds a drive).
        const int vmin = (has_hist || t0 >= Kh) ? 0 : Kh - (int)t0;
        // Two consecutive rows at a time, ra and ra + 1 (R is even, so ra + 1 is a
        // stage row; past the tile it is computed from stale data and not
        // stored).  Their local paths share K - 1 of their K + 1 drive rows.
        auto rows = [&](auto guard) {
            constexpr bool kGuard = decltype(guard)::value;
            for (int ra = 2 * r0, e0 = 2 * r0 * D; ra < n; ra += 2 * rpp, e0 += pair) {
                const bool second = ra + 1 < n;
                const int e1 = e0 + D;                         // element offsets of the rows
                float o[2][kCh], v[2][kCh];
                if (kHc) {
#pragma unroll
                    for (int q = 0; q < 2; ++q)
#pragma unroll
                        for (int e = 0; e < kCh; ++e) o[q][e] = 0.0f;
#pragma unroll
                    for (int h = 0; h < kHr; ++h) {
#pragma unroll
                        for (int q = 0; q < 2; ++q) {
                            V4<T>::lds(ys + (q ? e1 : e0) + h * dh + jc, v[q]);
#pragma unroll
                            for (int e = 0; e < kCh; ++e) o[q][e] = fmaf(cr[h], v[q][e], o[q][e]);
                        }
                    }
                } else {
#pragma unroll
                    for (int q = 0; q < 2; ++q) V4<T>::lds(ys + (q ? e1 : e0) + c, o[q]);
                }
                if (has_g) {
#pragma unroll
                    for (int q = 0; q < 2; ++q) {
                        V4<T>::lds(gs + (q ? e1 : e0) + c, v[q]);
#pragma unroll
                        for (int e = 0; e < kCh; ++e) o[q][e] *= gatef(v[q][e]);
                    }
                }
                if (K > 0) {
                    float l[2][kCh];
#pragma unroll
                    for (int q = 0; q < 2; ++q)
#pragma unroll
                        for (int e = 0; e < kCh; ++e) l[q][e] = 0.0f;
                    // Drive row j (j = 0..K) is token t0 + ra + 1 - j, stage row
                    // Kh + ra + 1 - j: tap j of row ra + 1 and tap j - 1 of row ra.
                    const int xtop = e1 + Kh * D + c;
#pragma unroll
                    for (int j = 0; j <= kKm; ++j) {
                        if (j > K) break;
                        int xe = xtop - j * D;
                        bool ok = true;
                        if (kGuard) {
                            ok = ra + 1 + Kh - j >= vmin;
                            xe = ok ? xe : vmin * D + c;             // any staged drive row
                        }
                        V4<T>::lds(xs + xe, v[0]);
                        if (kGuard && !ok) {
#pragma unroll
                            for (int e = 0; e < kCh; ++e) v[0][e] = 0.0f;
                        }
                        if (j < kKm && j < K) {
#pragma unroll
                            for (int e = 0; e < kCh; ++e) l[1][e] = fmaf(w[j < kKm ? j : 0][e], v[0][e], l[1][e]);
                        }
                        if (j >= 1) {
#pragma unroll
                            for (int e = 0; e < kCh; ++e) l[0][e] = fmaf(w[j >= 1 ? j - 1 : 0][e], v[0][e], l[0][e]);
                        }
                    }
#pragma unroll
                    for (int q = 0; q < 2; ++q)
#pragma unroll
                        for (int e = 0; e < kCh; ++e) o[q][e] = fmaf(sc[e], l[q][e], o[q][e]);
                }
                V4<T>::stg(zt + e0, o[0]);
                if (second) V4<T>::stg(zt + e1, o[1]);
            }
        };
        if (active) {
            if (vmin == 0)
                rows(std::false_type{});
            else
                rows(std::true_type{});
        }
        __syncwarp();
        if (lane == 0) bar_arrive(empty0 + 8u * s);
    }
}

template <typename T, int kHc, int kKm>
cudaError_t stream_launch(const StreamArgs &a, size_t smem, cudaStream_t st) {
    static bool configured = false;      // a repeated attribute call is harmless
    if (!configured) {
        const cudaError_t e = cudaFuncSetAttribute(k_mixer_stream<T, kHc, kKm>,
                                                   cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemMax);
        if (e != cudaSuccess) return e;
        configured = true;
    }
    const unsigned grid = (unsigned)std::min<int64_t>(a.ntiles, sm_count());
    k_mixer_stream<T, kHc, kKm><<<grid, kThreads, smem, st>>>(a);
    count_launches(1);
    return cudaGetLastError();
}

template <typename T, int kKm>
cudaError_t stream_h(const StreamArgs &a, int H, size_t smem, cudaStream_t st) {
    switch (H) {
        case 0: return stream_launch<T, 0, kKm>(a, smem, st);
        case 1: return stream_launch<T, 1, kKm>(a, smem, st);
        case 2: return stream_launch<T, 2, kKm>(a, smem, st);
        case 4: return stream_launch<T, 4, kKm>(a, smem, st);
        case 8: return stream_launch<T, 8, kKm>(a, smem, st);
        default: return stream_launch<T, 16, kKm>(a, smem, st);
    }
}

template <typename T>
cudaError_t stream_t(const StreamArgs &a, int H, size_t smem, cudaStream_t st) {
    return a.K <= 4 ? stream_h<T, 4>(a, H, smem, st) : stream_h<T, kMaxK>(a, H, smem, st);
}

}  // namespace

bool mixer_stream_supported(rlm_dtype dt, int D, int H) {
    const int64_t rb = (int64_t)D * (dt == RLM_BF16 ? 2 : 4);
    if (D < 8 || D % 8 != 0 || rb > kMaxRowBytes) return false;    // D / kCh <= 512 groups
    if (H == 0) return true;
    if (H != 1 && H != 2 && H != 4 && H != 8 && H != kMaxH) return false;
    return D % H == 0 && (D / H) % kCh == 0;
}

cudaError_t mixer_stream(const void *x, const void *g, void *z, const void *hist, const float *conv_w,
                         const float *scale, int K, const float *c_raw, float lambda_c, int H, rlm_dtype dt,
                         int64_t B, int64_t L, int D, cudaStream_t st) {
    const int64_t rb = (int64_t)D * (dt == RLM_BF16 ? 2 : 4);
    StreamArgs a{};
    a.x = x;
    a.g = g;
    a.hist = K > 1 ? hist : nullptr;
    a.z = z;
    a.conv_w = conv_w;
    a.scale = scale;
    a.c_raw = c_raw;
    a.lam = lambda_c;
    a.K = K;
    a.D = D;
    a.R = (int)std::max<int64_t>(2, std::min<int64_t>(64, 16384 / rb)) & ~1;   // even: rows go in pairs
    a.L = L;
    a.ntb = (L + a.R - 1) / a.R;
    a.ntiles = B * a.ntb;
    const int Kh = K > 1 ? K - 1 : 0;
    const int64_t xrows = K > 0 ? Kh + a.R : 0;
    a.off_y = (uint32_t)(xrows * rb);
    a.off_g = (uint32_t)((xrows + a.R) * rb);
    const int64_t bytes = (xrows + a.R + (g ? a.R : 0)) * rb;
    a.stage_bytes = (uint32_t)((bytes + 127) & ~int64_t(127));
    a.stages = (int)std::min<int64_t>(kMaxStages, (kSmemMax - kHdr) / a.stage_bytes);
    const size_t smem = kHdr + (size_t)a.stages * a.stage_bytes;
    if (dt == RLM_BF16) return stream_t<__nv_bfloat16>(a, H, smem, st);
    return stream_t<float>(a, H, smem, st);
}

cudaError_t read_and_clear_mixer_status(int *status, cudaStream_t st) {
    cudaError_t e = cudaMemcpyFromSymbolAsync(status, g_mixer_status, sizeof(int), 0, cudaMemcpyDeviceToHost, st);
    if (e != cudaSuccess) return e;
    if ((e = cudaStreamSynchronize(st)) != cudaSuccess) return e;
    const int zero = 0;
    if ((e = cudaMemcpyToSymbolAsync(g_mixer_status, &zero, sizeof(int), 0, cudaMemcpyHostToDevice, st)) !=
        cudaSuccess)
        return e;
    return cudaStreamSynchronize(st);
}

}  // namespace rlm
