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
// grid be scheduled (right after the wait; for the batched plain step, before
// it), which hides most of the per-step launch latency when decode steps are
// issued back to back or captured in a graph.
//
// The plain step (no mixer) takes k_decode_tile, whose blocks cover 8 or 16
// batch rows of the same channels so the coefficient rows come from L1.
#include "rlm_device.cuh"
#include "rlm_internal.h"
#include "rlm_mixer.cuh"

namespace rlm {
namespace {

constexpr int kDecodeBlock = 256;

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
__device__ __forceinline__ float as_float(float v) { return v; }
__device__ __forceinline__ float as_float(__nv_bfloat16 v) { return __bfloat162float(v); }

// One thread's share of the mixer step: the thread of rank g in its (b, d) group
// (tpg threads) loads history entries j = g, g + tpg, ... (at most one when
// tpg >= K - 1), weighs them, and later moves them one slot down; rank 0 also
// loads the gate and adds the current drive's tap.  The loads are issued before
// the state update.
template <typename T>
struct MixPart {
    float l;          // partial sum of w[k] u_{t-k}
    float gate;       // rank 0: g_t
    float sc;         // rank 0: the channel's scale
    T xr;             // rank 0: u_t as stored, appended to the history
    T hv[2];          // the history entries this thread owns (tpg >= 4 gives at most two)
};

template <typename T>
__device__ __forceinline__ MixPart<T> mix_part(const MixStep<T> &m, int64_t b, int d, int64_t bd, int D,
                                               int g, int tpg, const T *x_t) {
    MixPart<T> r;
    r.l = 0.0f;
    r.gate = 0.0f;
    r.sc = 0.0f;
    if (m.g && g == 0) r.gate = ld_elem(m.g + bd);
    if (m.K > 0) {
        const float *w = m.conv_w + (int64_t)d * m.K;
        if (g == 0) {
            // Every load of the step is issued here, before the reductions.
            r.xr = x_t[bd];
            r.sc = __ldg(m.scale + d);
            r.l = __ldg(w) * as_float(r.xr);
        }
        const T *h = m.hist + b * (m.K - 1) * (int64_t)D + d;
#pragma unroll
        for (int i = 0; i < 2; ++i) {
            const int j = g + i * tpg;              // entry j holds u_{t-(K-1-j)}
            if (j < m.K - 1) {
                r.hv[i] = h[(int64_t)j * D];
                r.l = fmaf(__ldg(w + (m.K - 1 - j)), as_float(r.hv[i]), r.l);
            }
        }
    }
    return r;
}

// After the group's reductions (which every thread's loads feed, so all loads of
// the old history are complete): shift the owned entries one slot down, rank 0
// appends the current drive.
template <typename T>
__device__ __forceinline__ void mix_shift(const MixStep<T> &m, const MixPart<T> &r, int64_t b, int d, int D, int g,
                                          int tpg) {
    if (m.K < 2) return;
    T *h = m.hist + b * (m.K - 1) * (int64_t)D + d;
#pragma unroll
    for (int i = 0; i < 2; ++i) {
        const int j = g + i * tpg;
        if (j >= 1 && j < m.K - 1) h[(int64_t)(j - 1) * D] = r.hv[i];
    }
    if (g == 0) h[(int64_t)(m.K - 2) * D] = r.xr;
}

__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
// Moves the line holding p into L2 without reading it into the thread: safe before
// the dependency wait even if the previous grid writes the line (L2 is where the
// writes land), and it overlaps the token's DRAM latency with the wait.
__device__ __forceinline__ void prefetch_l2(const void *p) {
    asm volatile("prefetch.global.L2 [%0];" ::"l"(p));
}
// The step's fresh inputs (token and gate rows: one line per 64 (b, d) pairs).
template <typename T>
__device__ __forceinline__ void prefetch_step(const T *x_t, const MixStep<T> &mix, bool is_mix, int64_t bd,
                                              int64_t BD, int g) {
    if (g != 0 || bd >= BD || (bd & 63) != 0) return;
    prefetch_l2(x_t + bd);
    if (is_mix && mix.g) prefetch_l2(mix.g + bd);
}
__device__ __forceinline__ void pdl_launch_dependents() {
    asm volatile("griddepcontrol.launch_dependents;" :::);
}

// M even with one mode pair per thread: a block of R
// warps covers the same 32 / tpg channels for R batch rows (warp w takes row
// R * blockIdx.y + w), so the coefficient rows that every batch row needs are
// fetched from L2 once per block and then hit in L1.  Within a warp the lanes
// cover consecutive (channel, pair) slots of one row: one contiguous 512-byte
// state access per warp.  R = 16 for batches of 16 to 256 rows, else 8: in a
// CUDA graph of steps at D = 256, M = 16, B = 64 took 1.82 us per step with
// R = 16 against 1.97 (R = 8), 1.99 (R = 12), 1.97 (R = 24) and 2.03 (R = 32);
// B = 8 took 1.16 with R = 8 and 1.29 with R = 16; B = 8192 (state above the L2
// size, bandwidth-bound) 88.5 with R = 8 and 93.4 with R = 16.  A single row
// (B = 1) took 1.05 us here against 1.37 with one block per 32 (b, d) pairs.
// kMix adds the mixer step: the group's ranks share the history loads and the
// shift, rank 0 takes the gate and the local path's sum; a group may then hold
// ranks without modes.
// The launch bound holds the kernel to 32 registers, so 64 warps stay resident
// per SM (the mixer step spills 8 bytes): at 40 registers the mixer step took
// 11.1 us a step at B = 64, D = 2048, M = 16 against 10.6.
template <typename T, int R, bool kMix>
__global__ void __launch_bounds__(R * 32, 2048 / (R * 32)) k_decode_tile(
    const T *__restrict__ x_t, T *__restrict__ y_t, int B, int D, int M, int log2_tpg,
    float4 *__restrict__ s, const float4 *__restrict__ coef, MixStep<T> mix, bool late) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int tpg = 1 << log2_tpg;
    const int g = lane & (tpg - 1);
    const int d = blockIdx.x * (32 >> log2_tpg) + (lane >> log2_tpg);
    const int b = blockIdx.y * R + warp;
    const bool rowok = b < B && d < D;
    const bool on = rowok && 2 * g < M;
    const int64_t bd = (int64_t)b * D + d;
    if (rowok && g == 0 && (d & 63) == 0) {
        prefetch_l2(x_t + bd);
        if (kMix && mix.g) prefetch_l2(mix.g + bd);
    }
    // The next step's grid is released once this one's wait has returned, or,
    // for a plain step whose grid fits on the GPU at once (`late`), at the end.
    // In a CUDA graph of steps (D = 256, M = 16, B = 8 / 64, us per step) the
    // release after the wait gave 1.05 / 1.95 for the plain step and 1.86 / 2.53
    // for the mixer step (K = 4, gate), against 1.20 / 2.08 and 1.95 / 3.91 with
    // the release before the wait.  At the end, the plain step took 0.98 / 1.87
    // against 1.24 / 1.97 in another harness, and the mixer step 1.72 / 2.76;
    // grids of more than one wave lost 8-10 % (B = 256: 3.56 against 3.25).
    pdl_wait();
    if (kMix || !late) pdl_launch_dependents();
    MixPart<T> mp{};
    if (kMix && rowok) mp = mix_part(mix, (int64_t)b, d, bd, D, g, tpg, x_t);  // every rank, with or without modes
    float acc = 0.0f;
    if (on) {
        const float4 c0 = __ldg(coef + d * M + 2 * g);
        const float4 c1 = __ldg(coef + d * M + 2 * g + 1);
        const float xv = ld_elem(x_t + bd);
        const int64_t si = (bd * M) / 2 + g;
        const float4 q = s[si];
        const float r0 = fmaf(c0.x, q.x, fmaf(-c0.y, q.y, xv));
        const float i0 = fmaf(c0.x, q.y, c0.y * q.x);
        const float r1 = fmaf(c1.x, q.z, fmaf(-c1.y, q.w, xv));
        const float i1 = fmaf(c1.x, q.w, c1.y * q.z);
        s[si] = make_float4(r0, i0, r1, i1);
        acc = fmaf(c0.z, r0, fmaf(-c0.w, i0, fmaf(c1.z, r1, -c1.w * i1)));
    }
    float lsum = mp.l;
    for (int o = tpg >> 1; o > 0; o >>= 1) {
        acc += __shfl_xor_sync(0xffffffffu, acc, o);
        if (kMix) lsum += __shfl_xor_sync(0xffffffffu, lsum, o);
    }
    if (kMix && rowok) {
        mix_shift(mix, mp, (int64_t)b, d, D, g, tpg);
        if (g == 0) {
            if (mix.g) acc *= 1.0f / (1.0f + expf(-mp.gate));
            if (mix.K > 0) acc = fmaf(mp.sc, lsum, acc);
        }
    }
    if (rowok && g == 0) st_elem(y_t + bd, acc);
    if (!kMix && late) pdl_launch_dependents();
}

// Any M: each thread owns up to MPT modes, accessed as float2.
template <typename T, bool kMix>
__global__ void __launch_bounds__(kDecodeBlock) k_decode_any(
    const T *__restrict__ x_t, T *__restrict__ y_t, int64_t BD, int D, int M, int log2_tpg,
    int mpt, float2 *__restrict__ s, const float4 *__restrict__ coef, MixStep<T> mix) {
    const int64_t gid = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const int64_t bd = gid >> log2_tpg;
    const int g = (int)(gid & ((1 << log2_tpg) - 1));
    prefetch_step(x_t, mix, kMix, bd, BD, g);
    pdl_wait();
    pdl_launch_dependents();
    const int tpg = 1 << log2_tpg;
    const int64_t b = bd / D;
    const int d = (int)(bd - b * D);
    MixPart<T> mp{};
    if (kMix && bd < BD) mp = mix_part(mix, b, d, bd, D, g, tpg, x_t);
    float acc = 0.0f;
    if (bd < BD) {
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
    float lsum = mp.l;
    for (int o = tpg >> 1; o > 0; o >>= 1) {
        acc += __shfl_xor_sync(0xffffffffu, acc, o);
        if (kMix) lsum += __shfl_xor_sync(0xffffffffu, lsum, o);
    }
    if (kMix && bd < BD) {
        mix_shift(mix, mp, b, d, D, g, tpg);
        if (g == 0) {
            if (mix.g) acc *= 1.0f / (1.0f + expf(-mp.gate));
            if (mix.K > 0) acc = fmaf(mp.sc, lsum, acc);
        }
    }
    if (bd < BD && g == 0) st_elem(y_t + bd, acc);
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
cudaError_t launch_pdl_block(Kern kern, dim3 grid, int block, cudaStream_t st, Args... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = dim3(block);
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

template <typename Kern, typename... Args>
cudaError_t launch_pdl(Kern kern, dim3 grid, cudaStream_t st, Args... args) {
    return launch_pdl_block(kern, grid, kDecodeBlock, st, args...);
}

// One decode step with head coupling (Sec. 3.4) in a single launch, one block per
// batch row, for rows of at most 512 channels and 4096 modes.  Right after the
// dependency wait every load of the step is issued at once: the thread of channel
// d (threadIdx.x) takes its token, gate, drive history and conv weights, and every
// thread takes its (at most four) float4 mode pairs of the row's state slab with
// their coefficients -- consecutive threads on consecutive pairs, so the M / 2
// threads of a channel form one aligned shuffle group.  Phase 1 updates the
// states and puts each channel's readout y_t[d] in shared memory (fp32); after
// the block barrier, phase 2 forms (C y_t)[d], applies the gate and the local
// path, shifts the history and writes z_t[d].  C depends on the parameters only,
// so it is built before the wait.  H = 0: no coupling (the mixer step alone).
constexpr int kCoupledBlock = 512;
constexpr int kCoupledIters = 4;               // mode pairs per thread
constexpr int kCoupledMaxModesPerRow = 2 * kCoupledIters * kCoupledBlock;   // D * M <= 4096
constexpr int kHistMax = RLM_MAX_LOCAL_K - 1;

template <typename T>
__global__ void __launch_bounds__(kCoupledBlock, 1) k_decode_coupled(
    const T *__restrict__ x_t, T *__restrict__ z_t, int D, int M, float4 *__restrict__ s,
    const float4 *__restrict__ coef, MixStep<T> mix, const float *__restrict__ c_raw, float lam, int H) {
    extern __shared__ __align__(16) float smf[];
    float *C = smf;                              // [H][H]
    float *ys = smf + ((H * H + 3) & ~3);        // [D]
    const int64_t b = blockIdx.x;
    if (H > 0) build_coupling(C, c_raw, lam, H);
    pdl_wait();
    pdl_launch_dependents();
    const T *xb = x_t + b * D;
    // ---- loads: phase 2's inputs (channel d2) ...
    const int d2 = threadIdx.x, K = mix.K;
    const bool ch = d2 < D;
    T xraw = T(0.0f), hv[kHistMax];
    float gv = 0.0f, sc = 0.0f, w0 = 0.0f, wj[kHistMax];   // wj[j]: the weight of history entry j
    T *hc = K > 1 ? mix.hist + b * (K - 1) * (int64_t)D + d2 : nullptr;   // used only when K > 1
    if (ch) {
        xraw = xb[d2];
        if (mix.g) gv = ld_elem(mix.g + b * D + d2);
        if (K > 0) {
            sc = __ldg(mix.scale + d2);
            w0 = __ldg(mix.conv_w + (int64_t)d2 * K);
#pragma unroll
            for (int j = 0; j < kHistMax; ++j) {
                if (j < K - 1) {
                    hv[j] = hc[(int64_t)j * D];
                    wj[j] = __ldg(mix.conv_w + (int64_t)d2 * K + (K - 1 - j));
                }
            }
        }
    }
    // ... and phase 1's states, coefficients and tokens.
    const int pairs = M / 2;                     // a power of two, at most 32
    const int lp = __ffs(pairs) - 1;
    const int n4 = D * pairs;
    float4 *sb = s + b * n4;
    float4 stv[kCoupledIters], c0v[kCoupledIters], c1v[kCoupledIters];
    float xv[kCoupledIters];
#pragma unroll
    for (int k = 0; k < kCoupledIters; ++k) {
        const int i = (int)threadIdx.x + k * kCoupledBlock;
        const int d = i >> lp, g = i & (pairs - 1);
        if (i < n4) {
            xv[k] = ld_elem(xb + d);
            stv[k] = sb[i];
            c0v[k] = __ldg(coef + (int64_t)d * M + 2 * g);
            c1v[k] = __ldg(coef + (int64_t)d * M + 2 * g + 1);
        }
    }
    // ---- phase 1: every thread runs every iteration, so whole warps shuffle
#pragma unroll
    for (int k = 0; k < kCoupledIters; ++k) {
        const int i = (int)threadIdx.x + k * kCoupledBlock;
        const bool on = i < n4;
        const int d = i >> lp, g = i & (pairs - 1);
        float acc = 0.0f;
        if (on) {
            const float4 st = stv[k], c0 = c0v[k], c1 = c1v[k];
            const float r0 = fmaf(c0.x, st.x, fmaf(-c0.y, st.y, xv[k]));
            const float i0 = fmaf(c0.x, st.y, c0.y * st.x);
            const float r1 = fmaf(c1.x, st.z, fmaf(-c1.y, st.w, xv[k]));
            const float i1 = fmaf(c1.x, st.w, c1.y * st.z);
            sb[i] = make_float4(r0, i0, r1, i1);
            acc = fmaf(c0.z, r0, fmaf(-c0.w, i0, fmaf(c1.z, r1, -c1.w * i1)));
        }
        for (int o = pairs >> 1; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
        if (on && g == 0) ys[d] = acc;
    }
    __syncthreads();
    // ---- phase 2
    if (!ch) return;
    float v = ys[d2];
    if (H > 0) {
        const int dh = D / H, gh = d2 / dh, jh = d2 % dh;
        v = 0.0f;
        for (int h = 0; h < H; ++h) v = fmaf(C[gh * H + h], ys[h * dh + jh], v);
    }
    if (mix.g) v *= gatef(gv);
    if (K > 0) {
        float l = w0 * as_float(xraw);
#pragma unroll
        for (int j = 0; j < kHistMax; ++j)
            if (j < K - 1) l = fmaf(wj[j], as_float(hv[j]), l);
#pragma unroll
        for (int j = 1; j < kHistMax; ++j)
            if (j < K - 1) hc[(int64_t)(j - 1) * D] = hv[j];
        if (K > 1) hc[(int64_t)(K - 2) * D] = xraw;
        v = fmaf(sc, l, v);
    }
    st_elem(z_t + b * D + d2, v);
}

template <typename T, bool kMix>
cudaError_t decode_t(const T *x_t, T *y_t, int B, int D, int M, float *s, const float *coef,
                     MixStep<T> mix, cudaStream_t st) {
    int pairs = (M + 1) / 2;
    int log2_tpg = 0;
    while ((1 << log2_tpg) < pairs && log2_tpg < 5) ++log2_tpg;
    // The mixer step spreads the K - 1 <= 7 history entries over the group, two
    // at most per rank: at least 4 ranks (extra ranks own no modes).
    if (kMix && log2_tpg < 2) log2_tpg = 2;
    const int tpg = 1 << log2_tpg;
    const int64_t BD = (int64_t)B * D;
    const int64_t threads = BD * tpg;
    const unsigned grid = (unsigned)((threads + kDecodeBlock - 1) / kDecodeBlock);
    const float4 *cf = reinterpret_cast<const float4 *>(coef);
    if (M % 2 == 0 && 2 * tpg >= M) {
        // Blocks of R batch rows sharing their channels' coefficient rows (the
        // mixer step: 8 rows, 10.2 us a step at B = 64, D = 2048, M = 16, K = 4
        // against 10.5 with 16 rows and 10.9 with 4).
        const int R = !kMix && B >= 16 && B <= 256 ? 16 : 8;
        const dim3 gr((unsigned)((D + (32 >> log2_tpg) - 1) / (32 >> log2_tpg)), (unsigned)((B + R - 1) / R));
        // One wave: every block resident at once (32 registers: 2048 threads per SM).
        const bool late = !kMix && (int64_t)gr.x * gr.y <= (int64_t)sm_count() * (2048 / (R * 32));
        if (R == 16)
            return launch_pdl_block(k_decode_tile<T, 16, kMix>, gr, 16 * 32, st, x_t, y_t, B, D, M, log2_tpg,
                                    reinterpret_cast<float4 *>(s), cf, mix, late);
        return launch_pdl_block(k_decode_tile<T, 8, kMix>, gr, 8 * 32, st, x_t, y_t, B, D, M, log2_tpg,
                                reinterpret_cast<float4 *>(s), cf, mix, late);
    }
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

bool mixer_decode_coupled_supported(int D, int M) {
    const int pairs = M / 2;
    return M % 2 == 0 && pairs >= 1 && pairs <= 32 && (pairs & (pairs - 1)) == 0 && D <= kCoupledBlock &&
           (int64_t)D * M <= kCoupledMaxModesPerRow;
}

cudaError_t mixer_decode_coupled(const void *x_t, const void *g_t, void *z_t, rlm_dtype dt, int B, int D, int M,
                                 float *s, const float *coef, void *hist, const float *conv_w, const float *scale,
                                 int K, const float *c_raw, float lambda_c, int H, cudaStream_t st) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)B);
    cfg.blockDim = dim3(kCoupledBlock);
    cfg.dynamicSmemBytes = (size_t)(((H * H + 3) & ~3) + D) * sizeof(float);
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    count_launches(1);
    float4 *s4 = reinterpret_cast<float4 *>(s);
    const float4 *cf = reinterpret_cast<const float4 *>(coef);
    if (dt == RLM_BF16) {
        using T = __nv_bfloat16;
        const MixStep<T> m{static_cast<const T *>(g_t), static_cast<T *>(hist), conv_w, scale, K};
        return cudaLaunchKernelEx(&cfg, k_decode_coupled<T>, static_cast<const T *>(x_t), static_cast<T *>(z_t), D,
                                  M, s4, cf, m, c_raw, lambda_c, H);
    }
    const MixStep<float> m{static_cast<const float *>(g_t), static_cast<float *>(hist), conv_w, scale, K};
    return cudaLaunchKernelEx(&cfg, k_decode_coupled<float>, static_cast<const float *>(x_t),
                              static_cast<float *>(z_t), D, M, s4, cf, m, c_raw, lambda_c, H);
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
