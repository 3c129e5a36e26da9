// rlm_prefill_tc.cu -- tcgen05 tensor-core prefill for bf16 I/O, M = 16 modes.
//
// The operator (Sec. 3.2, Eq. 2) is evaluated as a chunked complex-diagonal
// scan.  With chunks of C = 64 tokens, position p of chunk n of channel d:
//
//   y[nC+p] = sum_{q<=p} K[p-q] x[nC+q]            intra-chunk Toeplitz block
//           + sum_m Re(c_m lambda_m^(p+1) S_{n-1,m})  carried state, up-projected
//   L_n     = sum_q lambda^(C-1-q) x[nC+q]           chunk-local end state
//   S_n     = lambda^C S_{n-1} + L_n                 inter-chunk carry (fp32)
//
// Both contractions over the chunk's positions are dense matrix products per
// channel and run on the tensor cores (tcgen05.mma, kind::f16, bf16 operands,
// fp32 accumulators in TMEM):
//
//   D[0:64, n]   = T  (64x64)  X_n      Toeplitz block, T[p][q] = K[p-q]
//   D[64:96, n]  = W  (32x64)  X_n      local end state, (Re, Im) of 16 modes
//   D[0:64, n]  += U  (64x32)  S_{n-1}  up-projection of the carried state
//
// T and W share one A operand (rows 0-63 and 64-95 of a 128-row matrix), so a
// single MMA chain yields both.  The columns of D are the NT = 32 chunks of a
// 2048-token tile (MMA N = 32).  The carry between chunks is a sequential fp32
// complex scan in registers: one thread per state row, the two rows (Re, Im) of
// a mode exchange their values with one warp shuffle per chunk.
//
// One CTA owns one batch row b and one group of DG = 8 channels (a 16-byte
// slice of each token row) and walks the sequence tile by tile, carrying the
// state in registers, so no CTA waits on another.
//
// Data movement per tile (2048 tokens x 8 channels):
//   TMA (3-D map over [B][L][D], zero fill outside the sequence) -> smem ring
//   -> ldmatrix.trans / stmatrix into the per-channel K-major B operand (the
//      positions of a chunk reversed, so the Toeplitz block becomes a Hankel
//      block; see the A operand layout below)
//   -> tcgen05.mma -> TMEM -> scan warps -> B operand of the up-projection
//   -> tcgen05.mma -> TMEM -> epilogue warps (fp32 -> bf16, 8 channels packed
//      into one 16-byte row) -> smem ring -> TMA store.
// TMEM is double-buffered across tiles (2 x 8 channels x 32 columns).
//
// Warp roles (16 warps): TMEM lane quarter q = warp % 4 decides which rows of
// D a warp may read.  Quarters 0-1: epilogue (rows 0-63).  Quarter 2: scan
// (rows 64-95), two channels per warp.  Quarter 3: TMA producer (warp 3), MMA
// issuer (warp 7), TMA store issuer (warp 11), transposer (warp 15).
//
// Every wait is bounded: after kWaitLimitNs the waiting thread sets a shared
// abort flag and the device status word (RLM_ERR_TIMEOUT); all roles then leave
// their loops, drain what they issued and the CTA frees its TMEM and returns.
#include <cuda.h>

#include <mutex>
#include <vector>

#include "rlm_device.cuh"
#include "rlm_internal.h"

namespace rlm {

// Device status word: RLM_OK, or RLM_ERR_TIMEOUT once a bounded wait expired.
__device__ int g_device_status = 0;

namespace {

constexpr int kC = 64;                 // chunk length
constexpr int kNT = 32;                // chunks per tile = MMA N
constexpr int kTile = kC * kNT;        // 2048 tokens
constexpr int kDG = 8;                 // channels per CTA
constexpr int kModes = 16;             // M handled by this kernel
constexpr int kBox = 256;              // TMA box rows
constexpr int kBoxes = kTile / kBox;   // 8 per tile
constexpr int kXSlots = 4;             // x ring depth (boxes)
constexpr int kYSlots = 2;             // y ring depth (blocks of 8 chunks)
constexpr int kThreads = 512;
constexpr int kTmemCols = 512;
constexpr unsigned long long kWaitLimitNs = 1000000000ull;  // 1 s

// Shared memory map (bytes from a 1024-aligned base).
constexpr int kAtwStride = 12 * 1024;  // 96 real rows x 128 B; rows 96-127 alias the next buffer
constexpr int kAuStride = 4096;        // 64 real rows x 64 B;  rows 64-127 alias the next buffer
constexpr int kBxStride = 4096 + 16;   // 32 rows x 128 B, +16 so stmatrix rows hit distinct banks
constexpr int kBsLbo = 144, kBsSbo = 576, kBsStride = 4 * kBsSbo;
constexpr int kOffAtw = 0;
constexpr int kOffAu = kOffAtw + kDG * kAtwStride;          // 98304
constexpr int kOffBx = kOffAu + kDG * kAuStride;             // 131072
constexpr int kOffBs = kOffBx + kDG * kBxStride;             // 163968
constexpr int kOffX = 182400;                                // 128-aligned
constexpr int kOffY = kOffX + kXSlots * kBox * 16;           // 198784
constexpr int kOffBar = kOffY + kYSlots * 512 * 16;          // 215168
constexpr int kNumBars = 64;
constexpr int kOffMisc = kOffBar + kNumBars * 8;
constexpr int kSmemBytes = kOffMisc + 64 + 1024;             // + alignment slack
static_assert(kOffBs + kDG * kBsStride <= kOffX, "smem layout overlap");
static_assert(kOffX % 128 == 0 && kOffY % 128 == 0, "TMA buffers need 128-byte alignment");
static_assert(kOffBx + 8 * 64 * 16 * 4 + 8 * 64 * 4 <= kOffX, "prologue scratch does not fit");

// Barrier indices.
constexpr int kBarXFull = 0;        // [4]
constexpr int kBarXEmpty = 4;       // [4]
constexpr int kBarBxFull = 8;
constexpr int kBarBxEmpty = 9;
constexpr int kBarTwDone = 10;      // [2][8]
constexpr int kBarSFull = 26;       // [8]
constexpr int kBarUDone = 34;       // [2]
constexpr int kBarDEmpty = 36;      // [2]
constexpr int kBarYFull = 38;       // [2]
constexpr int kBarYEmpty = 40;      // [2]
constexpr int kBarFinal = 42;

// Instruction descriptor, kind::f16: fp32 accumulate, bf16 A and B, both
// K-major, M = 128, N = 32.
constexpr uint32_t kIdesc = (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(kNT >> 3) << 17) |
                            ((uint32_t)(128 >> 4) << 24);

// ------------------------------------------------------------ PTX wrappers
__device__ __forceinline__ uint32_t smem_u32(const void *p) {
    return (uint32_t)__cvta_generic_to_shared(p);
}
__device__ __forceinline__ uint64_t globaltimer() {
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
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
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes)
                 : "memory");
}

// Bounded wait on an mbarrier phase.  Returns false if this CTA aborted.
__device__ __forceinline__ bool wait_bar(uint32_t bar, uint32_t parity, volatile int *abort_flag) {
    if (bar_try(bar, parity)) return true;
    const uint64_t t0 = globaltimer();
    for (uint32_t it = 1;; ++it) {
        if (bar_try(bar, parity)) return true;
        if (*abort_flag) return false;
        if ((it & 63u) == 0 && globaltimer() - t0 > kWaitLimitNs) {
            *abort_flag = 1;
            atomicExch(&g_device_status, (int)RLM_ERR_TIMEOUT);
            return false;
        }
    }
}

__device__ __forceinline__ void fence_async_smem() {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_before() {
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

__device__ __forceinline__ void tma_load_3d(uint32_t dst, const CUtensorMap *map, int c0, int c1,
                                            int c2, uint32_t bar) {
    asm volatile(
        "cp.async.bulk.tensor.3d.shared::cluster.global.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%2, %3, %4}], [%5];" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(c2), "r"(bar)
        : "memory");
}
__device__ __forceinline__ void tma_store_3d(const CUtensorMap *map, uint32_t src, int c0, int c1,
                                             int c2) {
    asm volatile(
        "cp.async.bulk.tensor.3d.global.shared::cta.bulk_group [%0, {%1, %2, %3}], [%4];" ::"l"(
            reinterpret_cast<uint64_t>(map)),
        "r"(c0), "r"(c1), "r"(c2), "r"(src)
        : "memory");
}
__device__ __forceinline__ void tma_store_commit() {
    asm volatile("cp.async.bulk.commit_group;" ::: "memory");
}
__device__ __forceinline__ void tma_store_wait_read() {
    asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory");
}
__device__ __forceinline__ void tma_store_wait_all() {
    asm volatile("cp.async.bulk.wait_group 0;" ::: "memory");
}

// UMMA shared-memory descriptor: K-major, no swizzle.  LBO = byte distance of
// core matrices adjacent along K, SBO = along M/N; bit 46 = descriptor version.
__device__ __forceinline__ uint64_t umma_desc(uint32_t saddr, uint32_t lbo, uint32_t sbo) {
    return (uint64_t)((saddr >> 4) & 0x3FFFu) | ((uint64_t)((lbo >> 4) & 0x3FFFu) << 16) |
           ((uint64_t)((sbo >> 4) & 0x3FFFu) << 32) | ((uint64_t)1 << 46);
}
__device__ __forceinline__ void umma_f16(uint32_t d_tmem, uint64_t a, uint64_t b, uint32_t accum) {
    asm volatile(
        "{ .reg .pred p; setp.ne.b32 p, %4, 0;\n"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p; }" ::"r"(d_tmem),
        "l"(a), "l"(b), "r"(kIdesc), "r"(accum)
        : "memory");
}
__device__ __forceinline__ void umma_commit(uint32_t bar) {
    asm volatile(
        "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
        : "memory");
}

#define RLM_TMEM_LD32(taddr, v)                                                                   \
    asm volatile(                                                                                 \
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13," \
        "%14,%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"       \
        : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]),   \
          "=r"(v[7]), "=r"(v[8]), "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]),             \
          "=r"(v[13]), "=r"(v[14]), "=r"(v[15]), "=r"(v[16]), "=r"(v[17]), "=r"(v[18]),          \
          "=r"(v[19]), "=r"(v[20]), "=r"(v[21]), "=r"(v[22]), "=r"(v[23]), "=r"(v[24]),          \
          "=r"(v[25]), "=r"(v[26]), "=r"(v[27]), "=r"(v[28]), "=r"(v[29]), "=r"(v[30]),          \
          "=r"(v[31])                                                                             \
        : "r"(taddr))

__device__ __forceinline__ void tmem_ld2(uint32_t taddr, uint32_t &a, uint32_t &b) {
    asm volatile("tcgen05.ld.sync.aligned.32x32b.x2.b32 {%0, %1}, [%2];"
                 : "=r"(a), "=r"(b)
                 : "r"(taddr));
}
__device__ __forceinline__ void tmem_wait_ld() {
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
    uint32_t r;
    asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(hi), "f"(lo));
    return r;
}

struct TcArgs {
    const float *decay, *freq, *amp, *phase;
    float2 *state_out;   // nullable, [B][D][M]
    float4 *coef_out;    // nullable, [D][M]
    __nv_bfloat16 *y;    // for the plain stores of partially negative boxes
    int64_t L;
    int D;
    int ntiles;
    int64_t t0;          // first token of tile 0 (<= 0): tiles end exactly at L-1
};

__global__ void __launch_bounds__(kThreads, 1)
    k_prefill_tc(const __grid_constant__ CUtensorMap tmap_x,
                 const __grid_constant__ CUtensorMap tmap_y, const TcArgs args) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    const uint32_t sbase = smem_u32(smem);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int g = blockIdx.x, b = blockIdx.y;
    const int d0 = g * kDG;
    const int D = args.D;
    const int ntiles = args.ntiles;
    uint64_t *bars = reinterpret_cast<uint64_t *>(smem + kOffBar);
    auto bar = [&](int i) { return smem_u32(bars + i); };
    volatile int *abort_flag = reinterpret_cast<volatile int *>(smem + kOffMisc);
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(smem + kOffMisc + 16);

    if (tid == 0) {
        *abort_flag = 0;
        for (int i = 0; i < 4; ++i) {
            bar_init(bar(kBarXFull + i), 1);
            bar_init(bar(kBarXEmpty + i), 1);
        }
        bar_init(bar(kBarBxFull), 1);
        bar_init(bar(kBarBxEmpty), 1);
        for (int i = 0; i < 16; ++i) bar_init(bar(kBarTwDone + i), 1);
        for (int i = 0; i < 8; ++i) bar_init(bar(kBarSFull + i), 1);
        for (int i = 0; i < 2; ++i) {
            bar_init(bar(kBarUDone + i), 1);
            bar_init(bar(kBarDEmpty + i), 12);
            bar_init(bar(kBarYFull + i), 8);
            bar_init(bar(kBarYEmpty + i), 1);
        }
        bar_init(bar(kBarFinal), 1);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (warp == 7) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                         smem_u32(tmem_slot)),
                     "r"(kTmemCols));
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    // The producer starts the first loads before the constants are built.
    const int total_boxes = ntiles * kBoxes;
    int issued = 0;
    if (warp == 3 && lane == 0) {
        for (; issued < total_boxes && issued < kXSlots; ++issued) {
            const int jt = issued / kBoxes, q = issued % kBoxes;
            const uint32_t slot = issued % kXSlots;
            bar_expect_tx(bar(kBarXFull + slot), kBox * 16);
            tma_load_3d(sbase + kOffX + slot * (kBox * 16), &tmap_x, d0,
                        (int)(args.t0 + (int64_t)jt * kTile + q * kBox), b, bar(kBarXFull + slot));
        }
    }

    // ---------------------------------------------------- per-channel constants
    // Stage 1: thread (c, m, quarter) runs powers lambda^n, n in [16 qn, 16 qn + 16).
    {
        float *kt = reinterpret_cast<float *>(smem + kOffBx);  // [8][64][16] scratch
        const int c = tid >> 6, m = (tid >> 2) & 15, qn = tid & 3;
        const int pm = (d0 + c) * kModes + m;
        const float ga = args.decay[pm], om = args.freq[pm];
        const float2 lam = lambda_pow(ga, om, 1.0f);
        const float2 cf = mode_coef(args.amp[pm], args.phase[pm]);
        if (args.coef_out && b == 0 && qn == 0)
            args.coef_out[pm] = make_float4(lam.x, lam.y, cf.x, cf.y);
        float2 pw = lambda_pow(ga, om, (float)(16 * qn));
        uint8_t *atw = smem + kOffAtw + c * kAtwStride;
        uint8_t *au = smem + kOffAu + c * kAuStride;
        const int wrow = 64 + 2 * m;                 // W rows: Re at 64+2m, Im at 65+2m
        for (int h = 0; h < 2; ++h) {
            uint32_t re4[4], im4[4];
            for (int e = 0; e < 8; e += 2) {
                const int n = 16 * qn + 8 * h + e;
                const float2 p0 = pw;
                const float2 p1 = cmul(pw, lam);
                re4[e / 2] = pack_bf16x2(p0.x, p1.x);
                im4[e / 2] = pack_bf16x2(p0.y, p1.y);
                // K table contributions and U rows for n and n+1
                kt[(c * 64 + n) * 16 + m] = cf.x * p0.x - cf.y * p0.y;
                kt[(c * 64 + n + 1) * 16 + m] = cf.x * p1.x - cf.y * p1.y;
                const float2 q0 = cmul(cf, p1);      // c lambda^(n+1)
                const float2 p2 = cmul(p1, lam);
                const float2 q1 = cmul(cf, p2);      // c lambda^(n+2)
                *reinterpret_cast<uint32_t *>(au + (n / 8) * 512 + (m / 4) * 128 + (n % 8) * 16 +
                                              ((2 * m) % 8) * 2) = pack_bf16x2(q0.x, -q0.y);
                *reinterpret_cast<uint32_t *>(au + ((n + 1) / 8) * 512 + (m / 4) * 128 +
                                              ((n + 1) % 8) * 16 + ((2 * m) % 8) * 2) =
                    pack_bf16x2(q1.x, -q1.y);
                pw = p2;
            }
            const int kb = 2 * qn + h;
            *reinterpret_cast<uint4 *>(atw + (wrow / 8) * 1024 + kb * 128 + (wrow % 8) * 16) =
                make_uint4(re4[0], re4[1], re4[2], re4[3]);
            *reinterpret_cast<uint4 *>(atw + ((wrow + 1) / 8) * 1024 + kb * 128 +
                                       ((wrow + 1) % 8) * 16) =
                make_uint4(im4[0], im4[1], im4[2], im4[3]);
        }
    }
    __syncthreads();
    // Stage 2: K[c][n] = sum_m Re(c_m lambda_m^n)   (Eq. 1 at integer lags)
    {
        const float *kt = reinterpret_cast<const float *>(smem + kOffBx);
        float *kf = reinterpret_cast<float *>(smem + kOffBx + 8 * 64 * 16 * 4);
        const int c = tid >> 6, n = tid & 63;
        float s = 0.0f;
#pragma unroll
        for (int m = 0; m < kModes; ++m) s += kt[(c * 64 + n) * 16 + m];
        kf[c * 64 + n] = s;
    }
    __syncthreads();
    // Stage 3: Toeplitz rows in reversed-position coordinates: T[i][p'] = K[i + p' - 63].
    {
        const float *kf = reinterpret_cast<const float *>(smem + kOffBx + 8 * 64 * 16 * 4);
        const int c = tid >> 6, i = tid & 63;
        uint8_t *atw = smem + kOffAtw + c * kAtwStride;
        for (int kb = 0; kb < 8; ++kb) {
            float v[8];
#pragma unroll
            for (int e = 0; e < 8; ++e) {
                const int lag = i + 8 * kb + e - 63;
                v[e] = lag >= 0 ? kf[c * 64 + lag] : 0.0f;
            }
            *reinterpret_cast<uint4 *>(atw + (i / 8) * 1024 + kb * 128 + (i % 8) * 16) =
                make_uint4(pack_bf16x2(v[0], v[1]), pack_bf16x2(v[2], v[3]),
                           pack_bf16x2(v[4], v[5]), pack_bf16x2(v[6], v[7]));
        }
    }
    fence_async_smem();
    __syncthreads();

    const int quarter = warp & 3;
    if (warp == 3) {
        // ---------------------------------------------------- TMA producer
        if (lane == 0) {
            for (; issued < total_boxes; ++issued) {
                const int jt = issued / kBoxes, q = issued % kBoxes;
                const uint32_t slot = issued % kXSlots;
                const uint32_t fill = issued / kXSlots;
                if (!wait_bar(bar(kBarXEmpty + slot), (fill & 1) ^ 1, abort_flag)) break;
                bar_expect_tx(bar(kBarXFull + slot), kBox * 16);
                tma_load_3d(sbase + kOffX + slot * (kBox * 16), &tmap_x, d0,
                            (int)(args.t0 + (int64_t)jt * kTile + q * kBox), b,
                            bar(kBarXFull + slot));
            }
            // Drain: every issued load must land before this CTA may exit.
            const int first_unconsumed = issued > kXSlots ? issued - kXSlots : 0;
            for (int k = first_unconsumed; k < issued; ++k) {
                const uint32_t slot = k % kXSlots, fill = k / kXSlots;
                const uint64_t t0 = globaltimer();
                while (!bar_try(bar(kBarXFull + slot), fill & 1))
                    if (globaltimer() - t0 > kWaitLimitNs) break;
            }
        }
        __syncwarp();
    } else if (warp == 15) {
        // ---------------------------------------------------- transposer
        for (int j = 0; j < ntiles; ++j) {
            if (!wait_bar(bar(kBarBxEmpty), (j & 1) ^ 1, abort_flag)) break;
            bool ok = true;
            for (int q = 0; q < kBoxes && ok; ++q) {
                const int qg = j * kBoxes + q;
                const uint32_t slot = qg % kXSlots;
                if (!wait_bar(bar(kBarXFull + slot), (qg / kXSlots) & 1, abort_flag)) {
                    ok = false;
                    break;
                }
                const uint32_t xs = sbase + kOffX + slot * (kBox * 16);
#pragma unroll 2
                for (int sb = 0; sb < 8; ++sb) {
                    const uint32_t src = xs + (32 * sb + 8 * (lane >> 3) + (7 - (lane & 7))) * 16;
                    uint32_t r0, r1, r2, r3;
                    asm volatile(
                        "ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
                        : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
                        : "r"(src)
                        : "memory");
                    const int c = lane & 7, mq = lane >> 3;
                    const int tb = 32 * q + 4 * sb + mq;      // 8-token block in the tile
                    const int n = tb >> 3, kb = 7 - (tb & 7);
                    const uint32_t dst =
                        sbase + kOffBx + c * kBxStride + (n >> 3) * 1024 + kb * 128 + (n & 7) * 16;
                    asm volatile("stmatrix.sync.aligned.m8n8.x4.shared.b16 [%0], {%1,%2,%3,%4};" ::"r"(
                                     dst),
                                 "r"(r0), "r"(r1), "r"(r2), "r"(r3)
                                 : "memory");
                }
                __syncwarp();
                if (lane == 0) bar_arrive(bar(kBarXEmpty + slot));
            }
            if (!ok) break;
            fence_async_smem();
            __syncwarp();
            if (lane == 0) bar_arrive(bar(kBarBxFull));
        }
    } else if (warp == 7) {
        // ---------------------------------------------------- MMA issuer
        if (lane == 0) {
            for (int j = 0; j < ntiles; ++j) {
                const int buf = j & 1, use = j >> 1;
                if (!wait_bar(bar(kBarBxFull), j & 1, abort_flag)) break;
                if (!wait_bar(bar(kBarDEmpty + buf), (use & 1) ^ 1, abort_flag)) break;
                tc_fence_after();
                for (int c = 0; c < kDG; ++c) {
                    const uint32_t d = tmem + buf * 256 + c * 32;
                    const uint32_t a0 = sbase + kOffAtw + c * kAtwStride;
                    const uint32_t b0 = sbase + kOffBx + c * kBxStride;
#pragma unroll
                    for (int kk = 0; kk < 4; ++kk)
                        umma_f16(d, umma_desc(a0 + kk * 256, 128, 1024),
                                 umma_desc(b0 + kk * 256, 128, 1024), kk > 0);
                    umma_commit(bar(kBarTwDone + buf * 8 + c));
                }
                umma_commit(bar(kBarBxEmpty));
                bool ok = true;
                for (int c = 0; c < kDG; ++c) {
                    if (!wait_bar(bar(kBarSFull + c), j & 1, abort_flag)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t d = tmem + buf * 256 + c * 32;
                    const uint32_t a0 = sbase + kOffAu + c * kAuStride;
                    const uint32_t b0 = sbase + kOffBs + c * kBsStride;
#pragma unroll
                    for (int kk = 0; kk < 2; ++kk)
                        umma_f16(d, umma_desc(a0 + kk * 256, 128, 512),
                                 umma_desc(b0 + kk * 2 * kBsLbo, kBsLbo, kBsSbo), 1);
                }
                if (!ok) break;
                umma_commit(bar(kBarUDone + buf));
            }
            // Drain: all issued MMAs complete before TMEM is released.
            umma_commit(bar(kBarFinal));
            const uint64_t t0 = globaltimer();
            while (!bar_try(bar(kBarFinal), 0))
                if (globaltimer() - t0 > kWaitLimitNs) break;
        }
        __syncwarp();
    } else if (warp == 11) {
        // ---------------------------------------------------- y store issuer
        for (int j = 0; j < ntiles; ++j) {
            bool ok = true;
            for (int nb = 0; nb < 4; ++nb) {
                const int ng = j * 4 + nb;
                const uint32_t slot = ng % kYSlots;
                if (!wait_bar(bar(kBarYFull + slot), (ng / kYSlots) & 1, abort_flag)) {
                    ok = false;
                    break;
                }
                const uint32_t ys = sbase + kOffY + slot * 8192;
                for (int h = 0; h < 2; ++h) {
                    const int64_t start = args.t0 + (int64_t)j * kTile + nb * 512 + h * kBox;
                    if (start >= 0) {
                        if (lane == 0) tma_store_3d(&tmap_y, ys + h * 4096, d0, (int)start, b);
                    } else if (start + kBox > 0) {
                        // Partially before t = 0: plain 16-byte stores of the rows t >= 0.
                        const uint8_t *src = smem + kOffY + slot * 8192 + h * 4096;
                        for (int rr = (int)(-start) + lane; rr < kBox; rr += 32) {
                            const int64_t t = start + rr;
                            *reinterpret_cast<uint4 *>(args.y + ((int64_t)b * args.L + t) * D + d0) =
                                *reinterpret_cast<const uint4 *>(src + rr * 16);
                        }
                    }
                }
                if (lane == 0) {
                    tma_store_commit();
                    tma_store_wait_read();
                }
                __syncwarp();
                if (lane == 0) bar_arrive(bar(kBarYEmpty + slot));
            }
            if (!ok) break;
        }
        if (lane == 0) tma_store_wait_all();
    } else if (quarter == 2) {
        // ---------------------------------------------------- scan (rows 64..95)
        const int sidx = warp >> 2;                 // 0..3 -> channels 2 sidx, 2 sidx + 1
        const int r = lane, m = r >> 1, ri = r & 1;
        float2 LC[2], carry[2];
        for (int cc = 0; cc < 2; ++cc) {
            const int pm = (d0 + 2 * sidx + cc) * kModes + m;
            LC[cc] = lambda_pow(args.decay[pm], args.freq[pm], (float)kC);
            carry[cc] = make_float2(0.0f, 0.0f);
        }
        for (int j = 0; j < ntiles; ++j) {
            const int buf = j & 1, use = j >> 1;
            bool ok = true;
            for (int cc = 0; cc < 2; ++cc) {
                const int c = 2 * sidx + cc;
                if (!wait_bar(bar(kBarTwDone + buf * 8 + c), use & 1, abort_flag)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                uint32_t v[32];
                RLM_TMEM_LD32(tmem + (64u << 16) + buf * 256 + c * 32, v);
                tmem_wait_ld();
                uint8_t *bs = smem + kOffBs + c * kBsStride + (m / 4) * kBsLbo + ((2 * m) % 8) * 2;
                float2 S = carry[cc];
                const float2 lc = LC[cc];
#pragma unroll
                for (int n = 0; n < kNT; ++n) {
                    const float mine = __uint_as_float(v[n]);
                    const float other = __shfl_xor_sync(0xffffffffu, mine, 1);
                    const float2 Ln = ri ? make_float2(other, mine) : make_float2(mine, other);
                    if ((n >> 4) == ri)
                        *reinterpret_cast<uint32_t *>(bs + (n >> 3) * kBsSbo + (n & 7) * 16) =
                            pack_bf16x2(S.x, S.y);
                    S = cfma(lc, S, Ln);
                }
                carry[cc] = S;
                if (j == ntiles - 1 && args.state_out && ri == 0)
                    args.state_out[((int64_t)b * D + d0 + c) * kModes + m] = S;
                fence_async_smem();
                tc_fence_before();
                __syncwarp();
                if (lane == 0) bar_arrive(bar(kBarSFull + c));
            }
            if (!ok) break;
            if (lane == 0) bar_arrive(bar(kBarDEmpty + buf));
        }
    } else {
        // ---------------------------------------------------- epilogue (rows 0..63)
        const int e = warp >> 2;                     // 0..3: chunk pair within a block
        const int i = 32 * quarter + lane;           // position within the chunk
        for (int j = 0; j < ntiles; ++j) {
            const int buf = j & 1, use = j >> 1;
            if (!wait_bar(bar(kBarUDone + buf), use & 1, abort_flag)) break;
            tc_fence_after();
            bool ok = true;
            for (int nb = 0; nb < 4; ++nb) {
                const int ng = j * 4 + nb;
                const uint32_t slot = ng % kYSlots;
                const int n0 = 8 * nb + 2 * e;
                uint32_t v[kDG][2];
#pragma unroll
                for (int c = 0; c < kDG; ++c)
                    tmem_ld2(tmem + ((uint32_t)(32 * quarter) << 16) + buf * 256 + c * 32 + n0,
                             v[c][0], v[c][1]);
                tmem_wait_ld();
                if (!wait_bar(bar(kBarYEmpty + slot), ((ng / kYSlots) & 1) ^ 1, abort_flag)) {
                    ok = false;
                    break;
                }
                uint8_t *ys = smem + kOffY + slot * 8192;
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    uint4 row;
                    row.x = pack_bf16x2(__uint_as_float(v[0][h]), __uint_as_float(v[1][h]));
                    row.y = pack_bf16x2(__uint_as_float(v[2][h]), __uint_as_float(v[3][h]));
                    row.z = pack_bf16x2(__uint_as_float(v[4][h]), __uint_as_float(v[5][h]));
                    row.w = pack_bf16x2(__uint_as_float(v[6][h]), __uint_as_float(v[7][h]));
                    *reinterpret_cast<uint4 *>(ys + ((2 * e + h) * 64 + i) * 16) = row;
                }
                fence_async_smem();
                __syncwarp();
                if (lane == 0) bar_arrive(bar(kBarYFull + slot));
            }
            if (!ok) break;
            tc_fence_before();
            __syncwarp();
            if (lane == 0) bar_arrive(bar(kBarDEmpty + buf));
        }
    }

    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 7)
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem),
                     "r"(kTmemCols));
}

// ------------------------------------------------------------ host side
using EncodeTiledFn = CUresult (*)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *,
                                   const cuuint64_t *, const cuuint64_t *, const cuuint32_t *,
                                   const cuuint32_t *, CUtensorMapInterleave, CUtensorMapSwizzle,
                                   CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
    static EncodeTiledFn fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                             &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiledFn>(p);
    });
    return fn;
}

// 3-D map over a [B][L][D] bf16 field: dims (D, L, B), box (8, 256, 1).
bool make_field_map(CUtensorMap *map, const void *ptr, int64_t B, int64_t L, int D) {
    EncodeTiledFn fn = encode_fn();
    if (!fn) return false;
    cuuint64_t dims[3] = {(cuuint64_t)D, (cuuint64_t)L, (cuuint64_t)B};
    cuuint64_t strides[2] = {(cuuint64_t)D * 2, (cuuint64_t)L * D * 2};
    cuuint32_t box[3] = {(cuuint32_t)kDG, (cuuint32_t)kBox, 1};
    cuuint32_t estr[3] = {1, 1, 1};
    return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void *>(ptr), dims, strides, box,
              estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE,
              CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace

bool tc_prefill_supported(int64_t B, int64_t L, int D, int M, rlm_dtype dt) {
    return dt == RLM_BF16 && M == kModes && D % kDG == 0 && B >= 1 && B <= 65535 && L >= 1 &&
           L <= ((int64_t)1 << 31) - kTile && D / kDG <= 65535;
}

size_t tc_prefill_ws_bytes(int64_t, int64_t, int, int) { return 0; }

cudaError_t tc_prefill(const void *x, void *y, int64_t B, int64_t L, int D, int M,
                       const float *decay, const float *freq, const float *amp,
                       const float *phase, float *state_out, float *coef_out, void *,
                       cudaStream_t st) {
    (void)M;
    CUtensorMap mx, my;
    if (!make_field_map(&mx, x, B, L, D) || !make_field_map(&my, y, B, L, D))
        return cudaErrorInvalidValue;
    static std::mutex mu;
    static std::vector<int> configured;
    int dev = 0;
    cudaGetDevice(&dev);
    {
        std::lock_guard<std::mutex> lock(mu);
        if ((int)configured.size() <= dev) configured.resize(dev + 1, 0);
        if (!configured[dev]) {
            cudaError_t e = cudaFuncSetAttribute(k_prefill_tc, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                 kSmemBytes);
            if (e != cudaSuccess) return e;
            configured[dev] = 1;
        }
    }
    TcArgs a;
    a.decay = decay;
    a.freq = freq;
    a.amp = amp;
    a.phase = phase;
    a.state_out = reinterpret_cast<float2 *>(state_out);
    a.coef_out = reinterpret_cast<float4 *>(coef_out);
    a.y = static_cast<__nv_bfloat16 *>(y);
    a.L = L;
    a.D = D;
    a.ntiles = (int)((L + kTile - 1) / kTile);
    a.t0 = L - (int64_t)a.ntiles * kTile;
    dim3 grid((unsigned)(D / kDG), (unsigned)B);
    k_prefill_tc<<<grid, kThreads, kSmemBytes, st>>>(mx, my, a);
    count_launches(1);
    return cudaGetLastError();
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
