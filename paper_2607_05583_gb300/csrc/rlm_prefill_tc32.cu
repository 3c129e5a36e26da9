// rlm_prefill_tc32.cu -- tcgen05 tensor-core prefill for fp32 I/O, M <= 16 modes.
//
// The same chunked scan as the bf16 kernel (Sec. 3.2, Eq. 2; chunks of C = 64
// tokens, 2048-token tiles of N = 32 chunks):
//
//   D[0:64, n]   = T  (64x64)  X_n      Toeplitz block, T[p][q] = K[p-q]
//   D[64:96, n]  = W  (32x64)  X_n      local end state, (Re, Im) of 16 modes
//   D[0:64, n]  += U  (64x32)  S_{n-1}  up-projection of the carried state
//
// with fp32 operands represented as pairs of bf16 values, v = hi + lo, hi the
// bf16 rounding of v and lo the bf16 rounding of v - hi (16 significant bits in
// all).  Each product is accumulated in fp32 from three bf16 MMAs,
//
//   A B  ~  A_hi B_hi + A_hi B_lo + A_lo B_hi,
//
// dropping A_lo B_lo (relative size 2^-16): the drive X, the tables T, W, U and
// the carried state S are all split this way, so the contraction keeps about
// 16 bits, against a tolerance of 1e-4.  The carry between chunks, the
// accumulators and the output stay fp32.
//
// An initial state s_in (L a multiple of 64, so token 0 opens chunk n0 of tile
// 0) enters as the state carried into chunk n0: the up-projection then gives
// lambda^(i+1) s_in at its positions i and the scan carries lambda^64 s_in on.
//
// A CTA owns one batch row and a group of DG = 4 channels.  An fp32 token row of
// 4 channels is 16 bytes, the same slice of the [B][L][D] row as the bf16
// kernel's 8 channels, so loads and stores have the bf16 kernel's granularity
// with twice its bytes per token-channel.
// TMEM (512 columns): two accumulator buffers (tile v uses buffer v & 1), channel
// c's at columns 128 b + 32 c (32 chunks); its A operands hi / lo (128 lanes x 32
// columns of packed bf16 pairs) at columns 256 + 64 c and 256 + 64 c + 32.  With
// two buffers the chain of one tile (the Toeplitz/state MMAs) runs while the
// scan, up-projection and epilogue of the tile before still hold the other.
// Rows of channel c's accumulator (= TMEM lanes): its Toeplitz rows (positions
// 0-31, 32-63) in quarters 2, 3 for channels 0, 1 and in quarters 0, 1 for
// channels 2, 3; its 32 state rows (2 m + ri) in quarter c; zeros in the last
// quarter.  So every quarter holds the Toeplitz rows of two channels and the
// state rows of one.
//
// Warp roles (22 warps):
//   0-7    epilogue: warp (q = warp % 4, h = warp / 4) reads position
//          32 (q % 2) + lane of the two channels whose Toeplitz rows are in
//          quarter q, chunks 16h .. 16h+15, into the 8-byte half of each 16-byte
//          y row.
//   8-11   scan: the warp of quarter q carries channel q.
//   12-15  transposers (ring slot s: warp 12 + s mod 4): fp32 token rows -> hi / lo K-major
//          B operands.
//   16     TMA producer; 17 TMA store issuer and TMEM allocation.
//   18-21  MMA issue for one channel each: the thread polls the inputs of the
//          next Toeplitz/state chain and of the next up-projection and issues
//          whichever is ready.
// Warps 0-7 first build the per-channel constants.
//
// Every wait is bounded (about 2 s): the waiting thread then sets a shared abort
// flag and the device status word (RLM_ERR_TIMEOUT); all roles leave their loops,
// drain what they issued and the CTA frees its TMEM and returns.
#include <cuda.h>

#include <algorithm>
#include <mutex>
#include <vector>

#include "rlm_device.cuh"
#include "rlm_internal.h"

namespace rlm {

// Device status word of this kernel: RLM_OK, or RLM_ERR_TIMEOUT once a bounded
// wait expired.
__device__ int g_tc32_status = 0;

namespace {

constexpr int kC = 64;                 // chunk length
constexpr int kNT = 32;                // chunks per tile = MMA N
constexpr int kTile = kC * kNT;        // 2048 tokens
constexpr int kDG = 4;                 // channels per CTA
constexpr int kModes = 16;             // modes per channel in the tables (M <= 16 is padded)
constexpr int kBox = 256;              // TMA box rows (16 bytes each)
constexpr int kBoxes = kTile / kBox;   // 8 per tile
constexpr int kXSlots = 15;            // x ring depth (boxes)
constexpr int kYRows = 512;            // rows per y ring slot (8 chunks)
constexpr int kYPerTile = kTile / kYRows;
constexpr int kYSlots = 6;
constexpr int kWarps = 22;
constexpr int kThreads = kWarps * 32;
constexpr int kTmemCols = 512;
constexpr int kTmemA = 256;            // first TMEM column of the A operands
constexpr long long kWaitLimitCycles = 4000000000ll;  // about 2 s at 2 GHz
constexpr int kTransposers = 4;

// Shared memory map (bytes from a 1024-aligned base).
// U tables (hi, then lo): 64 rows x 64 B per channel, in the order of channels
// 2, 3, 0, 1.  The up-projection reads a 128-row A operand whose 64 real rows
// must meet the channel's Toeplitz lanes: rows 0-63 for channels 2, 3 (start at
// the table), rows 64-127 for channels 0, 1 (start one table earlier).  The
// other 64 rows read a neighbouring table into lanes nobody reads afterwards.
constexpr int kAuStride = 4096;
constexpr int kAuPart = kDG * kAuStride;           // 16 KB: the hi tables, then the lo tables
// B operand of a channel's drives (one part): K = 64 positions (reversed) x
// N = 32 chunks, K-major core matrices of 8 chunks x 16 B.  The parts are 4096 +
// 16 bytes apart, so the 8 rows one stmatrix writes (hi and lo of the 4
// channels) land in distinct banks.
constexpr int kBxLbo = 128, kBxSbo = 1024;
constexpr int kBxPart = 4 * kBxSbo + 16;            // 4112 bytes per channel and part
constexpr int kBxBuf = kDG * 2 * kBxPart;           // 32896: [channel][hi, lo]
// Carried-state operand (one part): K = 32 (Re, Im of 16 modes) x N = 32 chunks.
// LBO 144 spreads a chunk's 16 mode words over distinct banks; the lo part sits
// 16 banks after the hi part, so the two lanes of a mode write disjoint banks.
constexpr int kBsLbo = 144, kBsSbo = 576, kBsPart = 4 * kBsSbo + 64;
static_assert((kBsPart / 4) % 32 == 16, "hi and lo parts must use disjoint banks");
constexpr int kBsStride = 2 * kBsPart;              // per channel: hi, lo
constexpr int kOffAu = 0;
constexpr int kOffBx = kOffAu + 2 * kAuPart;                 // 32768
constexpr int kOffBs = kOffBx + 2 * kBxBuf;                  // 106496
constexpr int kOffX = kOffBs + kDG * kBsStride;
constexpr int kOffY = kOffX + kXSlots * kBox * 16;
constexpr int kOffBar = kOffY + kYSlots * kYRows * 16;
constexpr int kNumBars = 96;
constexpr int kOffMisc = kOffBar + kNumBars * 8;
constexpr int kSmemBytes = kOffMisc + 64 + 1024;             // + alignment slack
static_assert(kOffX % 128 == 0 && kOffY % 128 == 0, "TMA buffers need 128-byte alignment");
static_assert(kSmemBytes <= 232448, "shared memory budget");
// Prologue tables, in buffers no other role touches before the prologue ends:
// the W rows (hi, lo) in the y ring, word-major with rows innermost (stride 33
// words); the Toeplitz pair tables (hi, lo) and the partial sums of K in the
// carried-state buffers.
constexpr int kWtabStride = 33;
constexpr int kWtabPart = kDG * 32 * kWtabStride;      // words per part
constexpr int kTpairStride = 144;                      // words per channel and part: P0 at 0, P1 at 80
constexpr int kOffWtab = kOffY;
constexpr int kOffTpair = kOffBs;                      // [part][4 ch][144 words]
constexpr int kOffKp = kOffTpair + 2 * kDG * kTpairStride * 4;  // [2 halves][4 ch][64] fp32
static_assert(2 * kWtabPart * 4 <= kYSlots * kYRows * 16, "W tables do not fit the y ring");
static_assert(kOffKp + 2 * kDG * 64 * 4 <= kOffX, "prologue tables do not fit");
// Named barrier for the 8 warps that build the constants.
constexpr int kPrologueBarrier = 1;
constexpr int kPrologueThreads = 256;

// Barrier indices.
constexpr int kBarXFull = 0;                    // [kXSlots]
constexpr int kBarXEmpty = kXSlots;             // [kXSlots]
constexpr int kBarBxFull = 2 * kXSlots;         // [2]
constexpr int kBarBxEmpty = kBarBxFull + 2;     // [2]: released by the 4 scan warps
// Per channel c and accumulator buffer b (index 2 c + b), each completing once
// per tile of its buffer:
constexpr int kBarTwDone = kBarBxEmpty + 2;     // [4][2]: Toeplitz/state MMAs done
constexpr int kBarSFull = kBarTwDone + 2 * kDG; // [4][2]: carried states written
constexpr int kBarUDone = kBarSFull + 2 * kDG;  // [4][2]: up-projection done
constexpr int kBarDEmpty = kBarUDone + 2 * kDG; // [4][2]: accumulator read out
constexpr int kBarYFull = kBarDEmpty + 2 * kDG; // [kYSlots]
constexpr int kBarYEmpty = kBarYFull + kYSlots; // [kYSlots]
constexpr int kBarFinal = kBarYEmpty + kYSlots; // [4]
constexpr int kBarConsts = kBarFinal + kDG;     // the A operands and U tables are built
static_assert(kBarConsts + 1 <= kNumBars, "too many barriers");

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
// Non-blocking test of an mbarrier phase (for a thread that polls several).
__device__ __forceinline__ bool bar_test(uint32_t bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{ .reg .pred p; mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2; selp.u32 %0, 1, 0, p; }"
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

// Bounded wait on an mbarrier phase.  Returns false if this CTA aborted.  The
// bound is measured with the SM cycle counter, read every 1024 failed polls.
__device__ __forceinline__ bool wait_bar(uint32_t bar, uint32_t parity, volatile int *abort_flag) {
    if (bar_try(bar, parity)) return true;
    long long t0 = 0;
    for (uint32_t it = 1;; ++it) {
        if (bar_try(bar, parity)) return true;
        if ((it & 1023u) == 0) {
            if (*abort_flag) return false;
            const long long now = clock64();
            if (t0 == 0) {
                t0 = now;
            } else if (now - t0 > kWaitLimitCycles) {
                *abort_flag = 1;
                atomicExch(&g_tc32_status, (int)RLM_ERR_TIMEOUT);
                return false;
            }
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
// D (TMEM) (+)= A (shared memory) * B (shared memory)^T.
__device__ __forceinline__ void umma_ss(uint32_t d_tmem, uint64_t a, uint64_t b, uint32_t idesc,
                                        uint32_t accum) {
    asm volatile(
        "{ .reg .pred p; setp.ne.b32 p, %4, 0;\n"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p; }" ::"r"(d_tmem),
        "l"(a), "l"(b), "r"(idesc), "r"(accum)
        : "memory");
}
// D (TMEM) (+)= A (TMEM: lane = row, column c = K elements 2c, 2c+1) * B (smem)^T.
__device__ __forceinline__ void umma_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t b,
                                        uint32_t idesc, uint32_t accum) {
    asm volatile(
        "{ .reg .pred p; setp.ne.b32 p, %4, 0;\n"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p; }" ::"r"(d_tmem),
        "r"(a_tmem), "l"(b), "r"(idesc), "r"(accum)
        : "memory");
}
__device__ __forceinline__ void umma_commit(uint32_t bar) {
    asm volatile(
        "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
        : "memory");
}
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, uint32_t (&v)[16]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,"
        "%14,%15}, [%16];"
        : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]),
          "=r"(v[7]), "=r"(v[8]), "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]), "=r"(v[13]),
          "=r"(v[14]), "=r"(v[15])
        : "r"(taddr));
}
__device__ __forceinline__ void tmem_ld1(uint32_t taddr, uint32_t &v) {
    asm volatile("tcgen05.ld.sync.aligned.32x32b.x1.b32 {%0}, [%1];" : "=r"(v) : "r"(taddr));
}
__device__ __forceinline__ void tmem_wait_ld() {
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_st32(uint32_t taddr, const uint32_t (&w)[32]) {
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,"
        "%13,%14,%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};" ::"r"(
            taddr),
        "r"(w[0]), "r"(w[1]), "r"(w[2]), "r"(w[3]), "r"(w[4]), "r"(w[5]), "r"(w[6]), "r"(w[7]),
        "r"(w[8]), "r"(w[9]), "r"(w[10]), "r"(w[11]), "r"(w[12]), "r"(w[13]), "r"(w[14]),
        "r"(w[15]), "r"(w[16]), "r"(w[17]), "r"(w[18]), "r"(w[19]), "r"(w[20]), "r"(w[21]),
        "r"(w[22]), "r"(w[23]), "r"(w[24]), "r"(w[25]), "r"(w[26]), "r"(w[27]), "r"(w[28]),
        "r"(w[29]), "r"(w[30]), "r"(w[31])
        : "memory");
}
__device__ __forceinline__ void tmem_wait_st() {
    asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
    uint32_t r;
    asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(hi), "f"(lo));
    return r;
}
// The bf16 high part of v and the bf16 rounding of the remainder.
__device__ __forceinline__ float bf16_hi(float v) { return __bfloat162float(__float2bfloat16_rn(v)); }
// Packed (a, b) pairs of the high parts and of the low parts.
__device__ __forceinline__ void split_pack(float a, float b, uint32_t &hi, uint32_t &lo) {
    const float ah = bf16_hi(a), bh = bf16_hi(b);
    hi = pack_bf16x2(ah, bh);
    lo = pack_bf16x2(a - ah, b - bh);
}

// Instruction descriptor, kind::f16: fp32 accumulate, bf16 A and B, both K-major,
// M = 128, N = kNT.
constexpr uint32_t kIdesc = (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(kNT >> 3) << 17) |
                            ((uint32_t)(128 >> 4) << 24);

__device__ __forceinline__ int au_slot(int c) { return (c + 2) & 3; }
// First byte (from a U table area) of channel c's 128-row up-projection operand.
__device__ __forceinline__ int au_operand(int c) { return au_slot(c) * kAuStride - (c < 2 ? kAuStride : 0); }

struct Tc32Args {
    const float *decay, *freq, *amp, *phase;
    const float2 *state_in;  // nullable, [B][D][M]; L % 64 == 0 when set
    float2 *state_out;   // nullable, [B][D][M]
    float4 *coef_out;    // nullable, [D][M]
    float *y;            // for the plain stores of boxes that start before t = 0
    int64_t L;
    int D;
    int M;               // modes, 1..16; modes M..15 are padding (amplitude 0, never stored)
    int ntiles;
    int64_t t0;          // first token of tile 0 (<= 0): tiles end exactly at L-1
    int B, bpc;          // grid y covers batch rows in groups of bpc (kPacked)
};

enum : int { kPlain = 0, kPacked = 2 };

template <int kMode>
__global__ void __launch_bounds__(kThreads, 1)
    k_prefill_tc32(const __grid_constant__ CUtensorMap tmap_x, const __grid_constant__ CUtensorMap tmap_y,
                   const Tc32Args args) {
    constexpr bool kPack = kMode == kPacked;
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    uint8_t *smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
    const uint32_t sbase = smem_u32(smem);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int g = blockIdx.x;
    const int b = kPack ? (int)blockIdx.y * args.bpc : (int)blockIdx.y;   // the CTA's (first) batch row
    const int d0 = g * kDG;
    const int D = args.D;
    // Tiles of the CTA: packed, those of its batch rows, row after row.
    const int nV = kPack ? min(args.bpc, args.B - b) * args.ntiles : args.ntiles;
    auto real_tile = [&](int v) { return kPack ? v % args.ntiles : v; };
    auto row_of = [&](int v) { return kPack ? b + v / args.ntiles : b; };
    // Constant builders (warps 0-7) issue their parameter loads first.
    const bool builder = warp < 8;
    const int ptid = tid;                        // 0..255 for the builders
    float p_decay = 0.0f, p_freq = 0.0f, p_amp = 0.0f, p_phase = 0.0f;
    if (builder && ((ptid >> 2) & 15) < args.M) {
        const int pm = (d0 + (ptid >> 6)) * args.M + ((ptid >> 2) & 15);
        p_decay = args.decay[pm];
        p_freq = args.freq[pm];
        p_amp = args.amp[pm];
        p_phase = args.phase[pm];
    }
    uint64_t *bars = reinterpret_cast<uint64_t *>(smem + kOffBar);
    auto bar = [&](int i) { return smem_u32(bars + i); };
    volatile int *abort_flag = reinterpret_cast<volatile int *>(smem + kOffMisc);
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(smem + kOffMisc + 16);

    if (tid == 0) {
        *abort_flag = 0;
        for (int i = 0; i < kXSlots; ++i) {
            bar_init(bar(kBarXFull + i), 1);
            bar_init(bar(kBarXEmpty + i), 1);
        }
        for (int i = 0; i < 2; ++i) {
            bar_init(bar(kBarBxFull + i), kBoxes);
            bar_init(bar(kBarBxEmpty + i), kDG);
        }
        for (int i = 0; i < 2 * kDG; ++i) {
            bar_init(bar(kBarTwDone + i), 1);
            bar_init(bar(kBarSFull + i), 1);
            bar_init(bar(kBarUDone + i), 1);
            bar_init(bar(kBarDEmpty + i), 4);
        }
        for (int i = 0; i < kDG; ++i) bar_init(bar(kBarFinal + i), 1);
        for (int i = 0; i < kYSlots; ++i) {
            bar_init(bar(kBarYFull + i), 4);
            bar_init(bar(kBarYEmpty + i), 1);
        }
        bar_init(bar(kBarConsts), 1);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (warp == 17) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                         smem_u32(tmem_slot)),
                     "r"(kTmemCols));
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    // The producer fills the whole ring before the constants are built.
    const int total_boxes = nV * kBoxes;
    int issued = 0;
    if (warp == 16 && lane == 0) {
        for (; issued < total_boxes && issued < kXSlots; ++issued) {
            const int jt = real_tile(issued / kBoxes), q = issued % kBoxes, bq = row_of(issued / kBoxes);
            const uint32_t slot = issued % kXSlots;
            bar_expect_tx(bar(kBarXFull + slot), kBox * 16);
            tma_load_3d(sbase + kOffX + slot * (kBox * 16), &tmap_x, d0,
                        (int)(args.t0 + (int64_t)jt * kTile + q * kBox), bq, bar(kBarXFull + slot));
        }
    }

    // ---------------------------------------------------- per-channel constants
    // Stage 1: thread (c, m, qn) runs the powers lambda^n, n in [16 qn, 16 qn + 16),
    // of mode m of channel c: the U rows (Re, -Im of c lambda^(n+1), hi and lo),
    // the W-row words (lambda^n packed in pairs of n, hi and lo), and Re(c lambda^n)
    // summed over the eight modes of its warp into Kp[half][c][n].
    if (builder) {
        const int c = ptid >> 6, m = (ptid >> 2) & 15, qn = ptid & 3;
        const int pm = (d0 + c) * args.M + m;
        const float2 lam = lambda_pow(p_decay, p_freq, 1.0f);
        const float2 cf = mode_coef(p_amp, p_phase);
        if (args.coef_out && b == 0 && qn == 0 && m < args.M)
            args.coef_out[pm] = make_float4(lam.x, lam.y, cf.x, cf.y);
        float2 pw = lambda_pow(p_decay, p_freq, (float)(16 * qn));
        uint8_t *auh = smem + kOffAu + au_slot(c) * kAuStride + (m / 4) * 128 + ((2 * m) % 8) * 2;
        uint8_t *aul = auh + kAuPart;
        uint32_t wreh[8], wrel[8], wimh[8], wiml[8];
        float kv[16];
#pragma unroll
        for (int e = 0; e < 16; ++e) {
            const int n = 16 * qn + e;
            kv[e] = cf.x * pw.x - cf.y * pw.y;                          // Re(c lambda^n)
            const float2 nx = cmul(pw, lam);                             // lambda^(n+1)
            if ((e & 1) == 0) {
                split_pack(pw.x, nx.x, wreh[e >> 1], wrel[e >> 1]);
                split_pack(pw.y, nx.y, wimh[e >> 1], wiml[e >> 1]);
            }
            const float2 q = cmul(cf, nx);                               // c lambda^(n+1)
            uint32_t uh, ul;
            split_pack(q.x, -q.y, uh, ul);
            *reinterpret_cast<uint32_t *>(auh + (n / 8) * 512 + (n % 8) * 16) = uh;
            *reinterpret_cast<uint32_t *>(aul + (n / 8) * 512 + (n % 8) * 16) = ul;
            pw = nx;
        }
        uint32_t *wt = reinterpret_cast<uint32_t *>(smem + kOffWtab) + (c * 32 + 8 * qn) * kWtabStride + 2 * m;
#pragma unroll
        for (int k = 0; k < 8; ++k) {
            wt[k * kWtabStride] = wreh[k];
            wt[k * kWtabStride + 1] = wimh[k];
            wt[kWtabPart + k * kWtabStride] = wrel[k];
            wt[kWtabPart + k * kWtabStride + 1] = wiml[k];
        }
#pragma unroll
        for (int e = 0; e < 16; ++e) {
            float v = kv[e];
            v += __shfl_xor_sync(0xffffffffu, v, 4);
            v += __shfl_xor_sync(0xffffffffu, v, 8);
            v += __shfl_xor_sync(0xffffffffu, v, 16);
            kv[e] = v;
        }
        if ((lane >> 2) == 0) {
            float *kp = reinterpret_cast<float *>(smem + kOffKp) + ((m >> 3) * kDG + c) * 64 + 16 * qn;
#pragma unroll
            for (int e = 0; e < 16; ++e) kp[e] = kv[e];
        }
    }
    if (builder) asm volatile("bar.sync %0, %1;" ::"n"(kPrologueBarrier), "n"(kPrologueThreads) : "memory");
    // Stage 2: K[c][n] = Kp[0][c][n] + Kp[1][c][n] (Eq. 1 at integer lags), as
    // zero-padded pair tables kz(i) = K[i - 63] (0 for i < 63), hi and lo parts:
    // P0[c][i] = (kz(2i), kz(2i+1)), P1[c][i] = (kz(2i+1), kz(2i+2)).
    if (builder) {
        const float *kp = reinterpret_cast<const float *>(smem + kOffKp);
        const int c = ptid >> 6, i = ptid & 63;
        auto kz = [&](int idx) -> float {
            const int n = idx - 63;
            return (n >= 0 && n < 64) ? kp[c * 64 + n] + kp[(kDG + c) * 64 + n] : 0.0f;
        };
        uint32_t *tph = reinterpret_cast<uint32_t *>(smem + kOffTpair) + c * kTpairStride;
        uint32_t *tpl = tph + kDG * kTpairStride;
        split_pack(kz(2 * i), kz(2 * i + 1), tph[i], tpl[i]);
        split_pack(kz(2 * i + 1), kz(2 * i + 2), tph[80 + i], tpl[80 + i]);
    }
    if (builder) asm volatile("bar.sync %0, %1;" ::"n"(kPrologueBarrier), "n"(kPrologueThreads) : "memory");
    // Stage 3: the A operands into TMEM.  Warp (quarter q, rank e) writes lanes
    // 32 q + lane of channels e and e + 2, both parts:
    //   Toeplitz quarters: T[p][p'] = K[p + p' - 63] for position p = 32 (q % 2) + lane;
    //   quarter c:         W[k][p'] = (Re, Im) lambda_m^p' for state row k = lane;
    //   the remaining quarter: zero.
    if (builder) {
        const int q = warp & 3, e = warp >> 2;
        for (int cc = 0; cc < 2; ++cc) {
            const int c = e + 2 * cc;
            for (int part = 0; part < 2; ++part) {
                uint32_t w[32];
                if ((q >> 1) == (c < 2 ? 1 : 0)) {
                    const int pos = 32 * (q & 1) + lane;
                    const uint32_t *tp = reinterpret_cast<const uint32_t *>(smem + kOffTpair) +
                                         (part * kDG + c) * kTpairStride + ((pos & 1) ? 80 + (pos >> 1) : (pos >> 1));
#pragma unroll
                    for (int k = 0; k < 32; ++k) w[k] = tp[k];
                } else if (q == c) {
                    const uint32_t *wt = reinterpret_cast<const uint32_t *>(smem + kOffWtab) + part * kWtabPart +
                                         c * 32 * kWtabStride + lane;
#pragma unroll
                    for (int k = 0; k < 32; ++k) w[k] = wt[k * kWtabStride];
                } else {
#pragma unroll
                    for (int k = 0; k < 32; ++k) w[k] = 0u;
                }
                tmem_st32(tmem + ((uint32_t)(32 * q) << 16) + kTmemA + c * 64 + part * 32, w);
            }
        }
        tmem_wait_st();
        fence_async_smem();
        tc_fence_before();
        asm volatile("bar.sync %0, %1;" ::"n"(kPrologueBarrier), "n"(kPrologueThreads) : "memory");
        tc_fence_after();
        if (ptid == 0) bar_arrive(bar(kBarConsts));
    }

    const int quarter = warp & 3;
    if (warp == 16) {
        // ---------------------------------------------------- TMA producer
        if (lane == 0) {
            for (; issued < total_boxes; ++issued) {
                const int jt = real_tile(issued / kBoxes), q = issued % kBoxes, bq = row_of(issued / kBoxes);
                const uint32_t slot = issued % kXSlots;
                const uint32_t fill = issued / kXSlots;
                if (!wait_bar(bar(kBarXEmpty + slot), (fill & 1) ^ 1, abort_flag)) break;
                bar_expect_tx(bar(kBarXFull + slot), kBox * 16);
                tma_load_3d(sbase + kOffX + slot * (kBox * 16), &tmap_x, d0,
                            (int)(args.t0 + (int64_t)jt * kTile + q * kBox), bq, bar(kBarXFull + slot));
            }
            // Drain: every issued load must land before this CTA may exit.
            const int first = issued > kXSlots ? issued - kXSlots : 0;
            for (int k = first; k < issued; ++k) {
                const uint32_t slot = k % kXSlots, fill = k / kXSlots;
                const long long t0 = clock64();
                while (!bar_try(bar(kBarXFull + slot), fill & 1))
                    if (clock64() - t0 > kWaitLimitCycles) break;
            }
        }
        __syncwarp();
    } else if (warp >= 12 && warp < 12 + kTransposers) {
        // ---------------------------------------------------- transposers (ring slot s: warp 12 + s mod 4)
        // Per 8-token block (one K group of one chunk): ldmatrix.trans of the 8
        // token rows (in reversed order, so positions come out as p' = 63 - p)
        // gives thread t the half-word k = t / 4 (half k % 2 of channel k / 2) of
        // two tokens; one shuffle with thread t ^ 4 joins the two halves into the
        // fp32 values.  The thread of the even half then holds the bf16 high parts
        // of its channel's two positions, the thread of the odd half the low
        // parts: exactly row k of an 8 x 8 matrix whose rows are (channel, part),
        // which stmatrix writes into the 8 B operands (4 channels x hi, lo).
        // Each ring slot belongs to one transposer warp, so a warp waits on a slot's
        // full barrier only after it has itself consumed the slot's previous box (a
        // parity wait must never be two phases ahead of the barrier).
        const int tw = warp - 12;
        for (int k = tw; k < total_boxes;) {
            const int kn = (k % kXSlots) + kTransposers < kXSlots ? k + kTransposers
                                                                 : k - (k % kXSlots) + kXSlots + tw;
            const int j = k / kBoxes, tq = k % kBoxes;
            const int buf = j & 1, use = j >> 1;
            const uint32_t slot = k % kXSlots;
            if (!wait_bar(bar(kBarXFull + slot), (k / kXSlots) & 1, abort_flag)) break;
            const uint32_t xs = sbase + kOffX + slot * (kBox * 16);
            uint32_t r[8][4];
#pragma unroll
            for (int sb = 0; sb < 8; ++sb) {
                const uint32_t src = xs + (32 * sb + 8 * (lane >> 3) + (7 - (lane & 7))) * 16;
                asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
                             : "=r"(r[sb][0]), "=r"(r[sb][1]), "=r"(r[sb][2]), "=r"(r[sb][3])
                             : "r"(src)
                             : "memory");
            }
            // Join the halves and split into bf16 parts (even half: hi, odd: lo).
            const bool odd = (lane >> 2) & 1;
#pragma unroll
            for (int sb = 0; sb < 8; ++sb) {
#pragma unroll
                for (int mq = 0; mq < 4; ++mq) {
                    const uint32_t mine = r[sb][mq];
                    const uint32_t other = __shfl_xor_sync(0xffffffffu, mine, 4);
                    const uint32_t lo16 = odd ? other : mine, hi16 = odd ? mine : other;
                    const float fa = __uint_as_float(__byte_perm(lo16, hi16, 0x5410));
                    const float fb = __uint_as_float(__byte_perm(lo16, hi16, 0x7632));
                    const float ha = bf16_hi(fa), hb = bf16_hi(fb);
                    r[sb][mq] = odd ? pack_bf16x2(fa - ha, fb - hb) : pack_bf16x2(ha, hb);
                }
            }
            if (!wait_bar(bar(kBarBxEmpty + buf), (use & 1) ^ 1, abort_flag)) break;
            // stmatrix row address: thread t gives row t % 8 = (channel, part) of
            // matrix t / 8, i.e. of token block 32 tq + 4 sb + t / 8.
            const int rr = lane & 7, mq = lane >> 3;
            const uint32_t bx = sbase + kOffBx + buf * kBxBuf + ((rr >> 1) * 2 + (rr & 1)) * kBxPart;
#pragma unroll
            for (int sb = 0; sb < 8; ++sb) {
                const int tb = 32 * tq + 4 * sb + mq;    // 8-token block within the tile
                const int n = tb >> 3, kb = 7 - (tb & 7);
                const uint32_t dst = bx + (n >> 3) * kBxSbo + kb * kBxLbo + (n & 7) * 16;
                asm volatile("stmatrix.sync.aligned.m8n8.x4.shared.b16 [%0], {%1,%2,%3,%4};" ::"r"(dst),
                             "r"(r[sb][0]), "r"(r[sb][1]), "r"(r[sb][2]), "r"(r[sb][3])
                             : "memory");
            }
            fence_async_smem();
            __syncwarp();
            // The x slot is released only now that stmatrix has consumed the
            // ldmatrix registers.
            if (lane == 0) {
                bar_arrive(bar(kBarXEmpty + slot));
                bar_arrive(bar(kBarBxFull + buf));
            }
            k = kn;
        }
    } else if (warp == 17) {
        // ---------------------------------------------------- y store issuer
        const int nslots = nV * kYPerTile;
        int ng = 0;
        for (; ng < nslots; ++ng) {
            const uint32_t slot = ng % kYSlots;
            if (!wait_bar(bar(kBarYFull + slot), (ng / kYSlots) & 1, abort_flag)) break;
            const uint32_t ys = sbase + kOffY + slot * (kYRows * 16);
            const int vq = ng / kYPerTile, e = ng % kYPerTile;
            const int jt = real_tile(vq), bq = row_of(vq);
            for (int h = 0; h < kYRows / kBox; ++h) {
                const int64_t start = args.t0 + (int64_t)jt * kTile + e * kYRows + h * kBox;
                if (start >= 0) {
                    if (lane == 0) tma_store_3d(&tmap_y, ys + h * (kBox * 16), d0, (int)start, bq);
                } else if (start + kBox > 0) {
                    // Partially before t = 0: plain 16-byte stores of the rows t >= 0.
                    const uint8_t *src = smem + kOffY + slot * (kYRows * 16) + h * (kBox * 16);
                    for (int rr = (int)(-start) + lane; rr < kBox; rr += 32) {
                        const int64_t t = start + rr;
                        *reinterpret_cast<uint4 *>(args.y + ((int64_t)bq * args.L + t) * D + d0) =
                            *reinterpret_cast<const uint4 *>(src + rr * 16);
                    }
                }
            }
            if (lane == 0) {
                tma_store_commit();
                asm volatile("cp.async.bulk.wait_group.read %0;" ::"n"(kYSlots - 2) : "memory");
            }
            __syncwarp();
            const int freed = ng - (kYSlots - 2);
            if (lane == 0 && freed >= 0) bar_arrive(bar(kBarYEmpty + freed % kYSlots));
        }
        if (lane == 0) {
            tma_store_wait_read();
            for (int k = ng - (kYSlots - 2); k < ng; ++k)
                if (k >= 0) bar_arrive(bar(kBarYEmpty + k % kYSlots));
            tma_store_wait_all();
        }
        __syncwarp();
    } else if (warp >= 18) {
        // ---------------------------------------------------- MMA issuer, one channel
        // Tile v uses accumulator buffer v & 1 (and B-operand buffer v & 1).  The
        // thread issues whichever is ready: the Toeplitz/state chain of tile tw
        // (hi hi + hi lo + lo hi; its B operand full and its buffer's previous tile,
        // tw - 2, read out by the epilogue) or the up-projection of tile uu (same
        // three terms) once the scan has written that tile's carried states.  tw
        // stays at most two tiles ahead of uu, so no barrier runs a phase ahead of
        // this thread.
        const int c = warp - 18;
        const uint64_t dxh = umma_desc(sbase + kOffBx + c * 2 * kBxPart, kBxLbo, kBxSbo);
        const uint64_t dxl = umma_desc(sbase + kOffBx + c * 2 * kBxPart + kBxPart, kBxLbo, kBxSbo);
        const uint64_t duh = umma_desc(sbase + kOffAu + au_operand(c), 128, 512);
        const uint64_t dul = umma_desc(sbase + kOffAu + kAuPart + au_operand(c), 128, 512);
        const uint64_t dsh = umma_desc(sbase + kOffBs + c * kBsStride, kBsLbo, kBsSbo);
        const uint64_t dsl = umma_desc(sbase + kOffBs + c * kBsStride + kBsPart, kBsLbo, kBsSbo);
        const uint32_t aH = tmem + kTmemA + c * 64, aL = aH + 32;
        constexpr uint64_t kXStep = (2 * kBxLbo) >> 4;     // 16 K elements of the drive operand
        constexpr uint64_t kSStep = (2 * kBsLbo) >> 4;     // 16 K elements of the state operand
        if (lane == 0 && wait_bar(bar(kBarConsts), 0, abort_flag)) {
            tc_fence_after();
            int tw = 0, uu = 0;
            long long t_idle = 0;
            uint32_t polls = 0;
            while (uu < nV) {
                bool progress = false;
                if (uu < tw) {
                    const int bb = uu & 1, u = uu >> 1;
                    if (bar_test(bar(kBarSFull + 2 * c + bb), u & 1)) {
                        tc_fence_after();
                        const uint32_t d = tmem + bb * 128 + c * kNT;
#pragma unroll
                        for (int kk = 0; kk < 2; ++kk) umma_ss(d, duh + kk * 16, dsh + kk * kSStep, kIdesc, 1);
#pragma unroll
                        for (int kk = 0; kk < 2; ++kk) umma_ss(d, duh + kk * 16, dsl + kk * kSStep, kIdesc, 1);
#pragma unroll
                        for (int kk = 0; kk < 2; ++kk) umma_ss(d, dul + kk * 16, dsh + kk * kSStep, kIdesc, 1);
                        umma_commit(bar(kBarUDone + 2 * c + bb));
                        ++uu;
                        progress = true;
                    }
                }
                if (tw < nV && tw < uu + 2) {
                    const int bb = tw & 1, u = tw >> 1;
                    if (bar_test(bar(kBarBxFull + bb), u & 1) &&
                        (tw < 2 || bar_test(bar(kBarDEmpty + 2 * c + bb), (u - 1) & 1))) {
                        tc_fence_after();
                        const uint64_t xo = (uint64_t)((bb * kBxBuf) >> 4);
                        const uint32_t d = tmem + bb * 128 + c * kNT;
#pragma unroll
                        for (int kk = 0; kk < 4; ++kk) umma_ts(d, aH + kk * 8, dxh + xo + kk * kXStep, kIdesc, kk > 0);
#pragma unroll
                        for (int kk = 0; kk < 4; ++kk) umma_ts(d, aH + kk * 8, dxl + xo + kk * kXStep, kIdesc, 1);
#pragma unroll
                        for (int kk = 0; kk < 4; ++kk) umma_ts(d, aL + kk * 8, dxh + xo + kk * kXStep, kIdesc, 1);
                        umma_commit(bar(kBarTwDone + 2 * c + bb));
                        ++tw;
                        progress = true;
                    }
                }
                if (progress) {
                    t_idle = 0;
                    polls = 0;
                } else if ((++polls & 255u) == 0) {
                    // Bounded like wait_bar: give up after kWaitLimitCycles without progress.
                    if (*abort_flag) break;
                    const long long now = clock64();
                    if (t_idle == 0) {
                        t_idle = now;
                    } else if (now - t_idle > kWaitLimitCycles) {
                        *abort_flag = 1;
                        atomicExch(&g_tc32_status, (int)RLM_ERR_TIMEOUT);
                        break;
                    }
                }
            }
            // Drain: all MMAs this thread issued complete before TMEM is released.
            umma_commit(bar(kBarFinal + c));
            const long long t0 = clock64();
            while (!bar_try(bar(kBarFinal + c), 0))
                if (clock64() - t0 > kWaitLimitCycles) break;
        }
        __syncwarp();
    } else if (warp >= 8 && warp < 12) {
        // ---------------------------------------------------- scan, one channel
        // The warp of quarter q owns channel q, whose 32 state rows are its TMEM
        // lanes: lane 2m + ri reads row 2m + ri (Re or Im of mode m's chunk-local
        // end state) and one shuffle brings the other component, so both lanes of
        // a mode run S_n = lambda^C S_{n-1} + L_n in fp32.  Lane 2m writes the hi
        // part of S_{n-1} into the up-projection's B operand, lane 2m + 1 the lo part.
        const int ch = quarter;
        const uint32_t st_lane = 32u * (uint32_t)quarter;
        const int m = lane >> 1, ri = lane & 1;
        const bool mreal = m < args.M;                       // padded modes: gamma = omega = 0, never stored
        const int pm = (d0 + ch) * args.M + m;
        const float m_decay = mreal ? args.decay[pm] : 0.0f, m_freq = mreal ? args.freq[pm] : 0.0f;
        const float2 LC = lambda_pow(m_decay, m_freq, (float)kC);
        float2 S = make_float2(0.0f, 0.0f);
        // Chunk n0 of tile 0 opens at token 0; a batch row's initial state (zero
        // without one) is the state carried into it.
        const int n0 = (int)((-args.t0) >> 6);
        auto state_in_of = [&](int row) {
            return (args.state_in && mreal) ? args.state_in[((int64_t)row * D + d0 + ch) * args.M + m]
                                            : make_float2(0.0f, 0.0f);
        };
        float2 inj = kPack ? make_float2(0.0f, 0.0f) : state_in_of(b);
        uint8_t *bs = smem + kOffBs + ch * kBsStride + ri * kBsPart + (m / 4) * kBsLbo + (m % 4) * 4;
        for (int v = 0; v < nV; ++v) {
            const int bb = v & 1, u = v >> 1;
            if (kPack && real_tile(v) == 0) {
                S = make_float2(0.0f, 0.0f);   // a new batch row starts from zero (or its own s_in)
                inj = state_in_of(row_of(v));
            }
            const bool inj_tile = args.state_in != nullptr && real_tile(v) == 0;
            if (!wait_bar(bar(kBarTwDone + 2 * ch + bb), u & 1, abort_flag)) break;
            // The chain of tile v has completed, so its reads of B-operand buffer
            // v & 1 are done: release it (one arrival per channel).
            if (lane == 0) bar_arrive(bar(kBarBxEmpty + bb));
            // The carried-state operand is single-buffered: tile v - 1's
            // up-projection must have read it before it is rewritten.
            if (v > 0 && !wait_bar(bar(kBarUDone + 2 * ch + (bb ^ 1)), ((v - 1) >> 1) & 1, abort_flag)) break;
            tc_fence_after();
            if (!inj_tile) {
#pragma unroll
                for (int h = 0; h < kNT / 16; ++h) {
                    uint32_t va[16];
                    tmem_ld16(tmem + (st_lane << 16) + bb * 128 + ch * kNT + 16 * h, va);
                    tmem_wait_ld();
#pragma unroll
                    for (int n = 0; n < 16; ++n) {
                        const float a = __uint_as_float(va[n]);
                        const float other = __shfl_xor_sync(0xffffffffu, a, 1);
                        const float2 Ln = ri ? make_float2(other, a) : make_float2(a, other);
                        const int nn = 16 * h + n;
                        uint32_t hi, lo;
                        split_pack(S.x, S.y, hi, lo);
                        *reinterpret_cast<uint32_t *>(bs + (nn >> 3) * kBsSbo + (nn & 7) * 16) = ri ? lo : hi;
                        S = cfma(LC, S, Ln);
                    }
                }
            } else {
                // A row's first tile with an initial state: the same steps, one
                // chunk at a time (compact code, off the other tiles' path), the
                // state added where chunk n0 opens at token 0.
#pragma unroll 1
                for (int nn = 0; nn < kNT; ++nn) {
                    uint32_t r;
                    tmem_ld1(tmem + (st_lane << 16) + bb * 128 + ch * kNT + nn, r);
                    tmem_wait_ld();
                    const float a = __uint_as_float(r);
                    const float other = __shfl_xor_sync(0xffffffffu, a, 1);
                    const float2 Ln = ri ? make_float2(other, a) : make_float2(a, other);
                    if (nn == n0) S = make_float2(S.x + inj.x, S.y + inj.y);
                    uint32_t hi, lo;
                    split_pack(S.x, S.y, hi, lo);
                    *reinterpret_cast<uint32_t *>(bs + (nn >> 3) * kBsSbo + (nn & 7) * 16) = ri ? lo : hi;
                    S = cfma(LC, S, Ln);
                }
            }
            if ((kPack ? real_tile(v) == args.ntiles - 1 : v == nV - 1) && args.state_out && mreal && ri == 0)
                args.state_out[((int64_t)row_of(v) * D + d0 + ch) * args.M + m] = S;
            fence_async_smem();
            tc_fence_before();
            __syncwarp();
            if (lane == 0) bar_arrive(bar(kBarSFull + 2 * ch + bb));
        }
    } else if (warp < 8) {
        // ---------------------------------------------------- epilogue
        // Warp (quarter q, h) reads its quarter's Toeplitz lanes -- position
        // pos = 32 (q % 2) + lane of channels c0, c0+1 (c0 = 2 in quarters 0, 1 and
        // 0 in quarters 2, 3) -- for chunks 16h .. 16h+15, releasing each
        // accumulator as soon as it is read, and writes the 8-byte half (channels
        // c0, c0+1) of each token's 16-byte row into the y ring: slots 2h, 2h+1.
        const int h = warp >> 2;
        const int c0 = quarter < 2 ? 2 : 0;
        const int pos = 32 * (quarter & 1) + lane;
        const int hb = quarter < 2 ? 8 : 0;
        const uint32_t trow = tmem + ((uint32_t)(32 * quarter) << 16) + 16 * h;
        for (int j = 0; j < nV; ++j) {
            const int bb = j & 1, u = j >> 1;
            if (!wait_bar(bar(kBarUDone + 2 * c0 + bb), u & 1, abort_flag) ||
                !wait_bar(bar(kBarUDone + 2 * (c0 + 1) + bb), u & 1, abort_flag))
                break;
            tc_fence_after();
            uint32_t va[16], vb[16];
            tmem_ld16(trow + bb * 128 + c0 * kNT, va);
            tmem_ld16(trow + bb * 128 + (c0 + 1) * kNT, vb);
            tmem_wait_ld();
            tc_fence_before();
            __syncwarp();
            if (lane == 0) {
                bar_arrive(bar(kBarDEmpty + 2 * c0 + bb));
                bar_arrive(bar(kBarDEmpty + 2 * (c0 + 1) + bb));
            }
            bool ok = true;
#pragma unroll
            for (int sh = 0; sh < 2; ++sh) {
                const int ng = j * kYPerTile + 2 * h + sh;
                const uint32_t slot = ng % kYSlots;
                if (!wait_bar(bar(kBarYEmpty + slot), ((ng / kYSlots) & 1) ^ 1, abort_flag)) {
                    ok = false;
                    break;
                }
                uint8_t *ys = smem + kOffY + slot * (kYRows * 16) + hb;
#pragma unroll
                for (int n = 0; n < 8; ++n)
                    *reinterpret_cast<uint2 *>(ys + (n * kC + pos) * 16) = make_uint2(va[8 * sh + n], vb[8 * sh + n]);
                fence_async_smem();
                __syncwarp();
                if (lane == 0) bar_arrive(bar(kBarYFull + slot));
            }
            if (!ok) break;
        }
    }

    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 17)
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

// 3-D map over a [B][L][D] fp32 field: dims (D, L, B), box (4, 256, 1).
bool make_field_map32(CUtensorMap *map, const void *ptr, int64_t B, int64_t L, int D) {
    EncodeTiledFn fn = encode_fn();
    if (!fn) return false;
    cuuint64_t dims[3] = {(cuuint64_t)D, (cuuint64_t)L, (cuuint64_t)B};
    cuuint64_t strides[2] = {(cuuint64_t)D * 4, (cuuint64_t)L * D * 4};
    cuuint32_t box[3] = {(cuuint32_t)kDG, (cuuint32_t)kBox, 1};
    cuuint32_t estr[3] = {1, 1, 1};
    return fn(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 3, const_cast<void *>(ptr), dims, strides, box, estr,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Batch rows per CTA: as the bf16 kernel, runs in waves pay the CTAs' prologue and
// pipeline fill again, about six tiles' worth for a one-tile CTA.
int rows_per_cta32(int64_t B, int D, int ntiles) {
    const int64_t groups = D / kDG, sms = sm_count();
    const double fill = std::max(0, 6 - ntiles);
    int best = 1;
    double best_t = 0.0;
    for (int64_t r = 1; r <= B; ++r) {
        const int64_t ctas = groups * ((B + r - 1) / r);
        const double t = (double)((ctas + sms - 1) / sms) * (fill + (double)r * ntiles * (r > 1 ? 1.05 : 1.0));
        if (r == 1 || t < best_t - 1e-9) {
            best = (int)r;
            best_t = t;
        }
        if (ctas <= sms) break;
    }
    return best;
}

}  // namespace

bool tc32_prefill_supported(int64_t B, int64_t L, int D, int M, rlm_dtype dt) {
    return dt == RLM_F32 && M >= 1 && M <= kModes && D % kDG == 0 && B >= 1 && B <= 65535 && L >= 1 &&
           L <= ((int64_t)1 << 31) - kTile && D / kDG <= 65535;
}

cudaError_t tc32_prefill(const float *x, float *y, int64_t B, int64_t L, int D, int M, const float *decay,
                         const float *freq, const float *amp, const float *phase, const float *state_in,
                         float *state_out, float *coef_out, cudaStream_t st) {
    if (state_in && L % kC != 0) return cudaErrorInvalidValue;
    CUtensorMap mx, my;
    if (!make_field_map32(&mx, x, B, L, D) || !make_field_map32(&my, y, B, L, D)) return cudaErrorInvalidValue;
    static std::mutex mu;
    static std::vector<int> configured;
    int dev = 0;
    cudaGetDevice(&dev);
    {
        std::lock_guard<std::mutex> lock(mu);
        if ((int)configured.size() <= dev) configured.resize(dev + 1, 0);
        if (!configured[dev]) {
            cudaError_t e = cudaFuncSetAttribute(k_prefill_tc32<kPlain>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                 kSmemBytes);
            if (e == cudaSuccess)
                e = cudaFuncSetAttribute(k_prefill_tc32<kPacked>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         kSmemBytes);
            if (e != cudaSuccess) return e;
            configured[dev] = 1;
        }
    }
    Tc32Args a;
    a.decay = decay;
    a.freq = freq;
    a.amp = amp;
    a.phase = phase;
    a.state_in = reinterpret_cast<const float2 *>(state_in);
    a.state_out = reinterpret_cast<float2 *>(state_out);
    a.coef_out = reinterpret_cast<float4 *>(coef_out);
    a.y = y;
    a.L = L;
    a.D = D;
    a.M = M;
    a.ntiles = (int)((L + kTile - 1) / kTile);
    a.t0 = L - (int64_t)a.ntiles * kTile;
    a.B = (int)B;
    a.bpc = rows_per_cta32(B, D, a.ntiles);
    const dim3 grid((unsigned)(D / kDG), (unsigned)((B + a.bpc - 1) / a.bpc));
    if (a.bpc > 1)
        k_prefill_tc32<kPacked><<<grid, kThreads, kSmemBytes, st>>>(mx, my, a);
    else
        k_prefill_tc32<kPlain><<<grid, kThreads, kSmemBytes, st>>>(mx, my, a);
    count_launches(1);
    return cudaGetLastError();
}

cudaError_t read_and_clear_tc32_status(int *status, cudaStream_t st) {
    cudaError_t e = cudaMemcpyFromSymbolAsync(status, g_tc32_status, sizeof(int), 0, cudaMemcpyDeviceToHost, st);
    if (e != cudaSuccess) return e;
    if ((e = cudaStreamSynchronize(st)) != cudaSuccess) return e;
    const int zero = 0;
    if ((e = cudaMemcpyToSymbolAsync(g_tc32_status, &zero, sizeof(int), 0, cudaMemcpyHostToDevice, st)) !=
        cudaSuccess)
        return e;
    return cudaStreamSynchronize(st);
}

}  // namespace rlm
