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
// T and W share one A operand (64 Toeplitz rows and 32 state rows of a
// 128-row matrix) held in TMEM, so a single MMA chain yields both.  The columns
// of D are the NT = 32 chunks of a 2048-token tile (MMA N = 32).  A tcgen05.mma
// of this shape costs about the same whatever N is (N <= 64), so the number of
// MMAs per token, not their arithmetic, bounds the tensor pipe: the tile is as
// wide as TMEM allows.
// The carry between chunks is a sequential fp32 complex scan in registers: one
// thread per (channel, mode); a warp scans two channels, the two rows (Re, Im)
// of a mode exchanging their values with one warp shuffle per chunk.
//
// One CTA owns one batch row b and one group of DG = 8 channels (a 16-byte
// slice of each token row) and walks the sequence tile by tile, carrying the
// state in registers, so no CTA waits on another.
//
// Data movement per tile (2048 tokens x 8 channels):
//   TMA (3-D map over [B][L][D], zero fill outside the sequence) -> 15-box ring
//   -> ldmatrix.trans / stmatrix by three transposer warps into the per-channel
//      K-major B operand (double-buffered; the positions of a chunk reversed so
//      that the A operand's Toeplitz rows read K[i + p' - 63])
//   -> tcgen05.mma -> TMEM -> scan warps -> B operand of the up-projection
//   -> tcgen05.mma -> TMEM -> epilogue warps (fp32 -> bf16, 8 channels packed
//      into one 16-byte row) -> smem ring -> TMA store.
// TMEM (512 columns): one accumulator of 32 columns per channel (columns
// 0-255) and the 8 channels' A operands (128 lanes x 32 columns of packed bf16
// pairs, columns 256-511).  Each channel's accumulator passes through
// Toeplitz/state MMA -> scan -> up-projection MMA -> epilogue read and is then
// free for the next tile; the eight channels run this chain independently, so
// while one waits on its scan or epilogue the others keep the tensor pipe busy.
//
// TMEM lane quarter q (lanes 32q..32q+31) is readable only by warps with
// warp % 4 == q, which also run on SM sub-partition q.  The rows of each
// channel's A operand (and so of its accumulator) are placed so that every
// quarter carries the same load: quarter c/2 holds channel c's 32 state rows;
// the Toeplitz rows (positions 0-31, 32-63) sit in quarters 2, 3 for channels
// 0-3 and in quarters 0, 1 for channels 4-7; the fourth quarter is zero.
//
// Warp roles (26 warps):
//   0-7    epilogue: warp (q = warp % 4, h = warp / 4) converts positions
//          32 (q % 2) + lane of chunks 16h .. 16h+15 for the four channels whose
//          Toeplitz rows live in quarter q, into 8-byte halves of the y rows.
//   8-11   scan: the warp of quarter q carries channels 2q and 2q+1.
//   12-15  transposers (ring slot s: warp 12 + s mod 4); 16 TMA producer; 17 TMA store
//          issuer and TMEM allocation.
//   18-25  MMA issue for one channel each -- a tcgen05.mma occupies its issuing
//          thread for ~100 cycles, so eight issuing threads keep the pipe fed.
// Warps 0-11 and 18-21 first build the per-channel constants.
//
// Every wait is bounded: after wait_limit() cycles the waiting thread sets a shared
// abort flag and the device status word (RLM_ERR_TIMEOUT); all roles then leave
// their loops, drain what they issued and the CTA frees its TMEM and returns.
#include <cuda.h>

#include <algorithm>
#include <atomic>
#include <mutex>
#include <vector>

#include "rlm_device.cuh"
#include "rlm_internal.h"

namespace rlm {

// Device status word: RLM_OK, or RLM_ERR_TIMEOUT once a bounded wait expired.
__device__ int g_device_status = 0;

// Bound of every wait in the prefill kernel, in SM cycles: about 2 s at 2 GHz.
// The failure-detection test (rlm_test_stall_segments) shortens it to about 1 ms
// and makes the first sequence segment withhold its end-state flag, so that the
// later segments' waits expire; off (these values) by default.
constexpr long long kWaitLimitDefault = 4000000000ll;
__device__ long long g_wait_limit_cycles = kWaitLimitDefault;
__device__ int g_stall_segment0 = 0;
__device__ __forceinline__ long long wait_limit() {
    return *reinterpret_cast<volatile long long *>(&g_wait_limit_cycles);
}

namespace {

constexpr int kC = 64;                 // chunk length
constexpr int kNT = 32;                // chunks per tile = MMA N
constexpr int kTile = kC * kNT;        // 2048 tokens
constexpr int kDG = 8;                 // channels per CTA
constexpr int kBox = 256;              // TMA box rows
constexpr int kBoxes = kTile / kBox;   // 8 per tile
constexpr int kYRows = 512;            // rows per y ring slot (8 chunks)
constexpr int kYPerTile = kTile / kYRows;  // 4 slots per tile
constexpr int kWarps = 26;
constexpr int kThreads = kWarps * 32;
constexpr int kTmemCols = 512;
constexpr int kTmemA = 256;            // first TMEM column of the A operands
constexpr int kTransposers = 4;
constexpr int kBxStride = 4096 + 16;   // 32 rows x 128 B, +16 so stmatrix rows hit distinct banks
constexpr int kBxBuf = kDG * kBxStride;
// Carried-state operand: LBO 144 (not 128) spreads one chunk's 16 mode words
// over distinct banks; the channel stride is 16 banks (mod 32) so the two
// channels of a scan warp write disjoint banks as well.
constexpr int kBsLbo = 144;
// Prologue tables, in buffers no other role touches before the prologue ends
// (the transposers already fill the B operand meanwhile).  They are laid out for
// conflict-free reads when lane R of a warp fetches word k of row R: the W table
// is word-major with rows innermost (stride 33 words), and the second Toeplitz
// pair table starts 80 words (16 banks) after the first.
constexpr int kWtabStride = 33;
constexpr int kTpairStride = 144;      // words per channel: P0 at 0, P1 at 80
// Named barriers: the 16 warps that build the constants (0-11 and 18-21); the
// CTA's set-up, which the TMA producer warp only arrives at.
constexpr int kPrologueBarrier = 1;
constexpr int kPrologueThreads = 512;
constexpr int kSetupBarrier = 2;

// Layout of one kernel instance: kModes = 16 or 32 modes per channel in its
// tables (fewer are padded).  With 32 modes the A operand's fourth TMEM quarter
// holds the state rows of modes 16-31, the U tables and the carried-state
// operand double, and the x and y rings shrink to fit shared memory.
template <int kModes>
struct Cfg {
    static_assert(kModes == 16 || kModes == 32, "16 or 32 modes per instance");
    static constexpr int kXSlots = kModes == 16 ? 15 : 7;   // x ring depth (boxes)
    static constexpr int kYSlots = kModes == 16 ? 6 : 4;    // y ring depth
    // U tables: 64 rows x 2 kModes bf16 per channel (K-major core matrices: 8 rows
    // x 16 B, K groups 128 B apart, row groups kAuSbo apart), in the order of
    // channels 4-7, 0-3.  The up-projection reads a 128-row A operand whose 64
    // real rows must meet the channel's Toeplitz lanes: rows 0-63 for channels
    // 4-7 (start at the table), rows 64-127 for channels 0-3 (start one table
    // earlier).  The other 64 rows read a neighbouring table and land in state
    // lanes nobody reads afterwards.
    static constexpr int kAuSbo = 32 * kModes;
    static constexpr int kAuStride = 8 * kAuSbo;
    static constexpr int kBsSbo = (kModes / 4) * kBsLbo;
    static constexpr int kBsStride = 4 * kBsSbo + 64;
    static_assert((kBsStride / 4) % 32 == 16, "paired channels must use disjoint banks");
    static constexpr int kOffAu = 0;
    static constexpr int kOffBx = kOffAu + kDG * kAuStride;
    static constexpr int kOffBs = kOffBx + 2 * kBxBuf;
    static constexpr int kOffX = kOffBs + kDG * kBsStride;
    static constexpr int kOffY = kOffX + kXSlots * kBox * 16;
    static constexpr int kOffBar = kOffY + kYSlots * kYRows * 16;
    static constexpr int kNumBars = 96;
    static constexpr int kOffMisc = kOffBar + kNumBars * 8;
    static constexpr int kSmemBytes = kOffMisc + 64 + 1024;        // + alignment slack
    static_assert(kOffX % 128 == 0 && kOffY % 128 == 0, "TMA buffers need 128-byte alignment");
    static_assert(kSmemBytes <= 232448, "shared memory budget");
    // Prologue tables.  The W table (16 modes only; with 32 the W rows are formed
    // in registers) lives in the y ring, the others in the carried-state buffers.
    static constexpr int kOffWtab = kOffY;                          // [8 ch][32 words][33]
    static constexpr int kOffTpair = kOffBs;                        // [8 ch][144 words]: Toeplitz pairs
    static constexpr int kOffKp = kOffTpair + 8 * kTpairStride * 4; // [2 halves][8 ch][64] fp32 partial sums of K
    // [8 ch][kModes][5] float2: lambda, c, lambda^2, lambda^4, lambda^8 of each mode.
    static constexpr int kOffLtab = kOffKp + 2 * 8 * 64 * 4;
    static_assert(kModes != 16 || 8 * 32 * kWtabStride * 4 <= kYSlots * kYRows * 16, "W table does not fit the y ring");
    static_assert(kOffLtab + 8 * kModes * 5 * 8 <= kOffX, "prologue tables do not fit");
    // Barrier indices.
    static constexpr int kBarXFull = 0;                    // [kXSlots]
    static constexpr int kBarXEmpty = kXSlots;             // [kXSlots]
    static constexpr int kBarBxFull = 2 * kXSlots;         // [2]
    static constexpr int kBarBxEmpty = kBarBxFull + 2;     // [2]: released by the 8 MMA threads
    static constexpr int kBarTwDone = kBarBxEmpty + 2;     // [8]: Toeplitz/state MMAs of a channel done
    static constexpr int kBarSFull = kBarTwDone + 8;       // [8]: carried states of a channel written
    static constexpr int kBarUDone = kBarSFull + 8;        // [8]: up-projection of a channel done
    static constexpr int kBarDEmpty = kBarUDone + 8;       // [8]: accumulator of a channel read out
    static constexpr int kBarYFull = kBarDEmpty + 8;       // [kYSlots]
    static constexpr int kBarYEmpty = kBarYFull + kYSlots; // [kYSlots]
    static constexpr int kBarFinal = kBarYEmpty + kYSlots; // [8]
    static constexpr int kBarConsts = kBarFinal + 8;       // the A operands and U tables are built
    static constexpr int kBarGFull = kBarConsts + 1;       // [kYSlots] mixer: the gate rows of a z slot landed
    static_assert(kBarGFull + kYSlots <= kNumBars, "too many barriers");
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
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes)
                 : "memory");
}

// Bounded wait on an mbarrier phase.  Returns false if this CTA aborted.
// The bound is measured with the SM cycle counter, read only every 1024 failed
// polls: reading %globaltimer costs about half a microsecond, which would
// otherwise be added to every wait that does not succeed at once.
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
            } else if (now - t0 > wait_limit()) {
                *abort_flag = 1;
                atomicExch(&g_device_status, (int)RLM_ERR_TIMEOUT);
                return false;
            }
        }
    }
}

// Bounded wait until *flag == want (another CTA's release), with acquire
// semantics for the loads that follow.  Returns false if this CTA aborted.
__device__ __forceinline__ bool wait_flag(const unsigned long long *flag, unsigned long long want,
                                          volatile int *abort_flag) {
    long long t0 = 0;
    for (uint32_t it = 0;; ++it) {
        unsigned long long v;
        asm volatile("ld.acquire.gpu.global.u64 %0, [%1];" : "=l"(v) : "l"(flag) : "memory");
        if (v == want) return true;
        if ((it & 255u) == 0) {
            if (*abort_flag) return false;
            const long long now = clock64();
            if (t0 == 0) {
                t0 = now;
            } else if (now - t0 > wait_limit()) {
                *abort_flag = 1;
                atomicExch(&g_device_status, (int)RLM_ERR_TIMEOUT);
                return false;
            }
        }
        __nanosleep(64);
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
__device__ __forceinline__ void tmem_ld8(uint32_t taddr, uint32_t (&v)[8]) {
    asm volatile("tcgen05.ld.sync.aligned.32x32b.x8.b32 {%0,%1,%2,%3,%4,%5,%6,%7}, [%8];"
                 : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]),
                   "=r"(v[6]), "=r"(v[7])
                 : "r"(taddr));
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

// Instruction descriptors, kind::f16: fp32 accumulate, bf16 A and B, both K-major,
// M = 128, N = kNT.
constexpr uint32_t kIdesc = (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(kNT >> 3) << 17) |
                            ((uint32_t)(128 >> 4) << 24);

__device__ __forceinline__ int au_slot(int c) { return (c + 4) & 7; }
// First byte (from the U table area) of channel c's 128-row up-projection operand.
__device__ __forceinline__ int au_operand(int c, int stride) { return au_slot(c) * stride - (c < 4 ? stride : 0); }

struct TcArgs {
    const float *decay, *freq, *amp, *phase;
    const float2 *state_in;  // [B][D][M], the state before token 0 (kInj instances only)
    float2 *state_out;   // nullable, [B][D][M]
    float4 *coef_out;    // nullable, [D][M]
    __nv_bfloat16 *y;    // for the plain stores of boxes that start before t = 0
    int64_t L;
    int D;
    int M;               // modes of this pass, 1..kModes; modes M.. are padding (amplitude 0, never stored)
    int m0, Mt;          // first mode of this pass; modes per channel in the parameter/state layouts
    int add;             // kMix: the slot holds y so far (earlier passes); z = that + this pass's y
                         // (otherwise the slot holds the gate: z = sigma(g) y)
    int ntiles;
    int64_t t0;          // first token of tile 0 (<= 0): tiles end exactly at L-1
    // Unsegmented launches: grid y covers batch rows in groups of bpc; a CTA runs
    // its rows' tiles back to back as one stream (one prologue for all of them).
    int B, bpc;
    // Sequence segments (grid z): segment s owns tiles [s * seg_tiles, ...).
    int nseg, seg_tiles;
    float2 *seg_state;   // [B][nseg][D][M]: each segment's end state from a zero start
    unsigned long long *seg_flag;  // [B][nseg][D][M]: == epoch once that state is published
    unsigned long long epoch;      // distinct for every segmented launch of this process
};

// kMode: kPlain, one CTA per (channel group, batch row); kSegmented (kSeg), the
// grid's z dimension splits the sequence into segments; kPacked (kPack), a CTA
// runs args.bpc batch rows of its channel group back to back.  The plain instance
// keeps the tile count a kernel parameter (no register holds it), which the
// per-tile loops' register allocation depends on.
// kInj: the prefill starts from args.state_in instead of zero.  Token 0 sits at
// position p of chunk n0 of tile 0 (tiles end at L - 1); lambda^-p s_in is added
// to the state entering chunk n0, which gives lambda^(i+1-p) s_in at its positions
// i >= p (those before p are negative times, never stored) and lambda^(64-p) s_in
// carried on.  |lambda^-p| <= exp(63 gamma) stays bounded.
// kMix: a second field is loaded into the z ring and combined in the epilogue
// (unsegmented launches only): the gate of the mixer wrapper (Sec. 3.4),
// z = sigma(g) y, or (args.add, for M > 16 in passes of 16 modes) the output of
// the earlier passes, z = y_before + y.  The store issuer loads the field's rows
// of each z ring slot into the slot itself once the slot's previous store has
// been read out; every epilogue thread reads its 8 bytes there and overwrites them
// with z.
enum : int { kPlain = 0, kSegmented = 1, kPacked = 2 };

// kModes: 16, or 32 (kPlain and kPacked without the mixer field only).
template <int kMode, bool kInj, bool kMix, int kModes>
__global__ void __launch_bounds__(kThreads, 1)
    k_prefill_tc(const __grid_constant__ CUtensorMap tmap_x,
                 const __grid_constant__ CUtensorMap tmap_y, const __grid_constant__ CUtensorMap tmap_g,
                 const TcArgs args) {
    constexpr bool kSeg = kMode == kSegmented, kPack = kMode == kPacked;
    static_assert(!(kSeg && kMix), "the mixer epilogue is not built for segmented launches");
    static_assert(kModes == 16 || (!kSeg && !kMix), "32 modes: plain or packed launches without a second field");
    using Cf = Cfg<kModes>;
    constexpr int kXSlots = Cf::kXSlots, kYSlots = Cf::kYSlots, kAuStride = Cf::kAuStride, kAuSbo = Cf::kAuSbo;
    constexpr int kBsSbo = Cf::kBsSbo, kBsStride = Cf::kBsStride;
    constexpr int kOffAu = Cf::kOffAu, kOffBx = Cf::kOffBx, kOffBs = Cf::kOffBs, kOffX = Cf::kOffX, kOffY = Cf::kOffY;
    constexpr int kOffBar = Cf::kOffBar, kOffMisc = Cf::kOffMisc, kOffWtab = Cf::kOffWtab, kOffTpair = Cf::kOffTpair;
    constexpr int kOffKp = Cf::kOffKp, kOffLtab = Cf::kOffLtab;
    constexpr int kBarXFull = Cf::kBarXFull, kBarXEmpty = Cf::kBarXEmpty, kBarBxFull = Cf::kBarBxFull;
    constexpr int kBarBxEmpty = Cf::kBarBxEmpty, kBarTwDone = Cf::kBarTwDone, kBarSFull = Cf::kBarSFull;
    constexpr int kBarUDone = Cf::kBarUDone, kBarDEmpty = Cf::kBarDEmpty, kBarYFull = Cf::kBarYFull;
    constexpr int kBarYEmpty = Cf::kBarYEmpty, kBarFinal = Cf::kBarFinal, kBarConsts = Cf::kBarConsts;
    constexpr int kBarGFull = Cf::kBarGFull;
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    // Align with pointer arithmetic on the __shared__ array (not through an
    // integer), so the compiler keeps the shared address space and emits
    // shared-memory loads and stores instead of generic ones.
    uint8_t *smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
    const uint32_t sbase = smem_u32(smem);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int g = blockIdx.x, seg = kSeg ? (int)blockIdx.z : 0;
    const int b = kPack ? (int)blockIdx.y * args.bpc : (int)blockIdx.y;   // the CTA's (first) batch row
    const int d0 = g * kDG;
    const int D = args.D;
    // Virtual tiles.  Segmented: nA state-only passes over the segment's tiles
    // (every segment but the last publishes its end state for the later ones),
    // then nB output passes over the same tiles.  Packed: the tiles of the CTA's
    // batch rows, row after row (v -> row b + v / ntiles, tile v % ntiles).
    const int ja = kSeg ? seg * args.seg_tiles : 0;
    const int nB = kSeg ? min(args.ntiles, ja + args.seg_tiles) - ja
                        : kPack ? min(args.bpc, args.B - b) * args.ntiles : args.ntiles;
    const int nA = kSeg && seg < args.nseg - 1 ? nB : 0;
    const int nV = kSeg ? nA + nB : kPack ? nB : args.ntiles;
    auto real_tile = [&](int v) { return kPack ? v % args.ntiles : ja + (v < nA ? v : v - nA); };
    auto row_of = [&](int v) { return kPack ? b + v / args.ntiles : b; };
    // Constant builders: warps 0-11 and 18-21.  The first 128 of them (one per
    // (channel, mode)) form each mode's powers once for all builders and issue
    // their parameter loads first, so the DRAM latency overlaps the set-up.
    // (Computing these powers in warps 22-25 instead, the MMA issuers of channels
    // 4-7, made the steady state slower: 47.8 against 45.7 us at B = 4, L = 32768.)
    const bool builder = warp < 12 || (warp >= 18 && warp < 22);
    const int pq = warp & 3, pe = warp < 12 ? warp >> 2 : 3;
    const int ptid = (pe * 4 + pq) * 32 + lane;
    const bool lpow = builder && ptid < 8 * kModes;
    const int l_c = ptid / kModes, l_m = ptid % kModes;
    float p_decay = 0.0f, p_freq = 0.0f, p_amp = 0.0f, p_phase = 0.0f;
    if (lpow && l_m < args.M) {
        const int pm = (d0 + l_c) * args.Mt + args.m0 + l_m;
        p_decay = args.decay[pm];
        p_freq = args.freq[pm];
        p_amp = args.amp[pm];
        p_phase = args.phase[pm];
    }
    uint64_t *bars = reinterpret_cast<uint64_t *>(smem + kOffBar);
    auto bar = [&](int i) { return smem_u32(bars + i); };
    volatile int *abort_flag = reinterpret_cast<volatile int *>(smem + kOffMisc);
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(smem + kOffMisc + 16);

    // Set-up.  The TMA producer warp initialises the x ring's barriers, arrives
    // at the set-up barrier without waiting for it and fills the whole ring at
    // once (issuing a TMA load blocks its thread while the previous box is being
    // processed, so it must not hold up the others).  Thread 0 initialises the
    // other barriers, warp 17 allocates TMEM.
    const int total_boxes = nV * kBoxes;
    int issued = 0;
    uint32_t tmem = 0;
    if (warp == 16) {
        if (lane == 0) {
            *abort_flag = 0;
            asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmap_x)) : "memory");
            for (int i = 0; i < kXSlots; ++i) {
                bar_init(bar(kBarXFull + i), 1);
                bar_init(bar(kBarXEmpty + i), 1);
            }
            asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
            fence_async_smem();
        }
        __syncwarp();
        asm volatile("bar.arrive %0, %1;" ::"n"(kSetupBarrier), "n"(kThreads) : "memory");
        if (lane == 0) {
            for (; issued < total_boxes && issued < kXSlots; ++issued) {
                const int jt = real_tile(issued / kBoxes), q = issued % kBoxes, bq = row_of(issued / kBoxes);
                const uint32_t slot = issued % kXSlots;
                bar_expect_tx(bar(kBarXFull + slot), kBox * 16);
                tma_load_3d(sbase + kOffX + slot * (kBox * 16), &tmap_x, d0,
                            (int)(args.t0 + (int64_t)jt * kTile + q * kBox), bq, bar(kBarXFull + slot));
            }
        }
    } else {
        if (tid == 0) {
            for (int i = 0; i < 2; ++i) {
                bar_init(bar(kBarBxFull + i), kBoxes);
                bar_init(bar(kBarBxEmpty + i), kDG);
            }
            for (int i = 0; i < kDG; ++i) {
                bar_init(bar(kBarTwDone + i), 1);
                bar_init(bar(kBarSFull + i), kModes / 16);   // with 32 modes: two scan warps
                bar_init(bar(kBarUDone + i), 1);
                bar_init(bar(kBarDEmpty + i), 4);
                bar_init(bar(kBarFinal + i), 1);
            }
            for (int i = 0; i < kYSlots; ++i) {
                bar_init(bar(kBarYFull + i), 4);
                bar_init(bar(kBarYEmpty + i), 1);
            }
            bar_init(bar(kBarConsts), 1);
            if (kMix)
                for (int i = 0; i < kYSlots; ++i) bar_init(bar(kBarGFull + i), 1);
            asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        }
        if (warp == 17) {
            if (lane == 0) {
                asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmap_y)) : "memory");
                if (kMix) asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmap_g)) : "memory");
            }
            __syncwarp();
            asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                             smem_u32(tmem_slot)),
                         "r"(kTmemCols));
            asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
        }
        tc_fence_before();
        asm volatile("bar.sync %0, %1;" ::"n"(kSetupBarrier), "n"(kThreads) : "memory");
        tc_fence_after();
        tmem = *tmem_slot;
    }

    // Per-mode powers (builder threads 0-127, one per (channel, mode)): lambda and c
    // in full fp32 accuracy (also the mode coefficients for decode), lambda^2,
    // lambda^4 and lambda^8 by squaring.
    if (lpow) {
        const float2 lam = lambda_pow(p_decay, p_freq, 1.0f);
        const float2 cf = mode_coef(p_amp, p_phase);
        if (args.coef_out && b == 0 && seg == 0 && l_m < args.M)
            args.coef_out[(d0 + l_c) * args.Mt + args.m0 + l_m] = make_float4(lam.x, lam.y, cf.x, cf.y);
        const float2 l2 = cmul(lam, lam), l4 = cmul(l2, l2), l8 = cmul(l4, l4);
        float2 *lt = reinterpret_cast<float2 *>(smem + kOffLtab) + (l_c * kModes + l_m) * 5;
        lt[0] = lam;
        lt[1] = cf;
        lt[2] = l2;
        lt[3] = l4;
        lt[4] = l8;
    }

    // ---------------------------------------------------- per-channel constants
    // Built by warps 0-11 and 18-21 (synchronised by a named barrier), while the
    // transposers, the producer and the store issuer start their work.  Warp
    // (quarter q, rank e within its quarter) has prologue thread index ptid.
    // Stage 1: builder warp bw (channel c = bw / 2) runs the powers lambda^n of
    // its modes m = 4 (bw % 2) + lane % 4 + 8 j at the positions n = q8 + 8 e
    // (q8 = lane / 4, e < 8), by a recurrence with step lambda^8.  Per power it
    // writes the U row word (Re, -Im of c lambda^(n+1)), for even n the W-row
    // words (lambda^n, lambda^(n+1) packed), and adds Re(c lambda^n) to its
    // partial sum of K[n].  A warp's U stores cover every (n mod 8, m mod 4) pair,
    // i.e. 32 distinct banks.  The partial sums are reduced over the warp's four
    // lanes of equal q8 (a fixed shuffle tree) into Kp[bw % 2][c][n].
    if (builder) {
        asm volatile("bar.sync %0, %1;" ::"n"(kPrologueBarrier), "n"(kPrologueThreads) : "memory");
        const int c = ptid >> 6, q8 = lane >> 2;
        const int mb = 4 * ((ptid >> 5) & 1) + (lane & 3);
        float kv[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) kv[e] = 0.0f;
#pragma unroll
        for (int j = 0; j < kModes / 8; ++j) {
            const int m = mb + 8 * j;
            const float2 *lt = reinterpret_cast<const float2 *>(smem + kOffLtab) + (c * kModes + m) * 5;
            const float2 lam = lt[0], cf = lt[1], l2 = lt[2], l4 = lt[3], l8 = lt[4];
            float2 pw = (q8 & 1) ? lam : make_float2(1.0f, 0.0f);      // lambda^q8
            if (q8 & 2) pw = cmul(pw, l2);
            if (q8 & 4) pw = cmul(pw, l4);
            uint8_t *au = smem + kOffAu + au_slot(c) * kAuStride + (m / 4) * 128 + (m % 4) * 4 + q8 * 16;
            uint32_t *wt = reinterpret_cast<uint32_t *>(smem + kOffWtab) + (c * 32 + (q8 >> 1)) * kWtabStride + 2 * m;
#pragma unroll
            for (int e = 0; e < 8; ++e) {
                kv[e] = fmaf(cf.x, pw.x, fmaf(-cf.y, pw.y, kv[e]));        // += Re(c lambda^n)
                const float2 nx = cmul(pw, lam);                             // lambda^(n+1)
                if (kModes == 16 && (q8 & 1) == 0) {
                    wt[4 * e * kWtabStride] = pack_bf16x2(pw.x, nx.x);
                    wt[4 * e * kWtabStride + 1] = pack_bf16x2(pw.y, nx.y);
                }
                const float2 q = cmul(cf, nx);                               // c lambda^(n+1)
                *reinterpret_cast<uint32_t *>(au + e * kAuSbo) = pack_bf16x2(q.x, -q.y);
                pw = cmul(pw, l8);
            }
        }
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            float v = kv[e];
            v += __shfl_xor_sync(0xffffffffu, v, 1);
            v += __shfl_xor_sync(0xffffffffu, v, 2);
            kv[e] = v;
        }
        if ((lane & 3) == 0) {
            float *kp = reinterpret_cast<float *>(smem + kOffKp) + (((ptid >> 5) & 1) * 8 + c) * 64 + q8;
#pragma unroll
            for (int e = 0; e < 8; ++e) kp[8 * e] = kv[e];
        }
    }
    if (builder) asm volatile("bar.sync %0, %1;" ::"n"(kPrologueBarrier), "n"(kPrologueThreads) : "memory");
    // Stage 2: K[c][n] = Kp[0][c][n] + Kp[1][c][n] (Eq. 1 at integer lags), as
    // zero-padded pair tables kz(i) = K[i - 63] (0 for i < 63):
    // P0[c][i] = (kz(2i), kz(2i+1)), P1[c][i] = (kz(2i+1), kz(2i+2)).
    if (builder) {
        const float *kp = reinterpret_cast<const float *>(smem + kOffKp);
        const int c = ptid >> 6, i = ptid & 63;
        auto kz = [&](int idx) -> float {
            const int n = idx - 63;
            return (n >= 0 && n < 64) ? kp[c * 64 + n] + kp[(8 + c) * 64 + n] : 0.0f;
        };
        uint32_t *tp = reinterpret_cast<uint32_t *>(smem + kOffTpair) + c * kTpairStride;
        tp[i] = pack_bf16x2(kz(2 * i), kz(2 * i + 1));
        tp[80 + i] = pack_bf16x2(kz(2 * i + 1), kz(2 * i + 2));
    }
    if (builder) asm volatile("bar.sync %0, %1;" ::"n"(kPrologueBarrier), "n"(kPrologueThreads) : "memory");
    // Stage 3: the A operands into TMEM, lanes 32 q + lane of channels e and e + 4:
    //   Toeplitz quarters: T[p][p'] = K[p + p' - 63] (reversed positions) for
    //     position p = 32 (q % 2) + lane;
    //   quarter c / 2:     W[k][p'] = (Re, Im) lambda_m^p' for state row k = lane
    //     (k = 2m + ri);
    //   the remaining quarter, (c / 2) ^ 1: zero, or with 32 modes the W rows of
    //     modes 16-31 (row k = lane for mode 16 + k / 2).
    // With 32 modes the W rows are formed here, by the recurrence lambda^(p'+1) =
    // lambda^p' lambda from the per-mode table (the 16-mode instance reads the W
    // table written in stage 1).
    if (builder) {
        const int q = pq, e = pe;
        for (int cc = 0; cc < 2; ++cc) {
            const int c = e + 4 * cc;
            uint32_t w[32];
            if ((q >> 1) == (c < 4 ? 1 : 0)) {
                const int pos = 32 * (q & 1) + lane;
                const uint32_t *tp = reinterpret_cast<const uint32_t *>(smem + kOffTpair) + c * kTpairStride +
                                     ((pos & 1) ? 80 + (pos >> 1) : (pos >> 1));
#pragma unroll
                for (int k = 0; k < 32; ++k) w[k] = tp[k];
            } else if (kModes == 16 && q == (c >> 1)) {
                const uint32_t *wt = reinterpret_cast<const uint32_t *>(smem + kOffWtab) + c * 32 * kWtabStride + lane;
#pragma unroll
                for (int k = 0; k < 32; ++k) w[k] = wt[k * kWtabStride];
            } else if (kModes == 32) {
                const int m = (lane >> 1) + (q == (c >> 1) ? 0 : 16), ri = lane & 1;
                const float2 lam = reinterpret_cast<const float2 *>(smem + kOffLtab)[(c * kModes + m) * 5];
                float2 pw = make_float2(1.0f, 0.0f);
#pragma unroll
                for (int k = 0; k < 32; ++k) {
                    const float2 nx = cmul(pw, lam);
                    w[k] = ri ? pack_bf16x2(pw.y, nx.y) : pack_bf16x2(pw.x, nx.x);
                    pw = cmul(nx, lam);
                }
            } else {
#pragma unroll
                for (int k = 0; k < 32; ++k) w[k] = 0u;
            }
            tmem_st32(tmem + ((uint32_t)(32 * q) << 16) + kTmemA + c * 32, w);
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
                            (int)(args.t0 + (int64_t)jt * kTile + q * kBox), bq,
                            bar(kBarXFull + slot));
            }
            // Drain: every issued load must land before this CTA may exit.
            const int first = issued > kXSlots ? issued - kXSlots : 0;
            for (int k = first; k < issued; ++k) {
                const uint32_t slot = k % kXSlots, fill = k / kXSlots;
                const long long t0 = clock64();
                while (!bar_try(bar(kBarXFull + slot), fill & 1))
                    if (clock64() - t0 > wait_limit()) break;
            }
        }
        __syncwarp();
    } else if (warp >= 12 && warp < 12 + kTransposers) {
        // ---------------------------------------------------- transposers (ring slot s: warp 12 + s mod 4)
        // Each ring slot belongs to one transposer warp (slot s to warp s mod 4), so
        // a warp waits on a slot's full barrier only after it has itself consumed
        // the slot's previous box.  With boxes dealt round-robin instead, a warp
        // could wait for box k while box k - kXSlots (consumed by another warp) had
        // not landed yet; its parity wait then matched the phase of box k - 2 kXSlots
        // and passed at once (intermittent wrong tiles and launch failures with the
        // 7-slot ring of the 32-mode instance).
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
            if (!wait_bar(bar(kBarBxEmpty + buf), (use & 1) ^ 1, abort_flag)) break;
            const int c = lane & 7, mq = lane >> 3;
            const uint32_t bx = sbase + kOffBx + buf * kBxBuf + c * kBxStride;
#pragma unroll
            for (int sb = 0; sb < 8; ++sb) {
                const int tb = 32 * tq + 4 * sb + mq;    // 8-token block within the tile
                const int n = tb >> 3, kb = 7 - (tb & 7);
                const uint32_t dst = bx + (n >> 3) * 1024 + kb * 128 + (n & 7) * 16;
                asm volatile("stmatrix.sync.aligned.m8n8.x4.shared.b16 [%0], {%1,%2,%3,%4};" ::"r"(dst),
                             "r"(r[sb][0]), "r"(r[sb][1]), "r"(r[sb][2]), "r"(r[sb][3])
                             : "memory");
            }
            fence_async_smem();
            __syncwarp();
            // The x slot is released only now that stmatrix has consumed the
            // ldmatrix registers: releasing it right after issuing ldmatrix let
            // the next TMA load overwrite the box before it had been read.
            if (lane == 0) {
                bar_arrive(bar(kBarXEmpty + slot));
                bar_arrive(bar(kBarBxFull + buf));
            }
            k = kn;
        }
    } else if (warp == 17) {
        // ---------------------------------------------------- y store issuer
        // One bulk group per slot of 512 rows; up to kYSlots - 2 groups may still
        // be reading shared memory while the next slot is issued.
        const int nslots = nB * kYPerTile;
        // Mixer: the gate rows of z slot k go into the slot itself (two boxes of 256 rows).
        auto issue_g = [&](int k) {
            const uint32_t slot = k % kYSlots;
            if (lane != 0) return;
            bar_expect_tx(bar(kBarGFull + slot), kYRows * 16);
            const int vq = k / kYPerTile, e = k % kYPerTile;
            const int jt = kPack ? vq % args.ntiles : ja + vq, bq = row_of(vq);
            for (int h = 0; h < kYRows / kBox; ++h)
                tma_load_3d(sbase + kOffY + slot * (kYRows * 16) + h * (kBox * 16), &tmap_g, d0,
                            (int)(args.t0 + (int64_t)jt * kTile + e * kYRows + h * kBox), bq, bar(kBarGFull + slot));
        };
        // The prologue keeps its W table in the z ring until the constants are built.
        if (kMix && wait_bar(bar(kBarConsts), 0, abort_flag))
            for (int k = 0; k < kYSlots && k < nslots; ++k) issue_g(k);
        int ng = 0;
        for (; ng < nslots; ++ng) {
            const uint32_t slot = ng % kYSlots;
            if (!wait_bar(bar(kBarYFull + slot), (ng / kYSlots) & 1, abort_flag)) break;
            const uint32_t ys = sbase + kOffY + slot * (kYRows * 16);
            const int vq = ng / kYPerTile, e = ng % kYPerTile;
            const int jt = kPack ? vq % args.ntiles : ja + vq, bq = row_of(vq);
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
            if (kMix) {
                // The slot is refilled with gate rows a whole ring ahead, so its
                // read-out is awaited at once (the writes stay in flight).
                if (lane == 0) {
                    tma_store_commit();
                    tma_store_wait_read();
                }
                __syncwarp();
                if (ng + kYSlots < nslots) issue_g(ng + kYSlots);
                continue;
            }
            if (lane == 0) {
                tma_store_commit();
                asm volatile("cp.async.bulk.wait_group.read %0;" ::"n"(kYSlots - 2) : "memory");
            }
            __syncwarp();
            // Groups up to ng - (kYSlots - 2) have finished reading their slots.
            const int freed = ng - (kYSlots - 2);
            if (lane == 0 && freed >= 0) bar_arrive(bar(kBarYEmpty + freed % kYSlots));
        }
        if (lane == 0) {
            tma_store_wait_read();
            if (!kMix)
                for (int k = ng - (kYSlots - 2); k < ng; ++k)
                    if (k >= 0) bar_arrive(bar(kBarYEmpty + k % kYSlots));
            tma_store_wait_all();
        }
        __syncwarp();
    } else if (warp >= 18) {
        // ---------------------------------------------------- MMA issuer, one channel
        // Per tile: the Toeplitz/state chain into the channel's accumulator, then,
        // once the scan has written the carried states, the up-projection.  The
        // next tile's chain waits until the epilogue has read the accumulator
        // (after a state-only pass, until the scan has read it).
        const int c = warp - 18;
        const uint64_t dx0 = umma_desc(sbase + kOffBx + c * kBxStride, 128, 1024);
        const uint64_t du0 = umma_desc(sbase + kOffAu + au_operand(c, kAuStride), 128, kAuSbo);
        const uint64_t ds0 = umma_desc(sbase + kOffBs + c * kBsStride, kBsLbo, kBsSbo);
        const uint32_t aT = tmem + kTmemA + c * 32;
        const uint32_t d = tmem + c * kNT;
        if (lane == 0 && wait_bar(bar(kBarConsts), 0, abort_flag)) {
            tc_fence_after();
            for (int v = 0; v < nV; ++v) {
                const int buf = v & 1, use = v >> 1;
                if (!wait_bar(bar(kBarBxFull + buf), use & 1, abort_flag)) break;
                if (v > nA && !wait_bar(bar(kBarDEmpty + c), (v - 1 - nA) & 1, abort_flag)) break;
                tc_fence_after();
                const uint64_t xo = (uint64_t)((buf * kBxBuf) >> 4);
#pragma unroll
                for (int kk = 0; kk < 4; ++kk) umma_ts(d, aT + kk * 8, dx0 + xo + kk * 16, kIdesc, kk > 0);
                umma_commit(bar(kBarTwDone + c));
                if (!wait_bar(bar(kBarSFull + c), v & 1, abort_flag)) break;
                tc_fence_after();
                // The scan has seen this chain's commit, so its MMAs (and their
                // reads of the B operand) are complete: release the buffer.  A
                // second commit issued right behind the first was observed to
                // arrive while the chain was still reading shared memory.
                bar_arrive(bar(kBarBxEmpty + buf));
                if (v < nA) continue;  // state-only pass: no output
#pragma unroll
                for (int kk = 0; kk < kModes / 8; ++kk)
                    umma_ss(d, du0 + kk * 16, ds0 + kk * ((2 * kBsLbo) >> 4), kIdesc, 1);
                umma_commit(bar(kBarUDone + c));
            }
            // Drain: all MMAs this thread issued complete before TMEM is released.
            umma_commit(bar(kBarFinal + c));
            const long long t0 = clock64();
            while (!bar_try(bar(kBarFinal + c), 0))
                if (clock64() - t0 > wait_limit()) break;
        }
        __syncwarp();
    } else if (warp >= 8 && warp < 12) {
        // ---------------------------------------------------- scan, two channels
        if constexpr (kModes == 16) {
        // The warp of quarter q owns channels 2q and 2q+1, whose state rows are
        // its TMEM lanes.  Lane 2m carries mode m of the first channel, lane 2m+1
        // mode m of the second: each lane reads row 2m+ri of both channels and one
        // shuffle hands the partner the value it lacks.  S_n = lambda^C S_{n-1} +
        // L_n runs in fp32; S_{n-1} goes to the up-projection's B operand.
        const int cA = 2 * quarter, cB = cA + 1;
        const uint32_t st_lane = 32u * (uint32_t)quarter;
        const int m = lane >> 1, ri = lane & 1;
        const int ch = ri ? cB : cA;
        const bool mreal = m < args.M;                       // padded modes: gamma = omega = 0, never stored
        const int pm = (d0 + ch) * args.Mt + args.m0 + m;
        const float m_decay = mreal ? args.decay[pm] : 0.0f, m_freq = mreal ? args.freq[pm] : 0.0f;
        const float2 LC = lambda_pow(m_decay, m_freq, (float)kC);
        float2 S = make_float2(0.0f, 0.0f);
        float2 inj = make_float2(0.0f, 0.0f);
        int n0 = -1;
        if (kInj) {
            n0 = (int)((-args.t0) >> 6);
            const int p = (int)((-args.t0) & 63);
            if (!kPack && mreal)
                inj = cmul(lambda_pow(m_decay, m_freq, (float)(-p)), args.state_in[((int64_t)b * D + d0 + ch) * args.Mt + args.m0 + m]);
        }
        uint8_t *bs = smem + kOffBs + ch * kBsStride + (m / 4) * kBsLbo + (m % 4) * 4;
        const int64_t seg_row = (int64_t)b * args.nseg;
        // One tile of the carry: S_n = lambda^C S_{n-1} + L_n over its 32 chunks.
        auto scan_tile = [&](int v) -> bool {
            const bool row_start = real_tile(v) == 0;
            const bool inj_tile = kInj && row_start;
            if (kPack && row_start) {
                S = make_float2(0.0f, 0.0f);   // a new batch row starts from zero (or its own s_in)
                if (kInj && mreal)
                    inj = cmul(lambda_pow(m_decay, m_freq, (float)(-(int)((-args.t0) & 63))),
                               args.state_in[((int64_t)row_of(v) * D + d0 + ch) * args.Mt + args.m0 + m]);
            }
            if (!wait_bar(bar(kBarTwDone + cA), v & 1, abort_flag)) return false;
            if (!wait_bar(bar(kBarTwDone + cB), v & 1, abort_flag)) return false;
            tc_fence_after();
#pragma unroll
            for (int h = 0; h < kNT / 16; ++h) {
                uint32_t va[16], vb[16];
                tmem_ld16(tmem + (st_lane << 16) + cA * kNT + 16 * h, va);
                tmem_ld16(tmem + (st_lane << 16) + cB * kNT + 16 * h, vb);
                tmem_wait_ld();
#pragma unroll
                for (int n = 0; n < 16; ++n) {
                    const float a = __uint_as_float(va[n]), bb = __uint_as_float(vb[n]);
                    const float recv = __shfl_xor_sync(0xffffffffu, ri ? a : bb, 1);
                    const float2 Ln = ri ? make_float2(recv, bb) : make_float2(a, recv);
                    const int nn = 16 * h + n;
                    if (kInj && inj_tile && nn == n0) S = make_float2(S.x + inj.x, S.y + inj.y);
                    *reinterpret_cast<uint32_t *>(bs + (nn >> 3) * kBsSbo + (nn & 7) * 16) = pack_bf16x2(S.x, S.y);
                    S = cfma(LC, S, Ln);
                }
            }
            if ((kPack ? real_tile(v) == args.ntiles - 1 : v == nV - 1 && (!kSeg || seg == args.nseg - 1)) &&
                args.state_out && mreal)
                args.state_out[((int64_t)row_of(v) * D + d0 + ch) * args.Mt + args.m0 + m] = S;
            fence_async_smem();
            tc_fence_before();
            __syncwarp();
            if (lane == 0) {
                bar_arrive(bar(kBarSFull + cA));
                bar_arrive(bar(kBarSFull + cB));
            }
            return true;
        };
        bool ok = true;
        // State-only passes, then (segments with later ones) publish the end state
        // from a zero start: every lane stores its state, then releases its flag.
        for (int v = 0; v < nA && ok; ++v) ok = scan_tile(v);
        if (ok && nA > 0 && !(seg == 0 && *reinterpret_cast<volatile int *>(&g_stall_segment0))) {
            const int64_t at = ((seg_row + seg) * D + d0 + ch) * kModes + m;
            args.seg_state[at] = S;
            asm volatile("st.release.gpu.global.u64 [%0], %1;" ::"l"(args.seg_flag + at), "l"(args.epoch)
                         : "memory");
        }
        // Carry in for the output passes: the earlier segments' end states, each
        // advanced to the end of segment seg - 1 (full segments of seg_tiles tiles).
        if (kSeg && ok) {
            S = make_float2(0.0f, 0.0f);
            for (int r = 0; r < seg; ++r) {
                const int64_t at = ((seg_row + r) * D + d0 + ch) * kModes + m;
                if (!wait_flag(args.seg_flag + at, args.epoch, abort_flag)) {
                    ok = false;
                    break;
                }
                const float2 lr = __ldcg(args.seg_state + at);
                const float2 P = lambda_pow(m_decay, m_freq, (float)((int64_t)(seg - 1 - r) * args.seg_tiles * kTile));
                S = cfma(P, lr, S);
            }
        }
        for (int v = nA; v < nV && ok; ++v) ok = scan_tile(v);
        } else {
        // With 32 modes quarter q holds the state rows of modes 0-15 of channels
        // 2q, 2q+1 and of modes 16-31 of channels 2 (q ^ 1), 2 (q ^ 1) + 1, so each
        // channel's carried states come from two scan warps (SFull counts two).
        // Both warps of a quarter pair {q, q ^ 1} scan the channel pair of the even
        // quarter first and that of the odd quarter second, each as one chain of
        // 32 chunks like the 16-mode scan, so a pair's up-projection waits only for
        // that pair's scans.  Pass k covers channels 2 pr, 2 pr + 1 with pr =
        // 2 (q / 2) + k, at modes mo + m (mo = 0 if pr == q, else 16); lane 2m + ri
        // carries mode mo + m of channel 2 pr + ri.
        const uint32_t st_lane = 32u * (uint32_t)quarter;
        const int m = lane >> 1, ri = lane & 1;
        int chk[2], mok[2];
        bool realk[2];
        float deck[2], frqk[2];
        float2 LCk[2], Sk[2], injk[2];
        uint32_t bsk[2];
#pragma unroll
        for (int k = 0; k < 2; ++k) {
            const int pr = ((quarter >> 1) << 1) + k;
            chk[k] = 2 * pr + ri;
            mok[k] = pr == quarter ? 0 : 16;
            realk[k] = mok[k] + m < args.M;
            const int pm = (d0 + chk[k]) * args.Mt + args.m0 + mok[k] + m;
            deck[k] = realk[k] ? args.decay[pm] : 0.0f;
            frqk[k] = realk[k] ? args.freq[pm] : 0.0f;
            LCk[k] = lambda_pow(deck[k], frqk[k], (float)kC);
            Sk[k] = injk[k] = make_float2(0.0f, 0.0f);
            bsk[k] = sbase + kOffBs + chk[k] * kBsStride + ((mok[k] + m) / 4) * kBsLbo + (m % 4) * 4;
        }
        const int n0 = kInj ? (int)((-args.t0) >> 6) : -1;
        auto load_inj = [&](int row) {
            const float p = (float)(-(int)((-args.t0) & 63));
#pragma unroll
            for (int k = 0; k < 2; ++k)
                injk[k] = realk[k] ? cmul(lambda_pow(deck[k], frqk[k], p),
                                          args.state_in[((int64_t)row * D + d0 + chk[k]) * args.Mt + args.m0 + mok[k] + m])
                                   : make_float2(0.0f, 0.0f);
        };
        if (kInj && !kPack) load_inj(b);
        bool ok = true;
        for (int v = 0; v < nV && ok; ++v) {
            const bool row_start = real_tile(v) == 0;
            const bool inj_tile = kInj && row_start;
            if (kPack && row_start) {
                Sk[0] = Sk[1] = make_float2(0.0f, 0.0f);
                if (kInj) load_inj(row_of(v));
            }
#pragma unroll
            for (int k = 0; k < 2; ++k) {
                const int cA = 2 * (((quarter >> 1) << 1) + k), cB = cA + 1;
                if (!wait_bar(bar(kBarTwDone + cA), v & 1, abort_flag) ||
                    !wait_bar(bar(kBarTwDone + cB), v & 1, abort_flag)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                float2 S = Sk[k];
#pragma unroll
                for (int h = 0; h < kNT / 16; ++h) {
                    uint32_t va[16], vb[16];
                    tmem_ld16(tmem + (st_lane << 16) + cA * kNT + 16 * h, va);
                    tmem_ld16(tmem + (st_lane << 16) + cB * kNT + 16 * h, vb);
                    tmem_wait_ld();
#pragma unroll
                    for (int n = 0; n < 16; ++n) {
                        const float a = __uint_as_float(va[n]), bb = __uint_as_float(vb[n]);
                        const float recv = __shfl_xor_sync(0xffffffffu, ri ? a : bb, 1);
                        const float2 Ln = ri ? make_float2(recv, bb) : make_float2(a, recv);
                        const int nn = 16 * h + n;
                        if (kInj && inj_tile && nn == n0) S = make_float2(S.x + injk[k].x, S.y + injk[k].y);
                        asm volatile("st.shared.b32 [%0], %1;" ::"r"(bsk[k] + (nn >> 3) * kBsSbo + (nn & 7) * 16),
                                     "r"(pack_bf16x2(S.x, S.y))
                                     : "memory");
                        S = cfma(LCk[k], S, Ln);
                    }
                }
                Sk[k] = S;
                if ((kPack ? real_tile(v) == args.ntiles - 1 : v == nV - 1) && args.state_out && realk[k])
                    args.state_out[((int64_t)row_of(v) * D + d0 + chk[k]) * args.Mt + args.m0 + mok[k] + m] = S;
                fence_async_smem();
                tc_fence_before();
                __syncwarp();
                if (lane == 0) {
                    bar_arrive(bar(kBarSFull + cA));
                    bar_arrive(bar(kBarSFull + cB));
                }
            }
        }
        }
    } else if (warp < 8) {
        // ---------------------------------------------------- epilogue
        // Warp (quarter q, h) reads its quarter's Toeplitz lanes -- position
        // pos = 32 (q % 2) + lane of channels c0 .. c0+3 (c0 = 4 in quarters 0, 1
        // and 0 in quarters 2, 3) -- for chunks 16h .. 16h+15, a channel pair at a
        // time as its up-projections complete (releasing each accumulator as soon
        // as it is read), and writes the 8-byte half (channels c0 .. c0+3) of each
        // token's 16-byte row into the y ring: ring slots 2h and 2h+1 of the tile.
        const int h = warp >> 2;
        const int c0 = quarter < 2 ? 4 : 0;
        const int pos = 32 * (quarter & 1) + lane;
        const int hb = quarter < 2 ? 8 : 0;
        const uint32_t trow = tmem + ((uint32_t)(32 * quarter) << 16) + 16 * h;
        if constexpr (kMix) {
            for (int j = 0; j < nB; ++j) {
                const int ng0 = j * kYPerTile + 2 * h;
                if (!wait_bar(bar(kBarGFull + ng0 % kYSlots), (ng0 / kYSlots) & 1, abort_flag) ||
                    !wait_bar(bar(kBarGFull + (ng0 + 1) % kYSlots), ((ng0 + 1) / kYSlots) & 1, abort_flag))
                    break;
                bool ok = true;
#pragma unroll
                for (int p = 0; p < 2; ++p) {
                    const int cA = c0 + 2 * p, cB = cA + 1;
                    if (!wait_bar(bar(kBarUDone + cA), j & 1, abort_flag) ||
                        !wait_bar(bar(kBarUDone + cB), j & 1, abort_flag)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
#pragma unroll
                    for (int sh = 0; sh < 2; ++sh) {
                        uint32_t va[8], vb[8];
                        tmem_ld8(trow + cA * kNT + 8 * sh, va);
                        tmem_ld8(trow + cB * kNT + 8 * sh, vb);
                        tmem_wait_ld();
                        // The gate rows (and, once done, the z rows) of this 512-token block.
                        uint8_t *gs = smem + kOffY + ((ng0 + sh) % kYSlots) * (kYRows * 16) + hb + 4 * p;
#pragma unroll
                        for (int n8 = 0; n8 < 8; ++n8) {
                            uint32_t *gz = reinterpret_cast<uint32_t *>(gs + (n8 * kC + pos) * 16);
                            const __nv_bfloat162 g2 = *reinterpret_cast<const __nv_bfloat162 *>(gz);
                            float za = __uint_as_float(va[n8]), zb = __uint_as_float(vb[n8]);
                            if (args.add) {
                                za += __low2float(g2);
                                zb += __high2float(g2);
                            } else {
                                za *= __fdividef(1.0f, 1.0f + __expf(-__low2float(g2)));
                                zb *= __fdividef(1.0f, 1.0f + __expf(-__high2float(g2)));
                            }
                            *gz = pack_bf16x2(za, zb);
                        }
                    }
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0) {
                        bar_arrive(bar(kBarDEmpty + cA));
                        bar_arrive(bar(kBarDEmpty + cB));
                    }
                }
                if (!ok) break;
                fence_async_smem();
                __syncwarp();
                if (lane == 0) {
                    bar_arrive(bar(kBarYFull + ng0 % kYSlots));
                    bar_arrive(bar(kBarYFull + (ng0 + 1) % kYSlots));
                }
            }
        } else
        for (int j = 0; j < nB; ++j) {
            uint32_t pk[2][16];
            bool ok = true;
#pragma unroll
            for (int p = 0; p < 2; ++p) {
                const int cA = c0 + 2 * p, cB = cA + 1;
                if (!wait_bar(bar(kBarUDone + cA), j & 1, abort_flag) ||
                    !wait_bar(bar(kBarUDone + cB), j & 1, abort_flag)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
#pragma unroll
                for (int sh = 0; sh < 2; ++sh) {
                    uint32_t va[8], vb[8];
                    tmem_ld8(trow + cA * kNT + 8 * sh, va);
                    tmem_ld8(trow + cB * kNT + 8 * sh, vb);
                    tmem_wait_ld();
#pragma unroll
                    for (int n = 0; n < 8; ++n)
                        pk[p][8 * sh + n] = pack_bf16x2(__uint_as_float(va[n]), __uint_as_float(vb[n]));
                }
                tc_fence_before();
                __syncwarp();
                if (lane == 0) {
                    bar_arrive(bar(kBarDEmpty + cA));
                    bar_arrive(bar(kBarDEmpty + cB));
                }
            }
            if (!ok) break;
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
                    *reinterpret_cast<uint2 *>(ys + (n * kC + pos) * 16) = make_uint2(pk[0][8 * sh + n], pk[1][8 * sh + n]);
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

// Modes per channel of the segmented and mixer instances (their tables and the
// segment-state layout); plain and packed launches also come with 32.
constexpr int kModes16 = 16;

// Sequence segments: with fewer (batch row, channel group) CTAs than SMs, the
// sequence is cut into nseg runs of whole tiles so that nseg * B * D / 8 CTAs
// (at most one per SM, all resident at once) share the work.
struct Segments {
    int nseg, seg_tiles;
};

Segments segments(int64_t B, int64_t L, int D) {
    const int ntiles = (int)((L + kTile - 1) / kTile);
    const int64_t ctas = B * (int64_t)(D / kDG);
    // Segment offsets enter lambda^n with n below 2^24 (exact in fp32).
    int want = L > ((int64_t)1 << 24) ? 1
             : (int)std::min<int64_t>(ntiles, std::max<int64_t>(1, sm_count() / std::max<int64_t>(1, ctas)));
    Segments sg;
    sg.seg_tiles = (ntiles + want - 1) / want;
    sg.nseg = (ntiles + sg.seg_tiles - 1) / sg.seg_tiles;
    return sg;
}

size_t seg_state_bytes(int64_t B, int nseg, int D) {
    return ((size_t)B * nseg * D * kModes16 * sizeof(float2) + 255) / 256 * 256;
}

}  // namespace

bool tc_prefill_supported(int64_t B, int64_t L, int D, int M, rlm_dtype dt) {
    const bool shape = dt == RLM_BF16 && M >= 1 && D % kDG == 0 && B >= 1 && B <= 65535 && L >= 1 &&
                       L <= ((int64_t)1 << 31) - kTile && D / kDG <= 65535;
    if (!shape) return false;
    if (M <= kModes16) return true;
    // More modes (unsegmented launches only): up to 32 in one launch of the
    // 32-mode instance; beyond, passes of 16 modes, each later one adding to the
    // output of the earlier ones through the z ring.
    return M <= 4 * kModes16 && segments(B, L, D).nseg < 2;
}

bool tc_mixer_fused(int64_t B, int64_t L, int D, int M, rlm_dtype dt) {
    return M <= kModes16 && tc_prefill_supported(B, L, D, M, dt) && segments(B, L, D).nseg < 2;
}

size_t tc_prefill_ws_bytes(int64_t B, int64_t L, int D, int) {
    const Segments sg = segments(B, L, D);
    if (sg.nseg < 2) return 0;
    return 2 * seg_state_bytes(B, sg.nseg, D);  // states, then their epoch flags
}

template <int kMode>
void launch_unsegmented(bool field, bool inj, dim3 grid, const CUtensorMap &mx, const CUtensorMap &my,
                        const CUtensorMap &m2, const TcArgs &a, cudaStream_t st) {
    constexpr int sm = Cfg<16>::kSmemBytes;
    if (field) {
        if (inj)
            k_prefill_tc<kMode, true, true, 16><<<grid, kThreads, sm, st>>>(mx, my, m2, a);
        else
            k_prefill_tc<kMode, false, true, 16><<<grid, kThreads, sm, st>>>(mx, my, m2, a);
    } else if (inj) {
        k_prefill_tc<kMode, true, false, 16><<<grid, kThreads, sm, st>>>(mx, my, m2, a);
    } else {
        k_prefill_tc<kMode, false, false, 16><<<grid, kThreads, sm, st>>>(mx, my, m2, a);
    }
}

template <int kMode>
void launch_unsegmented32(bool inj, dim3 grid, const CUtensorMap &mx, const CUtensorMap &my, const TcArgs &a,
                          cudaStream_t st) {
    constexpr int sm = Cfg<32>::kSmemBytes;
    if (inj)
        k_prefill_tc<kMode, true, false, 32><<<grid, kThreads, sm, st>>>(mx, my, mx, a);
    else
        k_prefill_tc<kMode, false, false, 32><<<grid, kThreads, sm, st>>>(mx, my, mx, a);
}

// Batch rows per CTA of an unsegmented launch.  One CTA per SM (shared memory
// and TMEM), so a grid of more CTAs than SMs runs in waves, each paying the
// CTAs' prologue and pipeline fill again.  That cost is exposed only when a CTA
// has few tiles (with more, the producer fills the ring while the constants are
// built): measured at D = 256, about 6 tiles' worth for a one-tile CTA.  A CTA
// that runs several rows saves it, at a few per cent per tile (measured 5 % at
// D = 512, M = 32).  The count minimising waves * (max(0, 6 - tiles) + rows *
// tiles * cost) is taken.
int rows_per_cta(int64_t B, int D, int ntiles) {
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
        if (ctas <= sms) break;        // one wave: more rows per CTA only lengthen it
    }
    return best;
}

cudaError_t tc_prefill(const void *x, void *y, int64_t B, int64_t L, int D, int M,
                       const float *decay, const float *freq, const float *amp,
                       const float *phase, const float *state_in, float *state_out, float *coef_out,
                       const TcMix *mix, void *ws, cudaStream_t st) {
    CUtensorMap mx, my, mg;
    if (!make_field_map(&mx, x, B, L, D) || !make_field_map(&my, y, B, L, D))
        return cudaErrorInvalidValue;
    mg = mx;  // placeholder unless a gate field is given
    if (mix && (!mix->g || !make_field_map(&mg, mix->g, B, L, D))) return cudaErrorInvalidValue;
    static std::mutex mu;
    static std::vector<int> configured;
    int dev = 0;
    cudaGetDevice(&dev);
    {
        std::lock_guard<std::mutex> lock(mu);
        if ((int)configured.size() <= dev) configured.resize(dev + 1, 0);
        if (!configured[dev]) {
            const void *fns[] = {reinterpret_cast<const void *>(k_prefill_tc<kPlain, false, false, 16>),
                                 reinterpret_cast<const void *>(k_prefill_tc<kSegmented, false, false, 16>),
                                 reinterpret_cast<const void *>(k_prefill_tc<kPlain, true, false, 16>),
                                 reinterpret_cast<const void *>(k_prefill_tc<kSegmented, true, false, 16>),
                                 reinterpret_cast<const void *>(k_prefill_tc<kPlain, false, true, 16>),
                                 reinterpret_cast<const void *>(k_prefill_tc<kPlain, true, true, 16>),
                                 reinterpret_cast<const void *>(k_prefill_tc<kPacked, false, false, 16>),
                                 reinterpret_cast<const void *>(k_prefill_tc<kPacked, true, false, 16>),
                                 reinterpret_cast<const void *>(k_prefill_tc<kPacked, false, true, 16>),
                                 reinterpret_cast<const void *>(k_prefill_tc<kPacked, true, true, 16>)};
            const void *fns32[] = {reinterpret_cast<const void *>(k_prefill_tc<kPlain, false, false, 32>),
                                   reinterpret_cast<const void *>(k_prefill_tc<kPlain, true, false, 32>),
                                   reinterpret_cast<const void *>(k_prefill_tc<kPacked, false, false, 32>),
                                   reinterpret_cast<const void *>(k_prefill_tc<kPacked, true, false, 32>)};
            cudaError_t e = cudaSuccess;
            for (const void *f : fns)
                if (e == cudaSuccess)
                    e = cudaFuncSetAttribute(f, cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg<16>::kSmemBytes);
            for (const void *f : fns32)
                if (e == cudaSuccess)
                    e = cudaFuncSetAttribute(f, cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg<32>::kSmemBytes);
            if (e != cudaSuccess) return e;
            configured[dev] = 1;
        }
    }
    TcArgs a;
    a.decay = decay;
    a.freq = freq;
    a.amp = amp;
    a.phase = phase;
    a.state_in = reinterpret_cast<const float2 *>(state_in);
    a.state_out = reinterpret_cast<float2 *>(state_out);
    a.coef_out = reinterpret_cast<float4 *>(coef_out);
    a.y = static_cast<__nv_bfloat16 *>(y);
    a.L = L;
    a.D = D;
    a.M = std::min(M, kModes16);
    a.m0 = 0;
    a.Mt = M;
    a.add = 0;
    a.ntiles = (int)((L + kTile - 1) / kTile);
    a.t0 = L - (int64_t)a.ntiles * kTile;
    const Segments sg = segments(B, L, D);
    a.nseg = sg.nseg;
    a.seg_tiles = sg.seg_tiles;
    a.seg_state = nullptr;
    a.seg_flag = nullptr;
    a.epoch = 0;
    a.B = (int)B;
    a.bpc = sg.nseg < 2 ? rows_per_cta(B, D, a.ntiles) : 1;
    dim3 grid((unsigned)(D / kDG), (unsigned)((B + a.bpc - 1) / a.bpc), (unsigned)sg.nseg);
    // 16 < M <= 32: one launch of the 32-mode instance (unsegmented, no gate).
    const bool m32 = M > kModes16 && M <= 2 * kModes16;
    const int npass = m32 ? 1 : (M + kModes16 - 1) / kModes16;
    if ((mix || M > kModes16) && sg.nseg >= 2) return cudaErrorInvalidValue;  // callers check support
    if (mix && M > kModes16) return cudaErrorInvalidValue;
    if (m32) {
        a.M = M;
        if (a.bpc > 1)
            launch_unsegmented32<kPacked>(state_in != nullptr, grid, mx, my, a, st);
        else
            launch_unsegmented32<kPlain>(state_in != nullptr, grid, mx, my, a, st);
        count_launches(1);
        return cudaGetLastError();
    }
    if (sg.nseg < 2) {
        for (int p = 0; p < npass; ++p) {
            a.m0 = p * kModes16;
            a.M = std::min(kModes16, M - a.m0);
            a.add = p > 0;
            // Later passes load the output so far into the z ring and add to it.
            const CUtensorMap &m2 = p > 0 ? my : mg;
            if (a.bpc > 1) {
                launch_unsegmented<kPacked>(mix || p > 0, state_in != nullptr, grid, mx, my, m2, a, st);
            } else {
                launch_unsegmented<kPlain>(mix || p > 0, state_in != nullptr, grid, mx, my, m2, a, st);
            }
            count_launches(1);
            const cudaError_t e = cudaGetLastError();
            if (e != cudaSuccess) return e;
        }
        return cudaSuccess;
    }
    // Segments wait on the end states of earlier segments of the same rows: a
    // cooperative launch guarantees all CTAs are resident together.
    if (!ws) return cudaErrorInvalidValue;
    a.seg_state = static_cast<float2 *>(ws);
    a.seg_flag = reinterpret_cast<unsigned long long *>(static_cast<char *>(ws) + seg_state_bytes(B, sg.nseg, D));
    // Flags carry the launch's epoch, so values left by earlier launches (smaller
    // epochs) never pass for this one and the flags need no clearing.
    static std::atomic<unsigned long long> epoch{0x5eed0000ull};
    a.epoch = ++epoch;
    void *kargs[] = {&mx, &my, &mg, &a};
    const void *fn = state_in ? reinterpret_cast<const void *>(k_prefill_tc<kSegmented, true, false, 16>)
                              : reinterpret_cast<const void *>(k_prefill_tc<kSegmented, false, false, 16>);
    cudaError_t e = cudaLaunchCooperativeKernel(fn, grid, dim3(kThreads), kargs, (size_t)Cfg<16>::kSmemBytes, st);
    count_launches(1);
    return e;
}

cudaError_t set_segment_stall(int on) {
    const long long limit = on ? 2000000ll : kWaitLimitDefault;   // about 1 ms, or about 2 s
    cudaError_t e = cudaMemcpyToSymbol(g_wait_limit_cycles, &limit, sizeof(limit));
    if (e == cudaSuccess) e = cudaMemcpyToSymbol(g_stall_segment0, &on, sizeof(on));
    return e;
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
