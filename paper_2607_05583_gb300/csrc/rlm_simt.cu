// rlm_simt.cu -- chunked complex-diagonal scan on the CUDA cores (fp32).
//
// Runs the fp32-I/O prefill, every shape the tensor-core path does not cover,
// and the backward pass.  Three phases, each one launch:
//
//  1. chunk-local states: per (b, chunk k, d) and mode m, the state the chunk's
//     own drives leave at its last token when it starts from zero
//     (sum_j lambda^(C-1-j) x_j, the chunk form of the terminal state of
//     Sec. 3.2);
//  2. inter-chunk carry: per (b, d, m), a sequential scan over chunks,
//     S_k = lambda^C S_{k-1} + local_k, written back exclusive (the state each
//     chunk starts from) -- the final S is the prompt's terminal state;
//  3. chunk output: per (b, k, d), the recurrence of Eq. 4 restarted from the
//     carried state, with the readout y_t = sum_m Re(c s_t).
//
// Chunks are aligned to END at the last token: the first chunk may start at a
// negative time, whose drives count as zero.  With a zero initial state that
// leaves every state unchanged, so the carry needs no special last chunk.
//
// The backward pass runs the same phases in reverse time on dy (the adjoint of
// a causal convolution is the anti-causal one) and carries the Jordan partner
// R of the adjoint state as well, to form G = sum x S and P = sum x R.
#include <algorithm>

#include "rlm_device.cuh"
#include "rlm_internal.h"

namespace rlm {
namespace {

constexpr int kMgFwd = 16;  // modes per thread, forward phases
constexpr int kMgBwd = 8;   // modes per thread, backward output phase
constexpr int kBlock = 128;
constexpr int kTokBlock = 8;   // drives loaded ahead per thread in the per-token loops
constexpr int kCarryBlock = 64; // threads per block of the carry (one per (b, d, m): spread over all SMs)

int threads_per_channel(int M, int mg) {
    int t = (M + mg - 1) / mg;
    int p = 1;
    while (p < t) p <<= 1;
    return p;
}

struct ChunkGeom {
    int C;        // chunk length
    int nch;      // number of chunks
    int64_t t0;   // processing time of chunk 0's first token (<= 0)
};

ChunkGeom geom_c(int64_t L, int C) {
    ChunkGeom g;
    g.C = C;
    g.nch = (int)((L + g.C - 1) / g.C);
    g.t0 = L - (int64_t)g.nch * g.C;
    return g;
}

// The backward pass does ~26 M flop per token-channel in its two per-token
// phases, so it needs far fewer (b, chunk, channel) tuples than the forward to
// fill the GPU; longer chunks keep its workspace (16 bytes per (b, chunk, d, m))
// small enough to stay in L2 and shorten the sequential carry and the reduction.
int bwd_chunk_len(int64_t B, int64_t L, int D) {
    const int64_t target = (int64_t)sm_count() * 512;
    const int64_t per_chunk = std::max<int64_t>(1, B * (int64_t)D);
    int64_t nch = std::max<int64_t>(1, (target + per_chunk - 1) / per_chunk);
    int64_t C = (L + nch - 1) / nch;
    C = std::max<int64_t>(16, std::min<int64_t>(4096, C));
    return (int)C;
}

ChunkGeom geom(int64_t B, int64_t L, int D) {
    ChunkGeom g;
    g.C = simt_chunk_len(B, L, D);
    g.nch = (int)((L + g.C - 1) / g.C);
    g.t0 = L - (int64_t)g.nch * g.C;
    return g;
}

// Phase 1.  Grid (ceil(D*TPC/kBlock), nch, B).
template <typename T, int MG, bool REV, bool JORDAN>
__global__ void __launch_bounds__(kBlock) k_chunk_local(
    const T *__restrict__ x, int64_t L, int D, int M, int tpc, int C, int nch, int64_t t0,
    const float *__restrict__ decay, const float *__restrict__ freq, float2 *__restrict__ ws_s,
    float2 *__restrict__ ws_r) {
    const int gx = blockIdx.x * blockDim.x + threadIdx.x;
    const int d = gx / tpc, grp = gx % tpc;
    const int k = blockIdx.y, b = blockIdx.z;
    if (d >= D) return;
    float2 lam[MG], s[MG], r[MG];
#pragma unroll
    for (int j = 0; j < MG; ++j) {
        const int m = grp * MG + j;
        lam[j] = m < M ? lambda_pow(decay[d * M + m], freq[d * M + m], 1.0f) : make_float2(0, 0);
        s[j] = make_float2(0, 0);
        r[j] = make_float2(0, 0);
    }
    const int64_t tau0 = t0 + (int64_t)k * C;
    const int i0 = tau0 < 0 ? (int)(-tau0) : 0;
    // kTokBlock tokens' drives are loaded before their updates run.
    for (int i = i0; i < C; i += kTokBlock) {
        float xs[kTokBlock];
#pragma unroll
        for (int u = 0; u < kTokBlock; ++u) {
            const int64_t tau = tau0 + i + u;
            const int64_t t = REV ? (L - 1 - tau) : tau;
            xs[u] = i + u < C ? ld_elem(x + ((int64_t)b * L + t) * D + d) : 0.0f;
        }
#pragma unroll
        for (int u = 0; u < kTokBlock; ++u) {
            if (i + u >= C) break;
#pragma unroll
            for (int j = 0; j < MG; ++j) {
                if (JORDAN) r[j] = cmul(lam[j], make_float2(r[j].x + s[j].x, r[j].y + s[j].y));
                s[j] = cfma(lam[j], s[j], make_float2(xs[u], 0.0f));
            }
        }
    }
    const int64_t base = (((int64_t)b * nch + k) * D + d) * M;
#pragma unroll
    for (int j = 0; j < MG; ++j) {
        const int m = grp * MG + j;
        if (m < M) {
            ws_s[base + m] = s[j];
            if (JORDAN) ws_r[base + m] = r[j];
        }
    }
}

// Phase 2.  One thread per (b, d, m); grid over B*D*M.
// With state_in (forward only): chunk 0 is entered with the state before token 0
// (the output phase restarts its recurrence there, at time 0), and that state
// reaches the end of chunk 0 after C + t0 tokens.
template <bool JORDAN>
__global__ void __launch_bounds__(kCarryBlock) k_chunk_carry(
    int64_t B, int D, int M, int C, int nch, int64_t t0, const float *__restrict__ decay,
    const float *__restrict__ freq, const float *__restrict__ amp, const float *__restrict__ phase,
    float2 *__restrict__ ws_s, float2 *__restrict__ ws_r, const float2 *__restrict__ state_in,
    float2 *__restrict__ state_out, float4 *__restrict__ coef_out) {
    const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (idx >= B * D * M) return;
    const int m = (int)(idx % M);
    const int d = (int)((idx / M) % D);
    const int64_t b = idx / ((int64_t)M * D);
    const int pm = d * M + m;
    const float2 LC = lambda_pow(decay[pm], freq[pm], (float)C);
    const float Cf = (float)C;
    float2 S = state_in ? state_in[idx] : make_float2(0, 0), R = make_float2(0, 0);
    const float2 L0 = state_in ? lambda_pow(decay[pm], freq[pm], (float)(C + t0)) : LC;
    // The chunks' partials are read kCarryBatch at a time before the recurrence
    // runs over them (each slot is then overwritten with the state entering its
    // chunk), so a thread waits on memory once per batch, not once per chunk.
    constexpr int kCB = JORDAN ? 16 : 32;
    const int64_t stride = (int64_t)D * M;
    const int64_t off0 = (b * nch * D + d) * M + m;   // chunk 0; chunk k at off0 + k * stride
    for (int k0 = 0; k0 < nch; k0 += kCB) {
        float2 lsv[kCB], lrv[JORDAN ? kCB : 1];
#pragma unroll
        for (int j = 0; j < kCB; ++j) {
            if (k0 + j < nch) {
                lsv[j] = ws_s[off0 + (k0 + j) * stride];
                if (JORDAN) lrv[j] = ws_r[off0 + (k0 + j) * stride];
            }
        }
#pragma unroll
        for (int j = 0; j < kCB; ++j) {
            if (k0 + j >= nch) break;
            const int64_t off = off0 + (k0 + j) * stride;
            ws_s[off] = S;
            if (JORDAN) {
                ws_r[off] = R;
                R = cfma(LC, make_float2(fmaf(Cf, S.x, R.x), fmaf(Cf, S.y, R.y)), lrv[j]);
            }
            S = cfma(k0 + j == 0 ? L0 : LC, S, lsv[j]);
        }
    }
    if (state_out) state_out[idx] = S;
    if (coef_out && b == 0) {
        const float2 lam = lambda_pow(decay[pm], freq[pm], 1.0f);
        const float2 c = mode_coef(amp[pm], phase[pm]);
        coef_out[pm] = make_float4(lam.x, lam.y, c.x, c.y);
    }
}

// Phase 3 (forward).  Grid (ceil(D*TPC/kBlock), nch, B); the TPC threads of a
// channel split its modes and add their readouts with shuffles.
template <typename T, int MG, bool REV>
__global__ void __launch_bounds__(kBlock) k_chunk_output(
    const T *__restrict__ x, T *__restrict__ y, int64_t L, int D, int M, int tpc, int C, int nch,
    int64_t t0, const float *__restrict__ decay, const float *__restrict__ freq,
    const float *__restrict__ amp, const float *__restrict__ phase,
    const float2 *__restrict__ ws_s) {
    const int gx = blockIdx.x * blockDim.x + threadIdx.x;
    const int d = gx / tpc, grp = gx % tpc;
    const int k = blockIdx.y, b = blockIdx.z;
    const bool active = d < D;
    float2 lam[MG], c[MG], s[MG];
    const int64_t base = (((int64_t)b * nch + k) * D + d) * M;
#pragma unroll
    for (int j = 0; j < MG; ++j) {
        const int m = grp * MG + j;
        const bool on = active && m < M;
        lam[j] = on ? lambda_pow(decay[d * M + m], freq[d * M + m], 1.0f) : make_float2(0, 0);
        c[j] = on ? mode_coef(amp[d * M + m], phase[d * M + m]) : make_float2(0, 0);
        s[j] = on ? ws_s[base + m] : make_float2(0, 0);
    }
    const int64_t tau0 = t0 + (int64_t)k * C;
    const int i0 = tau0 < 0 ? (int)(-tau0) : 0;
    auto at = [&](int i) {
        const int64_t tau = tau0 + i;
        return ((int64_t)b * L + (REV ? (L - 1 - tau) : tau)) * D + d;
    };
    // kTokBlock tokens' drives are loaded before their updates run (the trip
    // counts are uniform across the warp, so every lane reaches the shuffles).
    for (int i = i0; i < C; i += kTokBlock) {
        float xs[kTokBlock];
#pragma unroll
        for (int u = 0; u < kTokBlock; ++u) xs[u] = active && i + u < C ? ld_elem(x + at(i + u)) : 0.0f;
#pragma unroll
        for (int u = 0; u < kTokBlock; ++u) {
            if (i + u >= C) break;
            float acc = 0.0f;
#pragma unroll
            for (int j = 0; j < MG; ++j) {
                s[j] = cfma(lam[j], s[j], make_float2(xs[u], 0.0f));
                acc = fmaf(c[j].x, s[j].x, fmaf(-c[j].y, s[j].y, acc));
            }
            for (int o = tpc >> 1; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
            if (active && grp == 0) st_elem(y + at(i + u), acc);
        }
    }
}

// Optional state terms of the backward (all [B][D][M] complex, null = absent).
struct StateTerms {
    const float2 *state_in;   // the forward's state before token 0
    const float2 *g;          // the loss gradient of the terminal state
    float2 *d_state_in;       // output: the loss gradient of state_in
    float2 *ws_j;             // with g: per-chunk partials of conj(g) J, next to ws_s / ws_r
};

// Phase 3 (backward).  Reverse time over dy; writes dx and, in place of the
// carried (S, R), the chunk's partial sums G = sum x S and P = sum x R.
// kG (a terminal-state gradient g): the second adjoint Phi_t = lambda^(L-1-t)
// conj(g) joins dx with readout 1, and J = sum x_t (L-1-t) lambda^(L-1-t) (the unit
// adjoint U and its Jordan partner Q, both closed-form at the chunk start) gives the
// partials conj(g) J.  The chunk that ends at token 0 holds S_0 and R_0: it adds the
// initial state's terms s_in lambda S_0 to G and s_in lambda (R_0 + S_0) to P (and
// conj(g) L lambda^L s_in to its J partial) and writes the gradient of s_in,
// conj(c lambda S_0) + g conj(lambda^L).
template <typename T, int MG, bool kG>
__global__ void __launch_bounds__(kBlock) k_chunk_backward(
    const T *__restrict__ dy, const T *__restrict__ x, T *__restrict__ dx, int64_t L, int D,
    int M, int tpc, int C, int nch, int64_t t0, const float *__restrict__ decay,
    const float *__restrict__ freq, const float *__restrict__ amp,
    const float *__restrict__ phase, float2 *__restrict__ ws_s, float2 *__restrict__ ws_r,
    const StateTerms stt) {
    const int gx = blockIdx.x * blockDim.x + threadIdx.x;
    const int d = gx / tpc, grp = gx % tpc;
    const int k = blockIdx.y, b = blockIdx.z;
    const bool active = d < D;
    float2 lam[MG], c[MG], s[MG], r[MG], G[MG], P[MG];
    float2 phi[MG], U[MG], Q[MG], J[MG];
    const int64_t base = (((int64_t)b * nch + k) * D + d) * M;
    const int64_t tau0 = t0 + (int64_t)k * C;
    const int i0 = tau0 < 0 ? (int)(-tau0) : 0;
#pragma unroll
    for (int j = 0; j < MG; ++j) {
        const int m = grp * MG + j;
        const bool on = active && m < M;
        lam[j] = on ? lambda_pow(decay[d * M + m], freq[d * M + m], 1.0f) : make_float2(0, 0);
        c[j] = on ? mode_coef(amp[d * M + m], phase[d * M + m]) : make_float2(0, 0);
        s[j] = on ? ws_s[base + m] : make_float2(0, 0);
        r[j] = on ? ws_r[base + m] : make_float2(0, 0);
        G[j] = make_float2(0, 0);
        P[j] = make_float2(0, 0);
        if (kG) {
            // At the first position (time L-1-tau, tau = tau0 + i0): lambda^tau.
            const float n = (float)(tau0 + i0);
            U[j] = on ? lambda_pow(decay[d * M + m], freq[d * M + m], n) : make_float2(0, 0);
            Q[j] = make_float2(n * U[j].x, n * U[j].y);
            const float2 gg = on ? stt.g[((int64_t)b * D + d) * M + m] : make_float2(0, 0);
            phi[j] = cmul(U[j], make_float2(gg.x, -gg.y));
            J[j] = make_float2(0, 0);
        }
    }
    // The next token's drives are loaded before this token's arithmetic.
    auto at = [&](int i) { return ((int64_t)b * L + (L - 1 - (tau0 + i))) * D + d; };
    float u_next = active && i0 < C ? ld_elem(dy + at(i0)) : 0.0f;
    float x_next = active && i0 < C ? ld_elem(x + at(i0)) : 0.0f;
    for (int i = i0; i < C; ++i) {
        const int64_t e = at(i);
        const float u = u_next, xv = x_next;
        if (active && i + 1 < C) {
            u_next = ld_elem(dy + at(i + 1));
            x_next = ld_elem(x + at(i + 1));
        }
        float acc = 0.0f;
#pragma unroll
        for (int j = 0; j < MG; ++j) {
            r[j] = cmul(lam[j], make_float2(r[j].x + s[j].x, r[j].y + s[j].y));
            s[j] = cfma(lam[j], s[j], make_float2(u, 0.0f));
            acc = fmaf(c[j].x, s[j].x, fmaf(-c[j].y, s[j].y, acc));
            G[j].x = fmaf(xv, s[j].x, G[j].x);
            G[j].y = fmaf(xv, s[j].y, G[j].y);
            P[j].x = fmaf(xv, r[j].x, P[j].x);
            P[j].y = fmaf(xv, r[j].y, P[j].y);
            if (kG) {
                acc += phi[j].x;
                J[j].x = fmaf(xv, Q[j].x, J[j].x);
                J[j].y = fmaf(xv, Q[j].y, J[j].y);
                phi[j] = cmul(lam[j], phi[j]);
                Q[j] = cmul(lam[j], make_float2(Q[j].x + U[j].x, Q[j].y + U[j].y));
                U[j] = cmul(lam[j], U[j]);
            }
        }
        for (int o = tpc >> 1; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
        if (active && grp == 0) st_elem(dx + e, acc);
    }
    const bool first_token = k == nch - 1;   // this chunk ends at token 0
#pragma unroll
    for (int j = 0; j < MG; ++j) {
        const int m = grp * MG + j;
        if (active && m < M) {
            const int64_t sm = ((int64_t)b * D + d) * M + m;
            const float2 gg = kG ? stt.g[sm] : make_float2(0, 0);
            float2 gj = kG ? cmul(make_float2(gg.x, -gg.y), J[j]) : make_float2(0, 0);
            if (first_token) {
                const float2 ls = cmul(lam[j], s[j]);   // lambda S_0
                if (stt.state_in) {
                    const float2 si = stt.state_in[sm];
                    G[j] = cfma(si, ls, G[j]);
                    P[j] = cfma(si, cmul(lam[j], make_float2(r[j].x + s[j].x, r[j].y + s[j].y)), P[j]);
                    if (kG) {
                        const float2 lL = lambda_pow(decay[d * M + m], freq[d * M + m], (float)L);
                        const float2 jin = cmul(si, lL);
                        gj = cfma(make_float2(gg.x, -gg.y), make_float2((float)L * jin.x, (float)L * jin.y), gj);
                    }
                }
                if (stt.d_state_in) {
                    const float2 cl = cmul(c[j], ls);
                    float2 ds = make_float2(cl.x, -cl.y);
                    if (kG) {
                        const float2 lL = lambda_pow(decay[d * M + m], freq[d * M + m], (float)L);
                        ds = cfma(gg, make_float2(lL.x, -lL.y), ds);
                    }
                    stt.d_state_in[sm] = ds;
                }
            }
            ws_s[base + m] = G[j];
            ws_r[base + m] = P[j];
            if (kG) stt.ws_j[base + m] = gj;
        }
    }
}

// Phase 4 (backward).  One thread per (d, m): fixed-order sum of the partials
// over (b, k), then the four gradients.  The sums are compensated (Kahan) fp32
// sums, so the result is reproducible and its error stays near one rounding
// however many chunk partials the SIMT path adds; the combination with
// c = A e^{i phi} (formed as the forward forms it, fp32 sincosf) uses fmaf for
// the differences.  Double precision made this launch 3-4x slower on this part
// (low FP64 rate): 4.8 against 1.4 us at D = 512, M = 32, four partials.
// ws_j (nullable): partials of conj(g) J from a terminal-state gradient, which
// add -Re and -Im of their sum to dgamma and domega.
struct KahanSum {
    float s = 0.0f, c = 0.0f;
    __device__ __forceinline__ void add(float v) {
        const float y = v - c;
        const float t = s + y;
        c = (t - s) - y;
        s = t;
    }
};
__global__ void __launch_bounds__(256) k_grad_reduce(
    int64_t B, int D, int M, int nch, const float *__restrict__ amp,
    const float *__restrict__ phase, const float2 *__restrict__ ws_s,
    const float2 *__restrict__ ws_r, const float2 *__restrict__ ws_j, float *__restrict__ g_decay,
    float *__restrict__ g_freq, float *__restrict__ g_amp, float *__restrict__ g_phase) {
    const int pm = blockIdx.x * blockDim.x + threadIdx.x;
    if (pm >= D * M) return;
    const float am = amp[pm], ph = phase[pm];
    KahanSum gr, gi, pr, pi, jr, ji;
    const int64_t n = B * nch, stride = (int64_t)D * M;
    // Four partials' loads in flight before their adds (the sum order is fixed).
    for (int64_t bk0 = 0; bk0 < n; bk0 += 4) {
        float2 g[4], p[4], j[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int64_t off = (bk0 + u) * stride + pm;
            const bool in = bk0 + u < n;
            g[u] = in ? ws_s[off] : make_float2(0.0f, 0.0f);
            p[u] = in ? ws_r[off] : make_float2(0.0f, 0.0f);
            j[u] = in && ws_j ? ws_j[off] : make_float2(0.0f, 0.0f);
        }
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            if (bk0 + u >= n) break;
            gr.add(g[u].x);
            gi.add(g[u].y);
            pr.add(p[u].x);
            pi.add(p[u].y);
            if (ws_j) {
                jr.add(j[u].x);
                ji.add(j[u].y);
            }
        }
    }
    float sph, cph;
    sincosf(ph, &sph, &cph);
    const float cr = am * cph, ci = am * sph;
    g_amp[pm] = fmaf(cph, gr.s, -sph * gi.s);            // Re(e^{i phi} G)
    g_phase[pm] = -fmaf(cr, gi.s, ci * gr.s);            // -Im(c G)
    g_decay[pm] = -fmaf(cr, pr.s, -ci * pi.s) - jr.s;    // -Re(c P) - Re(conj(g) J)
    g_freq[pm] = -fmaf(cr, pi.s, ci * pr.s) - ji.s;      // -Im(c P) - Im(conj(g) J)
}

template <typename T>
cudaError_t prefill_t(const T *x, T *y, int64_t B, int64_t L, int D, int M, const float *decay,
                      const float *freq, const float *amp, const float *phase, const float *state_in,
                      float *state_out, float *coef_out, void *ws, cudaStream_t st) {
    const ChunkGeom g = geom(B, L, D);
    const int tpc = threads_per_channel(M, kMgFwd);
    float2 *ws_s = reinterpret_cast<float2 *>(ws);
    dim3 grid((unsigned)((D * tpc + kBlock - 1) / kBlock), (unsigned)g.nch, (unsigned)B);
    k_chunk_local<T, kMgFwd, false, false><<<grid, kBlock, 0, st>>>(
        x, L, D, M, tpc, g.C, g.nch, g.t0, decay, freq, ws_s, nullptr);
    const int64_t n = B * D * M;
    k_chunk_carry<false><<<(unsigned)((n + kCarryBlock - 1) / kCarryBlock), kCarryBlock, 0, st>>>(
        B, D, M, g.C, g.nch, g.t0, decay, freq, amp, phase, ws_s, nullptr,
        reinterpret_cast<const float2 *>(state_in), reinterpret_cast<float2 *>(state_out),
        reinterpret_cast<float4 *>(coef_out));
    k_chunk_output<T, kMgFwd, false><<<grid, kBlock, 0, st>>>(
        x, y, L, D, M, tpc, g.C, g.nch, g.t0, decay, freq, amp, phase, ws_s);
    count_launches(3);
    return cudaGetLastError();
}

template <typename T>
cudaError_t backward_t(const T *dy, const T *x, T *dx, int64_t B, int64_t L, int D, int M,
                       const float *decay, const float *freq, const float *amp,
                       const float *phase, const float *state_in, const float *d_state_out,
                       float *d_state_in, float *gd, float *gf, float *ga, float *gp, void *ws,
                       cudaStream_t st) {
    const ChunkGeom g = geom_c(L, bwd_chunk_len(B, L, D));
    const int64_t n = B * (int64_t)g.nch * D * M;
    float2 *ws_s = reinterpret_cast<float2 *>(ws);
    float2 *ws_r = ws_s + n;
    StateTerms stt;
    stt.state_in = reinterpret_cast<const float2 *>(state_in);
    stt.g = reinterpret_cast<const float2 *>(d_state_out);
    stt.d_state_in = reinterpret_cast<float2 *>(d_state_in);
    stt.ws_j = d_state_out ? ws_r + n : nullptr;
    const int tpc1 = threads_per_channel(M, kMgFwd);
    dim3 grid1((unsigned)((D * tpc1 + kBlock - 1) / kBlock), (unsigned)g.nch, (unsigned)B);
    k_chunk_local<T, kMgFwd, true, true><<<grid1, kBlock, 0, st>>>(
        dy, L, D, M, tpc1, g.C, g.nch, g.t0, decay, freq, ws_s, ws_r);
    const int64_t nbdm = B * D * M;
    k_chunk_carry<true><<<(unsigned)((nbdm + kCarryBlock - 1) / kCarryBlock), kCarryBlock, 0, st>>>(
        B, D, M, g.C, g.nch, g.t0, decay, freq, amp, phase, ws_s, ws_r, nullptr, nullptr, nullptr);
    const int tpc3 = threads_per_channel(M, kMgBwd);
    dim3 grid3((unsigned)((D * tpc3 + kBlock - 1) / kBlock), (unsigned)g.nch, (unsigned)B);
    if (d_state_out)
        k_chunk_backward<T, kMgBwd, true><<<grid3, kBlock, 0, st>>>(
            dy, x, dx, L, D, M, tpc3, g.C, g.nch, g.t0, decay, freq, amp, phase, ws_s, ws_r, stt);
    else
        k_chunk_backward<T, kMgBwd, false><<<grid3, kBlock, 0, st>>>(
            dy, x, dx, L, D, M, tpc3, g.C, g.nch, g.t0, decay, freq, amp, phase, ws_s, ws_r, stt);
    k_grad_reduce<<<(unsigned)((D * M + 255) / 256), 256, 0, st>>>(
        B, D, M, g.nch, amp, phase, ws_s, ws_r, stt.ws_j, gd, gf, ga, gp);
    count_launches(4);
    return cudaGetLastError();
}

}  // namespace

int simt_chunk_len(int64_t B, int64_t L, int D) {
    // Enough (b, chunk, channel) threads for about two full waves of 1024
    // resident threads per SM; chunks of 16..1024 tokens.
    const int64_t target = (int64_t)sm_count() * 2048;
    const int64_t per_chunk = std::max<int64_t>(1, B * (int64_t)D);
    int64_t nch = (target + per_chunk - 1) / per_chunk;
    nch = std::max<int64_t>(1, nch);
    int64_t C = (L + nch - 1) / nch;
    C = std::max<int64_t>(16, std::min<int64_t>(1024, C));
    return (int)C;
}

size_t simt_prefill_ws_bytes(int64_t B, int64_t L, int D, int M) {
    const ChunkGeom g = geom(B, L, D);
    return (size_t)B * g.nch * D * M * sizeof(float2);
}

size_t simt_backward_ws_bytes(int64_t B, int64_t L, int D, int M) {
    const ChunkGeom g = geom_c(L, bwd_chunk_len(B, L, D));
    return 3 * (size_t)B * g.nch * D * M * sizeof(float2);   // G, P and conj(g) J partials
}

cudaError_t simt_prefill(const void *x, void *y, rlm_dtype dt, int64_t B, int64_t L, int D,
                         int M, const float *decay, const float *freq, const float *amp,
                         const float *phase, const float *state_in, float *state_out, float *coef_out,
                         void *ws, cudaStream_t st) {
    if (dt == RLM_BF16)
        return prefill_t(static_cast<const __nv_bfloat16 *>(x), static_cast<__nv_bfloat16 *>(y),
                         B, L, D, M, decay, freq, amp, phase, state_in, state_out, coef_out, ws, st);
    return prefill_t(static_cast<const float *>(x), static_cast<float *>(y), B, L, D, M, decay,
                     freq, amp, phase, state_in, state_out, coef_out, ws, st);
}

cudaError_t grad_reduce(int64_t nparts, int D, int M, const float *amp, const float *phase,
                        const float2 *G, const float2 *P, const float2 *J, float *g_decay, float *g_freq,
                        float *g_amp, float *g_phase, cudaStream_t st) {
    k_grad_reduce<<<(unsigned)((D * M + 255) / 256), 256, 0, st>>>(
        nparts, D, M, 1, amp, phase, G, P, J, g_decay, g_freq, g_amp, g_phase);
    count_launches(1);
    return cudaGetLastError();
}

cudaError_t simt_backward(const void *dy, const void *x, void *dx, rlm_dtype dt, int64_t B,
                          int64_t L, int D, int M, const float *decay, const float *freq,
                          const float *amp, const float *phase, const float *state_in,
                          const float *d_state_out, float *d_state_in, float *g_decay, float *g_freq,
                          float *g_amp, float *g_phase, void *ws, cudaStream_t st) {
    if (dt == RLM_BF16)
        return backward_t(static_cast<const __nv_bfloat16 *>(dy),
                          static_cast<const __nv_bfloat16 *>(x), static_cast<__nv_bfloat16 *>(dx),
                          B, L, D, M, decay, freq, amp, phase, state_in, d_state_out, d_state_in, g_decay,
                          g_freq, g_amp, g_phase, ws, st);
    return backward_t(static_cast<const float *>(dy), static_cast<const float *>(x),
                      static_cast<float *>(dx), B, L, D, M, decay, freq, amp, phase, state_in, d_state_out,
                      d_state_in, g_decay, g_freq, g_amp, g_phase, ws, st);
}

}  // namespace rlm
