// rlm_abi.cu -- the extern "C" boundary: host-side argument checks, workspace
// sizing and dispatch to the kernels.  Nothing here allocates device memory.
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <atomic>
#include <mutex>
#include <vector>

#include "rlm_internal.h"

namespace rlm {

static thread_local char g_err[512] = "";
static std::atomic<unsigned long long> g_launches{0};

void count_launches(int n) { g_launches.fetch_add((unsigned long long)n, std::memory_order_relaxed); }

void set_error(const char *fmt, ...) {
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(g_err, sizeof(g_err), fmt, ap);
    va_end(ap);
}

int sm_count() {
    static std::mutex mu;
    static std::vector<int> cache;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return 148;
    std::lock_guard<std::mutex> lock(mu);
    if ((int)cache.size() <= dev) cache.resize(dev + 1, 0);
    if (cache[dev] == 0) {
        int n = 0;
        if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0)
            n = 148;
        cache[dev] = n;
    }
    return cache[dev];
}

}  // namespace rlm

using namespace rlm;

namespace {

constexpr int kMaxModes = 64;

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

size_t elem_size(rlm_dtype dt) { return dt == RLM_BF16 ? 2 : 4; }

rlm_status fail(rlm_status s, const char *fmt, ...) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof(buf), fmt, ap);
    va_end(ap);
    set_error("%s", buf);
    return s;
}

rlm_status cuda_fail(cudaError_t e, const char *what) {
    return fail(RLM_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

rlm_status check_tensor(const rlm_tensor *t, const char *name) {
    if (!t) return fail(RLM_ERR_INVALID_ARG, "%s is NULL", name);
    if (!t->ptr) return fail(RLM_ERR_INVALID_ARG, "%s->ptr is NULL", name);
    if (!aligned16(t->ptr)) return fail(RLM_ERR_INVALID_ARG, "%s->ptr is not 16-byte aligned", name);
    if (t->dtype != RLM_F32 && t->dtype != RLM_BF16)
        return fail(RLM_ERR_INVALID_ARG, "%s->dtype %d is not RLM_F32 or RLM_BF16", name, (int)t->dtype);
    if (t->B < 1 || t->L < 1)
        return fail(RLM_ERR_INVALID_ARG, "%s has B=%lld L=%lld (need >= 1)", name, (long long)t->B,
                    (long long)t->L);
    if (t->D < 8 || t->D % 8 != 0)
        return fail(RLM_ERR_INVALID_ARG, "%s has D=%lld (need D >= 8 and D %% 8 == 0)", name,
                    (long long)t->D);
    if (t->D > (1 << 20)) return fail(RLM_ERR_UNSUPPORTED, "%s has D=%lld > 2^20", name, (long long)t->D);
    if (t->B > 65535) return fail(RLM_ERR_UNSUPPORTED, "%s has B=%lld > 65535", name, (long long)t->B);
    // lambda^n is formed from fp32 token counts n, exact up to 2^24.
    if (t->L > (int64_t)1 << 24)
        return fail(RLM_ERR_UNSUPPORTED, "%s has L=%lld > 2^24", name, (long long)t->L);
    return RLM_OK;
}

bool same_shape(const rlm_tensor *a, const rlm_tensor *b) {
    return a->B == b->B && a->L == b->L && a->D == b->D && a->dtype == b->dtype;
}

size_t tensor_bytes(const rlm_tensor *t) {
    return (size_t)t->B * (size_t)t->L * (size_t)t->D * elem_size(t->dtype);
}

bool overlap(const void *a, size_t na, const void *b, size_t nb) {
    const char *pa = static_cast<const char *>(a), *pb = static_cast<const char *>(b);
    return pa < pb + nb && pb < pa + na;
}

rlm_status check_params(const rlm_params *p, int64_t D) {
    if (!p) return fail(RLM_ERR_INVALID_ARG, "params is NULL");
    const float *ps[4] = {p->decay, p->freq, p->amp, p->phase};
    const char *nm[4] = {"decay", "freq", "amp", "phase"};
    for (int i = 0; i < 4; ++i) {
        if (!ps[i]) return fail(RLM_ERR_INVALID_ARG, "params->%s is NULL", nm[i]);
        if (!aligned16(ps[i])) return fail(RLM_ERR_INVALID_ARG, "params->%s is not 16-byte aligned", nm[i]);
    }
    if (p->M < 1 || p->M > kMaxModes)
        return fail(RLM_ERR_INVALID_ARG, "params->M=%d outside 1..%d", p->M, kMaxModes);
    if (p->D != D) return fail(RLM_ERR_INVALID_ARG, "params->D=%d does not match D=%lld", p->D, (long long)D);
    return RLM_OK;
}

rlm_status check_state(const rlm_state *s, int64_t B, int64_t D, int M, const char *name) {
    if (!s->s || !s->coef) return fail(RLM_ERR_INVALID_ARG, "%s has a NULL s or coef", name);
    if (!aligned16(s->s) || !aligned16(s->coef))
        return fail(RLM_ERR_INVALID_ARG, "%s buffers are not 16-byte aligned", name);
    if (s->B != B || s->D != D || s->M != M)
        return fail(RLM_ERR_INVALID_ARG, "%s is [B=%d][D=%d][M=%d], expected [%lld][%lld][%d]", name,
                    s->B, s->D, s->M, (long long)B, (long long)D, M);
    return RLM_OK;
}

rlm_status check_workspace(const rlm_launch *ln, size_t need) {
    if (!ln) return fail(RLM_ERR_INVALID_ARG, "launch is NULL");
    if (need == 0) return RLM_OK;
    if (!ln->workspace) return fail(RLM_ERR_INVALID_ARG, "workspace is NULL but %zu bytes are needed", need);
    if ((reinterpret_cast<uintptr_t>(ln->workspace) & 255u) != 0)
        return fail(RLM_ERR_INVALID_ARG, "workspace is not 256-byte aligned");
    if (ln->workspace_bytes < need)
        return fail(RLM_ERR_INVALID_ARG, "workspace has %zu bytes, %zu needed", ln->workspace_bytes, need);
    return RLM_OK;
}

int simt_chunks(int64_t B, int64_t L, int D) {
    const int C = simt_chunk_len(B, L, D);
    return (int)((L + C - 1) / C);
}

// The complex [B][D][M] buffer of an optional state argument (only ->s is used).
rlm_status check_state_s(const rlm_state *st, int64_t B, int64_t D, int M, const char *name) {
    if (!st) return RLM_OK;
    if (!st->s || !aligned16(st->s)) return fail(RLM_ERR_INVALID_ARG, "%s->s is NULL or not 16-byte aligned", name);
    if (st->B != B || st->D != D || st->M != M)
        return fail(RLM_ERR_INVALID_ARG, "%s is [B=%d][D=%d][M=%d], expected [%lld][%lld][%d]", name, st->B, st->D,
                    st->M, (long long)B, (long long)D, M);
    return RLM_OK;
}

// state_in / state_out of a prefill writing the field y: shapes, and no partial
// overlap (state_out may be state_in itself).
rlm_status check_prefill_states(const rlm_tensor *x, const rlm_tensor *y, const rlm_params *p,
                                const rlm_state *state_in, const rlm_state *state_out) {
    rlm_status s;
    if (state_out && (s = check_state(state_out, x->B, x->D, p->M, "state_out")) != RLM_OK) return s;
    const size_t sbytes = (size_t)x->B * x->D * p->M * 8;
    if (state_out) {
        const size_t cbytes = (size_t)x->D * p->M * 16;
        if (overlap(state_out->s, sbytes, x->ptr, tensor_bytes(x)) || overlap(state_out->s, sbytes, y->ptr, tensor_bytes(y)) ||
            overlap(state_out->coef, cbytes, x->ptr, tensor_bytes(x)) ||
            overlap(state_out->coef, cbytes, y->ptr, tensor_bytes(y)) || overlap(state_out->s, sbytes, state_out->coef, cbytes))
            return fail(RLM_ERR_INVALID_ARG, "state_out->s or state_out->coef overlaps the fields or each other");
    }
    if (state_in) {
        if (!state_in->s || !aligned16(state_in->s))
            return fail(RLM_ERR_INVALID_ARG, "state_in->s is NULL or not 16-byte aligned");
        if (state_in->B != x->B || state_in->D != x->D || state_in->M != p->M)
            return fail(RLM_ERR_INVALID_ARG, "state_in is [B=%d][D=%d][M=%d], expected [%lld][%lld][%d]",
                        state_in->B, state_in->D, state_in->M, (long long)x->B, (long long)x->D, p->M);
        if (overlap(state_in->s, sbytes, y->ptr, tensor_bytes(y)))
            return fail(RLM_ERR_INVALID_ARG, "state_in overlaps the output field");
        if (state_out && state_out->s != state_in->s && overlap(state_in->s, sbytes, state_out->s, sbytes))
            return fail(RLM_ERR_INVALID_ARG, "state_in and state_out overlap without being the same buffer");
    }
    return RLM_OK;
}

// The prefill path for a problem: the tcgen05 prefill (bf16, M <= 64), its
// time-reversed form (other bf16 M <= 32), the tcgen05 prefill for fp32 I/O
// (M <= 16), else the SIMT scan.  The tcgen05 forms work in 64-token chunks
// aligned to one end of the sequence; when L is not a
// multiple of 64, an initial state enters them through a negative power of
// lambda (up to lambda^-63), which overflows fp32 for decays above 88/63 per
// token.  Such calls run on the SIMT scan, whose powers of lambda are all
// positive, so every finite decay >= 0 is covered.
enum class PrefillPath { kTc, kRev, kTc32, kSimt };

bool state_in_needs_simt(int64_t L, bool with_state_in) { return with_state_in && L % 64 != 0; }

PrefillPath prefill_path(const rlm_tensor *x, int M, bool with_state_in) {
    const int D = (int)x->D;
    if (state_in_needs_simt(x->L, with_state_in)) return PrefillPath::kSimt;
    if (tc_prefill_supported(x->B, x->L, D, M, x->dtype)) return PrefillPath::kTc;
    if (tc_prefill_rev_supported(x->B, x->L, D, M, x->dtype)) return PrefillPath::kRev;
    if (tc32_prefill_supported(x->B, x->L, D, M, x->dtype)) return PrefillPath::kTc32;
    return PrefillPath::kSimt;
}

// Launches the mixing of x into y on the chosen path (arguments already checked).
cudaError_t launch_prefill(PrefillPath path, const rlm_tensor *x, const rlm_params *p, const float *sin,
                           void *y, float *so, float *co, const rlm_launch *ln) {
    cudaStream_t st = static_cast<cudaStream_t>(ln->stream);
    const int D = (int)x->D, M = p->M;
    switch (path) {
        case PrefillPath::kTc:
            return tc_prefill(x->ptr, y, x->B, x->L, D, M, p->decay, p->freq, p->amp, p->phase, sin, so, co,
                              nullptr, ln->workspace, st);
        case PrefillPath::kRev:
            return tc_prefill_rev(x->ptr, y, x->B, x->L, D, M, p->decay, p->freq, p->amp, p->phase, sin, so, co,
                                  ln->workspace, st);
        case PrefillPath::kTc32:
            return tc32_prefill(static_cast<const float *>(x->ptr), static_cast<float *>(y), x->B, x->L, D, M,
                                p->decay, p->freq, p->amp, p->phase, sin, so, co, st);
        default:
            return simt_prefill(x->ptr, y, x->dtype, x->B, x->L, D, M, p->decay, p->freq, p->amp, p->phase,
                                sin, so, co, ln->workspace, st);
    }
}

// The mixer's local path: K in range, D matching, weights present when K > 0.
rlm_status check_local(const rlm_local *lc, int64_t D, int *K) {
    *K = 0;
    if (!lc) return RLM_OK;
    if (lc->K < 0 || lc->K > RLM_MAX_LOCAL_K)
        return fail(RLM_ERR_INVALID_ARG, "local->K=%d outside 0..%d", lc->K, RLM_MAX_LOCAL_K);
    if (lc->K == 0) return RLM_OK;
    if (lc->D != D) return fail(RLM_ERR_INVALID_ARG, "local->D=%d does not match D=%lld", lc->D, (long long)D);
    if (!lc->conv_w || !lc->scale || !aligned16(lc->conv_w) || !aligned16(lc->scale))
        return fail(RLM_ERR_INVALID_ARG, "local->conv_w or local->scale is NULL or not 16-byte aligned");
    *K = lc->K;
    return RLM_OK;
}

// Head coupling: H heads dividing D, a finite strength, the raw matrix present.
rlm_status check_coupling(const rlm_coupling *cp, int64_t D) {
    if (!cp) return RLM_OK;
    if (cp->H < 1 || cp->H > 64) return fail(RLM_ERR_INVALID_ARG, "coupling->H=%d outside 1..64", cp->H);
    if (D % cp->H != 0)
        return fail(RLM_ERR_INVALID_ARG, "D=%lld is not a multiple of coupling->H=%d", (long long)D, cp->H);
    if (D > 8192) return fail(RLM_ERR_UNSUPPORTED, "head coupling supports D <= 8192 (got %lld)", (long long)D);
    if (!cp->c_raw || !aligned16(cp->c_raw))
        return fail(RLM_ERR_INVALID_ARG, "coupling->c_raw is NULL or not 16-byte aligned");
    if (!std::isfinite(cp->lambda_c)) return fail(RLM_ERR_INVALID_ARG, "coupling->lambda_c is not finite");
    return RLM_OK;
}

size_t conv_bytes(int64_t B, int64_t D, int K, rlm_dtype dt) {
    return K < 2 ? 0 : (size_t)B * (size_t)(K - 1) * (size_t)D * elem_size(dt);
}

// A drive-history argument (only checked when the local path has K >= 2).
rlm_status check_conv(const rlm_conv_state *c, int64_t B, int64_t D, int K, rlm_dtype dt, const char *name) {
    if (!c || K < 2) return RLM_OK;
    if (!c->u || !aligned16(c->u)) return fail(RLM_ERR_INVALID_ARG, "%s->u is NULL or not 16-byte aligned", name);
    if (c->B != B || c->D != D || c->K != K || c->dtype != dt)
        return fail(RLM_ERR_INVALID_ARG, "%s is [B=%lld][K-1=%d][D=%d] of dtype %d, expected [%lld][%d][%lld] of %d",
                    name, (long long)c->B, c->K - 1, c->D, (int)c->dtype, (long long)B, K - 1, (long long)D,
                    (int)dt);
    return RLM_OK;
}

}  // namespace

extern "C" {

const char *rlm_status_string(rlm_status s) {
    switch (s) {
        case RLM_OK: return "RLM_OK";
        case RLM_ERR_INVALID_ARG: return "RLM_ERR_INVALID_ARG";
        case RLM_ERR_UNSUPPORTED: return "RLM_ERR_UNSUPPORTED";
        case RLM_ERR_CUDA: return "RLM_ERR_CUDA";
        case RLM_ERR_TIMEOUT: return "RLM_ERR_TIMEOUT";
    }
    return "RLM_STATUS_UNKNOWN";
}

const char *rlm_last_error(void) { return g_err; }

int rlm_version(void) { return 100; }

unsigned long long rlm_kernels_launched(void) { return g_launches.load(std::memory_order_relaxed); }

size_t rlm_prefill_workspace_size(int64_t B, int64_t L, int D, int M, rlm_dtype dtype) {
    if (B < 1 || L < 1 || D < 1 || M < 1) return 0;
    size_t tc = 0;
    if (tc_prefill_supported(B, L, D, M, dtype)) tc = tc_prefill_ws_bytes(B, L, D, M);
    else if (tc_prefill_rev_supported(B, L, D, M, dtype)) tc = tc_prefill_rev_ws_bytes(B, L, D, M);
    else return simt_prefill_ws_bytes(B, L, D, M);
    // A call with an initial state and a ragged length runs on the SIMT scan.
    return state_in_needs_simt(L, true) ? std::max(tc, simt_prefill_ws_bytes(B, L, D, M)) : tc;
}

size_t rlm_backward_workspace_size(int64_t B, int64_t L, int D, int M, rlm_dtype dtype) {
    if (B < 1 || L < 1 || D < 1 || M < 1) return 0;
    if (tc_backward_supported(B, L, D, M, dtype)) return tc_backward_ws_bytes(B, L, D, M);
    return simt_backward_ws_bytes(B, L, D, M);
}

rlm_status rlm_mix_prefill(const rlm_tensor *x, const rlm_params *p, rlm_tensor *y,
                           rlm_state *state_out, const rlm_launch *ln) {
    return rlm_mix_prefill_from(x, p, nullptr, y, state_out, ln);
}

rlm_status rlm_mix_prefill_from(const rlm_tensor *x, const rlm_params *p, const rlm_state *state_in,
                                rlm_tensor *y, rlm_state *state_out, const rlm_launch *ln) {
    rlm_status s;
    if ((s = check_tensor(x, "x")) != RLM_OK) return s;
    if ((s = check_tensor(y, "y")) != RLM_OK) return s;
    if (!same_shape(x, y)) return fail(RLM_ERR_INVALID_ARG, "y must have x's shape and dtype");
    if (overlap(x->ptr, tensor_bytes(x), y->ptr, tensor_bytes(y)))
        return fail(RLM_ERR_INVALID_ARG, "x and y overlap");
    if ((s = check_params(p, x->D)) != RLM_OK) return s;
    if ((s = check_prefill_states(x, y, p, state_in, state_out)) != RLM_OK) return s;
    const PrefillPath path = prefill_path(x, p->M, state_in != nullptr);
    if (path == PrefillPath::kSimt && simt_chunks(x->B, x->L, (int)x->D) > 65535)
        return fail(RLM_ERR_UNSUPPORTED, "sequence too long for the chunk grid");
    const size_t need = rlm_prefill_workspace_size(x->B, x->L, (int)x->D, p->M, x->dtype);
    if ((s = check_workspace(ln, need)) != RLM_OK) return s;
    cudaError_t e = launch_prefill(path, x, p, state_in ? state_in->s : nullptr, y->ptr,
                                   state_out ? state_out->s : nullptr, state_out ? state_out->coef : nullptr, ln);
    if (e != cudaSuccess) return cuda_fail(e, "rlm_mix_prefill launch");
    return RLM_OK;
}

rlm_status rlm_mixer_prefill(const rlm_tensor *x, const rlm_tensor *g, const rlm_params *p, const rlm_local *local,
                             const rlm_coupling *coupling, const rlm_state *state_in, const rlm_conv_state *conv_in, rlm_tensor *z,
                             rlm_state *state_out, rlm_conv_state *conv_out, const rlm_launch *ln) {
    rlm_status s;
    if ((s = check_tensor(x, "x")) != RLM_OK) return s;
    if ((s = check_tensor(z, "z")) != RLM_OK) return s;
    if (!same_shape(x, z)) return fail(RLM_ERR_INVALID_ARG, "z must have x's shape and dtype");
    if (g) {
        if ((s = check_tensor(g, "g")) != RLM_OK) return s;
        if (!same_shape(x, g)) return fail(RLM_ERR_INVALID_ARG, "g must have x's shape and dtype");
        if (overlap(g->ptr, tensor_bytes(g), z->ptr, tensor_bytes(z)))
            return fail(RLM_ERR_INVALID_ARG, "g and z overlap");
    }
    if (overlap(x->ptr, tensor_bytes(x), z->ptr, tensor_bytes(z)))
        return fail(RLM_ERR_INVALID_ARG, "x and z overlap");
    if ((s = check_params(p, x->D)) != RLM_OK) return s;
    if ((s = check_prefill_states(x, z, p, state_in, state_out)) != RLM_OK) return s;
    int K = 0;
    if ((s = check_local(local, x->D, &K)) != RLM_OK) return s;
    if ((s = check_coupling(coupling, x->D)) != RLM_OK) return s;
    if ((s = check_conv(conv_in, x->B, x->D, K, x->dtype, "conv_in")) != RLM_OK) return s;
    if ((s = check_conv(conv_out, x->B, x->D, K, x->dtype, "conv_out")) != RLM_OK) return s;
    const size_t cb = conv_bytes(x->B, x->D, K, x->dtype);
    const void *hin = (conv_in && K >= 2) ? conv_in->u : nullptr;
    void *hout = (conv_out && K >= 2) ? conv_out->u : nullptr;
    if (hin && overlap(hin, cb, z->ptr, tensor_bytes(z)))
        return fail(RLM_ERR_INVALID_ARG, "conv_in overlaps z");
    if (hout) {
        if (overlap(hout, cb, z->ptr, tensor_bytes(z)) || overlap(hout, cb, x->ptr, tensor_bytes(x)) ||
            (g && overlap(hout, cb, g->ptr, tensor_bytes(g))))
            return fail(RLM_ERR_INVALID_ARG, "conv_out overlaps x, g or z");
        if (hin && hin != hout && overlap(hin, cb, hout, cb))
            return fail(RLM_ERR_INVALID_ARG, "conv_in and conv_out overlap without being the same buffer");
    }
    const PrefillPath path = prefill_path(x, p->M, state_in != nullptr);
    if (path == PrefillPath::kSimt && simt_chunks(x->B, x->L, (int)x->D) > 65535)
        return fail(RLM_ERR_UNSUPPORTED, "sequence too long for the chunk grid");
    const size_t need = rlm_prefill_workspace_size(x->B, x->L, (int)x->D, p->M, x->dtype);
    if ((s = check_workspace(ln, need)) != RLM_OK) return s;
    cudaStream_t st = static_cast<cudaStream_t>(ln->stream);
    // The gate alone is fused into the tcgen05 prefill's epilogue.  With a local
    // path, the mixing and one full-width pass over x, g and y are faster than
    // the fused kernel (whose 8-channel row slices cap its memory rate).
    const bool fused = g && K == 0 && !coupling && path == PrefillPath::kTc &&
                       tc_mixer_fused(x->B, x->L, (int)x->D, p->M, x->dtype);
    cudaError_t e;
    if (fused) {
        const TcMix mix{g->ptr};
        e = tc_prefill(x->ptr, z->ptr, x->B, x->L, (int)x->D, p->M, p->decay, p->freq, p->amp, p->phase,
                       state_in ? state_in->s : nullptr, state_out ? state_out->s : nullptr,
                       state_out ? state_out->coef : nullptr, &mix, ln->workspace, st);
    } else {
        e = launch_prefill(path, x, p, state_in ? state_in->s : nullptr, z->ptr, state_out ? state_out->s : nullptr,
                           state_out ? state_out->coef : nullptr, ln);
    }
    const int H = coupling ? coupling->H : 0;
    if (e == cudaSuccess && !fused && (g || K > 0 || coupling)) {
        if (mixer_stream_supported(x->dtype, (int)x->D, H)) {
            // Coupling, gate and local path in one pass over whole-row tiles.
            e = mixer_stream(x->ptr, g ? g->ptr : nullptr, z->ptr, hin, K > 0 ? local->conv_w : nullptr,
                             K > 0 ? local->scale : nullptr, K, coupling ? coupling->c_raw : nullptr,
                             coupling ? coupling->lambda_c : 0.0f, H, x->dtype, x->B, x->L, (int)x->D, st);
        } else {
            if (coupling)
                e = couple_heads(z->ptr, x->dtype, coupling->c_raw, coupling->lambda_c, H, x->B, x->L, (int)x->D,
                                 st);
            if (e == cudaSuccess && (g || K > 0))
                e = mixer_epilogue(x->ptr, g ? g->ptr : nullptr, z->ptr, hin, K > 0 ? local->conv_w : nullptr,
                                   K > 0 ? local->scale : nullptr, x->dtype, x->B, x->L, (int)x->D, K, st);
        }
    }
    if (e == cudaSuccess && hout) e = conv_tail(x->ptr, hin, hout, x->dtype, x->B, x->L, (int)x->D, K, st);
    if (e != cudaSuccess) return cuda_fail(e, "rlm_mixer_prefill launch");
    return RLM_OK;
}

rlm_status rlm_mix_decode(const rlm_tensor *x_t, rlm_state *state, rlm_tensor *y_t,
                          const rlm_launch *ln) {
    rlm_status s;
    if ((s = check_tensor(x_t, "x_t")) != RLM_OK) return s;
    if ((s = check_tensor(y_t, "y_t")) != RLM_OK) return s;
    if (x_t->L != 1) return fail(RLM_ERR_INVALID_ARG, "x_t must have L == 1 (got %lld)", (long long)x_t->L);
    if (!same_shape(x_t, y_t)) return fail(RLM_ERR_INVALID_ARG, "y_t must have x_t's shape and dtype");
    if (overlap(x_t->ptr, tensor_bytes(x_t), y_t->ptr, tensor_bytes(y_t)))
        return fail(RLM_ERR_INVALID_ARG, "x_t and y_t overlap");
    if (!state) return fail(RLM_ERR_INVALID_ARG, "state is NULL");
    if (state->M < 1 || state->M > kMaxModes)
        return fail(RLM_ERR_INVALID_ARG, "state->M=%d outside 1..%d", state->M, kMaxModes);
    if ((s = check_state(state, x_t->B, x_t->D, state->M, "state")) != RLM_OK) return s;
    if (!ln) return fail(RLM_ERR_INVALID_ARG, "launch is NULL");
    const size_t sbytes = (size_t)state->B * state->D * state->M * 8;
    if (overlap(state->s, sbytes, y_t->ptr, tensor_bytes(y_t)) ||
        overlap(state->s, sbytes, x_t->ptr, tensor_bytes(x_t)))
        return fail(RLM_ERR_INVALID_ARG, "state overlaps x_t or y_t");
    cudaError_t e = decode_step(x_t->ptr, y_t->ptr, x_t->dtype, (int)x_t->B, (int)x_t->D, state->M,
                                state->s, state->coef, static_cast<cudaStream_t>(ln->stream));
    if (e != cudaSuccess) return cuda_fail(e, "rlm_mix_decode launch");
    return RLM_OK;
}

rlm_status rlm_mixer_decode(const rlm_tensor *x_t, const rlm_tensor *g_t, rlm_state *state, const rlm_local *local,
                            const rlm_coupling *coupling, rlm_conv_state *conv, rlm_tensor *z_t, const rlm_launch *ln) {
    rlm_status s;
    if ((s = check_tensor(x_t, "x_t")) != RLM_OK) return s;
    if ((s = check_tensor(z_t, "z_t")) != RLM_OK) return s;
    if (x_t->L != 1) return fail(RLM_ERR_INVALID_ARG, "x_t must have L == 1 (got %lld)", (long long)x_t->L);
    if (!same_shape(x_t, z_t)) return fail(RLM_ERR_INVALID_ARG, "z_t must have x_t's shape and dtype");
    if (overlap(x_t->ptr, tensor_bytes(x_t), z_t->ptr, tensor_bytes(z_t)))
        return fail(RLM_ERR_INVALID_ARG, "x_t and z_t overlap");
    if (g_t) {
        if ((s = check_tensor(g_t, "g_t")) != RLM_OK) return s;
        if (!same_shape(x_t, g_t)) return fail(RLM_ERR_INVALID_ARG, "g_t must have x_t's shape and dtype");
        if (overlap(g_t->ptr, tensor_bytes(g_t), z_t->ptr, tensor_bytes(z_t)))
            return fail(RLM_ERR_INVALID_ARG, "g_t and z_t overlap");
    }
    if (!state) return fail(RLM_ERR_INVALID_ARG, "state is NULL");
    if (state->M < 1 || state->M > kMaxModes)
        return fail(RLM_ERR_INVALID_ARG, "state->M=%d outside 1..%d", state->M, kMaxModes);
    if ((s = check_state(state, x_t->B, x_t->D, state->M, "state")) != RLM_OK) return s;
    if (!ln) return fail(RLM_ERR_INVALID_ARG, "launch is NULL");
    const size_t sbytes = (size_t)state->B * state->D * state->M * 8;
    if (overlap(state->s, sbytes, z_t->ptr, tensor_bytes(z_t)) || overlap(state->s, sbytes, x_t->ptr, tensor_bytes(x_t)) ||
        (g_t && overlap(state->s, sbytes, g_t->ptr, tensor_bytes(g_t))))
        return fail(RLM_ERR_INVALID_ARG, "state overlaps x_t, g_t or z_t");
    int K = 0;
    if ((s = check_local(local, x_t->D, &K)) != RLM_OK) return s;
    if ((s = check_coupling(coupling, x_t->D)) != RLM_OK) return s;
    if (K >= 2 && !conv) return fail(RLM_ERR_INVALID_ARG, "conv is NULL but the local path has K=%d", K);
    if ((s = check_conv(conv, x_t->B, x_t->D, K, x_t->dtype, "conv")) != RLM_OK) return s;
    if (K >= 2) {
        const size_t cb = conv_bytes(x_t->B, x_t->D, K, x_t->dtype);
        if (overlap(conv->u, cb, z_t->ptr, tensor_bytes(z_t)) || overlap(conv->u, cb, x_t->ptr, tensor_bytes(x_t)) ||
            (g_t && overlap(conv->u, cb, g_t->ptr, tensor_bytes(g_t))) || overlap(conv->u, cb, state->s, sbytes))
            return fail(RLM_ERR_INVALID_ARG, "conv overlaps x_t, g_t, z_t or the state");
    }
    cudaStream_t st = static_cast<cudaStream_t>(ln->stream);
    cudaError_t e;
    // One block per batch row serves the coupled step; the uncoupled step runs on
    // the row-tiled decode kernel.
    const bool row_block = coupling != nullptr;
    if (row_block && mixer_decode_coupled_supported((int)x_t->D, state->M)) {
        // One launch: recurrence step, coupling (if any), gate, local path.
        e = mixer_decode_coupled(x_t->ptr, g_t ? g_t->ptr : nullptr, z_t->ptr, x_t->dtype, (int)x_t->B,
                                 (int)x_t->D, state->M, state->s, state->coef, K >= 2 ? conv->u : nullptr,
                                 K > 0 ? local->conv_w : nullptr, K > 0 ? local->scale : nullptr, K,
                                 coupling ? coupling->c_raw : nullptr, coupling ? coupling->lambda_c : 0.0f,
                                 coupling ? coupling->H : 0, st);
    } else if (coupling) {
        // The recurrence step writes y_t into z_t; one block per batch row then
        // couples the heads and applies the gate and the local path.
        e = decode_step(x_t->ptr, z_t->ptr, x_t->dtype, (int)x_t->B, (int)x_t->D, state->M, state->s, state->coef, st);
        if (e == cudaSuccess)
            e = mixer_finish_coupled(x_t->ptr, g_t ? g_t->ptr : nullptr, z_t->ptr, K >= 2 ? conv->u : nullptr,
                                     K > 0 ? local->conv_w : nullptr, K > 0 ? local->scale : nullptr, K,
                                     coupling->c_raw, coupling->lambda_c, coupling->H, x_t->dtype, (int)x_t->B,
                                     (int)x_t->D, st);
    } else {
        e = mixer_decode_step(x_t->ptr, g_t ? g_t->ptr : nullptr, z_t->ptr, x_t->dtype, (int)x_t->B, (int)x_t->D,
                              state->M, state->s, state->coef, K >= 2 ? conv->u : nullptr,
                              K > 0 ? local->conv_w : nullptr, K > 0 ? local->scale : nullptr, K, st);
    }
    if (e != cudaSuccess) return cuda_fail(e, "rlm_mixer_decode launch");
    return RLM_OK;
}

rlm_status rlm_state_init(rlm_state *state, const rlm_params *p, const rlm_launch *ln) {
    rlm_status s;
    if (!state) return fail(RLM_ERR_INVALID_ARG, "state is NULL");
    if ((s = check_params(p, state->D)) != RLM_OK) return s;
    if (state->B < 1 || state->D < 1) return fail(RLM_ERR_INVALID_ARG, "state has B or D < 1");
    if ((s = check_state(state, state->B, state->D, p->M, "state")) != RLM_OK) return s;
    if (!ln) return fail(RLM_ERR_INVALID_ARG, "launch is NULL");
    cudaError_t e = state_init(state->s, state->coef, state->B, state->D, state->M, p->decay, p->freq,
                               p->amp, p->phase, static_cast<cudaStream_t>(ln->stream));
    if (e != cudaSuccess) return cuda_fail(e, "rlm_state_init launch");
    return RLM_OK;
}

rlm_status rlm_mix_backward(const rlm_tensor *dy, const rlm_tensor *x, const rlm_params *p,
                            rlm_tensor *dx, rlm_grads *g, const rlm_launch *ln) {
    return rlm_mix_backward_from(dy, x, p, nullptr, nullptr, dx, g, nullptr, ln);
}


rlm_status rlm_mix_backward_from(const rlm_tensor *dy, const rlm_tensor *x, const rlm_params *p,
                                 const rlm_state *state_in, const rlm_state *d_state_out, rlm_tensor *dx,
                                 rlm_grads *g, rlm_state *d_state_in, const rlm_launch *ln) {
    rlm_status s;
    if ((s = check_tensor(dy, "dy")) != RLM_OK) return s;
    if ((s = check_tensor(x, "x")) != RLM_OK) return s;
    if ((s = check_tensor(dx, "dx")) != RLM_OK) return s;
    if (!same_shape(dy, x) || !same_shape(dx, x))
        return fail(RLM_ERR_INVALID_ARG, "dy, x and dx must share shape and dtype");
    if (overlap(dx->ptr, tensor_bytes(dx), x->ptr, tensor_bytes(x)) ||
        overlap(dx->ptr, tensor_bytes(dx), dy->ptr, tensor_bytes(dy)))
        return fail(RLM_ERR_INVALID_ARG, "dx overlaps x or dy");
    if ((s = check_params(p, x->D)) != RLM_OK) return s;
    if (!g) return fail(RLM_ERR_INVALID_ARG, "dparams is NULL");
    float *gs[4] = {g->decay, g->freq, g->amp, g->phase};
    for (int i = 0; i < 4; ++i)
        if (!gs[i] || !aligned16(gs[i]))
            return fail(RLM_ERR_INVALID_ARG, "dparams pointer %d is NULL or not 16-byte aligned", i);
    if (g->D != p->D || g->M != p->M) return fail(RLM_ERR_INVALID_ARG, "dparams shape differs from params");
    if ((s = check_state_s(state_in, x->B, x->D, p->M, "state_in")) != RLM_OK) return s;
    if ((s = check_state_s(d_state_out, x->B, x->D, p->M, "d_state_out")) != RLM_OK) return s;
    if ((s = check_state_s(d_state_in, x->B, x->D, p->M, "d_state_in")) != RLM_OK) return s;
    if (d_state_in) {
        const size_t sb = (size_t)x->B * x->D * p->M * 8;
        if (overlap(d_state_in->s, sb, dx->ptr, tensor_bytes(dx)) ||
            (state_in && overlap(d_state_in->s, sb, state_in->s, sb)) ||
            (d_state_out && overlap(d_state_in->s, sb, d_state_out->s, sb)))
            return fail(RLM_ERR_INVALID_ARG, "d_state_in overlaps dx, state_in or d_state_out");
        for (int i = 0; i < 4; ++i)
            if (overlap(d_state_in->s, sb, gs[i], (size_t)p->D * p->M * sizeof(float)))
                return fail(RLM_ERR_INVALID_ARG, "d_state_in overlaps dparams");
    }
    const float *sin = state_in ? state_in->s : nullptr;
    const float *gout = d_state_out ? d_state_out->s : nullptr;
    float *dsin = d_state_in ? d_state_in->s : nullptr;
    const int D = (int)x->D, M = p->M;
    const bool tc = tc_backward_supported(x->B, x->L, D, M, x->dtype);
    if (!tc && simt_chunks(x->B, x->L, D) > 65535)
        return fail(RLM_ERR_UNSUPPORTED, "sequence too long for the chunk grid");
    const size_t need = rlm_backward_workspace_size(x->B, x->L, D, M, x->dtype);
    if ((s = check_workspace(ln, need)) != RLM_OK) return s;
    cudaStream_t st = static_cast<cudaStream_t>(ln->stream);
    cudaError_t e =
        tc ? tc_backward(dy->ptr, x->ptr, dx->ptr, x->B, x->L, D, M, p->decay, p->freq, p->amp,
                         p->phase, sin, gout, dsin, g->decay, g->freq, g->amp, g->phase, ln->workspace, st)
           : simt_backward(dy->ptr, x->ptr, dx->ptr, x->dtype, x->B, x->L, D, M, p->decay, p->freq,
                           p->amp, p->phase, sin, gout, dsin, g->decay, g->freq, g->amp, g->phase,
                           ln->workspace, st);
    if (e != cudaSuccess) return cuda_fail(e, "rlm_mix_backward launch");
    return RLM_OK;
}

rlm_status rlm_validate_params(const rlm_params *p) {
    if (!p) return fail(RLM_ERR_INVALID_ARG, "params is NULL");
    rlm_status s;
    if ((s = check_params(p, p->D)) != RLM_OK) return s;
    if (p->D < 1) return fail(RLM_ERR_INVALID_ARG, "params->D < 1");
    const size_t n = (size_t)p->D * p->M;
    std::vector<float> h(n);
    const float *ps[4] = {p->decay, p->freq, p->amp, p->phase};
    const char *nm[4] = {"decay", "freq", "amp", "phase"};
    for (int i = 0; i < 4; ++i) {
        cudaError_t e = cudaMemcpy(h.data(), ps[i], n * sizeof(float), cudaMemcpyDeviceToHost);
        if (e != cudaSuccess) return cuda_fail(e, "rlm_validate_params copy");
        for (size_t k = 0; k < n; ++k) {
            if (!std::isfinite(h[k]))
                return fail(RLM_ERR_INVALID_ARG, "params->%s[%zu] is not finite", nm[i], k);
            if (i == 0 && h[k] < 0.0f)
                return fail(RLM_ERR_INVALID_ARG, "params->decay[%zu] = %g < 0", k, (double)h[k]);
        }
    }
    return RLM_OK;
}

rlm_status rlm_get_device_status(const rlm_launch *ln) {
    if (!ln) return fail(RLM_ERR_INVALID_ARG, "launch is NULL");
    int status = RLM_OK, bwd = RLM_OK, mix = RLM_OK, t32 = RLM_OK;
    cudaError_t e = read_and_clear_device_status(&status, static_cast<cudaStream_t>(ln->stream));
    if (e == cudaSuccess) e = read_and_clear_bwd_status(&bwd, static_cast<cudaStream_t>(ln->stream));
    if (e == cudaSuccess) e = read_and_clear_mixer_status(&mix, static_cast<cudaStream_t>(ln->stream));
    if (e == cudaSuccess) e = read_and_clear_tc32_status(&t32, static_cast<cudaStream_t>(ln->stream));
    if (e != cudaSuccess) return cuda_fail(e, "rlm_get_device_status");
    if (status == RLM_OK) status = bwd;
    if (status == RLM_OK) status = mix;
    if (status == RLM_OK) status = t32;
    if (status != RLM_OK) return fail((rlm_status)status, "a bounded device-side wait expired");
    return RLM_OK;
}

rlm_status rlm_test_stall_segments(int on) {
    const cudaError_t e = set_segment_stall(on ? 1 : 0);
    if (e != cudaSuccess) return cuda_fail(e, "rlm_test_stall_segments");
    return RLM_OK;
}

}  // extern "C"
