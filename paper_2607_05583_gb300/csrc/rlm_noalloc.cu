// rlm_noalloc.cu -- rlm_mix_prefill_noalloc: the chunked-scan prefill with its
// scratch in a fixed array that the library itself places in device memory, for
// callers that cannot hand the library a workspace.
//
// The scratch is a file-scope __device__ array of kNoAllocScratchBytes.  Every
// GPU on which the library's device code is loaded holds it until the process
// exits; under CUDA's default lazy module loading that happens when the first
// call of this entry point on the device looks the array up, so the memory is
// committed by that first call.  Host code must not pass the array's name to a
// kernel: on the host that name is only a stand-in, not a device address.  The
// device address is looked up with cudaGetSymbolAddress, once per device, with
// that device current, the first time this entry point runs on it.
#include <cuda_runtime.h>

#include <cstdarg>
#include <cstdio>
#include <cstdint>
#include <mutex>
#include <vector>

#include "rlm_internal.h"

namespace rlm {
namespace {

constexpr size_t kNoAllocScratchBytes = (size_t)64 << 20;  // 64 MiB

static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

std::mutex g_scratch_mu;
std::vector<void *> g_scratch_addr;  // per device; nullptr until looked up

// Device address of the scratch array on the current device (set-up on first use).
cudaError_t scratch_address(void **out) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    std::lock_guard<std::mutex> lock(g_scratch_mu);
    if ((int)g_scratch_addr.size() <= dev) g_scratch_addr.resize(dev + 1, nullptr);
    if (!g_scratch_addr[dev]) {
        void *p = nullptr;
        e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
        if (e != cudaSuccess) return e;
        g_scratch_addr[dev] = p;
    }
    *out = g_scratch_addr[dev];
    return cudaSuccess;
}

rlm_status reject(rlm_status s, const char *fmt, ...) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof(buf), fmt, ap);
    va_end(ap);
    set_error("%s", buf);
    return s;
}

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

rlm_status check_field(const rlm_tensor *t, const char *name) {
    if (!t || !t->ptr) return reject(RLM_ERR_INVALID_ARG, "%s is NULL", name);
    if (!aligned16(t->ptr)) return reject(RLM_ERR_INVALID_ARG, "%s->ptr is not 16-byte aligned", name);
    if (t->dtype != RLM_F32 && t->dtype != RLM_BF16)
        return reject(RLM_ERR_INVALID_ARG, "%s->dtype is not RLM_F32 or RLM_BF16", name);
    if (t->B < 1 || t->L < 1 || t->D < 8 || t->D % 8 != 0)
        return reject(RLM_ERR_INVALID_ARG, "%s has B=%lld L=%lld D=%lld (need B, L >= 1, D >= 8, D %% 8 == 0)",
                      name, (long long)t->B, (long long)t->L, (long long)t->D);
    if (t->B > 65535 || t->L > ((int64_t)1 << 30) || t->D > (1 << 20))
        return reject(RLM_ERR_UNSUPPORTED, "%s is larger than the kernels cover", name);
    return RLM_OK;
}

}  // namespace
}  // namespace rlm

using namespace rlm;

extern "C" rlm_status rlm_mix_prefill_noalloc(const rlm_tensor *x, const rlm_params *p,
                                              rlm_tensor *y, rlm_state *state_out, void *stream) {
    rlm_status s;
    if ((s = check_field(x, "x")) != RLM_OK) return s;
    if ((s = check_field(y, "y")) != RLM_OK) return s;
    if (x->B != y->B || x->L != y->L || x->D != y->D || x->dtype != y->dtype)
        return reject(RLM_ERR_INVALID_ARG, "y must have x's shape and dtype");
    const size_t nbytes = (size_t)x->B * x->L * x->D * (x->dtype == RLM_BF16 ? 2 : 4);
    const char *xa = static_cast<const char *>(x->ptr), *ya = static_cast<const char *>(y->ptr);
    if (xa < ya + nbytes && ya < xa + nbytes) return reject(RLM_ERR_INVALID_ARG, "x and y overlap");
    if (!p || !p->decay || !p->freq || !p->amp || !p->phase)
        return reject(RLM_ERR_INVALID_ARG, "params or one of its pointers is NULL");
    if (!aligned16(p->decay) || !aligned16(p->freq) || !aligned16(p->amp) || !aligned16(p->phase))
        return reject(RLM_ERR_INVALID_ARG, "params pointers must be 16-byte aligned");
    if (p->M < 1 || p->M > 64 || p->D != x->D)
        return reject(RLM_ERR_INVALID_ARG, "params is [D=%d][M=%d]; need D == %lld and 1 <= M <= 64",
                      p->D, p->M, (long long)x->D);
    if (state_out) {
        if (!state_out->s || !state_out->coef || !aligned16(state_out->s) || !aligned16(state_out->coef))
            return reject(RLM_ERR_INVALID_ARG, "state_out buffers are NULL or not 16-byte aligned");
        if (state_out->B != x->B || state_out->D != x->D || state_out->M != p->M)
            return reject(RLM_ERR_INVALID_ARG, "state_out shape does not match x and params");
        const char *sa = reinterpret_cast<const char *>(state_out->s);
        const char *ca = reinterpret_cast<const char *>(state_out->coef);
        const size_t sb = (size_t)x->B * x->D * p->M * 8, cb = (size_t)x->D * p->M * 16;
        auto hits = [](const char *a, size_t na, const char *b, size_t nb) { return a < b + nb && b < a + na; };
        if (hits(sa, sb, xa, nbytes) || hits(sa, sb, ya, nbytes) || hits(ca, cb, xa, nbytes) ||
            hits(ca, cb, ya, nbytes) || hits(sa, sb, ca, cb))
            return reject(RLM_ERR_INVALID_ARG, "state_out->s or state_out->coef overlaps x, y or each other");
    }
    if (stream) {
        // The scratch address is the current device's, so the stream must be that device's.
        int dev = 0, sdev = 0;
        if (cudaGetDevice(&dev) != cudaSuccess ||
            cudaStreamGetDevice(static_cast<cudaStream_t>(stream), &sdev) != cudaSuccess)
            return reject(RLM_ERR_INVALID_ARG, "rlm_mix_prefill_noalloc: the stream's device cannot be read");
        if (sdev != dev)
            return reject(RLM_ERR_INVALID_ARG,
                          "rlm_mix_prefill_noalloc: the stream belongs to device %d, the current device is %d",
                          sdev, dev);
    }
    const int D = (int)x->D, M = p->M;
    const int C = simt_chunk_len(x->B, x->L, D);
    if ((x->L + C - 1) / C > 65535) return reject(RLM_ERR_UNSUPPORTED, "sequence too long for the chunk grid");
    const size_t need = simt_prefill_ws_bytes(x->B, x->L, D, M);
    if (need > kNoAllocScratchBytes)
        return reject(RLM_ERR_UNSUPPORTED,
                      "rlm_mix_prefill_noalloc: this shape needs %zu bytes of scratch; the library's "
                      "fixed scratch array holds %zu bytes (use rlm_mix_prefill with a workspace)",
                      need, kNoAllocScratchBytes);
    void *scratch = nullptr;
    cudaError_t e = scratch_address(&scratch);
    if (e != cudaSuccess)
        return reject(RLM_ERR_CUDA, "rlm_mix_prefill_noalloc: cudaGetSymbolAddress: %s", cudaGetErrorString(e));
    e = simt_prefill(x->ptr, y->ptr, x->dtype, x->B, x->L, D, M, p->decay, p->freq, p->amp, p->phase,
                     nullptr, state_out ? state_out->s : nullptr, state_out ? state_out->coef : nullptr, scratch,
                     static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess)
        return reject(RLM_ERR_CUDA, "rlm_mix_prefill_noalloc launch: %s", cudaGetErrorString(e));
    return RLM_OK;
}
