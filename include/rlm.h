/*
 * rlm.h -- C ABI of the GB300 (sm_103a) causal resonant field mixing library.
 *
 * The operator is the attention replacement of ResonatorLM (arxiv 2607.05583):
 * every channel d of a (B, L, D) token field drives M damped resonators.  With
 * per-mode decay gamma, frequency omega, amplitude A and phase phi,
 *
 *   lambda_dm = exp(-gamma_dm) (cos omega_dm + i sin omega_dm)        (Eq. 5)
 *   c_dm      = A_dm exp(+i phi_dm)
 *   K_d[n]    = sum_m A_dm exp(-gamma_dm n) cos(omega_dm n + phi_dm)  (Eq. 1)
 *   y[b,t,d]  = sum_{j<=t} K_d[t-j] x[b,j,d]                          (Eq. 2)
 *
 * which is the same map as the complex recurrence s <- lambda s + x_t,
 * y_t = sum_m Re(c s) of Sec. 3.3 (Eq. 4), started from a zero state.  The
 * paper's readout Re(e^{-i phi} s) is taken as Re(e^{+i phi} s) so that decode
 * agrees with Eq. 1; the paper's single mode per head is the case M = 1, A = 1
 * with parameters tied across a head's channels.
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 *  - All tensor and parameter pointers are DEVICE pointers, 16-byte aligned.
 *    The caller owns every buffer; the library allocates nothing on any call
 *    path and keeps no pointer after a call returns.
 *  - Every call is asynchronous on launch->stream (a cudaStream_t passed as
 *    void*; NULL is the legacy default stream).
 *  - Argument checks run on the host before anything is enqueued; a failing
 *    check returns RLM_ERR_INVALID_ARG or RLM_ERR_UNSUPPORTED and enqueues
 *    nothing.  rlm_last_error() then describes the failure.
 *  - A failed kernel launch returns RLM_ERR_CUDA.
 *  - Kernels that wait on one another (the prefill's cross-block carry) wait a
 *    bounded number of iterations; on expiry they record RLM_ERR_TIMEOUT in a
 *    device status word and return without hanging.  rlm_get_device_status()
 *    reads and clears that word.
 *  - Shapes: B >= 1, L >= 1, D >= 8 with D % 8 == 0, 1 <= M <= 64.  Limits
 *    (RLM_ERR_UNSUPPORTED beyond): B <= 65535, D <= 2^20, L <= 2^24 (the kernels
 *    form lambda^n from fp32 token counts, which are exact up to 2^24).
 *  - Element types of x, y, dy, dx: RLM_F32 or RLM_BF16 (all four of one call
 *    share one type).  Parameters, gradients and the decode state are fp32.
 *  - Inputs and outputs of one call must not overlap.
 */
#ifndef RLM_H_
#define RLM_H_

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define RLM_API __attribute__((visibility("default")))
#else
#define RLM_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    RLM_OK = 0,
    RLM_ERR_INVALID_ARG = 1,  /* bad pointer, shape, dtype, alignment or size   */
    RLM_ERR_UNSUPPORTED = 2,  /* well-formed but outside what the kernels cover */
    RLM_ERR_CUDA = 3,         /* a CUDA runtime call or kernel launch failed    */
    RLM_ERR_TIMEOUT = 4       /* a bounded device-side wait expired             */
} rlm_status;

typedef enum { RLM_F32 = 0, RLM_BF16 = 1 } rlm_dtype;

/* Resonator parameters (Sec. 3.1 and Eq. 5), each fp32 [D][M] row-major on the
 * device, in the constrained space (gamma >= 0 and finite, any finite omega,
 * A and phi).  The paper's softplus/sigmoid reparameterisation lives outside
 * the operator. */
typedef struct {
    const float *decay;   /* gamma_dm */
    const float *freq;    /* omega_dm */
    const float *amp;     /* A_dm     */
    const float *phase;   /* phi_dm   */
    int D, M;
} rlm_params;

/* Gradients of a scalar loss with respect to rlm_params; same layout.
 * Overwritten (not accumulated) by rlm_mix_backward. */
typedef struct {
    float *decay, *freq, *amp, *phase;
    int D, M;
} rlm_grads;

/* A dense, contiguous [B][L][D] field on the device, channel innermost.
 * Single-token tensors of decode use L = 1. */
typedef struct {
    void *ptr;
    rlm_dtype dtype;
    int64_t B, L, D;
} rlm_tensor;

/* The fixed-size recurrent state of Sec. 3.3 (Eq. 4, "two real tensors", whose
 * size does not grow with decoded length), stored as interleaved complex fp32:
 *   s    [B][D][M][2]  (Re, Im) of s_bdm
 *   coef [D][M][4]     (Re lambda, Im lambda, Re c, Im c) of each mode
 * The coefficients travel with the state because decode takes no parameters.
 * rlm_mix_prefill (state_out) and rlm_state_init fill both. */
typedef struct {
    float *s;
    float *coef;
    int B, D, M;
} rlm_state;

/* Launch context: the stream, and a caller-owned device workspace of at least
 * the size the matching *_workspace_size() query returns (256-byte aligned). */
typedef struct {
    void *stream;
    void *workspace;
    size_t workspace_bytes;
} rlm_launch;

/* ------------------------------------------------------------------ prefill
 * Full-sequence causal mixing, Sec. 3.2 (Eq. 2; the paper evaluates it by FFT,
 * Eq. 3, this library by a chunked complex-diagonal scan with the same result
 * up to rounding), from a zero initial state.
 *   x          [B][L][D] input field (F32 or BF16)
 *   p          resonator parameters, p->D == x->D
 *   y          [B][L][D] output, same shape and dtype as x; overwritten
 *   state_out  nullable; if given (state_out->B == B, D, M matching), receives
 *              the prompt's terminal state s_{L-1} = sum_j lambda^{L-1-j} x_j
 *              (Sec. 3.2) and the mode coefficients, ready for decode.
 * Paths (all accumulate the state in fp32):
 *  - BF16, M <= 16: the tcgen05 tensor-core prefill (modes past M padded);
 *  - BF16, 16 < M <= 32: its 32-mode instance, one launch, where the shape needs
 *    no sequence segments (B * D / 8 of at least about the SM count); else the
 *    tcgen05 reverse-time scan of the reversed drive;
 *  - BF16, 32 < M <= 64 without segments: passes of 16 modes, each adding to y;
 *  - FP32, M <= 16: the tensor-core prefill with each product split into bf16
 *    high and low parts (three MMAs);
 *  - other cases: the SIMT chunked scan. */
RLM_API rlm_status rlm_mix_prefill(const rlm_tensor *x, const rlm_params *p, rlm_tensor *y,
                           rlm_state *state_out, const rlm_launch *launch);

/* Prefill from a given initial state (chunked or continued prefill: the terminal
 * state of an earlier prompt, or any state decode has reached), Sec. 3.2-3.3:
 *   s_{-1} = state_in,  s_t = lambda s_{t-1} + x_t,  y_t = sum_m Re(c_m s_t),
 * i.e. rlm_mix_prefill's y plus the free response sum_m Re(c_m lambda_m^{t+1} s_in).
 *   state_in   nullable (NULL = zero state, the same as rlm_mix_prefill); only
 *              state_in->s ([B][D][M] complex fp32, 16-byte aligned) is read,
 *              state_in->coef is ignored (p gives the coefficients).  It must
 *              not overlap y.  state_out may be the same buffer (in-place
 *              continuation); partial overlap is rejected.
 * Other arguments, the workspace (rlm_prefill_workspace_size) and the paths
 * taken are those of rlm_mix_prefill, except that a call with state_in whose L is
 * not a multiple of 64 runs on the SIMT chunked scan: the tensor-core forms work
 * in 64-token chunks aligned to the end of the sequence and would enter the state
 * through a negative power of lambda (up to lambda^-63), which overflows fp32 for
 * decays above 88/63 per token.  Every finite decay >= 0 is covered; chunked
 * prefills in pieces whose length is a multiple of 64 stay on the tensor cores. */
RLM_API rlm_status rlm_mix_prefill_from(const rlm_tensor *x, const rlm_params *p, const rlm_state *state_in,
                                        rlm_tensor *y, rlm_state *state_out, const rlm_launch *launch);

/* Bytes of workspace rlm_mix_prefill needs for this shape (0 is possible). */
RLM_API size_t rlm_prefill_workspace_size(int64_t B, int64_t L, int D, int M, rlm_dtype dtype);

/* rlm_mix_prefill_noalloc -- the paper has no counterpart; this entry point
 * exists for callers that cannot allocate device memory when they call the
 * library, such as serving runtimes that reserve all device memory up front and
 * forbid allocation afterwards, or plugin hosts that own every allocation and
 * cannot hand out a workspace.  It computes what rlm_mix_prefill computes (same
 * arguments, no workspace) with the chunked-scan kernels, whose scratch lives in
 * a fixed 64 MiB array that the library itself places in device memory: every
 * GPU that loads the library holds that array until the process exits.
 *  - The entry point allocates nothing: no cudaMalloc, cudaFree or allocating
 *    library routine on any path.
 *  - Shapes whose scratch would exceed 64 MiB (B * nchunks * D * M * 8 bytes)
 *    return RLM_ERR_UNSUPPORTED with the needed size in rlm_last_error().
 *  - The first call on a device looks up the array's device address (one
 *    cudaGetSymbolAddress with that device current); make that first call
 *    before any stream capture.  Under CUDA's default lazy module loading the
 *    array's device memory is committed by that same first call, so a runtime
 *    that reserves device memory up front should make it before reserving
 *    (or load modules eagerly, CUDA_MODULE_LOADING=EAGER).
 *  - stream must belong to the current device (RLM_ERR_INVALID_ARG otherwise);
 *    state_out's buffers must not overlap x, y or each other.
 *  - All calls share the one array, and it keeps the previous call's contents;
 *    every scratch element is written before it is read, so nothing needs
 *    clearing.  Calls whose executions overlap on the GPU (different streams,
 *    or host threads on one device) race on the array and must be serialised
 *    by the caller.
 *  - stream: a cudaStream_t passed as void* (NULL = legacy default stream). */
RLM_API rlm_status rlm_mix_prefill_noalloc(const rlm_tensor *x, const rlm_params *p, rlm_tensor *y,
                                           rlm_state *state_out, void *stream);

/* ------------------------------------------------------------------- decode
 * One autoregressive step of Sec. 3.3 (Eq. 4-5) for a batch of tokens:
 *   s_bdm <- lambda_dm s_bdm + x_t[b,d];   y_t[b,d] = sum_m Re(c_dm s_bdm)
 *   x_t    [B][1][D] input token field (F32 or BF16)
 *   state  in/out, updated in place (state->B == B, D, M matching)
 *   y_t    [B][1][D] output, same dtype as x_t
 * Needs no workspace (launch->workspace may be NULL). */
RLM_API rlm_status rlm_mix_decode(const rlm_tensor *x_t, rlm_state *state, rlm_tensor *y_t,
                          const rlm_launch *launch);

/* Zero state->s and fill state->coef from p (for decoding without a prompt). */
RLM_API rlm_status rlm_state_init(rlm_state *state, const rlm_params *p, const rlm_launch *launch);

/* ----------------------------------------------------------------- backward
 * Gradients of a scalar loss l through Eq. 2, given dy = dl/dy:
 *   dx[b,j,d] = sum_{t>=j} K_d[t-j] dy[b,t,d]        (anti-causal mixing)
 *   with G_dm = sum_{b,j} x_j S_j and P_dm = sum_{b,j} x_j R_j, where
 *   S_j = sum_{t>=j} lambda^{t-j} dy_t, R_j = sum_{t>=j} (t-j) lambda^{t-j} dy_t:
 *   dA = Re(e^{i phi} G), dphi = -Im(c G), dgamma = -Re(c P), domega = -Im(c P).
 *   dy, x   [B][L][D] (same dtype);  dx [B][L][D] output, overwritten
 *   dparams fp32 [D][M] each, overwritten; summed over batch and time in a
 *           fixed order (bit-reproducible run to run).
 * There is no gradient input for state_out: the loss depends on y only. */
RLM_API rlm_status rlm_mix_backward(const rlm_tensor *dy, const rlm_tensor *x, const rlm_params *p,
                            rlm_tensor *dx, rlm_grads *dparams, const rlm_launch *launch);

/* Backward of rlm_mix_prefill_from (training through a cached state), Sec. 3.2-3.3:
 * the loss may also depend on the terminal state s_L, and the forward may have
 * started from state_in.
 *   state_in     nullable; the forward's initial state (->s read, [B][D][M] complex).
 *   d_state_out  nullable; g = dl/d(Re s_L) + i dl/d(Im s_L) per (b, d, m) (->s read);
 *                the loss then has the extra term Re(conj(g) s_L).
 *   d_state_in   nullable output; dl/d(Re s_in) + i dl/d(Im s_in) (->s written); it
 *                must not overlap dx, dparams, state_in or d_state_out.
 * dx and dparams as for rlm_mix_backward, with the state terms included.  Paths:
 * bf16 with M <= 32 runs the tcgen05 backward (state_in and d_state_in are
 * per-(b, d, m) terms at its end; a d_state_out adds one launch that forms its
 * terms in closed form, conj(g) lambda^(L-1-t), on the tensor cores); fp32 or
 * M > 32, the SIMT backward.  rlm_backward_workspace_size covers the path taken. */
RLM_API rlm_status rlm_mix_backward_from(const rlm_tensor *dy, const rlm_tensor *x, const rlm_params *p,
                                         const rlm_state *state_in, const rlm_state *d_state_out, rlm_tensor *dx,
                                         rlm_grads *dparams, rlm_state *d_state_in, const rlm_launch *launch);

RLM_API size_t rlm_backward_workspace_size(int64_t B, int64_t L, int D, int M, rlm_dtype dtype);

/* ------------------------------------------------------------------ mixer
 * The mixer wrapper of Sec. 3.4 around the operator:
 *
 *   z_t[d] = sigma(g_t[d]) ybar_t[d] + s[d] l_t[d],   l_t[d] = sum_{k<K} w[d][k] u_{t-k}[d]
 *
 * ybar is y coupled across heads (below), or y itself without coupling.
 * u is the drive (x here), y its resonant mixing (as rlm_mix_prefill_from /
 * rlm_mix_decode compute it), g the gate pre-activation (the gate half of the
 * grouped input projection), sigma the logistic function, and l the local
 * lexical path: a causal depthwise convolution of kernel size K whose output is
 * scaled channel-wise by s.  The output projection that follows z is outside. */
#define RLM_MAX_LOCAL_K 8

/* Head coupling (Sec. 3.4): C = I + (lambda_c / sqrt(H)) tanh(c_raw) mixes the H
 * heads of each token, ybar[g*dh + i] = sum_h C[g][h] y[h*dh + i] with dh = D / H:
 * the D channels are the heads' dh channels, head-major.  c_raw [H][H] fp32
 * row-major; 1 <= H <= 64, D % H == 0, D <= 8192; lambda_c = 0 is the identity. */
typedef struct {
    const float *c_raw;
    float lambda_c;
    int H;
} rlm_coupling;

/* Local lexical path (Sec. 3.4).  conv_w [D][K] fp32: conv_w[d*K + k] multiplies
 * u_{t-k}[d]; scale [D] fp32 (s).  0 <= K <= RLM_MAX_LOCAL_K; K = 0 means no
 * local path (conv_w and scale are then not read). */
typedef struct {
    const float *conv_w;
    const float *scale;
    int D, K;
} rlm_local;

/* The local path's drive history: the K-1 drives before the next token, oldest
 * first, [B][K-1][D] in the element type of x: u[(b*(K-1) + j)*D + d] holds
 * u_{t-K+1+j}[d] when the next token is t.  Unused (may be NULL) when K <= 1. */
typedef struct {
    void *u;
    rlm_dtype dtype;
    int64_t B;
    int D, K;
} rlm_conv_state;

/* Mixer output over a sequence.
 *   x         [B][L][D] drive (F32 or BF16)
 *   g         nullable; [B][L][D] gate pre-activation, x's shape and dtype; NULL
 *             means no gate (sigma(g) taken as 1)
 *   p         resonator parameters
 *   local     nullable (no local path) or K = 0
 *   coupling  nullable (no coupling)
 *   state_in  nullable; the resonators' state before token 0 (as rlm_mix_prefill_from)
 *   conv_in   nullable; the drive history before token 0 (zero drives if NULL)
 *   z         [B][L][D] output, x's shape and dtype; must not overlap x, g, the
 *             parameters or the states
 *   state_out nullable; terminal state and coefficients (may alias state_in)
 *   conv_out  nullable; the history after token L-1 (may alias conv_in exactly)
 * Workspace: rlm_prefill_workspace_size.  With a gate only (no local path, no
 * coupling), bf16 with M <= 16 on unsegmented shapes applies the gate inside the
 * tcgen05 prefill's epilogue (one pass: x and g in, z out).  Otherwise the mixing
 * is written into z and one persistent pass over whole-row tiles applies the
 * coupling, the gate and the local path (rows of at most 2 KB; H in {1, 2, 4, 8,
 * 16} with D / H a multiple of 4); other shapes take a coupling pass and a
 * channel-pair pass. */
RLM_API rlm_status rlm_mixer_prefill(const rlm_tensor *x, const rlm_tensor *g, const rlm_params *p,
                                     const rlm_local *local, const rlm_coupling *coupling, const rlm_state *state_in,
                                     const rlm_conv_state *conv_in, rlm_tensor *z, rlm_state *state_out,
                                     rlm_conv_state *conv_out, const rlm_launch *launch);

/* One decode step of the mixer: the recurrence step of rlm_mix_decode, the
 * coupling, the gate, and the local path over the cached history.  Without
 * coupling: the decode kernel with the gate and the local path fused.  With
 * coupling: one kernel, one block per batch row, where D <= 512, D * M <= 4096
 * and M / 2 is a power of two; otherwise the recurrence step, then one kernel per
 * batch row for the coupling, the gate and the local path.
 *   x_t, g_t [B][1][D] (g_t nullable: no gate); state updated in place; conv
 *   ([B][K-1][D], required when K >= 2) shifted in place by one token; z_t
 *   [B][1][D] output.  No workspace. */
RLM_API rlm_status rlm_mixer_decode(const rlm_tensor *x_t, const rlm_tensor *g_t, rlm_state *state,
                                    const rlm_local *local, const rlm_coupling *coupling, rlm_conv_state *conv,
                                    rlm_tensor *z_t, const rlm_launch *launch);

/* ------------------------------------------------------------------ utility
 * rlm_validate_params: copies p to the host (synchronous) and checks that every
 * value is finite and every gamma >= 0 (Sec. 3.1 requires alpha > 0; gamma = 0
 * is accepted as the undamped limit).  The hot-path calls do not read
 * parameters on the host, so they do not perform this check. */
RLM_API rlm_status rlm_validate_params(const rlm_params *p);

/* Synchronises launch->stream, then reports and clears the device status word:
 * RLM_ERR_TIMEOUT if a bounded wait expired since the last call, else RLM_OK
 * (or RLM_ERR_CUDA if the stream reports an error). */
RLM_API rlm_status rlm_get_device_status(const rlm_launch *launch);

/* Static description of a status code. */
RLM_API const char *rlm_status_string(rlm_status status);

/* Test hook for failure detection; the paper has no counterpart.  on != 0 makes
 * the next prefills that split a sequence into segments (few batch rows, M <= 16,
 * bf16) run with a wait bound of about 1 ms instead of about 2 s, and makes the
 * first segment withhold the flag that publishes its end state: every later
 * segment's wait then expires, the kernel records RLM_ERR_TIMEOUT in the device
 * status word, drains what it issued, frees its tensor memory and returns (its
 * output is undefined).  on = 0 restores normal operation.  Synchronous (two
 * copies to device symbols on the current device); not for production use. */
RLM_API rlm_status rlm_test_stall_segments(int on);

/* Human-readable reason for the last non-OK status returned on this host
 * thread (valid until the next call on the thread). */
RLM_API const char *rlm_last_error(void);

/* Library version as major*10000 + minor*100 + patch. */
RLM_API int rlm_version(void);

/* Number of kernels this library has launched in this process so far (a
 * host-side count, incremented at each launch; for accounting in benchmarks). */
RLM_API unsigned long long rlm_kernels_launched(void);


#ifdef __cplusplus
}
#endif
#endif /* RLM_H_ */
