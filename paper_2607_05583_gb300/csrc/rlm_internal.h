// rlm_internal.h -- declarations shared by the library's translation units.
// Host-side only; device helpers live in rlm_device.cuh.
#pragma once

#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "../../include/rlm.h"

namespace rlm {

// Records a human-readable reason for the next rlm_last_error() on this thread.
void set_error(const char *fmt, ...);

// Multiprocessor count of the current device (cached per device).
int sm_count();

// Adds n to the process-wide count of kernels this library has launched.
void count_launches(int n);

// ---- SIMT chunked scan (rlm_simt.cu) --------------------------------------
// Chunk length the SIMT path uses for a problem; workspace and launch agree.
int simt_chunk_len(int64_t B, int64_t L, int D);
size_t simt_prefill_ws_bytes(int64_t B, int64_t L, int D, int M);
size_t simt_backward_ws_bytes(int64_t B, int64_t L, int D, int M);

// y = causal mixing of x (reverse=false) or the anti-causal mixing used by the
// backward pass for dx (reverse=true: time runs from L-1 down to 0).
// state_out/coef_out may be null.  ws must hold simt_prefill_ws_bytes().
// state_in ([B][D][M] complex, the state before token 0), state_out and
// coef_out may be null; state_out may alias state_in.
cudaError_t simt_prefill(const void *x, void *y, rlm_dtype dt, int64_t B, int64_t L, int D,
                         int M, const float *decay, const float *freq, const float *amp,
                         const float *phase, const float *state_in, float *state_out, float *coef_out,
                         void *ws, cudaStream_t st);

// dx and the four parameter gradients (deterministic reduction); optional state
// terms ([B][D][M] complex, null = absent): the forward's state_in, the loss
// gradient d_state_out of the terminal state, and the output d_state_in.
cudaError_t simt_backward(const void *dy, const void *x, void *dx, rlm_dtype dt, int64_t B,
                          int64_t L, int D, int M, const float *decay, const float *freq,
                          const float *amp, const float *phase, const float *state_in,
                          const float *d_state_out, float *d_state_in, float *g_decay,
                          float *g_freq, float *g_amp, float *g_phase, void *ws,
                          cudaStream_t st);

// Fixed-order (compensated fp32) sum of nparts partial (G, P) arrays of [D][M] each, then the
// four parameter gradients.  J (nullable): nparts partials of conj(g) J from a
// terminal-state gradient g, whose sum's -Re and -Im join dgamma and domega.
cudaError_t grad_reduce(int64_t nparts, int D, int M, const float *amp, const float *phase,
                        const float2 *G, const float2 *P, const float2 *J, float *g_decay, float *g_freq,
                        float *g_amp, float *g_phase, cudaStream_t st);

// ---- tcgen05 prefill for fp32 I/O (rlm_prefill_tc32.cu) ----------------------
// fp32 x and y, M <= 16, from a zero state or from state_in (L a multiple of
// 64); the contraction in three bf16 MMAs per product (hi and lo parts).  No
// workspace.  state_in / state_out / coef_out may be null.
bool tc32_prefill_supported(int64_t B, int64_t L, int D, int M, rlm_dtype dt);
cudaError_t tc32_prefill(const float *x, float *y, int64_t B, int64_t L, int D, int M, const float *decay,
                         const float *freq, const float *amp, const float *phase, const float *state_in,
                         float *state_out, float *coef_out, cudaStream_t st);
cudaError_t read_and_clear_tc32_status(int *status, cudaStream_t st);

// ---- tcgen05 backward (rlm_backward_tc.cu) -----------------------------------
bool tc_backward_supported(int64_t B, int64_t L, int D, int M, rlm_dtype dt);
size_t tc_backward_ws_bytes(int64_t B, int64_t L, int D, int M);
// state_in (the forward's initial state), d_state_out (the loss gradient of the
// terminal state) and d_state_in (output) may be null.
cudaError_t tc_backward(const void *dy, const void *x, void *dx, int64_t B, int64_t L, int D, int M,
                        const float *decay, const float *freq, const float *amp, const float *phase,
                        const float *state_in, const float *d_state_out, float *d_state_in, float *g_decay,
                        float *g_freq, float *g_amp, float *g_phase, void *ws, cudaStream_t st);
cudaError_t read_and_clear_bwd_status(int *status, cudaStream_t st);
// The causal prefill (bf16 I/O, M <= 32) as the same reverse-time tcgen05 scan
// applied to the time-reversed drive; used for the M the tcgen05 prefill does not
// cover.  state_out / coef_out may be null.
bool tc_prefill_rev_supported(int64_t B, int64_t L, int D, int M, rlm_dtype dt);
size_t tc_prefill_rev_ws_bytes(int64_t B, int64_t L, int D, int M);
cudaError_t tc_prefill_rev(const void *x, void *y, int64_t B, int64_t L, int D, int M, const float *decay,
                           const float *freq, const float *amp, const float *phase, const float *state_in,
                           float *state_out, float *coef_out, void *ws, cudaStream_t st);

// ---- decode (rlm_decode.cu) -----------------------------------------------
cudaError_t decode_step(const void *x_t, void *y_t, rlm_dtype dt, int B, int D, int M,
                        float *s, const float *coef, cudaStream_t st);
// The mixer step (Sec. 3.4) fused with the decode step: g_t nullable (no gate);
// hist [B][K-1][D] drive history shifted in place (unused when K <= 1).
cudaError_t mixer_decode_step(const void *x_t, const void *g_t, void *z_t, rlm_dtype dt, int B, int D, int M,
                              float *s, const float *coef, void *hist, const float *conv_w, const float *scale,
                              int K, cudaStream_t st);

// The mixer step in one launch, one block per batch row: recurrence step, C y_t
// (H = 0: no coupling, c_raw unused), gate and local path (with the history
// shift).  Covers M even with M / 2 a power of two, D <= 512 and D * M <= 4096.
bool mixer_decode_coupled_supported(int D, int M);
cudaError_t mixer_decode_coupled(const void *x_t, const void *g_t, void *z_t, rlm_dtype dt, int B, int D, int M,
                                 float *s, const float *coef, void *hist, const float *conv_w, const float *scale,
                                 int K, const float *c_raw, float lambda_c, int H, cudaStream_t st);

// ---- mixer epilogue for the unfused prefill paths (rlm_mixer.cu) ------------
// z <- sigma(g) z + s * (w * u) in place (g nullable; K = 0: no local path), the
// drives before token 0 from hist ([B][K-1][D], nullable = zeros).
cudaError_t mixer_epilogue(const void *x, const void *g, void *z, const void *hist, const float *conv_w,
                           const float *scale, rlm_dtype dt, int64_t B, int64_t L, int D, int K,
                           cudaStream_t st);
// Head coupling (Sec. 3.4) in place over z [B][L][D]: ybar = C y per token,
// C = I + lambda_c / sqrt(H) tanh(c_raw), channels head-major.
cudaError_t couple_heads(void *z, rlm_dtype dt, const float *c_raw, float lambda_c, int H, int64_t B, int64_t L,
                         int D, cudaStream_t st);
// One mixer decode step after the recurrence step wrote y_t into z_t: coupling,
// gate (g_t nullable), local path (K = 0: none) with the history shift.
cudaError_t mixer_finish_coupled(const void *x_t, const void *g_t, void *z_t, void *hist, const float *conv_w,
                                 const float *scale, int K, const float *c_raw, float lambda_c, int H, rlm_dtype dt,
                                 int B, int D, cudaStream_t st);
// The whole mixer pass after the mixing, z <- sigma(g) (C z) + s (w * u) in place,
// as one persistent kernel on whole-row tiles (rlm_mixer_stream.cu); g nullable,
// K = 0 (no local path), H = 0 (no coupling; c_raw unused).  Covers the shapes
// for which mixer_stream_supported() holds.
bool mixer_stream_supported(rlm_dtype dt, int D, int H);
cudaError_t mixer_stream(const void *x, const void *g, void *z, const void *hist, const float *conv_w,
                         const float *scale, int K, const float *c_raw, float lambda_c, int H, rlm_dtype dt,
                         int64_t B, int64_t L, int D, cudaStream_t st);
cudaError_t read_and_clear_mixer_status(int *status, cudaStream_t st);
// out = the last K-1 drives of hist || x (out may alias hist; no-op for K < 2).
cudaError_t conv_tail(const void *x, const void *hist, void *out, rlm_dtype dt, int64_t B, int64_t L, int D,
                      int K, cudaStream_t st);

cudaError_t state_init(float *s, float *coef, int B, int D, int M, const float *decay,
                       const float *freq, const float *amp, const float *phase,
                       cudaStream_t st);

// ---- tcgen05 prefill (rlm_prefill_tc.cu) ------------------------------------
// True when the tensor-core path covers this problem.
bool tc_prefill_supported(int64_t B, int64_t L, int D, int M, rlm_dtype dt);
// True when that path also applies the mixer's gate in its epilogue (unsegmented
// launches).
bool tc_mixer_fused(int64_t B, int64_t L, int D, int M, rlm_dtype dt);
size_t tc_prefill_ws_bytes(int64_t B, int64_t L, int D, int M);
// The gate field (Sec. 3.4) for the fused epilogue: [B][L][D] bf16, non-null.
struct TcMix {
    const void *g;
};
// mix non-null: y receives z = sigma(g) y (requires tc_mixer_fused).
cudaError_t tc_prefill(const void *x, void *y, int64_t B, int64_t L, int D, int M,
                       const float *decay, const float *freq, const float *amp,
                       const float *phase, const float *state_in, float *state_out, float *coef_out,
                       const TcMix *mix, void *ws, cudaStream_t st);
// Device status word written by bounded waits (RLM_OK or RLM_ERR_TIMEOUT).
cudaError_t read_and_clear_device_status(int *status, cudaStream_t st);
// Test hook of the failure-detection test: on = 1 shortens the prefill's wait
// bound to about 1 ms and makes sequence segment 0 withhold its end-state flag.
cudaError_t set_segment_stall(int on);

}  // namespace rlm
