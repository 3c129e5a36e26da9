/*
 * rlm_oracle.c -- plain, slow, fp64 CPU oracle for causal resonant field
 * mixing (ResonatorLM, arxiv 2607.05583).
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing in the product library calls, links or
 * loads this file.  Only the tests, the smoke check and the benchmark's
 * CPU-baseline leg use it.  It shares no code, header, table or constant
 * with the CUDA path.
 *
 * Notation (Sec. 3.1-3.3 of the paper, generalised to M modes per channel):
 *   x      [B][L][D]  drive (the token field), row-major, channel innermost
 *   decay  gamma [D][M], freq omega [D][M], amp A [D][M], phase phi [D][M]
 *   lambda = exp(-gamma) (cos omega + i sin omega)           (Eq. 5)
 *   c      = A exp(+i phi)                                    (reading Z1)
 *   K_d[n] = sum_m A exp(-gamma n) cos(omega n + phi)         (Eq. 1)
 *   y[b,t,d] = sum_{j<=t} K_d[t-j] x[b,j,d]                   (Eq. 2)
 *
 * Every quantity is computed in double precision (double complex where the
 * paper's state is complex).  Inputs arrive already promoted to double.
 */
#include <complex.h>
#include <math.h>
#include <stddef.h>
#include <stdint.h>
#include <stdlib.h>
#ifdef _OPENMP
#include <omp.h>
#endif

typedef double complex cplx;

int oracle_num_threads(void)
{
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}

/* Eq. 1 summed over the modes of one channel: the closed-form impulse
 * response of channel d at integer lag n >= 0. */
static double kernel_at(int M, const double *g, const double *w,
                        const double *a, const double *p, long n)
{
    double k = 0.0;
    for (int m = 0; m < M; ++m)
        k += a[m] * exp(-g[m] * (double)n) * cos(w[m] * (double)n + p[m]);
    return k;
}

/* K[d][n] for n = 0..L-1 (Eq. 1). */
void oracle_kernel_table(int D, int M, const double *decay, const double *freq,
                         const double *amp, const double *phase, long L,
                         double *K)
{
    for (int d = 0; d < D; ++d)
        for (long n = 0; n < L; ++n)
            K[(size_t)d * L + n] = kernel_at(M, decay + (size_t)d * M,
                                             freq + (size_t)d * M,
                                             amp + (size_t)d * M,
                                             phase + (size_t)d * M, n);
}

/* O1: direct O(L^2) causal convolution with the closed-form kernel
 * (Eq. 1 and Eq. 2).  y must hold B*L*D doubles.  With state_in
 * ([B][D][M][2], the state before token 0; NULL = zero), every output also gets
 * the free response of that state, evaluated in closed form (Eq. 5 powers):
 * sum_m Re(c_m lambda_m^(t+1) s_m) = sum_m A |s| exp(-gamma (t+1))
 * cos(omega (t+1) + phi + arg s). */
void oracle_conv_prefill(long B, long L, int D, int M, const double *x,
                         const double *decay, const double *freq,
                         const double *amp, const double *phase,
                         const double *state_in, double *y)
{
    double *K = (double *)malloc(sizeof(double) * (size_t)D * (size_t)L);
    oracle_kernel_table(D, M, decay, freq, amp, phase, L, K);
#pragma omp parallel for collapse(2) schedule(static)
    for (long b = 0; b < B; ++b)
        for (int d = 0; d < D; ++d) {
            const double *Kd = K + (size_t)d * L;
            for (long t = 0; t < L; ++t) {
                double acc = 0.0;
                for (long j = 0; j <= t; ++j)
                    acc += Kd[t - j] * x[((size_t)b * L + j) * D + d];
                if (state_in)
                    for (int m = 0; m < M; ++m) {
                        const size_t pm = (size_t)d * M + m;
                        const size_t o = (((size_t)b * D + d) * M + m) * 2;
                        const double mag = hypot(state_in[o], state_in[o + 1]);
                        const double arg = atan2(state_in[o + 1], state_in[o]);
                        const double n = (double)(t + 1);
                        acc += amp[pm] * mag * exp(-decay[pm] * n) * cos(freq[pm] * n + phase[pm] + arg);
                    }
                y[((size_t)b * L + t) * D + d] = acc;
            }
        }
    free(K);
}

static cplx mode_lambda(double g, double w) { return exp(-g) * (cos(w) + I * sin(w)); }
static cplx mode_coef(double a, double p) { return a * (cos(p) + I * sin(p)); }

/* O2: the sequential complex recurrence of Sec. 3.3 (Eq. 4-5), run over the
 * whole prompt:  s <- lambda s + x_t,  y_t = sum_m Re(c s), from the state
 * state_in ([B][D][M][2], the state before token 0) or, when it is NULL, from a
 * zero state.  The state after the last token is the prompt's terminal state of
 * Sec. 3.2 (the decay-weighted sum of past drives), returned as
 * state[B][D][M][2] (real, imaginary) when state is not NULL; it may alias
 * state_in. */
void oracle_rec_prefill(long B, long L, int D, int M, const double *x,
                        const double *decay, const double *freq,
                        const double *amp, const double *phase,
                        const double *state_in, double *y, double *state)
{
#pragma omp parallel for collapse(2) schedule(static)
    for (long b = 0; b < B; ++b)
        for (int d = 0; d < D; ++d) {
            for (long t = 0; t < L; ++t)
                y[((size_t)b * L + t) * D + d] = 0.0;
            for (int m = 0; m < M; ++m) {
                size_t pm = (size_t)d * M + m;
                cplx lam = mode_lambda(decay[pm], freq[pm]);
                cplx c = mode_coef(amp[pm], phase[pm]);
                const size_t o = (((size_t)b * D + d) * M + m) * 2;
                cplx s = state_in ? state_in[o] + I * state_in[o + 1] : 0.0;
                for (long t = 0; t < L; ++t) {
                    size_t i = ((size_t)b * L + t) * D + d;
                    s = lam * s + x[i];
                    y[i] += creal(c * s);
                }
                if (state) {
                    state[o] = creal(s);
                    state[o + 1] = cimag(s);
                }
            }
        }
}

/* One decode step of Sec. 3.3 (Eq. 4-5) for a batch of single tokens.
 * state_in/state_out: [B][D][M][2]; x_t, y_t: [B][D].  state_out may alias
 * state_in. */
void oracle_rec_decode(long B, int D, int M, const double *state_in,
                       const double *x_t, const double *decay,
                       const double *freq, const double *amp,
                       const double *phase, double *state_out, double *y_t)
{
    for (long b = 0; b < B; ++b)
        for (int d = 0; d < D; ++d) {
            double acc = 0.0;
            for (int m = 0; m < M; ++m) {
                size_t pm = (size_t)d * M + m;
                size_t o = (((size_t)b * D + d) * M + m) * 2;
                cplx s = state_in[o] + I * state_in[o + 1];
                s = mode_lambda(decay[pm], freq[pm]) * s + x_t[(size_t)b * D + d];
                acc += creal(mode_coef(amp[pm], phase[pm]) * s);
                state_out[o] = creal(s);
                state_out[o + 1] = cimag(s);
            }
            y_t[(size_t)b * D + d] = acc;
        }
}

/* O3, convolution route.  With loss l and dy = dl/dy, the chain rule through
 * Eq. 2 gives
 *   dx[b,j,d] = sum_{t>=j} K_d[t-j] dy[b,t,d]
 *   rho_d[n]  = sum_b sum_{t>=n} dy[b,t,d] x[b,t-n,d]   (dl/dK_d[n])
 * and, differentiating Eq. 1 term by term,
 *   dA   =  sum_n rho[n] exp(-g n) cos(w n + p)
 *   dphi = -sum_n rho[n] A exp(-g n) sin(w n + p)
 *   dg   = -sum_n rho[n] n A exp(-g n) cos(w n + p)
 *   dw   = -sum_n rho[n] n A exp(-g n) sin(w n + p).
 * Gradients are [D][M] and are overwritten. */
/* Optional state terms (all [B][D][M][2]; NULL = absent):
 *   state_in     the state before token 0 of the forward pass (Sec. 3.2-3.3);
 *   d_state_out  g, the loss gradient w.r.t. (Re, Im) of the terminal state,
 *                i.e. the loss has the extra term Re(conj(g) s_L);
 *   d_state_in   output: the loss gradient w.r.t. (Re, Im) of state_in.
 * Convolution route: every extra term as a direct sum of closed-form powers
 * (Eq. 5): with n = L-1-j, dx_j += |g| e^{-gamma n} cos(omega n - arg g);
 * W = sum_t dy_t lambda^(t+1), V = sum_t dy_t (t+1) lambda^(t+1),
 * J = sum_j (L-1-j) lambda^(L-1-j) x_j + L lambda^L s_in;
 * G += s_in W, P += s_in V, dgamma -= Re(conj(g) J), domega -= Im(conj(g) J),
 * d_state_in = conj(c W) + g conj(lambda^L). */
static cplx lam_pow_closed(double g, double w, double n)
{
    return exp(-g * n) * (cos(w * n) + I * sin(w * n));
}

void oracle_backward_conv(long B, long L, int D, int M, const double *x,
                          const double *dy, const double *decay,
                          const double *freq, const double *amp,
                          const double *phase, const double *state_in,
                          const double *d_state_out, double *dx, double *d_decay,
                          double *d_freq, double *d_amp, double *d_phase,
                          double *d_state_in)
{
    double *K = (double *)malloc(sizeof(double) * (size_t)D * (size_t)L);
    oracle_kernel_table(D, M, decay, freq, amp, phase, L, K);
#pragma omp parallel for schedule(static)
    for (int d = 0; d < D; ++d) {
        const double *Kd = K + (size_t)d * L;
        for (long b = 0; b < B; ++b)
            for (long j = 0; j < L; ++j) {
                double acc = 0.0;
                for (long t = j; t < L; ++t)
                    acc += Kd[t - j] * dy[((size_t)b * L + t) * D + d];
                dx[((size_t)b * L + j) * D + d] = acc;
            }
        double *rho = (double *)calloc((size_t)L, sizeof(double));
        for (long n = 0; n < L; ++n) {
            double r = 0.0;
            for (long b = 0; b < B; ++b)
                for (long t = n; t < L; ++t)
                    r += dy[((size_t)b * L + t) * D + d] *
                         x[((size_t)b * L + t - n) * D + d];
            rho[n] = r;
        }
        for (int m = 0; m < M; ++m) {
            size_t pm = (size_t)d * M + m;
            double g = decay[pm], w = freq[pm], a = amp[pm], p = phase[pm];
            double sa = 0, sp = 0, sg = 0, sw = 0;
            for (long n = 0; n < L; ++n) {
                double e = exp(-g * (double)n);
                double cs = cos(w * (double)n + p), sn = sin(w * (double)n + p);
                sa += rho[n] * e * cs;
                sp -= rho[n] * a * e * sn;
                sg -= rho[n] * (double)n * a * e * cs;
                sw -= rho[n] * (double)n * a * e * sn;
            }
            const cplx c = a * (cos(p) + I * sin(p));
            for (long b = 0; b < B; ++b) {
                const size_t o = (((size_t)b * D + d) * M + m) * 2;
                const cplx si = state_in ? state_in[o] + I * state_in[o + 1] : 0.0;
                const cplx gg = d_state_out ? d_state_out[o] + I * d_state_out[o + 1] : 0.0;
                cplx W = 0.0, V = 0.0, J = 0.0;
                for (long t = 0; t < L; ++t) {
                    const double u = dy[((size_t)b * L + t) * D + d];
                    const cplx pw = lam_pow_closed(g, w, (double)(t + 1));
                    W += u * pw;
                    V += u * (double)(t + 1) * pw;
                    J += (double)(L - 1 - t) * lam_pow_closed(g, w, (double)(L - 1 - t)) *
                         x[((size_t)b * L + t) * D + d];
                }
                J += (double)L * lam_pow_closed(g, w, (double)L) * si;
                const cplx Gi = si * W, Pi = si * V;
                sa += creal((cos(p) + I * sin(p)) * Gi);
                sp -= cimag(c * Gi);
                sg -= creal(c * Pi) + creal(conj(gg) * J);
                sw -= cimag(c * Pi) + cimag(conj(gg) * J);
                if (d_state_in) {
                    const cplx ds = conj(c * W) + gg * conj(lam_pow_closed(g, w, (double)L));
                    d_state_in[o] = creal(ds);
                    d_state_in[o + 1] = cimag(ds);
                }
                if (d_state_out) {
                    const double mag = cabs(gg), arg = carg(gg);
                    for (long j = 0; j < L; ++j) {
                        const double n = (double)(L - 1 - j);
                        dx[((size_t)b * L + j) * D + d] += mag * exp(-g * n) * cos(w * n - arg);
                    }
                }
            }
            d_amp[pm] = sa;
            d_phase[pm] = sp;
            d_decay[pm] = sg;
            d_freq[pm] = sw;
        }
        free(rho);
    }
    free(K);
}

/* O3, recurrence route (independent of the convolution route).  Reverse-time
 * adjoint of the Eq. 4 recurrence with its Jordan partner:
 *   S_j = lambda S_{j+1} + dy_j            (S_j = sum_{t>=j} lambda^{t-j} dy_t)
 *   R_j = lambda (R_{j+1} + S_{j+1})       (R_j = sum_{t>=j} (t-j) lambda^{t-j} dy_t)
 *   dx_j = sum_m Re(c S_j),  G = sum_{b,j} x_j S_j,  P = sum_{b,j} x_j R_j
 *   dA = Re(e^{i phi} G), dphi = -Im(c G), dgamma = -Re(c P), domega = -Im(c P). */
/* State terms (see oracle_backward_conv) by recurrences: the terminal-state
 * gradient is a second adjoint Phi_j = lambda Phi_{j+1}, Phi_{L-1} = conj(g),
 * read out with coefficient 1 (dx_j += Re Phi_j); J uses the unit adjoint
 * U_j = lambda U_{j+1} (U_{L-1} = 1) and its Jordan partner
 * Q_j = lambda (Q_{j+1} + U_{j+1}) (Q_j = (L-1-j) lambda^(L-1-j)): J = sum x Q +
 * s_in lambda (Q_0 + U_0); with the adjoint pair's end values S_0, R_0:
 * G += s_in lambda S_0, P += s_in lambda (R_0 + S_0),
 * d_state_in = conj(c lambda S_0) + g conj(lambda U_0). */
void oracle_backward_rec(long B, long L, int D, int M, const double *x,
                         const double *dy, const double *decay,
                         const double *freq, const double *amp,
                         const double *phase, const double *state_in,
                         const double *d_state_out, double *dx, double *d_decay,
                         double *d_freq, double *d_amp, double *d_phase,
                         double *d_state_in)
{
#pragma omp parallel for schedule(static)
    for (int d = 0; d < D; ++d) {
        for (long b = 0; b < B; ++b)
            for (long j = 0; j < L; ++j)
                dx[((size_t)b * L + j) * D + d] = 0.0;
        for (int m = 0; m < M; ++m) {
            size_t pm = (size_t)d * M + m;
            cplx lam = mode_lambda(decay[pm], freq[pm]);
            cplx c = mode_coef(amp[pm], phase[pm]);
            cplx G = 0.0, P = 0.0, GJ = 0.0;
            for (long b = 0; b < B; ++b) {
                const size_t o = (((size_t)b * D + d) * M + m) * 2;
                const cplx si = state_in ? state_in[o] + I * state_in[o + 1] : 0.0;
                const cplx gg = d_state_out ? d_state_out[o] + I * d_state_out[o + 1] : 0.0;
                cplx S = 0.0, R = 0.0, Phi = 0.0, U = 0.0, Q = 0.0, J = 0.0;
                for (long j = L - 1; j >= 0; --j) {
                    size_t i = ((size_t)b * L + j) * D + d;
                    R = lam * (R + S);
                    S = lam * S + dy[i];
                    if (j == L - 1) {
                        Phi = conj(gg);
                        U = 1.0;
                    } else {
                        Q = lam * (Q + U);
                        U = lam * U;
                        Phi = lam * Phi;
                    }
                    dx[i] += creal(c * S) + creal(Phi);
                    G += x[i] * S;
                    P += x[i] * R;
                    J += x[i] * Q;
                }
                J += si * lam * (Q + U);
                G += si * lam * S;
                P += si * lam * (R + S);
                GJ += conj(gg) * J;
                if (d_state_in) {
                    const cplx ds = conj(c * lam * S) + gg * conj(lam * U);
                    d_state_in[o] = creal(ds);
                    d_state_in[o + 1] = cimag(ds);
                }
            }
            d_amp[pm] = creal((cos(phase[pm]) + I * sin(phase[pm])) * G);
            d_phase[pm] = -cimag(c * G);
            d_decay[pm] = -creal(c * P) - creal(GJ);
            d_freq[pm] = -cimag(c * P) - cimag(GJ);
        }
    }
}
