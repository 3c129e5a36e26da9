"""fp64 CPU oracle for causal resonant field mixing (ResonatorLM, arxiv 2607.05583).

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
CPU-baseline / reference legs of ``bench.py`` may import this package.  The
product library (``paper_2607_05583_gb300``) never imports it, and it never
imports the product: the two share no code.

The arithmetic lives in ``rlm_oracle.c`` (plain C, double precision, optional
OpenMP over independent channels).  This module only compiles that file with
gcc and marshals numpy arrays into it.

Functions (all arrays float64, C-contiguous; shapes as in the paper's notation,
channel innermost):

* ``conv_prefill``   O1: direct O(L^2) causal convolution, Eq. 1-2 (plus the
                      closed-form free response of an initial state).
* ``rec_prefill``    O2: sequential complex recurrence, Eq. 4-5, from a zero or
                      given initial state, plus the prompt's terminal state
                      (Sec. 3.2).
* ``rec_decode``     one decode step, Eq. 4-5.
* ``backward_conv``  O3 via the convolution route (chain rule through Eq. 1-2).
* ``backward_rec``   O3 via the reverse-time Jordan recurrence.
* ``kernel_table``   K_d[n] of Eq. 1.
* ``local_conv``     the local lexical path of Sec. 3.4: causal depthwise
                      convolution of kernel size K over the drive history.
* ``coupling_matrix`` / ``couple_heads``
                     head coupling of Sec. 3.4: C = I + lambda_c / sqrt(H) tanh(C~),
                      ybar_g = sum_h C_gh y_h over head-major channels.
* ``mixer_prefill`` / ``mixer_decode``
                     the mixer output of Sec. 3.4: z = sigmoid(g) * ybar + s * l,
                      with ybar the (optionally coupled) resonant mixing above
                      (numpy, fp64).
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "rlm_oracle.c")
_BUILD_DIR = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD_DIR, "liboracle.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile rlm_oracle.c into oracle/_build/liboracle.so (gcc, -O2, OpenMP)."""
    os.makedirs(_BUILD_DIR, exist_ok=True)
    stale = (not os.path.exists(_LIB_PATH)
             or os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC))
    if force or stale:
        tmp = _LIB_PATH + f".{os.getpid()}.tmp"
        cmd = ["gcc", "-O2", "-std=c11", "-fopenmp", "-fPIC", "-shared",
               _SRC, "-o", tmp, "-lm"]
        subprocess.check_call(cmd)
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(build())
            dp = ctypes.POINTER(ctypes.c_double)
            L_, I_ = ctypes.c_long, ctypes.c_int
            lib.oracle_num_threads.restype = I_
            lib.oracle_kernel_table.argtypes = [I_, I_, dp, dp, dp, dp, L_, dp]
            lib.oracle_conv_prefill.argtypes = [L_, L_, I_, I_, dp, dp, dp, dp, dp, dp, dp]
            lib.oracle_rec_prefill.argtypes = [L_, L_, I_, I_, dp, dp, dp, dp, dp, dp, dp, dp]
            lib.oracle_rec_decode.argtypes = [L_, I_, I_, dp, dp, dp, dp, dp, dp, dp, dp]
            lib.oracle_backward_conv.argtypes = [L_, L_, I_, I_, dp, dp, dp, dp, dp, dp,
                                                 dp, dp, dp, dp, dp, dp, dp, dp]
            lib.oracle_backward_rec.argtypes = [L_, L_, I_, I_, dp, dp, dp, dp, dp, dp,
                                                dp, dp, dp, dp, dp, dp, dp, dp]
            _lib = lib
    return _lib


def _f64(a) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(a, dtype=np.float64))


def _ptr(a: np.ndarray):
    return a.ctypes.data_as(ctypes.POINTER(ctypes.c_double))


def _params(decay, freq, amp, phase):
    ps = [_f64(p) for p in (decay, freq, amp, phase)]
    D, M = ps[0].shape
    for p in ps:
        if p.shape != (D, M):
            raise ValueError("decay/freq/amp/phase must all be [D][M]")
    return ps, D, M


def num_threads() -> int:
    return int(_load().oracle_num_threads())


def kernel_table(decay, freq, amp, phase, L: int) -> np.ndarray:
    """K[d][n] = sum_m A exp(-gamma n) cos(omega n + phi), n < L (Eq. 1)."""
    ps, D, M = _params(decay, freq, amp, phase)
    K = np.empty((D, L), np.float64)
    _load().oracle_kernel_table(D, M, *map(_ptr, ps), L, _ptr(K))
    return K


def _state_pairs(state_in, B, D, M):
    """[B][D][M] complex -> [B][D][M][2] float64 (Re, Im), or None."""
    if state_in is None:
        return None
    s = np.asarray(state_in)
    if s.shape != (B, D, M):
        raise ValueError("state_in must be [B][D][M] complex")
    return np.ascontiguousarray(np.stack([s.real, s.imag], -1), np.float64)


def conv_prefill(x, decay, freq, amp, phase, state_in=None) -> np.ndarray:
    """O1: y[b,t,d] = sum_{j<=t} K_d[t-j] x[b,j,d] by direct summation (Eq. 2), plus,
    when state_in ([B][D][M] complex, the state before token 0) is given, its free
    response sum_m Re(c lambda^(t+1) s) in closed form."""
    x = _f64(x)
    ps, D, M = _params(decay, freq, amp, phase)
    B, L, Dx = x.shape
    assert Dx == D
    sin = _state_pairs(state_in, B, D, M)
    y = np.empty_like(x)
    _load().oracle_conv_prefill(B, L, D, M, _ptr(x), *map(_ptr, ps),
                                _ptr(sin) if sin is not None else None, _ptr(y))
    return y


def rec_prefill(x, decay, freq, amp, phase, state_in=None):
    """O2: sequential recurrence (Eq. 4-5) from state_in ([B][D][M] complex, the
    state before token 0), or from a zero state when it is None.

    Returns (y [B][L][D], state [B][D][M] complex128)."""
    x = _f64(x)
    ps, D, M = _params(decay, freq, amp, phase)
    B, L, Dx = x.shape
    assert Dx == D
    sin = _state_pairs(state_in, B, D, M)
    y = np.empty_like(x)
    st = np.empty((B, D, M, 2), np.float64)
    _load().oracle_rec_prefill(B, L, D, M, _ptr(x), *map(_ptr, ps),
                               _ptr(sin) if sin is not None else None, _ptr(y), _ptr(st))
    return y, st[..., 0] + 1j * st[..., 1]


def rec_decode(state, x_t, decay, freq, amp, phase):
    """One decode step (Eq. 4-5).  state: [B][D][M] complex; x_t: [B][D].

    Returns (y_t [B][D], new state [B][D][M] complex128)."""
    state = np.asarray(state)
    x_t = _f64(x_t)
    ps, D, M = _params(decay, freq, amp, phase)
    B = x_t.shape[0]
    sin = np.ascontiguousarray(np.stack([state.real, state.imag], -1), np.float64)
    sout = np.empty_like(sin)
    y = np.empty((B, D), np.float64)
    _load().oracle_rec_decode(B, D, M, _ptr(sin), _ptr(x_t), *map(_ptr, ps),
                              _ptr(sout), _ptr(y))
    return y, sout[..., 0] + 1j * sout[..., 1]


def _backward(fn, x, dy, decay, freq, amp, phase, state_in=None, d_state_out=None):
    x, dy = _f64(x), _f64(dy)
    ps, D, M = _params(decay, freq, amp, phase)
    B, L, Dx = x.shape
    assert Dx == D and dy.shape == x.shape
    sin = _state_pairs(state_in, B, D, M)
    gout = _state_pairs(d_state_out, B, D, M)
    want_ds = state_in is not None or d_state_out is not None
    ds = np.empty((B, D, M, 2), np.float64) if want_ds else None
    dx = np.empty_like(x)
    g = [np.empty((D, M), np.float64) for _ in range(4)]
    opt = lambda a: _ptr(a) if a is not None else None
    fn(B, L, D, M, _ptr(x), _ptr(dy), *map(_ptr, ps), opt(sin), opt(gout), _ptr(dx), *map(_ptr, g),
       opt(ds))
    out = {"decay": g[0], "freq": g[1], "amp": g[2], "phase": g[3]}
    if want_ds:
        out["state_in"] = ds[..., 0] + 1j * ds[..., 1]
    return dx, out


def backward_conv(x, dy, decay, freq, amp, phase, state_in=None, d_state_out=None):
    """O3 by the convolution route.  Returns (dx, {decay, freq, amp, phase}); with
    state_in (the forward's initial state) and/or d_state_out (the loss gradient of
    the terminal state, [B][D][M] complex) the dict also holds "state_in", the loss
    gradient of the initial state."""
    return _backward(_load().oracle_backward_conv, x, dy, decay, freq, amp, phase, state_in,
                     d_state_out)


def backward_rec(x, dy, decay, freq, amp, phase, state_in=None, d_state_out=None):
    """O3 by the reverse-time Jordan recurrence.  Same returns as backward_conv."""
    return _backward(_load().oracle_backward_rec, x, dy, decay, freq, amp, phase, state_in,
                     d_state_out)


# ------------------------------------------------------------------ mixer (Sec. 3.4)
def sigmoid(v) -> np.ndarray:
    """The gate nonlinearity gamma = sigma(g) of Sec. 3.1, in fp64."""
    v = _f64(v)
    return 1.0 / (1.0 + np.exp(-v))


def local_conv(u, conv_w, conv_in=None):
    """The local lexical path of Sec. 3.4: l_t[d] = sum_{k<K} w[d][k] u_{t-k}[d],
    a causal depthwise convolution of kernel size K.  Drives before token 0 come
    from conv_in ([B][K-1][D], oldest first: conv_in[:, K-2] is u_{-1}), or are zero.

    Returns (l [B][L][D], the last K-1 drives of conv_in || u, oldest first)."""
    u, w = _f64(u), _f64(conv_w)
    B, L, D = u.shape
    K = w.shape[1]
    if w.shape != (D, K):
        raise ValueError("conv_w must be [D][K]")
    hist = np.zeros((B, max(K - 1, 0), D)) if conv_in is None else _f64(conv_in)
    if hist.shape != (B, max(K - 1, 0), D):
        raise ValueError("conv_in must be [B][K-1][D]")
    ext = np.concatenate([hist, u], axis=1)          # ext[:, K-1+t] = u_t
    l = np.zeros((B, L, D))
    for k in range(K):
        l += w[:, k][None, None, :] * ext[:, K - 1 - k:K - 1 - k + L, :]
    tail = ext[:, ext.shape[1] - max(K - 1, 0):, :].copy()
    return l, tail


def coupling_matrix(c_raw, lambda_c) -> np.ndarray:
    """C = I + (lambda_c / sqrt(H)) tanh(C~) of Sec. 3.4, for C~ = c_raw [H][H]."""
    c = _f64(c_raw)
    H = c.shape[0]
    if c.shape != (H, H):
        raise ValueError("c_raw must be [H][H]")
    return np.eye(H) + (float(lambda_c) / np.sqrt(H)) * np.tanh(c)


def couple_heads(y, C) -> np.ndarray:
    """ybar[..., g*dh + i] = sum_h C[g, h] y[..., h*dh + i] (Sec. 3.4): the channels of
    a token are the H heads' dh channels, head-major (d = h*dh + i)."""
    y, C = _f64(y), _f64(C)
    H = C.shape[0]
    D = y.shape[-1]
    if D % H:
        raise ValueError("D must be a multiple of H")
    dh = D // H
    out = np.zeros_like(y)
    for g in range(H):
        for h in range(H):
            out[..., g * dh:(g + 1) * dh] += C[g, h] * y[..., h * dh:(h + 1) * dh]
    return out


def mixer_prefill(x, g, decay, freq, amp, phase, conv_w, scale, state_in=None, conv_in=None, coupling=None):
    """Mixer output over a sequence (Sec. 3.4): z_t = sigma(g_t) * ybar_t + s * l_t,
    ybar the resonant mixing of the drive x (O2, from state_in), coupled across
    heads when coupling = (c_raw [H][H], lambda_c) is given, and l the local path
    over conv_in || x.  g = None means no gate (gamma = 1).  Returns (z, terminal
    state [B][D][M] complex, last K-1 drives)."""
    y, st = rec_prefill(x, decay, freq, amp, phase, state_in=state_in)
    if coupling is not None:
        y = couple_heads(y, coupling_matrix(*coupling))
    l, tail = local_conv(x, conv_w, conv_in)
    gate = 1.0 if g is None else sigmoid(g)
    return gate * y + _f64(scale)[None, None, :] * l, st, tail


def mixer_decode(state, conv, x_t, g_t, decay, freq, amp, phase, conv_w, scale, coupling=None):
    """One decode step of the mixer: the recurrence step (Eq. 4-5), the head
    coupling (if given), the gate and the local path over the K-1 cached drives.
    state [B][D][M] complex, conv [B][K-1][D], x_t and g_t [B][D] (g_t None: no
    gate).  Returns (z_t, new state, new conv)."""
    y, st = rec_decode(state, x_t, decay, freq, amp, phase)
    if coupling is not None:
        y = couple_heads(y, coupling_matrix(*coupling))
    x_t = _f64(x_t)
    l, tail = local_conv(x_t[:, None, :], conv_w, conv)
    gate = 1.0 if g_t is None else sigmoid(g_t)
    return gate * y + _f64(scale)[None, :] * l[:, 0, :], st, tail
