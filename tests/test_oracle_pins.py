"""Pins for the fp64 CPU oracle: each test checks the oracle against something
other than itself (hand-derived closed forms, textbook special cases, library
routines, the paper's FFT route, brute-force finite differences, invariants).

A plausible mistake in the oracle (dropped term, flipped phase sign, off-by-one
lag, wrong decay sign, transposed operand) fails at least one of these.
"""
import math
import os

import numpy as np
import pytest
import scipy.signal

import oracle
from synth import make_inputs

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _parse_expr(tok: str) -> float:
    env = {"pi": math.pi, "ln2": math.log(2.0)}
    return float(eval(tok, {"__builtins__": {}}, env))


def _load_impulse_golden():
    cases = []
    with open(os.path.join(GOLDEN, "impulse_closed_form.txt")) as f:
        for line in f:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            lhs, rhs = line.split("|")
            modes = [[_parse_expr(t) for t in m.split()] for m in lhs.split(";")]
            vals = [float(v) for v in rhs.split()]
            cases.append((np.array(modes, np.float64), np.array(vals)))
    return cases


def _golden_kv(name):
    out = {}
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.split("#")[0].strip()
            if line:
                k, v = line.split()
                out[k] = float(v)
    return out


def _one_channel_params(modes):
    # modes rows: alpha omega phi A  ->  [D=1][M] arrays
    g, w, p, a = modes[:, 0], modes[:, 1], modes[:, 2], modes[:, 3]
    return g[None], w[None], a[None], p[None]


# ---------------------------------------------------------------- Eq. 1 / I1
@pytest.mark.parametrize("case", range(len(_load_impulse_golden())))
def test_impulse_matches_hand_derived_closed_form(case):
    """I1: a unit impulse reproduces the hand-derived damped sinusoid (Eq. 1).

    The phi = pi/2 lines pin the phase sign of the readout (cos(omega t + phi),
    not cos(omega t - phi)); the ln2 lines pin the decay sign."""
    modes, want = _load_impulse_golden()[case]
    decay, freq, amp, phase = _one_channel_params(modes)
    L = len(want)
    x = np.zeros((1, L, 1))
    x[0, 0, 0] = 1.0
    y1 = oracle.conv_prefill(x, decay, freq, amp, phase)[0, :, 0]
    y2, _ = oracle.rec_prefill(x, decay, freq, amp, phase)
    np.testing.assert_allclose(y1, want, rtol=0, atol=1e-14)
    np.testing.assert_allclose(y2[0, :, 0], want, rtol=0, atol=1e-14)
    np.testing.assert_allclose(oracle.kernel_table(decay, freq, amp, phase, L)[0], want,
                               rtol=0, atol=1e-14)


def test_impulse_at_offset_and_channel_independence():
    """An impulse at t0 in channel 1 only gives K_1[t - t0] in channel 1, zero elsewhere."""
    inp = make_inputs(1, 40, 3, 2, "f32", seed=3)
    x = np.zeros((1, 40, 3))
    x[0, 7, 1] = 1.0
    K = oracle.kernel_table(*inp.params(), 40)
    for y in (oracle.conv_prefill(x, *inp.params()), oracle.rec_prefill(x, *inp.params())[0]):
        np.testing.assert_array_equal(y[0, :, 0], 0.0)
        np.testing.assert_array_equal(y[0, :, 2], 0.0)
        np.testing.assert_array_equal(y[0, :7, 1], 0.0)
        np.testing.assert_allclose(y[0, 7:, 1], K[1, :33], rtol=1e-12, atol=1e-14)


# ---------------------------------------------------------------- I4 cumsum
def test_zero_damping_zero_frequency_is_cumulative_sum():
    """I4: gamma = 0, omega = 0, phi = 0, A = 1, M = 1 gives the inclusive cumsum
    (pins the lag-0 term, reading Z2)."""
    rng = np.random.default_rng(1)
    x = rng.standard_normal((2, 100, 3))
    z, o = np.zeros((3, 1)), np.ones((3, 1))
    want = np.cumsum(x, axis=1)
    np.testing.assert_allclose(oracle.conv_prefill(x, z, z, o, z), want, rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(oracle.rec_prefill(x, z, z, o, z)[0], want, rtol=1e-12, atol=1e-12)


# ------------------------------------------------- library IIR filter (scipy)
def _lfilter_reference(x, decay, freq, amp, phase):
    """Each mode is the first-order complex IIR filter 1/(1 - lambda z^-1);
    scipy.signal.lfilter runs it, the readout takes Re(c s)."""
    B, L, D = x.shape
    y = np.zeros((B, L, D))
    for d in range(D):
        for m in range(decay.shape[1]):
            lam = np.exp(-float(decay[d, m]) + 1j * float(freq[d, m]))
            c = float(amp[d, m]) * np.exp(1j * float(phase[d, m]))
            s = scipy.signal.lfilter([1.0], [1.0, -lam], x[:, :, d].astype(np.complex128), axis=1)
            y[:, :, d] += (c * s).real
    return y


def test_recurrence_and_convolution_match_scipy_lfilter():
    inp = make_inputs(2, 300, 5, 3, "f32", seed=5)
    want = _lfilter_reference(inp.x.astype(np.float64), *inp.params())
    np.testing.assert_allclose(oracle.conv_prefill(inp.x, *inp.params()), want,
                               rtol=1e-10, atol=1e-10)
    np.testing.assert_allclose(oracle.rec_prefill(inp.x, *inp.params())[0], want,
                               rtol=1e-10, atol=1e-10)


# ------------------------------------------------ Eq. 3 (the paper's FFT route)
def test_convolution_matches_fft_route_of_eq3():
    """Eq. 3: y = F^-1(F(u) . F(k)), zero-padded to the next power of two >= 2L.
    The kernel comes from scipy's impulse response, not from the oracle."""
    inp = make_inputs(1, 513, 4, 4, "f32", seed=7)
    B, L, D = inp.x.shape
    delta = np.zeros((1, L, D))
    delta[0, 0, :] = 1.0
    k = _lfilter_reference(delta, *inp.params())[0]          # [L][D]
    n = 1 << (2 * L - 1).bit_length()
    Y = np.fft.irfft(np.fft.rfft(inp.x.astype(np.float64), n, axis=1)
                     * np.fft.rfft(k, n, axis=0)[None], n, axis=1)[:, :L]
    np.testing.assert_allclose(oracle.conv_prefill(inp.x, *inp.params()), Y,
                               rtol=1e-9, atol=1e-9)


# ---------------------------------------------------------------- I2
def test_convolution_equals_recurrence():
    """I2: O1 (direct convolution) and O2 (recurrence) agree to ~1e-12."""
    inp = make_inputs(2, 777, 6, 5, "f32", seed=11)
    y1 = oracle.conv_prefill(inp.x, *inp.params())
    y2, _ = oracle.rec_prefill(inp.x, *inp.params())
    assert np.linalg.norm(y1 - y2) / np.linalg.norm(y1) < 1e-12


# ---------------------------------------------------------------- I8
def test_constant_drive_is_geometric_series():
    """I8: x = 1 gives y_t = Re sum_m c (1 - lambda^(t+1)) / (1 - lambda)."""
    inp = make_inputs(1, 200, 3, 4, "f32", seed=13)
    x = np.ones((1, 200, 3))
    t = np.arange(200)[:, None, None]
    lam = np.exp(-inp.decay.astype(np.float64) + 1j * inp.freq)[None]
    c = (inp.amp.astype(np.float64) * np.exp(1j * inp.phase.astype(np.float64)))[None]
    want = (c * (1 - lam ** (t + 1)) / (1 - lam)).real.sum(-1)
    np.testing.assert_allclose(oracle.conv_prefill(x, *inp.params())[0], want, rtol=1e-10, atol=1e-10)
    np.testing.assert_allclose(oracle.rec_prefill(x, *inp.params())[0][0], want, rtol=1e-10, atol=1e-10)


def test_terminal_state_is_decay_weighted_sum_of_drives():
    """Sec. 3.2: the prompt's terminal state is sum_j lambda^(L-1-j) x_j (per mode),
    computed here with numpy.polyval (Horner) as an independent route."""
    inp = make_inputs(2, 150, 3, 4, "f32", seed=17)
    _, st = oracle.rec_prefill(inp.x, *inp.params())
    lam = np.exp(-inp.decay.astype(np.float64) + 1j * inp.freq)
    for b in range(2):
        for d in range(3):
            for m in range(4):
                want = np.polyval(inp.x[b, :, d].astype(np.complex128), lam[d, m])
                assert abs(st[b, d, m] - want) <= 1e-10 * max(1.0, abs(want))


# ---------------------------------------------------------------- I3
def test_prefill_then_decode_equals_longer_prefill():
    """I3: prefill(x[0..L]) == prefill(x[0..L-1]) followed by decode(x_L)."""
    inp = make_inputs(3, 65, 4, 3, "f32", seed=19)
    y_full, st_full = oracle.rec_prefill(inp.x, *inp.params())
    _, st = oracle.rec_prefill(inp.x[:, :64], *inp.params())
    y_t, st2 = oracle.rec_decode(st, inp.x[:, 64], *inp.params())
    np.testing.assert_allclose(y_t, y_full[:, 64], rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(st2, st_full, rtol=1e-12, atol=1e-12)
    y_conv = oracle.conv_prefill(inp.x, *inp.params())
    np.testing.assert_allclose(y_t, y_conv[:, 64], rtol=1e-10, atol=1e-10)


def test_many_decode_steps_equal_prefill():
    inp = make_inputs(2, 40, 3, 2, "f32", seed=23)
    st = np.zeros((2, 3, 2), np.complex128)
    ys = []
    for t in range(40):
        y_t, st = oracle.rec_decode(st, inp.x[:, t], *inp.params())
        ys.append(y_t)
    want = oracle.conv_prefill(inp.x, *inp.params())
    np.testing.assert_allclose(np.stack(ys, 1), want, rtol=1e-11, atol=1e-11)


# ---------------------------------------------------------------- I6
def test_causality_prefix_unchanged_by_suffix_perturbation():
    """I6 (Sec. 3.5, Table 2): perturbing x[t >= t0] must not change y[t < t0].
    The paper reports a maximum prefix error below 1e-6; the oracle's is 0."""
    kv = _golden_kv("physics_diagnostics.txt")
    inp = make_inputs(2, 300, 4, 3, "f32", seed=29)
    x2 = inp.x.astype(np.float64).copy()
    x2[:, 123:] += np.random.default_rng(0).standard_normal(x2[:, 123:].shape)
    for f in (oracle.conv_prefill, lambda *a: oracle.rec_prefill(*a)[0]):
        y1, y2 = f(inp.x, *inp.params()), f(x2, *inp.params())
        err = np.abs(y1[:, :123] - y2[:, :123]).max()
        assert err == 0.0 and err < kv["causality_threshold"]
        assert np.abs(y1[:, 123:] - y2[:, 123:]).max() > 1e-3


# ---------------------------------------------------------------- I7
def test_zero_drive_state_energy_decays_as_exp_minus_2_gamma_t():
    """I7 (Sec. 3.5): with zero drive, |s_t|^2 = exp(-2 gamma t) |s_0|^2 per mode."""
    inp = make_inputs(2, 50, 3, 4, "f32", seed=31)
    _, st0 = oracle.rec_prefill(inp.x, *inp.params())
    st = st0
    z = np.zeros((2, 3))
    for t in range(1, 21):
        _, st = oracle.rec_decode(st, z, *inp.params())
        want = np.exp(-2 * inp.decay.astype(np.float64) * t)[None] * np.abs(st0) ** 2
        np.testing.assert_allclose(np.abs(st) ** 2, want, rtol=1e-12)


@pytest.mark.parametrize("key", ["half_life_min", "half_life_max"])
def test_half_life_of_a_mode(key):
    """Half-life log(2)/alpha (Sec. 3.5; range 2..2048 in Table 2): after h zero-drive
    steps the state's magnitude halves, and the impulse envelope at lag h is 1/2."""
    h = int(_golden_kv("physics_diagnostics.txt")[key])
    g = np.array([[math.log(2.0) / h]])
    w, p, a = np.array([[0.7]]), np.array([[0.0]]), np.array([[1.0]])
    st = np.array([[[3.0 - 4.0j]]])
    z = np.zeros((1, 1))
    for _ in range(h):
        _, st = oracle.rec_decode(st, z, g, w, a, p)
    assert abs(abs(st[0, 0, 0]) - 2.5) < 1e-9
    K = oracle.kernel_table(g, np.zeros((1, 1)), a, p, h + 1)[0]
    assert abs(K[h] - 0.5) < 1e-12


# ---------------------------------------------------------------- I9
def test_linearity_and_time_shift_equivariance():
    inp = make_inputs(1, 200, 3, 3, "f32", seed=37)
    rng = np.random.default_rng(2)
    x1, x2 = rng.standard_normal((2, 1, 200, 3))
    f = lambda x: oracle.conv_prefill(x, *inp.params())
    np.testing.assert_allclose(f(2.5 * x1 - 0.75 * x2), 2.5 * f(x1) - 0.75 * f(x2),
                               rtol=1e-11, atol=1e-11)
    xs = np.zeros_like(x1)
    xs[:, 17:] = x1[:, :-17]
    np.testing.assert_allclose(f(xs)[:, 17:], f(x1)[:, :-17], rtol=1e-11, atol=1e-11)
    np.testing.assert_array_equal(f(xs)[:, :17], 0.0)


# ---------------------------------------------------------------- I5 backward
def _loss(x, dy, params):
    return float(np.sum(dy * oracle.conv_prefill(x, *params)))


# ------------------------------------------------- prefill from an initial state
def test_prefill_from_state_continues_the_sequence():
    """Prefill of x1 || x2 from zero equals prefill of x2 started from the state
    that x1 leaves (Sec. 3.2 terminal state carried on, Eq. 4-5)."""
    inp = make_inputs(2, 300, 6, 5, "f32", seed=21)
    y_all, s_all = oracle.rec_prefill(inp.x, *inp.params())
    y1, s1 = oracle.rec_prefill(inp.x[:, :123], *inp.params())
    y2, s2 = oracle.rec_prefill(inp.x[:, 123:], *inp.params(), state_in=s1)
    np.testing.assert_allclose(y2, y_all[:, 123:], rtol=1e-11, atol=1e-12)
    np.testing.assert_allclose(s2, s_all, rtol=1e-11, atol=1e-12)


def test_initial_state_routes_agree():
    """O1 (closed-form free response added to the convolution) against O2 (the
    recurrence started from the state): independent code."""
    inp = make_inputs(2, 200, 5, 4, "f32", seed=22)
    rng = np.random.default_rng(3)
    s0 = rng.normal(size=(2, 5, 4)) + 1j * rng.normal(size=(2, 5, 4))
    y_rec, _ = oracle.rec_prefill(inp.x, *inp.params(), state_in=s0)
    y_conv = oracle.conv_prefill(inp.x, *inp.params(), state_in=s0)
    np.testing.assert_allclose(y_conv, y_rec, rtol=1e-10, atol=1e-10)


def test_free_response_hand_derived():
    """Zero drive from s = 1: one mode with half-life 10 tokens (gamma = ln2 / 10),
    omega = pi / 2, A = 2, phi = 0 rings as 2 * 2^(-(t+1)/10) cos(pi (t+1) / 2):
    0, -2^0.8, 0, 2^0.6 for t = 0..3, and leaves the state 2^(-0.4)."""
    g = np.array([[math.log(2.0) / 10.0]])
    w = np.array([[math.pi / 2.0]])
    a = np.array([[2.0]])
    ph = np.array([[0.0]])
    x = np.zeros((1, 4, 1))
    s0 = np.ones((1, 1, 1), complex)
    want = np.array([0.0, -2.0 ** 0.8, 0.0, 2.0 ** 0.6])
    y, st = oracle.rec_prefill(x, g, w, a, ph, state_in=s0)
    np.testing.assert_allclose(y[0, :, 0], want, rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(st[0, 0, 0], 2.0 ** -0.4, rtol=1e-12, atol=1e-12)
    yc = oracle.conv_prefill(x, g, w, a, ph, state_in=s0)
    np.testing.assert_allclose(yc[0, :, 0], want, rtol=1e-12, atol=1e-12)


def test_zero_initial_state_is_plain_prefill_and_response_is_linear():
    inp = make_inputs(1, 150, 4, 3, "f32", seed=23)
    y0, s0 = oracle.rec_prefill(inp.x, *inp.params())
    z = np.zeros((1, 4, 3), complex)
    yz, sz = oracle.rec_prefill(inp.x, *inp.params(), state_in=z)
    assert np.array_equal(y0, yz) and np.array_equal(s0, sz)
    rng = np.random.default_rng(4)
    si = rng.normal(size=(1, 4, 3)) + 1j * rng.normal(size=(1, 4, 3))
    ys, ss = oracle.rec_prefill(inp.x, *inp.params(), state_in=si)
    yf, sf = oracle.rec_prefill(np.zeros_like(inp.x), *inp.params(), state_in=si)
    np.testing.assert_allclose(ys, y0 + yf, rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(ss, s0 + sf, rtol=1e-12, atol=1e-12)


@pytest.mark.parametrize("seed", [41, 43])
def test_backward_matches_central_finite_differences(seed):
    """I5: both backward routes match central differences of l = sum(dy * y)
    (y by the direct convolution) at a tiny size, h = 1e-6 max(1, |p|)."""
    inp = make_inputs(1, 37, 2, 2, "f32", seed=seed, with_dy=True)
    x = inp.x.astype(np.float64)
    dy = inp.dy.astype(np.float64)
    params = [p.astype(np.float64) for p in inp.params()]
    names = ["decay", "freq", "amp", "phase"]
    dx_c, g_c = oracle.backward_conv(x, dy, *params)
    dx_r, g_r = oracle.backward_rec(x, dy, *params)
    # parameters
    for k, name in enumerate(names):
        fd = np.zeros_like(params[k])
        for idx in np.ndindex(*params[k].shape):
            h = 1e-6 * max(1.0, abs(params[k][idx]))
            pp = [q.copy() for q in params]
            pm = [q.copy() for q in params]
            pp[k][idx] += h
            pm[k][idx] -= h
            fd[idx] = (_loss(x, dy, pp) - _loss(x, dy, pm)) / (2 * h)
        scale = max(1.0, np.abs(fd).max())
        assert np.abs(g_c[name] - fd).max() / scale < 2e-7, name
        assert np.abs(g_r[name] - fd).max() / scale < 2e-7, name
    # input (the loss is linear in x, so central differences are exact up to rounding)
    fdx = np.zeros_like(x)
    for idx in [(0, 0, 0), (0, 5, 1), (0, 36, 0), (0, 20, 1)]:
        xp, xm = x.copy(), x.copy()
        xp[idx] += 1e-3
        xm[idx] -= 1e-3
        fdx[idx] = (_loss(xp, dy, params) - _loss(xm, dy, params)) / 2e-3
        assert abs(dx_c[idx] - fdx[idx]) < 1e-8
        assert abs(dx_r[idx] - fdx[idx]) < 1e-8


def _loss_state(x, dy, params, s_in, g):
    """l = sum(dy * y) + sum Re(conj(g) s_L) for the prefill from s_in (O2)."""
    y, sL = oracle.rec_prefill(x, *params, state_in=s_in)
    return float(np.sum(dy * y) + np.sum(np.real(np.conj(g) * sL)))


@pytest.mark.parametrize("seed", [5, 6])
def test_backward_with_state_terms_matches_central_finite_differences(seed):
    """Backward of a prefill from an initial state with a loss on its terminal
    state: both routes against central differences of that loss (in the
    parameters, in x, and in Re / Im of the initial state)."""
    inp = make_inputs(1, 29, 2, 2, "f32", seed=seed, with_dy=True)
    x, dy = inp.x.astype(np.float64), inp.dy.astype(np.float64)
    params = [p.astype(np.float64) for p in inp.params()]
    rng = np.random.default_rng(seed)
    s_in = rng.normal(size=(1, 2, 2)) + 1j * rng.normal(size=(1, 2, 2))
    g = rng.normal(size=(1, 2, 2)) + 1j * rng.normal(size=(1, 2, 2))
    outs = [oracle.backward_conv(x, dy, *params, state_in=s_in, d_state_out=g),
            oracle.backward_rec(x, dy, *params, state_in=s_in, d_state_out=g)]
    for k, name in enumerate(["decay", "freq", "amp", "phase"]):
        fd = np.zeros_like(params[k])
        for idx in np.ndindex(*params[k].shape):
            h = 1e-6 * max(1.0, abs(params[k][idx]))
            pp = [q.copy() for q in params]
            pm = [q.copy() for q in params]
            pp[k][idx] += h
            pm[k][idx] -= h
            fd[idx] = (_loss_state(x, dy, pp, s_in, g) - _loss_state(x, dy, pm, s_in, g)) / (2 * h)
        scale = max(1.0, np.abs(fd).max())
        for _, gr in outs:
            assert np.abs(gr[name] - fd).max() / scale < 2e-7, name
    for idx in [(0, 0, 0), (0, 7, 1), (0, 28, 0), (0, 28, 1)]:
        xp, xm = x.copy(), x.copy()
        xp[idx] += 1e-3
        xm[idx] -= 1e-3
        fdx = (_loss_state(xp, dy, params, s_in, g) - _loss_state(xm, dy, params, s_in, g)) / 2e-3
        for dx, _ in outs:
            assert abs(dx[idx] - fdx) < 1e-8, idx
    for idx in np.ndindex(1, 2, 2):
        for part, unit in (("re", 1.0), ("im", 1j)):
            sp, sm = s_in.copy(), s_in.copy()
            sp[idx] += 1e-4 * unit
            sm[idx] -= 1e-4 * unit
            fds = (_loss_state(x, dy, params, sp, g) - _loss_state(x, dy, params, sm, g)) / 2e-4
            for _, gr in outs:
                got = gr["state_in"][idx].real if part == "re" else gr["state_in"][idx].imag
                assert abs(got - fds) < 1e-8 * max(1.0, abs(fds)), (idx, part)


def test_backward_state_terms_routes_agree_and_vanish_when_zero():
    inp = make_inputs(2, 300, 3, 4, "f32", seed=41, with_dy=True)
    rng = np.random.default_rng(9)
    s_in = rng.normal(size=(2, 3, 4)) + 1j * rng.normal(size=(2, 3, 4))
    g = rng.normal(size=(2, 3, 4)) + 1j * rng.normal(size=(2, 3, 4))
    dxc, gc = oracle.backward_conv(inp.x, inp.dy, *inp.params(), state_in=s_in, d_state_out=g)
    dxr, gr = oracle.backward_rec(inp.x, inp.dy, *inp.params(), state_in=s_in, d_state_out=g)
    np.testing.assert_allclose(dxc, dxr, rtol=1e-9, atol=1e-9)
    for k in ("decay", "freq", "amp", "phase", "state_in"):
        np.testing.assert_allclose(gc[k], gr[k], rtol=1e-9, atol=1e-9 * np.abs(gr[k]).max())
    z = np.zeros((2, 3, 4), complex)
    dx0, g0 = oracle.backward_rec(inp.x, inp.dy, *inp.params())
    dxz, gz = oracle.backward_rec(inp.x, inp.dy, *inp.params(), state_in=z, d_state_out=z)
    assert np.array_equal(dx0, dxz)
    for k in ("decay", "freq", "amp", "phase"):
        assert np.array_equal(g0[k], gz[k])


def test_backward_routes_agree():
    inp = make_inputs(2, 211, 4, 5, "f32", seed=47, with_dy=True)
    dx_c, g_c = oracle.backward_conv(inp.x, inp.dy, *inp.params())
    dx_r, g_r = oracle.backward_rec(inp.x, inp.dy, *inp.params())
    assert np.linalg.norm(dx_c - dx_r) / np.linalg.norm(dx_c) < 1e-11
    for k in g_c:
        assert np.linalg.norm(g_c[k] - g_r[k]) / np.linalg.norm(g_c[k]) < 1e-10, k


def test_backward_dx_is_time_reversed_forward():
    """dx = reverse(conv(K, reverse(dy))): the adjoint of a causal convolution is
    the anti-causal one."""
    inp = make_inputs(2, 120, 3, 3, "f32", seed=53, with_dy=True)
    dx, _ = oracle.backward_rec(inp.x, inp.dy, *inp.params())
    want = oracle.conv_prefill(inp.dy[:, ::-1], *inp.params())[:, ::-1]
    np.testing.assert_allclose(dx, want, rtol=1e-11, atol=1e-11)


def test_oracle_threads_reported():
    assert oracle.num_threads() >= 1


# ------------------------------------------------------------------ mixer (Sec. 3.4)
def _mixer_case(B=2, L=37, D=5, M=3, K=4, seed=3):
    from synth import make_mixer_inputs
    inp = make_inputs(B, L, D, M, "f32", seed=seed)
    return inp, make_mixer_inputs(inp, K, seed=seed)


@pytest.mark.parametrize("K", [1, 2, 4, 7])
def test_local_conv_is_an_fir_filter(K):
    """The local path against scipy's direct-form FIR filter, run per channel over
    the drive history followed by the sequence (zero initial conditions)."""
    inp, mx = _mixer_case(K=K)
    l, tail = oracle.local_conv(inp.x, mx.conv_w, mx.conv_in)
    ext = np.concatenate([mx.conv_in.astype(np.float64), inp.x.astype(np.float64)], axis=1)
    for b in range(inp.B):
        for d in range(inp.D):
            want = scipy.signal.lfilter(mx.conv_w[d].astype(np.float64), [1.0], ext[b, :, d])
            np.testing.assert_allclose(l[b, :, d], want[K - 1:], rtol=1e-13, atol=1e-13)
    np.testing.assert_array_equal(tail, ext[:, ext.shape[1] - (K - 1):, :])


def test_local_conv_unit_lag_is_a_causal_shift():
    """w = e_k gives l_t = u_{t-k}: the lag runs into the past (a mistaken
    anti-causal or reversed kernel fails), and the history supplies t < k."""
    inp, mx = _mixer_case(K=4)
    for k in range(4):
        w = np.zeros((inp.D, 4))
        w[:, k] = 1.0
        l, _ = oracle.local_conv(inp.x, w, mx.conv_in)
        np.testing.assert_array_equal(l[:, k:], inp.x[:, :inp.L - k].astype(np.float64))
        for t in range(k):
            np.testing.assert_array_equal(l[:, t], mx.conv_in[:, 3 - k + t].astype(np.float64))


def test_mixer_reduces_to_its_parts():
    """sigma is scipy's expit; with zero amplitudes (y = 0) z is s * FIR(x); with a
    zero local kernel z is expit(g) * y; with no gate z is y + s * l."""
    import scipy.special
    inp, mx = _mixer_case()
    np.testing.assert_allclose(oracle.sigmoid(mx.g), scipy.special.expit(mx.g.astype(np.float64)),
                               rtol=1e-15)
    assert oracle.sigmoid(0.0) == 0.5
    zero_amp = np.zeros_like(inp.amp)
    z, _, _ = oracle.mixer_prefill(inp.x, mx.g, inp.decay, inp.freq, zero_amp, inp.phase,
                                   mx.conv_w, mx.scale, conv_in=mx.conv_in)
    ext = np.concatenate([mx.conv_in, inp.x], axis=1).astype(np.float64)
    fir = scipy.signal.lfilter(mx.conv_w.astype(np.float64)[0], [1.0], ext[0, :, 0])[mx.K - 1:]
    np.testing.assert_allclose(z[0, :, 0], mx.scale[0] * fir, rtol=1e-13, atol=1e-13)
    z, _, _ = oracle.mixer_prefill(inp.x, mx.g, *inp.params(), np.zeros_like(mx.conv_w), mx.scale)
    y, _ = oracle.conv_prefill(inp.x, *inp.params()), None
    np.testing.assert_allclose(z, scipy.special.expit(mx.g.astype(np.float64)) * y, rtol=1e-10,
                               atol=1e-12)
    z, _, _ = oracle.mixer_prefill(inp.x, None, *inp.params(), mx.conv_w, mx.scale)
    l, _ = oracle.local_conv(inp.x, mx.conv_w)
    np.testing.assert_allclose(z, y + mx.scale[None, None, :] * l, rtol=1e-10, atol=1e-12)


def test_mixer_split_prefill_and_decode_continue_the_sequence():
    """Prefill of x1, then prefill of x2 from (state, drive history), then decode
    steps, reproduce one prefill of the whole sequence: z, state and history."""
    inp, mx = _mixer_case(L=40, K=3)
    args = (*inp.params(), mx.conv_w, mx.scale)
    z, st, tail = oracle.mixer_prefill(inp.x, mx.g, *args, conv_in=mx.conv_in)
    z1, st1, t1 = oracle.mixer_prefill(inp.x[:, :17], mx.g[:, :17], *args, conv_in=mx.conv_in)
    z2, st2, t2 = oracle.mixer_prefill(inp.x[:, 17:35], mx.g[:, 17:35], *args, state_in=st1,
                                       conv_in=t1)
    np.testing.assert_allclose(np.concatenate([z1, z2], 1), z[:, :35], rtol=1e-10, atol=1e-12)
    s, c = st2, t2
    for t in range(35, 40):
        zt, s, c = oracle.mixer_decode(s, c, inp.x[:, t], mx.g[:, t], *args)
        np.testing.assert_allclose(zt, z[:, t], rtol=1e-10, atol=1e-12)
    np.testing.assert_allclose(s, st, rtol=1e-10, atol=1e-12)
    np.testing.assert_array_equal(c, tail)


def test_coupling_hand_derived_two_heads():
    """H = 2, dh = 1: C = [[1, l/sqrt2 tanh a], [l/sqrt2 tanh b, 1]] applied to one
    token (a transposed C or a dropped identity fails)."""
    a, b_, lam = 0.7, -1.3, 0.5
    C = oracle.coupling_matrix([[0.0, a], [b_, 0.0]], lam)
    k = lam / math.sqrt(2.0)
    np.testing.assert_allclose(C, [[1.0, k * math.tanh(a)], [k * math.tanh(b_), 1.0]], rtol=1e-15)
    y = np.array([[[2.0, -3.0]]])
    yb = oracle.couple_heads(y, C)
    np.testing.assert_allclose(yb[0, 0], [2.0 + k * math.tanh(a) * -3.0, k * math.tanh(b_) * 2.0 - 3.0], rtol=1e-15)


def test_coupling_is_a_head_major_einsum_and_identity_when_off():
    rng = np.random.default_rng(5)
    H, dh = 4, 3
    y = rng.standard_normal((2, 7, H * dh))
    c_raw = rng.standard_normal((H, H))
    C = oracle.coupling_matrix(c_raw, 0.8)
    want = np.einsum("gh,blhi->blgi", C, y.reshape(2, 7, H, dh)).reshape(2, 7, H * dh)
    np.testing.assert_allclose(oracle.couple_heads(y, C), want, rtol=1e-13, atol=1e-14)
    # a field living in head 1 only spreads to head g with weight C[g, 1]
    y1 = np.zeros_like(y)
    y1[..., dh:2 * dh] = y[..., dh:2 * dh]
    out = oracle.couple_heads(y1, C)
    for g in range(H):
        np.testing.assert_allclose(out[..., g * dh:(g + 1) * dh], C[g, 1] * y[..., dh:2 * dh], rtol=1e-13)
    np.testing.assert_array_equal(oracle.couple_heads(y, oracle.coupling_matrix(c_raw, 0.0)), y)
    np.testing.assert_array_equal(oracle.couple_heads(y, oracle.coupling_matrix(np.zeros((H, H)), 0.9)), y)


def test_coupled_mixer_decode_continues_the_prefill():
    inp, mx = _mixer_case(B=2, L=30, D=6, M=2, K=3)
    cp = (np.random.default_rng(1).standard_normal((3, 3)), 0.6)
    args = (*inp.params(), mx.conv_w, mx.scale)
    z, st, tail = oracle.mixer_prefill(inp.x, mx.g, *args, conv_in=mx.conv_in, coupling=cp)
    z1, s, c = oracle.mixer_prefill(inp.x[:, :25], mx.g[:, :25], *args, conv_in=mx.conv_in, coupling=cp)
    np.testing.assert_allclose(z1, z[:, :25], rtol=1e-12, atol=1e-12)
    for t in range(25, 30):
        zt, s, c = oracle.mixer_decode(s, c, inp.x[:, t], mx.g[:, t], *args, coupling=cp)
        np.testing.assert_allclose(zt, z[:, t], rtol=1e-10, atol=1e-12)
