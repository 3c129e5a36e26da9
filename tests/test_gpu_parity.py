"""GPU parity: the CUDA path through the C ABI against the fp64 CPU oracle on the
same seeded inputs, element by element, at sizes the oracle finishes in seconds
(several chunks/tiles plus ragged tails) and at the full workload sizes on
sampled channels (channels and batch rows are independent, so a sampled
channel's oracle result is exact)."""
import numpy as np
import pytest

import oracle
from synth import make_inputs
from tests._util import TOL, assert_close, rel_errors, to_dev, to_np

torch = pytest.importorskip("torch")
rlm = pytest.importorskip("paper_2607_05583_gb300")

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    from paper_2607_05583_gb300 import build
    build.build()
    rlm.load_library()
    yield
    torch.cuda.synchronize()
    assert rlm.rlm_get_device_status() == rlm.RLM_OK


def _prefill(inp, with_state=True):
    x = to_dev(inp.x, inp.dtype)
    p = rlm.Params.from_arrays(*inp.params())
    y = torch.empty_like(x)
    st = rlm.State.empty(inp.B, inp.D, inp.M) if with_state else None
    rlm.rlm_mix_prefill(x, p, y, st)
    torch.cuda.synchronize()
    return y, st


def _sub(inp, chans):
    """Oracle inputs restricted to the sampled channels."""
    return (inp.x[:, :, chans], inp.decay[chans], inp.freq[chans], inp.amp[chans],
            inp.phase[chans])


def _state_err(st, ref, tol, what="state"):
    s = st.complex().cpu().numpy()
    assert_close(s.real, ref.real, tol, what + " re")
    assert_close(s.imag, ref.imag, tol, what + " im")


# --------------------------------------------------------------------- prefill
def test_prefill_tiny_fp32_against_direct_convolution():
    """fp32 single mixing op: B=1, L=256, D=64, M=4 against the O(L^2) oracle."""
    inp = make_inputs(1, 256, 64, 4, "f32", seed=0)
    y, st = _prefill(inp)
    ref = oracle.conv_prefill(inp.x, *inp.params())
    assert_close(to_np(y), ref, TOL["f32"], "y")
    _, st_ref = oracle.rec_prefill(inp.x, *inp.params())
    _state_err(st, st_ref, TOL["f32"])


def test_prefill_layer6m_bf16():
    """6M-scale layer: B=8, L=2048, D=256, M=16, bf16 I/O, plus the final state."""
    inp = make_inputs(8, 2048, 256, 16, "bf16", seed=0)
    y, st = _prefill(inp)
    ref, st_ref = oracle.rec_prefill(inp.x, *inp.params())
    assert_close(to_np(y), ref, TOL["bf16"], "y")
    _state_err(st, st_ref, TOL["bf16"])
    chans = np.array([0, 37, 128, 255])
    ref1 = oracle.conv_prefill(*_sub(inp, chans))
    assert_close(to_np(y)[:, :, chans], ref1, TOL["bf16"], "y vs direct convolution")


@pytest.mark.parametrize("B,L,D,M,with_state_in,bitwise", [
    (8, 2048, 256, 16, False, True),          # the 6M layer: two rows per CTA, one wave
    (9, 704, 256, 7, True, True),             # three rows per CTA, padded modes, an initial state
    (3, 2048 * 2 + 64, 2048, 16, True, True), # more channel groups than SMs: three rows per CTA, ragged tile
    (3, 2048 * 2 + 77, 2048, 16, True, False), # L not a multiple of 64 with a state: the SIMT scan
    (5, 2048 + 3, 512, 32, False, False),     # 32 modes in one launch, rows in CTAs of three (a partial last one)
    (6, 2048 * 2 + 64, 1024, 24, True, True), # 32-mode instance: modes 24-31 padded, an initial state
    (9, 704, 512, 32, False, True),           # 32-mode instance, one tile per row
])
def test_packed_rows_prefill(B, L, D, M, with_state_in, bitwise):
    """Where the (batch row, channel group) CTAs would take more than one wave, a
    CTA runs several rows' tiles back to back (one prologue).  Against the oracle,
    and bit for bit against prefilling each row alone where that call is
    unsegmented too (y and the terminal state)."""
    inp = make_inputs(B, L, D, M, "bf16", seed=B * 100 + L)
    rng = np.random.default_rng(L)
    s_in = (rng.standard_normal((B, D, M)) + 1j * rng.standard_normal((B, D, M))) if with_state_in else None
    x = to_dev(inp.x, "bf16")
    p = rlm.Params.from_arrays(*inp.params())
    y, st = torch.empty_like(x), rlm.State.empty(B, D, M)
    si = None
    if with_state_in:
        si = rlm.State.empty(B, D, M)
        si.s.copy_(torch.from_numpy(np.stack([s_in.real, s_in.imag], -1).astype(np.float32)))
    rlm.rlm_mix_prefill_from(x, p, si, y, st)
    torch.cuda.synchronize()
    ref, st_ref = oracle.rec_prefill(inp.x, *inp.params(), state_in=s_in)
    assert_close(to_np(y), ref, TOL["bf16"], "y")
    _state_err(st, st_ref, TOL["bf16"])
    if bitwise:
        for b in range(B):
            yb, stb = torch.empty_like(x[b:b + 1]), rlm.State.empty(1, D, M)
            sib = None
            if with_state_in:
                sib = rlm.State.empty(1, D, M)
                sib.s.copy_(si.s[b:b + 1])
            rlm.rlm_mix_prefill_from(x[b:b + 1].contiguous(), p, sib, yb, stb)
            torch.cuda.synchronize()
            assert torch.equal(yb[0], y[b]), b
            assert torch.equal(stb.s[0], st.s[b]), b


@pytest.mark.parametrize("B,L,D,M,dtype", [
    (1, 1, 8, 1, "f32"), (1, 1, 8, 16, "bf16"), (2, 7, 16, 3, "f32"), (3, 65, 24, 16, "bf16"),
    (1, 1000, 8, 64, "f32"), (2, 2049, 64, 16, "bf16"), (1, 4097, 32, 5, "bf16"),
    (2, 3000, 40, 33, "f32"), (1, 6143, 256, 16, "bf16"), (3, 2048 * 3 + 17, 64, 16, "bf16"),
    # few rows: the sequence is split into segments (one per tile; two tiles each
    # with a shorter last segment)
    (1, 2048 * 5 + 100, 8, 16, "bf16"), (1, 2048 * 24 + 5, 64, 16, "bf16"),
    # bf16 with M < 16: the tcgen05 prefill with the modes padded to 16 (one token,
    # D not a multiple of 64, the paper's single mode per channel, segmented and not)
    (1, 1, 8, 3, "bf16"), (2, 2048 * 2 + 7, 24, 8, "bf16"), (1, 2048 * 3, 64, 1, "bf16"),
    (4, 2048 + 5, 256, 1, "bf16"), (1, 3000, 8, 15, "bf16"),
    # bf16 with 16 < M <= 32: the time-reversed tcgen05 scan -- one token, a tail
    # shorter than a chunk, one token past a tile, D not a multiple of 64
    (1, 1, 8, 17, "bf16"), (2, 65, 16, 32, "bf16"), (1, 2100, 8, 31, "bf16"),
    (2, 2048 * 2 + 7, 24, 20, "bf16"),
    # bf16 with 16 < M <= 32 on unsegmented shapes: the 32-mode tcgen05 instance
    # (several tiles and a ragged first tile; 17 modes; a packed launch)
    (4, 2048 * 2 + 100, 160, 20, "bf16"), (1, 2048 + 1, 1024, 17, "bf16"),
    (2, 3 * 2048 + 17, 640, 32, "bf16"),
    # bf16 with M > 32: the SIMT path
    (1, 500, 8, 40, "bf16"),
])
def test_prefill_edge_and_ragged_shapes(B, L, D, M, dtype):
    inp = make_inputs(B, L, D, M, dtype, seed=B * 1000 + L)
    y, st = _prefill(inp)
    ref, st_ref = oracle.rec_prefill(inp.x, *inp.params())
    assert_close(to_np(y), ref, TOL[dtype], "y")
    _state_err(st, st_ref, TOL[dtype])


@pytest.mark.parametrize("B,L", [(1, 8192), (1, 16384), (1, 32768), (4, 8192), (4, 16384),
                                 (4, 32768)])
def test_prefill_long_context_sweep(B, L):
    """Long-context sweep at the benchmark's launch configuration (D=256, M=16, bf16),
    every channel of y and of the terminal state against the sequential recurrence
    (O2) run in full: B * L * 256 * 16 complex updates, a few seconds on the host."""
    inp = make_inputs(B, L, 256, 16, "bf16", seed=0)
    y, st = _prefill(inp)
    ref, st_ref = oracle.rec_prefill(inp.x, *inp.params())
    assert_close(to_np(y), ref, TOL["bf16"], "y")
    _state_err(st, st_ref, TOL["bf16"])
    # Per channel too: a fault confined to one 8-channel CTA group must not hide
    # in the whole-tensor norms.
    yg = to_np(y)
    for d0 in range(0, 256, 8):
        assert_close(yg[:, :, d0:d0 + 8], ref[:, :, d0:d0 + 8], TOL["bf16"], f"y channels {d0}..{d0 + 7}")


def test_prefill_training_shape_m32():
    """Forward of the training workload (B=4, L=32768, D=512, M=32, bf16): every
    channel of y and of the terminal state against O2 run in full, and the mode
    coefficients of every channel."""
    inp = make_inputs(4, 32768, 512, 32, "bf16", seed=0)
    y, st = _prefill(inp)
    ref, st_ref = oracle.rec_prefill(inp.x, *inp.params())
    assert_close(to_np(y), ref, TOL["bf16"], "y")
    _state_err(st, st_ref, TOL["bf16"])
    chans = np.arange(512)
    coef = st.coef.cpu().numpy()[chans]
    lam = np.exp(-inp.decay[chans].astype(np.float64) + 1j * inp.freq[chans].astype(np.float64))
    np.testing.assert_allclose(coef[..., 0], lam.real, rtol=0, atol=1e-6)
    np.testing.assert_allclose(coef[..., 1], lam.imag, rtol=0, atol=1e-6)


def test_time_reversed_prefill_is_causal_bit_exact():
    """The bf16 prefill with 16 < M <= 32 runs as a reverse-time scan of the reversed
    drive; perturbing x[t >= t0] must still leave y[t < t0] bit-identical."""
    inp = make_inputs(2, 5000, 64, 24, "bf16", seed=6)
    y1, _ = _prefill(inp, False)
    inp2 = make_inputs(2, 5000, 64, 24, "bf16", seed=6)
    inp2.x = inp.x.copy()
    inp2.x[:, 2999:] = -inp2.x[:, 2999:] + 1.0
    y2, _ = _prefill(inp2, False)
    a, b = y1.cpu(), y2.cpu()
    assert torch.equal(a[:, :2999], b[:, :2999])
    assert not torch.equal(a[:, 2999:], b[:, 2999:])


def _state_from(inp, s_np):
    st = rlm.State.empty(inp.B, inp.D, inp.M)
    st.s.copy_(torch.from_numpy(np.stack([s_np.real, s_np.imag], -1).astype(np.float32)))
    return st


@pytest.mark.parametrize("B,L,D,M,dtype", [
    (2, 2048 * 2, 64, 16, "bf16"),        # tcgen05 prefill, token 0 at a tile start
    (8, 5056, 256, 16, "bf16"),           # ... token 0 inside the first tile (at a chunk start)
    (1, 3008, 16, 16, "bf16"),            # ... segmented sequence
    (3, 2048 + 64, 128, 16, "bf16"),      # ... segmented, several rows
    (8, 5000, 256, 16, "bf16"),           # L not a multiple of 64: the SIMT scan
    (3, 2048 + 77, 128, 16, "bf16"),      # ... the same for a segmented shape
    (2, 1000, 8, 32, "bf16"),             # time-reversed scan, L not a chunk multiple
    (1, 4096, 16, 20, "bf16"),            # time-reversed scan, L a chunk multiple
    (1, 4096, 16, 7, "bf16"),             # tcgen05 prefill, 7 modes padded to 16 (segmented)
    (4, 3001, 256, 1, "bf16"),            # ... one mode per channel, unsegmented
    (2, 1000, 16, 7, "f32"),              # SIMT (L not a multiple of 64)
    (2, 4096, 16, 7, "f32"),              # fp32 tcgen05 prefill, 7 modes padded to 16
    (3, 2048 + 64 * 5, 64, 16, "f32"),    # ... token 0 inside the first tile
    (9, 704, 256, 16, "f32"),             # ... several rows per CTA, each from its own state
    (1, 500, 8, 40, "bf16"),              # SIMT, bf16 with M > 32
    (2, 4096, 640, 32, "bf16"),           # 32-mode tcgen05 instance, two rows per CTA
    (1, 2048 * 2 + 64 * 3, 1024, 24, "bf16"),  # ... one row per CTA, token 0 inside the first tile
])
def test_prefill_from_initial_state_matches_oracle(B, L, D, M, dtype):
    """Prefill started from a state (chunked / continued prefill) against the
    oracle's recurrence from the same state; the state is one a 300-token
    prompt leaves, so its size is that of real use."""
    inp = make_inputs(B, L, D, M, dtype, seed=L + 7 * M)
    pre = make_inputs(B, 300, D, M, dtype, seed=1 + M)
    _, s_in = oracle.rec_prefill(pre.x, *inp.params())
    x = to_dev(inp.x, dtype)
    p = rlm.Params.from_arrays(*inp.params())
    y = torch.empty_like(x)
    si = _state_from(inp, s_in)
    so = rlm.State.empty(B, D, M)
    rlm.rlm_mix_prefill_from(x, p, si, y, so)
    torch.cuda.synchronize()
    ref, st_ref = oracle.rec_prefill(inp.x, *inp.params(), state_in=s_in)
    assert_close(to_np(y), ref, TOL[dtype], "y")
    _state_err(so, st_ref, TOL[dtype])


@pytest.mark.parametrize("B,L,D,M", [(2, 1000, 8, 32), (1, 4001, 16, 24)])
def test_prefill_from_state_with_fast_decays_on_ragged_lengths(B, L, D, M):
    """Decays of 1.5-3 per token (half-lives under half a token) with an initial
    state on shapes whose zero-state prefill takes the time-reversed tcgen05 path
    and L not a multiple of 64: the state must enter without a negative power of
    lambda, so y and the terminal state stay finite and match the oracle."""
    inp = make_inputs(B, L, D, M, "bf16", seed=L + M)
    rng = np.random.default_rng(L)
    decay = inp.decay.copy()
    fast = rng.random(decay.shape) < 0.5
    decay[fast] = rng.uniform(1.5, 3.0, size=int(fast.sum())).astype(np.float32)
    params = (decay, inp.freq, inp.amp, inp.phase)
    pre = make_inputs(B, 300, D, M, "bf16", seed=2 + M)
    _, s_in = oracle.rec_prefill(pre.x, *params)
    x = to_dev(inp.x, "bf16")
    p = rlm.Params.from_arrays(*params)
    y = torch.empty_like(x)
    si = _state_from(inp, s_in)
    so = rlm.State.empty(B, D, M)
    rlm.rlm_mix_prefill_from(x, p, si, y, so)
    torch.cuda.synchronize()
    assert torch.isfinite(y.float()).all() and torch.isfinite(so.s).all()
    ref, st_ref = oracle.rec_prefill(inp.x, *params, state_in=s_in)
    assert_close(to_np(y), ref, TOL["bf16"], "y")
    _state_err(so, st_ref, TOL["bf16"])


@pytest.mark.parametrize("M", [16, 32])
def test_split_prefill_with_in_place_state_equals_whole_prefill(M):
    """Prefill of x1 then prefill_from(x2) with state_out = state_in (in place)
    equals one prefill of x1 || x2 (bf16, ragged split)."""
    inp = make_inputs(2, 6000, 64, M, "bf16", seed=31)
    x = to_dev(inp.x, "bf16")
    p = rlm.Params.from_arrays(*inp.params())
    y_all = torch.empty_like(x)
    st_all = rlm.State.empty(2, 64, M)
    rlm.rlm_mix_prefill(x, p, y_all, st_all)
    x1, x2 = x[:, :2345].contiguous(), x[:, 2345:].contiguous()
    y1, y2 = torch.empty_like(x1), torch.empty_like(x2)
    st = rlm.State.empty(2, 64, M)
    rlm.rlm_mix_prefill(x1, p, y1, st)
    rlm.rlm_mix_prefill_from(x2, p, st, y2, st)
    torch.cuda.synchronize()
    ref, st_ref = oracle.rec_prefill(inp.x, *inp.params())
    assert_close(to_np(y2), ref[:, 2345:], TOL["bf16"], "y of the continuation")
    assert_close(to_np(torch.cat([y1, y2], 1)), to_np(y_all), TOL["bf16"], "split vs whole")
    _state_err(st, st_ref, TOL["bf16"])


@pytest.mark.parametrize("L", [3008, 3000])
def test_prefill_from_zero_state_equals_prefill(L):
    """A zero initial state gives the zero-state prefill bit for bit where both take
    the same path (L a multiple of 64); with L = 3000 the call with a state runs on
    the SIMT scan and agrees within the tolerance."""
    inp = make_inputs(2, L, 64, 16, "bf16", seed=33)
    x = to_dev(inp.x, "bf16")
    p = rlm.Params.from_arrays(*inp.params())
    y0, y1 = torch.empty_like(x), torch.empty_like(x)
    rlm.rlm_mix_prefill(x, p, y0)
    z = rlm.State.empty(2, 64, 16)
    z.s.zero_()
    rlm.rlm_mix_prefill_from(x, p, z, y1)
    y2 = torch.empty_like(x)
    rlm.rlm_mix_prefill_from(x, p, None, y2)
    torch.cuda.synchronize()
    assert torch.equal(y0, y2)
    if L % 64 == 0:
        assert torch.equal(y0, y1)
    else:
        assert_close(to_np(y1), to_np(y0), TOL["bf16"], "zero state on the SIMT scan")


def test_prefill_is_causal_bit_exact():
    """I6: perturbing x[t >= t0] leaves y[t < t0] bit-identical on the GPU."""
    for dtype in ("bf16", "f32"):
        inp = make_inputs(2, 5000, 64, 16, dtype, seed=5)
        y1, _ = _prefill(inp, False)
        x2 = inp.x.copy()
        x2[:, 3001:] = -x2[:, 3001:] + 1.0
        inp2 = make_inputs(2, 5000, 64, 16, dtype, seed=5)
        inp2.x = x2
        y2, _ = _prefill(inp2, False)
        a, b = y1.cpu(), y2.cpu()
        assert torch.equal(a[:, :3001], b[:, :3001])
        assert not torch.equal(a[:, 3001:], b[:, 3001:])


def test_prefill_is_deterministic():
    inp = make_inputs(2, 4100, 128, 16, "bf16", seed=9)
    y1, s1 = _prefill(inp)
    y2, s2 = _prefill(inp)
    assert torch.equal(y1, y2) and torch.equal(s1.s, s2.s) and torch.equal(s1.coef, s2.coef)


def test_segmented_prefill_reuses_one_workspace():
    """Few batch rows split the sequence into segments that publish their end
    states in the workspace (epoch-tagged flags, never cleared): consecutive calls
    with different inputs and one workspace must each match the oracle."""
    B, L, D, M = 1, 2048 * 6 + 300, 64, 16
    assert rlm.rlm_prefill_workspace_size(B, L, D, M, torch.bfloat16) > 0
    work = torch.empty(rlm.rlm_prefill_workspace_size(B, L, D, M, torch.bfloat16),
                       dtype=torch.uint8, device="cuda")
    for seed in (31, 32, 33):
        inp = make_inputs(B, L, D, M, "bf16", seed=seed)
        x = to_dev(inp.x, "bf16")
        p = rlm.Params.from_arrays(*inp.params())
        y = torch.empty_like(x)
        st = rlm.State.empty(B, D, M)
        rlm.rlm_mix_prefill(x, p, y, st, workspace=work)
        torch.cuda.synchronize()
        ref, st_ref = oracle.rec_prefill(inp.x, *inp.params())
        assert_close(to_np(y), ref, TOL["bf16"], f"y (seed {seed})")
        _state_err(st, st_ref, TOL["bf16"])


def test_prefill_does_not_write_outside_y():
    inp = make_inputs(2, 777, 64, 16, "bf16", seed=13)
    x = to_dev(inp.x, "bf16")
    p = rlm.Params.from_arrays(*inp.params())
    n = x.numel()
    guard = 4096
    buf = torch.full((n + 2 * guard,), 7.0, dtype=torch.bfloat16, device="cuda")
    y = buf[guard:guard + n].view_as(x)
    rlm.rlm_mix_prefill(x, p, y)
    torch.cuda.synchronize()
    assert torch.all(buf[:guard] == 7.0) and torch.all(buf[guard + n:] == 7.0)
    ref, _ = oracle.rec_prefill(inp.x, *inp.params())
    assert_close(to_np(y), ref, TOL["bf16"], "y")


def test_linearity_on_gpu():
    """I9 on the GPU (fp32 I/O): y(2 x1 - 3 x2) = 2 y(x1) - 3 y(x2) to fp32 rounding."""
    a = make_inputs(1, 3000, 32, 8, "f32", seed=21)
    b = make_inputs(1, 3000, 32, 8, "f32", seed=22)
    b.decay, b.freq, b.amp, b.phase = a.decay, a.freq, a.amp, a.phase
    c = make_inputs(1, 3000, 32, 8, "f32", seed=21)
    c.x = (2 * a.x - 3 * b.x).astype(np.float32)
    ya, yb, yc = (to_np(_prefill(i, False)[0]) for i in (a, b, c))
    assert_close(yc, 2 * ya - 3 * yb, 1e-5, "linearity")


# ---------------------------------------------------------------------- decode
@pytest.mark.parametrize("dtype,M", [("bf16", 16), ("f32", 16), ("f32", 5), ("bf16", 64),
                                     ("f32", 1)])
def test_decode_steps_match_oracle(dtype, M):
    B, L, D, T = 3, 500, 24, 40
    inp = make_inputs(B, L, D, M, dtype, seed=M, decode_steps=T)
    _, st = _prefill(inp)
    ys = []
    for t in range(T):
        xt = to_dev(inp.tokens[t], dtype)
        yt = torch.empty_like(xt)
        rlm.rlm_mix_decode(xt, st, yt)
        ys.append(to_np(yt))
    xcat = np.concatenate([inp.x, inp.tokens.transpose(1, 0, 2)], axis=1)
    ref, st_ref = oracle.rec_prefill(xcat, *inp.params())
    assert_close(np.stack(ys, 1), ref[:, L:], TOL[dtype], "y_t")
    _state_err(st, st_ref, TOL[dtype])


def test_prefill_plus_one_decode_equals_longer_prefill_on_gpu():
    """I3 with both sides on the GPU."""
    for dtype in ("f32", "bf16"):
        inp = make_inputs(2, 4097, 64, 16, dtype, seed=3)
        y_full, st_full = _prefill(inp)
        short = make_inputs(2, 4097, 64, 16, dtype, seed=3)
        short.x = inp.x[:, :4096].copy()
        short.L = 4096
        _, st = _prefill(short)
        xt = to_dev(inp.x[:, 4096], dtype)
        yt = torch.empty_like(xt)
        rlm.rlm_mix_decode(xt, st, yt)
        torch.cuda.synchronize()
        assert_close(to_np(yt), to_np(y_full[:, 4096]), TOL[dtype], "y_L")
        _state_err(st, st_full.complex().cpu().numpy(), TOL[dtype])


@pytest.mark.parametrize("B", [1, 8, 64])
def test_decode_after_32k_prefill(B):
    """Decode workload: state from a 32768-token prefill (D=256, M=16), then 4096
    single-token steps, checked against a prefill of the concatenated sequence
    (oracle on sampled channels)."""
    L, D, M, T = 32768, 256, 16, 4096
    inp = make_inputs(B, L, D, M, "bf16", seed=0, decode_steps=T)
    _, st = _prefill(inp)
    toks = to_dev(inp.tokens, "bf16")                  # [T][B][D]
    out = torch.empty_like(toks)
    for t in range(T):
        rlm.rlm_mix_decode(toks[t], st, out[t])
    torch.cuda.synchronize()
    chans = np.array([3, 130, 254])
    xcat = np.concatenate([inp.x[:, :, chans], inp.tokens[:, :, chans].transpose(1, 0, 2)], 1)
    ref, st_ref = oracle.rec_prefill(xcat, inp.decay[chans], inp.freq[chans], inp.amp[chans],
                                     inp.phase[chans])
    got = to_np(out)[:, :, chans].transpose(1, 0, 2)
    assert_close(got, ref[:, L:], TOL["bf16"], "decode y_t")
    s = st.complex().cpu().numpy()[:, chans]
    assert_close(s.real, st_ref.real, TOL["bf16"], "state re")


@pytest.mark.parametrize("B,D", [(8, 1024), (8, 8192), (64, 4096)])
def test_decode_grids_of_one_and_several_waves(B, D):
    """The row-tiled step on a grid that fits on the GPU at once (8 x 1024: 256
    blocks) and on grids of several waves (8 x 8192: 2048 blocks of 8 rows;
    64 x 4096: 4096 blocks of 16 rows), which release the next step at different
    points: chained steps after a short prefill against the oracle on sampled
    channels, the first and last included."""
    L, M, T = 5, 16, 6
    inp = make_inputs(B, L, D, M, "bf16", seed=D + B, decode_steps=T)
    _, st = _prefill(inp)
    toks = to_dev(inp.tokens, "bf16")                  # [T][B][D]
    out = torch.empty_like(toks)
    for t in range(T):
        rlm.rlm_mix_decode(toks[t], st, out[t])
    torch.cuda.synchronize()
    chans = np.unique(np.r_[np.random.default_rng(B).choice(D, 61, replace=False), 0, D // 2, D - 1])
    xcat = np.concatenate([inp.x[:, :, chans], inp.tokens[:, :, chans].transpose(1, 0, 2)], 1)
    ref, st_ref = oracle.rec_prefill(xcat, inp.decay[chans], inp.freq[chans], inp.amp[chans],
                                     inp.phase[chans])
    got = to_np(out)[:, :, chans].transpose(1, 0, 2)
    assert_close(got, ref[:, L:], TOL["bf16"], "decode y_t")
    s = st.complex().cpu().numpy()[:, chans]
    assert_close(s.real, st_ref.real, TOL["bf16"], "state re")
    assert_close(s.imag, st_ref.imag, TOL["bf16"], "state im")


def test_state_init_then_decode_equals_prefill():
    inp = make_inputs(2, 50, 16, 16, "f32", seed=4)
    p = rlm.Params.from_arrays(*inp.params())
    st = rlm.State.empty(2, 16, 16)
    rlm.rlm_state_init(st, p)
    ys = []
    for t in range(50):
        xt = to_dev(inp.x[:, t], "f32")
        yt = torch.empty_like(xt)
        rlm.rlm_mix_decode(xt, st, yt)
        ys.append(to_np(yt))
    ref = oracle.conv_prefill(inp.x, *inp.params())
    assert_close(np.stack(ys, 1), ref, TOL["f32"], "y")


def test_zero_drive_decode_energy_decay():
    """I7 on the GPU: with zero drive |s_t|^2 = exp(-2 gamma t) |s_0|^2."""
    inp = make_inputs(2, 300, 16, 8, "f32", seed=6)
    _, st = _prefill(inp)
    s0 = st.complex().cpu().numpy().copy()
    z = torch.zeros(2, 16, device="cuda")
    y = torch.empty_like(z)
    for _ in range(25):
        rlm.rlm_mix_decode(z, st, y)
    s = st.complex().cpu().numpy()
    want = np.exp(-2 * 25 * inp.decay.astype(np.float64))[None] * np.abs(s0) ** 2
    np.testing.assert_allclose(np.abs(s) ** 2, want, rtol=2e-5, atol=1e-12)


# -------------------------------------------------------------------- backward
def _backward(inp):
    x, dy = to_dev(inp.x, inp.dtype), to_dev(inp.dy, inp.dtype)
    p = rlm.Params.from_arrays(*inp.params())
    dx = torch.empty_like(x)
    g = rlm.Grads.empty(inp.D, inp.M)
    rlm.rlm_mix_backward(dy, x, p, dx, g)
    torch.cuda.synchronize()
    return dx, g


@pytest.mark.parametrize("B,L,D,M,dtype", [
    (1, 256, 64, 4, "f32"), (2, 1000, 16, 7, "f32"), (2, 3001, 64, 16, "bf16"),
    (1, 4096, 32, 32, "bf16"), (1, 1, 8, 1, "f32"),
    # tensor-core path: one token; a ragged tail shorter than a chunk with an odd
    # mode count; one token past two tiles with M = 31; a slowly decaying mode
    # whose dgamma is a near-cancelling projection of a large P (needs the
    # high + low parts of the lambda^i tables)
    (1, 1, 8, 1, "bf16"), (3, 65, 8, 5, "bf16"), (1, 2 * 2048 + 1, 16, 31, "bf16"),
    (1, 2100, 8, 32, "bf16"),
    # bf16 with M > 32 runs the SIMT path
    (1, 700, 8, 40, "bf16"),
])
def test_backward_matches_oracle(B, L, D, M, dtype):
    inp = make_inputs(B, L, D, M, dtype, seed=L + M, with_dy=True)
    dx, g = _backward(inp)
    dx_ref, g_ref = oracle.backward_rec(inp.x, inp.dy, *inp.params())
    assert_close(to_np(dx), dx_ref, TOL[dtype], "dx")
    for k in ("decay", "freq", "amp", "phase"):
        assert_close(getattr(g, k).cpu().numpy(), g_ref[k], TOL[dtype], "d" + k)


@pytest.mark.parametrize("B,L,D,M,dtype,with_s,with_g", [
    # tensor-core backward: state_in and its gradient
    (2, 3001, 16, 16, "bf16", True, False),
    (1, 2 * 2048 + 1, 8, 32, "bf16", True, False),
    (3, 65, 8, 5, "bf16", True, False),
    (2, 3001, 16, 16, "bf16", False, False),
    # ... with a terminal-state gradient (the closed-form terminal-state launch)
    (2, 3001, 16, 16, "bf16", True, True),
    (1, 700, 8, 32, "bf16", False, True),
    (3, 65, 8, 5, "bf16", True, True),
    (1, 2 * 2048, 8, 32, "bf16", True, True),
    (2, 1, 8, 16, "bf16", True, True),
    # SIMT: fp32, bf16 with M > 32
    (2, 1000, 16, 7, "f32", True, True),
    (1, 1, 8, 3, "f32", True, True),
    (1, 700, 8, 40, "bf16", True, False),
    (1, 700, 8, 40, "bf16", True, True),
])
def test_backward_with_state_terms_matches_oracle(B, L, D, M, dtype, with_s, with_g):
    """Backward of prefill_from (Sec. 3.2-3.3 with an initial state): dx, the four
    parameter gradients and the initial-state gradient, for a loss
    sum(dy * y) + Re<g, state_out>, against the oracle's adjoint recurrence."""
    inp = make_inputs(B, L, D, M, dtype, seed=L + 3 * M, with_dy=True)
    rng = np.random.default_rng(L + M)
    pre = make_inputs(B, 300, D, M, dtype, seed=2 + M)
    s_in = oracle.rec_prefill(pre.x, *inp.params())[1] if with_s else None
    g_out = ((rng.standard_normal((B, D, M)) + 1j * rng.standard_normal((B, D, M)))
             if with_g else None)
    x, dy = to_dev(inp.x, dtype), to_dev(inp.dy, dtype)
    p = rlm.Params.from_arrays(*inp.params())
    dx = torch.empty_like(x)
    g = rlm.Grads.empty(D, M)
    ds = rlm.State.empty(B, D, M)
    rlm.rlm_mix_backward_from(dy, x, p, _state_from(inp, s_in) if with_s else None,
                              _state_from(inp, g_out) if with_g else None, dx, g, ds)
    torch.cuda.synchronize()
    # a zero initial state leaves the forward unchanged and makes the oracle return
    # the initial-state gradient
    s_ref = s_in if with_s else np.zeros((B, D, M), np.complex128)
    dx_ref, g_ref = oracle.backward_rec(inp.x, inp.dy, *inp.params(), state_in=s_ref,
                                        d_state_out=g_out)
    assert_close(to_np(dx), dx_ref, TOL[dtype], "dx")
    for k in ("decay", "freq", "amp", "phase"):
        assert_close(getattr(g, k).cpu().numpy(), g_ref[k], TOL[dtype], "d" + k)
    ds_np = ds.complex().cpu().numpy()
    want = g_ref["state_in"]
    for part, got, ref in (("re", ds_np.real, want.real), ("im", ds_np.imag, want.imag)):
        assert_close(got, ref, TOL[dtype], "dstate_in " + part)


@pytest.mark.parametrize("decay_scale,L", [(1.0, 3001), (40.0, 2077)])
def test_terminal_gradient_with_silent_modes_matches_oracle(decay_scale, L):
    """A terminal-state gradient reaches modes with zero amplitude (c = 0: they add
    nothing to y, but the terminal state still depends on them), and fast decays
    with a ragged sequence end (the chunk holding token L - 1, summed directly
    on the tensor-core route)."""
    B, D, M = 2, 16, 16
    inp = make_inputs(B, L, D, M, "bf16", seed=L, with_dy=True)
    decay, freq, amp, phase = (a.copy() for a in inp.params())
    amp[:, ::3] = 0.0
    decay *= decay_scale
    rng = np.random.default_rng(L)
    g_out = rng.standard_normal((B, D, M)) + 1j * rng.standard_normal((B, D, M))
    s_in = rng.standard_normal((B, D, M)) + 1j * rng.standard_normal((B, D, M))
    x, dy = to_dev(inp.x, "bf16"), to_dev(inp.dy, "bf16")
    p = rlm.Params.from_arrays(decay, freq, amp, phase)
    dx, g, ds = torch.empty_like(x), rlm.Grads.empty(D, M), rlm.State.empty(B, D, M)
    rlm.rlm_mix_backward_from(dy, x, p, _state_from(inp, s_in), _state_from(inp, g_out), dx, g, ds)
    torch.cuda.synchronize()
    dx_ref, g_ref = oracle.backward_rec(inp.x, inp.dy, decay, freq, amp, phase, state_in=s_in,
                                        d_state_out=g_out)
    assert_close(to_np(dx), dx_ref, TOL["bf16"], "dx")
    for k in ("decay", "freq", "amp", "phase"):
        assert_close(getattr(g, k).cpu().numpy(), g_ref[k], TOL["bf16"], "d" + k)
    ds_np = ds.complex().cpu().numpy()
    assert_close(ds_np.real, g_ref["state_in"].real, TOL["bf16"], "dstate_in re")
    assert_close(ds_np.imag, g_ref["state_in"].imag, TOL["bf16"], "dstate_in im")


@pytest.mark.parametrize("L,M,with_s", [
    (63, 7, False),            # no chunk ends before L: all of it from the direct sum
    (64, 32, True),            # one chunk ending exactly at L - 1
    (2049, 32, False),         # the last tile holds only the one-token chunk
    (4095, 5, True),           # a ragged chunk inside the last tile
    (3 * 2048 + 100, 32, True),  # weights carried across tiles by lambda^2048
    (2 ** 18 + 77, 8, True),   # ... over 128 tiles
])
def test_terminal_state_terms_at_tile_edges(L, M, with_s):
    """The terminal-state terms of the tcgen05 backward (dx, the decay and frequency
    gradients through conj(g) J, the gradient of s_in) at the chunk and tile edges
    of its closed form, against the recurrence oracle."""
    B, D = 2, 8
    inp = make_inputs(B, L, D, M, "bf16", seed=L + 3 * M, with_dy=True)
    rng = np.random.default_rng(L + M)
    g_out = rng.standard_normal((B, D, M)) + 1j * rng.standard_normal((B, D, M))
    s_in = rng.standard_normal((B, D, M)) + 1j * rng.standard_normal((B, D, M)) if with_s else None
    x, dy = to_dev(inp.x, "bf16"), to_dev(inp.dy, "bf16")
    p = rlm.Params.from_arrays(*inp.params())
    dx, g, ds = torch.empty_like(x), rlm.Grads.empty(D, M), rlm.State.empty(B, D, M)
    rlm.rlm_mix_backward_from(dy, x, p, _state_from(inp, s_in) if with_s else None, _state_from(inp, g_out),
                              dx, g, ds)
    torch.cuda.synchronize()
    dx_ref, g_ref = oracle.backward_rec(inp.x, inp.dy, *inp.params(), state_in=s_in, d_state_out=g_out)
    assert_close(to_np(dx), dx_ref, TOL["bf16"], "dx")
    for k in ("decay", "freq", "amp", "phase"):
        assert_close(getattr(g, k).cpu().numpy(), g_ref[k], TOL["bf16"], "d" + k)
    ds_np = ds.complex().cpu().numpy()
    assert_close(ds_np.real, g_ref["state_in"].real, TOL["bf16"], "dstate_in re")
    assert_close(ds_np.imag, g_ref["state_in"].imag, TOL["bf16"], "dstate_in im")


def test_backward_from_without_state_terms_equals_backward():
    """No state arguments: the same kernels and bit-identical results as rlm_mix_backward."""
    inp = make_inputs(2, 3001, 64, 16, "bf16", seed=12, with_dy=True)
    dx0, g0 = _backward(inp)
    x, dy = to_dev(inp.x, "bf16"), to_dev(inp.dy, "bf16")
    p = rlm.Params.from_arrays(*inp.params())
    dx1 = torch.empty_like(x)
    g1 = rlm.Grads.empty(inp.D, inp.M)
    rlm.rlm_mix_backward_from(dy, x, p, None, None, dx1, g1)
    torch.cuda.synchronize()
    assert torch.equal(dx0, dx1)
    for k in ("decay", "freq", "amp", "phase"):
        assert torch.equal(getattr(g0, k), getattr(g1, k))


def test_split_backward_chains_state_gradients():
    """Backward through a split sequence x1 || x2: the second half's backward with
    state_in = state after x1 gives d_state_in, which fed as d_state_out into the
    first half's backward reproduces the whole sequence's gradients (bf16; the
    first half's backward takes the terminal-state gradient)."""
    B, L, D, M, cut = 2, 5000, 16, 16, 2345
    inp = make_inputs(B, L, D, M, "bf16", seed=41, with_dy=True)
    x, dy = to_dev(inp.x, "bf16"), to_dev(inp.dy, "bf16")
    p = rlm.Params.from_arrays(*inp.params())
    st = rlm.State.empty(B, D, M)
    x1, x2 = x[:, :cut].contiguous(), x[:, cut:].contiguous()
    y1 = torch.empty_like(x1)
    dy1, dy2 = dy[:, :cut].contiguous(), dy[:, cut:].contiguous()
    rlm.rlm_mix_prefill(x1, p, y1, st)
    dx2, g2, ds = torch.empty_like(x2), rlm.Grads.empty(D, M), rlm.State.empty(B, D, M)
    rlm.rlm_mix_backward_from(dy2, x2, p, st, None, dx2, g2, ds)
    dx1, g1 = torch.empty_like(x1), rlm.Grads.empty(D, M)
    rlm.rlm_mix_backward_from(dy1, x1, p, None, ds, dx1, g1)
    torch.cuda.synchronize()
    dx_ref, g_ref = oracle.backward_rec(inp.x, inp.dy, *inp.params())
    assert_close(to_np(torch.cat([dx1, dx2], 1)), dx_ref, TOL["bf16"], "dx")
    for k in ("decay", "freq", "amp", "phase"):
        got = getattr(g1, k).cpu().numpy() + getattr(g2, k).cpu().numpy()
        assert_close(got, g_ref[k], TOL["bf16"], "d" + k)


def test_backward_training_workload_sampled():
    """Training path: B=4, L=32768, D=512, M=32, bf16 I/O; dx and all four parameter
    gradients of sampled channels against the oracle."""
    inp = make_inputs(4, 32768, 512, 32, "bf16", seed=0, with_dy=True)
    dx, g = _backward(inp)
    groups = np.arange(64)
    chans = 8 * groups + (5 * groups) % 8    # one channel of every 8-channel group, at cycling offsets
    dx_ref, g_ref = oracle.backward_rec(inp.x[:, :, chans], inp.dy[:, :, chans],
                                        inp.decay[chans], inp.freq[chans], inp.amp[chans],
                                        inp.phase[chans])
    assert_close(to_np(dx)[:, :, chans], dx_ref, TOL["bf16"], "dx")
    for k in ("decay", "freq", "amp", "phase"):
        assert_close(getattr(g, k).cpu().numpy()[chans], g_ref[k], TOL["bf16"], "d" + k)


@pytest.mark.parametrize("B,L,D,M,dtype", [
    (4, 32768, 256, 16, "bf16"),     # the 16-mode tensor-core prefill (15-slot x ring)
    (4, 32768, 512, 32, "bf16"),     # the 32-mode instance (7-slot x ring, two CTA waves)
    (4, 32768, 256, 16, "f32"),      # the fp32 tensor-core prefill
    (1, 2048 * 24 + 5, 64, 16, "bf16"),  # segmented, with published segment states
])
def test_prefill_is_bit_reproducible(B, L, D, M, dtype):
    """Each call is a fixed sequence of fp32 operations, so repeated calls give
    identical bits (y and the terminal state).  Runs each shape five times: a
    pipeline hazard that lets a stage read a stale buffer shows up as a
    difference between calls."""
    inp = make_inputs(B, L, D, M, dtype, seed=21)
    x = to_dev(inp.x, dtype)
    p = rlm.Params.from_arrays(*inp.params())
    ws = torch.empty(max(256, rlm.rlm_prefill_workspace_size(B, L, D, M, x.dtype)), dtype=torch.uint8,
                     device=x.device)
    ref_y, ref_s = None, None
    for it in range(5):
        y, st = torch.empty_like(x), rlm.State.empty(B, D, M)
        rlm.rlm_mix_prefill(x, p, y, st, workspace=ws)
        torch.cuda.synchronize()
        if ref_y is None:
            ref_y, ref_s = y, st.s.clone()
        else:
            assert torch.equal(y, ref_y), it
            assert torch.equal(st.s, ref_s), it


def test_backward_is_deterministic():
    inp = make_inputs(2, 5000, 64, 16, "bf16", seed=8, with_dy=True)
    dx1, g1 = _backward(inp)
    dx2, g2 = _backward(inp)
    assert torch.equal(dx1, dx2)
    for k in ("decay", "freq", "amp", "phase"):
        assert torch.equal(getattr(g1, k), getattr(g2, k))


def test_backward_with_state_terms_is_deterministic():
    """The tcgen05 backward with state_in and d_state_out (the main pass, then the
    closed-form terminal-state launch) gives the same bits on every call."""
    B, L, D, M = 2, 5000, 64, 32
    inp = make_inputs(B, L, D, M, "bf16", seed=9, with_dy=True)
    rng = np.random.default_rng(9)
    g_out = rng.standard_normal((B, D, M)) + 1j * rng.standard_normal((B, D, M))
    s_in = rng.standard_normal((B, D, M)) + 1j * rng.standard_normal((B, D, M))
    x, dy = to_dev(inp.x, "bf16"), to_dev(inp.dy, "bf16")
    p = rlm.Params.from_arrays(*inp.params())
    outs = []
    for _ in range(3):
        dx, g, ds = torch.empty_like(x), rlm.Grads.empty(D, M), rlm.State.empty(B, D, M)
        rlm.rlm_mix_backward_from(dy, x, p, _state_from(inp, s_in), _state_from(inp, g_out), dx, g, ds)
        outs.append((dx, g, ds))
    torch.cuda.synchronize()
    for dx, g, ds in outs[1:]:
        assert torch.equal(dx, outs[0][0])
        for k in ("decay", "freq", "amp", "phase"):
            assert torch.equal(getattr(g, k), getattr(outs[0][1], k))
        assert torch.equal(ds.s, outs[0][2].s)


def test_backward_gpu_finite_differences_tiny():
    """Gradients against central differences of the GPU's own fp32 forward at a tiny
    size (loss sum(dy * y)); loose bound because the forward is fp32."""
    inp = make_inputs(1, 40, 8, 2, "f32", seed=77, with_dy=True)
    dx, g = _backward(inp)
    p0 = [q.astype(np.float64) for q in inp.params()]
    dy = inp.dy.astype(np.float64)

    def loss(ps):
        i2 = make_inputs(1, 40, 8, 2, "f32", seed=77)
        i2.decay, i2.freq, i2.amp, i2.phase = (q.astype(np.float32) for q in ps)
        y, _ = _prefill(i2, False)
        return float(np.sum(dy * to_np(y)))

    names = ["decay", "freq", "amp", "phase"]
    for k, name in enumerate(names):
        idx = (3, 1)
        h = 5e-4 if name == "decay" else 1e-3
        pp = [q.copy() for q in p0]
        pm = [q.copy() for q in p0]
        pp[k][idx] += h
        pm[k][idx] -= h
        fd = (loss(pp) - loss(pm)) / (2 * h)
        got = float(getattr(g, name).cpu().numpy()[idx])
        assert abs(got - fd) <= 2e-2 * max(1.0, abs(fd)), (name, got, fd)


def test_tied_heads_match_the_paper_kernel():
    """The paper's heads (one mode, A = 1, parameters shared by the head's channels)
    through Params.tied_heads: y against the direct convolution with
    k_h[t] = exp(-alpha_h t) cos(omega_h t + phi_h) (Sec. 3.1), per head."""
    H, d_h, B, L = 8, 32, 2, 3000
    rng = np.random.default_rng(17)
    alpha = np.exp(rng.uniform(np.log(1e-3), np.log(0.3), H)).astype(np.float32)
    omega = rng.uniform(0.0, np.pi, H).astype(np.float32)
    phi = rng.uniform(-np.pi, np.pi, H).astype(np.float32)
    inp = make_inputs(B, L, H * d_h, 1, "bf16", seed=18)
    p = rlm.Params.tied_heads(alpha, omega, phi, d_h)
    x = to_dev(inp.x, "bf16")
    y = torch.empty_like(x)
    rlm.rlm_mix_prefill(x, p, y)
    torch.cuda.synchronize()
    n = np.arange(L, dtype=np.float64)
    for h in (0, 3, 7):
        k = np.exp(-np.float64(alpha[h]) * n) * np.cos(np.float64(omega[h]) * n + np.float64(phi[h]))
        for c in (h * d_h, h * d_h + d_h - 1):
            ref = np.stack([np.convolve(inp.x[b, :, c].astype(np.float64), k)[:L] for b in range(B)])
            assert_close(to_np(y)[:, :, c], ref, TOL["bf16"], f"head {h} channel {c}")


@pytest.mark.parametrize("B,L,D,M,with_state_in", [
    (2, 3000, 512, 32, False),        # one launch of the 32-mode instance (128 CTAs: unsegmented)
    (1, 2048 + 64, 1024, 40, True),   # three passes, the last with 8 modes; from an initial state
    (2, 4160, 512, 64, True),         # four passes
    (4, 2048 * 2, 512, 17, False),    # the 32-mode instance with 15 padded modes
    (2, 2048 * 2, 512, 33, False),    # three passes, the last with one mode
])
def test_multi_pass_prefill_matches_oracle(B, L, D, M, with_state_in):
    """bf16 with M > 16 on unsegmented shapes: one launch of the 32-mode instance
    for M <= 32, else passes of 16 modes, each later pass adding to the output of
    the earlier ones; y, the terminal state and the mode coefficients of every
    mode on sampled channels against the oracle."""
    inp = make_inputs(B, L, D, M, "bf16", seed=M + L)
    s_in = None
    if with_state_in:
        pre = make_inputs(B, 200, D, M, "bf16", seed=M)
        s_in = oracle.rec_prefill(pre.x, *inp.params())[1]
    x = to_dev(inp.x, "bf16")
    p = rlm.Params.from_arrays(*inp.params())
    y = torch.empty_like(x)
    so = rlm.State.empty(B, D, M)
    n0 = rlm.rlm_kernels_launched()
    rlm.rlm_mix_prefill_from(x, p, _state_from(inp, s_in) if with_state_in else None, y, so)
    torch.cuda.synchronize()
    assert rlm.rlm_kernels_launched() - n0 == (1 if M <= 32 else (M + 15) // 16)
    ch = np.array([0, 9, D // 2 + 3, D - 1])
    ref, st_ref = oracle.rec_prefill(inp.x[:, :, ch], inp.decay[ch], inp.freq[ch], inp.amp[ch], inp.phase[ch],
                                     state_in=s_in[:, ch] if with_state_in else None)
    assert_close(to_np(y)[:, :, ch], ref, TOL["bf16"], "y")
    s = so.complex().cpu().numpy()[:, ch]
    assert_close(s.real, st_ref.real, TOL["bf16"], "state re")
    assert_close(s.imag, st_ref.imag, TOL["bf16"], "state im")
    coef = so.coef.cpu().numpy()[ch]
    lam = np.exp(-inp.decay[ch].astype(np.float64) + 1j * inp.freq[ch].astype(np.float64))
    np.testing.assert_allclose(coef[..., 0], lam.real, rtol=0, atol=1e-6)
    np.testing.assert_allclose(coef[..., 1], lam.imag, rtol=0, atol=1e-6)


def test_prefill_million_token_sequence():
    """One sequence of 2^20 + 3 tokens (B = 1, D = 8, M = 16, bf16): the segmented
    tcgen05 prefill with its longest segment offsets, y on sampled stretches and
    the terminal state against the oracle's recurrence over the whole sequence."""
    L = (1 << 20) + 3
    inp = make_inputs(1, L, 8, 16, "bf16", seed=20)
    y, st = _prefill(inp)
    ref, st_ref = oracle.rec_prefill(inp.x, *inp.params())
    yn = to_np(y)
    for a in (0, 2048 * 100 + 7, L - 5000):
        assert_close(yn[:, a:a + 5000], ref[:, a:a + 5000], TOL["bf16"], f"y at {a}")
    _state_err(st, st_ref, TOL["bf16"])
