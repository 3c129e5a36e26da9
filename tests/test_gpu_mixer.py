"""GPU parity of the mixer wrapper (Sec. 3.4: gate and local path around the
operator) through the C ABI against the fp64 oracle, on every prefill path and
in decode."""
import numpy as np
import pytest

import oracle
from synth import make_inputs, make_mixer_inputs
from tests._util import TOL, assert_close, to_dev, to_np

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


def _state_from(B, D, M, s_np):
    st = rlm.State.empty(B, D, M)
    st.s.copy_(torch.from_numpy(np.stack([s_np.real, s_np.imag], -1).astype(np.float32)))
    return st


def _run_prefill(inp, mx, with_g=True, with_hist=True, s_in=None):
    dt = inp.dtype
    x = to_dev(inp.x, dt)
    g = to_dev(mx.g, dt) if with_g else None
    p = rlm.Params.from_arrays(*inp.params())
    local = rlm.Local.from_arrays(mx.conv_w, mx.scale) if mx.K > 0 else None
    cin = rlm.ConvState(to_dev(mx.conv_in, dt)) if with_hist and mx.K > 0 else None
    cout = rlm.ConvState.empty(inp.B, inp.D, max(mx.K, 1), dtype=x.dtype) if mx.K > 0 else None
    si = _state_from(inp.B, inp.D, inp.M, s_in) if s_in is not None else None
    so = rlm.State.empty(inp.B, inp.D, inp.M)
    z = torch.empty_like(x)
    rlm.rlm_mixer_prefill(x, g, p, local, z, state_in=si, conv_in=cin, state_out=so, conv_out=cout)
    torch.cuda.synchronize()
    return z, so, cout


def _check_prefill(inp, mx, z, so, cout, with_g, with_hist, s_in=None):
    tol = TOL[inp.dtype]
    zr, sr, tr = oracle.mixer_prefill(inp.x, mx.g if with_g else None, *inp.params(), mx.conv_w, mx.scale,
                                      state_in=s_in, conv_in=mx.conv_in if with_hist else None)
    assert_close(to_np(z), zr, tol, "z")
    s = so.complex().cpu().numpy()
    assert_close(s.real, sr.real, tol, "state re")
    assert_close(s.imag, sr.imag, tol, "state im")
    if cout is not None and mx.K > 1:
        np.testing.assert_array_equal(to_np(cout.u), tr)   # the history is a copy: bit-exact


@pytest.mark.parametrize("B,L,D,M,K,dtype,with_g,with_hist", [
    (2, 2 * 2048 + 77, 64, 16, 4, "bf16", True, True),    # tcgen05 prefill (M = 16), ragged tail
    (1, 3000, 16, 16, 8, "bf16", True, False),             # ... segmented sequence, K = 8, zero history
    (3, 1000, 32, 16, 1, "bf16", False, False),            # ... no gate, pointwise local path
    (2, 1000, 8, 16, 0, "bf16", True, False),              # ... gate only
    (2, 1000, 8, 32, 4, "bf16", True, True),               # time-reversed tcgen05 prefill
    (2, 1000, 16, 7, 3, "f32", True, True),                # SIMT, fp32
    (1, 500, 8, 40, 2, "bf16", True, True),                # SIMT, bf16 with M > 32
    (1, 5, 8, 16, 8, "bf16", True, True),                  # L shorter than the history
    (1, 700, 2048, 16, 4, "bf16", True, True),             # 4 KB rows: the channel-pair pass instead
    (1, 300, 1024, 7, 3, "f32", True, False),              # ... and in fp32
    (1, 130, 16, 16, 8, "bf16", True, True),               # 64-token tiles: the history rows of tile 2
])
def test_mixer_prefill_matches_oracle(B, L, D, M, K, dtype, with_g, with_hist):
    inp = make_inputs(B, L, D, M, dtype, seed=L + K)
    mx = make_mixer_inputs(inp, K, seed=L + K)
    z, so, cout = _run_prefill(inp, mx, with_g, with_hist)
    _check_prefill(inp, mx, z, so, cout, with_g, with_hist)


def test_mixer_prefill_from_state_matches_oracle():
    inp = make_inputs(2, 3001, 64, 16, "bf16", seed=5)
    mx = make_mixer_inputs(inp, 4, seed=5)
    pre = make_inputs(2, 300, 64, 16, "bf16", seed=6)
    _, s_in = oracle.rec_prefill(pre.x, *inp.params())
    z, so, cout = _run_prefill(inp, mx, True, True, s_in=s_in)
    _check_prefill(inp, mx, z, so, cout, True, True, s_in=s_in)


def test_mixer_without_gate_or_local_path_is_the_mixing():
    inp = make_inputs(2, 3000, 64, 16, "bf16", seed=9)
    x = to_dev(inp.x, "bf16")
    p = rlm.Params.from_arrays(*inp.params())
    y, z = torch.empty_like(x), torch.empty_like(x)
    rlm.rlm_mix_prefill(x, p, y)
    rlm.rlm_mixer_prefill(x, None, p, None, z)
    torch.cuda.synchronize()
    assert torch.equal(y, z)


@pytest.mark.parametrize("M", [16, 32])
def test_mixer_split_prefill_in_place_equals_whole(M):
    """Prefill of x1, then of x2 continuing from the state and drive history, both
    updated in place, equals one prefill of x1 || x2."""
    B, L, D, K, cut = 2, 5000, 64, 4, 2345
    inp = make_inputs(B, L, D, M, "bf16", seed=21)
    mx = make_mixer_inputs(inp, K, seed=21)
    x, g = to_dev(inp.x, "bf16"), to_dev(mx.g, "bf16")
    p = rlm.Params.from_arrays(*inp.params())
    local = rlm.Local.from_arrays(mx.conv_w, mx.scale)
    st = rlm.State.empty(B, D, M)
    cs = rlm.ConvState.empty(B, D, K, dtype=torch.bfloat16)
    x1, x2 = x[:, :cut].contiguous(), x[:, cut:].contiguous()
    g1, g2 = g[:, :cut].contiguous(), g[:, cut:].contiguous()
    z1, z2 = torch.empty_like(x1), torch.empty_like(x2)
    rlm.rlm_mixer_prefill(x1, g1, p, local, z1, state_out=st, conv_out=cs)
    rlm.rlm_mixer_prefill(x2, g2, p, local, z2, state_in=st, conv_in=cs, state_out=st, conv_out=cs)
    torch.cuda.synchronize()
    zr, sr, tr = oracle.mixer_prefill(inp.x, mx.g, *inp.params(), mx.conv_w, mx.scale)
    assert_close(to_np(torch.cat([z1, z2], 1)), zr, TOL["bf16"], "z")
    s = st.complex().cpu().numpy()
    assert_close(s.real, sr.real, TOL["bf16"], "state re")
    np.testing.assert_array_equal(to_np(cs.u), tr)


@pytest.mark.parametrize("dtype,M,K,B", [("bf16", 16, 4, 3), ("f32", 7, 3, 3), ("bf16", 40, 8, 3), ("bf16", 16, 1, 3),
                                       ("f32", 1, 8, 3), ("bf16", 2, 6, 3), ("bf16", 6, 8, 3),
                                       ("bf16", 16, 4, 12), ("f32", 2, 6, 12), ("bf16", 40, 8, 12)])
def test_mixer_decode_continues_the_prefill(dtype, M, K, B):
    """Prefill of 300 tokens then 40 fused mixer decode steps reproduce the oracle's
    mixer output over all 340 tokens, and the final state and history (row-tiled
    step: 3 rows in one block of 8, 12 rows over two; M = 1, 7 on the any-M
    kernel)."""
    D, L0, T = 32, 300, 40
    inp = make_inputs(B, L0 + T, D, M, dtype, seed=M + K)
    mx = make_mixer_inputs(inp, K, seed=M + K)
    x, g = to_dev(inp.x, dtype), to_dev(mx.g, dtype)
    p = rlm.Params.from_arrays(*inp.params())
    local = rlm.Local.from_arrays(mx.conv_w, mx.scale)
    st = rlm.State.empty(B, D, M)
    cs = rlm.ConvState.empty(B, D, K, dtype=x.dtype)
    z0 = torch.empty_like(x[:, :L0])
    rlm.rlm_mixer_prefill(x[:, :L0].contiguous(), g[:, :L0].contiguous(), p, local, z0, state_out=st, conv_out=cs)
    zs = []
    for t in range(L0, L0 + T):
        zt = torch.empty_like(x[:, t])
        rlm.rlm_mixer_decode(x[:, t].contiguous(), g[:, t].contiguous(), st, local, cs, zt)
        zs.append(zt)
    torch.cuda.synchronize()
    zr, sr, tr = oracle.mixer_prefill(inp.x, mx.g, *inp.params(), mx.conv_w, mx.scale)
    assert_close(to_np(z0), zr[:, :L0], TOL[dtype], "prefill z")
    assert_close(to_np(torch.stack(zs, 1)), zr[:, L0:], TOL[dtype], "decode z")
    s = st.complex().cpu().numpy()
    assert_close(s.real, sr.real, TOL[dtype], "state re")
    if K > 1:
        np.testing.assert_array_equal(to_np(cs.u), tr)


@pytest.mark.parametrize("B,D", [(8, 256), (64, 2048)])
def test_mixer_decode_on_one_and_several_waves(B, D):
    """The row-tiled mixer step on a grid that fits on the GPU at once (8 x 256)
    and on one of several waves (64 x 2048: 4096 blocks), chained over 5 steps
    after a 6-token prefill: output, state and history against the oracle on
    sampled channels, the first and last included."""
    M, K, L0, T = 16, 4, 6, 5
    inp = make_inputs(B, L0 + T, D, M, "bf16", seed=D)
    mx = make_mixer_inputs(inp, K, seed=D)
    x, g = to_dev(inp.x, "bf16"), to_dev(mx.g, "bf16")
    p = rlm.Params.from_arrays(*inp.params())
    local = rlm.Local.from_arrays(mx.conv_w, mx.scale)
    st = rlm.State.empty(B, D, M)
    cs = rlm.ConvState.empty(B, D, K, dtype=x.dtype)
    z0 = torch.empty_like(x[:, :L0])
    rlm.rlm_mixer_prefill(x[:, :L0].contiguous(), g[:, :L0].contiguous(), p, local, z0, state_out=st, conv_out=cs)
    zs = []
    for t in range(L0, L0 + T):
        zt = torch.empty_like(x[:, t])
        rlm.rlm_mixer_decode(x[:, t].contiguous(), g[:, t].contiguous(), st, local, cs, zt)
        zs.append(zt)
    torch.cuda.synchronize()
    chans = np.unique(np.r_[np.random.default_rng(B).choice(D, 45, replace=False), 0, D - 1])
    zr, sr, tr = oracle.mixer_prefill(inp.x[:, :, chans], mx.g[:, :, chans], inp.decay[chans], inp.freq[chans],
                                      inp.amp[chans], inp.phase[chans], mx.conv_w[chans], mx.scale[chans])
    assert_close(to_np(torch.stack(zs, 1))[:, :, chans], zr[:, L0:], TOL["bf16"], "decode z")
    s = st.complex().cpu().numpy()[:, chans]
    assert_close(s.real, sr.real, TOL["bf16"], "state re")
    assert_close(s.imag, sr.imag, TOL["bf16"], "state im")
    np.testing.assert_array_equal(to_np(cs.u)[:, :, chans], tr)


def test_mixer_decode_without_gate_or_local_path_is_the_decode():
    inp = make_inputs(4, 1, 64, 16, "bf16", seed=2)
    x = to_dev(inp.x[:, 0], "bf16")
    p = rlm.Params.from_arrays(*inp.params())
    s1, s2 = rlm.State.empty(4, 64, 16), rlm.State.empty(4, 64, 16)
    rlm.rlm_state_init(s1, p)
    rlm.rlm_state_init(s2, p)
    y, z = torch.empty_like(x), torch.empty_like(x)
    for _ in range(3):
        rlm.rlm_mix_decode(x, s1, y)
        rlm.rlm_mixer_decode(x, None, s2, None, None, z)
    torch.cuda.synchronize()
    assert torch.equal(y, z) and torch.equal(s1.s, s2.s)


def test_mixer_prefill_is_causal_bit_exact():
    """Changing x and g from token t0 on leaves z before t0 bit-identical."""
    inp = make_inputs(2, 4100, 64, 16, "bf16", seed=4)
    mx = make_mixer_inputs(inp, 4, seed=4)
    x, g = to_dev(inp.x, "bf16"), to_dev(mx.g, "bf16")
    p = rlm.Params.from_arrays(*inp.params())
    local = rlm.Local.from_arrays(mx.conv_w, mx.scale)
    z1, z2 = torch.empty_like(x), torch.empty_like(x)
    rlm.rlm_mixer_prefill(x, g, p, local, z1)
    t0 = 2049
    x2, g2 = x.clone(), g.clone()
    x2[:, t0:] = torch.randn_like(x2[:, t0:])
    g2[:, t0:] = torch.randn_like(g2[:, t0:])
    rlm.rlm_mixer_prefill(x2, g2, p, local, z2)
    torch.cuda.synchronize()
    assert torch.equal(z1[:, :t0], z2[:, :t0])
    assert not torch.equal(z1[:, t0:], z2[:, t0:])


def test_mixer_prefill_long_context_sampled():
    """The long-context workload shape (B=4, L=32768, D=256, M=16, K=4, bf16) on
    sampled channels against the oracle."""
    inp = make_inputs(4, 32768, 256, 16, "bf16", seed=0)
    mx = make_mixer_inputs(inp, 4, seed=0)
    z, so, cout = _run_prefill(inp, mx, True, True)
    ch = np.array([0, 7, 8, 129, 255])
    zr, sr, tr = oracle.mixer_prefill(inp.x[:, :, ch], mx.g[:, :, ch], inp.decay[ch], inp.freq[ch], inp.amp[ch],
                                      inp.phase[ch], mx.conv_w[ch], mx.scale[ch], conv_in=mx.conv_in[:, :, ch])
    assert_close(to_np(z)[:, :, ch], zr, TOL["bf16"], "z")
    np.testing.assert_array_equal(to_np(cout.u)[:, :, ch], tr)


# ---- the gate fused into the tcgen05 epilogue (bf16, M = 16, unsegmented: >= 77
# channel groups x rows); with a local path the mixing is followed by one full-width pass
def _launches(fn):
    before = rlm.rlm_kernels_launched()
    fn()
    torch.cuda.synchronize()
    return rlm.rlm_kernels_launched() - before


@pytest.mark.parametrize("B,L,D,K,with_g,with_hist", [
    (2, 2 * 2048 + 77, 512, 0, True, False),   # gate only: fused; ragged, token 0 inside tile 0
    (1, 3 * 2048, 1024, 0, True, False),       # gate only: fused; tiles aligned with the sequence
    (2, 2 * 2048 + 77, 512, 4, True, True),    # local path: mixing + pass + history tail
    (1, 3 * 2048, 1024, 8, True, True),
    (2, 2048 + 3, 512, 2, False, True),
    (8, 2048, 256, 0, True, False),            # gate only, two batch rows per CTA (the 6M layer)
    (9, 700, 256, 0, True, False),             # ... three rows per CTA, one tile each
])
def test_tcgen05_shape_mixer_prefill_matches_oracle(B, L, D, K, with_g, with_hist):
    inp = make_inputs(B, L, D, 16, "bf16", seed=L + D + K)
    mx = make_mixer_inputs(inp, K, seed=L + K)
    out = {}

    def run():
        out["r"] = _run_prefill(inp, mx, with_g, with_hist)

    n = _launches(run)
    # fused gate: one launch; otherwise the tcgen05 prefill, the pass and (K >= 2)
    # the history tail
    assert n == (1 if K == 0 else 2 + (1 if K >= 2 else 0)), n
    z, so, cout = out["r"]
    _check_prefill(inp, mx, z, so, cout, with_g, with_hist)


@pytest.mark.parametrize("M,K", [(32, 4), (24, 0), (40, 4)])
def test_multi_pass_mixer_prefill_matches_oracle(M, K):
    """M > 16 on an unsegmented shape: the prefill (one launch of the 32-mode
    instance for M <= 32, else passes of 16 modes), then the mixer pass (the gate
    is not fused with more than 16 modes)."""
    inp = make_inputs(2, 3000, 512, M, "bf16", seed=M + K)
    mx = make_mixer_inputs(inp, K, seed=M)
    out = {}

    def run():
        out["r"] = _run_prefill(inp, mx, True, K > 0)

    n = _launches(run)
    passes = 1 if M <= 32 else (M + 15) // 16
    assert n == passes + 1 + (1 if K >= 2 else 0), n
    z, so, cout = out["r"]
    _check_prefill(inp, mx, z, so, cout, True, K > 0)


@pytest.mark.parametrize("K", [0, 4])
def test_tcgen05_shape_mixer_prefill_from_state_and_split_in_place(K):
    B, L, D, cut = 2, 6000, 512, 2345
    inp = make_inputs(B, L, D, 16, "bf16", seed=77)
    mx = make_mixer_inputs(inp, K, seed=77)
    x, g = to_dev(inp.x, "bf16"), to_dev(mx.g, "bf16")
    p = rlm.Params.from_arrays(*inp.params())
    local = rlm.Local.from_arrays(mx.conv_w, mx.scale) if K else None
    st = rlm.State.empty(B, D, 16)
    cs = rlm.ConvState(to_dev(mx.conv_in, "bf16")) if K else None
    x1, x2 = x[:, :cut].contiguous(), x[:, cut:].contiguous()
    g1, g2 = g[:, :cut].contiguous(), g[:, cut:].contiguous()
    z1, z2 = torch.empty_like(x1), torch.empty_like(x2)
    rlm.rlm_mixer_prefill(x1, g1, p, local, z1, conv_in=cs, state_out=st, conv_out=cs)
    rlm.rlm_mixer_prefill(x2, g2, p, local, z2, state_in=st, conv_in=cs, state_out=st, conv_out=cs)
    torch.cuda.synchronize()
    zr, sr, tr = oracle.mixer_prefill(inp.x, mx.g, *inp.params(), mx.conv_w, mx.scale,
                                      conv_in=mx.conv_in if K else None)
    assert_close(to_np(torch.cat([z1, z2], 1)), zr, TOL["bf16"], "z")
    s = st.complex().cpu().numpy()
    assert_close(s.real, sr.real, TOL["bf16"], "state re")
    assert_close(s.imag, sr.imag, TOL["bf16"], "state im")
    if K:
        np.testing.assert_array_equal(to_np(cs.u), tr)


@pytest.mark.parametrize("K", [0, 8])
def test_tcgen05_shape_mixer_prefill_is_causal_bit_exact(K):
    inp = make_inputs(2, 4100, 512, 16, "bf16", seed=14)
    mx = make_mixer_inputs(inp, K, seed=14)
    x, g = to_dev(inp.x, "bf16"), to_dev(mx.g, "bf16")
    p = rlm.Params.from_arrays(*inp.params())
    local = rlm.Local.from_arrays(mx.conv_w, mx.scale) if K else None
    z1, z2 = torch.empty_like(x), torch.empty_like(x)
    rlm.rlm_mixer_prefill(x, g, p, local, z1)
    for t0 in (2048, 2049, 4095):
        x2, g2 = x.clone(), g.clone()
        x2[:, t0:] = torch.randn_like(x2[:, t0:])
        g2[:, t0:] = torch.randn_like(g2[:, t0:])
        rlm.rlm_mixer_prefill(x2, g2, p, local, z2)
        torch.cuda.synchronize()
        assert torch.equal(z1[:, :t0], z2[:, :t0]), t0
        assert not torch.equal(z1[:, t0:], z2[:, t0:])


def test_packed_rows_gate_from_state_matches_oracle():
    """The gate in the epilogue of a prefill whose CTAs run several batch rows
    (B = 9, L = 704, D = 256: three rows per CTA), each row from its own initial
    state."""
    B, L, D, M = 9, 704, 256, 16
    inp = make_inputs(B, L, D, M, "bf16", seed=77)
    mx = make_mixer_inputs(inp, 0, seed=77)
    rng = np.random.default_rng(77)
    s_in = rng.standard_normal((B, D, M)) + 1j * rng.standard_normal((B, D, M))
    x, g = to_dev(inp.x, "bf16"), to_dev(mx.g, "bf16")
    p = rlm.Params.from_arrays(*inp.params())
    so, z = rlm.State.empty(B, D, M), torch.empty_like(x)
    assert _launches(lambda: rlm.rlm_mixer_prefill(x, g, p, None, z, state_in=_state_from(B, D, M, s_in),
                                                   state_out=so)) == 1
    zr, sr, _ = oracle.mixer_prefill(inp.x, mx.g, *inp.params(), mx.conv_w, mx.scale, state_in=s_in)
    assert_close(to_np(z), zr, TOL["bf16"], "z")
    s = so.complex().cpu().numpy()
    assert_close(s.real, sr.real, TOL["bf16"], "state re")
    assert_close(s.imag, sr.imag, TOL["bf16"], "state im")


def test_fused_and_unfused_gate_agree():
    """The gate through the fused epilogue (D = 512) and, 64 channels at a time,
    through the segmented prefill and the separate pass: within one bf16 rounding
    of z (the unfused route rounds y before the gate)."""
    inp = make_inputs(2, 3000, 512, 16, "bf16", seed=3)
    mx = make_mixer_inputs(inp, 0, seed=3)
    x, g = to_dev(inp.x, "bf16"), to_dev(mx.g, "bf16")
    p = rlm.Params.from_arrays(*inp.params())
    zf = torch.empty_like(x)
    assert _launches(lambda: rlm.rlm_mixer_prefill(x, g, p, None, zf)) == 1
    zu = torch.empty_like(x)
    for c0 in range(0, 512, 64):
        sl = slice(c0, c0 + 64)
        ps = rlm.Params(*(t[sl].contiguous() for t in (p.decay, p.freq, p.amp, p.phase)))
        zs = torch.empty_like(x[:, :, sl].contiguous())
        assert _launches(lambda: rlm.rlm_mixer_prefill(x[:, :, sl].contiguous(), g[:, :, sl].contiguous(), ps,
                                                       None, zs)) == 2
        zu[:, :, sl] = zs
    torch.cuda.synchronize()
    d = (zf.float() - zu.float()).abs().max().item()
    assert d <= 2.0 ** -6 * zu.float().abs().max().item(), d


# ---- head coupling (NEXT 3): C = I + lambda_c/sqrt(H) tanh(C~) before the gate
def _coupling(H, seed, lam=0.7):
    return np.random.default_rng(seed).standard_normal((H, H)), lam


@pytest.mark.parametrize("B,L,D,M,K,H,dtype,with_g", [
    (2, 3001, 64, 16, 4, 8, "bf16", True),          # tcgen05 prefill (segmented), K = 4
    (2, 2 * 2048 + 77, 512, 16, 0, 8, "bf16", True), # unsegmented shape: the gate is not fused with coupling
    (2, 1000, 16, 7, 3, 4, "f32", True),             # SIMT, fp32
    (1, 700, 8, 40, 2, 2, "bf16", False),            # SIMT, bf16 with M > 32, no gate
    (2, 1000, 32, 32, 0, 1, "bf16", True),           # time-reversed prefill, H = 1 (a scalar gain)
    (2, 1000, 24, 16, 4, 8, "bf16", True),           # head width 3: one position per thread
    (2, 1000, 64, 16, 2, 32, "f32", True),           # 32 heads: whole rows staged in shared memory
    (2, 3001, 64, 16, 4, 16, "bf16", True),          # 16 heads (the largest unrolled case)
    (1, 700, 48, 16, 3, 12, "bf16", True),           # 12 heads: H not unrolled, head width 4
    (1, 50, 8, 4, 2, 8, "f32", True),                # one channel per head
    (2, 1000, 128, 16, 4, 16, "bf16", True),         # 16 heads of width 8: coupling in the whole-row pass
    (2, 1000, 96, 16, 4, 12, "bf16", True),          # 12 heads of width 8: separate passes
    (2, 700, 64, 7, 3, 4, "f32", True),              # ... fp32, 4 heads
    (2, 600, 64, 16, 0, 4, "bf16", False),           # coupling alone, in the whole-row pass
    (1, 300, 1024, 16, 2, 8, "f32", True),           # 4 KB rows: separate coupling and mixer passes
    (1, 300, 8192, 16, 4, 64, "bf16", True),         # the largest coupling: D = 8192, 64 heads of 128
])
def test_coupled_mixer_prefill_matches_oracle(B, L, D, M, K, H, dtype, with_g):
    inp = make_inputs(B, L, D, M, dtype, seed=L + H)
    mx = make_mixer_inputs(inp, K, seed=L + H)
    c_raw, lam = _coupling(H, H)
    x = to_dev(inp.x, dtype)
    g = to_dev(mx.g, dtype) if with_g else None
    p = rlm.Params.from_arrays(*inp.params())
    local = rlm.Local.from_arrays(mx.conv_w, mx.scale) if K else None
    cin = rlm.ConvState(to_dev(mx.conv_in, dtype)) if K else None
    so = rlm.State.empty(B, D, M)
    z = torch.empty_like(x)
    rlm.rlm_mixer_prefill(x, g, p, local, z, conv_in=cin, state_out=so,
                          coupling=rlm.Coupling.from_arrays(c_raw, lam))
    torch.cuda.synchronize()
    zr, sr, _ = oracle.mixer_prefill(inp.x, mx.g if with_g else None, *inp.params(), mx.conv_w, mx.scale,
                                     conv_in=mx.conv_in if K else None, coupling=(c_raw, lam))
    assert_close(to_np(z), zr, TOL[dtype], "z")
    s = so.complex().cpu().numpy()
    assert_close(s.real, sr.real, TOL[dtype], "state re")


@pytest.mark.parametrize("dtype,M,K,H,B,D,launches", [
    # one launch per step (M / 2 a power of two, D <= 512, D * M <= 4096): one block per batch row
    ("bf16", 16, 4, 8, 3, 64, 1), ("bf16", 16, 0, 2, 3, 64, 1), ("bf16", 2, 8, 16, 3, 64, 1),
    ("bf16", 16, 4, 8, 1, 64, 1), ("f32", 16, 3, 4, 3, 64, 1), ("bf16", 64, 4, 8, 2, 64, 1),
    ("bf16", 8, 8, 16, 2, 512, 1),
    # two launches: the recurrence step, then coupling, gate and local path
    ("f32", 7, 3, 4, 3, 64, 2), ("bf16", 12, 2, 4, 2, 64, 2), ("bf16", 32, 4, 8, 2, 512, 2),
    ("bf16", 64, 4, 8, 2, 128, 2),
    ("bf16", 16, 4, 64, 2, 8192, 2),                 # the largest coupling (48 KB of C and y_t per block)
])
def test_coupled_mixer_decode_continues_the_prefill(dtype, M, K, H, B, D, launches):
    L0, T = 300, 30
    inp = make_inputs(B, L0 + T, D, M, dtype, seed=M + K + H)
    mx = make_mixer_inputs(inp, K, seed=M + K + H)
    c_raw, lam = _coupling(H, 3 * H)
    cp = rlm.Coupling.from_arrays(c_raw, lam)
    x, g = to_dev(inp.x, dtype), to_dev(mx.g, dtype)
    p = rlm.Params.from_arrays(*inp.params())
    local = rlm.Local.from_arrays(mx.conv_w, mx.scale) if K else None
    st = rlm.State.empty(B, D, M)
    cs = rlm.ConvState.empty(B, D, max(K, 1), dtype=x.dtype)
    z0 = torch.empty_like(x[:, :L0])
    rlm.rlm_mixer_prefill(x[:, :L0].contiguous(), g[:, :L0].contiguous(), p, local, z0, state_out=st,
                          conv_out=cs if K else None, coupling=cp)
    zs = []
    n0 = rlm.rlm_kernels_launched()
    for t in range(L0, L0 + T):
        zt = torch.empty_like(x[:, t])
        rlm.rlm_mixer_decode(x[:, t].contiguous(), g[:, t].contiguous(), st, local, cs if K else None, zt,
                             coupling=cp)
        zs.append(zt)
    torch.cuda.synchronize()
    assert rlm.rlm_kernels_launched() - n0 == launches * T
    zr, sr, tr = oracle.mixer_prefill(inp.x, mx.g, *inp.params(), mx.conv_w, mx.scale, coupling=(c_raw, lam))
    assert_close(to_np(z0), zr[:, :L0], TOL[dtype], "prefill z")
    assert_close(to_np(torch.stack(zs, 1)), zr[:, L0:], TOL[dtype], "decode z")
    if K > 1:
        np.testing.assert_array_equal(to_np(cs.u), tr)


@pytest.mark.parametrize("D,H,passes", [(256, 8, 1), (64, 16, 1), (96, 12, 2), (2048, 8, 2)])
def test_coupled_mixer_prefill_launches(D, H, passes):
    """Coupling, gate and local path after the mixing: one whole-row pass where
    the rows fit (at most 2 KB), H is 1, 2, 4, 8 or 16 and each head is a
    multiple of 4 channels wide; else a coupling pass and a channel-pair pass;
    then the history tail."""
    inp = make_inputs(1, 300, D, 16, "bf16", seed=D + H)
    mx = make_mixer_inputs(inp, 4, seed=D + H)
    x, g = to_dev(inp.x, "bf16"), to_dev(mx.g, "bf16")
    p = rlm.Params.from_arrays(*inp.params())
    local = rlm.Local.from_arrays(mx.conv_w, mx.scale)
    cin = rlm.ConvState(to_dev(mx.conv_in, "bf16"))
    cout = rlm.ConvState.empty(1, D, 4, dtype=x.dtype)
    z = torch.empty_like(x)
    cp = rlm.Coupling.from_arrays(*_coupling(H, H))
    n = _launches(lambda: rlm.rlm_mixer_prefill(x, g, p, local, z, conv_in=cin, conv_out=cout, coupling=cp))
    assert n == 1 + passes + 1, n


def test_zero_strength_coupling_is_no_coupling():
    inp = make_inputs(2, 3001, 64, 16, "bf16", seed=6)
    mx = make_mixer_inputs(inp, 4, seed=6)
    x, g = to_dev(inp.x, "bf16"), to_dev(mx.g, "bf16")
    p = rlm.Params.from_arrays(*inp.params())
    local = rlm.Local.from_arrays(mx.conv_w, mx.scale)
    z0, z1 = torch.empty_like(x), torch.empty_like(x)
    rlm.rlm_mixer_prefill(x, g, p, local, z0)
    rlm.rlm_mixer_prefill(x, g, p, local, z1, coupling=rlm.Coupling.from_arrays(np.ones((8, 8)), 0.0))
    torch.cuda.synchronize()
    assert torch.equal(z0, z1)
