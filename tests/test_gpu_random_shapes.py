"""Seeded random configurations through every entry point against the fp64 oracle:
prefill (from an initial state or not), the backward with its state terms, and
the mixer wrapper (gate, local path, coupling).  Each configuration draws B, L, D,
M, the element type, the state arguments and the mixer's options, so the sweep
reaches combinations of paths (segmented or not, passes of 16 modes, time
reversal, SIMT) that the hand-picked cases do not."""
import numpy as np
import pytest

import oracle
from synth import make_inputs, make_mixer_inputs
from tests._util import TOL, assert_close, to_dev, to_np

torch = pytest.importorskip("torch")
rlm = pytest.importorskip("paper_2607_05583_gb300")

pytestmark = pytest.mark.gpu

N_CONFIGS = 64


def _config(i):
    r = np.random.default_rng([2025, i])
    dtype = "bf16" if r.random() < 0.75 else "f32"
    B = int(r.choice([1, 2, 3, 4]))
    D = int(8 * r.integers(1, 17))
    M = int(r.choice([1, 2, 5, 8, 15, 16, 17, 24, 32, 40]))
    L = int(r.choice([1, 2, 63, 64, 65, 777, 2047, 2048, 2049, 3001]))
    K = int(r.choice([0, 1, 3, 4, 8]))
    H = int(r.choice([0, 0, 1, 2, 4, 8]))
    if H and D % H:
        H = 0
    with_state = bool(r.random() < 0.5)
    with_gate = bool(r.random() < 0.7)
    with_gout = bool(r.random() < 0.5)   # drawn last: the earlier draws stay as they were
    return dict(dtype=dtype, B=B, D=D, M=M, L=L, K=K, H=H, with_state=with_state, with_gate=with_gate,
                with_gout=with_gout, seed=1000 + i)


def _state_dev(B, D, M, s_np):
    st = rlm.State.empty(B, D, M)
    st.s.copy_(torch.from_numpy(np.stack([s_np.real, s_np.imag], -1).astype(np.float32)))
    return st


@pytest.mark.parametrize("i", range(N_CONFIGS))
def test_random_configuration(i):
    c = _config(i)
    dtype, B, D, M, L = c["dtype"], c["B"], c["D"], c["M"], c["L"]
    tol = TOL[dtype]
    inp = make_inputs(B, L, D, M, dtype, seed=c["seed"], with_dy=True)
    s_in = None
    if c["with_state"]:
        pre = make_inputs(B, 100, D, M, dtype, seed=c["seed"] + 1)
        s_in = oracle.rec_prefill(pre.x, *inp.params())[1]
    x, dy = to_dev(inp.x, dtype), to_dev(inp.dy, dtype)
    p = rlm.Params.from_arrays(*inp.params())
    si = _state_dev(B, D, M, s_in) if s_in is not None else None

    # prefill
    y = torch.empty_like(x)
    so = rlm.State.empty(B, D, M)
    rlm.rlm_mix_prefill_from(x, p, si, y, so)
    torch.cuda.synchronize()
    y_ref, st_ref = oracle.rec_prefill(inp.x, *inp.params(), state_in=s_in)
    assert_close(to_np(y), y_ref, tol, f"{c} y")
    s = so.complex().cpu().numpy()
    assert_close(s.real, st_ref.real, tol, f"{c} state re")
    assert_close(s.imag, st_ref.imag, tol, f"{c} state im")

    # backward with the state terms (the initial-state gradient whenever there is
    # an initial state or a terminal-state gradient)
    g_out = None
    if c["with_gout"]:
        rg = np.random.default_rng(c["seed"] + 2)
        g_out = rg.standard_normal((B, D, M)) + 1j * rg.standard_normal((B, D, M))
    dx = torch.empty_like(x)
    g = rlm.Grads.empty(D, M)
    ds = rlm.State.empty(B, D, M) if (s_in is not None or g_out is not None) else None
    rlm.rlm_mix_backward_from(dy, x, p, si, _state_dev(B, D, M, g_out) if g_out is not None else None, dx, g, ds)
    torch.cuda.synchronize()
    dx_ref, g_ref = oracle.backward_rec(inp.x, inp.dy, *inp.params(), state_in=s_in, d_state_out=g_out)
    assert_close(to_np(dx), dx_ref, tol, f"{c} dx")
    for k in ("decay", "freq", "amp", "phase"):
        assert_close(getattr(g, k).cpu().numpy(), g_ref[k], tol, f"{c} d{k}")
    if ds is not None:
        d = ds.complex().cpu().numpy()
        assert_close(d.real, g_ref["state_in"].real, tol, f"{c} dstate re")

    # the mixer wrapper
    K, H = c["K"], c["H"]
    mx = make_mixer_inputs(inp, K, seed=c["seed"])
    gt = to_dev(mx.g, dtype) if c["with_gate"] else None
    local = rlm.Local.from_arrays(mx.conv_w, mx.scale) if K else None
    cp = None
    cpl = None
    if H:
        cp = (np.random.default_rng(c["seed"]).standard_normal((H, H)), 0.6)
        cpl = rlm.Coupling.from_arrays(*cp)
    hin = rlm.ConvState(to_dev(mx.conv_in, dtype)) if K else None
    z = torch.empty_like(x)
    rlm.rlm_mixer_prefill(x, gt, p, local, z, state_in=si, conv_in=hin, coupling=cpl)
    torch.cuda.synchronize()
    z_ref, _, _ = oracle.mixer_prefill(inp.x, mx.g if c["with_gate"] else None, *inp.params(), mx.conv_w,
                                       mx.scale, state_in=s_in, conv_in=mx.conv_in if K else None, coupling=cp)
    assert_close(to_np(z), z_ref, tol, f"{c} z")


N_DECODE = 24


def _decode_config(i):
    r = np.random.default_rng([2026, i])
    dtype = "bf16" if r.random() < 0.75 else "f32"
    B = int(r.choice([1, 2, 7, 8, 9, 16, 33, 64, 200]))
    D = int(r.choice([8, 24, 64, 256, 520, 2048, 4096]))
    M = int(r.choice([1, 2, 5, 6, 8, 16, 17, 32, 40, 64]))
    K = int(r.choice([0, 1, 3, 4, 8]))
    H = int(r.choice([0, 0, 0, 2, 8]))
    mixer = bool(r.random() < 0.6)
    with_gate = bool(r.random() < 0.7)
    if H and (D % H or (D // H) % 4 or B * D * M > (1 << 21)):
        H = 0
    return dict(dtype=dtype, B=B, D=D, M=M, K=K, H=H, mixer=mixer, with_gate=with_gate, seed=5000 + i)


@pytest.mark.parametrize("i", range(N_DECODE))
def test_random_decode_configuration(i):
    """Seeded decode configurations: 1 to 200 batch rows (grids of one or several
    waves, blocks of 8 or 16 rows), D up to 4096, M from 1 to 64 (one mode pair
    per thread, widened groups, several modes per thread), plain steps or the
    mixer's (gate, local path, coupling).  A 3-token prefill, then 4 chained
    steps, against the oracle over the whole sequence on sampled channels (all
    channels with coupling), outputs and terminal state."""
    c = _decode_config(i)
    dtype, B, D, M, K, H = c["dtype"], c["B"], c["D"], c["M"], c["K"], c["H"]
    tol = TOL[dtype]
    L0, T = 3, 4
    inp = make_inputs(B, L0 + T, D, M, dtype, seed=c["seed"])
    x = to_dev(inp.x, dtype)
    p = rlm.Params.from_arrays(*inp.params())
    st = rlm.State.empty(B, D, M)
    if H:
        chans = np.arange(D)
    else:
        pick = np.random.default_rng(c["seed"]).choice(D, min(D, 40), replace=False)
        chans = np.unique(np.r_[pick, D - 1])
    params = (inp.decay[chans], inp.freq[chans], inp.amp[chans], inp.phase[chans])
    outs = []
    if not c["mixer"]:
        y0 = torch.empty_like(x[:, :L0])
        rlm.rlm_mix_prefill(x[:, :L0].contiguous(), p, y0, st)
        for t in range(L0, L0 + T):
            yt = torch.empty_like(x[:, t])
            rlm.rlm_mix_decode(x[:, t].contiguous(), st, yt)
            outs.append(yt)
        torch.cuda.synchronize()
        ref, st_ref = oracle.rec_prefill(inp.x[:, :, chans], *params)
    else:
        mx = make_mixer_inputs(inp, K, seed=c["seed"])
        g = to_dev(mx.g, dtype) if c["with_gate"] else None
        local = rlm.Local.from_arrays(mx.conv_w, mx.scale) if K else None
        cp = (np.random.default_rng(c["seed"]).standard_normal((H, H)), 0.6) if H else None
        cpl = rlm.Coupling.from_arrays(*cp) if H else None
        hin = rlm.ConvState(to_dev(mx.conv_in, dtype)) if K else None
        hout = rlm.ConvState.empty(B, D, K, dtype=x.dtype) if K else None
        z0 = torch.empty_like(x[:, :L0])
        rlm.rlm_mixer_prefill(x[:, :L0].contiguous(), g[:, :L0].contiguous() if g is not None else None, p, local,
                              z0, conv_in=hin, state_out=st, conv_out=hout, coupling=cpl)
        for t in range(L0, L0 + T):
            zt = torch.empty_like(x[:, t])
            rlm.rlm_mixer_decode(x[:, t].contiguous(), g[:, t].contiguous() if g is not None else None, st, local,
                                 hout, zt, coupling=cpl)
            outs.append(zt)
        torch.cuda.synchronize()
        ref, st_ref, _ = oracle.mixer_prefill(inp.x[:, :, chans], mx.g[:, :, chans] if c["with_gate"] else None,
                                              *params, mx.conv_w[chans], mx.scale[chans],
                                              conv_in=mx.conv_in[:, :, chans] if K else None, coupling=cp)
    assert_close(to_np(torch.stack(outs, 1))[:, :, chans], ref[:, L0:], tol, f"{c} outputs")
    s = st.complex().cpu().numpy()[:, chans]
    assert_close(s.real, st_ref.real, tol, f"{c} state re")
    assert_close(s.imag, st_ref.imag, tol, f"{c} state im")
