"""rlm_mix_prefill_noalloc: the prefill for callers that cannot allocate device
memory (serving runtimes that reserve all memory up front, plugin hosts that own
every allocation).  Its scratch is the library's one fixed device array, which
keeps whatever the previous call left there.  So consecutive calls of different
shapes -- a large one, then a smaller one that lands on the stale scratch of the
first, then the large one again with new inputs -- must each reproduce the fp64
oracle on their own inputs.

This file is collected last on purpose (its name sorts after the others)."""
import ctypes

import numpy as np
import pytest

import oracle
from synth import make_inputs
from tests._util import TOL, assert_close, to_dev, to_np

torch = pytest.importorskip("torch")
rlm = pytest.importorskip("paper_2607_05583_gb300")

pytestmark = pytest.mark.gpu

# (B, L, D): the first shape's chunk states fill far more of the scratch than the
# second's; the third repeats the first with new inputs.
CALLS = [(4, 8000, 64), (1, 700, 64), (4, 8000, 64)]


@pytest.fixture(scope="module")
def lib():
    from paper_2607_05583_gb300 import build
    build.build()
    return rlm.load_library()


def _noalloc(lib, x, params, y, state):
    xt, yt = rlm._field(x), rlm._field(y)
    st = state._c() if state is not None else None
    return lib.rlm_mix_prefill_noalloc(ctypes.byref(xt), ctypes.byref(params._c()),
                                       ctypes.byref(yt), ctypes.byref(st) if st is not None else None,
                                       ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))


def _check_coef(coef, inp):
    """coef[d][m] = (Re lambda, Im lambda, Re c, Im c) with lambda = exp(-gamma + i omega)
    (Eq. 5) and c = A exp(i phi)."""
    lam = np.exp(-inp.decay.astype(np.float64) + 1j * inp.freq.astype(np.float64))
    c = inp.amp.astype(np.float64) * np.exp(1j * inp.phase.astype(np.float64))
    got = coef.cpu().numpy().astype(np.float64)
    for k, want in enumerate((lam.real, lam.imag, c.real, c.imag)):
        np.testing.assert_allclose(got[..., k], want, rtol=0, atol=2e-6)


@pytest.mark.parametrize("dtype,M", [("f32", 8), ("bf16", 16)])
def test_noalloc_prefill_matches_oracle_on_consecutive_calls(lib, dtype, M):
    for call, (B, L, D) in enumerate(CALLS):
        inp = make_inputs(B, L, D, M, dtype, seed=100 + 7 * call + M)
        x = to_dev(inp.x, dtype)
        p = rlm.Params.from_arrays(*inp.params())
        y = torch.full_like(x, float("nan"))
        st = rlm.State.empty(B, D, M)
        st.s.fill_(float("nan"))
        st.coef.fill_(float("nan"))
        status = _noalloc(lib, x, p, y, st)
        assert status == rlm.RLM_OK, lib.rlm_last_error().decode()
        torch.cuda.synchronize()
        y_ref, s_ref = oracle.rec_prefill(inp.x, *inp.params())
        assert_close(to_np(y), y_ref, TOL[dtype], f"y (call {call}, B={B} L={L})")
        s = st.complex().cpu().numpy()
        assert_close(s.real, s_ref.real, TOL[dtype], f"state re (call {call})")
        assert_close(s.imag, s_ref.imag, TOL[dtype], f"state im (call {call})")
        _check_coef(st.coef, inp)
    assert rlm.rlm_get_device_status() == rlm.RLM_OK


def test_noalloc_prefill_without_state_out(lib):
    """state_out = NULL: only y is written."""
    for call, (B, L, D) in enumerate(CALLS[:2]):
        inp = make_inputs(B, L, D, 4, "f32", seed=300 + call)
        x = to_dev(inp.x, "f32")
        y = torch.full_like(x, float("nan"))
        status = _noalloc(lib, x, rlm.Params.from_arrays(*inp.params()), y, None)
        assert status == rlm.RLM_OK, lib.rlm_last_error().decode()
        torch.cuda.synchronize()
        y_ref, _ = oracle.rec_prefill(inp.x, *inp.params())
        assert_close(to_np(y), y_ref, TOL["f32"], f"y (call {call})")


def test_noalloc_rejects_shapes_beyond_its_scratch(lib):
    B, L, D, M = 64, 32768, 256, 64
    x = torch.empty(B, L, D, dtype=torch.float32, device="cuda")
    y = torch.empty_like(x)
    p = rlm.Params(*(torch.zeros(D, M, device="cuda") for _ in range(4)))
    st = rlm.State.empty(B, D, M)
    status = _noalloc(lib, x, p, y, st)
    assert status == rlm.RLM_ERR_UNSUPPORTED
    msg = lib.rlm_last_error().decode()
    assert "scratch" in msg and str(64 << 20) in msg
