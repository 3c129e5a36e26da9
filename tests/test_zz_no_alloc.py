"""rlm_mix_prefill_noalloc: the prefill for callers that cannot allocate device
memory (serving runtimes that reserve all memory up front, plugin hosts that own
every allocation).  Its scratch is the library's fixed device array, so two
calls in a row must each reproduce what rlm_mix_prefill (caller workspace)
computes, whatever the previous call left in that array.

This file is collected last on purpose (its name sorts after the others)."""
import ctypes

import pytest

from synth import make_inputs
from tests._util import TOL, assert_close, to_dev, to_np

torch = pytest.importorskip("torch")
rlm = pytest.importorskip("paper_2607_05583_gb300")

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def lib():
    from paper_2607_05583_gb300 import build
    build.build()
    return rlm.load_library()


def _noalloc(lib, x, params, y, state):
    xt, yt = rlm._field(x), rlm._field(y)
    st = state._c()
    return lib.rlm_mix_prefill_noalloc(ctypes.byref(xt), ctypes.byref(params._c()),
                                       ctypes.byref(yt), ctypes.byref(st),
                                       ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))


@pytest.mark.parametrize("dtype,M", [("f32", 8), ("bf16", 16)])
def test_noalloc_prefill_matches_workspace_prefill_on_two_calls(lib, dtype, M):
    B, L, D = 2, 3001, 64
    inp = make_inputs(B, L, D, M, dtype, seed=M)
    x = to_dev(inp.x, dtype)
    p = rlm.Params.from_arrays(*inp.params())
    y_ref = torch.empty_like(x)
    st_ref = rlm.State.empty(B, D, M)
    rlm.rlm_mix_prefill(x, p, y_ref, st_ref)
    torch.cuda.synchronize()
    for call in range(2):
        y = torch.full_like(x, float("nan"))
        st = rlm.State.empty(B, D, M)
        status = _noalloc(lib, x, p, y, st)
        assert status == rlm.RLM_OK, lib.rlm_last_error().decode()
        torch.cuda.synchronize()
        assert_close(to_np(y), to_np(y_ref), TOL[dtype], f"y (call {call})")
        s, s_ref = st.complex().cpu().numpy(), st_ref.complex().cpu().numpy()
        assert_close(s.real, s_ref.real, TOL[dtype], f"state re (call {call})")
        assert_close(s.imag, s_ref.imag, TOL[dtype], f"state im (call {call})")
        assert torch.equal(st.coef, st_ref.coef) or dtype == "bf16"
    assert rlm.rlm_get_device_status() == rlm.RLM_OK


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
