"""Failure detection on the GPU without a fault: a bounded device wait is made to
expire on purpose and must end in RLM_ERR_TIMEOUT, not a hang, with the CUDA
context left usable.

The prefill splits a long sequence with few batch rows into segments run by
different thread blocks; a block waits (bounded) for the end states that the
blocks of earlier segments publish.  The test hook rlm_test_stall_segments
shortens that bound to about 1 ms and makes the first segment withhold its flag,
so every later segment's wait runs out: those blocks set the device status word,
drain what they issued, free their tensor memory and return."""
import time

import pytest

import oracle
from synth import make_inputs
from tests._util import TOL, assert_close, to_dev, to_np

torch = pytest.importorskip("torch")
rlm = pytest.importorskip("paper_2607_05583_gb300")

pytestmark = pytest.mark.gpu


def test_expired_segment_wait_reports_timeout_and_the_context_recovers():
    from paper_2607_05583_gb300 import build
    build.build()
    lib = rlm.load_library()
    torch.cuda.synchronize()
    assert rlm.rlm_get_device_status() == rlm.RLM_OK
    B, L, D, M = 1, 8192, 256, 16
    # One batch row: the sequence is split into segments (the call needs a workspace for them).
    assert rlm.rlm_prefill_workspace_size(B, L, D, M, torch.bfloat16) > 0
    inp = make_inputs(B, L, D, M, "bf16", seed=11)
    x = to_dev(inp.x, "bf16")
    p = rlm.Params.from_arrays(*inp.params())
    y = torch.empty_like(x)
    st = rlm.State.empty(B, D, M)
    assert lib.rlm_test_stall_segments(1) == rlm.RLM_OK
    try:
        t0 = time.perf_counter()
        rlm.rlm_mix_prefill(x, p, y, st)
        torch.cuda.synchronize()
        elapsed = time.perf_counter() - t0
        assert rlm.rlm_get_device_status() == rlm.RLM_ERR_TIMEOUT
        assert elapsed < 1.0, f"the stalled call took {elapsed:.3f} s: the short bound did not apply"
    finally:
        assert lib.rlm_test_stall_segments(0) == rlm.RLM_OK
    # The status word was read and cleared, and the same call now runs normally.
    y.fill_(float("nan"))
    rlm.rlm_mix_prefill(x, p, y, st)
    torch.cuda.synchronize()
    assert rlm.rlm_get_device_status() == rlm.RLM_OK
    y_ref, s_ref = oracle.rec_prefill(inp.x, *inp.params())
    assert_close(to_np(y), y_ref, TOL["bf16"], "y after recovery")
    s = st.complex().cpu().numpy()
    assert_close(s.real, s_ref.real, TOL["bf16"], "state re after recovery")
    assert_close(s.imag, s_ref.imag, TOL["bf16"], "state im after recovery")
