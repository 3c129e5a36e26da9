"""Host-side checks of the C ABI that need no GPU: the library builds and loads,
exports every entry point include/rlm.h declares, and rejects bad arguments
on the host before anything is enqueued (no pointer is dereferenced, so fake
device addresses are enough)."""
import ctypes
import os
import re

import pytest

import paper_2607_05583_gb300 as rlm
from paper_2607_05583_gb300 import build as cbuild

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    cbuild.build()
    return rlm.load_library()


def _declared_entry_points():
    names = []
    for fn in os.listdir(os.path.join(ROOT, "include")):
        if fn.endswith(".h"):
            src = open(os.path.join(ROOT, "include", fn)).read()
            names += re.findall(r"RLM_API\s+[\w\s\*]+?\b(rlm_\w+)\s*\(", src)
    return sorted(set(names))


def test_header_declares_the_boundary():
    names = _declared_entry_points()
    for want in ("rlm_mix_prefill", "rlm_mix_prefill_from", "rlm_mix_decode", "rlm_mix_backward",
                 "rlm_mix_backward_from", "rlm_mixer_prefill", "rlm_mixer_decode", "rlm_prefill_workspace_size", "rlm_backward_workspace_size",
                 "rlm_state_init", "rlm_validate_params", "rlm_get_device_status",
                 "rlm_status_string", "rlm_last_error"):
        assert want in names


def test_library_exports_every_declared_symbol(lib):
    for name in _declared_entry_points():
        assert hasattr(lib, name), name


def test_sources_target_sm103a_only():
    assert cbuild.ARCH == ["-gencode", "arch=compute_103a,code=sm_103a"]


def test_status_strings(lib):
    assert rlm.rlm_status_string(rlm.RLM_OK) == "RLM_OK"
    assert rlm.rlm_status_string(rlm.RLM_ERR_TIMEOUT) == "RLM_ERR_TIMEOUT"
    assert rlm.rlm_version() >= 100


FAKE = 0x7F0000000000          # 256-byte aligned fake device address, never dereferenced


def _t(ptr, B, L, D, dt=rlm.RLM_BF16):
    return rlm._Tensor(ptr, dt, B, L, D)


def _p(D, M, base=FAKE + (1 << 32)):
    return rlm._Params(base, base + 4096, base + 8192, base + 12288, D, M)


def _launch(ws=0, nbytes=0):
    return rlm._Launch(None, ws or None, nbytes)


def _prefill(lib, x, p, y, st=None, ln=None):
    ln = ln or _launch(FAKE + (1 << 34), 1 << 40)
    return lib.rlm_mix_prefill(ctypes.byref(x), ctypes.byref(p), ctypes.byref(y),
                               ctypes.byref(st) if st else None, ctypes.byref(ln))


@pytest.mark.parametrize("case", [
    "null_x", "misaligned_x", "bad_dtype", "d_not_multiple_of_8", "zero_length",
    "shape_mismatch", "dtype_mismatch", "overlap", "m_zero", "m_too_big", "param_d_mismatch",
    "misaligned_param", "state_shape", "ws_too_small", "ws_misaligned"])
def test_prefill_rejects_bad_arguments_on_host(lib, case):
    B, L, D, M = 2, 100, 64, 16
    x = _t(FAKE, B, L, D)
    y = _t(FAKE + (1 << 30), B, L, D)
    p = _p(D, M)
    st = None
    ln = None
    if case == "null_x":
        x = _t(0, B, L, D)
    elif case == "misaligned_x":
        x = _t(FAKE + 8, B, L, D)
    elif case == "bad_dtype":
        x = _t(FAKE, B, L, D, 7)
    elif case == "d_not_multiple_of_8":
        x, y, p = _t(FAKE, B, L, 12), _t(FAKE + (1 << 30), B, L, 12), _p(12, M)
    elif case == "zero_length":
        x, y = _t(FAKE, B, 0, D), _t(FAKE + (1 << 30), B, 0, D)
    elif case == "shape_mismatch":
        y = _t(FAKE + (1 << 30), B, L + 1, D)
    elif case == "dtype_mismatch":
        y = _t(FAKE + (1 << 30), B, L, D, rlm.RLM_F32)
    elif case == "overlap":
        y = _t(FAKE + 256, B, L, D)
    elif case == "m_zero":
        p = _p(D, 0)
    elif case == "m_too_big":
        p = _p(D, 65)
    elif case == "param_d_mismatch":
        p = _p(D + 8, M)
    elif case == "misaligned_param":
        p = _p(D, M, base=FAKE + (1 << 32) + 4)
    elif case == "state_shape":
        st = rlm._State(FAKE + (1 << 33), FAKE + (1 << 33) + (1 << 20), B + 1, D, M)
    elif case in ("ws_too_small", "ws_misaligned"):
        # fp32 I/O runs the chunked SIMT path, which needs a workspace
        x, y = _t(FAKE, B, L, D, rlm.RLM_F32), _t(FAKE + (1 << 30), B, L, D, rlm.RLM_F32)
        assert lib.rlm_prefill_workspace_size(B, L, D, M, rlm.RLM_F32) > 16
        ln = (_launch(FAKE + (1 << 34), 16) if case == "ws_too_small"
              else _launch(FAKE + (1 << 34) + 16, 1 << 40))
    status = _prefill(lib, x, p, y, st, ln)
    assert status == rlm.RLM_ERR_INVALID_ARG, (case, lib.rlm_last_error())
    assert lib.rlm_last_error().decode()


def test_sequences_past_2_to_24_tokens_are_unsupported(lib):
    # The kernels form lambda^n from fp32 token counts, exact up to 2^24.
    B, L, D, M = 1, (1 << 24) + 1, 8, 4
    x, y = _t(FAKE, B, L, D), _t(FAKE + (1 << 36), B, L, D)
    assert _prefill(lib, x, _p(D, M), y, None, None) == rlm.RLM_ERR_UNSUPPORTED
    assert "2^24" in lib.rlm_last_error().decode()


def test_prefill_from_rejects_bad_initial_states_on_host(lib):
    B, L, D, M = 2, 100, 64, 16
    x = _t(FAKE, B, L, D)
    y = _t(FAKE + (1 << 30), B, L, D)
    p = _p(D, M)
    ln = _launch(FAKE + (1 << 34), 1 << 40)
    sbase = FAKE + (1 << 36)

    def call(si, so=None):
        return lib.rlm_mix_prefill_from(ctypes.byref(x), ctypes.byref(p),
                                        ctypes.byref(si) if si else None, ctypes.byref(y),
                                        ctypes.byref(so) if so else None, ctypes.byref(ln))

    def state(ptr, b=B, d=D, m=M, coef=0):
        return rlm._State(ptr, coef, b, d, m)

    assert call(state(0)) == rlm.RLM_ERR_INVALID_ARG                      # NULL s
    assert call(state(sbase + 8)) == rlm.RLM_ERR_INVALID_ARG              # misaligned s
    assert call(state(sbase, b=B + 1)) == rlm.RLM_ERR_INVALID_ARG         # batch mismatch
    assert call(state(sbase, m=M - 1)) == rlm.RLM_ERR_INVALID_ARG         # mode mismatch
    assert call(state(y.ptr)) == rlm.RLM_ERR_INVALID_ARG                  # overlaps y
    so = state(sbase + 256, coef=sbase + (1 << 24))                       # partial overlap
    assert call(state(sbase), so) == rlm.RLM_ERR_INVALID_ARG


def test_prefills_reject_state_out_overlapping_fields_on_host(lib):
    """state_out's complex buffer and its coefficient buffer may overlap neither x,
    y nor each other (rlm_mix_prefill and rlm_mix_prefill_noalloc)."""
    B, L, D, M = 2, 100, 64, 16
    x = _t(FAKE, B, L, D)
    y = _t(FAKE + (1 << 30), B, L, D)
    p = _p(D, M)
    ln = _launch(FAKE + (1 << 34), 1 << 40)
    sbase = FAKE + (1 << 36)
    cases = [(x.ptr + 4096, sbase), (y.ptr, sbase), (sbase, x.ptr + 256), (sbase, y.ptr + 512),
             (sbase, sbase + 256)]
    for s_ptr, c_ptr in cases:
        so = rlm._State(s_ptr, c_ptr, B, D, M)
        assert lib.rlm_mix_prefill(ctypes.byref(x), ctypes.byref(p), ctypes.byref(y), ctypes.byref(so),
                                   ctypes.byref(ln)) == rlm.RLM_ERR_INVALID_ARG, (s_ptr, c_ptr)
        assert lib.rlm_mix_prefill_noalloc(ctypes.byref(x), ctypes.byref(p), ctypes.byref(y), ctypes.byref(so),
                                           None) == rlm.RLM_ERR_INVALID_ARG, (s_ptr, c_ptr)
        assert "overlaps" in lib.rlm_last_error().decode()


def test_decode_rejects_bad_arguments_on_host(lib):
    B, D, M = 4, 64, 16
    st = rlm._State(FAKE + (1 << 33), FAKE + (1 << 33) + (1 << 20), B, D, M)
    ln = _launch()
    call = lambda xt, s, yt: lib.rlm_mix_decode(ctypes.byref(xt), ctypes.byref(s),
                                                ctypes.byref(yt), ctypes.byref(ln))
    # L must be 1
    assert call(_t(FAKE, B, 2, D), st, _t(FAKE + (1 << 30), B, 2, D)) == rlm.RLM_ERR_INVALID_ARG
    # state batch mismatch
    bad = rlm._State(st.s, st.coef, B + 1, D, M)
    assert call(_t(FAKE, B, 1, D), bad, _t(FAKE + (1 << 30), B, 1, D)) == rlm.RLM_ERR_INVALID_ARG
    # y overlaps the state
    assert call(_t(FAKE, B, 1, D), st, _t(st.s, B, 1, D)) == rlm.RLM_ERR_INVALID_ARG
    # M out of range
    bad = rlm._State(st.s, st.coef, B, D, 0)
    assert call(_t(FAKE, B, 1, D), bad, _t(FAKE + (1 << 30), B, 1, D)) == rlm.RLM_ERR_INVALID_ARG


def test_backward_rejects_bad_arguments_on_host(lib):
    B, L, D, M = 1, 50, 16, 2
    dy, x, dx = _t(FAKE, B, L, D), _t(FAKE + (1 << 30), B, L, D), _t(FAKE + (1 << 31), B, L, D)
    p = _p(D, M)
    g = rlm._Params(FAKE + (1 << 35), FAKE + (1 << 35) + 4096, FAKE + (1 << 35) + 8192,
                    FAKE + (1 << 35) + 12288, D, M)
    ln = _launch(FAKE + (1 << 34), 1 << 40)
    call = lambda dy, x, dx, g: lib.rlm_mix_backward(ctypes.byref(dy), ctypes.byref(x),
                                                     ctypes.byref(p), ctypes.byref(dx),
                                                     ctypes.byref(g), ctypes.byref(ln))
    assert call(dy, x, _t(x.ptr, B, L, D), g) == rlm.RLM_ERR_INVALID_ARG        # dx aliases x
    gbad = rlm._Params(g.decay, g.freq, g.amp, g.phase, D, M + 1)
    assert call(dy, x, dx, gbad) == rlm.RLM_ERR_INVALID_ARG                      # grad shape
    gnull = rlm._Params(g.decay, 0, g.amp, g.phase, D, M)
    assert call(dy, x, dx, gnull) == rlm.RLM_ERR_INVALID_ARG
    assert call(dy, _t(FAKE + (1 << 30), B, L, D, rlm.RLM_F32), dx, g) == rlm.RLM_ERR_INVALID_ARG


def test_backward_from_rejects_bad_state_arguments_on_host(lib):
    B, L, D, M = 2, 100, 16, 4
    dy, x, dx = _t(FAKE, B, L, D), _t(FAKE + (1 << 30), B, L, D), _t(FAKE + (1 << 31), B, L, D)
    p = _p(D, M)
    g = rlm._Params(FAKE + (1 << 35), FAKE + (1 << 35) + 4096, FAKE + (1 << 35) + 8192,
                    FAKE + (1 << 35) + 12288, D, M)
    ln = _launch(FAKE + (1 << 34), 1 << 40)
    sbase = FAKE + (1 << 36)
    ref = lambda st: ctypes.byref(st) if st else None

    def call(si=None, go=None, ds=None):
        return lib.rlm_mix_backward_from(ctypes.byref(dy), ctypes.byref(x), ctypes.byref(p),
                                         ref(si), ref(go), ctypes.byref(dx), ctypes.byref(g),
                                         ref(ds), ctypes.byref(ln))

    def state(ptr, b=B, d=D, m=M):
        return rlm._State(ptr, 0, b, d, m)

    assert call(state(0)) == rlm.RLM_ERR_INVALID_ARG                       # NULL s
    assert call(None, state(sbase + 4)) == rlm.RLM_ERR_INVALID_ARG         # misaligned s
    assert call(state(sbase, b=B + 1)) == rlm.RLM_ERR_INVALID_ARG          # batch mismatch
    assert call(None, state(sbase, d=D - 1)) == rlm.RLM_ERR_INVALID_ARG    # width mismatch
    assert call(None, None, state(sbase, m=M + 1)) == rlm.RLM_ERR_INVALID_ARG
    assert call(None, None, state(dx.ptr)) == rlm.RLM_ERR_INVALID_ARG      # d_state_in overlaps dx
    assert call(state(sbase), None, state(sbase)) == rlm.RLM_ERR_INVALID_ARG  # ... the state_in
    assert call(None, None, state(g.decay)) == rlm.RLM_ERR_INVALID_ARG     # ... a gradient


RLM_MAX_K = 8


def test_mixer_rejects_bad_arguments_on_host(lib):
    B, L, D, M, K = 2, 100, 16, 4, 4
    x, z = _t(FAKE, B, L, D), _t(FAKE + (1 << 30), B, L, D)
    g = _t(FAKE + (1 << 31), B, L, D)
    p = _p(D, M)
    ln = _launch(FAKE + (1 << 34), 1 << 40)
    wbase = FAKE + (1 << 37)
    cbase = FAKE + (1 << 38)
    ref = lambda v: ctypes.byref(v) if v is not None else None

    def local(k=K, d=D, w=wbase):
        return rlm._Local(w, w + 4096, d, k)

    def conv(ptr=cbase, b=B, d=D, k=K, dt=rlm.RLM_BF16):
        return rlm._ConvState(ptr, dt, b, d, k)

    def call(gt=g, lc=None, cin=None, zt=z, cout=None, cp=None):
        return lib.rlm_mixer_prefill(ctypes.byref(x), ref(gt), ctypes.byref(p), ref(lc), ref(cp), None, ref(cin),
                                     ctypes.byref(zt), None, ref(cout), ctypes.byref(ln))

    assert call(lc=local(k=RLM_MAX_K + 1)) == rlm.RLM_ERR_INVALID_ARG          # K too large
    assert call(lc=local(k=-1)) == rlm.RLM_ERR_INVALID_ARG
    assert call(lc=local(d=D + 8)) == rlm.RLM_ERR_INVALID_ARG                  # D mismatch
    assert call(lc=local(w=0)) == rlm.RLM_ERR_INVALID_ARG                      # NULL weights
    assert call(gt=_t(FAKE + (1 << 31), B, L + 1, D)) == rlm.RLM_ERR_INVALID_ARG   # g shape
    assert call(gt=_t(z.ptr, B, L, D)) == rlm.RLM_ERR_INVALID_ARG               # g overlaps z
    assert call(lc=local(), cin=conv(k=K + 1)) == rlm.RLM_ERR_INVALID_ARG       # history shape
    assert call(lc=local(), cin=conv(dt=rlm.RLM_F32)) == rlm.RLM_ERR_INVALID_ARG  # history dtype
    assert call(lc=local(), cin=conv(ptr=cbase + 8)) == rlm.RLM_ERR_INVALID_ARG   # misaligned
    assert call(lc=local(), cin=conv(), cout=conv(ptr=cbase + 64)) == rlm.RLM_ERR_INVALID_ARG  # partial overlap
    assert call(lc=local(), cout=conv(ptr=z.ptr)) == rlm.RLM_ERR_INVALID_ARG     # history overlaps z
    cpl = lambda h=4, ptr=wbase + 8192, lam=0.5: rlm._Coupling(ptr, lam, h)
    assert call(cp=cpl(h=3)) == rlm.RLM_ERR_INVALID_ARG                          # D % H != 0
    assert call(cp=cpl(h=65)) == rlm.RLM_ERR_INVALID_ARG                         # H > 64
    assert call(cp=cpl(ptr=0)) == rlm.RLM_ERR_INVALID_ARG                        # no matrix
    assert call(cp=cpl(lam=float("nan"))) == rlm.RLM_ERR_INVALID_ARG             # strength not finite
    st = rlm._State(FAKE + (1 << 33), FAKE + (1 << 33) + (1 << 20), B, D, M)
    x1, z1 = _t(FAKE, B, 1, D), _t(FAKE + (1 << 30), B, 1, D)
    dec = lambda lc, cv: lib.rlm_mixer_decode(ctypes.byref(x1), None, ctypes.byref(st), ref(lc), None, ref(cv),
                                              ctypes.byref(z1), ctypes.byref(ln))
    assert dec(local(), None) == rlm.RLM_ERR_INVALID_ARG                         # history required for K >= 2
    assert dec(local(), conv(b=B + 1)) == rlm.RLM_ERR_INVALID_ARG
    assert dec(local(), conv(ptr=st.s)) == rlm.RLM_ERR_INVALID_ARG               # history overlaps the state


def test_prefill_workspace_only_when_the_sequence_is_segmented(lib):
    # The tensor-core prefill splits the sequence when batch rows x channel groups
    # leave SMs idle; it then needs room for each segment's end state and flag.
    few = rlm.rlm_prefill_workspace_size(1, 32768, 256, 16, rlm.RLM_BF16)
    many = rlm.rlm_prefill_workspace_size(64, 32768, 256, 16, rlm.RLM_BF16)
    assert many == 0
    assert few > 0 and few % 256 == 0
    # states and epoch flags: 2 x 8 bytes per (b, segment, d, m)
    assert few % (2 * 256 * 16 * 8) == 0


def test_workspace_queries_are_host_only_and_monotone(lib):
    a = lib.rlm_prefill_workspace_size(1, 1000, 64, 4, rlm.RLM_F32)
    b = lib.rlm_prefill_workspace_size(4, 100000, 64, 4, rlm.RLM_F32)
    assert b >= a
    assert lib.rlm_backward_workspace_size(2, 5000, 64, 8, rlm.RLM_BF16) > 0
    assert lib.rlm_prefill_workspace_size(0, 10, 8, 1, rlm.RLM_F32) == 0


def test_tensor_core_backward_workspace(lib):
    # bf16 I/O with M <= 32 runs the tensor-core backward: channel-major copies of
    # x, dy and dx ([B*D][Lp] bf16, Lp = L rounded up to 2048-token tiles, each
    # rounded up to 1 KiB) plus the per-(b, d, m) partial sums of G and P of the
    # main pass and of conj(g) J of the terminal-state terms.
    B, L, D, M = 4, 32768, 512, 32
    field = B * D * L * 2
    parts = 3 * B * D * M * 8
    assert rlm.rlm_backward_workspace_size(B, L, D, M, rlm.RLM_BF16) == 3 * field + parts
    B, L, D, M = 1, 2049, 8, 5
    field = (B * D * 4096 * 2 + 1023) // 1024 * 1024
    parts = 3 * ((B * D * M * 8 + 255) // 256 * 256)
    assert rlm.rlm_backward_workspace_size(B, L, D, M, rlm.RLM_BF16) == 3 * field + parts
    # fp32 I/O and M > 32 keep the SIMT path and its chunk workspace.
    assert rlm.rlm_backward_workspace_size(4, 32768, 512, 32, rlm.RLM_F32) < 3 * 4 * 512 * 32768 * 2
    parts40 = 2 * ((8 * 40 * 8 + 255) // 256 * 256)
    assert rlm.rlm_backward_workspace_size(1, 2049, 8, 40, rlm.RLM_BF16) != 3 * field + parts40


def test_binding_fails_loudly_without_library(monkeypatch, tmp_path):
    monkeypatch.setattr(rlm, "_lib", None)
    monkeypatch.setattr(cbuild, "LIB", str(tmp_path / "missing.so"))
    with pytest.raises(RuntimeError, match="not built"):
        rlm.load_library()
