"""Python binding of the GB300 causal resonant field mixing library (``librlm.so``).

Argument marshalling only: every step of the operator runs in the library's
CUDA kernels, reached through the C ABI declared in ``include/rlm.h`` with the
same function names.  PyTorch supplies device memory and the current stream.
There is no fallback: if the compiled library is missing the calls raise.

Names follow the paper (ResonatorLM, arxiv 2607.05583): x is the drive field
[B][L][D]; decay gamma, frequency omega, amplitude A and phase phi are the
per-mode resonator parameters [D][M]; the state is the complex recurrent state
of Sec. 3.3, [B][D][M] complex fp32 plus its mode coefficients.
"""
from __future__ import annotations

import ctypes
import os
from dataclasses import dataclass

import torch

from . import build as _build_mod

__all__ = [
    "RlmError", "Params", "Grads", "State", "load_library", "library_path",
    "rlm_mix_prefill", "rlm_mix_prefill_from", "rlm_mix_prefill_noalloc", "rlm_mix_decode", "rlm_mix_backward",
    "rlm_mix_backward_from", "rlm_state_init", "Local", "ConvState", "Coupling", "rlm_mixer_prefill",
    "rlm_mixer_decode",
    "rlm_prefill_workspace_size", "rlm_backward_workspace_size",
    "rlm_validate_params", "rlm_get_device_status", "rlm_status_string",
    "rlm_version", "rlm_kernels_launched", "RLM_OK", "RLM_ERR_INVALID_ARG", "RLM_ERR_UNSUPPORTED",
    "RLM_ERR_CUDA", "RLM_ERR_TIMEOUT", "RLM_F32", "RLM_BF16",
]

RLM_OK, RLM_ERR_INVALID_ARG, RLM_ERR_UNSUPPORTED, RLM_ERR_CUDA, RLM_ERR_TIMEOUT = range(5)
RLM_F32, RLM_BF16 = 0, 1


class _Tensor(ctypes.Structure):
    _fields_ = [("ptr", ctypes.c_void_p), ("dtype", ctypes.c_int),
                ("B", ctypes.c_int64), ("L", ctypes.c_int64), ("D", ctypes.c_int64)]


class _Params(ctypes.Structure):
    _fields_ = [("decay", ctypes.c_void_p), ("freq", ctypes.c_void_p),
                ("amp", ctypes.c_void_p), ("phase", ctypes.c_void_p),
                ("D", ctypes.c_int), ("M", ctypes.c_int)]


_Grads = _Params


class _State(ctypes.Structure):
    _fields_ = [("s", ctypes.c_void_p), ("coef", ctypes.c_void_p),
                ("B", ctypes.c_int), ("D", ctypes.c_int), ("M", ctypes.c_int)]


class _Local(ctypes.Structure):
    _fields_ = [("conv_w", ctypes.c_void_p), ("scale", ctypes.c_void_p),
                ("D", ctypes.c_int), ("K", ctypes.c_int)]


class _Coupling(ctypes.Structure):
    _fields_ = [("c_raw", ctypes.c_void_p), ("lambda_c", ctypes.c_float), ("H", ctypes.c_int)]


class _ConvState(ctypes.Structure):
    _fields_ = [("u", ctypes.c_void_p), ("dtype", ctypes.c_int), ("B", ctypes.c_int64),
                ("D", ctypes.c_int), ("K", ctypes.c_int)]


class _Launch(ctypes.Structure):
    _fields_ = [("stream", ctypes.c_void_p), ("workspace", ctypes.c_void_p),
                ("workspace_bytes", ctypes.c_size_t)]


class RlmError(RuntimeError):
    def __init__(self, status: int, where: str, detail: str):
        super().__init__(f"{where}: {rlm_status_string(status)}: {detail}")
        self.status = status


_lib = None


def library_path() -> str:
    return _build_mod.LIB


def load_library(build_if_missing: bool = False) -> ctypes.CDLL:
    """Load librlm.so (raises if it has not been built)."""
    global _lib
    if _lib is not None:
        return _lib
    path = _build_mod.LIB
    if not os.path.exists(path):
        if not build_if_missing:
            raise RuntimeError(
                f"the CUDA library {path} is not built; run "
                "`python -c 'import __graft_entry__ as g; g.build()'` first")
        _build_mod.build()
    lib = ctypes.CDLL(path)
    P = ctypes.POINTER
    lib.rlm_mix_prefill.argtypes = [P(_Tensor), P(_Params), P(_Tensor), P(_State), P(_Launch)]
    lib.rlm_mix_prefill_from.argtypes = [P(_Tensor), P(_Params), P(_State), P(_Tensor), P(_State),
                                         P(_Launch)]
    lib.rlm_mix_decode.argtypes = [P(_Tensor), P(_State), P(_Tensor), P(_Launch)]
    lib.rlm_mix_backward.argtypes = [P(_Tensor), P(_Tensor), P(_Params), P(_Tensor),
                                     P(_Grads), P(_Launch)]
    lib.rlm_mix_backward_from.argtypes = [P(_Tensor), P(_Tensor), P(_Params), P(_State), P(_State),
                                          P(_Tensor), P(_Grads), P(_State), P(_Launch)]
    lib.rlm_mixer_prefill.argtypes = [P(_Tensor), P(_Tensor), P(_Params), P(_Local), P(_Coupling), P(_State),
                                      P(_ConvState), P(_Tensor), P(_State), P(_ConvState), P(_Launch)]
    lib.rlm_mixer_decode.argtypes = [P(_Tensor), P(_Tensor), P(_State), P(_Local), P(_Coupling), P(_ConvState),
                                     P(_Tensor), P(_Launch)]
    lib.rlm_state_init.argtypes = [P(_State), P(_Params), P(_Launch)]
    lib.rlm_validate_params.argtypes = [P(_Params)]
    lib.rlm_get_device_status.argtypes = [P(_Launch)]
    lib.rlm_test_stall_segments.argtypes = [ctypes.c_int]
    for f in ("rlm_prefill_workspace_size", "rlm_backward_workspace_size"):
        getattr(lib, f).argtypes = [ctypes.c_int64, ctypes.c_int64, ctypes.c_int,
                                    ctypes.c_int, ctypes.c_int]
        getattr(lib, f).restype = ctypes.c_size_t
    for f in ("rlm_mix_prefill", "rlm_mix_prefill_from", "rlm_mix_decode", "rlm_mix_backward",
              "rlm_mix_backward_from", "rlm_mixer_prefill", "rlm_mixer_decode", "rlm_state_init",
              "rlm_validate_params", "rlm_get_device_status"):
        getattr(lib, f).restype = ctypes.c_int
    lib.rlm_status_string.argtypes = [ctypes.c_int]
    lib.rlm_status_string.restype = ctypes.c_char_p
    lib.rlm_last_error.restype = ctypes.c_char_p
    lib.rlm_version.restype = ctypes.c_int
    lib.rlm_kernels_launched.restype = ctypes.c_ulonglong
    lib.rlm_mix_prefill_noalloc.argtypes = [P(_Tensor), P(_Params), P(_Tensor), P(_State),
                                            ctypes.c_void_p]
    lib.rlm_mix_prefill_noalloc.restype = ctypes.c_int
    _lib = lib
    return lib


# --------------------------------------------------------------- containers
@dataclass
class Params:
    """Resonator parameters, each a float32 CUDA tensor [D][M]."""
    decay: torch.Tensor
    freq: torch.Tensor
    amp: torch.Tensor
    phase: torch.Tensor

    @property
    def D(self) -> int:
        return int(self.decay.shape[0])

    @property
    def M(self) -> int:
        return int(self.decay.shape[1])

    @classmethod
    def from_arrays(cls, decay, freq, amp, phase, device="cuda"):
        t = lambda a: torch.as_tensor(a, dtype=torch.float32).contiguous().to(device)
        return cls(t(decay), t(freq), t(amp), t(phase))

    @classmethod
    def tied_heads(cls, decay, freq, phase, d_h: int, device="cuda"):
        """The paper's parameterisation (Sec. 3.1): one damped mode per head, no
        amplitude (A = 1), shared by the head's d_h channels (head-major).  decay,
        freq, phase: [H].  Gives [H * d_h][1] parameters, which the bf16 prefill
        runs on its tcgen05 path (M = 1)."""
        t = lambda a: torch.as_tensor(a, dtype=torch.float32).reshape(-1).repeat_interleave(d_h)
        dec, fr, ph = t(decay), t(freq), t(phase)
        amp = torch.ones_like(dec)
        return cls(*(v.reshape(-1, 1).contiguous().to(device) for v in (dec, fr, amp, ph)))

    def _c(self) -> _Params:
        return _Params(*(_ptr(t, torch.float32, 2) for t in
                         (self.decay, self.freq, self.amp, self.phase)), self.D, self.M)


@dataclass
class Grads(Params):
    """Parameter gradients, same layout as Params (overwritten by backward)."""

    @classmethod
    def empty(cls, D: int, M: int, device="cuda"):
        return cls(*(torch.empty(D, M, dtype=torch.float32, device=device) for _ in range(4)))


@dataclass
class State:
    """Recurrent state of Sec. 3.3: s [B][D][M][2] (Re, Im) and coef [D][M][4]."""
    s: torch.Tensor
    coef: torch.Tensor

    @classmethod
    def empty(cls, B: int, D: int, M: int, device="cuda"):
        return cls(torch.empty(B, D, M, 2, dtype=torch.float32, device=device),
                   torch.empty(D, M, 4, dtype=torch.float32, device=device))

    @property
    def shape(self):
        B, D, M, _ = self.s.shape
        return int(B), int(D), int(M)

    def complex(self) -> torch.Tensor:
        return torch.view_as_complex(self.s.contiguous())

    def _c(self) -> _State:
        B, D, M = self.shape
        return _State(_ptr(self.s, torch.float32, 4), _ptr(self.coef, torch.float32, 3), B, D, M)


@dataclass
class Local:
    """Local lexical path of Sec. 3.4: depthwise causal kernel conv_w [D][K] (conv_w[d][k]
    multiplies u_{t-k}) and channel scale [D], both float32 CUDA tensors."""
    conv_w: torch.Tensor
    scale: torch.Tensor

    @property
    def K(self) -> int:
        return int(self.conv_w.shape[1])

    @classmethod
    def from_arrays(cls, conv_w, scale, device="cuda"):
        t = lambda a: torch.as_tensor(a, dtype=torch.float32).contiguous().to(device)
        return cls(t(conv_w), t(scale))

    def _c(self) -> _Local:
        D, K = self.conv_w.shape
        if K == 0:
            return _Local(None, None, int(D), 0)
        return _Local(_ptr(self.conv_w, torch.float32, 2), _ptr(self.scale, torch.float32, 1), int(D), int(K))


@dataclass
class Coupling:
    """Head coupling of Sec. 3.4: raw matrix c_raw [H][H] (float32 CUDA tensor) and
    strength lambda_c; C = I + lambda_c / sqrt(H) tanh(c_raw) mixes the heads of
    head-major channels."""
    c_raw: torch.Tensor
    lambda_c: float

    @classmethod
    def from_arrays(cls, c_raw, lambda_c, device="cuda"):
        return cls(torch.as_tensor(c_raw, dtype=torch.float32).contiguous().to(device), float(lambda_c))

    def _c(self) -> _Coupling:
        H = int(self.c_raw.shape[0])
        return _Coupling(_ptr(self.c_raw, torch.float32, 2), float(self.lambda_c), H)


@dataclass
class ConvState:
    """Drive history of the local path: u [B][K-1][D] in the field's dtype, oldest first."""
    u: torch.Tensor

    @property
    def K(self) -> int:
        return int(self.u.shape[1]) + 1

    @classmethod
    def empty(cls, B: int, D: int, K: int, dtype=torch.bfloat16, device="cuda"):
        return cls(torch.empty(B, max(K - 1, 0), D, dtype=dtype, device=device))

    def _c(self) -> _ConvState:
        if self.u.dtype not in _DT or not self.u.is_cuda or not self.u.is_contiguous() or self.u.dim() != 3:
            raise ValueError("ConvState.u must be a contiguous CUDA [B][K-1][D] float32 or bfloat16 tensor")
        B, K1, D = self.u.shape
        return _ConvState(self.u.data_ptr() if K1 > 0 else None, _DT[self.u.dtype], int(B), int(D), int(K1) + 1)


# --------------------------------------------------------------- marshalling
_DT = {torch.float32: RLM_F32, torch.bfloat16: RLM_BF16}


def _ptr(t: torch.Tensor, dtype, ndim) -> int:
    if not isinstance(t, torch.Tensor):
        raise TypeError("expected a torch.Tensor")
    if t.dtype != dtype or t.dim() != ndim or not t.is_contiguous() or not t.is_cuda:
        raise ValueError(f"expected a contiguous CUDA {dtype} tensor of rank {ndim}, got "
                         f"{t.dtype} {tuple(t.shape)} on {t.device}")
    return t.data_ptr()


def _field(t: torch.Tensor) -> _Tensor:
    if t.dtype not in _DT:
        raise ValueError(f"unsupported dtype {t.dtype}")
    if not t.is_cuda or not t.is_contiguous():
        raise ValueError("fields must be contiguous CUDA tensors")
    if t.dim() == 3:
        B, L, D = t.shape
    elif t.dim() == 2:     # a single token per batch row: [B][D]
        (B, D), L = t.shape, 1
    else:
        raise ValueError(f"fields are [B][L][D] (or [B][D] for one token), got {tuple(t.shape)}")
    return _Tensor(t.data_ptr(), _DT[t.dtype], B, L, D)


def _stream(stream) -> int:
    if stream is None:
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, torch.cuda.Stream):
        return stream.cuda_stream
    return int(stream)


def _launch(stream, workspace) -> _Launch:
    if workspace is None:
        return _Launch(_stream(stream), None, 0)
    return _Launch(_stream(stream), workspace.data_ptr(),
                   workspace.numel() * workspace.element_size())


def _check(status: int, where: str):
    if status != RLM_OK:
        raise RlmError(status, where, load_library().rlm_last_error().decode())


def _workspace(nbytes: int, device) -> torch.Tensor | None:
    if nbytes == 0:
        return None
    return torch.empty(nbytes, dtype=torch.uint8, device=device)


# --------------------------------------------------------------- entry points
def rlm_status_string(status: int) -> str:
    return load_library().rlm_status_string(status).decode()


def rlm_version() -> int:
    return load_library().rlm_version()


def rlm_kernels_launched() -> int:
    """Kernels the library has launched in this process (host-side count)."""
    return int(load_library().rlm_kernels_launched())


def rlm_prefill_workspace_size(B: int, L: int, D: int, M: int, dtype) -> int:
    return load_library().rlm_prefill_workspace_size(B, L, D, M, _DT.get(dtype, dtype))


def rlm_backward_workspace_size(B: int, L: int, D: int, M: int, dtype) -> int:
    return load_library().rlm_backward_workspace_size(B, L, D, M, _DT.get(dtype, dtype))


def rlm_mix_prefill(x: torch.Tensor, params: Params, y: torch.Tensor,
                    state_out: State | None = None, workspace: torch.Tensor | None = None,
                    stream=None) -> None:
    """Causal mixing y = K * x (Eq. 2) from a zero state; optional terminal state.

    ``workspace`` defaults to a fresh buffer of rlm_prefill_workspace_size bytes."""
    lib = load_library()
    xt, yt = _field(x), _field(y)
    if workspace is None:
        workspace = _workspace(lib.rlm_prefill_workspace_size(xt.B, xt.L, xt.D, params.M, xt.dtype),
                               x.device)
    st = state_out._c() if state_out is not None else None
    _check(lib.rlm_mix_prefill(ctypes.byref(xt), ctypes.byref(params._c()), ctypes.byref(yt),
                               ctypes.byref(st) if st is not None else None,
                               ctypes.byref(_launch(stream, workspace))), "rlm_mix_prefill")


def rlm_mix_prefill_from(x: torch.Tensor, params: Params, state_in: State | None, y: torch.Tensor,
                         state_out: State | None = None, workspace: torch.Tensor | None = None,
                         stream=None) -> None:
    """Causal mixing from an initial state (chunked or continued prefill): y = K * x
    plus the free response of ``state_in`` (its ``s``; None = zero state).
    ``state_out`` may be ``state_in`` itself (in-place continuation)."""
    lib = load_library()
    xt, yt = _field(x), _field(y)
    if workspace is None:
        workspace = _workspace(lib.rlm_prefill_workspace_size(xt.B, xt.L, xt.D, params.M, xt.dtype),
                               x.device)
    si = state_in._c() if state_in is not None else None
    so = state_out._c() if state_out is not None else None
    _check(lib.rlm_mix_prefill_from(ctypes.byref(xt), ctypes.byref(params._c()),
                                    ctypes.byref(si) if si is not None else None, ctypes.byref(yt),
                                    ctypes.byref(so) if so is not None else None,
                                    ctypes.byref(_launch(stream, workspace))), "rlm_mix_prefill_from")


def rlm_mix_prefill_noalloc(x: torch.Tensor, params: Params, y: torch.Tensor,
                            state_out: State | None = None, stream=None) -> None:
    """rlm_mix_prefill without a workspace, for callers that cannot allocate device
    memory: the scratch is the library's fixed 64 MiB device array (see rlm.h).
    Calls that overlap on the GPU race on that array."""
    lib = load_library()
    xt, yt = _field(x), _field(y)
    st = state_out._c() if state_out is not None else None
    _check(lib.rlm_mix_prefill_noalloc(ctypes.byref(xt), ctypes.byref(params._c()),
                                       ctypes.byref(yt),
                                       ctypes.byref(st) if st is not None else None,
                                       _stream(stream)), "rlm_mix_prefill_noalloc")


def rlm_mix_decode(x_t: torch.Tensor, state: State, y_t: torch.Tensor, stream=None) -> None:
    """One decode step (Eq. 4-5); the state is updated in place."""
    lib = load_library()
    xt, yt = _field(x_t), _field(y_t)
    _check(lib.rlm_mix_decode(ctypes.byref(xt), ctypes.byref(state._c()), ctypes.byref(yt),
                              ctypes.byref(_launch(stream, None))), "rlm_mix_decode")


def rlm_state_init(state: State, params: Params, stream=None) -> None:
    lib = load_library()
    _check(lib.rlm_state_init(ctypes.byref(state._c()), ctypes.byref(params._c()),
                              ctypes.byref(_launch(stream, None))), "rlm_state_init")


def rlm_mix_backward(dy: torch.Tensor, x: torch.Tensor, params: Params, dx: torch.Tensor,
                     dparams: Grads, workspace: torch.Tensor | None = None, stream=None) -> None:
    """dx and the four parameter gradients of l given dy = dl/dy."""
    lib = load_library()
    dyt, xt, dxt = _field(dy), _field(x), _field(dx)
    if workspace is None:
        workspace = _workspace(lib.rlm_backward_workspace_size(xt.B, xt.L, xt.D, params.M,
                                                               xt.dtype), x.device)
    _check(lib.rlm_mix_backward(ctypes.byref(dyt), ctypes.byref(xt), ctypes.byref(params._c()),
                                ctypes.byref(dxt), ctypes.byref(dparams._c()),
                                ctypes.byref(_launch(stream, workspace))), "rlm_mix_backward")


def rlm_mix_backward_from(dy: torch.Tensor, x: torch.Tensor, params: Params, state_in: State | None,
                          d_state_out: State | None, dx: torch.Tensor, dparams: Grads,
                          d_state_in: State | None = None, workspace: torch.Tensor | None = None,
                          stream=None) -> None:
    """Backward of rlm_mix_prefill_from: dx, the parameter gradients and (if
    ``d_state_in`` is given) the gradient of the initial state, for a loss that may
    also depend on the terminal state (its gradient ``d_state_out``).  Only the
    ``s`` buffers of the state arguments are used."""
    lib = load_library()
    dyt, xt, dxt = _field(dy), _field(x), _field(dx)
    if workspace is None:
        workspace = _workspace(lib.rlm_backward_workspace_size(xt.B, xt.L, xt.D, params.M, xt.dtype),
                               x.device)
    opt = lambda st: ctypes.byref(st._c()) if st is not None else None
    _check(lib.rlm_mix_backward_from(ctypes.byref(dyt), ctypes.byref(xt), ctypes.byref(params._c()),
                                     opt(state_in), opt(d_state_out), ctypes.byref(dxt),
                                     ctypes.byref(dparams._c()), opt(d_state_in),
                                     ctypes.byref(_launch(stream, workspace))), "rlm_mix_backward_from")


def rlm_validate_params(params: Params) -> None:
    _check(load_library().rlm_validate_params(ctypes.byref(params._c())), "rlm_validate_params")


def rlm_get_device_status(stream=None) -> int:
    """Synchronise the stream and return (and clear) the device status word."""
    return load_library().rlm_get_device_status(ctypes.byref(_launch(stream, None)))


def rlm_mixer_prefill(x: torch.Tensor, g: torch.Tensor | None, params: Params, local: Local | None,
                      z: torch.Tensor, state_in: State | None = None, conv_in: ConvState | None = None,
                      state_out: State | None = None, conv_out: ConvState | None = None,
                      workspace: torch.Tensor | None = None, stream=None,
                      coupling: Coupling | None = None) -> None:
    """Mixer output of Sec. 3.4 over a sequence: z = sigmoid(g) * y + s * (w * x), y the
    resonant mixing of x from ``state_in``; the local path reads its drives before
    token 0 from ``conv_in``.  ``state_out`` / ``conv_out`` receive the terminal
    state and drive history (each may be its input, for in-place continuation)."""
    lib = load_library()
    xt, zt = _field(x), _field(z)
    gt = _field(g) if g is not None else None
    if workspace is None:
        workspace = _workspace(lib.rlm_prefill_workspace_size(xt.B, xt.L, xt.D, params.M, xt.dtype),
                               x.device)
    ref = lambda c: ctypes.byref(c) if c is not None else None
    opt = lambda o: ref(o._c()) if o is not None else None
    _check(lib.rlm_mixer_prefill(ctypes.byref(xt), ref(gt), ctypes.byref(params._c()), opt(local), opt(coupling),
                                 opt(state_in),
                                 opt(conv_in), ctypes.byref(zt), opt(state_out), opt(conv_out),
                                 ctypes.byref(_launch(stream, workspace))), "rlm_mixer_prefill")


def rlm_mixer_decode(x_t: torch.Tensor, g_t: torch.Tensor | None, state: State, local: Local | None,
                     conv: ConvState | None, z_t: torch.Tensor, stream=None, coupling: Coupling | None = None) -> None:
    """One mixer decode step: recurrence, gate and local path in one kernel; the state
    and the drive history advance in place."""
    lib = load_library()
    xt, zt = _field(x_t), _field(z_t)
    gt = _field(g_t) if g_t is not None else None
    ref = lambda c: ctypes.byref(c) if c is not None else None
    opt = lambda o: ref(o._c()) if o is not None else None
    _check(lib.rlm_mixer_decode(ctypes.byref(xt), ref(gt), ctypes.byref(state._c()), opt(local), opt(coupling),
                                opt(conv),
                                ctypes.byref(zt), ctypes.byref(_launch(stream, None))), "rlm_mixer_decode")
