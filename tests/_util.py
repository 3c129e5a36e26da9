"""Helpers shared by the GPU tests (comparison metrics and tensor transfer)."""
import numpy as np

# Tolerances of the operator's parity bar: relative error <= 1e-4 for fp32 I/O and
# <= 2e-2 for bf16 I/O with fp32 state, each measured both as ||d||_2/||ref||_2 and
# as max|d|/max|ref| per output tensor.
TOL = {"f32": 1e-4, "bf16": 2e-2}


def rel_errors(got, ref):
    got = np.asarray(got, np.float64)
    ref = np.asarray(ref, np.float64)
    d = got - ref
    l2 = np.linalg.norm(d) / max(np.linalg.norm(ref), 1e-300)
    mx = np.abs(d).max() / max(np.abs(ref).max(), 1e-300) if d.size else 0.0
    return float(l2), float(mx)


def assert_close(got, ref, tol, what=""):
    l2, mx = rel_errors(got, ref)
    assert l2 <= tol and mx <= tol, f"{what}: l2 rel {l2:.3e}, max rel {mx:.3e} > {tol}"
    return l2, mx


def torch_dtype(dtype):
    import torch
    return torch.bfloat16 if dtype == "bf16" else torch.float32


def to_dev(a, dtype, device="cuda"):
    import torch
    return torch.from_numpy(np.ascontiguousarray(a)).to(device=device, dtype=torch_dtype(dtype))


def to_np(t):
    return t.float().cpu().numpy().astype(np.float64)
