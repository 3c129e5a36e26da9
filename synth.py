"""Seeded synthetic inputs for causal resonant field mixing.

Shared by the tests, the benchmark and the smoke check; used identically for
the CUDA path and the CPU oracle.  This module holds none of the operator's
arithmetic: it only draws random numbers and rounds them to the storage dtype.

Draw order (numpy ``default_rng(seed)``, PCG64), fixed so that every consumer
sees the same buffers: x, decay, freq, amp, phase, dy, decode tokens.

Distributions follow the paper's 6M-parameter workload as generalised to M
modes per channel:
  x ~ N(0,1); decay gamma ~ U[0.001, 0.1] (half-lives 6.9-693 tokens, inside
  the 2-2048 range of Table 2); frequency omega ~ U[0, pi]; amplitude
  A ~ N(0, 1/M) (variance 1/M); phase phi ~ U[0, 2 pi); dy ~ N(0,1).
The paper's corpora (WikiText-2/103, TinyStories) are not used: the operator's
cost and numerics do not depend on the data beyond these shapes and scales.
"""
from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np


def round_to_bf16(a: np.ndarray) -> np.ndarray:
    """Round float32 values to the nearest bfloat16 (ties to even); float32 out."""
    a = np.ascontiguousarray(a, dtype=np.float32)
    u = a.view(np.uint32).astype(np.uint64)
    r = ((u + 0x7FFF + ((u >> 16) & 1)) >> 16) << 16
    out = r.astype(np.uint32).view(np.float32)
    nan = np.isnan(a)
    if nan.any():
        out = out.copy()
        out[nan] = np.float32("nan")
    return out


def to_bf16_bits(a: np.ndarray) -> np.ndarray:
    """uint16 bit patterns of float32 values that are already bf16-representable."""
    a = np.ascontiguousarray(a, dtype=np.float32)
    return (a.view(np.uint32) >> 16).astype(np.uint16)


@dataclass
class Inputs:
    B: int
    L: int
    D: int
    M: int
    dtype: str               # storage dtype of x / y / dy / dx: "f32" or "bf16"
    x: np.ndarray            # [B][L][D] float32 (bf16-representable when dtype == "bf16")
    decay: np.ndarray        # [D][M] float32
    freq: np.ndarray
    amp: np.ndarray
    phase: np.ndarray
    dy: np.ndarray | None = None          # [B][L][D]
    tokens: np.ndarray | None = None      # [T][B][D] decode tokens
    extra: dict = field(default_factory=dict)

    def params(self):
        return self.decay, self.freq, self.amp, self.phase


def make_inputs(B: int, L: int, D: int, M: int, dtype: str = "bf16", seed: int = 0,
                with_dy: bool = False, decode_steps: int = 0,
                decay_range=(0.001, 0.1)) -> Inputs:
    """Draw one seeded problem instance (see module docstring for the recipe)."""
    if dtype not in ("f32", "bf16"):
        raise ValueError(dtype)
    rng = np.random.default_rng(seed)
    x = rng.standard_normal((B, L, D), dtype=np.float32)
    decay = rng.uniform(decay_range[0], decay_range[1], (D, M)).astype(np.float32)
    freq = rng.uniform(0.0, np.pi, (D, M)).astype(np.float32)
    amp = (rng.standard_normal((D, M)) / np.sqrt(M)).astype(np.float32)
    phase = rng.uniform(0.0, 2.0 * np.pi, (D, M)).astype(np.float32)
    dy = rng.standard_normal((B, L, D), dtype=np.float32) if with_dy else None
    tokens = (rng.standard_normal((decode_steps, B, D), dtype=np.float32)
              if decode_steps else None)
    if dtype == "bf16":
        x = round_to_bf16(x)
        dy = round_to_bf16(dy) if dy is not None else None
        tokens = round_to_bf16(tokens) if tokens is not None else None
    return Inputs(B, L, D, M, dtype, x, decay, freq, amp, phase, dy, tokens)


@dataclass
class MixerInputs:
    """The mixer wrapper's extra inputs around the resonant operator (Sec. 3.4):
    the gate pre-activation g (the gate half of the grouped input projection), the
    local path's depthwise causal kernel w and its channel scale s, and the drive
    history and gate of decode steps."""
    K: int
    g: np.ndarray            # [B][L][D] float32 (bf16-representable for bf16 I/O)
    conv_w: np.ndarray       # [D][K] float32
    scale: np.ndarray        # [D] float32
    conv_in: np.ndarray      # [B][K-1][D] float32: drives before token 0
    g_tokens: np.ndarray | None = None   # [T][B][D] gate of decode steps


def make_mixer_inputs(inp: Inputs, K: int, seed: int = 0) -> MixerInputs:
    """Draw the mixer's extra inputs for an Inputs instance, from a generator of
    their own (default_rng([seed, 1])) so the operator's draws are unchanged.
    g ~ N(0, 1); w ~ N(0, 1/K) (variance 1/K, unit-variance output for unit
    drives); s ~ U[0.5, 1.5]; the drive history ~ N(0, 1); decode-step gates
    ~ N(0, 1), one per decode token of inp."""
    rng = np.random.default_rng([seed, 1])
    B, L, D = inp.B, inp.L, inp.D
    g = rng.standard_normal((B, L, D), dtype=np.float32)
    conv_w = (rng.standard_normal((D, max(K, 0))) / np.sqrt(max(K, 1))).astype(np.float32)
    scale = rng.uniform(0.5, 1.5, D).astype(np.float32)
    conv_in = rng.standard_normal((B, max(K - 1, 0), D), dtype=np.float32)
    T = 0 if inp.tokens is None else inp.tokens.shape[0]
    g_tokens = rng.standard_normal((T, B, D), dtype=np.float32) if T else None
    if inp.dtype == "bf16":
        g = round_to_bf16(g)
        conv_in = round_to_bf16(conv_in)
        g_tokens = round_to_bf16(g_tokens) if g_tokens is not None else None
    return MixerInputs(K, g, conv_w, scale, conv_in, g_tokens)


# The workloads, named by what they are (B, L, D, M, dtype).
WORKLOADS = {
    "tiny_f32_prefill": dict(B=1, L=256, D=64, M=4, dtype="f32"),
    "layer6m_prefill": dict(B=8, L=2048, D=256, M=16, dtype="bf16"),
    "long_prefill_b1_8k": dict(B=1, L=8192, D=256, M=16, dtype="bf16"),
    "long_prefill_b1_16k": dict(B=1, L=16384, D=256, M=16, dtype="bf16"),
    "long_prefill_b1_32k": dict(B=1, L=32768, D=256, M=16, dtype="bf16"),
    "long_prefill_b4_8k": dict(B=4, L=8192, D=256, M=16, dtype="bf16"),
    "long_prefill_b4_16k": dict(B=4, L=16384, D=256, M=16, dtype="bf16"),
    "long_prefill_b4_32k": dict(B=4, L=32768, D=256, M=16, dtype="bf16"),
    "train_b4_32k_d512_m32": dict(B=4, L=32768, D=512, M=32, dtype="bf16"),
}
