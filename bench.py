"""Benchmark of the causal resonant field mixing operator on GB300.

Headline (``value``): prefill throughput in Mtok/s at L = 32768 on the long-context
workload (B=4, L=32768, D=256, M=16, bf16 I/O, fp32 state), inputs resident in HBM,
L2 flushed (a 512 MiB write) before every timed step.  One step = one
rlm_mix_prefill call: parameter precompute, intra-chunk Toeplitz contraction,
inter-chunk carry, state up-projection, epilogue and terminal state.

Also reported on the same line:
  decode    4096 single-token rlm_mix_decode steps at B=64 (D=256, M=16) after a
            32768-token prefill, captured in a CUDA graph; tok/s and % of HBM.
  backward  rlm_mix_backward at B=4, L=32768, D=512, M=32 (bf16 I/O), with the
            training step's forward (rlm_mix_prefill) on the same shape.
  roofline  achieved algorithmic GB/s of the prefill against the measured HBM peak.
  e2e       the same prefill metric through the C ABI with pinned HOST buffers
            (host->device copy of x and device->host copy of y inside the timing).
  cpu_baseline  the fp64 CPU oracle (sequential recurrence) on the host cores.

``--impl reference`` times the CPU oracle itself as the reference arm.
``--only backward`` runs only the backward measurement and prints its object
(a diagnostic mode for profiling that path; not the benchmark line).
Multi-GPU (torchrun, N > 1): every rank runs its own independent batch of the
same workload (weak scaling, replicas only; the operator has no cross-GPU
exchange); rank 0 prints value = all ranks' tokens / max time over ranks.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "mix prefill Mtok/s at L=32K (% of roofline); decode tok/s at B=64 (% HBM)"
PREFILL = dict(B=4, L=32768, D=256, M=16)
DECODE = dict(B=64, L=32768, D=256, M=16, T=4096)
BACKWARD = dict(B=4, L=32768, D=512, M=32)
MIXER = dict(B=4, L=32768, D=256, M=16, K=4, H=8, decode_B=64, T=4096)
L2_FLUSH_BYTES = 512 << 20


def _peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            pk = json.load(f)
        return float(pk["hbm_gbs"]), float(pk["bf16_tflops"]), "measured"
    except Exception:
        return 6800.0, 1900.0, "fallback"


def prefill_bytes(B, L, D, M, elem=2):
    """Algorithmic HBM bytes of one prefill: read x, write y (elem = 2 B each per
    token-channel in bf16, 4 in fp32), write the terminal state (8 B per (b,d,m))
    and its coefficients (16 B per (d,m)), read the parameters (16 B per (d,m))."""
    return B * L * D * 2 * elem + B * D * M * 8 + D * M * 32


def decode_bytes(B, D, M):
    """Per decode step: state read+write (16 B per (b,d,m)), token in and out
    (bf16, 4 B per (b,d)), coefficients (16 B per (d,m))."""
    return 16 * B * D * M + 4 * B * D + 16 * D * M


def mixer_prefill_bytes(B, L, D, M, K):
    """Algorithmic HBM bytes of one mixer prefill (Sec. 3.4): read x and g, write z
    (bf16, 6 B per token-channel), the state and parameters as for the prefill,
    and with a local path (K > 0) the drive history in and out (2 B per (b, k, d))
    and its weights (4 B per (d, k) and per d)."""
    extra = 2 * 2 * B * (K - 1) * D + 4 * D * (K + 1) if K > 0 else 0
    return prefill_bytes(B, L, D, M) + 2 * B * L * D + extra


def mixer_decode_bytes(B, D, M, K):
    """Per mixer decode step: the decode step's bytes, the gate (2 B per (b,d)),
    the drive history read and written (4 B per (b, k, d)) and the weights."""
    return decode_bytes(B, D, M) + 2 * B * D + 4 * B * (K - 1) * D + 4 * D * (K + 1)


def backward_bytes(B, L, D, M):
    """Per backward call: read x and dy, write dx (bf16, 6 B per token-channel),
    read params and write four gradients (32 B per (d,m))."""
    return 6 * B * L * D + 32 * D * M


def backward_moved_bytes(B, L, D):
    """DRAM bytes the tensor-core backward's data path moves per call (bf16,
    L a multiple of 2048): the transpose of x and dy to channel-major (read 4 B,
    write 4 B per token-channel), the tcgen05 kernel (read 4 B, write 2 B) and
    the transpose of dx back (read 2 B, write 2 B): 18 B per token-channel."""
    return 18 * B * L * D


# ---------------------------------------------------------------- clocks
class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index=0):
        self.gpu = gpu_index
        self.proc = None
        self.lines = []

    def __enter__(self):
        cmd = ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}",
               "--format=csv,noheader,nounits", "-lms", "200"]
        try:
            # nvidia-smi block-buffers into a pipe; stdbuf makes it line-buffered.
            import shutil
            if shutil.which("stdbuf"):
                cmd = ["stdbuf", "-oL"] + cmd
            self.proc = subprocess.Popen(cmd, stdout=subprocess.PIPE, stderr=subprocess.DEVNULL,
                                         text=True)
            self._t = threading.Thread(target=self._read, daemon=True)
            self._t.start()
        except Exception:
            self.proc = None
        return self

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def __exit__(self, *a):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self):
        sm, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            parts = [p.strip() for p in ln.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                mx = float(parts[2])
            except ValueError:
                continue
            for nm, v in zip(names, parts[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(nm)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": mx, "reasons": [], "samples": 0}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": mx, "reasons": sorted(reasons),
                "samples": len(sm)}


# ---------------------------------------------------------------- helpers
def _dist():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def _barrier_max(t, ws):
    """Maximum of t over the ranks (the job's step time is its slowest rank's)."""
    if ws == 1:
        return t
    import torch
    import torch.distributed as dist
    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    v = torch.tensor([t], dtype=torch.float64, device=dev)
    dist.all_reduce(v, op=dist.ReduceOp.MAX)
    return float(v.item())


def _barrier(ws):
    if ws > 1:
        import torch.distributed as dist
        dist.barrier()


def _traffic_from_profiles(kernel_tag):
    """DRAM bytes per launch recorded in profiles/<kernel_tag>.md, valid only while
    the kernel source hash recorded there matches the current source."""
    import hashlib
    path = os.path.join(ROOT, "profiles", f"{kernel_tag}.md")
    if not os.path.exists(path):
        return None
    kv = {}
    for line in open(path):
        if line.startswith("- ") and ":" in line:
            k, v = line[2:].split(":", 1)
            kv[k.strip()] = v.strip().strip("`")
    src = kv.get("source")
    if not src or "dram_bytes_per_full_launch" not in kv:
        return None
    try:
        h = hashlib.sha256(open(os.path.join(ROOT, src), "rb").read()).hexdigest()[:16]
    except OSError:
        return None
    if h != kv.get("source_sha256_16"):
        return None
    return float(kv["dram_bytes_per_full_launch"])


# ---------------------------------------------------------------- our arm
def run_ours(args):
    import torch

    import paper_2607_05583_gb300 as rlm
    from synth import make_inputs

    ws, rank, local = _dist()
    torch.cuda.set_device(local)
    if ws > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl")
    dev = torch.device("cuda", local)
    rlm.load_library()
    hbm_peak, bf16_peak, peak_kind = _peaks()
    stream = torch.cuda.current_stream()

    # ---------------- prefill (headline)
    P = PREFILL
    inp = make_inputs(P["B"], P["L"], P["D"], P["M"], "bf16", seed=rank)
    x = torch.from_numpy(inp.x).to(dev, torch.bfloat16)
    params = rlm.Params.from_arrays(*inp.params(), device=dev)
    y = torch.empty_like(x)
    st = rlm.State.empty(P["B"], P["D"], P["M"], device=dev)
    wsz = rlm.rlm_prefill_workspace_size(P["B"], P["L"], P["D"], P["M"], torch.bfloat16)
    work = torch.empty(max(wsz, 256), dtype=torch.uint8, device=dev)
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=dev)

    def step():
        rlm.rlm_mix_prefill(x, params, y, st, workspace=work)

    for _ in range(args.warmup):
        flush.zero_()
        step()
    torch.cuda.synchronize()
    starts = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    ends = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    with ClockSampler(local) as clk:
        # The clock sampler (200 ms period) needs a loaded GPU for longer than the
        # timed steps last: soak with the same kernel first, then time.
        t_end = time.perf_counter() + args.soak
        while time.perf_counter() < t_end:
            for _ in range(20):
                step()
            torch.cuda.synchronize()
        _barrier(ws)
        torch.cuda.synchronize()
        n0 = rlm.rlm_kernels_launched()
        for i in range(args.steps):
            flush.zero_()
            starts[i].record(stream)
            step()
            ends[i].record(stream)
        torch.cuda.synchronize()
        n_launch = rlm.rlm_kernels_launched() - n0
    _barrier(ws)
    times = [s.elapsed_time(e) for s, e in zip(starts, ends)]
    ms = statistics.mean(times)
    ms_max = _barrier_max(ms, ws)
    tokens = P["B"] * P["L"]
    value = ws * tokens / (ms_max * 1e-3) / 1e6
    alg = prefill_bytes(P["B"], P["L"], P["D"], P["M"])
    achieved = alg / (ms * 1e-3) / 1e9
    roofline = {"bound": "hbm", "achieved": round(achieved, 1), "peak": hbm_peak,
                "unit": "GB/s", "frac": round(achieved / hbm_peak, 4),
                "traffic": _traffic_from_profiles("prefill_tc_long_b4_32k"),
                "peak_kind": peak_kind, "frac_of_8TBps": round(achieved / 8000.0, 4),
                "algorithmic_bytes_per_launch": alg,
                "kernel": "rlm_mix_prefill (whole call)", "median_ms": statistics.median(times)}

    # ---------------- e2e through the C ABI with host buffers
    # Every step copies its input from pinned host memory, runs the prefill and
    # copies its output back.  Consecutive steps overlap as a serving pipeline
    # would: the copy-in, the prefill and the copy-out run on their own streams
    # over two device buffer pairs, ordered by events (buffer k is refilled only
    # after the prefill two steps back has read it, and rewritten only after its
    # output has been copied out).
    xh = torch.from_numpy(inp.x).to(torch.bfloat16).pin_memory()
    yhs = [torch.empty_like(xh).pin_memory() for _ in range(2)]
    xs, ys = [x, torch.empty_like(x)], [y, torch.empty_like(y)]
    s_in, s_comp, s_out = torch.cuda.Stream(), torch.cuda.Stream(), torch.cuda.Stream()
    ev_in = [torch.cuda.Event() for _ in range(2)]
    ev_comp = [torch.cuda.Event() for _ in range(2)]
    ev_out = [torch.cuda.Event() for _ in range(2)]

    def e2e_steps(n):
        for ev in ev_comp + ev_out:
            ev.record(stream)
        for s_ in (s_in, s_comp, s_out):
            s_.wait_stream(stream)
        for i in range(n):
            k = i % 2
            s_in.wait_event(ev_comp[k])
            with torch.cuda.stream(s_in):
                xs[k].copy_(xh, non_blocking=True)
            ev_in[k].record(s_in)
            s_comp.wait_event(ev_in[k])
            s_comp.wait_event(ev_out[k])
            rlm.rlm_mix_prefill(xs[k], params, ys[k], st, workspace=work, stream=s_comp)
            ev_comp[k].record(s_comp)
            s_out.wait_event(ev_comp[k])
            with torch.cuda.stream(s_out):
                yhs[k].copy_(ys[k], non_blocking=True)
            ev_out[k].record(s_out)
        for s_ in (s_in, s_comp, s_out):
            stream.wait_stream(s_)

    e2e_steps(3)
    torch.cuda.synchronize()
    reps = max(6, args.steps // 2)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    e2e_steps(reps)
    e1.record(stream)
    torch.cuda.synchronize()
    e2e_ms = e0.elapsed_time(e1) / reps
    # The same schedule without the prefill: what the host link alone allows with
    # both directions busy (the bound on e2e; the prefill hides under the copies).
    def copy_steps(n):
        for s_ in (s_in, s_out):
            s_.wait_stream(stream)
        for i in range(n):
            k = i % 2
            with torch.cuda.stream(s_in):
                xs[k].copy_(xh, non_blocking=True)
            with torch.cuda.stream(s_out):
                yhs[k].copy_(ys[k], non_blocking=True)
        for s_ in (s_in, s_out):
            stream.wait_stream(s_)

    copy_steps(3)
    torch.cuda.synchronize()
    e0.record(stream)
    copy_steps(reps)
    e1.record(stream)
    torch.cuda.synchronize()
    copy_ms = e0.elapsed_time(e1) / reps
    e2e = {"value": round(tokens / (e2e_ms * 1e-3) / 1e6, 2), "unit": "Mtok/s",
           "h2d_bytes_per_step": xh.numel() * 2, "d2h_bytes_per_step": yhs[0].numel() * 2,
           "schedule": "copy-in, prefill and copy-out of consecutive steps overlapped on three streams",
           "copy_only_ms_per_step": round(copy_ms, 4),
           "link_GBps_each_way": round(xh.numel() * 2 / (copy_ms * 1e-3) / 1e9, 1),
           "frac_of_copy_only": round(copy_ms / e2e_ms, 4)}
    del xh, yhs, xs, ys

    # ---------------- per-L sweep (same launch configuration)
    sweep = {}
    if not args.quick:
        for (B, L) in ((1, 8192), (1, 16384), (1, 32768), (4, 8192), (4, 16384)):
            sweep[f"B{B}_L{L}"] = _time_prefill(rlm, torch, dev, B, L, P["D"], P["M"], flush,
                                                hbm_peak, reps=max(5, args.steps // 2))
        # the 6M layer's prefill (B = 8, L = 2048)
        sweep["layer6m_B8_L2048"] = _time_prefill(rlm, torch, dev, 8, 2048, P["D"], P["M"], flush,
                                                  hbm_peak, reps=max(5, args.steps // 2))
        # fp32 I/O on the headline shape (the fp32 tcgen05 prefill; 8 B per token-channel)
        sweep[f"fp32_B{P['B']}_L{P['L']}"] = _time_prefill(rlm, torch, dev, P["B"], P["L"], P["D"], P["M"],
                                                           flush, hbm_peak, reps=max(5, args.steps // 2),
                                                           dtype="f32")
    sweep[f"B{P['B']}_L{P['L']}"] = {"Mtok_s": round(tokens / (ms * 1e-3) / 1e6, 1),
                                     "frac": roofline["frac"]}
    del x, y, work

    # ---------------- decode
    decode = None if args.quick else _bench_decode(rlm, torch, dev, hbm_peak)
    if decode is not None:
        decode["other_batch_sizes"] = {f"B{b}": {k: v for k, v in _bench_decode(rlm, torch, dev, hbm_peak, B=b).items()
                                                 if k in ("tok_s", "us_per_step", "frac_hbm")}
                                       for b in (1, 8)}
        decode["large_batch"] = _bench_decode_large_batch(rlm, torch, dev, hbm_peak)
    # ---------------- backward
    backward = None if args.quick else _bench_backward(rlm, torch, dev, hbm_peak, args, flush)
    # ---------------- mixer wrapper (gate + local path, fused)
    mixer = None if args.quick else _bench_mixer(rlm, torch, dev, hbm_peak, flush, ms)
    # ---------------- the paper's tied heads, and its FFT evaluation as the comparison
    paper_form = None if args.quick else _bench_tied_and_fft(rlm, torch, dev, hbm_peak, flush)

    cpu = None
    if rank == 0 and ws == 1 and not args.no_cpu:
        cpu = cpu_baseline(seconds=args.cpu_seconds)

    if rank == 0:
        line = {
            "metric": METRIC, "value": round(value, 2), "unit": "Mtok/s", "n_gpus": ws,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms_max, 5),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "bf16", "data": "synthetic (seeded N(0,1) drives, paper-range resonator params)",
            "config": {"workload": "long-context prefill B=4 L=32768 D=256 M=16 bf16 I/O fp32 state",
                       "B": P["B"], "L": P["L"], "D": P["D"], "M": P["M"],
                       "parallelism": f"replicas x{ws}" if ws > 1 else "single GPU",
                       "l2": "flushed (512 MiB write) before every timed step"},
            "roofline": roofline, "cpu_baseline": cpu, "e2e": e2e,
            "gpu_launches": n_launch,
            "clocks": clk.summary(), "sweep": sweep, "decode": decode, "backward": backward, "mixer": mixer,
            "paper_form": paper_form,
        }
        print(json.dumps(line), flush=True)
    if ws > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


def _time_prefill(rlm, torch, dev, B, L, D, M, flush, hbm_peak, reps=5, dtype="bf16"):
    from synth import make_inputs
    inp = make_inputs(B, L, D, M, dtype, seed=1)
    x = torch.from_numpy(inp.x).to(dev, torch.bfloat16 if dtype == "bf16" else torch.float32)
    p = rlm.Params.from_arrays(*inp.params(), device=dev)
    y = torch.empty_like(x)
    st = rlm.State.empty(B, D, M, device=dev)
    wsz = rlm.rlm_prefill_workspace_size(B, L, D, M, x.dtype)
    work = torch.empty(max(wsz, 256), dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream()
    for _ in range(3):
        rlm.rlm_mix_prefill(x, p, y, st, workspace=work)
    ts = []
    for _ in range(reps):
        flush.zero_()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        rlm.rlm_mix_prefill(x, p, y, st, workspace=work)
        b.record(stream)
        torch.cuda.synchronize()
        ts.append(a.elapsed_time(b))
    ms = statistics.mean(ts)
    gbs = prefill_bytes(B, L, D, M, 2 if dtype == "bf16" else 4) / (ms * 1e-3) / 1e9
    return {"Mtok_s": round(B * L / (ms * 1e-3) / 1e6, 1), "ms": round(ms, 5),
            "frac": round(gbs / hbm_peak, 4)}


def _bench_decode(rlm, torch, dev, hbm_peak, B=None):
    from synth import make_inputs
    P = DECODE
    B = P["B"] if B is None else B
    L, D, M, T = P["L"], P["D"], P["M"], P["T"]
    inp = make_inputs(B, L, D, M, "bf16", seed=0, decode_steps=T)
    x = torch.from_numpy(inp.x).to(dev, torch.bfloat16)
    p = rlm.Params.from_arrays(*inp.params(), device=dev)
    y = torch.empty_like(x)
    st = rlm.State.empty(B, D, M, device=dev)
    rlm.rlm_mix_prefill(x, p, y, st)
    del x, y
    toks = torch.from_numpy(inp.tokens).to(dev, torch.bfloat16)     # [T][B][D]
    outs = torch.empty_like(toks)
    s0 = st.s.clone()
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):          # warm up on a side stream before capture
        for t in range(8):
            rlm.rlm_mix_decode(toks[t], st, outs[t])
    torch.cuda.current_stream().wait_stream(side)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        for t in range(T):
            rlm.rlm_mix_decode(toks[t], st, outs[t])
    stream = torch.cuda.current_stream()
    res = []
    for rep in range(4):
        st.s.copy_(s0)
        torch.cuda.synchronize()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        g.replay()
        b.record(stream)
        torch.cuda.synchronize()
        if rep:
            res.append(a.elapsed_time(b))
    ms = statistics.median(res)
    us_step = ms * 1e3 / T
    per_step = decode_bytes(B, D, M)
    gbs = per_step / (us_step * 1e-6) / 1e9
    return {"workload": f"decode B={B} D={D} M={M}, {T} steps after a {L}-token prefill, CUDA graph",
            "tok_s": round(B * T / (ms * 1e-3), 1), "us_per_step": round(us_step, 4),
            "achieved_GBps": round(gbs, 1), "frac_hbm": round(gbs / hbm_peak, 4),
            "bytes_per_step": per_step, "launches": T}


def _bench_decode_large_batch(rlm, torch, dev, hbm_peak, B=8192, T=64):
    """The decode kernel where moving the state, not latency, sets the step time:
    B = 8192 (a 256 MiB fp32 state, above the L2 size, read and written every
    step).  The state is seeded with N(0, 1) values (rlm_state_init, then a fill)
    instead of a 32768-token prefill, which at this batch would need 137 GB of
    drive."""
    from synth import make_inputs
    P = DECODE
    D, M = P["D"], P["M"]
    inp = make_inputs(1, 1, D, M, "bf16", seed=0)
    p = rlm.Params.from_arrays(*inp.params(), device=dev)
    st = rlm.State.empty(B, D, M, device=dev)
    rlm.rlm_state_init(st, p)
    gen = torch.Generator(device="cpu").manual_seed(3)
    s0 = torch.randn(B, D, M, 2, generator=gen).to(dev)
    toks = torch.randn(T, B, D, generator=gen).to(dev, torch.bfloat16)
    outs = torch.empty_like(toks)
    st.s.copy_(s0)
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        for t in range(8):
            rlm.rlm_mix_decode(toks[t], st, outs[t])
    torch.cuda.current_stream().wait_stream(side)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        for t in range(T):
            rlm.rlm_mix_decode(toks[t], st, outs[t])
    stream = torch.cuda.current_stream()
    res = []
    for rep in range(4):
        st.s.copy_(s0)
        torch.cuda.synchronize()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        g.replay()
        b.record(stream)
        torch.cuda.synchronize()
        if rep:
            res.append(a.elapsed_time(b))
    us_step = statistics.median(res) * 1e3 / T
    per_step = decode_bytes(B, D, M)
    gbs = per_step / (us_step * 1e-6) / 1e9
    return {"workload": f"decode B={B} D={D} M={M}, {T} steps from a seeded state, CUDA graph (beyond the "
                        f"configured batch sizes: the bandwidth-bound regime of the same kernel)",
            "us_per_step": round(us_step, 4), "tok_s": round(B / (us_step * 1e-6), 1),
            "achieved_GBps": round(gbs, 1), "frac_hbm": round(gbs / hbm_peak, 4), "bytes_per_step": per_step}


def _bench_mixer(rlm, torch, dev, hbm_peak, flush, mix_ms, with_decode=True):
    """The mixer wrapper of Sec. 3.4 on the headline prefill shape: the gate alone
    (fused into the tcgen05 prefill) and the gate with the local path K = 4 and
    drive history (the prefill, then one pass over whole-row tiles that also
    applies the head coupling when there is one); and the fused decode step
    (B = 64) in a CUDA graph."""
    from synth import make_inputs, make_mixer_inputs
    P = MIXER
    B, L, D, M, K = P["B"], P["L"], P["D"], P["M"], P["K"]
    inp = make_inputs(B, L, D, M, "bf16", seed=2)
    mx = make_mixer_inputs(inp, K, seed=2)
    x = torch.from_numpy(inp.x).to(dev, torch.bfloat16)
    g = torch.from_numpy(mx.g).to(dev, torch.bfloat16)
    p = rlm.Params.from_arrays(*inp.params(), device=dev)
    local = rlm.Local.from_arrays(mx.conv_w, mx.scale, device=dev)
    hin = rlm.ConvState(torch.from_numpy(mx.conv_in).to(dev, torch.bfloat16))
    hout = rlm.ConvState.empty(B, D, K, dtype=torch.bfloat16, device=dev)
    z = torch.empty_like(x)
    st = rlm.State.empty(B, D, M, device=dev)
    wsz = rlm.rlm_prefill_workspace_size(B, L, D, M, torch.bfloat16)
    work = torch.empty(max(wsz, 256), dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream()

    H = P["H"]
    coupling = rlm.Coupling.from_arrays(np.random.default_rng(5).standard_normal((H, H)), 0.5, device=dev)

    def measure(kk, cp=None):
        loc = local if kk else None

        def call():
            rlm.rlm_mixer_prefill(x, g, p, loc, z, conv_in=hin if kk else None, state_out=st,
                                  conv_out=hout if kk else None, workspace=work, coupling=cp)

        for _ in range(3):
            flush.zero_()
            call()
        torch.cuda.synchronize()
        ts = []
        n0 = rlm.rlm_kernels_launched()
        for _ in range(10):
            flush.zero_()
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record(stream)
            call()
            b.record(stream)
            torch.cuda.synchronize()
            ts.append(a.elapsed_time(b))
        launches = (rlm.rlm_kernels_launched() - n0) // 10
        ms = statistics.mean(ts)
        alg = mixer_prefill_bytes(B, L, D, M, kk) + (4 * H * H if cp is not None else 0)
        gbs = alg / (ms * 1e-3) / 1e9
        what = "gate fused into the tcgen05 prefill" if kk == 0 else \
            f"gate and local path K={kk} with drive history: prefill then one whole-row pass"
        if cp is not None:
            what = f"head coupling H={H}, " + what.replace("one whole-row pass", "one whole-row pass with the coupling")
        return {"workload": f"mixer prefill B={B} L={L} D={D} M={M} bf16, {what}",
                "ms": round(ms, 5), "Mtok_s": round(B * L / (ms * 1e-3) / 1e6, 1),
                "achieved_GBps": round(gbs, 1), "frac_hbm": round(gbs / hbm_peak, 4),
                "algorithmic_bytes": alg, "launches_per_call": launches,
                "vs_mix_only": round(ms / mix_ms, 3)}

    prefill_gate = measure(0)
    prefill = measure(K)
    prefill_coupled = measure(K, coupling)
    del x, g, z, work
    if not with_decode:
        return {"prefill_gate": prefill_gate, "prefill": prefill, "prefill_coupled": prefill_coupled}

    Bd, T = P["decode_B"], P["T"]
    dinp = make_inputs(Bd, 1, D, M, "bf16", seed=3, decode_steps=T)
    dmx = make_mixer_inputs(dinp, K, seed=3)
    toks = torch.from_numpy(dinp.tokens).to(dev, torch.bfloat16)      # [T][B][D]
    gts = torch.from_numpy(np.ascontiguousarray(
        np.random.default_rng(4).standard_normal((T, Bd, D)).astype(np.float32))).to(dev, torch.bfloat16)
    outs = torch.empty_like(toks)
    dp = rlm.Params.from_arrays(*dinp.params(), device=dev)
    dlocal = rlm.Local.from_arrays(dmx.conv_w, dmx.scale, device=dev)
    dst = rlm.State.empty(Bd, D, M, device=dev)
    rlm.rlm_state_init(dst, dp)
    hist = rlm.ConvState(torch.zeros(Bd, K - 1, D, dtype=torch.bfloat16, device=dev))
    s0 = dst.s.clone()
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        for t in range(8):
            rlm.rlm_mixer_decode(toks[t], gts[t], dst, dlocal, hist, outs[t])
    torch.cuda.current_stream().wait_stream(side)
    torch.cuda.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        for t in range(T):
            rlm.rlm_mixer_decode(toks[t], gts[t], dst, dlocal, hist, outs[t])
    def replay_us(gr):
        res = []
        for rep in range(4):
            dst.s.copy_(s0)
            torch.cuda.synchronize()
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record(stream)
            gr.replay()
            b.record(stream)
            torch.cuda.synchronize()
            if rep:
                res.append(a.elapsed_time(b))
        return statistics.median(res) * 1e3 / T

    us = replay_us(graph)
    per = mixer_decode_bytes(Bd, D, M, K)
    dgbs = per / (us * 1e-6) / 1e9
    decode = {"workload": f"fused mixer decode B={Bd} D={D} M={M} K={K}, {T} steps, CUDA graph",
              "us_per_step": round(us, 4), "tok_s": round(Bd / (us * 1e-6), 1),
              "achieved_GBps": round(dgbs, 1), "frac_hbm": round(dgbs / hbm_peak, 4), "bytes_per_step": per}
    dcp = rlm.Coupling.from_arrays(np.random.default_rng(6).standard_normal((H, H)), 0.5, device=dev)
    graph_c = torch.cuda.CUDAGraph()
    n0 = rlm.rlm_kernels_launched()
    with torch.cuda.graph(graph_c):
        for t in range(T):
            rlm.rlm_mixer_decode(toks[t], gts[t], dst, dlocal, hist, outs[t], coupling=dcp)
    lps = (rlm.rlm_kernels_launched() - n0) / T
    uc = replay_us(graph_c)
    decode_coupled = {"workload": f"mixer decode with head coupling H={H}, B={Bd} D={D} M={M} K={K}: one block "
                                  f"per batch row (recurrence step, coupling, gate, local path); {T} steps, "
                                  f"CUDA graph",
                      "us_per_step": round(uc, 4), "tok_s": round(Bd / (uc * 1e-6), 1), "launches_per_step": lps}
    return {"prefill_gate": prefill_gate, "prefill": prefill, "prefill_coupled": prefill_coupled, "decode": decode,
            "decode_coupled": decode_coupled}


def _bench_tied_and_fft(rlm, torch, dev, hbm_peak, flush):
    """The paper's tied heads (Sec. 3.1: H = 8 heads x 32 channels, one mode, no
    amplitude) on the long-context shape through the library (the tcgen05 prefill
    with M = 1), and the paper's own evaluation of Eq. 2 by FFT (Eq. 3: zero
    padding to a power of two; cuFFT through torch.fft in fp32) on the same drive
    and kernels, timed as the prior-art comparison and checked against the
    library's output."""
    B, L, H, dh = 4, 32768, 8, 32
    D = H * dh
    rng = np.random.default_rng(9)
    alpha = np.exp(rng.uniform(np.log(1e-3), np.log(0.3), H)).astype(np.float32)
    omega = rng.uniform(0.0, np.pi, H).astype(np.float32)
    phi = rng.uniform(-np.pi, np.pi, H).astype(np.float32)
    x = torch.randn(B, L, D, device=dev).to(torch.bfloat16)
    p = rlm.Params.tied_heads(alpha, omega, phi, dh, device=dev)
    y = torch.empty_like(x)
    stream = torch.cuda.current_stream()

    def timed(fn, reps=8):
        for _ in range(3):
            flush.zero_()
            fn()
        torch.cuda.synchronize()
        ts = []
        for _ in range(reps):
            flush.zero_()
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record(stream)
            fn()
            b.record(stream)
            torch.cuda.synchronize()
            ts.append(a.elapsed_time(b))
        return statistics.mean(ts)

    ms = timed(lambda: rlm.rlm_mix_prefill(x, p, y))
    alg = prefill_bytes(B, L, D, 1)
    tied = {"workload": f"tied heads B={B} L={L} H={H} d_h={dh} (one mode per head, A = 1), bf16",
            "ms": round(ms, 5), "Mtok_s": round(B * L / (ms * 1e-3) / 1e6, 1),
            "frac_hbm": round(alg / (ms * 1e-3) / 1e9 / hbm_peak, 4)}
    nfft = 1 << (2 * L - 1).bit_length()
    n = torch.arange(L, device=dev, dtype=torch.float32)
    a_t, w_t, f_t = (torch.from_numpy(v).to(dev)[:, None] for v in (alpha, omega, phi))
    k = torch.exp(-a_t * n) * torch.cos(w_t * n + f_t)                       # [H][L], Sec. 3.1
    out = {}

    def fft_route():
        kf = torch.fft.rfft(k, nfft)
        xf = torch.fft.rfft(x.float().view(B, L, H, dh).permute(0, 2, 3, 1), nfft)
        yh = torch.fft.irfft(xf * kf[None, :, None, :], nfft)[..., :L]
        out["y"] = yh.permute(0, 3, 1, 2).reshape(B, L, D).to(torch.bfloat16)

    fms = timed(fft_route, reps=4)
    d = (out["y"].float() - y.float()).norm() / y.float().norm()
    fft = {"workload": "the same problem by Eq. 3: rfft of drive and kernels (zero padded to "
                       f"{nfft}), product, irfft, fp32 (cuFFT through torch.fft)",
           "ms": round(fms, 4), "Mtok_s": round(B * L / (fms * 1e-3) / 1e6, 1),
           "rel_l2_vs_library": round(float(d), 6), "library_speedup": round(fms / ms, 1)}
    del x, y, out
    return {"tied_heads": tied, "fft_eq3": fft}


def _bench_backward(rlm, torch, dev, hbm_peak, args, flush):
    """Training step at B=4 L=32768 D=512 M=32 (bf16): backward, forward and the
    backward with state terms.  Each timed call follows an L2 flush, which also
    keeps the GPU busy while the host enqueues the call (no host latency inside
    the events)."""
    from synth import make_inputs
    P = BACKWARD
    B, L, D, M = P["B"], P["L"], P["D"], P["M"]
    inp = make_inputs(B, L, D, M, "bf16", seed=0, with_dy=True)
    x = torch.from_numpy(inp.x).to(dev, torch.bfloat16)
    dy = torch.from_numpy(inp.dy).to(dev, torch.bfloat16)
    p = rlm.Params.from_arrays(*inp.params(), device=dev)
    dx = torch.empty_like(x)
    g = rlm.Grads.empty(D, M, device=dev)
    wsz = rlm.rlm_backward_workspace_size(B, L, D, M, torch.bfloat16)
    work = torch.empty(max(wsz, 256), dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream()

    def _timed(fn, reps=5):
        for _ in range(2):
            fn()
        out = []
        for _ in range(reps):
            flush.zero_()
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record(stream)
            fn()
            b.record(stream)
            torch.cuda.synchronize()
            out.append(a.elapsed_time(b))
        return statistics.mean(out)

    ms = _timed(lambda: rlm.rlm_mix_backward(dy, x, p, dx, g, workspace=work))
    # The training step's forward on the same shape (bf16, M = 32: one launch of
    # the 32-mode tensor-core prefill).
    y = torch.empty_like(x)
    st = rlm.State.empty(B, D, M, device=dev)
    fw = torch.empty(max(256, rlm.rlm_prefill_workspace_size(B, L, D, M, torch.bfloat16)), dtype=torch.uint8,
                     device=dev)
    fms = _timed(lambda: rlm.rlm_mix_prefill(x, p, y, st, workspace=fw))
    del y, st, fw
    # Backward with the state terms of a segmented training step: an initial state
    # (its gradient returned), and a terminal-state gradient as well (one more
    # launch that forms its terms in closed form).
    gen = torch.Generator(device="cpu").manual_seed(1)
    s_in, ds_out, ds_in = (rlm.State.empty(B, D, M, device=dev) for _ in range(3))
    s_in.s.copy_(torch.randn(B, D, M, 2, generator=gen))
    ds_out.s.copy_(torch.randn(B, D, M, 2, generator=gen))

    ms_init = _timed(lambda: rlm.rlm_mix_backward_from(dy, x, p, s_in, None, dx, g, ds_in, workspace=work))
    ms_term = _timed(lambda: rlm.rlm_mix_backward_from(dy, x, p, s_in, ds_out, dx, g, ds_in, workspace=work))
    del s_in, ds_out, ds_in
    gbs = backward_bytes(B, L, D, M) / (ms * 1e-3) / 1e9
    moved = backward_moved_bytes(B, L, D) / (ms * 1e-3) / 1e9
    return {"workload": "backward B=4 L=32768 D=512 M=32 bf16", "ms": round(ms, 4),
            "Mtok_s": round(B * L / (ms * 1e-3) / 1e6, 2), "achieved_GBps": round(gbs, 1),
            "frac_hbm": round(gbs / hbm_peak, 4),
            "data_path": "transpose to channel-major, tcgen05 kernel, transpose back, fixed-order reduction",
            "moved_GBps": round(moved, 1), "moved_frac_hbm": round(moved / hbm_peak, 4),
            "forward_ms": round(fms, 4), "forward_plus_backward_ms": round(fms + ms, 4),
            "with_state_in_ms": round(ms_init, 4),
            "with_state_in_and_d_state_out_ms": round(ms_term, 4),
            "state_terms_route": "tcgen05; d_state_out adds one launch (k_terminal_tc) forming "
                                 "conj(g) lambda^(L-1-t) terms in closed form on the tensor cores"}


def run_backward_only(args):
    import torch

    import paper_2607_05583_gb300 as rlm
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    rlm.load_library()
    hbm_peak, _, peak_kind = _peaks()
    n0 = rlm.rlm_kernels_launched()
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=dev)
    out = _bench_backward(rlm, torch, dev, hbm_peak, args, flush)
    out.update({"mode": "backward only", "peak_kind": peak_kind,
                "gpu_launches": rlm.rlm_kernels_launched() - n0})
    print(json.dumps(out), flush=True)


def run_kernels_only(args):
    """One representative workload per kernel that the headline path does not
    time, for their ncu captures: each case runs 3 warm-up and 5 timed calls (L2
    flushed before each) and the line reports its mean time and algorithmic
    bytes.  Cases and the kernels they launch:
      fp32_prefill        B=4 L=32768 D=256 M=16 fp32: k_prefill_tc32
      fp32_prefill_state  the same with an initial state: k_prefill_tc32
      fp32_prefill_state_ragged  B=4 L=32767 with an initial state (the SIMT chunked scan):
                          k_chunk_local, k_chunk_carry, k_chunk_output
      decode_b64 / b1     one plain decode step: k_decode_tile
      mixer_decode_plain  mixer step without coupling, B=64 D=2048 K=4 (rows past the
                          one-block step): k_decode_tile (mixer)
      mixer_decode_b64    coupled mixer step H=8 K=4 (D=256): k_decode_coupled
      mixer_prefill_d2048 coupled mixer prefill B=1 L=32768 D=2048 H=8 K=4 (4 KB rows):
                          k_prefill_tc, k_couple_small, k_mixer_epilogue, k_mixer_tail
      mixer_decode_d2048  coupled mixer step B=64 D=2048 H=8 K=4: k_decode_tile, k_mixer_finish"""
    import torch

    import paper_2607_05583_gb300 as rlm
    from synth import make_inputs, make_mixer_inputs
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    rlm.load_library()
    hbm_peak, _, peak_kind = _peaks()
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream()
    out = {}

    def timed(name, fn, alg_bytes):
        for _ in range(3):
            flush.zero_()
            fn()
        torch.cuda.synchronize()
        ts = []
        for _ in range(5):
            flush.zero_()
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record(stream)
            fn()
            b.record(stream)
            torch.cuda.synchronize()
            ts.append(a.elapsed_time(b))
        ms = statistics.mean(ts)
        gbs = alg_bytes / (ms * 1e-3) / 1e9
        out[name] = {"ms": round(ms, 5), "algorithmic_bytes": alg_bytes, "achieved_GBps": round(gbs, 1),
                     "frac_hbm": round(gbs / hbm_peak, 4)}

    # fp32 prefill on the tensor cores, from a zero state and from an initial state;
    # with an initial state and a length that is not a multiple of 64, the SIMT
    # chunked scan
    B, L, D, M = 4, 32768, 256, 16
    inp = make_inputs(B, L, D, M, "f32", seed=1)
    x = torch.from_numpy(inp.x).to(dev)
    p = rlm.Params.from_arrays(*inp.params(), device=dev)
    y = torch.empty_like(x)
    st = rlm.State.empty(B, D, M, device=dev)
    s_in = rlm.State.empty(B, D, M, device=dev)
    s_in.s.copy_(torch.randn(B, D, M, 2, generator=torch.Generator(device="cpu").manual_seed(2)))
    work = torch.empty(max(rlm.rlm_prefill_workspace_size(B, L, D, M, torch.float32), 256), dtype=torch.uint8,
                       device=dev)
    timed("fp32_prefill", lambda: rlm.rlm_mix_prefill(x, p, y, st, workspace=work), prefill_bytes(B, L, D, M, 4))
    timed("fp32_prefill_state", lambda: rlm.rlm_mix_prefill_from(x, p, s_in, y, st, workspace=work),
          prefill_bytes(B, L, D, M, 4))
    xr = x[:, :L - 1].contiguous()
    yr = torch.empty_like(xr)
    timed("fp32_prefill_state_ragged", lambda: rlm.rlm_mix_prefill_from(xr, p, s_in, yr, st, workspace=work),
          prefill_bytes(B, L - 1, D, M, 4))
    del x, y, xr, yr, work, s_in

    # plain decode steps
    for Bd in (64, 1):
        dinp = make_inputs(Bd, 1, D, M, "bf16", seed=3, decode_steps=2)
        dp = rlm.Params.from_arrays(*dinp.params(), device=dev)
        dst = rlm.State.empty(Bd, D, M, device=dev)
        rlm.rlm_state_init(dst, dp)
        tok = torch.from_numpy(dinp.tokens[0]).to(dev, torch.bfloat16)
        yt = torch.empty_like(tok)
        timed(f"decode_b{Bd}", lambda: rlm.rlm_mix_decode(tok, dst, yt), decode_bytes(Bd, D, M))

    # mixer decode step without coupling on rows past the one-block step (the
    # row-tiled recurrence step with gate and local path)
    H, K = 8, 4
    Bd, Dm = 64, 2048
    dinp = make_inputs(Bd, 1, Dm, M, "bf16", seed=4, decode_steps=2)
    dmx = make_mixer_inputs(dinp, K, seed=4)
    dp = rlm.Params.from_arrays(*dinp.params(), device=dev)
    dst = rlm.State.empty(Bd, Dm, M, device=dev)
    rlm.rlm_state_init(dst, dp)
    loc = rlm.Local.from_arrays(dmx.conv_w, dmx.scale, device=dev)
    hist = rlm.ConvState(torch.zeros(Bd, K - 1, Dm, dtype=torch.bfloat16, device=dev))
    tok = torch.from_numpy(dinp.tokens[0]).to(dev, torch.bfloat16)
    gt = torch.randn(Bd, 1, Dm, device=dev).to(torch.bfloat16).view_as(tok)
    zt = torch.empty_like(tok)
    timed("mixer_decode_plain", lambda: rlm.rlm_mixer_decode(tok, gt, dst, loc, hist, zt),
          decode_bytes(Bd, Dm, M) + 2 * Bd * Dm * (K - 1) * 2 + 2 * Bd * Dm)

    # coupled mixer decode step, fused (D = 256) and with the finishing pass (D = 2048)
    for Dm in (256, 2048):
        Bd = 64
        dinp = make_inputs(Bd, 1, Dm, M, "bf16", seed=4, decode_steps=2)
        dmx = make_mixer_inputs(dinp, K, seed=4)
        dp = rlm.Params.from_arrays(*dinp.params(), device=dev)
        dst = rlm.State.empty(Bd, Dm, M, device=dev)
        rlm.rlm_state_init(dst, dp)
        loc = rlm.Local.from_arrays(dmx.conv_w, dmx.scale, device=dev)
        cp = rlm.Coupling.from_arrays(np.random.default_rng(5).standard_normal((H, H)), 0.5, device=dev)
        hist = rlm.ConvState(torch.zeros(Bd, K - 1, Dm, dtype=torch.bfloat16, device=dev))
        tok = torch.from_numpy(dinp.tokens[0]).to(dev, torch.bfloat16)
        gt = torch.randn(Bd, 1, Dm, device=dev).to(torch.bfloat16).view_as(tok)
        zt = torch.empty_like(tok)
        name = "mixer_decode_b64" if Dm == 256 else "mixer_decode_d2048"
        alg = decode_bytes(Bd, Dm, M) + 2 * Bd * Dm * (K - 1) * 2 + 2 * Bd * Dm
        timed(name, lambda: rlm.rlm_mixer_decode(tok, gt, dst, loc, hist, zt, coupling=cp), alg)

    # coupled mixer prefill on 4 KB rows (the separate coupling and channel-pair passes)
    B, L, Dm = 1, 32768, 2048
    inp = make_inputs(B, L, Dm, M, "bf16", seed=6)
    mx = make_mixer_inputs(inp, K, seed=6)
    x = torch.from_numpy(inp.x).to(dev, torch.bfloat16)
    g = torch.from_numpy(mx.g).to(dev, torch.bfloat16)
    p = rlm.Params.from_arrays(*inp.params(), device=dev)
    loc = rlm.Local.from_arrays(mx.conv_w, mx.scale, device=dev)
    cp = rlm.Coupling.from_arrays(np.random.default_rng(7).standard_normal((H, H)), 0.5, device=dev)
    z = torch.empty_like(x)
    work = torch.empty(max(rlm.rlm_prefill_workspace_size(B, L, Dm, M, torch.bfloat16), 256), dtype=torch.uint8,
                       device=dev)
    timed("mixer_prefill_d2048",
          lambda: rlm.rlm_mixer_prefill(x, g, p, loc, z, workspace=work, coupling=cp),
          mixer_prefill_bytes(B, L, Dm, M, K) + 4 * H * H)
    print(json.dumps({"kernels_only": out, "peak_GBps": hbm_peak, "peak_kind": peak_kind}), flush=True)


def run_mixer_only(args):
    """The mixer prefill measurements alone (used for their ncu captures)."""
    import torch

    import paper_2607_05583_gb300 as rlm
    from synth import make_inputs
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    rlm.load_library()
    hbm_peak, _, peak_kind = _peaks()
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=dev)
    P = MIXER
    inp = make_inputs(P["B"], P["L"], P["D"], P["M"], "bf16", seed=2)
    x = torch.from_numpy(inp.x).to(dev, torch.bfloat16)
    p = rlm.Params.from_arrays(*inp.params(), device=dev)
    y = torch.empty_like(x)
    for _ in range(3):
        rlm.rlm_mix_prefill(x, p, y)
    ts = []
    for _ in range(5):
        flush.zero_()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record()
        rlm.rlm_mix_prefill(x, p, y)
        b.record()
        torch.cuda.synchronize()
        ts.append(a.elapsed_time(b))
    del x, y
    n0 = rlm.rlm_kernels_launched()
    out = _bench_mixer(rlm, torch, dev, hbm_peak, flush, statistics.mean(ts), with_decode=False)
    out.update({"mode": "mixer prefill only", "peak_kind": peak_kind,
                "gpu_launches": rlm.rlm_kernels_launched() - n0})
    print(json.dumps(out), flush=True)


# ---------------------------------------------------------------- CPU oracle
def cpu_baseline(seconds=10.0):
    """The fp64 oracle's sequential recurrence (as it stands) on the host cores, on
    a bounded sample of the prefill workload: whole sequences of the B=4, L=32768,
    D=256, M=16 problem, repeated until about ``seconds`` of CPU time."""
    import oracle
    from synth import make_inputs
    P = PREFILL
    inp = make_inputs(1, P["L"], P["D"], P["M"], "bf16", seed=0)
    x64 = inp.x.astype(np.float64)
    prm = [q.astype(np.float64) for q in inp.params()]
    oracle.rec_prefill(x64[:, :1024], *prm)          # load/compile outside the timing
    t0 = time.perf_counter()
    n = 0
    while True:
        oracle.rec_prefill(x64, *prm)
        n += 1
        if time.perf_counter() - t0 >= seconds:
            break
    dt = time.perf_counter() - t0
    out = {"value": round(n * P["L"] / dt / 1e6, 4), "unit": "Mtok/s", "cores": oracle.num_threads(),
           "kind": "oracle",
           "sample": f"{n} x one sequence (B=1, L={P['L']}, D={P['D']}, M={P['M']}) of the "
                     f"prefill workload through the fp64 sequential recurrence, {dt:.1f} s"}
    out["other_workloads"] = _cpu_other_workloads(seconds=max(1.0, seconds / 4))
    return out


def _cpu_other_workloads(seconds):
    """The oracle on the other workloads, each for about ``seconds``: the 6M layer's
    prefill (O2), decode steps at B = 64 (O2's step), and the O(L^2) direct
    convolution (O1) at L = 8192 on a sample of channels (the analogue of the
    paper's quadratic causal reference)."""
    import oracle
    from synth import make_inputs

    def loop(fn):
        t0 = time.perf_counter()
        n = 0
        while True:
            fn()
            n += 1
            if time.perf_counter() - t0 >= seconds:
                return n, time.perf_counter() - t0

    res = {}
    inp = make_inputs(8, 2048, 256, 16, "bf16", seed=0)
    x64, prm = inp.x.astype(np.float64), [q.astype(np.float64) for q in inp.params()]
    n, dt = loop(lambda: oracle.rec_prefill(x64, *prm))
    res["layer6m_prefill_B8_L2048"] = {"Mtok_s": round(n * 8 * 2048 / dt / 1e6, 4),
                                       "sample": f"{n} calls of the whole problem, {dt:.1f} s"}
    dec = make_inputs(64, 1, 256, 16, "bf16", seed=0)
    _, st = oracle.rec_prefill(dec.x.astype(np.float64), *[q.astype(np.float64) for q in dec.params()])
    xt = dec.x[:, 0].astype(np.float64)
    dprm = [q.astype(np.float64) for q in dec.params()]
    box = {"s": st}

    def step():
        _, box["s"] = oracle.rec_decode(box["s"], xt, *dprm)

    n, dt = loop(step)
    res["decode_B64"] = {"tok_s": round(n * 64 / dt, 1), "us_per_step": round(dt / n * 1e6, 1),
                         "sample": f"{n} steps, {dt:.1f} s"}
    ch = 16
    conv = make_inputs(1, 8192, ch, 16, "bf16", seed=0)
    cx, cprm = conv.x.astype(np.float64), [q.astype(np.float64) for q in conv.params()]
    n, dt = loop(lambda: oracle.conv_prefill(cx, *cprm))
    # scale to the full 256 channels: channels are independent work
    res["direct_convolution_L8192"] = {"Mtok_s_at_D256": round(n * 8192 * ch / 256 / dt / 1e6, 6),
                                       "sample": f"{n} calls on {ch} of 256 channels, {dt:.1f} s"}
    return res


def run_reference(args):
    """Reference arm: the CPU oracle as it stands, on the host cores."""
    ws, rank, _ = _dist()
    if rank != 0:
        return
    import oracle
    from synth import make_inputs
    P = PREFILL
    inp = make_inputs(1, P["L"], P["D"], P["M"], "bf16", seed=0)
    x64 = inp.x.astype(np.float64)
    prm = [q.astype(np.float64) for q in inp.params()]
    for _ in range(args.warmup):
        oracle.rec_prefill(x64[:, :4096], *prm)
    t0 = time.perf_counter()
    for _ in range(args.steps):
        oracle.rec_prefill(x64, *prm)
    dt = time.perf_counter() - t0
    val = args.steps * P["L"] / dt / 1e6
    cpu = {"value": round(val, 4), "unit": "Mtok/s", "cores": oracle.num_threads(), "kind": "oracle",
           "sample": f"each step one sequence (B=1, L={P['L']}, D={P['D']}, M={P['M']}) of the "
                     f"prefill workload through the fp64 sequential recurrence"}
    print(json.dumps({
        "impl": "reference", "metric": METRIC, "value": round(val, 4), "unit": "Mtok/s",
        "n_gpus": ws, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round(dt / args.steps * 1e3, 3), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": "long-context prefill B=4 L=32768 D=256 M=16 bf16 I/O fp32 state",
                   "sample": "B=1 per step"},
        "cpu_baseline": cpu,
        "e2e": {"value": round(val, 4), "unit": "Mtok/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0}}), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--quick", action="store_true", help="prefill only (no sweep/decode/backward)")
    ap.add_argument("--no-cpu", action="store_true", help="skip the CPU-oracle baseline")
    ap.add_argument("--cpu-seconds", type=float, default=10.0)
    ap.add_argument("--only", default="all", choices=["all", "backward", "mixer", "kernels"],
                    help="backward / mixer / kernels: run only that measurement (diagnostic, ncu captures)")
    ap.add_argument("--soak", type=float, default=1.5,
                    help="seconds of untimed prefill before the timed steps (clock sampling)")
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3
    if args.impl == "reference":
        run_reference(args)
    elif args.only == "backward":
        run_backward_only(args)
    elif args.only == "mixer":
        run_mixer_only(args)
    elif args.only == "kernels":
        run_kernels_only(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
