"""The bench's multi-process host logic on CPU: two ranks under the gloo backend
(one process per rank, rendezvous on 127.0.0.1).  Each rank's step time is
reduced to the slowest rank's, every rank takes part in the barriers, and the
reference arm runs on rank 0 only."""
import importlib.util
import os
import socket

import pytest

torch = pytest.importorskip("torch")
import torch.distributed as dist  # noqa: E402
import torch.multiprocessing as mp  # noqa: E402

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _bench():
    spec = importlib.util.spec_from_file_location("bench", os.path.join(ROOT, "bench.py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, ws, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(ws), LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=ws)
    try:
        bench = _bench()
        assert bench._dist() == (ws, rank, rank)
        bench._barrier(ws)
        out[rank] = bench._barrier_max(1.0 + 2.0 * rank, ws)
        bench._barrier(ws)
    finally:
        dist.destroy_process_group()


def test_step_time_is_the_slowest_rank():
    ws = 2
    out = mp.Manager().dict()
    mp.spawn(_rank_main, args=(ws, _free_port(), out), nprocs=ws, join=True)
    assert dict(out) == {0: 3.0, 1: 3.0}


def test_reference_arm_runs_on_rank_zero_only(monkeypatch, capsys):
    bench = _bench()
    monkeypatch.setenv("WORLD_SIZE", "2")
    monkeypatch.setenv("RANK", "1")
    monkeypatch.setenv("LOCAL_RANK", "1")

    class Args:
        steps, warmup = 1, 3

    bench.run_reference(Args())          # rank 1: returns at once, prints nothing
    assert capsys.readouterr().out == ""
