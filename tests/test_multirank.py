"""The multi-rank host logic of bench.py on the CPU (gloo, world size 2): the job time is the
slowest rank's, the value counts every rank's frames, and the reference arm runs on rank 0
only.  The path has no data-path collective (independent chunks per rank)."""
import json
import os
import socket

import pytest
import torch.multiprocessing as mp

import bench


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, local_ms, out):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        dist.barrier()
        m = bench.reduce_max_ms(local_ms[rank], world, "cpu")
        out.put((rank, m, bench.whole_job_value(world, 8, 10, m)))
    finally:
        dist.destroy_process_group()


def test_job_time_is_max_over_ranks():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    local = [12.5, 20.0]
    ps = [ctx.Process(target=_worker, args=(r, 2, port, local, q)) for r in range(2)]
    for p in ps:
        p.start()
    res = sorted(q.get(timeout=120) for _ in range(2))
    for p in ps:
        p.join(timeout=60)
        assert p.exitcode == 0
    for rank, m, v in res:
        assert m == 20.0                              # the slowest rank
        assert v == pytest.approx(2 * 8 * 10 / 0.020)  # frames of both ranks per second


def test_single_rank_is_identity():
    assert bench.reduce_max_ms(7.0, 1, "cpu") == 7.0


def test_reference_arm_runs_on_rank_zero_only(monkeypatch, capsys):
    monkeypatch.setattr(bench, "_oracle_sample", lambda *a, **k: (2.0, 0.5, "stub sample"))
    monkeypatch.setattr(bench, "_par_input", lambda wl: None)
    monkeypatch.setattr(bench.W, "block_step_inputs", lambda wl: {})
    args = type("A", (), {"steps": 2, "warmup": 3})()
    monkeypatch.setenv("RANK", "1")
    monkeypatch.setenv("WORLD_SIZE", "2")
    bench.run_reference(args)
    assert capsys.readouterr().out == ""
    monkeypatch.setenv("RANK", "0")
    bench.run_reference(args)
    line = json.loads(capsys.readouterr().out.strip())
    assert line["impl"] == "reference" and line["n_gpus"] == 2
    assert line["value"] == pytest.approx(bench.WL.n_cur * 2 / 4.0)
    assert line["e2e"]["value"] == line["value"]
