"""Host logic of the multi-GPU benchmark path, on CPU with the gloo backend (world size 2).

The connection op is token-parallel: every rank runs the whole step on its own tokens (weak
scaling, no collective on the data path).  What crosses ranks is the timing: the timed region is
the slowest rank's, and the reported rate counts every rank's tokens.  The reference arm runs on
rank 0 only; the other ranks exit without work."""
import os
import socket
import sys

import torch
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out_dir):
    sys.path.insert(0, ROOT)
    import bench
    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank, world_size=world)
    try:
        ms, value = bench.job_rate(10.0 + 5.0 * rank, 1000, 4, world, "cpu")
        with open(os.path.join(out_dir, f"r{rank}.txt"), "w") as f:
            f.write(f"{ms!r} {value!r}\n")
    finally:
        dist.destroy_process_group()


def test_job_rate_takes_the_slowest_rank_and_counts_every_rank(tmp_path):
    world = 2
    mp.start_processes(_rank_main, args=(world, _free_port(), str(tmp_path)), nprocs=world,
                       join=True, start_method="spawn")
    for r in range(world):
        ms, value = (float(v) for v in (tmp_path / f"r{r}.txt").read_text().split())
        assert ms == 15.0
        assert abs(value - world * 1000 * 4 / 0.015) < 1e-6 * value


def test_job_rate_single_rank_needs_no_process_group():
    sys.path.insert(0, ROOT)
    import bench
    ms, value = bench.job_rate(20.0, 500, 2, 1)
    assert ms == 20.0 and abs(value - 500 * 2 / 0.02) < 1e-9


def test_reference_arm_runs_on_rank0_only(monkeypatch, capsys):
    sys.path.insert(0, ROOT)
    import bench

    class A:
        ref_tokens, steps, warmup, gpus = 4, 1, 0, 2

    monkeypatch.setenv("RANK", "1")
    bench.run_reference(A, "flash4")
    assert capsys.readouterr().out == ""
