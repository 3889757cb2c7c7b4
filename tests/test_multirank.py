"""The multi-GPU path on CPU: bench.py runs one replica per rank (the step
shards by sequence with no exchange on the data path), then reduces its
figures over the ranks.  Two gloo ranks check that reduction: times take the
slowest rank, token counts add.  A non-zero rank of the reference arm exits
without work."""
import os
import socket
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket(socket.AF_INET, socket.SOCK_STREAM) as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out_dir):
    sys.path.insert(0, ROOT)
    import torch.distributed as dist

    import bench
    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank, world_size=world)
    try:
        # rank r: device times (10 + r, 2 r) ms, tokens (100 r + 7, 3)
        times, counts = bench.aggregate_ranks([10.0 + rank, 2.0 * rank], [100.0 * rank + 7.0, 3.0], world, "cpu")
        dist.barrier()
    finally:
        dist.destroy_process_group()
    with open(os.path.join(out_dir, f"rank{rank}.txt"), "w") as f:
        f.write(" ".join(repr(x) for x in times + counts))


def test_two_rank_reduction_takes_max_time_and_summed_tokens(tmp_path):
    import torch.multiprocessing as mp
    world, port = 2, _free_port()
    mp.start_processes(_rank_main, args=(world, port, str(tmp_path)), nprocs=world, join=True,
                       start_method="spawn")
    expect = [11.0, 2.0, 107.0 + 7.0, 6.0]
    for r in range(world):
        got = [float(x) for x in (tmp_path / f"rank{r}.txt").read_text().split()]
        assert got == expect


def test_single_rank_figures_pass_through():
    sys.path.insert(0, ROOT)
    import bench
    times, counts = bench.aggregate_ranks([1.5, 2.5], [9, 4], 1, "cpu")
    assert times == [1.5, 2.5] and counts == [9.0, 4.0]


def test_reference_arm_runs_on_rank_zero_only(monkeypatch, capsys):
    sys.path.insert(0, ROOT)
    import bench
    monkeypatch.setenv("RANK", "1")
    monkeypatch.setenv("WORLD_SIZE", "2")
    monkeypatch.setattr(sys, "argv", ["bench.py", "--impl", "reference", "--gpus", "2"])
    assert bench.main() == 0
    assert capsys.readouterr().out == ""
