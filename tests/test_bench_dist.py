"""The multi-rank bench path on CPU (gloo, world size 2): independent
problems per rank, timings reduced with MAX and unit counts with SUM."""
import os
import socket

import pytest

torch = pytest.importorskip("torch")
import torch.multiprocessing as mp  # noqa: E402


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, out):
    import sys

    import torch.distributed as dist

    sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
    import bench

    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank, world_size=world)
    mx = bench.reduce_across_ranks(10.0 + rank, "max")
    sm = bench.reduce_across_ranks(1000 * (rank + 1), "sum")
    dist.barrier()
    dist.destroy_process_group()
    with open(os.path.join(out, f"r{rank}"), "w") as f:
        f.write(f"{mx} {sm}")


def test_two_rank_reduction(tmp_path):
    port = _free_port()
    mp.spawn(_rank, args=(2, port, str(tmp_path)), nprocs=2, join=True)
    for r in range(2):
        mx, sm = map(float, open(tmp_path / f"r{r}").read().split())
        assert mx == 11.0 and sm == 3000.0


def test_single_process_is_identity():
    import sys

    sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
    import bench

    assert bench.reduce_across_ranks(3.5, "max") == 3.5
    assert bench.reduce_across_ranks(7, "sum") == 7.0
