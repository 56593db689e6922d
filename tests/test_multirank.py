"""Multi-rank host logic of bench.py on CPU: two gloo ranks.

The path shards into independent chunk streams (one per rank, no data exchange);
the only collective is the max-reduction of the timing.  These tests check that
reduction, the weak-scaling aggregate and the per-rank seeds with world_size 2.
"""

import json
import os
import socket
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out_dir):
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    import torch.distributed as dist

    import bench

    dist.init_process_group("gloo", rank=rank, world_size=world)
    own = 0.010 + 0.005 * rank  # rank 1 is the slower one
    t = bench.max_over_ranks(own, world, "cpu")
    res = {"rank": rank, "max": t, "seed": bench.rank_seed(rank),
           "value": bench.whole_job_tflops(16.15e12, t, world)}
    dist.barrier()
    dist.destroy_process_group()
    with open(os.path.join(out_dir, f"r{rank}.json"), "w") as f:
        json.dump(res, f)


def test_two_rank_timing_reduction(tmp_path):
    world = 2
    mp.start_processes(_rank_main, args=(world, _free_port(), str(tmp_path)), nprocs=world, join=True,
                       start_method="spawn")
    res = [json.load(open(tmp_path / f"r{r}.json")) for r in range(world)]
    # every rank sees the slowest rank's time
    assert all(r["max"] == pytest.approx(0.015) for r in res)
    # weak scaling: both ranks' FLOP over the max time
    assert res[0]["value"] == pytest.approx(2 * 16.15e12 / 0.015 / 1e12)
    # independent synthetic streams per rank
    assert res[0]["seed"] != res[1]["seed"]


def _heads_main(rank, world, port, out_dir):
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    import torch
    import torch.distributed as dist

    from paper_2607_21848_gb300 import api

    dist.init_process_group("gloo", rank=rank, world_size=world)
    out = {}
    for H in (2, 3, 12, 40, 41):
        h0, nh = api.head_range(H, rank, world)
        # this rank's view of a [L, N, H, d] tensor is exactly its heads
        t = torch.arange(2 * 3 * H * 4).reshape(2, 3, H, 4)
        v = api.head_view(t, h0, nh)
        assert v.shape[2] == nh and torch.equal(v, t[:, :, h0:h0 + nh])
        got = [None] * world
        dist.all_gather_object(got, (h0, nh))
        out[H] = got
    dist.barrier()
    dist.destroy_process_group()
    with open(os.path.join(out_dir, f"h{rank}.json"), "w") as f:
        json.dump(out, f)


def test_two_ranks_cover_the_heads_disjointly_and_completely(tmp_path):
    """Each gloo rank takes its head range (api.head_range) and builds its views; the ranges
    the ranks report to each other tile [0, H) with no overlap and no gap."""
    world = 2
    mp.start_processes(_heads_main, args=(world, _free_port(), str(tmp_path)), nprocs=world, join=True,
                       start_method="spawn")
    res = [json.load(open(tmp_path / f"h{r}.json")) for r in range(world)]
    assert res[0] == res[1]  # every rank sees the same split
    for H, ranges in res[0].items():
        covered = []
        for h0, nh in ranges:
            assert nh >= 1
            covered.extend(range(h0, h0 + nh))
        assert covered == list(range(int(H))), (H, ranges)  # disjoint, complete, in rank order


def test_single_rank_needs_no_process_group():
    sys.path.insert(0, ROOT)
    import bench

    assert bench.max_over_ranks(0.25, 1, "cpu") == 0.25
    assert bench.whole_job_tflops(1e12, 0.5, 1) == pytest.approx(2.0)
