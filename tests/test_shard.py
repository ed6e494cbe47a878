"""Sharding a batch of images across ranks (CPU, gloo, world size 2).

Images are independent, so ranks take contiguous image ranges and need no
data-path exchange.  The per-rank computation here is the oracle pipeline
(merge, merge, compose, gather) standing in for each rank's GPU; the test
checks that the partition covers every image once, is balanced, and that
the per-rank results gathered over gloo equal the single-process result.
"""

from __future__ import annotations

import os
import socket

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

from paper_2604_05718_gb300.shard import partition_images, shard_for_rank


def test_partition_covers_and_balances():
    rng = np.random.default_rng(0)
    for world in (1, 2, 3, 8):
        for _ in range(20):
            sizes = rng.choice([0, 1, 64, 1024, 1600, 2304, 4096], size=int(rng.integers(1, 40)))
            ranges = partition_images(sizes, world)
            assert len(ranges) == world
            assert ranges[0][0] == 0 and ranges[-1][1] == len(sizes)
            for (a, b), (c, d) in zip(ranges, ranges[1:]):
                assert b == c and a <= b
            cost = sizes.astype(float) ** 2
            loads = [cost[a:b].sum() for a, b in ranges]
            assert max(loads) <= cost.sum() / world + cost.max() + 1e-9


def test_shard_slices():
    offsets = np.array([0, 100, 100, 400, 401, 1000])
    covered = []
    for r in range(3):
        sh = shard_for_rank(offsets, r, 3)
        lo = sh.local_offsets(offsets)
        assert lo[0] == 0 and lo[-1] == sh.row_end - sh.row_start
        covered += list(range(sh.image_start, sh.image_end))
    assert covered == list(range(5))


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank: int, world: int, port: int, out_dir: str) -> None:
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import oracle
        from workloads import make_custom

        batch = make_custom([90, 1, 0, 250, 33, 120, 7], 16, "f32", seed=4)
        x = batch.tokens.double().numpy()
        sh = shard_for_rank(batch.offsets, rank, world)
        lo = sh.local_offsets(batch.offsets)
        xs = x[sh.row_start:sh.row_end]
        m1 = oracle.merge_batch(xs, lo)
        m2 = oracle.merge_batch(m1.x_out, m1.out_offsets)
        rs = oracle.compose_batch(m1.r, lo, m2.r, m1.out_offsets)
        up = oracle.gather_batch(m2.x_out, m2.out_offsets, rs, lo)
        parts = [None] * world
        dist.all_gather_object(parts, (sh.image_start, sh.image_end, up, rs, np.diff(m2.out_offsets)))
        # Max-over-ranks timing, as bench.py reports it.
        t = torch.tensor([float(rank + 1)], dtype=torch.float64)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        if rank == 0:
            full1 = oracle.merge_batch(x, batch.offsets)
            full2 = oracle.merge_batch(full1.x_out, full1.out_offsets)
            rs_full = oracle.compose_batch(full1.r, batch.offsets, full2.r, full1.out_offsets)
            up_full = oracle.gather_batch(full2.x_out, full2.out_offsets, rs_full, batch.offsets)
            got_up = np.concatenate([p[2] for p in parts])
            got_rs = np.concatenate([p[3] for p in parts])
            got_counts = np.concatenate([p[4] for p in parts])
            ok = (np.array_equal(got_up, up_full) and np.array_equal(got_rs, rs_full)
                  and np.array_equal(got_counts, np.diff(full2.out_offsets))
                  and [p[0] for p in parts] == sorted(p[0] for p in parts)
                  and float(t.item()) == float(world))
            with open(os.path.join(out_dir, "result.txt"), "w") as f:
                f.write("ok" if ok else "mismatch")
        dist.barrier()
    finally:
        dist.destroy_process_group()


@pytest.mark.timeout(300)
def test_two_rank_gloo_shards_concatenate_to_single_result(tmp_path):
    world = 2
    port = _free_port()
    mp.start_processes(_rank_main, args=(world, port, str(tmp_path)), nprocs=world, start_method="spawn")
    assert (tmp_path / "result.txt").read_text() == "ok"
