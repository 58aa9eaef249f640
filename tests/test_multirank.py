"""Host-side multi-rank logic (replicas and batch shards, max/sum over ranks),
run as two gloo processes on the CPU."""
import os
import socket
import sys

import pytest
import torch.multiprocessing as mp

from paper_2608_22099_gb300 import multirank


def test_shard_ranges_partition_the_batch():
    for batch in (0, 1, 7, 4096, 4097):
        for world in (1, 2, 3, 8):
            spans = [multirank.shard_range(batch, r, world) for r in range(world)]
            assert spans[0][0] == 0 and spans[-1][1] == batch
            assert all(a[1] == b[0] for a, b in zip(spans, spans[1:]))
            sizes = [b1 - b0 for b0, b1 in spans]
            assert max(sizes) - min(sizes) <= 1
    with pytest.raises(ValueError):
        multirank.shard_range(10, 2, 2)


def test_rank_info_defaults_and_env():
    assert multirank.rank_info({}) == (0, 1, 0)
    assert multirank.rank_info({"RANK": "3", "WORLD_SIZE": "4", "LOCAL_RANK": "1"}) == (3, 4, 1)


def test_single_process_reductions_are_identity():
    assert multirank.max_over_ranks(2.5) == 2.5
    assert multirank.sum_over_ranks(2.5) == 2.5
    assert multirank.job_throughput(10.0, 2.0) == 5.0


def _free_port() -> int:
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _worker(rank, world, port, out_dir):
    import torch.distributed as dist

    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world),
                      LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        r, w, lr = multirank.rank_info()
        assert (r, w, lr) == (rank, world, rank)
        # every rank times its own shard; the job's time is the slowest rank's
        local_time = 1.0 + rank
        t = multirank.max_over_ranks(local_time)
        b0, b1 = multirank.shard_range(4097, rank, world)
        total = multirank.sum_over_ranks(b1 - b0)
        value = multirank.job_throughput(total, t)
        with open(os.path.join(out_dir, f"rank{rank}.txt"), "w") as f:
            f.write(f"{t} {total} {value}\n")
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks(tmp_path):
    world = 2
    mp.start_processes(_worker, args=(world, _free_port(), str(tmp_path)), nprocs=world, start_method="spawn")
    rows = [open(tmp_path / f"rank{r}.txt").read().split() for r in range(world)]
    for t, total, value in rows:
        assert float(t) == 2.0                      # max over ranks of 1.0 and 2.0
        assert float(total) == 4097.0               # the shards cover the batch
        assert float(value) == 4097.0 / 2.0
