"""The bench's multi-rank path on CPU: two gloo ranks, the way torchrun starts
them (RANK / WORLD_SIZE / MASTER_* in the environment). Each rank runs its own
replica (weak scaling, no collective on the data path); the job time is the max
over ranks and the token count the sum."""
import os
import socket

import pytest
import torch.multiprocessing as mp


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _rank_main(rank, world, port, out):
    os.environ.update({"RANK": str(rank), "WORLD_SIZE": str(world), "LOCAL_RANK": str(rank),
                       "MASTER_ADDR": "127.0.0.1", "MASTER_PORT": str(port),
                       "HWKV_BENCH_BACKEND": "gloo"})
    import bench
    import torch.distributed as dist
    w, r, local = bench.dist_setup(world)
    assert (w, r, local) == (world, rank, rank)
    bench.barrier(w)
    t = bench.max_over_ranks(10.0 + rank, w)      # slowest rank sets the job time
    n = bench.sum_over_ranks(16.0 * (rank + 1), w)  # every rank's tokens count
    out[rank] = (t, n)
    dist.destroy_process_group()


@pytest.mark.parametrize("world", [2])
def test_two_rank_aggregation(world):
    port = _free_port()
    with mp.Manager() as m:
        out = m.dict()
        mp.spawn(_rank_main, args=(world, port, out), nprocs=world, join=True)
        res = dict(out)
    assert res[0] == res[1] == (11.0, 48.0)


def test_ranks_get_distinct_inputs():
    """Replicas differ only in their seed: rank r draws from seed + 1000003 r."""
    import hwkv_gen
    a = hwkv_gen.fill_host(hwkv_gen.desc(0), hwkv_gen.K, 0, 1, 0, 4, 1, 8)
    b = hwkv_gen.fill_host(hwkv_gen.desc(1000003), hwkv_gen.K, 0, 1, 0, 4, 1, 8)
    assert (a != b).any()
