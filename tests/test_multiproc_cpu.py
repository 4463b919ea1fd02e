"""bench.py's multi-replica host logic on CPU: world size 2 over gloo (one process per rank, the
way torchrun launches them). Each rank times its own replica; rank 0 reports the max elapsed over
ranks and the tokens summed over ranks (weak scaling, no data-path collective)."""
import os
import socket

import pytest
import torch.multiprocessing as mp


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    p = s.getsockname()[1]
    s.close()
    return p


def _worker(rank, world, port, q):
    import torch.distributed as dist

    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench

    r, w, lr = bench.dist_env()
    el, units = bench.aggregate(elapsed_s=1.0 + rank, units=100.0 * (rank + 1), world=w)
    q.put((r, w, lr, el, units, bench.replica_seed(0, r)))
    dist.barrier()
    dist.destroy_process_group()


@pytest.mark.parametrize("world", [2])
def test_aggregate_over_gloo(world):
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    out = sorted(q.get(timeout=120) for _ in range(world))
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for r, (rank, w, lr, el, units, seed) in enumerate(out):
        assert (rank, w, lr) == (r, world, r)
        assert el == 2.0            # max over ranks
        assert units == 300.0       # sum over ranks
    assert len({o[5] for o in out}) == world  # every replica decodes its own streams


def test_single_rank_is_identity():
    import bench

    assert bench.aggregate(1.5, 10.0, 1) == (1.5, 10.0)
