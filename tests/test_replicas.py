"""Host logic of running N independent replicas (world size 2, gloo, CPU):
every rank draws its own batch, the timed region is lined up by barriers and
the slowest rank's time is what every rank sees."""
import os
import socket

import pytest
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    os.environ.update(RANK=str(rank), LOCAL_RANK=str(rank), WORLD_SIZE=str(world),
                      MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    from paper_2609_18145_gb300 import replicas
    r, lr, w = replicas.env_world()
    assert (r, lr, w) == (rank, rank, world)
    replicas.init("gloo")
    replicas.barrier()
    t = replicas.max_over_ranks(1.5 + rank)          # rank 1 is the slow one
    s = replicas.sum_over_ranks(100.0 * (rank + 1))
    out.put((rank, t, s, replicas.batch_seed(0, rank)))
    replicas.finish()


def test_two_replicas_max_time_and_distinct_batches():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert [r[1] for r in res] == [2.5, 2.5]
    assert [r[2] for r in res] == [300.0, 300.0]
    assert res[0][3] != res[1][3]


def test_single_process_is_identity():
    from paper_2609_18145_gb300 import replicas
    for k in ("RANK", "WORLD_SIZE", "LOCAL_RANK"):
        assert k not in os.environ or os.environ[k] in ("0", "1")
    assert replicas.max_over_ranks(3.25) == 3.25
    assert replicas.sum_over_ranks(2.0) == 2.0
