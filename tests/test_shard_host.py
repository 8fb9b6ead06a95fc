"""Column sharding, host side (no GPU): the column split, the ordered exchange through the C ABI
(adpsgd_shard_combine) between threads and between two gloo processes, and refused arguments.

Every shard must end up with the same totals, equal to the partial sums added in shard order
from 0, so that every shard of a column-split run takes the same decisions."""
import os
import socket
import sys
import threading

import numpy as np
import pytest

from paper_2007_06134_gb300 import abi, shard

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.mark.parametrize("P,g", [(0, 1), (3, 1), (4, 2), (4099, 3), (11_689_512, 8), (138_357_544, 4), (10, 4)])
def test_column_split_covers_the_columns(P, g):
    ranges = [shard.column_split(P, g, r) for r in range(g)]
    assert ranges[0][0] == 0
    for (a0, an), (b0, _) in zip(ranges, ranges[1:]):
        assert b0 == a0 + an
    assert ranges[-1][0] + ranges[-1][1] == P
    assert all(c0 % 4 == 0 and cn >= 0 for c0, cn in ranges)
    assert all(cn % 4 == 0 for _, cn in ranges[:-1])  # only the last shard is ragged
    full = [cn // 4 for _, cn in ranges]
    assert max(full) - min(full) <= 1
    with pytest.raises(ValueError):
        shard.column_split(P, g, g)


def _ordered_sum(parts):
    out = np.zeros_like(parts[0])
    for p in parts:
        out = out + p
    return out


def test_combine_between_threads_sums_in_shard_order():
    g, count = 3, 5
    rng = np.random.default_rng(1)
    # values whose sum depends on the order (so a wrong order shows)
    parts = [rng.standard_normal(count) * 10.0 ** rng.integers(-8, 8, count) for _ in range(g)]
    tg = shard.ThreadGather(g)
    results = [None] * g

    def work(r):
        sh = abi.make_shard(g, r, 4 * r, 4 * g, tg.callbacks[r])
        results[r] = abi.adpsgd_shard_combine(sh, parts[r])

    threads = [threading.Thread(target=work, args=(r,)) for r in range(g)]
    for t in threads:
        t.start()
    for t in threads:
        t.join(60)
    want = _ordered_sum(parts)
    for r in range(g):
        assert np.array_equal(results[r], want), r


def test_single_shard_needs_no_gather():
    sh = abi.make_shard(1, 0, 0, 16)
    assert np.array_equal(abi.adpsgd_shard_combine(sh, [1.5, -2.0]), np.array([1.5, -2.0]))


def test_refused_arguments_and_failed_exchange():
    bad = [abi.make_shard(0, 0, 0, 4), abi.make_shard(2, 2, 0, 8), abi.make_shard(2, 0, 2, 8),
           abi.make_shard(2, 0, -4, 8), abi.make_shard(2, 0, 0, 8)]  # the last: no gather with 2 shards
    for sh in bad:
        with pytest.raises(abi.AdpsgdError) as e:
            abi.adpsgd_shard_combine(sh, [1.0])
        assert e.value.status == abi.E_INVAL
    failing = abi.GATHER_FN(lambda local, count, gathered, user: 3)
    with pytest.raises(abi.AdpsgdError) as e:
        abi.adpsgd_shard_combine(abi.make_shard(2, 0, 0, 8, failing), [1.0, 2.0])
    assert e.value.status == abi.E_PEER and "3" in str(e.value)
    with pytest.raises(abi.AdpsgdError) as e:
        abi._check(abi.load().adpsgd_set_shard(None, None), "adpsgd_set_shard")
    assert e.value.status == abi.E_INVAL


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _gloo_worker(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    sys.path.insert(0, ROOT)
    import torch.distributed as dist

    from paper_2007_06134_gb300 import abi as A
    from paper_2007_06134_gb300 import shard as S
    dist.init_process_group("gloo", rank=rank, world_size=world)
    cb, _ = S.dist_gather()
    col0, cols = S.column_split(4099, world, rank)
    sh = A.make_shard(world, rank, col0, 4099, cb)
    local = np.array([1e16 if rank == 0 else 1.0, 0.1 * (rank + 1), -3.0 * rank])
    got = A.adpsgd_shard_combine(sh, local)
    q.put((rank, got.tolist()))
    dist.destroy_process_group()


def test_combine_between_two_gloo_processes():
    import torch.multiprocessing as mp
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_gloo_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(180)
        assert p.exitcode == 0
    got = dict(q.get(timeout=10) for _ in range(2))
    want = [(0.0 + 1e16) + 1.0, (0.0 + 0.1) + 0.2, (0.0 + -0.0) + -3.0]
    assert got[0] == got[1] == want


def _replica_worker(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    sys.path.insert(0, ROOT)
    import torch
    import torch.distributed as dist

    from paper_2007_06134_gb300 import abi as A
    from paper_2007_06134_gb300 import shard as S
    dist.init_process_group("gloo", rank=rank, world_size=world)
    n_locals = [2, 1]
    P = 4 * 5 + 3
    x = torch.arange(n_locals[rank] * P, dtype=torch.float32).reshape(n_locals[rank], P) + 1000.0 * rank
    c0, cols = S.column_split(P, world, rank)
    chunk = torch.full((sum(n_locals), cols), -1.0)
    coll = S.DistReplicaCollective(x, chunk, n_locals)
    assert coll.callback(A.SCATTER_COLUMNS, None) == 0
    scattered = chunk.clone()
    chunk[0] = 0.5 + rank + torch.arange(cols, dtype=torch.float32)  # stands in for the chunk's mean
    assert coll.callback(A.GATHER_AVERAGE, None) == 0
    q.put((rank, scattered.tolist(), x.tolist()))
    dist.destroy_process_group()


def test_replica_split_collectives_between_two_gloo_processes():
    # The all-to-all leaves every process all replicas' values of its column chunk, rows in global
    # replica order (process 0's two replicas, then process 1's); the all-gather writes every
    # chunk's row 0 into every local replica.
    import torch.multiprocessing as mp
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_replica_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(180)
        assert p.exitcode == 0
    got = dict((r, (np.array(a), np.array(b))) for r, a, b in (q.get(timeout=10) for _ in range(2)))
    P = 23
    x_all = np.concatenate([np.arange(2 * P, dtype=np.float32).reshape(2, P),
                            np.arange(P, dtype=np.float32).reshape(1, P) + 1000.0])
    mean_row = np.concatenate([0.5 + r + np.arange(shard.column_split(P, 2, r)[1], dtype=np.float32)
                               for r in range(2)])
    for r in range(2):
        c0, cols = shard.column_split(P, 2, r)
        scattered, x_after = got[r]
        assert np.array_equal(scattered, x_all[:, c0:c0 + cols])
        assert np.array_equal(x_after, np.repeat(mean_row[None, :], x_after.shape[0], axis=0))


def _leaving_worker(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    sys.path.insert(0, ROOT)
    import datetime

    import torch.distributed as dist

    from paper_2007_06134_gb300 import abi as A
    from paper_2007_06134_gb300 import shard as S
    dist.init_process_group("gloo", rank=rank, world_size=world, timeout=datetime.timedelta(seconds=20))
    group = dist.new_group(backend="gloo", timeout=datetime.timedelta(seconds=5))
    cb, _ = S.dist_gather(group)
    def report(value):
        q.put((rank, value))
        q.close()
        q.join_thread()  # the message is sent before the process ends

    if rank == 1:
        report("left")
        os._exit(0)  # this rank leaves between syncs, without a word to the others
    sh = A.make_shard(world, rank, 0, 8, cb)
    try:
        A.adpsgd_shard_combine(sh, [1.0, 2.0])
        report("no error")
    except A.AdpsgdError as e:
        report(e.status)
    os._exit(0)


def test_a_rank_that_leaves_is_reported_as_a_peer_failure():
    # Failure detection on the host: when a shard's process is gone, the exchange runs out its
    # process-group timeout and the library reports ADPSGD_E_PEER instead of hanging.
    import torch.multiprocessing as mp
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_leaving_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    got = dict(q.get(timeout=120) for _ in range(2))
    for p in procs:
        p.join(60)
    assert got[1] == "left"
    assert got[0] == abi.E_PEER
