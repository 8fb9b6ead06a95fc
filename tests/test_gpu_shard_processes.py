"""Column shards as separate processes on one GPU, exchanging their partial sums through
torch.distributed (gloo) with shard.dist_gather -- the plumbing bench.py uses under torchrun.
Two spawned processes each hold half the columns of one problem; every column's x and v must equal
the unsharded run's bit for bit, and both processes must report the same schedule.  (No kernel
of one process waits on the other: the exchange is a host all-gather between syncs.)"""
import os
import socket
import sys

import numpy as np
import pytest

from paper_2007_06134_gb300 import abi, inputs

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
N, P, K = 8, 4 * 3000 + 3, 36


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _problem():
    w = inputs.WORKLOADS["resnet18-n8"]
    h, c = inputs.draw_h(P, w.h_dist, 21), inputs.draw_c(P, 1.0, 21)
    x, v = inputs.random_state(N, P, 21)
    return w.seed, h, c, x, v


def _schedule(A):
    return A.make_schedule(A.ADPSGD, K, 2, K_s=8, lr0=0.1, milestones=(20,))


def _config(A, cols, seed):
    return A.make_config(N, cols, momentum=0.9, weight_decay=5e-4, noise_sigma=0.8, seed=seed, fuse_sync_step=True)


def _rank(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    sys.path.insert(0, ROOT)
    import torch as T
    import torch.distributed as dist

    from paper_2007_06134_gb300 import abi as A
    from paper_2007_06134_gb300 import shard as S
    try:
        dist.init_process_group("gloo", rank=rank, world_size=world)
        seed, h, c, x, v = _problem()
        col0, cols = S.column_split(P, world, rank)
        dev = lambda a: T.from_numpy(np.ascontiguousarray(a)).to("cuda:0")
        xd, vd = dev(x[:, col0:col0 + cols]), dev(v[:, col0:col0 + cols])
        gather, _ = S.dist_gather()
        sched = _schedule(A)
        tr = A.TraceBuffers(K + 1)
        with A.adpsgd_init(_config(A, cols, seed), xd, vd, dev(h[col0:col0 + cols]), dev(c[col0:col0 + cols])) as ctx:
            A.adpsgd_set_shard(ctx, A.make_shard(world, rank, col0, P, gather))
            A.adpsgd_run(ctx, sched, A.adpsgd_state_init(sched), trace=tr)
        T.cuda.synchronize()
        t = tr.arrays()
        q.put((rank, col0, xd.cpu().numpy(), vd.cpu().numpy(), t["k"], t["p"], t["S"]))
        dist.destroy_process_group()
    except Exception as e:  # reported to the parent
        q.put((rank, repr(e)))
        raise


def test_two_processes_share_one_problem_by_columns():
    import torch.multiprocessing as mp
    seed, h, c, x, v = _problem()
    dev = lambda a: torch.from_numpy(np.ascontiguousarray(a)).to("cuda:0")
    xd, vd = dev(x), dev(v)
    sched = _schedule(abi)
    tr = abi.TraceBuffers(K + 1)
    with abi.adpsgd_init(_config(abi, P, seed), xd, vd, dev(h), dev(c)) as ctx:
        abi.adpsgd_run(ctx, sched, abi.adpsgd_state_init(sched), trace=tr)
    torch.cuda.synchronize()
    ux, uv, ut = xd.cpu().numpy(), vd.cpu().numpy(), tr.arrays()

    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    got = [q.get(timeout=300) for _ in range(2)]
    for p in procs:
        p.join(120)
    assert all(len(g) == 7 for g in got), got
    for rank, col0, gx, gv, k, p_, S in got:
        cols = gx.shape[1]
        assert np.array_equal(gx.view(np.uint32), ux[:, col0:col0 + cols].view(np.uint32)), rank
        assert np.array_equal(gv.view(np.uint32), uv[:, col0:col0 + cols].view(np.uint32)), rank
        assert np.array_equal(k, ut["k"]) and np.array_equal(p_, ut["p"])
        # a ragged P: the last shard's scalar kernels against the float4 groups of one context
        assert np.all(np.abs(S - ut["S"]) <= 1e-6 * np.abs(ut["S"]))
    assert np.array_equal(got[0][6], got[1][6])  # both processes saw the same totals
    assert all(p.exitcode == 0 for p in procs)
