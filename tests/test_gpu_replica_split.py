"""The replica split (the paper's mapping: each process holds whole replicas, averaging is an
allreduce) on one GPU: g host threads, each a context over its replicas on its own stream, the
allreduce's two halves done by device copies between the threads' buffers
(shard.ThreadReplicaCollective) around the library's averaging kernel on each thread's column
chunk, and the chunk sums exchanged by shard.ThreadGather.  Against one context holding every
replica: each replica's x and v bit-exact, the sync iterations, periods and phases identical, S and
the loss equal up to summation order; and against the oracle."""
import threading

import numpy as np
import pytest

from oracle import oracle as O
from paper_2007_06134_gb300 import abi, inputs, shard

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
DEV = "cuda:0"
SUM_ORDER = 1e-12
GROUP_ROUNDING = 1e-6  # ragged P: scalar kernels against float4 chunks (fp32 group sums of 4 columns)


def _dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).to(DEV)


def _cfg(n, P, bf16, seed):
    return abi.make_config(n, P, momentum=0.9, weight_decay=5e-4, noise_sigma=0.8, seed=seed, want_loss=True,
                           noise_mode=abi.NOISE_BF16 if bf16 else abi.NOISE_PHILOX)


def _problem(n, P):
    w = inputs.WORKLOADS["resnet18-n8"]
    h, c = inputs.draw_h(P, w.h_dist, 14), inputs.draw_c(P, 1.0, 14)
    x, v = inputs.random_state(n, P, 14)
    return w.seed, h, c, x, v


def _single(n, P, sched, bf16, K):
    seed, h, c, x, v = _problem(n, P)
    xd, vd = _dev(x), _dev(v)
    nd = None
    if bf16:
        nd = torch.empty((n, P), dtype=torch.int16, device=DEV)
        abi.adpsgd_noise_fill_bf16(seed, n, P, nd)
    tr = abi.TraceBuffers(K + 1)
    with abi.adpsgd_init(_cfg(n, P, bf16, seed), xd, vd, _dev(h), _dev(c), nd) as ctx:
        stats = abi.adpsgd_run(ctx, sched, abi.adpsgd_state_init(sched), trace=tr)
    torch.cuda.synchronize()
    return xd.cpu().numpy(), vd.cpu().numpy(), tr.arrays(), stats


def _split(n, P, g, sched, bf16, K):
    seed, h, c, x, v = _problem(n, P)
    n_local = n // g
    coll = shard.ThreadReplicaCollective(g, P)
    tg = shard.ThreadGather(g)
    out, errors = [None] * g, []
    ready = threading.Barrier(g, timeout=120)

    def work(r):
        try:
            row0 = r * n_local
            c0, cols = shard.column_split(P, g, r)
            stream = torch.cuda.Stream(device=DEV)
            with torch.cuda.stream(stream):
                xd, vd = _dev(x[row0:row0 + n_local]), _dev(v[row0:row0 + n_local])
                hd, cd = _dev(h), _dev(c)
                chunk = torch.zeros((n, cols), device=DEV)
                nd = None
                if bf16:
                    nd = torch.empty((n_local, P), dtype=torch.int16, device=DEV)
                    abi.adpsgd_noise_fill_bf16_part(seed, n_local, P, row0, 0, nd, stream)
            stream.synchronize()
            coll.register(r, xd, chunk, row0, stream)
            ready.wait()
            tr = abi.TraceBuffers(K + 1)
            with abi.adpsgd_init(_cfg(n_local, P, bf16, seed), xd, vd, hd, cd, nd, stream) as ctx:
                split = abi.make_replica_split(g, r, row0, n, c0, cols, chunk, coll.callbacks[r], tg.callbacks[r])
                abi.adpsgd_set_replica_split(ctx, split)
                stats = abi.adpsgd_run(ctx, sched, abi.adpsgd_state_init(sched), trace=tr)
            stream.synchronize()
            out[r] = (row0, xd.cpu().numpy(), vd.cpu().numpy(), tr.arrays(), stats)
        except Exception as e:  # surfaced below
            errors.append((r, repr(e)))
            coll.barrier.abort()
            tg.barrier.abort()
            ready.abort()

    threads = [threading.Thread(target=work, args=(r,)) for r in range(g)]
    for t in threads:
        t.start()
    for t in threads:
        t.join(300)
    assert not errors, errors
    return out


def _rel(a, b):
    return np.abs(a - b) / np.maximum(np.abs(b), 1e-300)


@pytest.mark.parametrize("n,P,g,bf16", [(4, 4 * 1000 + 2, 4, False), (4, 1 << 16, 2, False), (8, 4 * 3001, 4, True)])
def test_replica_split_equals_one_context(n, P, g, bf16):
    K = 40
    sched = abi.make_schedule(abi.ADPSGD, K, 2, K_s=10, lr0=0.1, milestones=(25,))
    ux, uv, ut, ustats = _single(n, P, sched, bf16, K)
    tol = SUM_ORDER if P % 4 == 0 else GROUP_ROUNDING
    for row0, x, v, t, stats in _split(n, P, g, sched, bf16, K):
        rows = slice(row0, row0 + x.shape[0])
        assert np.array_equal(x.view(np.uint32), ux[rows].view(np.uint32)), row0
        assert np.array_equal(v.view(np.uint32), uv[rows].view(np.uint32)), row0
        for key in ("k", "p", "phase"):
            assert np.array_equal(t[key], ut[key]), key
        for key in ("S", "loss", "C2"):
            assert np.all(_rel(t[key], ut[key]) <= tol), key
        assert stats.rounds == ustats.rounds and stats.wire_bytes_per_node == ustats.wire_bytes_per_node


def test_replica_split_matches_the_oracle():
    n, P, g, K = 4, 4 * 2500, 4, 30
    seed, h, c, x, v = _problem(n, P)
    sched = abi.make_schedule(abi.ADPSGD, K, 3, K_s=9, lr0=0.1)
    parts = _split(n, P, g, sched, False, K)
    spec = O.ScheduleSpec(kind=abi.ADPSGD, K=K, p_init=3, K_s=9, lr0=0.1)
    otr = O.run(x, v, h, c, spec=spec, seed=seed, mu=0.9, wd=5e-4, sigma=0.8)
    for row0, gx, gv, t, _ in parts:
        assert np.array_equal(gx.view(np.uint32), x[row0:row0 + gx.shape[0]].view(np.uint32))
        assert np.array_equal(gv.view(np.uint32), v[row0:row0 + gv.shape[0]].view(np.uint32))
        assert np.array_equal(t["k"], otr.k) and np.array_equal(t["p"], otr.p)
        assert np.all(_rel(t["S"], otr.S) <= 1e-4) and np.all(_rel(t["loss"], otr.loss) <= 1e-4)


def test_replica_split_arguments():
    n, P = 2, 64
    xd = torch.zeros((n, P), device=DEV)
    z = torch.zeros(P, device=DEV)
    chunk = torch.zeros((4, 32), device=DEV)
    noop = abi.COLLECTIVE_FN(lambda op, user: 0)
    gather = abi.GATHER_FN(lambda local, count, gathered, user: 0)
    with abi.adpsgd_init(abi.make_config(n, P), xd, torch.zeros_like(xd), z, z) as ctx:
        bad = [abi.make_replica_split(2, 0, 3, 4, 0, 32, chunk, noop, gather),   # replicas past n_total
               abi.make_replica_split(2, 0, 0, 4, 2, 32, chunk, noop, gather),   # col0 not a multiple of 4
               abi.make_replica_split(2, 0, 0, 4, 40, 32, chunk, noop, gather),  # chunk past P
               abi.make_replica_split(2, 0, 0, 4, 0, 32, chunk, noop, None),     # no gather, two processes
               abi.make_replica_split(2, 2, 0, 4, 0, 32, chunk, noop, gather)]   # rank out of range
        for rs in bad:
            with pytest.raises(abi.AdpsgdError) as e:
                abi.adpsgd_set_replica_split(ctx, rs)
            assert e.value.status == abi.E_INVAL
        with pytest.raises(abi.AdpsgdError) as e:
            abi.adpsgd_set_replica_split(ctx, abi.make_replica_split(1, 0, 0, 2, 0, 32, chunk[:, 1:], noop))
        assert e.value.status == abi.E_ALIGN
    cfg = abi.make_config(n, P, fuse_sync_step=True)
    with abi.adpsgd_init(cfg, xd, torch.zeros_like(xd), z, z) as ctx:
        with pytest.raises(abi.AdpsgdError) as e:
            abi.adpsgd_set_replica_split(ctx, abi.make_replica_split(1, 0, 0, 2, 0, 32, chunk, noop))
        assert e.value.status == abi.E_INVAL
