"""Column sharding on one GPU: a problem split into g column ranges, each a context of its own on
its own stream and host thread, exchanging the two fp64 partial sums at every sync through the
C ABI's gather callback (shard.ThreadGather).  Against the unsharded run of the same problem: x and
v bit-exact on every column (the noise of column j is drawn from the global Philox block j div 4),
the sync iterations, periods and phases identical, S and the loss equal up to the order of fp64
additions.  The same with the bf16 noise tensor filled per shard, with fused sync steps and fused
intervals, with the per-iteration variance record, and against the oracle."""
import threading

import numpy as np
import pytest

from oracle import oracle as O
from paper_2007_06134_gb300 import abi, inputs, shard

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
DEV = "cuda:0"
# S and the loss of a sharded run against the unsharded run.  With P % 4 == 0 every shard takes
# the same float4 column groups as the unsharded run, whose fp32 group sums are then identical, and
# only the order of the fp64 additions differs.  A ragged P runs the scalar kernels (one fp64 add
# per column instead of one per fp32 group sum of four columns) where the shards' float4 kernels
# differ from it by the fp32 rounding of those group sums, about 2^-24 relative.
SUM_ORDER = 1e-12
GROUP_ROUNDING = 1e-6


def _dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).to(DEV)


def _cfg(n, P, *, bf16, mode, seed):
    return abi.make_config(n, P, momentum=0.9, weight_decay=5e-4, noise_sigma=0.8, seed=seed, want_loss=True,
                           noise_mode=abi.NOISE_BF16 if bf16 else abi.NOISE_PHILOX,
                           fuse_sync_step=mode == "sync_step", fuse_intervals=mode == "intervals")


def _problem(n, P):
    w = inputs.WORKLOADS["resnet18-n8"]
    h, c = inputs.draw_h(P, w.h_dist, 12), inputs.draw_c(P, 1.0, 12)
    x, v = inputs.random_state(n, P, 12)
    return w.seed, h, c, x, v


def _unsharded(n, P, sched, *, bf16, mode, track, K):
    seed, h, c, x, v = _problem(n, P)
    xd, vd = _dev(x), _dev(v)
    nd = None
    if bf16:
        nd = torch.empty((n, P), dtype=torch.int16, device=DEV)
        abi.adpsgd_noise_fill_bf16(seed, n, P, nd)
    tr = abi.TraceBuffers(K + 1, var_cap=K if track else 0)
    with abi.adpsgd_init(_cfg(n, P, bf16=bf16, mode=mode, seed=seed), xd, vd, _dev(h), _dev(c), nd) as ctx:
        stats = abi.adpsgd_run(ctx, sched, abi.adpsgd_state_init(sched), trace=tr)
    torch.cuda.synchronize()
    return xd.cpu().numpy(), vd.cpu().numpy(), tr.arrays(), stats


def _sharded(n, P, g, sched, *, bf16, mode, track, K):
    seed, h, c, x, v = _problem(n, P)
    tg = shard.ThreadGather(g)
    out = [None] * g
    errors = []

    def work(r):
        try:
            col0, cols = shard.column_split(P, g, r)
            stream = torch.cuda.Stream(device=DEV)
            with torch.cuda.stream(stream):
                xd = _dev(x[:, col0:col0 + cols])
                vd = _dev(v[:, col0:col0 + cols])
                hd, cd = _dev(h[col0:col0 + cols]), _dev(c[col0:col0 + cols])
                nd = None
                if bf16:
                    nd = torch.empty((n, cols), dtype=torch.int16, device=DEV)
                    abi.adpsgd_noise_fill_bf16_part(seed, n, cols, 0, col0, nd, stream)
            stream.synchronize()
            tr = abi.TraceBuffers(K + 1, var_cap=K if track else 0)
            with abi.adpsgd_init(_cfg(n, cols, bf16=bf16, mode=mode, seed=seed), xd, vd, hd, cd, nd, stream) as ctx:
                abi.adpsgd_set_shard(ctx, abi.make_shard(g, r, col0, P, tg.callbacks[r]))
                stats = abi.adpsgd_run(ctx, sched, abi.adpsgd_state_init(sched), trace=tr)
            stream.synchronize()
            out[r] = (col0, cols, xd.cpu().numpy(), vd.cpu().numpy(), tr.arrays(), stats)
        except Exception as e:  # surfaced below
            errors.append((r, e))
            tg.barrier.abort()

    threads = [threading.Thread(target=work, args=(r,)) for r in range(g)]
    for t in threads:
        t.start()
    for t in threads:
        t.join(300)
    assert not errors, errors
    return out


def _rel(a, b):
    return np.abs(a - b) / np.maximum(np.abs(b), 1e-300)


@pytest.mark.parametrize("n,P,g,bf16,mode,track", [
    (8, 4 * 1000 + 3, 3, False, "unfused", True),      # ragged last shard, variance record
    (8, 1 << 18, 2, False, "sync_step", False),         # the bench's launch form
    (4, 4 * 777, 4, False, "intervals", False),
    (16, 4 * 2049, 2, True, "sync_step", False),        # bf16 noise tensor filled per shard
    (12, 4 * 3001, 3, False, "sync_step", False),       # the two-halves form of the fused step
])
def test_sharded_run_equals_unsharded_run(n, P, g, bf16, mode, track):
    K = 48
    sched = abi.make_schedule(abi.ADPSGD, K, 2, K_s=12, lr0=0.1, milestones=(30,))
    ux, uv, ut, ustats = _unsharded(n, P, sched, bf16=bf16, mode=mode, track=track, K=K)
    parts = _sharded(n, P, g, sched, bf16=bf16, mode=mode, track=track, K=K)
    tol = SUM_ORDER if P % 4 == 0 else GROUP_ROUNDING
    for col0, cols, x, v, t, stats in parts:
        assert np.array_equal(x.view(np.uint32), ux[:, col0:col0 + cols].view(np.uint32)), col0
        assert np.array_equal(v.view(np.uint32), uv[:, col0:col0 + cols].view(np.uint32)), col0
        for key in ("k", "p", "phase"):
            assert np.array_equal(t[key], ut[key]), key
        for key in ("S", "loss", "C2"):
            assert np.all(_rel(t[key], ut[key]) <= tol), key
        if track:
            assert np.all((_rel(t["var"][1:], ut["var"][1:]) <= tol))
        assert stats.rounds == ustats.rounds
        assert stats.wire_bytes_per_node == ustats.wire_bytes_per_node  # accounted on the whole P
    # every shard saw the same totals, bit for bit
    for _, _, _, _, t, _ in parts[1:]:
        assert np.array_equal(t["S"], parts[0][4]["S"]) and np.array_equal(t["loss"], parts[0][4]["loss"])


def test_sharded_run_matches_the_oracle():
    n, P, g, K = 8, 4 * 5000 + 2, 3, 40
    seed, h, c, x, v = _problem(n, P)
    sched = abi.make_schedule(abi.ADPSGD, K, 3, K_s=10, lr0=0.1)
    parts = _sharded(n, P, g, sched, bf16=False, mode="sync_step", track=False, K=K)
    spec = O.ScheduleSpec(kind=abi.ADPSGD, K=K, p_init=3, K_s=10, lr0=0.1)
    otr = O.run(x, v, h, c, spec=spec, seed=seed, mu=0.9, wd=5e-4, sigma=0.8)
    for col0, cols, gx, gv, t, _ in parts:
        assert np.array_equal(gx.view(np.uint32), x[:, col0:col0 + cols].view(np.uint32))
        assert np.array_equal(gv.view(np.uint32), v[:, col0:col0 + cols].view(np.uint32))
        assert np.array_equal(t["k"], otr.k) and np.array_equal(t["p"], otr.p)
        assert np.all(_rel(t["S"], otr.S) <= 1e-4) and np.all(_rel(t["loss"], otr.loss) <= 1e-4)


def test_shard_arguments_checked_against_the_context():
    n, P = 2, 64
    xd = torch.zeros((n, P), device=DEV)
    z = torch.zeros(P, device=DEV)
    with abi.adpsgd_init(abi.make_config(n, P), xd, torch.zeros_like(xd), z, z) as ctx:
        for sh in (abi.make_shard(1, 0, 0, P - 1),          # P_total < col0 + P
                   abi.make_shard(1, 0, 4 << 32, (4 << 32) + P),  # Philox block beyond 2^32
                   abi.make_shard(2, 1, 8, 128)):           # no gather for two shards
            with pytest.raises(abi.AdpsgdError) as e:
                abi.adpsgd_set_shard(ctx, sh)
            assert e.value.status == abi.E_INVAL
        abi.adpsgd_set_shard(ctx, abi.make_shard(1, 0, 0, P))
        D, _ = abi.adpsgd_average_and_variance(ctx)
        assert D == 0.0
