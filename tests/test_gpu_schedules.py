"""Schedule variants and the per-iteration variance record through the C ABI on the GPU.

Piecewise-constant periods (the strategies of Sec. III-A, the decreasing period of Sec. V-B)
must sync where the oracle syncs (the paper's counts: 750, 750, 500) with bit-exact state, and
the recorded Var[W_k] (Sec. II-B) must match the oracle's within 1e-4, exactly 0 after syncs."""
import numpy as np
import pytest

from oracle import oracle as O
from paper_2007_06134_gb300 import abi, diagnostics, inputs

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
DEV = "cuda:0"
REL = 1e-4


def dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).to(DEV)


def _run(w, n, P, sched, spec, var=False, fused=False):
    h, c = inputs.problem(w, P)
    x, v = inputs.zero_state(n, P)
    xd, vd = dev(x), dev(v)
    cfg = abi.make_config(n, P, momentum=w.mu, weight_decay=w.wd, noise_sigma=w.sigma, seed=w.seed,
                          fuse_intervals=fused)
    tr = abi.TraceBuffers(sched.K + 1, var_cap=sched.K if var else 0)
    with abi.adpsgd_init(cfg, xd, vd, dev(h), dev(c)) as ctx:
        stats = abi.adpsgd_run(ctx, sched, abi.adpsgd_state_init(sched), trace=tr)
    torch.cuda.synchronize()
    otr = O.run(x, v, h, c, spec=spec, seed=w.seed, mu=w.mu, wd=w.wd, sigma=w.sigma, track_variance=var)
    return tr.arrays(), stats, xd.cpu().numpy(), vd.cpu().numpy(), otr, x, v


@pytest.mark.parametrize("p0,p1,expect", [(4, 8, 750), (8, 4, 750), (20, 5, 500)])
@pytest.mark.parametrize("fused", [False, True])
def test_piecewise_strategies(p0, p1, expect, fused):
    w = inputs.WORKLOADS["strategies-n16"]
    n, P, K = 4, 1031, 4000
    sched = abi.make_schedule(abi.PIECEWISE, K, p0, lr0=w.lr0, lr_factor=w.lr_factor, milestones=w.milestones,
                              period_changes=((2000, p1),))
    spec = O.ScheduleSpec(kind=2, K=K, p_init=p0, lr0=w.lr0, lr_factor=w.lr_factor, milestones=w.milestones,
                          period_changes=((2000, p1),))
    gt, stats, gx, gv, otr, x, v = _run(w, n, P, sched, spec, fused=fused)
    assert stats.rounds == expect == otr.syncs
    assert np.array_equal(gt["k"], otr.k) and np.array_equal(gt["p"], otr.p)
    assert np.array_equal(gx, x) and np.array_equal(gv, v)


@pytest.mark.parametrize("kind", [abi.ADPSGD, abi.CPSGD])
def test_variance_record_matches_oracle(kind):
    w = inputs.WORKLOADS["quadratic-n4-P1M"]
    n, P, K = 4, 4099, 60
    K_s = 15 if kind == abi.ADPSGD else 0
    sched = abi.make_schedule(kind, K, 3, K_s=K_s, lr0=w.lr0)
    spec = O.ScheduleSpec(kind=kind, K=K, p_init=3, K_s=K_s, lr0=w.lr0)
    gt, stats, gx, gv, otr, x, v = _run(w, n, P, sched, spec, var=True)
    var, ovar = gt["var"], otr.var
    assert var.shape == ovar.shape == (K,)
    for k in range(K):
        if ovar[k] == 0.0:
            assert var[k] == 0.0, k
        else:
            assert abs(var[k] - ovar[k]) <= REL * ovar[k], (k, var[k], ovar[k])
    assert var[0] == 0.0 and all(var[k + 1] == 0.0 for k in gt["k"] if k + 1 < K)
    # the paper's summaries agree too
    Vt, oVt = diagnostics.interval_means(var, gt["k"]), diagnostics.interval_means(ovar, otr.k)
    assert np.allclose(Vt, oVt, rtol=REL)
    assert np.array_equal(gx, x)


def test_variance_record_rejected_with_fused_intervals():
    w = inputs.WORKLOADS["quadratic-n4-P1M"]
    n, P = 2, 64
    sched = abi.make_schedule(abi.CPSGD, 8, 2, lr0=0.05)
    xd = torch.zeros((n, P), device=DEV)
    z = torch.zeros(P, device=DEV)
    tr = abi.TraceBuffers(16, var_cap=8)
    with abi.adpsgd_init(abi.make_config(n, P, fuse_intervals=True), xd, torch.zeros_like(xd), z, z) as ctx:
        with pytest.raises(abi.AdpsgdError) as e:
            abi.adpsgd_run(ctx, sched, abi.adpsgd_state_init(sched), trace=tr)
    assert e.value.status == abi.E_INVAL


def test_imagenet_style_schedule_run():
    # Sec. IV-C: step-size warm-up stairs, averaging every iteration during the warm-up (K_w), then
    # Algorithm 2; the run must match the oracle bit for bit.
    w = inputs.WORKLOADS["quadratic-n4-P1M"]
    n, P, L = 4, 2053, 5
    kw = dict(lr0=0.01, lr_factor=0.1, milestones=(30 * L, 60 * L), lr_warmup_steps=8, lr_warmup_len=L)
    K = 90 * L
    sched = abi.make_schedule(abi.ADPSGD, K, 4, K_s=8 * L + 100, K_w=8 * L, **kw)
    spec = O.ScheduleSpec(kind=1, K=K, p_init=4, K_s=8 * L + 100, K_w=8 * L, **kw)
    gt, stats, gx, gv, otr, x, v = _run(w, n, P, sched, spec)
    assert np.array_equal(gt["k"], otr.k) and np.array_equal(gt["p"], otr.p)
    assert list(gt["k"][:8 * L]) == list(range(8 * L))
    assert np.array_equal(gx, x) and np.array_equal(gv, v)


@pytest.mark.parametrize("fused", [False, True])
def test_piecewise_change_inside_an_interval(fused):
    w = inputs.WORKLOADS["quadratic-n4-P1M"]
    sched = abi.make_schedule(abi.PIECEWISE, 12, 4, lr0=w.lr0, period_changes=((6, 2),))
    spec = O.ScheduleSpec(kind=2, K=12, p_init=4, lr0=w.lr0, period_changes=((6, 2),))
    gt, stats, gx, gv, otr, x, v = _run(w, 3, 515, sched, spec, fused=fused)
    assert list(gt["k"]) == [3, 6, 8, 10] == list(otr.k)
    assert np.array_equal(gx, x) and np.array_equal(gv, v)
