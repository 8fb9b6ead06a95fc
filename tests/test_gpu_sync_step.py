"""The fused sync step (cfg.fuse_sync_step): the local step of every iteration that ends with a
sync, and that averaging, run as one kernel.  Whole runs must match the oracle exactly as the
unfused path does (x, v, the mean and the schedule bit-exact; D and the loss within 1e-4), and
match the unfused path itself.  Shapes the kernel does not take fall back to the separate
kernels: P not a multiple of 4, more than 16 replicas."""
import numpy as np
import pytest

from oracle import oracle as O
from paper_2007_06134_gb300 import abi, inputs

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
DEV = "cuda:0"
REL = 1e-4


def dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).to(DEV)


def host(t):
    torch.cuda.synchronize()
    return t.cpu().numpy()


def rel(a, b):
    return abs(a - b) / max(abs(b), 1e-300)


def _run(n, P, K, kind, p, *, fused, wd=5e-4, bf16=False, loss=True, K_s=0, milestones=(), seed=3,
         track=False, state=None):
    w = inputs.WORKLOADS["resnet18-n8"]
    h, c = inputs.draw_h(P, w.h_dist, seed), inputs.draw_c(P, 1.0, seed)
    x, v = inputs.random_state(n, P, seed)
    noise = O.noise_bf16(w.seed, n, P) if bf16 else None
    xd, vd = dev(x), dev(v)
    cfg = abi.make_config(n, P, momentum=0.9, weight_decay=wd, noise_sigma=0.8, seed=w.seed, want_loss=loss,
                          noise_mode=abi.NOISE_BF16 if bf16 else abi.NOISE_PHILOX, fuse_sync_step=fused)
    sched = abi.make_schedule(kind, K, p, K_s=K_s, lr0=0.1, milestones=milestones)
    tr = abi.TraceBuffers(K + 1, var_cap=K if track else 0)
    with abi.adpsgd_init(cfg, xd, vd, dev(h), dev(c), dev(noise.view(np.int16)) if bf16 else None) as ctx:
        stats = abi.adpsgd_run(ctx, sched, abi.adpsgd_state_init(sched), trace=tr)
    return dict(trace=tr.arrays(), stats=stats, x=host(xd), v=host(vd), inputs=(h, c, x, v, noise),
                spec=O.ScheduleSpec(kind=kind, K=K, p_init=p, K_s=K_s, lr0=0.1, milestones=milestones),
                wd=wd, seed=w.seed)


def _against_oracle(r, loss=True):
    h, c, x, v, noise = r["inputs"]
    otr = O.run(x, v, h, c, spec=r["spec"], seed=r["seed"], mu=0.9, wd=r["wd"], sigma=0.8, noise=noise)
    g = r["trace"]
    assert np.array_equal(g["k"], otr.k) and np.array_equal(g["p"], otr.p) and np.array_equal(g["phase"], otr.phase)
    for a, b in zip(g["S"], otr.S):
        assert rel(a, b) < REL
    if loss:
        for a, b in zip(g["loss"], otr.loss):
            assert rel(a, b) < REL
    assert np.array_equal(r["x"].view(np.uint32), x.view(np.uint32))
    assert np.array_equal(r["v"].view(np.uint32), v.view(np.uint32))


# Up to 8 replicas take the register form, 9..16 with Philox noise the two-halves form and 9..16
# with the bf16 noise tensor the 16-replica register form.
@pytest.mark.parametrize("n,bf16", [(1, False), (2, False), (3, False), (5, False), (8, False), (9, False),
                                    (12, False), (16, False), (12, True), (16, True)])
@pytest.mark.parametrize("kind", [abi.ADPSGD, abi.CPSGD])
def test_runs_match_the_oracle(n, bf16, kind):
    P, K = 4096 + 4 * 37, 60
    r = _run(n, P, K, kind, 4, fused=True, bf16=bf16, K_s=16 if kind == abi.ADPSGD else 0, milestones=(30,))
    assert r["stats"].sync_step_launches > 0
    assert r["stats"].sync_step_launches + r["stats"].average_launches == r["stats"].rounds
    _against_oracle(r)


@pytest.mark.parametrize("bf16,wd,loss", [(True, 0.0, True), (False, 0.0, False), (True, 5e-4, False)])
def test_noise_modes_weight_decay_and_no_loss(bf16, wd, loss):
    r = _run(8, 8192, 40, abi.ADPSGD, 3, fused=True, wd=wd, bf16=bf16, loss=loss, K_s=9)
    assert r["stats"].sync_step_launches > 0
    _against_oracle(r, loss=loss)


@pytest.mark.parametrize("n", [3, 4, 6, 8, 12])
def test_several_groups_per_thread(n):
    # At 2^20 + 148 columns every thread of the fused step's persistent grid takes several column
    # groups in its grid-stride loop: whole runs bit-exact against the oracle (all host cores).
    P, K = (1 << 20) + 4 * 37, 12
    w = inputs.WORKLOADS["resnet18-n8"]
    h, c = inputs.draw_h(P, w.h_dist, 8), inputs.draw_c(P, 1.0, 8)
    x, v = inputs.random_state(n, P, 8)
    xd, vd = dev(x), dev(v)
    cfg = abi.make_config(n, P, momentum=0.9, weight_decay=5e-4, noise_sigma=0.8, seed=w.seed, fuse_sync_step=True)
    sched = abi.make_schedule(abi.ADPSGD, K, 2, K_s=4, lr0=0.1)
    tr = abi.TraceBuffers(K + 1)
    with abi.adpsgd_init(cfg, xd, vd, dev(h), dev(c)) as ctx:
        st = abi.adpsgd_run(ctx, sched, abi.adpsgd_state_init(sched), trace=tr)
    assert st.sync_step_launches > 0
    spec = O.ScheduleSpec(kind=abi.ADPSGD, K=K, p_init=2, K_s=4, lr0=0.1)
    otr = O.run(x, v, h, c, spec=spec, seed=w.seed, mu=0.9, wd=5e-4, sigma=0.8, threads=O.host_threads())
    g = tr.arrays()
    assert np.array_equal(g["k"], otr.k) and np.array_equal(g["p"], otr.p)
    for a, b in zip(g["S"], otr.S):
        assert rel(a, b) < REL
    for a, b in zip(g["loss"], otr.loss):
        assert rel(a, b) < REL
    assert np.array_equal(host(xd).view(np.uint32), x.view(np.uint32))
    assert np.array_equal(host(vd).view(np.uint32), v.view(np.uint32))


def test_two_halves_form_at_2_24_columns():
    # 16 replicas with Philox noise take the two-halves form; at 2^24 columns every thread of its
    # persistent grid takes dozens of column groups.  Every sync against the all-core oracle, and
    # x, v bit-exact at the end.
    n, P, K = 16, 1 << 24, 24
    w = inputs.WORKLOADS["resnet18-n8"]
    h, c = inputs.draw_h(P, w.h_dist, 11), inputs.draw_c(P, 1.0, 11)
    x, v = inputs.random_state(n, P, 11)
    xd, vd = dev(x), dev(v)
    cfg = abi.make_config(n, P, momentum=0.9, weight_decay=5e-4, noise_sigma=0.8, seed=w.seed, fuse_sync_step=True)
    sched = abi.make_schedule(abi.ADPSGD, K, 2, K_s=6, lr0=0.1)
    tr = abi.TraceBuffers(K + 1)
    with abi.adpsgd_init(cfg, xd, vd, dev(h), dev(c)) as ctx:
        st = abi.adpsgd_run(ctx, sched, abi.adpsgd_state_init(sched), trace=tr)
    # syncs one iteration apart (p = 1) keep the two kernels for the step enqueued ahead of a wait
    assert st.sync_step_launches > 0 and st.sync_step_launches + st.average_launches == st.rounds
    spec = O.ScheduleSpec(kind=abi.ADPSGD, K=K, p_init=2, K_s=6, lr0=0.1)
    otr = O.run(x, v, h, c, spec=spec, seed=w.seed, mu=0.9, wd=5e-4, sigma=0.8, threads=O.host_threads())
    g = tr.arrays()
    assert np.array_equal(g["k"], otr.k) and np.array_equal(g["p"], otr.p) and np.array_equal(g["phase"], otr.phase)
    for a, b in zip(g["S"], otr.S):
        assert rel(a, b) < REL
    for a, b in zip(g["loss"], otr.loss):
        assert rel(a, b) < REL
    assert np.array_equal(host(xd).view(np.uint32), x.view(np.uint32))
    assert np.array_equal(host(vd).view(np.uint32), v.view(np.uint32))


def test_fused_equals_unfused_at_a_larger_size():
    args = dict(n=8, P=(1 << 20) + 4 * 11, K=120, kind=abi.ADPSGD, p=4, K_s=30, milestones=(60, 90))
    a = _run(fused=False, **args)
    b = _run(fused=True, **args)
    assert a["stats"].sync_step_launches == 0 and b["stats"].sync_step_launches > 0
    for key in ("k", "p", "phase"):
        assert np.array_equal(a["trace"][key], b["trace"][key])
    assert np.array_equal(a["x"], b["x"]) and np.array_equal(a["v"], b["v"])
    # S (and C2, built from it) differ only by the order of fp64 additions
    for key in ("S", "C2"):
        for s1, s2 in zip(a["trace"][key], b["trace"][key]):
            assert rel(s1, s2) < 1e-6


@pytest.mark.parametrize("n,P", [(17, 4096), (8, 4099), (4, 1), (12, 4094)])
def test_unsupported_shapes_fall_back(n, P):
    r = _run(n, P, 30, abi.CPSGD, 3, fused=True)
    assert r["stats"].sync_step_launches == 0 and r["stats"].average_launches == r["stats"].rounds
    _against_oracle(r)


def test_variance_record_with_fused_sync_steps():
    a = _run(4, 4096, 40, abi.ADPSGD, 3, fused=False, K_s=10, track=True)
    b = _run(4, 4096, 40, abi.ADPSGD, 3, fused=True, K_s=10, track=True)
    assert b["stats"].sync_step_launches > 0
    for s1, s2 in zip(a["trace"]["var"], b["trace"]["var"]):
        assert rel(s1, s2) < 1e-6 or s1 == s2 == 0.0
    assert np.array_equal(a["x"], b["x"])


def test_kernel_times_count_the_sync_steps():
    n, P, K = 4, 4096, 24
    x, v = inputs.random_state(n, P, 1)
    xd, vd = dev(x), dev(v)
    z = torch.zeros(P, device=DEV)
    cfg = abi.make_config(n, P, fuse_sync_step=True, time_kernels=1)
    sched = abi.make_schedule(abi.CPSGD, K, 4, lr0=0.1)
    with abi.adpsgd_init(cfg, xd, vd, z, z) as ctx:
        st = abi.adpsgd_run(ctx, sched, abi.adpsgd_state_init(sched))
        t = abi.adpsgd_kernel_times(ctx)
    assert st.sync_step_launches == t["sync_step_launches"] == 6
    assert t["local_step_launches"] == K - 6 and t["average_launches"] == 0 and t["sync_step_ms"] > 0


@pytest.mark.parametrize("split", [17, 20, 33])
def test_resume_with_fused_sync_steps(split):
    # One call against two calls split at iteration `split` (CPSGD p = 4: 20 ends right after a
    # sync, 17 and 33 fall inside an interval): x, v and the schedule are bit-identical.
    n, P, K = 8, 4096 + 64, 48
    w = inputs.WORKLOADS["resnet18-n8"]
    h, c = inputs.draw_h(P, w.h_dist, 4), inputs.draw_c(P, 1.0, 4)
    x0, v0 = inputs.random_state(n, P, 4)
    cfg = abi.make_config(n, P, momentum=0.9, weight_decay=5e-4, noise_sigma=0.8, seed=9, fuse_sync_step=True)
    sched = abi.make_schedule(abi.CPSGD, K, 4, lr0=0.1)
    out = []
    for calls in ([K], [split, K]):
        xd, vd = dev(x0), dev(v0)
        tr = abi.TraceBuffers(K + 1)
        with abi.adpsgd_init(cfg, xd, vd, dev(h), dev(c)) as ctx:
            st = abi.adpsgd_state_init(sched)
            for k_end in calls:
                abi.adpsgd_run(ctx, sched, st, k_end=k_end, trace=tr)
        out.append((host(xd), host(vd), tr.arrays(), st))
    (xa, va, ta, sa), (xb, vb, tb, sb) = out
    assert np.array_equal(xa.view(np.uint32), xb.view(np.uint32))
    assert np.array_equal(va.view(np.uint32), vb.view(np.uint32))
    assert np.array_equal(ta["k"], tb["k"]) and np.array_equal(ta["p"], tb["p"])
    for s1, s2 in zip(ta["S"], tb["S"]):
        assert rel(s1, s2) < 1e-12
    assert (sa.k_next, sa.cnt, sa.p, sa.rounds) == (sb.k_next, sb.cnt, sb.p, sb.rounds)


@pytest.mark.parametrize("fused", [False, True])
def test_noise_free_identical_replicas(fused):
    # sigma = 0 from a shared start: the replicas stay identical, every sync reports D = 0 exactly
    # (the exact-zero test, no fp64 path) and Algorithm 2 keeps p (0 is neither < 0.7 nor > 1.3
    # times gamma C2 = 0).  x matches the oracle bit for bit.
    n, P, K = 8, 4096, 40
    w = inputs.WORKLOADS["resnet18-n8"]
    h, c = inputs.draw_h(P, w.h_dist, 6), inputs.draw_c(P, 1.0, 6)
    base, _ = inputs.random_state(1, P, 6)
    x = np.repeat(base, n, axis=0)
    v = np.zeros_like(x)
    xd, vd = dev(x), dev(v)
    cfg = abi.make_config(n, P, momentum=0.9, weight_decay=5e-4, noise_sigma=0.0, seed=1, fuse_sync_step=fused)
    sched = abi.make_schedule(abi.ADPSGD, K, 3, K_s=9, lr0=0.1)
    tr = abi.TraceBuffers(K + 1)
    with abi.adpsgd_init(cfg, xd, vd, dev(h), dev(c)) as ctx:
        st = abi.adpsgd_run(ctx, sched, abi.adpsgd_state_init(sched), trace=tr)
    g = tr.arrays()
    assert (st.sync_step_launches > 0) == fused
    assert np.all(g["S"] == 0.0) and np.all(g["p"] == 3) and np.all(g["C2"] == 0.0)
    spec = O.ScheduleSpec(kind=abi.ADPSGD, K=K, p_init=3, K_s=9, lr0=0.1)
    otr = O.run(x, v, h, c, spec=spec, seed=1, mu=0.9, wd=5e-4, sigma=0.0)
    assert np.array_equal(g["k"], otr.k) and np.all(otr.S == 0.0)
    assert np.array_equal(host(xd).view(np.uint32), x.view(np.uint32))
