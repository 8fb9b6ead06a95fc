"""Temporal fusion (cfg.fuse_intervals): every stretch of local steps up to the next sync and the
sync's averaging run as one kernel.  It must give the oracle's bits exactly like the unfused
path: x, v, the mean and the schedule bit-exact, D and the loss within 1e-4."""
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


def _problem(P, seed=1):
    w = inputs.WORKLOADS["resnet18-n8"]
    return inputs.draw_h(P, w.h_dist, seed), inputs.draw_c(P, 1.0, seed)


@pytest.mark.parametrize("n", [1, 3, 8, 32])
@pytest.mark.parametrize("P", [1, 5, 4099, 65536 + 3, 4096])
@pytest.mark.parametrize("wd", [0.0, 5e-4])
def test_fused_local_steps_bit_exact(n, P, wd):
    h, c = _problem(P)
    x, v = inputs.random_state(n, P, 7)
    seed, k0 = 0xFEEDFACE, 11
    lrs = [0.1, 0.05, 0.05, 0.01, 0.2]
    xd, vd = dev(x), dev(v)
    cfg = abi.make_config(n, P, momentum=0.9, weight_decay=wd, noise_sigma=0.5, seed=seed, fuse_intervals=True)
    with abi.adpsgd_init(cfg, xd, vd, dev(h), dev(c)) as ctx:
        abi.adpsgd_local_steps(ctx, k0, lrs)
        gx, gv = host(xd), host(vd)
    for t, lr in enumerate(lrs):
        O.local_step(x, v, h, c, seed=seed, k=k0 + t, gamma=lr, mu=0.9, wd=wd, sigma=0.5)
    assert np.array_equal(gx.view(np.uint32), x.view(np.uint32))
    assert np.array_equal(gv.view(np.uint32), v.view(np.uint32))


@pytest.mark.parametrize("n,P", [(16, 4096), (4, 4099)])
def test_fused_local_steps_bf16_noise(n, P):
    h, c = _problem(P, 2)
    x, v = inputs.random_state(n, P, 8)
    noise = O.noise_bf16(77, n, P)
    xd, vd = dev(x), dev(v)
    cfg = abi.make_config(n, P, noise_sigma=1.0, seed=77, noise_mode=abi.NOISE_BF16, fuse_intervals=True)
    with abi.adpsgd_init(cfg, xd, vd, dev(h), dev(c), dev(noise.view(np.int16))) as ctx:
        abi.adpsgd_local_steps(ctx, 0, [0.05] * 3)
        gx, gv = host(xd), host(vd)
    for k in range(3):
        O.local_step(x, v, h, c, seed=77, k=k, gamma=0.05, mu=0.9, wd=0.0, sigma=1.0, noise=noise)
    assert np.array_equal(gx, x) and np.array_equal(gv, v)


def _run(w, P, K, kind, p, fused, *, K_s=0, K_w=0, milestones=(), literal=False, n=None):
    n = w.n if n is None else n
    h, c = inputs.problem(w, P)
    x, v = inputs.zero_state(n, P)
    xd, vd = dev(x), dev(v)
    cfg = abi.make_config(n, P, momentum=w.mu, weight_decay=w.wd, noise_sigma=w.sigma, seed=w.seed,
                          fuse_intervals=fused, time_kernels=True)
    sched = abi.make_schedule(kind, K, p, K_s=K_s, K_w=K_w, lr0=w.lr0, lr_factor=w.lr_factor,
                              milestones=milestones, literal_phase=literal)
    tr = abi.TraceBuffers(K + 1)
    with abi.adpsgd_init(cfg, xd, vd, dev(h), dev(c)) as ctx:
        stats = abi.adpsgd_run(ctx, sched, abi.adpsgd_state_init(sched), trace=tr)
        times = abi.adpsgd_kernel_times(ctx)
    return tr.arrays(), stats, times, host(xd), host(vd), (h, c, x, v)


def _oracle(w, P, K, kind, p, hcxv, *, K_s=0, K_w=0, milestones=(), literal=False):
    h, c, x, v = hcxv
    spec = O.ScheduleSpec(kind=kind, K=K, p_init=p, K_s=K_s, K_w=K_w, lr0=w.lr0, lr_factor=w.lr_factor,
                          milestones=milestones, literal_phase=int(literal))
    return O.run(x, v, h, c, spec=spec, seed=w.seed, mu=w.mu, wd=w.wd, sigma=w.sigma), x, v


def _assert_same(gt, otr):
    assert np.array_equal(gt["k"], otr.k) and np.array_equal(gt["p"], otr.p)
    assert np.array_equal(gt["phase"], otr.phase)
    for a, b in zip(gt["S"], otr.S):
        assert rel(a, b) < REL
    for a, b in zip(gt["loss"], otr.loss):
        assert rel(a, b) < REL


@pytest.mark.parametrize("kind", [abi.ADPSGD, abi.CPSGD])
def test_fused_run_full_small_workload(kind):
    w = inputs.WORKLOADS["quadratic-n4-P1M"]
    K_s = w.K_s if kind == abi.ADPSGD else 0
    gt, stats, times, gx, gv, hcxv = _run(w, w.P, w.K, kind, 4, True, K_s=K_s)
    assert stats.interval_launches == stats.rounds and stats.local_step_launches == 0
    assert times["interval_launches"] == stats.rounds
    otr, x, v = _oracle(w, w.P, w.K, kind, 4, hcxv, K_s=K_s)
    _assert_same(gt, otr)
    assert np.array_equal(gx.view(np.uint32), x.view(np.uint32))
    assert np.array_equal(gv.view(np.uint32), v.view(np.uint32))


def test_fused_equals_unfused_with_step_size_milestones():
    w = inputs.WORKLOADS["resnet18-n8"]
    P, K = (1 << 16) + 13, 400
    a = _run(w, P, K, abi.ADPSGD, 4, False, K_s=100, milestones=(200, 300))
    b = _run(w, P, K, abi.ADPSGD, 4, True, K_s=100, milestones=(200, 300))
    for key in ("k", "p", "phase", "C2"):
        assert np.array_equal(a[0][key], b[0][key])
    assert np.array_equal(a[3], b[3]) and np.array_equal(a[4], b[4])
    for s1, s2 in zip(a[0]["S"], b[0]["S"]):
        assert rel(s1, s2) < 1e-6


@pytest.mark.parametrize("p,K,literal,K_w", [(300, 700, False, 0), (3, 20, True, 0), (5, 40, False, 7)])
def test_fused_long_intervals_literal_phase_and_warmup(p, K, literal, K_w):
    # p > 256 splits an interval into chunks; Algorithm 1's literal phase and a warm-up change
    # where the syncs fall.
    w = inputs.WORKLOADS["quadratic-n4-P1M"]
    P = 1031
    kind = abi.CPSGD if K_w == 0 else abi.ADPSGD
    K_s = 0 if K_w == 0 else K_w + p + 1
    gt, stats, _, gx, gv, hcxv = _run(w, P, K, kind, p, True, K_s=K_s, K_w=K_w, literal=literal)
    otr, x, v = _oracle(w, P, K, kind, p, hcxv, K_s=K_s, K_w=K_w, literal=literal)
    _assert_same(gt, otr)
    assert np.array_equal(gx, x) and np.array_equal(gv, v)


def test_fused_requires_at_most_32_replicas():
    n, P = 33, 64
    xd = torch.zeros((n, P), device=DEV)
    z = torch.zeros(P, device=DEV)
    with pytest.raises(abi.AdpsgdError) as e:
        abi.adpsgd_init(abi.make_config(n, P, fuse_intervals=True), xd, torch.zeros_like(xd), z, z)
    assert e.value.status == abi.E_INVAL
