"""Parity at the workloads' full sizes, in the launch configuration the bench times.

The adaptive runs the bench times (Algorithm 2, p_init 4, K_s = K / 4, the loss at every sync;
with fused sync steps, and with fused intervals) are compared with the oracle's chunked all-core
run over all columns at every sync: k, p and the phase bit-exact, S, the loss and C_2 within
1e-4, the final x and v bit-exact.

The surrogate objective is separable per column and the constant-period schedule does not
depend on the data, so the oracle can also follow a full-size constant-period run exactly on a
sample of columns: bit-exact x and v there after every iteration of the run.  The averaging
kernel is checked over all columns (the oracle's averaging is cheap).
"""
import dataclasses

import numpy as np
import pytest

from oracle import oracle as O
from paper_2007_06134_gb300 import abi, inputs

pytestmark = [pytest.mark.gpu, pytest.mark.slow]

torch = pytest.importorskip("torch")
DEV = "cuda:0"
REL = 1e-4
SAMPLE_WIDTH = 1024


def _dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).to(DEV)


def _rel(a, b):
    return abs(a - b) / max(abs(b), 1e-300)


def _sample_ranges(P, count=6):
    """Disjoint column ranges: the first and last SAMPLE_WIDTH columns and one random range
    (start a multiple of 4) inside each of `count` equal segments in between."""
    rng = np.random.default_rng(P)
    ranges = [(0, SAMPLE_WIDTH)]
    seg = (P - 2 * SAMPLE_WIDTH) // count
    for t in range(count):
        lo = SAMPLE_WIDTH + t * seg
        start = lo + 4 * int(rng.integers(0, max(1, (seg - SAMPLE_WIDTH) // 4)))
        ranges.append((start, start + SAMPLE_WIDTH))
    ranges.append((P - SAMPLE_WIDTH, P))
    assert all(a[1] <= b[0] for a, b in zip(ranges, ranges[1:]))
    return ranges


def _cfg(w, noise=False, mode="unfused"):
    return abi.make_config(w.n, w.P, momentum=w.mu, weight_decay=w.wd, noise_sigma=w.sigma, seed=w.seed,
                           noise_mode=abi.NOISE_BF16 if noise else abi.NOISE_PHILOX,
                           fuse_intervals=mode == "intervals", fuse_sync_step=mode == "sync_step")


def _oracle_noise_on_ranges(w, ranges):
    """The bf16 noise tensor on the sampled columns, from the oracle (zero elsewhere)."""
    noise = np.zeros((w.n, w.P), np.uint16)
    for j0, j1 in ranges:
        for i in range(w.n):
            noise[i, j0:j1] = O.to_bf16(O.normals(w.seed, 1, i, 0, j0, j1 - j0))
    return noise


# "sync_step" is the launch configuration bench.py times.
@pytest.mark.parametrize("name,p,mode", [("resnet18-n8", 8, "unfused"), ("vgg16-n8", 8, "unfused"),
                                         ("resnet50-n16-bf16noise", 4, "unfused"), ("resnet18-n8", 8, "intervals"),
                                         ("resnet50-n16-bf16noise", 4, "intervals"), ("resnet18-n8", 8, "sync_step"),
                                         ("vgg16-n8", 8, "sync_step"), ("resnet50-n16-bf16noise", 4, "sync_step")])
def test_full_size_constant_period_run_on_sampled_columns(name, p, mode):
    w = inputs.WORKLOADS[name]
    bf16 = w.noise == "bf16"
    h, c = inputs.problem(w)
    ranges = _sample_ranges(w.P)
    # GPU: the whole run at full size
    xd = torch.zeros((w.n, w.P), dtype=torch.float32, device=DEV)
    vd = torch.zeros_like(xd)
    nd = None
    if bf16:
        nd = torch.empty((w.n, w.P), dtype=torch.int16, device=DEV)
        abi.adpsgd_noise_fill_bf16(w.seed, w.n, w.P, nd)
    sched = abi.make_schedule(abi.CPSGD, w.K, p, lr0=w.lr0, lr_factor=w.lr_factor, milestones=w.milestones)
    tr = abi.TraceBuffers(w.K)
    with abi.adpsgd_init(_cfg(w, bf16, mode), xd, vd, _dev(h), _dev(c), nd) as ctx:
        stats = abi.adpsgd_run(ctx, sched, abi.adpsgd_state_init(sched), trace=tr)
    torch.cuda.synchronize()
    rounds = w.K // p
    assert stats.rounds == rounds
    launches = {"unfused": (w.K, rounds, 0, 0), "intervals": (0, 0, rounds, 0),
                "sync_step": (w.K - rounds, 0, 0, rounds)}[mode]
    assert (stats.local_step_launches, stats.average_launches, stats.interval_launches,
            stats.sync_step_launches) == launches
    # oracle: the same run on the sampled columns only
    x = np.zeros((w.n, w.P), np.float32)
    v = np.zeros((w.n, w.P), np.float32)
    noise = _oracle_noise_on_ranges(w, ranges) if bf16 else None
    if bf16:
        for j0, j1 in ranges:
            gn = nd[:, j0:j1].cpu().numpy().view(np.uint16)
            assert np.array_equal(gn, noise[:, j0:j1])
    spec = O.ScheduleSpec(kind=0, K=w.K, p_init=p, lr0=w.lr0, lr_factor=w.lr_factor, milestones=w.milestones)
    for k in range(w.K):
        g = O.gamma(spec, k)
        for j0, j1 in ranges:
            O.local_step(x, v, h, c, seed=w.seed, k=k, gamma=g, mu=w.mu, wd=w.wd, sigma=w.sigma, noise=noise,
                         j0=j0, j1=j1)
        if (k + 1) % p == 0:
            for j0, j1 in ranges:
                O.average_variance(x, h, c, j0, j1)
    for j0, j1 in ranges:
        gx = xd[:, j0:j1].cpu().numpy()
        gv = vd[:, j0:j1].cpu().numpy()
        assert np.array_equal(gx.view(np.uint32), x[:, j0:j1].view(np.uint32)), (name, j0)
        assert np.array_equal(gv.view(np.uint32), v[:, j0:j1].view(np.uint32)), (name, j0)


@pytest.mark.parametrize("name", ["resnet18-n8", "vgg16-n8", "resnet50-n16-bf16noise"])
def test_full_size_average_and_variance(name):
    w = inputs.WORKLOADS[name]
    h, c = inputs.problem(w)
    x, _ = inputs.random_state(w.n, w.P, 5)
    xd = _dev(x)
    with abi.adpsgd_init(_cfg(w), xd, torch.empty_like(xd), _dev(h), _dev(c)) as ctx:
        D, L = abi.adpsgd_average_and_variance(ctx)
    torch.cuda.synchronize()
    Do, Lo = O.average_variance(x, h, c)
    assert _rel(D, Do) < REL and _rel(L, Lo) < REL
    got = xd.cpu().numpy()
    assert np.array_equal(got.view(np.uint32), x.view(np.uint32))


@pytest.mark.parametrize("mode", ["unfused", "sync_step"])
def test_full_size_adaptive_first_interval_and_rule_replay(mode):
    # resnet18-n8 at full size, Algorithm 2 (p_init 4, K_s 500): the first sync (after 4 local
    # steps from x0 = 0) against the oracle over all columns, and the whole trace against
    # Algorithm 2 replayed on the S values the run reported.
    w = inputs.WORKLOADS["resnet18-n8"]
    h, c = inputs.problem(w)
    xd = torch.zeros((w.n, w.P), dtype=torch.float32, device=DEV)
    vd = torch.zeros_like(xd)
    sched = abi.make_schedule(abi.ADPSGD, w.K, w.p_init, K_s=w.K_s, lr0=w.lr0, lr_factor=w.lr_factor,
                              milestones=w.milestones)
    tr = abi.TraceBuffers(w.K)
    with abi.adpsgd_init(_cfg(w, mode=mode), xd, vd, _dev(h), _dev(c)) as ctx:
        stats = abi.adpsgd_run(ctx, sched, abi.adpsgd_state_init(sched), trace=tr)
    t = tr.arrays()
    assert stats.rounds == len(t["k"]) and t["k"][0] == w.p_init - 1
    assert (stats.sync_step_launches > 0) == (mode == "sync_step")

    x, v = inputs.zero_state(w.n, w.P)
    for k in range(w.p_init):
        O.local_step(x, v, h, c, seed=w.seed, k=k, gamma=np.float32(w.lr0), mu=w.mu, wd=w.wd, sigma=w.sigma)
    D0, L0 = O.average_variance(x, h, c)
    assert _rel(t["S"][0], D0 / w.n) < REL and _rel(t["loss"][0], L0) < REL

    spec = O.ScheduleSpec(kind=1, K=w.K, p_init=w.p_init, K_s=w.K_s, lr0=w.lr0, lr_factor=w.lr_factor,
                          milestones=w.milestones)
    st = O.new_state(spec)
    k_expect = w.p_init - 1
    for s in range(len(t["k"])):
        assert t["k"][s] == k_expect
        O.on_sync(spec, st, int(t["k"][s]), float(t["S"][s]), O.gamma(spec, int(t["k"][s])))
        assert t["p"][s] == st.p and t["C2"][s] == st.C2
        k_expect += st.p
    assert k_expect >= w.K


# Iterations of the whole adaptive runs below: resnet18-n8 runs its full schedule; vgg16-n8 and
# resnet50-n16 run a shortened one (the same per-iteration work, fewer iterations), which keeps
# the oracle's share of the GPU test run to a few minutes on the host's cores.
FULL_RUN_K = {"resnet18-n8": 2000, "vgg16-n8": 100, "resnet50-n16-bf16noise": 200}


@pytest.mark.parametrize("name", list(FULL_RUN_K))
def test_full_size_adaptive_run_against_oracle_at_every_sync(name):
    # Both launch forms the bench times: fused sync steps (the headline) and fused intervals (its
    # fused_intervals figure), each against one oracle run.
    w = inputs.WORKLOADS[name]
    K = FULL_RUN_K[name]
    if K != w.K:
        w = dataclasses.replace(w, K=K, milestones=tuple(m * K // w.K for m in w.milestones))
    bf16 = w.noise == "bf16"
    h, c = inputs.problem(w)
    sched = abi.make_schedule(abi.ADPSGD, w.K, w.p_init, K_s=w.K_s, lr0=w.lr0, lr_factor=w.lr_factor,
                              milestones=w.milestones)
    runs = {}
    hd, cd = _dev(h), _dev(c)
    nd = None
    if bf16:
        nd = torch.empty((w.n, w.P), dtype=torch.int16, device=DEV)
        abi.adpsgd_noise_fill_bf16(w.seed, w.n, w.P, nd)
    for mode in ("sync_step", "intervals"):
        xd = torch.zeros((w.n, w.P), dtype=torch.float32, device=DEV)
        vd = torch.zeros_like(xd)
        tr = abi.TraceBuffers(w.K)
        cfg = abi.make_config(w.n, w.P, momentum=w.mu, weight_decay=w.wd, noise_sigma=w.sigma, seed=w.seed,
                              noise_mode=abi.NOISE_BF16 if bf16 else abi.NOISE_PHILOX, want_loss=True,
                              fuse_sync_step=mode == "sync_step", fuse_intervals=mode == "intervals")
        with abi.adpsgd_init(cfg, xd, vd, hd, cd, nd) as ctx:
            stats = abi.adpsgd_run(ctx, sched, abi.adpsgd_state_init(sched), trace=tr)
        torch.cuda.synchronize()
        if mode == "sync_step":
            assert stats.sync_step_launches > 0
            assert stats.sync_step_launches + stats.average_launches == stats.rounds
        else:
            assert stats.interval_launches >= stats.rounds > 0
        runs[mode] = (stats, tr.arrays(), xd.cpu().numpy(), vd.cpu().numpy())
        del xd, vd
        torch.cuda.empty_cache()
    del hd, cd, nd
    # oracle: the same run over all columns on every host core
    x, v = inputs.zero_state(w.n, w.P)
    noise = O.noise_bf16(w.seed, w.n, w.P) if bf16 else None
    spec = O.ScheduleSpec(kind=1, K=w.K, p_init=w.p_init, K_s=w.K_s, lr0=w.lr0, lr_factor=w.lr_factor,
                          milestones=w.milestones)
    otr = O.run(x, v, h, c, spec=spec, seed=w.seed, mu=w.mu, wd=w.wd, sigma=w.sigma, noise=noise,
                threads=O.host_threads())
    # every adaptive decision well away from the thresholds, so that the bit-exact comparison of
    # the schedule is well posed (S agrees to far better than 1e-6)
    C2_before = np.concatenate([[0.0], otr.C2[:-1]])
    for k, S, C2b, ph in zip(otr.k, otr.S, C2_before, otr.phase):
        if ph == O.PHASE_ADAPTING and C2b > 0.0:
            ratio = S / (np.float64(O.gamma(spec, int(k))) * C2b)
            assert min(abs(ratio - 0.7) / 0.7, abs(ratio - 1.3) / 1.3) > 1e-6, (name, k, ratio)
    for mode, (stats, t, gx, gv) in runs.items():
        assert stats.rounds == otr.syncs == len(t["k"]), mode
        assert np.array_equal(t["k"], otr.k) and np.array_equal(t["p"], otr.p), mode
        assert np.array_equal(t["phase"], otr.phase), mode
        for key in ("S", "loss", "C2"):
            for s_idx, (a, b) in enumerate(zip(t[key], getattr(otr, key))):
                assert _rel(a, b) < REL or (a == 0.0 and b == 0.0), (name, mode, key, s_idx, a, b)
        assert np.array_equal(gx.view(np.uint32), x.view(np.uint32)), (name, mode)
        assert np.array_equal(gv.view(np.uint32), v.view(np.uint32)), (name, mode)


def _cfg_big(n, P, mu, wd, sigma, seed, mode):
    return abi.make_config(n, P, momentum=mu, weight_decay=wd, noise_sigma=sigma, seed=seed,
                           fuse_sync_step=mode == "sync_step", fuse_intervals=mode == "intervals")


def test_more_than_2_31_elements():
    # n P = 2^31 + 8 elements per array: the 64-bit index arithmetic of the local step, the
    # averaging, the fused sync step and the fused interval, on columns on both sides of 2^30
    # and at the end (x and v bit-exact against the oracle).  About 26 GB of HBM; the host arrays
    # are lazily zeroed, so only the sampled columns' pages are touched.
    n, P = 2, (1 << 30) + 4
    ranges = [(0, 64), ((1 << 29) - 32, (1 << 29) + 32), ((1 << 30) - 32, (1 << 30) + 4)]
    gen = torch.Generator(device=DEV).manual_seed(31)
    hd = 0.1 + 0.9 * torch.rand(P, device=DEV, generator=gen)
    cd = torch.randn(P, device=DEV, generator=gen)
    h = np.zeros(P, np.float32)
    c = np.zeros(P, np.float32)
    for j0, j1 in ranges:
        h[j0:j1] = hd[j0:j1].cpu().numpy()
        c[j0:j1] = cd[j0:j1].cpu().numpy()
    seed, mu, wd, sigma, lr = 77, 0.9, 5e-4, 0.5, 0.05
    sched = abi.make_schedule(abi.CPSGD, 4, 4, lr0=lr)
    for mode in ("unfused", "sync_step", "intervals"):
        xd = torch.zeros((n, P), dtype=torch.float32, device=DEV)
        vd = torch.zeros_like(xd)
        with abi.adpsgd_init(_cfg_big(n, P, mu, wd, sigma, seed, mode), xd, vd, hd, cd) as ctx:
            st = abi.adpsgd_run(ctx, sched, abi.adpsgd_state_init(sched))
        assert st.rounds == 1
        assert (st.sync_step_launches, st.interval_launches) == {"unfused": (0, 0), "sync_step": (1, 0),
                                                                 "intervals": (0, 1)}[mode]
        x = np.zeros((n, P), np.float32)
        v = np.zeros((n, P), np.float32)
        for j0, j1 in ranges:
            for k in range(4):
                O.local_step(x, v, h, c, seed=seed, k=k, gamma=np.float32(lr), mu=mu, wd=wd, sigma=sigma,
                             j0=j0, j1=j1)
            O.average_variance(x, h, c, j0, j1)
            gx = xd[:, j0:j1].cpu().numpy()
            gv = vd[:, j0:j1].cpu().numpy()
            assert np.array_equal(gx.view(np.uint32), x[:, j0:j1].view(np.uint32)), (mode, j0)
            assert np.array_equal(gv.view(np.uint32), v[:, j0:j1].view(np.uint32)), (mode, j0)
        del xd, vd
        torch.cuda.empty_cache()
