"""Averaging at the edges of the fp32 range, against the oracle.

The kernels square deviations and loss terms in fp32 and add them in fp64; the oracle squares in
fp64.  The two agree within 1e-4 as long as no fp32 square underflows or overflows.  Replicas that
differ by less than about 2^-63 (subnormal parameters) or by more than about 2^63 break that.  For
such columns the kernels redo the column in fp64, so the results follow the definition (Sec. II-B,
Var[W_k]) over the whole fp32 range.  These cases pin that:
- tiny and huge values;
- identical replicas and negative zeros;
- zero curvatures and minimisers hit exactly;
- NaN and infinity.
Each case runs through every averaging path:
- the context entry point, with write-back and loss;
- the variance-only entry point;
- the entry point without a context;
- the fused interval kernel and the fused sync step inside a run.
The replica counts cover every register-resident variant and the any-n variant.
"""
import numpy as np
import pytest

from oracle import oracle as O
from paper_2007_06134_gb300 import abi

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
DEV = "cuda:0"
REL = 1e-4
F32 = np.float32


def _dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).to(DEV)


def _host(t):
    torch.cuda.synchronize()
    return t.cpu().numpy()


def _close(a, b):
    if np.isnan(b):
        return bool(np.isnan(a))
    if np.isinf(b) or b == 0.0:
        return a == b
    return abs(a - b) <= REL * abs(b)


def _same_bits(a, b):
    """Bit-exact, except that NaN encodings differ between the CPU and the GPU (both quiet NaNs)."""
    na, nb = np.isnan(a), np.isnan(b)
    return np.array_equal(na, nb) and np.array_equal(a[~na].view(np.uint32), b[~nb].view(np.uint32))


def _problem(n, P, kind, seed):
    """x [n, P], h, c for one kind of extreme input; the column pattern repeats every 5 columns."""
    rng = np.random.default_rng(seed)
    x = rng.standard_normal((n, P)).astype(F32)
    c = (0.1 * rng.standard_normal(P)).astype(F32)
    h = rng.uniform(0.1, 1.0, P).astype(F32)
    j = np.arange(P)
    h[j % 11 == 0] = 0.0                           # zero curvature: loss term exactly 0
    if kind == "tiny":                             # subnormal and near-subnormal deviations
        x = (x * F32(1e-39)).astype(F32)
        x[:, j % 3 == 0] = (x[:, j % 3 == 0] * F32(1e-5)).astype(F32)
        c = (c * F32(1e-38)).astype(F32)
    elif kind == "huge":                           # squares above the fp32 range
        x = (x * F32(1e30)).astype(F32)
        c = (c * F32(1e30)).astype(F32)
    elif kind in ("mixed-tiny", "mixed-huge"):     # some groups redone, the rest written normally
        s = F32(1e-39) if kind == "mixed-tiny" else F32(1e30)
        x[:, j % 5 == 0] = (x[:, j % 5 == 0] * s).astype(F32)
        x[:, j % 5 == 1] = x[0, j % 5 == 1]        # identical replicas ...
        c[j % 5 == 1] = x[0, j % 5 == 1]           # ... sitting exactly on the minimiser
        x[:, j % 5 == 2] = F32(-0.0)               # negative zeros (the mean is +0)
    elif kind == "nonfinite":
        x[:, j % 97 == 5] = np.inf                 # every replica +inf: mean NaN
        x[n - 1, j % 89 == 7] = np.nan
        x[0, j % 83 == 3] = np.inf                 # one replica +inf
    return x, h, c


KINDS = ["tiny", "huge", "mixed-tiny", "mixed-huge", "nonfinite"]
NS = [1, 2, 3, 8, 16, 32, 40]  # register-resident variants for n <= 32; n = 40 re-reads x


@pytest.mark.parametrize("kind", KINDS)
@pytest.mark.parametrize("n", NS)
@pytest.mark.parametrize("P", [4096, 4099])
def test_average_and_variance_entry_points(kind, n, P):
    x, h, c = _problem(n, P, kind, seed=17 * n + P)
    Dv = O.variance(x.copy())
    xo = x.copy()
    Do, Lo = O.average_variance(xo, h, c)

    xd = _dev(x)
    with abi.adpsgd_init(abi.make_config(n, P), xd, torch.zeros_like(xd), _dev(h), _dev(c)) as ctx:
        D_var = abi.adpsgd_variance(ctx)
        assert _same_bits(_host(xd), x), "the variance-only pass must not write"
        D, L = abi.adpsgd_average_and_variance(ctx)
    assert _same_bits(_host(xd), xo)
    assert _close(D_var, Dv) and _close(D, Do) and _close(L, Lo), (D_var, Dv, D, Do, L, Lo)

    xs = _dev(x)
    Ds, Ls = abi.adpsgd_average_and_variance_static(xs, _dev(h), _dev(c), n, P)
    assert _same_bits(_host(xs), xo)
    assert _close(Ds, Do) and _close(Ls, Lo), (Ds, Do, Ls, Lo)


def test_identical_replicas_give_exact_zero():
    # n identical replicas (the state right after a sync): D = 0 exactly, no fp64 path needed.
    n, P = 8, (1 << 16) + 4
    x, h, c = _problem(1, P, "normal", seed=3)
    x = np.repeat(x, n, axis=0)
    xd = _dev(x)
    with abi.adpsgd_init(abi.make_config(n, P), xd, torch.zeros_like(xd), _dev(h), _dev(c)) as ctx:
        assert abi.adpsgd_variance(ctx) == 0.0
        D, L = abi.adpsgd_average_and_variance(ctx)
    Do, Lo = O.average_variance(x, h, c)
    assert D == 0.0 and Do == 0.0 and _close(L, Lo)
    assert _same_bits(_host(xd), x)


@pytest.mark.parametrize("n", [4, 6, 12])
@pytest.mark.parametrize("kind", ["tiny", "huge"])
@pytest.mark.parametrize("mode", ["unfused", "intervals", "sync_step"])
def test_run_at_extreme_scales(kind, mode, n):
    # A short CPSGD run whose steps and syncs stay at the scale of the data: tiny values with tiny
    # noise (every sum subnormal), or huge values whose squares leave fp32.  Six replicas run the
    # kernels built for up to 8 with two slots unused, four those built for exactly 4, and twelve
    # the fused step's two-halves form, whose averaging reads the new x from shared memory.
    K, p = 6, 2
    P = 1032 if mode == "sync_step" else 1031  # the fused sync step takes P % 4 == 0 only
    x, h, c = _problem(n, P, kind, seed=5)
    scale = 1e-39 if kind == "tiny" else 1e30
    v = (0.1 * x).astype(F32)
    sigma, seed = scale, 0x5EED
    xd, vd = _dev(x), _dev(v)
    cfg = abi.make_config(n, P, momentum=0.9, weight_decay=0.0, noise_sigma=sigma, seed=seed,
                          fuse_intervals=mode == "intervals", fuse_sync_step=mode == "sync_step")
    sched = abi.make_schedule(abi.CPSGD, K, p, lr0=0.1)
    tr = abi.TraceBuffers(K + 1)
    with abi.adpsgd_init(cfg, xd, vd, _dev(h), _dev(c)) as ctx:
        stats = abi.adpsgd_run(ctx, sched, abi.adpsgd_state_init(sched), trace=tr)
    assert (stats.interval_launches > 0) == (mode == "intervals")
    assert (stats.sync_step_launches > 0) == (mode == "sync_step")
    g = tr.arrays()
    spec = O.ScheduleSpec(kind=abi.CPSGD, K=K, p_init=p, lr0=0.1)
    otr = O.run(x, v, h, c, spec=spec, seed=seed, mu=0.9, wd=0.0, sigma=sigma)
    assert np.array_equal(g["k"], otr.k)
    for a, b in zip(g["S"], otr.S):
        assert b != 0.0 and _close(a, b), (a, b)
    for a, b in zip(g["loss"], otr.loss):
        assert _close(a, b), (a, b)
    assert _same_bits(_host(xd), x) and _same_bits(_host(vd), v)
