"""Properties of the CUDA path that hold at any size, checked at sizes the oracle cannot follow,
plus randomised shapes against the oracle.

- The spread of the replicas after m noisy steps from a common start has the exact second moment
  of the linear recurrence (Sec. II-B's Var[W_k], statistical at 5 sigma): this pins the noise
  scale, the momentum form and D = sum_i ||x_i - xbar||^2 on the GPU without the oracle.
- Averaging preserves the replica mean and leaves zero variance at P = 2^26.
"""
import numpy as np
import pytest

from oracle import oracle as O
from paper_2007_06134_gb300 import abi, inputs

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
DEV = "cuda:0"


def _second_moment(h, gamma, sigma, mu, m, n):
    """E[D] after m noisy steps from identical replicas: (n - 1) sum_j sum_t (impulse_t)^2, where the
    impulse is the x-response of (y, v) <- M (y, v) + b z, M = [[1 - g h, -g mu], [h, mu]],
    b = (-g sigma, sigma)."""
    h = h.astype(np.float64)
    y = np.full(h.size, -gamma * sigma)
    v = np.full(h.size, sigma)
    acc = np.zeros(h.size)
    for _ in range(m):
        acc += y * y
        y, v = (1 - gamma * h) * y - gamma * mu * v, h * y + mu * v
    return (n - 1) * acc.sum()


@pytest.mark.parametrize("mu,m", [(0.0, 3), (0.9, 6)])
def test_spread_second_moment_at_large_P(mu, m):
    n, P, gamma, sigma = 8, 1 << 24, 0.1, 0.5
    h = inputs.draw_h(P, "uniform:0.1:1", 9)
    c = inputs.draw_c(P, 1.0, 9)
    xd = torch.zeros((n, P), device=DEV)
    vd = torch.zeros_like(xd)
    cfg = abi.make_config(n, P, momentum=mu, noise_sigma=sigma, seed=0xC0FFEE)
    with abi.adpsgd_init(cfg, xd, vd, torch.from_numpy(h).to(DEV), torch.from_numpy(c).to(DEV)) as ctx:
        abi.adpsgd_local_steps(ctx, 0, [gamma] * m)
        D = abi.adpsgd_variance(ctx)
    ED = _second_moment(h, np.float64(np.float32(gamma)), sigma, mu, m, n)
    assert abs(D / ED - 1.0) < 5 * np.sqrt(2.0 / ((n - 1) * P)), (D, ED)


def test_mean_preserved_and_variance_zero_at_large_P():
    n, P = 16, 1 << 26
    gen = torch.Generator(device=DEV).manual_seed(3)
    xd = torch.randn((n, P), device=DEV, generator=gen)
    before = xd.double().mean(dim=0)
    z = torch.zeros(P, device=DEV)
    with abi.adpsgd_init(abi.make_config(n, P, want_loss=False), xd, xd, z, z) as ctx:
        D1, _ = abi.adpsgd_average_and_variance(ctx, want_loss=False)
        D2, _ = abi.adpsgd_average_and_variance(ctx, want_loss=False)
    assert D1 > 0 and D2 == 0.0
    assert torch.equal(xd[0], xd[n - 1])
    err = (xd[0].double() - before).abs()
    bound = n * 2.0 ** -23 * (xd.double() - xd[0].double()).abs().max() + 2.0 ** -23 * before.abs()
    assert bool((err <= bound + 1e-30).all()) or float(err.max()) < 1e-5


@pytest.mark.parametrize("case", range(8))
def test_random_shapes_against_oracle(case):
    rng = np.random.default_rng(1000 + case)
    n = int(rng.integers(1, 41))
    P = int(rng.integers(1, 70000))
    wd = float(rng.choice([0.0, 1e-3]))
    mu = float(rng.choice([0.0, 0.5, 0.9]))
    k0 = int(rng.integers(0, 1 << 31))
    lrs = [float(v) for v in rng.uniform(0.001, 0.2, int(rng.integers(1, 4)))]
    seed = int(rng.integers(0, 1 << 63))
    w = inputs.WORKLOADS["resnet18-n8"]
    h = inputs.draw_h(P, w.h_dist, case)
    c = inputs.draw_c(P, 1.0, case)
    x, v = inputs.random_state(n, P, case)
    xd, vd = torch.from_numpy(x).to(DEV), torch.from_numpy(v).to(DEV)
    cfg = abi.make_config(n, P, momentum=mu, weight_decay=wd, noise_sigma=0.7, seed=seed,
                          fuse_intervals=bool(case % 2) and n <= 32)
    with abi.adpsgd_init(cfg, xd, vd, torch.from_numpy(h).to(DEV), torch.from_numpy(c).to(DEV)) as ctx:
        abi.adpsgd_local_steps(ctx, k0, lrs)
        D, L = abi.adpsgd_average_and_variance(ctx)
    for t, lr in enumerate(lrs):
        O.local_step(x, v, h, c, seed=seed, k=k0 + t, gamma=np.float32(lr), mu=mu, wd=wd, sigma=0.7)
    Do, Lo = O.average_variance(x, h, c)
    torch.cuda.synchronize()
    assert np.array_equal(xd.cpu().numpy(), x) and np.array_equal(vd.cpu().numpy(), v), (n, P)
    assert (D == 0.0 and Do == 0.0) or abs(D - Do) <= 1e-4 * Do
    assert abs(L - Lo) <= 1e-4 * Lo
