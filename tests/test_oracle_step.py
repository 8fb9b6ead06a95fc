"""Pins of the oracle's local step and its averaging + variance.

Local step: Algorithm 1 / Algorithm 2 update line with SGD momentum (Sec. IV-A)
on the surrogate f(x) = 1/2 sum_j h_j (x_j - c_j)^2.  Pinned by closed forms of
the linear recurrence (computed here by fp64 matrix powers, a different route
from iterating), by the special case h = 0 where the update is a plain sum of
the drawn noise, and by the exact second moment of the noise-driven spread.

Averaging: Algorithm 2 averaging and S_k lines, Var[W_k] of Sec. II-B.  Pinned
by n = 1 (identity), "variance is zero after each synchronization"
(Sec. III-B), an exactly representable closed form, and fp64 brute force.
"""
import numpy as np
import pytest

from oracle import oracle as O
from paper_2007_06134_gb300 import inputs


def _problem(P, seed=3, hlo=0.1, hhi=1.0):
    h = inputs.draw_h(P, f"uniform:{hlo}:{hhi}", seed)
    c = inputs.draw_c(P, 1.0, seed)
    return h, c


def _matrix_power_solution(h, c, wd, mu, gamma, K, x0, v0):
    """Noise-free trajectory via M^K on (x - x*, v), x* = h c / (h + wd)."""
    h = h.astype(np.float64)
    c = c.astype(np.float64)
    a = h + wd
    xstar = h * c / a
    out_x = np.empty_like(h)
    out_v = np.empty_like(h)
    for j in range(h.size):
        M = np.array([[1.0 - gamma * a[j], -gamma * mu], [a[j], mu]])
        s = np.linalg.matrix_power(M, K) @ np.array([x0[j] - xstar[j], v0[j]])
        out_x[j] = s[0] + xstar[j]
        out_v[j] = s[1]
    return out_x, out_v


@pytest.mark.parametrize("mu,wd", [(0.0, 0.0), (0.9, 0.0), (0.9, 5e-4), (0.5, 1e-2)])
def test_noise_free_step_matches_matrix_power(mu, wd):
    n, P, K, gamma = 2, 257, 60, 0.05
    h, c = _problem(P)
    x = np.zeros((n, P), np.float32)
    v = np.zeros((n, P), np.float32)
    for k in range(K):
        O.local_step(x, v, h, c, seed=1, k=k, gamma=gamma, mu=mu, wd=wd, sigma=0.0)
    ex, ev = _matrix_power_solution(h, c, wd, mu, np.float64(np.float32(gamma)), K,
                                    np.zeros(P), np.zeros(P))
    scale = np.abs(c).max()
    assert np.abs(x[0] - ex).max() <= 1e-5 * scale
    assert np.abs(v[0] - ev).max() <= 1e-5 * scale
    assert np.array_equal(x[0], x[1])  # no noise: replicas identical


def test_plain_gd_closed_form():
    # mu = 0, wd = 0, sigma = 0: x_K - c = (1 - gamma h)^K (x_0 - c) (Eq. gd).
    P, K, gamma = 1000, 40, 0.1
    h, c = _problem(P)
    x = np.ones((1, P), np.float32)
    v = np.zeros((1, P), np.float32)
    for k in range(K):
        O.local_step(x, v, h, c, seed=0, k=k, gamma=gamma, mu=0.0, wd=0.0, sigma=0.0)
    g = np.float64(np.float32(gamma))
    expect = c + (1.0 - g * h.astype(np.float64)) ** K * (1.0 - c)
    assert np.abs(x[0] - expect).max() <= 1e-5 * np.abs(c).max()


def test_weight_decay_fixed_point():
    P = 64
    h, c = _problem(P, hlo=0.5)
    wd = 0.25
    x = np.zeros((1, P), np.float32)
    v = np.zeros((1, P), np.float32)
    for k in range(3000):
        O.local_step(x, v, h, c, seed=0, k=k, gamma=0.05, mu=0.9, wd=wd, sigma=0.0)
    xstar = h.astype(np.float64) * c / (h.astype(np.float64) + wd)
    assert np.abs(x[0] - xstar).max() <= 1e-5


def test_zero_curvature_is_a_sum_of_noise():
    # h = 0, mu = 0: x_K = x_0 - gamma sigma sum_k z[i, j, k]: pins the replica index, the
    # step index fed to the generator, and the sign and scale of the noise term.
    n, P, K, gamma, sigma = 3, 37, 5, 0.25, 0.5
    h = np.zeros(P, np.float32)
    c = np.zeros(P, np.float32)
    x = np.zeros((n, P), np.float32)
    v = np.zeros((n, P), np.float32)
    for k in range(K):
        O.local_step(x, v, h, c, seed=99, k=k, gamma=gamma, mu=0.0, wd=0.0, sigma=sigma)
    for i in range(n):
        zs = sum(O.normals(99, 0, i, k, 0, P).astype(np.float64) for k in range(K))
        assert np.abs(x[i] - (-gamma * sigma * zs)).max() <= 1e-6


def test_bf16_noise_mode_uses_the_tensor_every_step():
    n, P = 2, 19
    h = np.zeros(P, np.float32)
    c = np.zeros(P, np.float32)
    noise = O.noise_bf16(4, n, P)
    z = (noise.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    x = np.zeros((n, P), np.float32)
    v = np.zeros((n, P), np.float32)
    for k in range(3):
        O.local_step(x, v, h, c, seed=4, k=k, gamma=0.5, mu=0.0, wd=0.0, sigma=1.0, noise=noise)
    assert np.abs(x - (-1.5 * z)).max() <= 1e-6


def test_column_ranges_compose_exactly():
    n, P = 3, 103
    h, c = _problem(P)
    x1, v1 = inputs.random_state(n, P, 5)
    x2, v2 = x1.copy(), v1.copy()
    kw = dict(seed=8, k=17, gamma=0.05, mu=0.9, wd=5e-4, sigma=0.5)
    O.local_step(x1, v1, h, c, **kw)
    O.local_step(x2, v2, h, c, j0=0, j1=41, **kw)
    O.local_step(x2, v2, h, c, j0=41, j1=P, **kw)
    assert np.array_equal(x1, x2) and np.array_equal(v1, v2)


def _noise_spread_expectation(h, gamma, sigma, mu, m, n):
    """E[D] after m noisy steps from identical replicas: (n-1) sum_j sum_t (impulse_t)^2."""
    total = 0.0
    for hj in h.astype(np.float64):
        M = np.array([[1.0 - gamma * hj, -gamma * mu], [hj, mu]])
        b = np.array([-gamma * sigma, sigma])  # noise enters g: v += sigma z, x -= gamma sigma z
        acc = 0.0
        resp = b.copy()
        for _ in range(m):
            acc += resp[0] ** 2
            resp = M @ resp
        total += acc
    return (n - 1) * total


@pytest.mark.parametrize("mu", [0.0, 0.9])
def test_variance_after_m_steps_matches_second_moment(mu):
    # Statistical pin of the noise scale and of D = sum_i ||x_i - xbar||^2 (Sec. II-B).
    n, P, m, gamma, sigma = 4, 1 << 14, 6, 0.1, 0.5
    h, c = _problem(P)
    x = np.zeros((n, P), np.float32)
    v = np.zeros((n, P), np.float32)
    for k in range(m):
        O.local_step(x, v, h, c, seed=123, k=k, gamma=gamma, mu=mu, wd=0.0, sigma=sigma)
    D, _ = O.average_variance(x, h, c)
    ED = _noise_spread_expectation(h, np.float64(np.float32(gamma)), sigma, mu, m, n)
    rel_sd = np.sqrt(2.0 / ((n - 1) * P))
    assert abs(D / ED - 1.0) < 5 * rel_sd


# ---------------------------------------------------------------------------------------------
# averaging + variance
# ---------------------------------------------------------------------------------------------

def test_single_replica_is_identity():
    x, _ = inputs.random_state(1, 1001, 7)
    before = x.copy()
    h, c = _problem(1001)
    D, loss = O.average_variance(x, h, c)
    assert D == 0.0 and np.array_equal(x, before)
    assert loss == pytest.approx(0.5 * np.sum(h.astype(np.float64) * (before[0].astype(np.float64) - c) ** 2), rel=1e-12)


@pytest.mark.parametrize("n", [2, 3, 5, 8, 16, 33])
def test_variance_is_zero_after_averaging(n):
    x, _ = inputs.random_state(n, 513, n)
    D1, _ = O.average_variance(x)
    assert D1 > 0
    after = x.copy()
    D2, _ = O.average_variance(x)
    assert D2 == 0.0 and np.array_equal(x, after)
    assert all(np.array_equal(x[0], x[i]) for i in range(n))


@pytest.mark.parametrize("n", [2, 3, 4, 7, 16, 32])
def test_mean_and_variance_against_fp64(n):
    P = 2049
    x, _ = inputs.random_state(n, P, 11 + n)
    x64 = x.astype(np.float64)
    mean = x64.mean(axis=0)
    D_ref = ((x64 - mean) ** 2).sum()
    dev_max = np.abs(x64 - x64[0]).max(axis=0)
    D, _ = O.average_variance(x)
    xbar = x[0].astype(np.float64)
    bound = np.spacing(np.abs(xbar).astype(np.float32)) + n * 2.0 ** -23 * dev_max
    assert np.all(np.abs(xbar - mean) <= bound)
    # D uses the fp32 mean: D = D_ref + n sum_j (xbar_j - mean_j)^2 >= D_ref
    assert abs(D - D_ref) <= 1e-6 * D_ref


@pytest.mark.parametrize("n", [2, 3, 4, 8, 16, 32])
def test_exact_offsets_closed_form(n):
    # x_ij = b_j + i d with b_j on a 2^-12 grid and d = 2^-10: every value and the mean are
    # exact in fp32, so D = P d^2 n (n^2 - 1) / 12 exactly and xbar_j = b_j + d (n - 1) / 2.
    P = 4099
    rng = np.random.default_rng(n)
    b = (rng.integers(-8192, 8192, P) * 2.0 ** -12).astype(np.float32)
    d = 2.0 ** -10
    x = np.stack([b + np.float32(i * d) for i in range(n)]).astype(np.float32)
    D, _ = O.average_variance(x)
    assert D == P * d * d * n * (n * n - 1) / 12.0
    assert np.array_equal(x[0], (b.astype(np.float64) + d * (n - 1) / 2.0).astype(np.float32))


def test_sweep_recipe_shared_draw_closed_form():
    # The sweep recipe x_i = N(0,1) + i 1e-3 with one shared draw: D ~= P 1e-6 n (n^2 - 1) / 12,
    # up to the fp32 rounding of the offsets (relative error ~ 2^-24 |x| / 1e-3).
    n, P = 8, 1 << 14
    x = inputs.sweep_replicas(n, P, 5, shared=True)
    D, _ = O.average_variance(x)
    assert D == pytest.approx(P * 1e-6 * n * (n * n - 1) / 12.0, rel=5e-3)


def test_loss_closed_forms():
    P = 100
    h = np.full(P, 2.0, np.float32)
    c = np.zeros(P, np.float32)
    x = np.ones((3, P), np.float32)
    D, loss = O.average_variance(x, h, c)
    assert D == 0.0 and loss == P * 0.5 * 2.0 * 1.0
    x = np.stack([c, c]).astype(np.float32)
    assert O.average_variance(x, h, c)[1] == 0.0


def test_average_column_ranges_compose():
    x1, _ = inputs.random_state(5, 300, 2)
    x2 = x1.copy()
    h, c = _problem(300)
    D1, L1 = O.average_variance(x1, h, c)
    Da, La = O.average_variance(x2, h, c, 0, 123)
    Db, Lb = O.average_variance(x2, h, c, 123, 300)
    assert np.array_equal(x1, x2)
    assert Da + Db == pytest.approx(D1, rel=1e-13) and La + Lb == pytest.approx(L1, rel=1e-13)


def test_variance_only_matches_average():
    x, _ = inputs.random_state(6, 777, 3)
    D0 = O.variance(x)
    D1, _ = O.average_variance(x.copy())
    assert D0 == D1
