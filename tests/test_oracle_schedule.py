"""Pins of the oracle's schedules: Algorithm 1 (constant period) and Algorithm 2 (adaptive).

Pinned by the sync-count arithmetic the paper prints (Sec. III-A: 2000/4 + 2000/8
= 750 and 4000/5 = 800; Sec. V-B: 2000/20 + 2000/5 = 500 = 4000/8; Sec. III-B:
4000/498 ~ 8.03), by Algorithm 2's own logic on scripted variances (strict
comparisons at 0.7 and 1.3, cumulative-mean C_2, p >= 1), and by closed forms of
the noise-free run.
"""
import numpy as np
import pytest

from oracle import oracle as O
from paper_2007_06134_gb300 import inputs


def cps(K, p, **kw):
    return O.ScheduleSpec(kind=0, K=K, p_init=p, lr0=0.1, **kw)


def ads(K, p_init, K_s, **kw):
    return O.ScheduleSpec(kind=1, K=K, p_init=p_init, K_s=K_s, lr0=0.1, **kw)


@pytest.mark.parametrize("K,p", [(100, 4), (500, 8), (4000, 8), (4000, 5), (2000, 20), (7, 3)])
def test_constant_period_counts(K, p):
    syncs, ks, ps = O.schedule_only(cps(K, p), [])
    assert syncs == K // p
    assert list(ks) == [p - 1 + p * t for t in range(K // p)]
    assert set(ps) <= {p}


@pytest.mark.parametrize("K,p", [(100, 4), (500, 8), (7, 3)])
def test_literal_algorithm1_phase(K, p):
    # Algorithm 1 as printed syncs when k mod p == 0, k from 0: ceil(K / p) syncs.
    syncs, ks, _ = O.schedule_only(cps(K, p, literal_phase=1), [])
    assert syncs == -(-K // p)
    assert list(ks) == list(range(0, K, p))


def test_paper_sync_count_arithmetic():
    count = lambda K, p: O.schedule_only(cps(K, p), [])[0]
    assert count(2000, 4) + count(2000, 8) == 750   # strategies 1 and 2 (Sec. III-A)
    assert count(4000, 5) == 800                    # strategy 4
    assert count(2000, 20) + count(2000, 5) == 500  # decreasing period of Sec. V-B
    assert count(4000, 8) == 500
    assert round(4000 / 498) == 8                   # equal-budget constant period (Sec. III-B)


def test_adaptive_without_adaptation_is_constant_period():
    K = 300
    rng = np.random.default_rng(0)
    S = rng.uniform(0.0, 10.0, 400)
    a = O.schedule_only(ads(K, 4, K_s=K), S)
    b = O.schedule_only(cps(K, 4), S)
    assert a[0] == b[0] and np.array_equal(a[1], b[1]) and np.array_equal(a[2], b[2])


def test_constant_ratio_keeps_period():
    # S = gamma C_2 every sync: after sampling, neither 0.7 nor 1.3 is crossed.
    spec = ads(400, 4, K_s=100)
    S = np.full(1000, 0.1 * 3.0)  # gamma = 0.1 throughout, S / gamma = 3 = C_2
    syncs, ks, ps = O.schedule_only(spec, S)
    assert set(ps) == {4} and syncs == 100


def test_shrinking_variance_grows_period_by_one_per_sync():
    spec = ads(2000, 4, K_s=100)
    S = np.concatenate([np.full(25, 1.0), 0.5 ** np.arange(1, 200)])
    syncs, ks, ps = O.schedule_only(spec, S)
    assert list(ps[:25]) == [4] * 25         # sampling phase: syncs at k = 3, 7, ..., 99
    assert ks[24] == 99
    assert list(ps[25:30]) == [5, 6, 7, 8, 9]
    assert np.all(np.diff(ks[25:30]) == [5, 6, 7, 8])  # the new p governs the next interval


def test_large_variance_shrinks_period_to_one_and_clamps():
    spec = ads(400, 4, K_s=20)
    S = np.concatenate([np.full(5, 1.0), np.full(1000, 100.0)])
    syncs, ks, ps = O.schedule_only(spec, S)
    assert list(ps[5:9]) == [3, 2, 1, 1]
    assert ps[-1] == 1 and np.all(np.diff(ks[8:]) == 1)


def test_p_max_clamp():
    spec = ads(400, 4, K_s=20, p_max=6)
    S = np.concatenate([np.full(5, 1.0), np.full(1000, 1e-9)])
    _, _, ps = O.schedule_only(spec, S)
    assert ps.max() == 6


def test_zero_variance_keeps_period():
    # sigma = 0: S = 0 and C_2 = 0; 0 < 0.7 * 0 and 0 > 1.3 * 0 are both false.
    spec = ads(300, 4, K_s=50)
    _, _, ps = O.schedule_only(spec, np.zeros(500))
    assert set(ps) == {4}


def test_comparisons_are_strict():
    spec = ads(100, 2, K_s=2)
    st = O.new_state(spec)
    O.on_sync(spec, st, 1, 4.0, 2.0)    # sampling: C_2 = 2
    assert st.C2 == 2.0
    for S, p in ((0.7 * 2.0 * 2.0, 2), (1.3 * 2.0 * 2.0, 2), (0.7 * 4.0 - 1e-12, 3),
                 (1.3 * 4.0 + 1e-12, 2)):
        O.on_sync(spec, st, 10, S, 2.0)
        assert st.p == p


def test_running_average_is_cumulative_mean():
    spec = ads(10 ** 6, 1, K_s=10 ** 6)
    st = O.new_state(spec)
    rng = np.random.default_rng(3)
    S = rng.uniform(0, 5, 200)
    g = rng.uniform(0.01, 0.1, 200)
    for t in range(200):
        assert O.on_sync(spec, st, t, S[t], g[t]) == O.PHASE_SAMPLING
    assert st.m == 200
    assert st.C2 == pytest.approx(np.mean(S / g), rel=1e-12)


def test_warmup_syncs_every_iteration_unsampled():
    spec = ads(60, 4, K_s=30, K_w=10)
    syncs, ks, ps = O.schedule_only(spec, np.full(100, 1.0))
    assert list(ks[:10]) == list(range(10))
    assert ks[10] == 13  # p_init = 4 after the warm-up


def test_step_size_schedule():
    spec = O.ScheduleSpec(kind=1, K=2000, p_init=4, K_s=500, lr0=0.1, lr_factor=0.1,
                          milestones=(1000, 1500))
    assert O.gamma(spec, 0) == np.float32(0.1) and O.gamma(spec, 999) == np.float32(0.1)
    assert O.gamma(spec, 1000) == np.float32(0.01) and O.gamma(spec, 1499) == np.float32(0.01)
    assert O.gamma(spec, 1500) == np.float32(0.001) and O.gamma(spec, 1999) == np.float32(0.001)


def test_noise_free_run_closed_form_loss():
    # sigma = 0, mu = 0: replicas never drift apart (S = 0) and after k + 1 steps from x_0 = 0
    # the loss at a sync is 1/2 sum_j h_j c_j^2 (1 - gamma h_j)^(2(k+1)).
    n, P = 3, 500
    h = inputs.draw_h(P, "uniform:0.1:1", 1)
    c = inputs.draw_c(P, 1.0, 1)
    x, v = inputs.zero_state(n, P)
    spec = cps(40, 4)
    spec.lr0 = 0.05
    tr = O.run(x, v, h, c, spec=spec, seed=0, mu=0.0, wd=0.0, sigma=0.0)
    g = np.float64(np.float32(0.05))
    for k, S, loss in zip(tr.k, tr.S, tr.loss):
        assert S == 0.0
        expect = 0.5 * np.sum(h * c.astype(np.float64) ** 2 * (1 - g * h) ** (2 * (k + 1)))
        assert loss == pytest.approx(expect, rel=1e-5)


def test_run_resume_is_bit_identical():
    n, P = 3, 301
    w = inputs.WORKLOADS["quadratic-n4-P1M"]
    h, c = inputs.problem(w, P)
    spec = O.ScheduleSpec(kind=1, K=60, p_init=2, K_s=15, lr0=0.05)
    kw = dict(seed=5, mu=0.9, wd=5e-4, sigma=0.5)
    x1, v1 = inputs.zero_state(n, P)
    t1 = O.run(x1, v1, h, c, spec=spec, **kw)
    x2, v2 = inputs.zero_state(n, P)
    st = O.new_state(spec)
    ta = O.run(x2, v2, h, c, spec=spec, state=st, k_begin=0, k_end=27, **kw)
    tb = O.run(x2, v2, h, c, spec=spec, state=st, k_begin=27, k_end=60, **kw)
    assert np.array_equal(x1, x2) and np.array_equal(v1, v2)
    assert list(t1.k) == list(ta.k) + list(tb.k)
    assert list(t1.p) == list(ta.p) + list(tb.p)
    assert list(t1.S) == list(ta.S) + list(tb.S)


def test_run_trace_semantics():
    # S is D / n of the pre-average replicas, and the rule sees the gamma of the sync iteration.
    n, P = 4, 256
    h = inputs.draw_h(P, "uniform:0.1:1", 2)
    c = inputs.draw_c(P, 1.0, 2)
    spec = O.ScheduleSpec(kind=0, K=8, p_init=4, lr0=0.05)
    x, v = inputs.zero_state(n, P)
    tr = O.run(x, v, h, c, spec=spec, seed=3, mu=0.9, wd=0.0, sigma=0.5)
    x2, v2 = inputs.zero_state(n, P)
    for k in range(4):
        O.local_step(x2, v2, h, c, seed=3, k=k, gamma=0.05, mu=0.9, wd=0.0, sigma=0.5)
    D = O.variance(x2)
    assert tr.k[0] == 3 and tr.S[0] == D / n and tr.phase[0] == O.PHASE_CONSTANT


# ---------------------------------------------------------------------------------------------
# wire accounting
# ---------------------------------------------------------------------------------------------

def _simulate_ring_allreduce_bytes(n, P, elem=4):
    """Count the bytes one node sends in a ring allreduce of P elements, chunk by chunk."""
    chunks = [P // n + (1 if r < P % n else 0) for r in range(n)]
    sent = 0
    for step in range(n - 1):                 # reduce-scatter: node 0 sends chunk (0 - step) mod n
        sent += chunks[(0 - step) % n] * elem
    for step in range(n - 1):                 # all-gather: node 0 forwards chunk (1 - step) mod n
        sent += chunks[(1 - step) % n] * elem
    return sent


@pytest.mark.parametrize("n,P", [(2, 1000), (4, 1 << 20), (16, 25_557_032), (8, 11_689_512)])
def test_wire_bytes_match_ring_simulation(n, P):
    per_node, total = O.wire_bytes(n, P, 1, with_scalar=False)
    sim = _simulate_ring_allreduce_bytes(n, P)
    assert abs(per_node - sim) <= 2 * 4 * n  # the formula spreads uneven chunks evenly
    assert total == pytest.approx(per_node * n)


def test_wire_bytes_ratios():
    assert O.wire_bytes(1, 1000, 50) == (0.0, 0.0)
    K, P, n = 4000, 1000, 16
    full = O.wire_bytes(n, P, K, with_scalar=False)[0]
    adp = O.wire_bytes(n, P, K // 8, with_scalar=False)[0]
    # 8-bit gradient quantisation moves 1/4 of full communication and twice ADPSGD (Sec. IV-B).
    assert full / adp == pytest.approx(8.0) and (full / 4) / adp == pytest.approx(2.0)


def test_sync_at_K_s_is_not_sampled():
    # Algorithm 2 samples only while k < K_s: a sync exactly at k = K_s already adapts.
    spec = ads(200, 4, K_s=99)
    S = np.concatenate([np.full(24, 1.0), np.full(100, 1e-6)])
    _, ks, ps = O.schedule_only(spec, S)
    assert ks[24] == 99 and ps[23] == 4
    assert ps[24] == 5  # sync 25 sees S << 0.7 gamma C2 and is not sampled


def test_step_size_of_each_iteration_in_a_run():
    # mu = 0, sigma = 0, one milestone: x after iterations 0..k is c + prod_t (1 - gamma_t h)(x0 - c).
    n, P = 2, 64
    h = inputs.draw_h(P, "uniform:0.1:1", 4)
    c = inputs.draw_c(P, 1.0, 4)
    spec = O.ScheduleSpec(kind=0, K=8, p_init=1, lr0=0.5, lr_factor=0.1, milestones=(4,))
    x, v = inputs.zero_state(n, P)
    tr = O.run(x, v, h, c, spec=spec, seed=0, mu=0.0, wd=0.0, sigma=0.0)
    fac = np.ones(P)
    for k in range(8):
        g = np.float64(np.float32(0.5 if k < 4 else 0.05))
        fac = fac * (1.0 - g * h.astype(np.float64))
        xk = c.astype(np.float64) * (1.0 - fac)
        expect = 0.5 * np.sum(h * (xk - c) ** 2)
        assert tr.loss[k] == pytest.approx(expect, rel=1e-5)


def test_piecewise_strategies_sync_counts():
    # Sec. III-A: strategy 1 (p = 4 for 2000 iterations, then 8) and strategy 2 (8, then 4) both
    # sync 750 times in 4000 iterations; Sec. V-B: 20 then 5 syncs 500 times.
    def count(p0, p1):
        spec = O.ScheduleSpec(kind=2, K=4000, p_init=p0, period_changes=((2000, p1),))
        return O.schedule_only(spec, [])
    s1, k1, p1 = count(4, 8)
    s2, _, _ = count(8, 4)
    s3, _, _ = count(20, 5)
    assert (s1, s2, s3) == (750, 750, 500)
    assert k1[499] == 1999 and k1[500] == 2007 and set(p1[:500]) == {4} and set(p1[500:]) == {8}


def test_variance_trace_resets_at_syncs_and_matches_second_moment():
    # Var[W_k] (Sec. II-B) recorded at the start of every iteration: exactly 0 at k = 0 and right
    # after every sync, and t steps into an interval its mean is the second moment of the spread.
    n, P, p, K = 4, 1 << 14, 4, 40
    gamma, sigma = 0.1, 0.5
    h = inputs.draw_h(P, "uniform:0.1:1", 6)
    c = inputs.draw_c(P, 1.0, 6)
    x, v = inputs.zero_state(n, P)
    spec = O.ScheduleSpec(kind=0, K=K, p_init=p, lr0=gamma)
    tr = O.run(x, v, h, c, spec=spec, seed=17, mu=0.0, wd=0.0, sigma=sigma, track_variance=True)
    var = tr.var
    assert var[0] == 0.0 and all(var[k] == 0.0 for k in range(p, K, p))
    g = np.float64(np.float32(gamma))
    hh = h.astype(np.float64)
    for t in range(1, p):
        # E[D] after t steps from identical replicas, mu = 0: (n-1) sum_j g^2 sigma^2 sum_{s<t} (1-g h)^(2s)
        ED = (n - 1) * np.sum(g * g * sigma * sigma * sum((1 - g * hh) ** (2 * s) for s in range(t)))
        got = np.mean([var[k] for k in range(t, K, p)]) * n
        assert abs(got / ED - 1) < 5 * np.sqrt(2.0 / ((n - 1) * P * (K // p)))


def test_imagenet_step_size_schedule():
    # Sec. IV-C: warm-up from 0.1, +0.1 per epoch for 8 epochs (0.8), x0.1 at epochs 30 and 60.
    L = 10  # iterations per epoch
    spec = O.ScheduleSpec(kind=0, K=90 * L, p_init=1, lr0=0.1, lr_factor=0.1, milestones=(30 * L, 60 * L),
                          lr_warmup_steps=8, lr_warmup_len=L)
    expect = {0: 0.1, L - 1: 0.1, L: 0.2, 3 * L + 5: 0.4, 7 * L: 0.8, 8 * L: 0.8, 29 * L + 9: 0.8,
              30 * L: 0.08, 59 * L: 0.08, 60 * L: 0.008, 89 * L: 0.008}
    for k, g in expect.items():
        assert O.gamma(spec, k) == np.float32(g), (k, O.gamma(spec, k), g)


def test_piecewise_change_inside_an_interval():
    # p = 4 until iteration 5, p = 2 from iteration 6 on: iterations 4, 5, 6 count 1, 2, 3, and at
    # k = 6 the period in force is already 2, so the sync falls at 6; then every 2 iterations.
    spec = O.ScheduleSpec(kind=2, K=12, p_init=4, period_changes=((6, 2),))
    syncs, ks, ps = O.schedule_only(spec, [])
    assert list(ks) == [3, 6, 8, 10] and list(ps) == [4, 2, 2, 2]


def test_piecewise_ignores_the_variance():
    # A set period is never adapted, whatever S the syncs report.
    spec = O.ScheduleSpec(kind=2, K=400, p_init=4, K_s=0, period_changes=((200, 8),))
    _, ks, ps = O.schedule_only(spec, np.full(200, 5.0))
    assert set(ps[:50]) == {4} and set(ps[50:]) == {8}
    st = O.new_state(spec)
    assert O.on_sync(spec, st, 10, 5.0, 0.1) == O.PHASE_CONSTANT and st.p == 4
