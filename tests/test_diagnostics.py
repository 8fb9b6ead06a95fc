"""The paper's variance summaries (Eq. vt, Eq. metric2) from a recorded series, pinned by hand
examples and closed forms."""
import numpy as np
import pytest

from paper_2007_06134_gb300 import diagnostics as dg


def test_interval_means_hand_example():
    var = [0.0, 1.0, 2.0, 3.0, 0.0, 5.0, 7.0]
    # syncs after iterations 3 and 6: intervals {0..3} and {4..6}
    assert np.allclose(dg.interval_means(var, [3, 6]), [1.5, 4.0])


def test_interval_means_linear_growth_closed_form():
    # Var[W_k] = (k - last sync start): mean over an interval of p iterations = (p - 1) / 2
    p, T = 8, 50
    var = np.tile(np.arange(p, dtype=float), T)
    sync_k = [p * t + p - 1 for t in range(T)]
    assert np.allclose(dg.interval_means(var, sync_k), (p - 1) / 2.0)


def test_weighted_variance_matches_interval_form_for_constant_gamma():
    # With a constant step size Eq. metric2 over whole intervals equals the mean of V_t (Eq. equals).
    rng = np.random.default_rng(0)
    p, T = 5, 40
    var = rng.uniform(0, 1, p * T)
    sync_k = [p * t + p - 1 for t in range(T)]
    assert dg.weighted_variance(var, np.full(p * T, 0.1)) == pytest.approx(dg.interval_means(var, sync_k).mean())


def test_weighted_variance_weights_by_step_size():
    var = [1.0, 1.0, 4.0, 4.0]
    g = [0.1, 0.1, 0.01, 0.01]
    assert dg.weighted_variance(var, g) == pytest.approx((0.2 * 1 + 0.02 * 4) / 0.22)
    assert dg.phase_means(var, [0, 2, 4]) == [1.0, 4.0]
