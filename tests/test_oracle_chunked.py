"""The oracle's chunked all-core run against its single-thread run (no GPU).

The chunked form runs the same per-element code on fixed column chunks in parallel and adds the
fp64 partial sums of D and the loss in chunk order.  So x, v, the sync iterations, the periods
and the phases must equal the single-thread run bit for bit, at any thread count; S, the loss and
the per-iteration variance may differ only by the order of fp64 additions: two orders of a sum of
m nonnegative terms are each within (m - 1) 2^-53 of the exact sum (recursive summation), so
within 2 m 2^-53 of each other.  The chunked sums do not depend on the thread count at all.
"""
import numpy as np
import pytest

from oracle import oracle as O
from paper_2007_06134_gb300 import inputs

U = 2.0 ** -53


def _case(n, P, noise):
    w = inputs.WORKLOADS["resnet50-n16-bf16noise" if noise else "resnet18-n8"]
    h, c = inputs.problem(w, P)
    nz = O.noise_bf16(w.seed, n, P) if noise else None
    return w, h, c, nz


@pytest.mark.parametrize("n,P,chunk,noise,kind", [
    (3, 4099, 64, False, 1),      # ragged P, 65 chunks, the last one short
    (8, 1 << 14, 1 << 12, False, 1),
    (4, 1000, 4, False, 0),       # one Philox block per chunk, constant period
    (5, 777, 1 << 16, True, 1),   # a single chunk larger than P, bf16 noise tensor
])
def test_chunked_run_equals_single_thread_run(n, P, chunk, noise, kind):
    w, h, c, nz = _case(n, P, noise)
    spec = O.ScheduleSpec(kind=kind, K=40, p_init=2, K_s=12, lr0=w.lr0, milestones=(25,))
    x0, v0 = inputs.random_state(n, P, 3)
    ref_x, ref_v = x0.copy(), v0.copy()
    ref = O.run(ref_x, ref_v, h, c, spec=spec, seed=w.seed, mu=w.mu, wd=5e-4, sigma=w.sigma, noise=nz,
                track_variance=True)
    sums = {}
    for threads in (1, 3, O.host_threads()):
        x, v = x0.copy(), v0.copy()
        tr = O.run(x, v, h, c, spec=spec, seed=w.seed, mu=w.mu, wd=5e-4, sigma=w.sigma, noise=nz,
                   track_variance=True, threads=threads, chunk=chunk)
        assert np.array_equal(x.view(np.uint32), ref_x.view(np.uint32))
        assert np.array_equal(v.view(np.uint32), ref_v.view(np.uint32))
        assert tr.syncs == ref.syncs
        for key in ("k", "p", "phase"):
            assert np.array_equal(getattr(tr, key), getattr(ref, key)), key
        bound = 2 * n * P * U
        for key in ("S", "loss"):
            a, b = getattr(tr, key), getattr(ref, key)
            assert np.all(np.abs(a - b) <= bound * np.abs(b)), key
        assert np.all(np.abs(tr.C2 - ref.C2) <= 4 * bound * np.abs(ref.C2))
        assert np.all(np.abs(tr.var - ref.var) <= bound * np.abs(ref.var))
        sums[threads] = (tr.S.copy(), tr.loss.copy(), tr.var.copy())
    first = sums[1]
    for got in sums.values():
        for a, b in zip(got, first):
            assert np.array_equal(a, b), "the chunked sums depend on the thread count"


def test_chunk_must_be_a_multiple_of_4():
    w, h, c, _ = _case(2, 64, False)
    x, v = inputs.zero_state(2, 64)
    spec = O.ScheduleSpec(kind=0, K=4, p_init=2)
    with pytest.raises(ValueError):
        O.run(x, v, h, c, spec=spec, seed=1, mu=0.9, wd=0.0, sigma=1.0, threads=2, chunk=6)
