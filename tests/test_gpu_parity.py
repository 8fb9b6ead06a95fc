"""GPU parity: the CUDA path through the C ABI against the CPU oracle, element by element.

Bar (stated for fp32 in the target): Philox words, normals, the bf16 noise tensor, x, v,
the replica mean and the period schedule bit-exact; D (sum_i ||x_i - xbar||^2) and the
loss within relative 1e-4 (the kernel sums fp32 column terms in a tree, the oracle sums the
definition in fp64 in index order; the observed gap is ~1e-7).  Sizes span several blocks
and ragged tails (P mod 4 != 0, P < 4), n = 1 and n above the register-resident limit.
"""
import ctypes as C
import os
import subprocess

import numpy as np
import pytest

from oracle import oracle as O
from paper_2007_06134_gb300 import abi, inputs

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
DEV = "cuda:0"
REL_D = 1e-4


def dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).to(DEV)


def host(t):
    torch.cuda.synchronize()
    return t.cpu().numpy()


def rel(a, b):
    return abs(a - b) / max(abs(b), 1e-300)


# ---------------------------------------------------------------------------------------------
# generator
# ---------------------------------------------------------------------------------------------

@pytest.mark.parametrize("seed,tag,k", [(0, 0, 0), (0x2007061340000001, 0, 7), (0xFFFFFFFFFFFFFFFF, 1, 0),
                                        (12345, 0, (1 << 32) - 1), (1 << 40, 3, 99999)])
def test_philox_words_bit_exact(seed, tag, k):
    n, nq = 5, 1037
    out = torch.zeros((n, nq, 4), dtype=torch.int32, device=DEV)
    abi.adpsgd_philox_fill(seed, tag, n, nq, k, out)
    got = host(out).view(np.uint32)
    for i in range(n):
        assert np.array_equal(got[i], O.philox_words(seed, tag, i, k, 0, nq))


@pytest.fixture(scope="module")
def curand_ref(tmp_path_factory):
    src = os.path.join(os.path.dirname(__file__), "cuda", "curand_philox_ref.cu")
    so = str(tmp_path_factory.mktemp("curand") / "libcurand_ref.so")
    subprocess.check_call(["nvcc", "-gencode", "arch=compute_103a,code=sm_103a", "-O2", "-shared",
                           "-Xcompiler", "-fPIC", "-cudart", "static", "-o", so, src])
    lib = C.CDLL(so)
    lib.curand_ref_fill.argtypes = [C.c_uint64, C.c_uint32, C.c_int, C.c_longlong, C.c_uint32, C.c_void_p,
                                    C.c_void_p]
    return lib


@pytest.mark.parametrize("seed,tag,k", [(0, 0, 0), (0xDEADBEEFCAFEF00D, 0, 123), (7, 1, 0)])
def test_philox_matches_curand(curand_ref, seed, tag, k):
    # cuRAND's Philox4x32-10 is an independent implementation of the same published generator.
    n, nq = 3, 777
    raw = torch.zeros((n, nq, 4), dtype=torch.int32, device=DEV)
    api = torch.zeros_like(raw)
    torch.cuda.synchronize()
    assert curand_ref.curand_ref_fill(seed, tag, n, nq, k, raw.data_ptr(), api.data_ptr()) == 0
    mine = torch.zeros_like(raw)
    abi.adpsgd_philox_fill(seed, tag, n, nq, k, mine)
    m, r, a = host(mine), host(raw), host(api)
    assert np.array_equal(m, r)
    assert np.array_equal(m, a)
    assert np.array_equal(r[0].view(np.uint32), O.philox_words(seed, tag, 0, k, 0, nq))


@pytest.mark.parametrize("P", [1, 3, 4, 5, 1023, 4099, 65539])
@pytest.mark.parametrize("k", [0, 17])
def test_normals_bit_exact(P, k):
    n, seed = 3, 0x5EED
    out = torch.empty((n, P), dtype=torch.float32, device=DEV)
    abi.adpsgd_noise_fill_f32(seed, 0, n, P, k, out)
    got = host(out)
    for i in range(n):
        assert np.array_equal(got[i].view(np.uint32), O.normals(seed, 0, i, k, 0, P).view(np.uint32))


def test_normals_exhaustive_words_sample():
    # A large sample (2^22 normals) of the stream, bit for bit.
    n, P, seed = 4, 1 << 20, 0xABCDEF
    out = torch.empty((n, P), dtype=torch.float32, device=DEV)
    abi.adpsgd_noise_fill_f32(seed, 0, n, P, 3, out)
    got = host(out)
    for i in range(n):
        assert np.array_equal(got[i].view(np.uint32), O.normals(seed, 0, i, 3, 0, P).view(np.uint32))


@pytest.mark.parametrize("n,P", [(1, 1), (2, 7), (16, 4099), (3, 100000)])
def test_bf16_noise_bit_exact(n, P):
    out = torch.empty((n, P), dtype=torch.int16, device=DEV)
    abi.adpsgd_noise_fill_bf16(99, n, P, out)
    assert np.array_equal(host(out).view(np.uint16), O.noise_bf16(99, n, P))


# ---------------------------------------------------------------------------------------------
# local step
# ---------------------------------------------------------------------------------------------

def _problem(P, seed=1):
    w = inputs.WORKLOADS["resnet18-n8"]
    return inputs.draw_h(P, w.h_dist, seed), inputs.draw_c(P, 1.0, seed)


@pytest.mark.parametrize("n", [1, 3, 8])
@pytest.mark.parametrize("P", [1, 3, 5, 1024, 4099, 65536 + 3])
@pytest.mark.parametrize("wd", [0.0, 5e-4])
def test_local_steps_bit_exact(n, P, wd):
    h, c = _problem(P)
    x, v = inputs.random_state(n, P, 7)
    seed, k0, lrs = 0x1234567890, 5, [0.1, 0.05, 0.01]
    xd, vd, hd, cd = dev(x), dev(v), dev(h), dev(c)
    cfg = abi.make_config(n, P, momentum=0.9, weight_decay=wd, noise_sigma=0.5, seed=seed)
    with abi.adpsgd_init(cfg, xd, vd, hd, cd) as ctx:
        abi.adpsgd_local_steps(ctx, k0, lrs)
        gx, gv = host(xd), host(vd)
    for t, lr in enumerate(lrs):
        O.local_step(x, v, h, c, seed=seed, k=k0 + t, gamma=lr, mu=0.9, wd=wd, sigma=0.5)
    assert np.array_equal(gx.view(np.uint32), x.view(np.uint32))
    assert np.array_equal(gv.view(np.uint32), v.view(np.uint32))


@pytest.mark.parametrize("n,P", [(16, 4096), (4, 4099), (2, 2)])
def test_local_steps_bf16_noise_bit_exact(n, P):
    h, c = _problem(P, 2)
    x, v = inputs.random_state(n, P, 8)
    noise = O.noise_bf16(77, n, P)
    xd, vd, hd, cd = dev(x), dev(v), dev(h), dev(c)
    nd = dev(noise.view(np.int16))
    cfg = abi.make_config(n, P, momentum=0.9, noise_sigma=1.0, seed=77, noise_mode=abi.NOISE_BF16)
    with abi.adpsgd_init(cfg, xd, vd, hd, cd, nd) as ctx:
        abi.adpsgd_local_steps(ctx, 0, [0.05, 0.05])
        gx, gv = host(xd), host(vd)
    for k in range(2):
        O.local_step(x, v, h, c, seed=77, k=k, gamma=0.05, mu=0.9, wd=0.0, sigma=1.0, noise=noise)
    assert np.array_equal(gx.view(np.uint32), x.view(np.uint32))
    assert np.array_equal(gv.view(np.uint32), v.view(np.uint32))


def test_last_step_index_of_the_counter():
    n, P = 2, 64
    h, c = _problem(P)
    x, v = inputs.random_state(n, P, 9)
    xd, vd = dev(x), dev(v)
    cfg = abi.make_config(n, P, noise_sigma=1.0, seed=3)
    with abi.adpsgd_init(cfg, xd, vd, dev(h), dev(c)) as ctx:
        abi.adpsgd_local_steps(ctx, (1 << 32) - 1, [0.1])
        with pytest.raises(abi.AdpsgdError):
            abi.adpsgd_local_steps(ctx, (1 << 32) - 1, [0.1, 0.1])
        gx = host(xd)
    O.local_step(x, v, h, c, seed=3, k=(1 << 32) - 1, gamma=0.1, mu=0.9, wd=0.0, sigma=1.0)
    assert np.array_equal(gx, x)


# ---------------------------------------------------------------------------------------------
# averaging + variance
# ---------------------------------------------------------------------------------------------

@pytest.mark.parametrize("n", [1, 2, 3, 4, 5, 8, 13, 16, 17, 32, 33, 40])
@pytest.mark.parametrize("P", [1, 7, 4, 4096, 4099, 100003, 1024 * 300 + 12, 512 * 77 + 8])
def test_average_and_variance(n, P):
    h, c = _problem(P, 3)
    x, _ = inputs.random_state(n, P, 10 + n)
    xd = dev(x)
    cfg = abi.make_config(n, P)
    with abi.adpsgd_init(cfg, xd, torch.zeros_like(xd), dev(h), dev(c)) as ctx:
        Dv = abi.adpsgd_variance(ctx)
        assert np.array_equal(host(xd), x)       # variance only: no write-back
        D, L = abi.adpsgd_average_and_variance(ctx)
        gx = host(xd)
        D2, _ = abi.adpsgd_average_and_variance(ctx)
    Do, Lo = O.average_variance(x, h, c)
    assert np.array_equal(gx.view(np.uint32), x.view(np.uint32))
    if n == 1:
        assert D == 0.0 and Dv == 0.0
    else:
        assert rel(D, Do) < REL_D and rel(Dv, Do) < REL_D
    assert rel(L, Lo) < REL_D
    assert D2 == 0.0  # variance is exactly zero right after averaging


def test_average_exact_offsets_closed_form():
    n, P, d = 8, 4096 * 3 + 1, 2.0 ** -10
    rng = np.random.default_rng(0)
    b = (rng.integers(-8192, 8192, P) * 2.0 ** -12).astype(np.float32)
    x = np.stack([b + np.float32(i * d) for i in range(n)]).astype(np.float32)
    xd = dev(x)
    with abi.adpsgd_init(abi.make_config(n, P, want_loss=False), xd, torch.zeros_like(xd), dev(b), dev(b)) as ctx:
        D, _ = abi.adpsgd_average_and_variance(ctx, want_loss=False)
    assert D == P * d * d * n * (n * n - 1) / 12.0


# ---------------------------------------------------------------------------------------------
# whole schedules
# ---------------------------------------------------------------------------------------------

def _run_both(w: inputs.Workload, P, K, kind, p, *, K_s=0, milestones=(), n=None, lr0=None, sample=None):
    n = w.n if n is None else n
    lr0 = w.lr0 if lr0 is None else lr0
    h, c = inputs.problem(w, P)
    x, v = inputs.zero_state(n, P)
    noise = O.noise_bf16(w.seed, n, P) if w.noise == "bf16" else None
    xd, vd = dev(x), dev(v)
    cfg = abi.make_config(n, P, momentum=w.mu, weight_decay=w.wd, noise_sigma=w.sigma, seed=w.seed,
                          noise_mode=abi.NOISE_BF16 if noise is not None else abi.NOISE_PHILOX)
    sched = abi.make_schedule(kind, K, p, K_s=K_s, lr0=lr0, lr_factor=w.lr_factor, milestones=milestones)
    tr = abi.TraceBuffers(100000)
    nd = dev(noise.view(np.int16)) if noise is not None else None
    with abi.adpsgd_init(cfg, xd, vd, dev(h), dev(c), nd) as ctx:
        st = abi.adpsgd_state_init(sched)
        stats = abi.adpsgd_run(ctx, sched, st, trace=tr)
        gx, gv = host(xd), host(vd)
    spec = O.ScheduleSpec(kind=kind, K=K, p_init=p, K_s=K_s, lr0=lr0, lr_factor=w.lr_factor,
                          milestones=milestones)
    otr = O.run(x, v, h, c, spec=spec, seed=w.seed, mu=w.mu, wd=w.wd, sigma=w.sigma, noise=noise)
    return tr.arrays(), stats, gx, gv, otr, x, v


def _decision_margin(otr, spec_lo=0.7, spec_hi=1.3, lr_of=None):
    """Smallest relative distance of S / (gamma C_2) from the 0.7 and 1.3 thresholds over the
    oracle's adaptive decisions (the GPU's S differs from the oracle's by ~1e-8 relative, so a
    margin far above that makes the bit-exact schedule comparison well posed)."""
    margin = np.inf
    for k, S, C2_before, phase in zip(otr.k, otr.S, np.concatenate([[0.0], otr.C2[:-1]]), otr.phase):
        if phase != O.PHASE_ADAPTING or C2_before == 0.0:
            continue
        ratio = S / (lr_of(int(k)) * C2_before)
        margin = min(margin, abs(ratio - spec_lo) / spec_lo, abs(ratio - spec_hi) / spec_hi)
    return margin


def _assert_trace(gt, otr, lr_of=None):
    if lr_of is not None:
        assert _decision_margin(otr, lr_of=lr_of) > 1e-6
    assert np.array_equal(gt["k"], otr.k)
    assert np.array_equal(gt["p"], otr.p)
    assert np.array_equal(gt["phase"], otr.phase)
    for a, b in zip(gt["S"], otr.S):
        assert rel(a, b) < REL_D
    for a, b in zip(gt["loss"], otr.loss):
        assert rel(a, b) < REL_D
    for a, b in zip(gt["C2"], otr.C2):
        assert rel(a, b) < REL_D or (a == 0 and b == 0)


@pytest.mark.parametrize("kind", [abi.ADPSGD, abi.CPSGD])
def test_quadratic_n4_P1M_full_run(kind):
    # The small workload at full size: n = 4, P = 2^20, 100 iterations, ADPSGD (p_init 4,
    # K_s = 25) and CPSGD (p = 4), trace and final state.
    w = inputs.WORKLOADS["quadratic-n4-P1M"]
    gt, stats, gx, gv, otr, x, v = _run_both(w, w.P, w.K, kind, 4, K_s=w.K_s if kind == abi.ADPSGD else 0)
    _assert_trace(gt, otr, lr_of=lambda k: np.float64(np.float32(w.lr0)))
    assert stats.rounds == otr.syncs and stats.local_step_launches == w.K
    assert np.array_equal(gx.view(np.uint32), x.view(np.uint32))
    assert np.array_equal(gv.view(np.uint32), v.view(np.uint32))
    if kind == abi.CPSGD:
        assert stats.rounds == 25


def test_resnet18_shape_scaled_run_with_lr_steps():
    # The n = 8 workload's schedule shape (lr 0.1 stepped x0.1 at 50% / 75%, wd 5e-4, sigma 1) on a
    # smaller P with a ragged tail, ADPSGD and the equal-budget CPSGD.
    w = inputs.WORKLOADS["resnet18-n8"]
    P, K = (1 << 16) + 13, 400
    gt, stats, gx, gv, otr, x, v = _run_both(w, P, K, abi.ADPSGD, 4, K_s=100, milestones=(200, 300))
    spec = O.ScheduleSpec(kind=1, K=K, p_init=4, K_s=100, lr0=w.lr0, lr_factor=w.lr_factor, milestones=(200, 300))
    _assert_trace(gt, otr, lr_of=lambda k: np.float64(O.gamma(spec, k)))
    assert np.array_equal(gx, x) and np.array_equal(gv, v)
    p_eq = max(1, round(K / stats.rounds))
    gt2, stats2, gx2, _, otr2, x2, _ = _run_both(w, P, K, abi.CPSGD, p_eq, milestones=(200, 300))
    _assert_trace(gt2, otr2)
    assert np.array_equal(gx2, x2)


def test_bf16_noise_run():
    w = inputs.WORKLOADS["resnet50-n16-bf16noise"]
    gt, stats, gx, gv, otr, x, v = _run_both(w, 4096 * 5 + 2, 60, abi.ADPSGD, 4, K_s=15)
    _assert_trace(gt, otr)
    assert np.array_equal(gx, x) and np.array_equal(gv, v)


def test_resume_is_bit_identical():
    # A run split at k = 33, checkpointed to the host (x, v, scheduler state) and resumed in a
    # fresh context, gives the same bits as the unsplit run: the noise is keyed by the absolute step.
    w = inputs.WORKLOADS["quadratic-n4-P1M"]
    n, P, K = 4, 10007, 80
    h, c = inputs.problem(w, P)
    sched = abi.make_schedule(abi.ADPSGD, K, 2, K_s=20, lr0=0.05)
    cfg = abi.make_config(n, P, momentum=0.9, noise_sigma=0.5, seed=11)
    x0, v0 = inputs.zero_state(n, P)

    xd, vd = dev(x0), dev(v0)
    ta = abi.TraceBuffers(1000)
    with abi.adpsgd_init(cfg, xd, vd, dev(h), dev(c)) as ctx:
        abi.adpsgd_run(ctx, sched, abi.adpsgd_state_init(sched), trace=ta)
        xa, va = host(xd), host(vd)

    xd, vd = dev(x0), dev(v0)
    tb = abi.TraceBuffers(1000)
    with abi.adpsgd_init(cfg, xd, vd, dev(h), dev(c)) as ctx:
        st = abi.adpsgd_state_init(sched)
        abi.adpsgd_run(ctx, sched, st, k_end=33, trace=tb)
        xs, vs = host(xd), host(vd)
    st2 = abi.State.from_buffer_copy(st)
    assert st2.k_next == 33
    xd2, vd2 = dev(xs), dev(vs)
    with abi.adpsgd_init(cfg, xd2, vd2, dev(h), dev(c)) as ctx2:
        abi.adpsgd_run(ctx2, sched, st2, trace=tb)
        xb, vb = host(xd2), host(vd2)
    assert np.array_equal(xa, xb) and np.array_equal(va, vb)
    A, B = ta.arrays(), tb.arrays()
    for key in ("k", "p", "S", "C2", "loss", "phase"):
        assert np.array_equal(A[key], B[key])


def test_bounded_wait_times_out_and_context_survives():
    n, P = 2, 4096
    h, c = _problem(P)
    xd = torch.zeros((n, P), device=DEV)
    cfg = abi.make_config(n, P, wait_timeout_ms=200)
    with abi.adpsgd_init(cfg, xd, torch.zeros_like(xd), dev(h), dev(c)) as ctx:
        abi.adpsgd_test_force_incomplete(ctx, True)
        with pytest.raises(abi.AdpsgdError) as e:
            abi.adpsgd_average_and_variance(ctx)
        assert e.value.status == abi.E_TIMEOUT
        abi.adpsgd_test_force_incomplete(ctx, False)
        torch.cuda.synchronize()
        D, _ = abi.adpsgd_average_and_variance(ctx)
        assert D == 0.0


def test_loss_requires_want_loss():
    n, P = 2, 16
    xd = torch.zeros((n, P), device=DEV)
    cfg = abi.make_config(n, P, want_loss=False)
    z = torch.zeros(P, device=DEV)
    with abi.adpsgd_init(cfg, xd, torch.zeros_like(xd), z, z) as ctx:
        with pytest.raises(abi.AdpsgdError) as e:
            abi.adpsgd_average_and_variance(ctx, want_loss=True)
        assert e.value.status == abi.E_STATE


def test_kernel_timing_counts_launches():
    n, P = 4, 1 << 16
    h, c = _problem(P)
    xd = torch.zeros((n, P), device=DEV)
    cfg = abi.make_config(n, P, time_kernels=True)
    sched = abi.make_schedule(abi.CPSGD, 20, 4, lr0=0.05)
    with abi.adpsgd_init(cfg, xd, torch.zeros_like(xd), dev(h), dev(c)) as ctx:
        st = abi.adpsgd_state_init(sched)
        stats = abi.adpsgd_run(ctx, sched, st)
        t = abi.adpsgd_kernel_times(ctx)
    assert t["local_step_launches"] == 20 and t["average_launches"] == 5
    assert stats.local_step_launches == 20 and stats.average_launches == 5
    assert t["local_step_ms"] > 0 and t["average_ms"] > 0
