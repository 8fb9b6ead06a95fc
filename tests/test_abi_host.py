"""The C-ABI library on a machine without a GPU: it loads, exports every entry point its
header declares, and its host-side logic (Algorithm 2's period rule, the step-size
schedule, the wire accounting, argument checks) agrees with the oracle.  No call here
launches GPU work."""
import ctypes as C

import numpy as np
import pytest

from oracle import oracle as O
from paper_2007_06134_gb300 import abi


def test_library_exports_every_header_entry_point():
    lib = abi.load()
    names = abi.header_entry_points()
    assert len(names) >= 18
    for name in names:
        assert hasattr(lib, name), name
    assert set(names) == set(abi._SIGS)


def test_strerror_covers_every_status():
    for st in (abi.OK, abi.E_INVAL, abi.E_ALIGN, abi.E_CUDA, abi.E_TIMEOUT, abi.E_NOMEM, abi.E_STATE, abi.E_PEER):
        assert abi.strerror(st) and abi.strerror(st) != "unknown status"
    assert abi.strerror(12345) == "unknown status"


def _pair(kind, K, p_init, **kw):
    ms = kw.pop("milestones", ())
    lib_s = abi.make_schedule(kind, K, p_init, milestones=ms, **kw)
    orc_s = O.ScheduleSpec(kind=kind, K=K, p_init=p_init, milestones=ms, **kw)
    return lib_s, orc_s


@pytest.mark.parametrize("seed", range(6))
def test_period_rule_matches_oracle_on_random_scripts(seed):
    rng = np.random.default_rng(seed)
    K = 3000
    lib_s, orc_s = _pair(abi.ADPSGD, K, int(rng.integers(1, 6)), K_s=int(rng.integers(100, 600)),
                         K_w=int(rng.integers(0, 20)), lr0=0.1, lr_factor=0.1, milestones=(1000, 2000),
                         p_max=int(rng.integers(0, 2)) * 30)
    if orc_s.K_s < orc_s.K_w + orc_s.p_init:
        orc_s.K_s = lib_s.K_s = orc_s.K_w + orc_s.p_init
    st = abi.adpsgd_state_init(lib_s)
    ost = O.new_state(orc_s)
    # drive both rules with the same sync iterations and scripted variances
    S_scale = rng.uniform(0.1, 10.0)
    for k in range(K):
        g = abi.adpsgd_gamma(lib_s, k)
        assert g == O.gamma(orc_s, k)
        if rng.random() < 0.15:
            S = S_scale * rng.lognormal(0.0, 0.6) * g
            ph = abi.adpsgd_sched_on_sync(lib_s, st, k, S, g)
            oph = O.on_sync(orc_s, ost, k, S, g)
            assert (ph, st.p, st.C2, st.m) == (oph, ost.p, ost.C2, ost.m)


@pytest.mark.parametrize("changes", [((2000, 8),), ((2000, 4),), ((2000, 5),), ((10, 3), (17, 9), (400, 1))])
def test_piecewise_period_matches_oracle(changes):
    K, p0 = 4000, 4
    lib_s = abi.make_schedule(abi.PIECEWISE, K, p0, period_changes=changes)
    orc_s = O.ScheduleSpec(kind=2, K=K, p_init=p0, period_changes=changes)
    syncs, ks, ps = O.schedule_only(orc_s, [])
    # drive the library's rule through the same iterations: it only ever reports constant phase
    st = abi.adpsgd_state_init(lib_s)
    for k in ks[:50]:
        assert abi.adpsgd_sched_on_sync(lib_s, st, int(k), 1.0, 0.1) == abi.PHASE_CONSTANT


def test_wire_bytes_match_oracle():
    for n, P, R in ((1, 10, 5), (8, 11_689_512, 250), (16, 25_557_032, 125), (3, 7, 0)):
        assert abi.adpsgd_wire_bytes(n, P, R, True) == O.wire_bytes(n, P, R, True)
        assert abi.adpsgd_wire_bytes(n, P, R, False) == O.wire_bytes(n, P, R, False)


def test_schedule_validation():
    ok = abi.make_schedule(abi.ADPSGD, 100, 4, K_s=25)
    abi.adpsgd_state_init(ok)
    bad = [abi.make_schedule(abi.ADPSGD, 100, 4, K_s=3),          # C_2 would never be sampled
           abi.make_schedule(abi.ADPSGD, 100, 0, K_s=25),         # p < 1
           abi.make_schedule(abi.CPSGD, -1, 4),
           abi.make_schedule(abi.ADPSGD, 100, 4, K_s=25, lo=1.5, hi=1.3),
           abi.make_schedule(abi.CPSGD, 100, 4, p_min=0),
           abi.make_schedule(abi.CPSGD, 100, 4, lr0=0.0),
           abi.make_schedule(abi.ADPSGD, 100, 4, K_s=25, literal_phase=True),
           abi.make_schedule(3, 100, 4),
           abi.make_schedule(abi.PIECEWISE, 100, 4, period_changes=((50, 8), (40, 2))),
           abi.make_schedule(abi.PIECEWISE, 100, 4, period_changes=((50, 0),))]
    for s in bad:
        with pytest.raises(abi.AdpsgdError) as e:
            abi.adpsgd_state_init(s)
        assert e.value.status == abi.E_INVAL


def test_init_argument_checks_before_any_cuda_call():
    lib = abi.load()
    out = C.c_void_p(123)
    cfg = abi.make_config(4, 1024)
    assert lib.adpsgd_init(C.byref(cfg), None, 16, 16, 16, None, None, C.byref(out)) == abi.E_INVAL
    assert out.value is None
    assert lib.adpsgd_init(C.byref(cfg), 16, 32, 48, 8, None, None, C.byref(out)) == abi.E_ALIGN
    for n, P in ((0, 10), (4, 0), (-1, 5)):
        bad = abi.make_config(n, P)
        assert lib.adpsgd_init(C.byref(bad), 16, 32, 48, 64, None, None, C.byref(out)) == abi.E_INVAL
    bf = abi.make_config(4, 1024, noise_mode=abi.NOISE_BF16)
    assert lib.adpsgd_init(C.byref(bf), 16, 32, 48, 64, None, None, C.byref(out)) == abi.E_INVAL
    assert lib.adpsgd_local_steps(None, 0, 1, None) == abi.E_INVAL
    assert lib.adpsgd_init_replicas(None, 16) == abi.E_INVAL
    assert lib.adpsgd_philox_fill(0, 0, 1, 4, 0, None, None) == abi.E_INVAL
    assert lib.adpsgd_philox_fill(0, 0, 1, 4, 0, 8, None) == abi.E_ALIGN
    assert lib.adpsgd_philox_fill(0, 0, 1, 4, 1 << 32, 16, None) == abi.E_INVAL
    assert lib.adpsgd_philox_fill(0, 0, 1 << 20, 1 << 30, 0, 16, None) == abi.E_INVAL
    assert lib.adpsgd_noise_fill_f32(0, 0, 1 << 10, 1 << 34, 0, 16, None) == abi.E_INVAL
    assert lib.adpsgd_noise_fill_bf16(0, 1 << 10, 1 << 34, 16, None) == abi.E_INVAL
    assert lib.adpsgd_noise_fill_bf16(0, 1, (1 << 34) + 1, 16, None) == abi.E_INVAL
    big = abi.make_config(1 << 10, 1 << 34)
    assert lib.adpsgd_init(C.byref(big), 16, 32, 48, 64, None, None, C.byref(out)) == abi.E_INVAL
    lib.adpsgd_destroy(None)


def test_step_size_warmup_matches_oracle():
    L = 7
    kw = dict(lr0=0.1, lr_factor=0.1, milestones=(30 * L, 60 * L), lr_warmup_steps=8, lr_warmup_len=L)
    lib_s = abi.make_schedule(abi.CPSGD, 90 * L, 1, **kw)
    orc_s = O.ScheduleSpec(kind=0, K=90 * L, p_init=1, **kw)
    for k in range(90 * L):
        assert abi.adpsgd_gamma(lib_s, k) == O.gamma(orc_s, k)
    with pytest.raises(abi.AdpsgdError):
        abi.adpsgd_state_init(abi.make_schedule(abi.CPSGD, 10, 1, lr_warmup_steps=2, lr_warmup_len=0))
