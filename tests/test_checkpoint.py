"""Checkpoint files: the scheduler state and arrays round-trip exactly (CPU), and a run resumed
from a file in a fresh context continues with the same bits as an unsplit run (GPU)."""
import numpy as np
import pytest

from paper_2007_06134_gb300 import abi, checkpoint, inputs


def test_state_and_arrays_round_trip(tmp_path):
    st = abi.State(k_next=1234, cnt=3, p=17, C2=0.123456789012345, m=42, rounds=99)
    x = np.random.default_rng(0).standard_normal((3, 7)).astype(np.float32)
    v = -x
    trace = {"k": np.arange(5), "S": np.linspace(0, 1, 5)}
    path = str(tmp_path / "ck.npz")
    checkpoint.save(path, x, v, st, trace)
    x2, v2, st2, tr2 = checkpoint.load(path)
    assert np.array_equal(x, x2) and np.array_equal(v, v2)
    assert checkpoint.state_to_dict(st) == checkpoint.state_to_dict(st2)
    assert np.array_equal(tr2["k"], trace["k"]) and np.array_equal(tr2["S"], trace["S"])


@pytest.mark.gpu
def test_resume_from_file_is_bit_identical(tmp_path):
    torch = pytest.importorskip("torch")
    w = inputs.WORKLOADS["quadratic-n4-P1M"]
    n, P, K = 4, 8195, 70
    h, c = inputs.problem(w, P)
    hd, cd = torch.from_numpy(h).cuda(), torch.from_numpy(c).cuda()
    sched = abi.make_schedule(abi.ADPSGD, K, 3, K_s=20, lr0=w.lr0)
    cfg = abi.make_config(n, P, momentum=0.9, noise_sigma=0.5, seed=21)
    xa = torch.zeros((n, P), device="cuda")
    va = torch.zeros_like(xa)
    ta = abi.TraceBuffers(K)
    with abi.adpsgd_init(cfg, xa, va, hd, cd) as ctx:
        abi.adpsgd_run(ctx, sched, abi.adpsgd_state_init(sched), trace=ta)
    xb = torch.zeros((n, P), device="cuda")
    vb = torch.zeros_like(xb)
    tb = abi.TraceBuffers(K)
    path = str(tmp_path / "mid.npz")
    with abi.adpsgd_init(cfg, xb, vb, hd, cd) as ctx:
        st = abi.adpsgd_state_init(sched)
        abi.adpsgd_run(ctx, sched, st, k_end=41, trace=tb)
        checkpoint.save(path, xb, vb, st, tb.arrays())
    x2, v2, st2, tr = checkpoint.load(path)
    xc, vc = torch.from_numpy(x2).cuda(), torch.from_numpy(v2).cuda()
    tc = abi.TraceBuffers(K)
    with abi.adpsgd_init(cfg, xc, vc, hd, cd) as ctx:
        abi.adpsgd_run(ctx, sched, st2, trace=tc)
    torch.cuda.synchronize()
    assert torch.equal(xa, xc) and torch.equal(va, vc)
    A, C = ta.arrays(), tc.arrays()
    assert np.array_equal(A["k"], np.concatenate([tr["k"], C["k"]]))
    assert np.array_equal(A["S"], np.concatenate([tr["S"], C["S"]]))
