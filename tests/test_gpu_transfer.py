"""Host <-> device transfers through the C ABI (adpsgd_copy_h2d / adpsgd_copy_d2h).

Page-locked host buffers go through the library's copy kernel; other host memory through
cudaMemcpyAsync.  Both must deliver every byte, including ragged tails, interior pointers of a
pinned allocation, and empty copies.  Bad arguments are refused before anything is enqueued.
A whole run fed and read back through these calls matches the oracle.
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


def _bytes(nbytes, seed, pinned):
    g = torch.Generator().manual_seed(seed)
    t = torch.randint(0, 256, (nbytes,), dtype=torch.uint8, generator=g)
    return t.pin_memory() if pinned else t


@pytest.mark.parametrize("pinned", [True, False])
@pytest.mark.parametrize("nbytes", [0, 1, 15, 16, 17, 4096 + 3, (1 << 20) + 5, (64 << 20) + 7])
def test_round_trip(nbytes, pinned):
    src = _bytes(nbytes, nbytes, pinned)
    dev = torch.full((nbytes + 64,), 0xAB, dtype=torch.uint8, device=DEV)
    back = torch.zeros(nbytes + 64, dtype=torch.uint8)
    back = back.pin_memory() if pinned else back
    abi.adpsgd_copy_h2d(dev, src, nbytes)
    abi.adpsgd_copy_d2h(back, dev, nbytes)
    torch.cuda.synchronize()
    assert torch.equal(dev[:nbytes].cpu(), src)
    assert bool((dev[nbytes:] == 0xAB).all()), "wrote past the end"
    assert torch.equal(back[:nbytes], src) and bool((back[nbytes:] == 0).all())


def test_interior_pointers_of_a_pinned_allocation():
    big = _bytes(1 << 22, 3, True)
    dev = torch.zeros(1 << 22, dtype=torch.uint8, device=DEV)
    for off, ln in [(16, 1000), (4096, 123457), ((1 << 21) + 48, (1 << 20) + 1)]:
        abi.adpsgd_copy_h2d(dev[off:], big[off:], ln)
    torch.cuda.synchronize()
    for off, ln in [(16, 1000), (4096, 123457), ((1 << 21) + 48, (1 << 20) + 1)]:
        assert torch.equal(dev[off:off + ln].cpu(), big[off:off + ln])
    out = torch.zeros(1 << 22, dtype=torch.uint8).pin_memory()
    abi.adpsgd_copy_d2h(out[32:], dev[4096:], 123457)
    torch.cuda.synchronize()
    assert torch.equal(out[32:32 + 123457], big[4096:4096 + 123457])


def test_copies_are_stream_ordered():
    s = torch.cuda.Stream()
    src = torch.arange(1 << 20, dtype=torch.float32).pin_memory()
    dev = torch.zeros(1 << 20, device=DEV)
    out = torch.zeros(1 << 20, dtype=torch.float32).pin_memory()
    with torch.cuda.stream(s):
        abi.adpsgd_copy_h2d(dev, src, stream=s)
        dev.mul_(2.0)
        abi.adpsgd_copy_d2h(out, dev, stream=s)
    s.synchronize()
    assert torch.equal(out, 2.0 * src)


@pytest.fixture(scope="module")
def managed(tmp_path_factory):
    src = os.path.join(os.path.dirname(__file__), "cuda", "managed_alloc.cu")
    so = str(tmp_path_factory.mktemp("managed") / "libmanaged_alloc.so")
    subprocess.check_call(["nvcc", "-gencode", "arch=compute_103a,code=sm_103a", "-O2", "-shared",
                           "-Xcompiler", "-fPIC", "-o", so, src])
    lib = C.CDLL(so)
    lib.test_alloc_managed.argtypes = [C.c_size_t]
    lib.test_alloc_managed.restype = C.c_void_p
    lib.test_free_managed.argtypes = [C.c_void_p]
    lib.test_free_managed.restype = C.c_int
    return lib


@pytest.mark.parametrize("nbytes", [16, 4096 + 3, (8 << 20) + 5])
def test_managed_device_side(managed, nbytes):
    # The copy kernel takes only device memory of the current device; a managed buffer goes
    # through cudaMemcpyAsync and must still receive and return every byte.
    torch.cuda.synchronize()
    ptr = managed.test_alloc_managed(nbytes + 16)
    assert ptr
    try:
        src = _bytes(nbytes, 7 + nbytes, True)
        abi.adpsgd_copy_h2d(ptr, src, nbytes)
        torch.cuda.synchronize()
        got = np.ctypeslib.as_array((C.c_uint8 * nbytes).from_address(ptr)).copy()
        assert np.array_equal(got, src.numpy())
        back = torch.zeros(nbytes, dtype=torch.uint8).pin_memory()
        abi.adpsgd_copy_d2h(back, ptr, nbytes)
        torch.cuda.synchronize()
        assert torch.equal(back, src)
    finally:
        torch.cuda.synchronize()
        assert managed.test_free_managed(ptr) == 0


def test_bad_arguments_are_refused():
    host = torch.zeros(64, dtype=torch.uint8).pin_memory()
    pageable = torch.zeros(64, dtype=torch.uint8)
    dev = torch.zeros(64, dtype=torch.uint8, device=DEV)
    cases = [
        (abi.adpsgd_copy_h2d, (dev[4:], host, 16), abi.E_ALIGN),
        (abi.adpsgd_copy_h2d, (dev, host[4:], 16), abi.E_ALIGN),
        (abi.adpsgd_copy_h2d, (host, pageable, 16), abi.E_INVAL),   # device side is host memory
        (abi.adpsgd_copy_h2d, (pageable, host, 16), abi.E_INVAL),
        (abi.adpsgd_copy_d2h, (host, host, 16), abi.E_INVAL),
        (abi.adpsgd_copy_d2h, (dev, dev, 16), abi.E_INVAL),          # host side is device memory
        (abi.adpsgd_copy_h2d, (dev, host, -1), abi.E_INVAL),
        (abi.adpsgd_copy_h2d, (None, host, 16), abi.E_INVAL),
    ]
    for fn, args, status in cases:
        with pytest.raises(abi.AdpsgdError) as e:
            fn(*args)
        assert e.value.status == status, (fn.__name__, status, e.value.status)
    abi.adpsgd_copy_h2d(None, None, 0)  # empty copy: nothing to check, nothing done
    torch.cuda.synchronize()


def test_run_fed_and_read_back_through_the_transfer_calls():
    w = inputs.WORKLOADS["quadratic-n4-P1M"]
    n, P, K = w.n, (1 << 16) + 12, 40
    h, c = inputs.problem(w, P)
    x, v = inputs.random_state(n, P, 11)
    xh, vh = torch.from_numpy(x).pin_memory(), torch.from_numpy(v).pin_memory()
    hh, ch = torch.from_numpy(h).pin_memory(), torch.from_numpy(c).pin_memory()
    xd, vd = torch.empty((n, P), device=DEV), torch.empty((n, P), device=DEV)
    hd, cd = torch.empty(P, device=DEV), torch.empty(P, device=DEV)
    for d, s in ((xd, xh), (vd, vh), (hd, hh), (cd, ch)):
        abi.adpsgd_copy_h2d(d, s)
    cfg = abi.make_config(n, P, momentum=w.mu, weight_decay=w.wd, noise_sigma=w.sigma, seed=w.seed)
    sched = abi.make_schedule(abi.ADPSGD, K, 4, K_s=10, lr0=w.lr0)
    tr = abi.TraceBuffers(K + 1)
    with abi.adpsgd_init(cfg, xd, vd, hd, cd) as ctx:
        abi.adpsgd_run(ctx, sched, abi.adpsgd_state_init(sched), trace=tr)
    xo = torch.empty((n, P), dtype=torch.float32).pin_memory()
    abi.adpsgd_copy_d2h(xo, xd)
    torch.cuda.synchronize()
    spec = O.ScheduleSpec(kind=abi.ADPSGD, K=K, p_init=4, K_s=10, lr0=w.lr0)
    otr = O.run(x, v, h, c, spec=spec, seed=w.seed, mu=w.mu, wd=w.wd, sigma=w.sigma)
    g = tr.arrays()
    assert np.array_equal(g["k"], otr.k) and np.array_equal(g["p"], otr.p)
    assert np.array_equal(xo.numpy().view(np.uint32), x.view(np.uint32))


def _w0(P, seed):
    g = torch.Generator().manual_seed(seed)
    return torch.randn(P, generator=g, dtype=torch.float32)


@pytest.mark.parametrize("where", ["pinned", "pageable", "device", "row_of_x", "inner_row_of_x"])
@pytest.mark.parametrize("n,P", [(1, 8), (3, 4099), (8, 1 << 20), (5, (1 << 18) + 4)])
def test_init_replicas(where, n, P):
    # Algorithms 1 and 2 start every replica from the same model with zero momentum: every row of
    # x equals w0 bit for bit, v is zero, and nothing outside x and v is written.
    w0 = _w0(P, n * 7 + P)
    xbuf = torch.full((n * P + 64,), 3.5, dtype=torch.float32, device=DEV)
    vbuf = torch.full((n * P + 64,), -1.25, dtype=torch.float32, device=DEV)
    xd, vd = xbuf[:n * P].view(n, P), vbuf[:n * P].view(n, P)
    z = torch.zeros(P, device=DEV)
    if where == "pinned":
        src = w0.pin_memory()
    elif where == "pageable":
        src = w0
    elif where == "device":
        src = w0.to(DEV)
    else:
        r = 0 if where == "row_of_x" else n - 1
        xd[r].copy_(w0.to(DEV))
        src = xd[r]
    with abi.adpsgd_init(abi.make_config(n, P), xd, vd, z, z) as ctx:
        abi.adpsgd_init_replicas(ctx, src)
        torch.cuda.synchronize()
    want = w0.numpy().view(np.uint32)
    got = xd.cpu().numpy().view(np.uint32)
    assert all(np.array_equal(got[i], want) for i in range(n))
    assert bool((vd == 0).all()) and not bool(torch.signbit(vd).any())
    assert bool((xbuf[n * P:] == 3.5).all()) and bool((vbuf[n * P:] == -1.25).all()), "wrote past x or v"


def test_init_replicas_refuses_null():
    n, P = 2, 64
    xd, vd, z = torch.zeros((n, P), device=DEV), torch.zeros((n, P), device=DEV), torch.zeros(P, device=DEV)
    with abi.adpsgd_init(abi.make_config(n, P), xd, vd, z, z) as ctx:
        with pytest.raises(abi.AdpsgdError) as e:
            abi.adpsgd_init_replicas(ctx, None)
        assert e.value.status == abi.E_INVAL


@pytest.mark.parametrize("kind", [abi.ADPSGD, abi.CPSGD])
def test_run_from_one_initial_model_against_the_oracle(kind):
    # The end-to-end form: one host row w0 broadcast to every replica (zero momentum), h and c
    # copied in, a whole run, and the result read back: one row when the run ends with a sync
    # (CPSGD p = 4 over 40 iterations does), every row otherwise.
    w = inputs.WORKLOADS["quadratic-n4-P1M"]
    n, P, K = w.n, (1 << 16) + 12, 40
    h, c = inputs.problem(w, P)
    w0 = _w0(P, 5)
    hh, ch = torch.from_numpy(h).pin_memory(), torch.from_numpy(c).pin_memory()
    xd, vd = torch.full((n, P), 7.0, device=DEV), torch.full((n, P), 7.0, device=DEV)
    hd, cd = torch.empty(P, device=DEV), torch.empty(P, device=DEV)
    abi.adpsgd_copy_h2d(hd, hh)
    abi.adpsgd_copy_h2d(cd, ch)
    cfg = abi.make_config(n, P, momentum=w.mu, weight_decay=w.wd, noise_sigma=w.sigma, seed=w.seed)
    K_s = 10 if kind == abi.ADPSGD else 0
    sched = abi.make_schedule(kind, K, 4, K_s=K_s, lr0=w.lr0)
    tr = abi.TraceBuffers(K + 1)
    with abi.adpsgd_init(cfg, xd, vd, hd, cd) as ctx:
        abi.adpsgd_init_replicas(ctx, w0.pin_memory())
        abi.adpsgd_run(ctx, sched, abi.adpsgd_state_init(sched), trace=tr)
    g = tr.arrays()
    one_row = g["k"][-1] == K - 1
    assert one_row or kind == abi.ADPSGD
    xo = torch.empty((1 if one_row else n, P), dtype=torch.float32).pin_memory()
    abi.adpsgd_copy_d2h(xo, xd, xo.numel() * 4)
    torch.cuda.synchronize()
    x = np.repeat(w0.numpy()[None, :], n, axis=0)
    v = np.zeros((n, P), np.float32)
    spec = O.ScheduleSpec(kind=kind, K=K, p_init=4, K_s=K_s, lr0=w.lr0)
    otr = O.run(x, v, h, c, spec=spec, seed=w.seed, mu=w.mu, wd=w.wd, sigma=w.sigma)
    assert np.array_equal(g["k"], otr.k) and np.array_equal(g["p"], otr.p)
    assert np.array_equal(xo.numpy().view(np.uint32), x[:xo.shape[0]].view(np.uint32))
    assert np.array_equal(xd.cpu().numpy().view(np.uint32), x.view(np.uint32))
    assert np.array_equal(vd.cpu().numpy().view(np.uint32), v.view(np.uint32))
