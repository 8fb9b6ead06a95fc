"""Every value the generator's Box-Muller can produce, on the GPU against the oracle.

The radius depends only on the top 23 bits of the radius word (u1 = 1 - (w >> 9) 2^-23) and the
angle only on the top 23 bits of the angle word, so two sweeps of 2^23 word pairs cover every
radius (with the angle fixed) and every (sin, cos) pair (with the radius fixed).  The library's
device code (noise.cuh, built into a probe with the library's arithmetic flags) must give the
oracle's z0 and z1 bit for bit on all of them."""
import ctypes as C
import os
import subprocess

import numpy as np
import pytest

from oracle import oracle as O
from paper_2007_06134_gb300 import build as B

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
HERE = os.path.dirname(os.path.abspath(__file__))


@pytest.fixture(scope="module")
def probe(tmp_path_factory):
    so = str(tmp_path_factory.mktemp("probe") / "libbox_muller_probe.so")
    flags = [f for f in B.NVCC_FLAGS if f not in ("-Xptxas", "-v")]
    subprocess.check_call(["nvcc", *B.ARCH, *flags, "-shared", "-I", B.CSRC, "-I", B.INCLUDE,
                           "-o", so, os.path.join(HERE, "cuda", "box_muller_probe.cu")])
    lib = C.CDLL(so)
    lib.box_muller_probe.argtypes = [C.c_void_p] * 2 + [C.c_int64] + [C.c_void_p] * 2
    lib.box_muller_probe.restype = C.c_int
    return lib


def _device_box_muller(lib, wr, wa):
    d = lambda a: torch.from_numpy(np.ascontiguousarray(a).view(np.int32)).to("cuda:0")
    dwr, dwa = d(wr), d(wa)
    z0 = torch.empty(wr.size, dtype=torch.float32, device="cuda:0")
    z1 = torch.empty_like(z0)
    assert lib.box_muller_probe(dwr.data_ptr(), dwa.data_ptr(), wr.size, z0.data_ptr(), z1.data_ptr()) == 0
    return z0.cpu().numpy(), z1.cpu().numpy()


@pytest.mark.parametrize("sweep", ["radius", "angle"])
def test_every_radius_and_every_angle(probe, sweep):
    k = np.arange(1 << 23, dtype=np.uint32) << np.uint32(9)
    rng = np.random.default_rng(7)
    low = rng.integers(0, 1 << 9, size=k.size, dtype=np.uint32)  # the ignored low bits
    fixed = np.full(k.size, 0x5A5A5A5A, dtype=np.uint32)
    wr, wa = (k | low, fixed) if sweep == "radius" else (fixed, k | low)
    g0, g1 = _device_box_muller(probe, wr, wa)
    o0, o1 = O.box_muller_array(wr, wa)
    assert np.array_equal(g0.view(np.uint32), o0.view(np.uint32))
    assert np.array_equal(g1.view(np.uint32), o1.view(np.uint32))
