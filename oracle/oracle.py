"""Python access to the plain CPU oracle in ``adpsgd_oracle.c``.

TEST INFRASTRUCTURE ONLY: the tests, ``__graft_entry__.smoke()`` and the CPU
baseline leg of ``bench.py`` may use this module; the product path never does.
It shares no code with the CUDA library: it compiles its own C file with gcc
(``-O2 -ffp-contract=off``, no fast-math, so every fp32 operation is one IEEE
rounding; ``-fopenmp`` for the chunked all-core run) and marshals numpy arrays
through ctypes.

Every function cites the part of the paper it follows (Jiang & Agrawal,
"Adaptive Periodic Averaging", arXiv 2007.06134); the C file states the
readings taken where the paper is silent.
"""
from __future__ import annotations

import ctypes as C
import os
import subprocess
import threading
from dataclasses import dataclass, field

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "adpsgd_oracle.c")
_LIB = os.path.join(_HERE, "liboracle_adpsgd.so")
_lock = threading.Lock()
_lib = None

CFLAGS = ["-O2", "-std=c11", "-fPIC", "-shared", "-fopenmp", "-ffp-contract=off", "-fno-fast-math",
          "-fno-unsafe-math-optimizations"]
CHUNK_COLUMNS = 1 << 16  # columns per chunk of the all-core run


def build(force: bool = False) -> str:
    """Compile the oracle library with gcc if it is missing or stale."""
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", *CFLAGS, "-o", tmp, _SRC, "-lm"])
        os.replace(tmp, _LIB)
    return _LIB


def _f32p(a):
    return a.ctypes.data_as(C.POINTER(C.c_float))


def _u32p(a):
    return a.ctypes.data_as(C.POINTER(C.c_uint32))


def _u16p(a):
    return a.ctypes.data_as(C.POINTER(C.c_uint16))


def _f64p(a):
    return a.ctypes.data_as(C.POINTER(C.c_double))


def _i64p(a):
    return a.ctypes.data_as(C.POINTER(C.c_int64))


def _i32p(a):
    return a.ctypes.data_as(C.POINTER(C.c_int32))


class Schedule(C.Structure):
    """Mirror of the oracle's ``orc_schedule`` (Algorithm 1 / Algorithm 2 knobs)."""
    _fields_ = [
        ("kind", C.c_int32), ("p_init", C.c_int32), ("K", C.c_int64), ("K_s", C.c_int64),
        ("K_w", C.c_int64), ("lo", C.c_double), ("hi", C.c_double), ("p_min", C.c_int32),
        ("p_max", C.c_int32), ("lr0", C.c_double), ("lr_factor", C.c_double),
        ("n_milestones", C.c_int32), ("literal_phase", C.c_int32),
        ("milestones", C.POINTER(C.c_int64)), ("n_period_changes", C.c_int32), ("pad", C.c_int32),
        ("period_change_k", C.POINTER(C.c_int64)), ("period_values", C.POINTER(C.c_int32)),
        ("lr_warmup_steps", C.c_int32), ("pad2", C.c_int32), ("lr_warmup_len", C.c_int64),
    ]


class State(C.Structure):
    _fields_ = [("cnt", C.c_int32), ("p", C.c_int32), ("C2", C.c_double), ("m", C.c_int64)]


class Trace(C.Structure):
    _fields_ = [
        ("k", C.POINTER(C.c_int64)), ("p", C.POINTER(C.c_int32)), ("S", C.POINTER(C.c_double)),
        ("C2", C.POINTER(C.c_double)), ("loss", C.POINTER(C.c_double)),
        ("phase", C.POINTER(C.c_int32)), ("cap", C.c_int64), ("var", C.POINTER(C.c_double)),
        ("var_cap", C.c_int64),
    ]


PHASE_CONSTANT, PHASE_WARMUP, PHASE_SAMPLING, PHASE_ADAPTING = 0, 1, 2, 3


def lib():
    global _lib
    with _lock:
        if _lib is None:
            build()
            L = C.CDLL(_LIB)
            L.orc_philox4x32_10.argtypes = [C.POINTER(C.c_uint32)] * 3
            L.orc_philox_words.argtypes = [C.c_uint64, C.c_uint32, C.c_uint32, C.c_uint32,
                                           C.c_int64, C.c_int64, C.POINTER(C.c_uint32)]
            L.orc_ln.argtypes = [C.c_float]
            L.orc_ln.restype = C.c_float
            L.orc_ln_array.argtypes = [C.POINTER(C.c_float), C.POINTER(C.c_float), C.c_int64]
            L.orc_sincos_array.argtypes = [C.POINTER(C.c_float)] * 3 + [C.c_int64]
            L.orc_normals.argtypes = [C.c_uint64, C.c_uint32, C.c_uint32, C.c_uint32, C.c_int64,
                                      C.c_int64, C.POINTER(C.c_float)]
            L.orc_box_muller_words.argtypes = [C.c_uint32, C.c_uint32, C.POINTER(C.c_float),
                                               C.POINTER(C.c_float)]
            L.orc_box_muller_array.argtypes = [C.POINTER(C.c_uint32), C.POINTER(C.c_uint32), C.c_int64,
                                               C.POINTER(C.c_float), C.POINTER(C.c_float)]
            L.orc_to_bf16_array.argtypes = [C.POINTER(C.c_float), C.POINTER(C.c_uint16), C.c_int64]
            L.orc_noise_bf16.argtypes = [C.c_uint64, C.c_int32, C.c_int64, C.POINTER(C.c_uint16)]
            L.orc_local_step.argtypes = [C.c_int32, C.c_int64, C.c_int64, C.c_int64,
                                         C.POINTER(C.c_float), C.POINTER(C.c_float),
                                         C.POINTER(C.c_float), C.POINTER(C.c_float),
                                         C.POINTER(C.c_uint16), C.c_uint64, C.c_int64,
                                         C.c_float, C.c_float, C.c_float, C.c_float]
            L.orc_average_variance.argtypes = [C.c_int32, C.c_int64, C.c_int64, C.c_int64,
                                               C.POINTER(C.c_float), C.POINTER(C.c_float),
                                               C.POINTER(C.c_float), C.POINTER(C.c_double),
                                               C.POINTER(C.c_double)]
            L.orc_variance.argtypes = [C.c_int32, C.c_int64, C.POINTER(C.c_float)]
            L.orc_variance.restype = C.c_double
            L.orc_gamma.argtypes = [C.POINTER(Schedule), C.c_int64]
            L.orc_gamma.restype = C.c_float
            L.orc_on_sync.argtypes = [C.POINTER(Schedule), C.POINTER(State), C.c_int64,
                                      C.c_double, C.c_double]
            L.orc_on_sync.restype = C.c_int32
            L.orc_state_init.argtypes = [C.POINTER(Schedule), C.POINTER(State)]
            L.orc_run.argtypes = [C.c_int32, C.c_int64, C.POINTER(C.c_float), C.POINTER(C.c_float),
                                  C.POINTER(C.c_float), C.POINTER(C.c_float), C.POINTER(C.c_uint16),
                                  C.c_uint64, C.c_float, C.c_float, C.c_float,
                                  C.POINTER(Schedule), C.POINTER(State), C.c_int64, C.c_int64,
                                  C.POINTER(Trace)]
            L.orc_run.restype = C.c_int64
            L.orc_run_chunked.argtypes = [C.c_int32, C.c_int64] + L.orc_run.argtypes
            L.orc_run_chunked.restype = C.c_int64
            L.orc_schedule_only.argtypes = [C.POINTER(Schedule), C.POINTER(C.c_double), C.c_int64,
                                            C.POINTER(C.c_int64), C.POINTER(C.c_int32), C.c_int64]
            L.orc_schedule_only.restype = C.c_int64
            L.orc_wire_bytes.argtypes = [C.c_int32, C.c_int64, C.c_int64, C.c_int32,
                                         C.POINTER(C.c_double), C.POINTER(C.c_double)]
            _lib = L
    return _lib


# --------------------------------------------------------------------------
# Generator pieces (Philox4x32-10, Salmon et al. SC'11; Box-Muller 1958).
# --------------------------------------------------------------------------

def philox4x32_10(ctr, key) -> np.ndarray:
    """One Philox4x32-10 block: four 32-bit counter words, two key words."""
    c = np.ascontiguousarray(ctr, dtype=np.uint32)
    k = np.ascontiguousarray(key, dtype=np.uint32)
    out = np.zeros(4, dtype=np.uint32)
    lib().orc_philox4x32_10(_u32p(c), _u32p(k), _u32p(out))
    return out


def philox_words(seed: int, tag: int, i: int, k: int, q0: int, nq: int) -> np.ndarray:
    """Words of the noise stream for blocks q0..q0+nq-1 of replica i, step k: [nq, 4]."""
    out = np.zeros((nq, 4), dtype=np.uint32)
    lib().orc_philox_words(seed, tag, i, k, q0, nq, _u32p(out))
    return out


def ln(u) -> np.ndarray:
    """The oracle's own natural log on fp32 values (Cody-Waite + atanh series)."""
    u = np.ascontiguousarray(u, dtype=np.float32)
    out = np.empty_like(u)
    lib().orc_ln_array(_f32p(u), _f32p(out), u.size)
    return out


def sincos_turn(u):
    """(sin 2*pi*u, cos 2*pi*u) on fp32 u in [0, 1) (quarter-turn reduction + Taylor)."""
    u = np.ascontiguousarray(u, dtype=np.float32)
    s = np.empty_like(u)
    c = np.empty_like(u)
    lib().orc_sincos_array(_f32p(u), _f32p(s), _f32p(c), u.size)
    return s, c


def normals(seed: int, tag: int, i: int, k: int, j0: int, m: int) -> np.ndarray:
    """Gaussian noise z[i, j0:j0+m] at step k (the surrogate's mini-batch noise, Eq. eg)."""
    out = np.empty(m, dtype=np.float32)
    lib().orc_normals(seed, tag, i, k, j0, m, _f32p(out))
    return out


def box_muller_words(w_radius: int, w_angle: int):
    """(z0, z1) = radius * (cos, sin) of the angle, from two raw 32-bit words."""
    z0 = C.c_float()
    z1 = C.c_float()
    lib().orc_box_muller_words(w_radius, w_angle, C.byref(z0), C.byref(z1))
    return z0.value, z1.value


def box_muller_array(w_radius, w_angle):
    """(z0, z1) arrays of Box-Muller on word pairs: radius sqrt(-2 ln u1), angle 2 pi u2."""
    wr = np.ascontiguousarray(w_radius, dtype=np.uint32)
    wa = np.ascontiguousarray(w_angle, dtype=np.uint32)
    z0 = np.empty(wr.size, np.float32)
    z1 = np.empty(wr.size, np.float32)
    lib().orc_box_muller_array(_u32p(wr), _u32p(wa), wr.size, _f32p(z0), _f32p(z1))
    return z0, z1


def to_bf16(x) -> np.ndarray:
    """The oracle's fp32 -> bf16 rounding (raw bits as uint16)."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    out = np.empty(x.shape, dtype=np.uint16)
    lib().orc_to_bf16_array(_f32p(x), _u16p(out), x.size)
    return out


def noise_bf16(seed: int, n: int, P: int) -> np.ndarray:
    """The pre-materialised bf16 noise tensor [n, P] (raw bf16 bits as uint16)."""
    out = np.empty((n, P), dtype=np.uint16)
    lib().orc_noise_bf16(seed, n, P, _u16p(out))
    return out


# --------------------------------------------------------------------------
# Hot-path pieces (Algorithm 2).
# --------------------------------------------------------------------------

def _check_state(x, v=None):
    assert x.dtype == np.float32 and x.flags.c_contiguous and x.ndim == 2
    if v is not None:
        assert v.dtype == np.float32 and v.flags.c_contiguous and v.shape == x.shape


def local_step(x, v, h, c, *, seed, k, gamma, mu, wd, sigma, noise=None, j0=0, j1=None):
    """In-place local step of every replica on columns [j0, j1) (Algorithm 2, update line)."""
    _check_state(x, v)
    n, P = x.shape
    j1 = P if j1 is None else j1
    h = np.ascontiguousarray(h, dtype=np.float32)
    c = np.ascontiguousarray(c, dtype=np.float32)
    nz = None if noise is None else _u16p(np.ascontiguousarray(noise, dtype=np.uint16))
    lib().orc_local_step(n, P, j0, j1, _f32p(x), _f32p(v), _f32p(h), _f32p(c), nz, seed, k,
                         gamma, mu, wd, sigma)


def average_variance(x, h=None, c=None, j0=0, j1=None):
    """In-place averaging of columns [j0, j1); returns (D, loss) in fp64 (Algorithm 2, sync)."""
    _check_state(x)
    n, P = x.shape
    j1 = P if j1 is None else j1
    D = C.c_double(0.0)
    L = C.c_double(0.0)
    if h is None:
        lib().orc_average_variance(n, P, j0, j1, _f32p(x), None, None, C.byref(D), None)
        return D.value, None
    h = np.ascontiguousarray(h, dtype=np.float32)
    c = np.ascontiguousarray(c, dtype=np.float32)
    lib().orc_average_variance(n, P, j0, j1, _f32p(x), _f32p(h), _f32p(c), C.byref(D), C.byref(L))
    return D.value, L.value


def variance(x) -> float:
    """D = sum_i ||x_i - xbar||^2 without averaging (Sec. II-B, Var[W_k] times n)."""
    _check_state(x)
    return lib().orc_variance(x.shape[0], x.shape[1], _f32p(x))


@dataclass
class ScheduleSpec:
    """Algorithm 1 (kind=0, constant p), Algorithm 2 (kind=1) with its knobs, or a piecewise-constant
    period (kind=2: p_init, then period_values[t] from iteration period_change_k[t] on)."""
    kind: int
    K: int
    p_init: int
    K_s: int = 0
    K_w: int = 0
    lo: float = 0.7
    hi: float = 1.3
    p_min: int = 1
    p_max: int = 0
    lr0: float = 0.1
    lr_factor: float = 0.1
    milestones: tuple = ()
    literal_phase: int = 0
    period_changes: tuple = ()   # ((k, p), ...) for kind 2
    lr_warmup_steps: int = 0     # step-size warm-up stairs (Sec. IV-C), each lr_warmup_len iterations
    lr_warmup_len: int = 1
    _ms: np.ndarray = field(default=None, repr=False)
    _pk: np.ndarray = field(default=None, repr=False)
    _pv: np.ndarray = field(default=None, repr=False)

    def c(self) -> Schedule:
        self._ms = np.ascontiguousarray(self.milestones if self.milestones else [0], dtype=np.int64)
        ch = self.period_changes if self.period_changes else ((0, self.p_init),)
        self._pk = np.ascontiguousarray([k for k, _ in ch], dtype=np.int64)
        self._pv = np.ascontiguousarray([p for _, p in ch], dtype=np.int32)
        return Schedule(self.kind, self.p_init, self.K, self.K_s, self.K_w, self.lo, self.hi,
                        self.p_min, self.p_max, self.lr0, self.lr_factor, len(self.milestones),
                        self.literal_phase, _i64p(self._ms), len(self.period_changes), 0,
                        _i64p(self._pk), _i32p(self._pv), self.lr_warmup_steps, 0, self.lr_warmup_len)


def gamma(spec: ScheduleSpec, k: int) -> float:
    s = spec.c()
    return lib().orc_gamma(C.byref(s), k)


def new_state(spec: ScheduleSpec) -> State:
    st = State()
    s = spec.c()
    lib().orc_state_init(C.byref(s), C.byref(st))
    return st


def on_sync(spec: ScheduleSpec, st: State, k: int, S: float, g: float) -> int:
    s = spec.c()
    return lib().orc_on_sync(C.byref(s), C.byref(st), k, S, g)


@dataclass
class RunTrace:
    k: np.ndarray
    p: np.ndarray
    S: np.ndarray
    C2: np.ndarray
    loss: np.ndarray
    phase: np.ndarray
    syncs: int
    var: np.ndarray = None


def host_threads() -> int:
    """Host cores this process may run on."""
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:  # pragma: no cover - Linux has sched_getaffinity
        return os.cpu_count() or 1


def run(x, v, h, c, *, spec: ScheduleSpec, seed, mu, wd, sigma, noise=None, state=None,
        k_begin=0, k_end=None, cap=100000, track_variance=False, threads=None,
        chunk=CHUNK_COLUMNS) -> RunTrace:
    """Algorithm 2 (or 1) end to end on the [n, P] arrays, in place; returns the sync trace and,
    with track_variance, Var[W_k] at the start of every iteration k (Sec. II-B, Eq. vt).
    threads=None runs on one thread in column order; threads=t (e.g. host_threads()) runs the
    chunked all-core form: the same x, v and schedule, D and the loss summed per chunk of `chunk`
    columns in chunk order."""
    _check_state(x, v)
    n, P = x.shape
    k_end = spec.K if k_end is None else k_end
    st = new_state(spec) if state is None else state
    arrs = dict(k=np.zeros(cap, np.int64), p=np.zeros(cap, np.int32), S=np.zeros(cap),
                C2=np.zeros(cap), loss=np.zeros(cap), phase=np.zeros(cap, np.int32))
    var = np.full(k_end, np.nan) if track_variance else None
    tr = Trace(_i64p(arrs["k"]), _i32p(arrs["p"]), _f64p(arrs["S"]), _f64p(arrs["C2"]),
               _f64p(arrs["loss"]), _i32p(arrs["phase"]), cap,
               _f64p(var) if var is not None else None, k_end if var is not None else 0)
    s = spec.c()
    h = np.ascontiguousarray(h, dtype=np.float32)
    c = np.ascontiguousarray(c, dtype=np.float32)
    nz = None if noise is None else _u16p(np.ascontiguousarray(noise, dtype=np.uint16))
    args = (n, P, _f32p(x), _f32p(v), _f32p(h), _f32p(c), nz, seed, mu, wd, sigma,
            C.byref(s), C.byref(st), k_begin, k_end, C.byref(tr))
    if threads is None:
        syncs = lib().orc_run(*args)
    else:
        syncs = lib().orc_run_chunked(threads, chunk, *args)
        if syncs < 0:
            raise ValueError(f"chunked run refused: chunk {chunk} must be a positive multiple of 4")
    m = min(syncs, cap)
    return RunTrace(**{a: b[:m].copy() for a, b in arrs.items()}, syncs=syncs, var=var)


def schedule_only(spec: ScheduleSpec, S_script, cap=100000):
    """Sync iterations and periods of a schedule when sync t reports S_script[t]."""
    S = np.ascontiguousarray(S_script, dtype=np.float64)
    ks = np.zeros(cap, np.int64)
    ps = np.zeros(cap, np.int32)
    s = spec.c()
    syncs = lib().orc_schedule_only(C.byref(s), _f64p(S) if S.size else None, S.size,
                                    _i64p(ks), _i32p(ps), cap)
    m = min(syncs, cap)
    return syncs, ks[:m].copy(), ps[:m].copy()


def wire_bytes(n: int, P: int, rounds: int, with_scalar: bool = True):
    """(per-node, total) ring-allreduce bytes for `rounds` syncs of P fp32 (+ the S_k scalar)."""
    pn = C.c_double()
    tot = C.c_double()
    lib().orc_wire_bytes(n, P, rounds, int(with_scalar), C.byref(pn), C.byref(tot))
    return pn.value, tot.value
