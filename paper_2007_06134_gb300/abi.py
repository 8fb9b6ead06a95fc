"""ctypes binding of ``libadpsgd.so`` (include/adpsgd.h), one Python function per C entry point.

Argument marshalling only: tensors become device pointers (``data_ptr()``), the stream
becomes its ``cudaStream_t`` handle, and a nonzero status becomes an ``AdpsgdError``.
Every step of the hot path runs in the library's CUDA kernels; if the library cannot be
built or loaded this module raises, it never falls back to another implementation.
"""
from __future__ import annotations

import ctypes as C
import os
import re
import threading

from . import build as _build

_lock = threading.Lock()
_lib = None

OK, E_INVAL, E_ALIGN, E_CUDA, E_TIMEOUT, E_NOMEM, E_STATE, E_PEER = 0, -1, -2, -3, -4, -5, -6, -7
NOISE_PHILOX, NOISE_BF16 = 0, 1
CPSGD, ADPSGD, PIECEWISE = 0, 1, 2
PHASE_CONSTANT, PHASE_WARMUP, PHASE_SAMPLING, PHASE_ADAPTING = 0, 1, 2, 3


class AdpsgdError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        detail = last_error() if status in (E_CUDA, E_TIMEOUT, E_PEER) else ""
        super().__init__(f"{where}: {strerror(status)} ({status}){': ' + detail if detail else ''}")


class Config(C.Structure):
    _fields_ = [("n", C.c_int32), ("noise_mode", C.c_int32), ("P", C.c_int64), ("momentum", C.c_float),
                ("weight_decay", C.c_float), ("noise_sigma", C.c_float), ("want_loss", C.c_int32),
                ("seed", C.c_uint64), ("wait_timeout_ms", C.c_int64), ("time_kernels", C.c_int32),
                ("fuse_intervals", C.c_int32), ("fuse_sync_step", C.c_int32)]


class Schedule(C.Structure):
    _fields_ = [("kind", C.c_int32), ("p_init", C.c_int32), ("K", C.c_int64), ("K_s", C.c_int64),
                ("K_w", C.c_int64), ("lo", C.c_double), ("hi", C.c_double), ("p_min", C.c_int32),
                ("p_max", C.c_int32), ("lr0", C.c_double), ("lr_factor", C.c_double),
                ("n_milestones", C.c_int32), ("literal_phase", C.c_int32),
                ("milestones", C.POINTER(C.c_int64)), ("n_period_changes", C.c_int32), ("reserved", C.c_int32),
                ("period_change_k", C.POINTER(C.c_int64)), ("period_values", C.POINTER(C.c_int32)),
                ("lr_warmup_steps", C.c_int32), ("reserved2", C.c_int32), ("lr_warmup_len", C.c_int64)]


class State(C.Structure):
    _fields_ = [("k_next", C.c_int64), ("cnt", C.c_int32), ("p", C.c_int32), ("C2", C.c_double),
                ("m", C.c_int64), ("rounds", C.c_int64)]


class Trace(C.Structure):
    _fields_ = [("cap", C.c_int64), ("len", C.c_int64), ("k", C.POINTER(C.c_int64)),
                ("p", C.POINTER(C.c_int32)), ("S", C.POINTER(C.c_double)), ("C2", C.POINTER(C.c_double)),
                ("loss", C.POINTER(C.c_double)), ("phase", C.POINTER(C.c_int32)), ("var_cap", C.c_int64),
                ("var", C.POINTER(C.c_double))]


class Stats(C.Structure):
    _fields_ = [("rounds", C.c_int64), ("equiv_period", C.c_double), ("wire_bytes_per_node", C.c_double),
                ("wire_bytes_total", C.c_double), ("fullsgd_wire_bytes_per_node", C.c_double),
                ("local_step_launches", C.c_int64), ("average_launches", C.c_int64),
                ("interval_launches", C.c_int64), ("sync_step_launches", C.c_int64)]


class KernelTiming(C.Structure):
    _fields_ = [("local_step_ms", C.c_double), ("local_step_launches", C.c_int64), ("average_ms", C.c_double),
                ("average_launches", C.c_int64), ("interval_ms", C.c_double), ("interval_launches", C.c_int64),
                ("sync_step_ms", C.c_double), ("sync_step_launches", C.c_int64)]


# int gather(const double* local, int64_t count, double* gathered, void* user)
GATHER_FN = C.CFUNCTYPE(C.c_int, C.POINTER(C.c_double), C.c_int64, C.POINTER(C.c_double), C.c_void_p)


SCATTER_COLUMNS, GATHER_AVERAGE = 0, 1
# int collective(int32_t op, void* user)
COLLECTIVE_FN = C.CFUNCTYPE(C.c_int, C.c_int32, C.c_void_p)


class ReplicaSplit(C.Structure):
    _fields_ = [("processes", C.c_int32), ("rank", C.c_int32), ("replica0", C.c_int32), ("n_total", C.c_int32),
                ("col0", C.c_int64), ("P_chunk", C.c_int64), ("chunk_x", C.c_void_p),
                ("collective", COLLECTIVE_FN), ("gather", GATHER_FN), ("user", C.c_void_p)]


class Shard(C.Structure):
    _fields_ = [("shards", C.c_int32), ("index", C.c_int32), ("col0", C.c_int64), ("P_total", C.c_int64),
                ("gather", GATHER_FN), ("user", C.c_void_p)]


_P = C.c_void_p
_SIGS = {
    "adpsgd_init": (C.c_int, [C.POINTER(Config), _P, _P, _P, _P, _P, _P, C.POINTER(_P)]),
    "adpsgd_local_steps": (C.c_int, [_P, C.c_int64, C.c_int32, C.POINTER(C.c_float)]),
    "adpsgd_average_and_variance": (C.c_int, [_P, C.POINTER(C.c_double), C.POINTER(C.c_double)]),
    "adpsgd_variance": (C.c_int, [_P, C.POINTER(C.c_double)]),
    "adpsgd_average_and_variance_static": (C.c_int, [_P, _P, _P, C.c_int32, C.c_int64, C.POINTER(C.c_double),
                                                     C.POINTER(C.c_double), C.c_int64, _P]),
    "adpsgd_state_init": (C.c_int, [C.POINTER(Schedule), C.POINTER(State)]),
    "adpsgd_run": (C.c_int, [_P, C.POINTER(Schedule), C.POINTER(State), C.c_int64, C.POINTER(Trace),
                             C.POINTER(Stats)]),
    "adpsgd_sched_on_sync": (C.c_int, [C.POINTER(Schedule), C.POINTER(State), C.c_int64, C.c_double,
                                       C.c_double, C.POINTER(C.c_int32)]),
    "adpsgd_gamma": (C.c_int, [C.POINTER(Schedule), C.c_int64, C.POINTER(C.c_float)]),
    "adpsgd_wire_bytes": (C.c_int, [C.c_int32, C.c_int64, C.c_int64, C.c_int32, C.POINTER(C.c_double),
                                    C.POINTER(C.c_double)]),
    "adpsgd_philox_fill": (C.c_int, [C.c_uint64, C.c_uint32, C.c_int32, C.c_int64, C.c_int64, _P, _P]),
    "adpsgd_noise_fill_f32": (C.c_int, [C.c_uint64, C.c_uint32, C.c_int32, C.c_int64, C.c_int64, _P, _P]),
    "adpsgd_noise_fill_bf16": (C.c_int, [C.c_uint64, C.c_int32, C.c_int64, _P, _P]),
    "adpsgd_set_shard": (C.c_int, [_P, C.POINTER(Shard)]),
    "adpsgd_set_replica_split": (C.c_int, [_P, C.POINTER(ReplicaSplit)]),
    "adpsgd_shard_combine": (C.c_int, [C.POINTER(Shard), C.POINTER(C.c_double), C.c_int64, C.POINTER(C.c_double)]),
    "adpsgd_noise_fill_bf16_part": (C.c_int, [C.c_uint64, C.c_int32, C.c_int64, C.c_int32, C.c_int64, _P, _P]),
    "adpsgd_copy_h2d": (C.c_int, [_P, _P, C.c_int64, _P]),
    "adpsgd_init_replicas": (C.c_int, [_P, _P]),
    "adpsgd_copy_d2h": (C.c_int, [_P, _P, C.c_int64, _P]),
    "adpsgd_kernel_times": (C.c_int, [_P, C.POINTER(KernelTiming)]),
    "adpsgd_reset_kernel_times": (C.c_int, [_P]),
    "adpsgd_test_force_incomplete": (C.c_int, [_P, C.c_int32]),
    "adpsgd_destroy": (None, [_P]),
    "adpsgd_strerror": (C.c_char_p, [C.c_int]),
    "adpsgd_last_error": (C.c_char_p, []),
}


def library_path() -> str:
    return _build.LIB


def load(build_if_stale: bool = True):
    """Load (building first if needed) the CUDA library; raise if that is impossible."""
    global _lib
    with _lock:
        if _lib is None:
            if build_if_stale:
                _build.build()
            if not os.path.exists(_build.LIB):
                raise RuntimeError(f"CUDA library missing: {_build.LIB} (build with paper_2007_06134_gb300.build)")
            L = C.CDLL(_build.LIB)
            for name, (res, args) in _SIGS.items():
                f = getattr(L, name)
                f.restype = res
                f.argtypes = args
            _lib = L
    return _lib


def header_entry_points() -> list[str]:
    """Names of the functions include/adpsgd.h declares."""
    hdr = os.path.join(_build.INCLUDE, "adpsgd.h")
    text = open(hdr).read()
    return sorted(set(re.findall(r"^\s*(?:int|void|const char\*)\s+(adpsgd_\w+)\s*\(", text, re.M)))


def strerror(status: int) -> str:
    return load().adpsgd_strerror(status).decode()


def last_error() -> str:
    return load().adpsgd_last_error().decode()


def _check(status: int, where: str):
    if status != OK:
        raise AdpsgdError(status, where)


def _ptr(t) -> int | None:
    if t is None:
        return None
    if isinstance(t, int):
        return t
    return t.data_ptr()


def _stream(stream) -> int | None:
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def make_config(n, P, *, momentum=0.9, weight_decay=0.0, noise_sigma=1.0, seed=0, noise_mode=NOISE_PHILOX,
                want_loss=True, wait_timeout_ms=60000, time_kernels=False, fuse_intervals=False,
                fuse_sync_step=False) -> Config:
    return Config(n, noise_mode, P, momentum, weight_decay, noise_sigma, int(bool(want_loss)),
                  seed & 0xFFFFFFFFFFFFFFFF, wait_timeout_ms, int(time_kernels), int(bool(fuse_intervals)),
                  int(bool(fuse_sync_step)))


def make_schedule(kind, K, p_init, *, K_s=0, K_w=0, lo=0.7, hi=1.3, p_min=1, p_max=0, lr0=0.1, lr_factor=0.1,
                  milestones=(), literal_phase=False, period_changes=(), lr_warmup_steps=0,
                  lr_warmup_len=1) -> Schedule:
    """period_changes: ((k, p), ...) for PIECEWISE: p from iteration k on.  lr_warmup_steps > 0: the
    step size climbs lr0, 2 lr0, ... over that many stairs of lr_warmup_len iterations (Sec. IV-C)."""
    ms = (C.c_int64 * max(1, len(milestones)))(*milestones)
    pk = (C.c_int64 * max(1, len(period_changes)))(*[k for k, _ in period_changes])
    pv = (C.c_int32 * max(1, len(period_changes)))(*[p for _, p in period_changes])
    s = Schedule(kind, p_init, K, K_s, K_w, lo, hi, p_min, p_max, lr0, lr_factor, len(milestones),
                 int(bool(literal_phase)), C.cast(ms, C.POINTER(C.c_int64)), len(period_changes), 0,
                 C.cast(pk, C.POINTER(C.c_int64)), C.cast(pv, C.POINTER(C.c_int32)), lr_warmup_steps, 0,
                 lr_warmup_len)
    s._keep = (ms, pk, pv)  # keep the host arrays alive with the struct
    return s


class Context:
    """An ``adpsgd_ctx*`` over caller-owned device tensors; ``close()`` calls adpsgd_destroy."""

    def __init__(self, handle: int, keep: tuple):
        self.handle = handle
        self._keep = keep  # tensors the context borrows

    def close(self):
        if self.handle:
            load().adpsgd_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()


def adpsgd_init(cfg: Config, x, v, h, c, noise_bf16=None, stream=None) -> Context:
    out = C.c_void_p()
    _check(load().adpsgd_init(C.byref(cfg), _ptr(x), _ptr(v), _ptr(h), _ptr(c), _ptr(noise_bf16),
                              _stream(stream), C.byref(out)), "adpsgd_init")
    return Context(out.value, (x, v, h, c, noise_bf16))


def make_shard(shards: int, index: int, col0: int, P_total: int, gather=None) -> Shard:
    """gather: a GATHER_FN (or None with one shard); the struct keeps a reference to it."""
    sh = Shard(shards, index, col0, P_total, gather if gather is not None else GATHER_FN(), None)
    sh._keep = gather
    return sh


def adpsgd_set_shard(ctx: Context, shard: Shard) -> None:
    _check(load().adpsgd_set_shard(ctx.handle, C.byref(shard)), "adpsgd_set_shard")
    ctx._shard = shard  # the context calls shard.gather until it is destroyed


def make_replica_split(processes: int, rank: int, replica0: int, n_total: int, col0: int, P_chunk: int, chunk_x,
                       collective, gather=None) -> ReplicaSplit:
    """collective: a COLLECTIVE_FN; gather: a GATHER_FN (None with one process)."""
    rs = ReplicaSplit(processes, rank, replica0, n_total, col0, P_chunk, _ptr(chunk_x), collective,
                      gather if gather is not None else GATHER_FN(), None)
    rs._keep = (chunk_x, collective, gather)
    return rs


def adpsgd_set_replica_split(ctx: Context, split: ReplicaSplit) -> None:
    _check(load().adpsgd_set_replica_split(ctx.handle, C.byref(split)), "adpsgd_set_replica_split")
    ctx._split = split  # the context calls split.collective and split.gather until it is destroyed


def adpsgd_shard_combine(shard: Shard, local):
    """Every shard's values through shard.gather, summed in shard order (pure host code)."""
    import numpy as np
    loc = np.ascontiguousarray(local, dtype=np.float64)
    out = np.zeros_like(loc)
    _check(load().adpsgd_shard_combine(C.byref(shard), loc.ctypes.data_as(C.POINTER(C.c_double)), loc.size,
                                       out.ctypes.data_as(C.POINTER(C.c_double))), "adpsgd_shard_combine")
    return out


def adpsgd_local_steps(ctx: Context, k0: int, lr) -> None:
    lr = list(lr)
    arr = (C.c_float * max(1, len(lr)))(*lr)
    _check(load().adpsgd_local_steps(ctx.handle, k0, len(lr), arr), "adpsgd_local_steps")


def adpsgd_average_and_variance(ctx: Context, want_loss: bool = True):
    D = C.c_double()
    L = C.c_double()
    _check(load().adpsgd_average_and_variance(ctx.handle, C.byref(D), C.byref(L) if want_loss else None),
           "adpsgd_average_and_variance")
    return D.value, (L.value if want_loss else None)


def adpsgd_average_and_variance_static(x, h, c, n: int, P: int, want_loss: bool = True,
                                       wait_timeout_ms: int = 60000, stream=None):
    """Averaging without a context or any allocation (fixed scratch inside the library)."""
    D = C.c_double()
    L = C.c_double()
    _check(load().adpsgd_average_and_variance_static(_ptr(x), _ptr(h), _ptr(c), n, P, C.byref(D),
                                                     C.byref(L) if want_loss else None, wait_timeout_ms,
                                                     _stream(stream)),
           "adpsgd_average_and_variance_static")
    return D.value, (L.value if want_loss else None)


def adpsgd_variance(ctx: Context) -> float:
    D = C.c_double()
    _check(load().adpsgd_variance(ctx.handle, C.byref(D)), "adpsgd_variance")
    return D.value


def adpsgd_state_init(sched: Schedule) -> State:
    st = State()
    _check(load().adpsgd_state_init(C.byref(sched), C.byref(st)), "adpsgd_state_init")
    return st


class TraceBuffers:
    """Host arrays for an adpsgd_trace; var_cap > 0 also records Var[W_k] per iteration."""

    def __init__(self, cap: int, var_cap: int = 0):
        import numpy as np
        self.k = np.zeros(cap, np.int64)
        self.p = np.zeros(cap, np.int32)
        self.S = np.zeros(cap)
        self.C2 = np.zeros(cap)
        self.loss = np.zeros(cap)
        self.phase = np.zeros(cap, np.int32)
        self.var = np.full(max(1, var_cap), np.nan)
        self.c = Trace(cap, 0, self.k.ctypes.data_as(C.POINTER(C.c_int64)),
                       self.p.ctypes.data_as(C.POINTER(C.c_int32)), self.S.ctypes.data_as(C.POINTER(C.c_double)),
                       self.C2.ctypes.data_as(C.POINTER(C.c_double)),
                       self.loss.ctypes.data_as(C.POINTER(C.c_double)),
                       self.phase.ctypes.data_as(C.POINTER(C.c_int32)), var_cap,
                       self.var.ctypes.data_as(C.POINTER(C.c_double)) if var_cap > 0 else None)

    @property
    def len(self) -> int:
        return self.c.len

    def arrays(self):
        m = self.c.len
        return dict(k=self.k[:m].copy(), p=self.p[:m].copy(), S=self.S[:m].copy(), C2=self.C2[:m].copy(),
                    loss=self.loss[:m].copy(), phase=self.phase[:m].copy(),
                    var=self.var[:self.c.var_cap].copy())


def adpsgd_run(ctx: Context, sched: Schedule, state: State, k_end: int | None = None,
               trace: TraceBuffers | None = None) -> Stats:
    stats = Stats()
    k_end = sched.K if k_end is None else k_end
    _check(load().adpsgd_run(ctx.handle, C.byref(sched), C.byref(state), k_end,
                             C.byref(trace.c) if trace is not None else None, C.byref(stats)), "adpsgd_run")
    return stats


def adpsgd_sched_on_sync(sched: Schedule, state: State, k: int, S: float, gamma: float) -> int:
    ph = C.c_int32()
    _check(load().adpsgd_sched_on_sync(C.byref(sched), C.byref(state), k, S, gamma, C.byref(ph)),
           "adpsgd_sched_on_sync")
    return ph.value


def adpsgd_gamma(sched: Schedule, k: int) -> float:
    g = C.c_float()
    _check(load().adpsgd_gamma(C.byref(sched), k, C.byref(g)), "adpsgd_gamma")
    return g.value


def adpsgd_wire_bytes(n: int, P: int, rounds: int, with_scalar: bool = True):
    pn = C.c_double()
    tot = C.c_double()
    _check(load().adpsgd_wire_bytes(n, P, rounds, int(with_scalar), C.byref(pn), C.byref(tot)),
           "adpsgd_wire_bytes")
    return pn.value, tot.value


def adpsgd_philox_fill(seed: int, tag: int, n: int, nq: int, k: int, out, stream=None) -> None:
    _check(load().adpsgd_philox_fill(seed & 0xFFFFFFFFFFFFFFFF, tag, n, nq, k, _ptr(out), _stream(stream)),
           "adpsgd_philox_fill")


def adpsgd_noise_fill_f32(seed: int, tag: int, n: int, P: int, k: int, out, stream=None) -> None:
    _check(load().adpsgd_noise_fill_f32(seed & 0xFFFFFFFFFFFFFFFF, tag, n, P, k, _ptr(out), _stream(stream)),
           "adpsgd_noise_fill_f32")


def adpsgd_noise_fill_bf16(seed: int, n: int, P: int, out, stream=None) -> None:
    _check(load().adpsgd_noise_fill_bf16(seed & 0xFFFFFFFFFFFFFFFF, n, P, _ptr(out), _stream(stream)),
           "adpsgd_noise_fill_bf16")


def adpsgd_noise_fill_bf16_part(seed: int, n: int, P: int, replica0: int, col0: int, out, stream=None) -> None:
    """Rows [replica0, replica0 + n) and columns [col0, col0 + P) of the bf16 noise tensor."""
    _check(load().adpsgd_noise_fill_bf16_part(seed & 0xFFFFFFFFFFFFFFFF, n, P, replica0, col0, _ptr(out),
                                              _stream(stream)), "adpsgd_noise_fill_bf16_part")


def _nbytes(t, nbytes):
    return t.numel() * t.element_size() if nbytes is None else nbytes


def adpsgd_copy_h2d(dst, src, nbytes: int | None = None, stream=None) -> None:
    """Host tensor src -> device tensor dst (nbytes: all of src by default), enqueued on stream."""
    _check(load().adpsgd_copy_h2d(_ptr(dst), _ptr(src), _nbytes(src, nbytes), _stream(stream)), "adpsgd_copy_h2d")


def adpsgd_init_replicas(ctx: Context, w0) -> None:
    """Every replica row of x set to w0 (fp32 [P], host or device tensor) and v to zero, on the
    context's stream."""
    _check(load().adpsgd_init_replicas(ctx.handle, _ptr(w0)), "adpsgd_init_replicas")


def adpsgd_copy_d2h(dst, src, nbytes: int | None = None, stream=None) -> None:
    """Device tensor src -> host tensor dst (nbytes: all of src by default), enqueued on stream."""
    _check(load().adpsgd_copy_d2h(_ptr(dst), _ptr(src), _nbytes(src, nbytes), _stream(stream)), "adpsgd_copy_d2h")


def adpsgd_kernel_times(ctx: Context):
    t = KernelTiming()
    _check(load().adpsgd_kernel_times(ctx.handle, C.byref(t)), "adpsgd_kernel_times")
    return {name: getattr(t, name) for name, _ in KernelTiming._fields_}


def adpsgd_reset_kernel_times(ctx: Context) -> None:
    _check(load().adpsgd_reset_kernel_times(ctx.handle), "adpsgd_reset_kernel_times")


def adpsgd_test_force_incomplete(ctx: Context, on: bool) -> None:
    _check(load().adpsgd_test_force_incomplete(ctx.handle, int(bool(on))), "adpsgd_test_force_incomplete")


def adpsgd_destroy(ctx: Context) -> None:
    ctx.close()


def adpsgd_strerror(status: int) -> str:
    return strerror(status)


def adpsgd_last_error() -> str:
    return last_error()
