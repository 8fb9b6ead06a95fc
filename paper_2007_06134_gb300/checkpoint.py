"""Checkpoint and resume of a run: x, v and the scheduler state.

The noise of step k is a pure function of (seed, replica, k, element), so x, v and the
scheduler state (next iteration, Algorithm 2's cnt and p, the sampled C_2 and its sample count,
the rounds so far) are all a run needs to resume with the same bits.  The per-sync trace can be
saved along.  The file is a numpy .npz archive.
"""
from __future__ import annotations

import numpy as np

from . import abi

_STATE_FIELDS = ("k_next", "cnt", "p", "C2", "m", "rounds")


def state_to_dict(state: abi.State) -> dict:
    return {name: getattr(state, name) for name in _STATE_FIELDS}


def state_from_dict(d) -> abi.State:
    st = abi.State()
    for name in _STATE_FIELDS:
        setattr(st, name, type(getattr(st, name))(d[name]))
    return st


def save(path: str, x, v, state: abi.State, trace: dict | None = None) -> None:
    """Write x, v (torch tensors or arrays [n, P] fp32), the scheduler state and an optional
    trace (the dict of TraceBuffers.arrays())."""
    def host(a):
        return a.detach().cpu().numpy() if hasattr(a, "detach") else np.asarray(a)
    payload = {"x": host(x), "v": host(v)}
    payload.update({"state_" + k: np.asarray(val) for k, val in state_to_dict(state).items()})
    for k, val in (trace or {}).items():
        payload["trace_" + k] = np.asarray(val)
    np.savez(path, **payload)


def load(path: str):
    """(x, v, state, trace) from a file written by save(); x and v as numpy arrays."""
    with np.load(path) as f:
        x, v = f["x"], f["v"]
        state = state_from_dict({k: f["state_" + k][()] for k in _STATE_FIELDS})
        trace = {k[len("trace_"):]: f[k] for k in f.files if k.startswith("trace_")}
    return x, v, state, trace
