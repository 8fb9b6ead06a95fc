"""Diagnostics of a run from its recorded trace (host-side, O(K)).

The paper measures how far the replicas drift apart with Var[W_k] (Sec. II-B) and summarises a
schedule by the interval means V_t (Eq. vt) and the step-size-weighted mean variance (Eq.
metric2), which bounds the convergence metric of Eq. metric1 (Eq. bound1).  With the trace
option `var`, adpsgd_run records Var[W_k] at the start of every iteration k; these functions
turn that series into the paper's quantities.
"""
from __future__ import annotations

import numpy as np


def interval_means(var, sync_k, k_begin: int = 0):
    """V_t (Eq. vt): the mean of Var[W_k] over the iterations of each sync interval, from the
    iteration after the previous sync (or k_begin) up to and including the sync iteration."""
    var = np.asarray(var, dtype=np.float64)
    out = []
    start = k_begin
    for k in sync_k:
        k = int(k)
        out.append(var[start:k + 1].mean())
        start = k + 1
    return np.asarray(out)


def weighted_variance(var, gammas):
    """Eq. metric2: sum_k gamma_k Var[W_k] / sum_k gamma_k over the recorded iterations."""
    var = np.asarray(var, dtype=np.float64)
    g = np.asarray(gammas, dtype=np.float64)[: var.size]
    return float(np.sum(g * var) / np.sum(g))


def phase_means(var, edges):
    """Mean Var[W_k] over consecutive iteration ranges [edges[t], edges[t + 1])."""
    var = np.asarray(var, dtype=np.float64)
    return [float(var[a:b].mean()) for a, b in zip(edges[:-1], edges[1:])]
