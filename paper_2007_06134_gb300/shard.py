"""Column sharding of one problem over several processes (one GPU each), or over threads.

The local step is elementwise and the averaging reduces over replicas column by column, so one
problem can be cut into contiguous column ranges, one per shard (``adpsgd_set_shard`` in the C
ABI).  The only exchange is each shard's two fp64 partial sums at every sync; the library adds
them in shard order.  This module holds the plumbing around that call and none of the method's
arithmetic:

- ``column_split`` chooses the shards' column ranges (starts on multiples of 4, so that every
  Philox block of four columns lies in one shard);
- ``dist_gather`` moves the partial sums between processes with ``torch.distributed``
  (all-gather over a CPU group);
- ``ThreadGather`` moves them between threads of one process (shards that share a GPU).
"""
from __future__ import annotations

import ctypes as C
import threading

from . import abi


def column_split(P: int, shards: int, index: int):
    """(col0, P_index): shard `index`'s contiguous column range of a P-column problem.  The blocks
    of four columns are dealt out as evenly as possible; the ragged tail (P % 4) goes to the last
    shard."""
    if shards < 1 or not 0 <= index < shards or P < 0:
        raise ValueError((P, shards, index))
    blocks = P // 4
    base, extra = divmod(blocks, shards)
    start = index * base + min(index, extra)
    count = base + (1 if index < extra else 0)
    col0 = 4 * start
    cols = 4 * count
    if index == shards - 1:
        cols = P - col0
    return col0, cols


def _fill(gathered, values):
    for t, val in enumerate(values):
        gathered[t] = val


def dist_gather(group=None):
    """A GATHER_FN that all-gathers `count` doubles per shard over torch.distributed, shard r =
    rank r of `group` (a CPU-capable group, e.g. gloo; default: a new gloo group over the world).
    Returns (callback, group).  The callback returns 1 on any exception (the library then reports
    ADPSGD_E_PEER)."""
    import torch
    import torch.distributed as dist
    if group is None:
        group = dist.new_group(backend="gloo")
    world = dist.get_world_size(group)

    def gather(local, count, gathered, _user):
        try:
            mine = torch.tensor([local[t] for t in range(count)], dtype=torch.float64)
            parts = [torch.empty(count, dtype=torch.float64) for _ in range(world)]
            dist.all_gather(parts, mine, group=group)
            _fill(gathered, [float(x) for part in parts for x in part.tolist()])
            return 0
        except Exception:  # reported to the caller as ADPSGD_E_PEER
            return 1

    return abi.GATHER_FN(gather), group


class ThreadGather:
    """The exchange between `shards` threads of one process (each running one shard's context):
    every thread deposits its values and waits at a barrier for the others."""

    def __init__(self, shards: int, timeout: float = 120.0):
        self.shards = shards
        self.barrier = threading.Barrier(shards, timeout=timeout)
        self.slots = [None] * shards
        self.callbacks = [abi.GATHER_FN(self._make(r)) for r in range(shards)]

    def _make(self, index):
        def gather(local, count, gathered, _user):
            try:
                self.slots[index] = [local[t] for t in range(count)]
                self.barrier.wait()
                _fill(gathered, [v for r in range(self.shards) for v in self.slots[r]])
                self.barrier.wait()  # nobody overwrites its slot before everyone has read
                return 0
            except threading.BrokenBarrierError:
                return 1
        return gather
