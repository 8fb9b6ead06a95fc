"""Splitting one problem over several processes (one GPU each), or over threads.

Column shards (``adpsgd_set_shard``): the local step is elementwise and the averaging reduces over
replicas column by column, so one problem can be cut into contiguous column ranges, one per
shard.  The only exchange is each shard's two fp64 partial sums at every sync; the library adds
them in shard order.

Replica split (``adpsgd_set_replica_split``): the paper's own mapping, each process holding whole
replicas.  A sync is an allreduce in two halves around the library's averaging kernel: an
all-to-all that gives each process all replicas' values of its column chunk, then an all-gather of
the chunks' means.

This module holds the plumbing around those calls and none of the method's arithmetic:

- ``column_split`` chooses column ranges (starts on multiples of 4, so that every Philox block of
  four columns lies in one range);
- ``dist_gather`` moves the partial sums between processes with ``torch.distributed``
  (all-gather over a CPU group); ``ThreadGather`` moves them between threads of one process;
- ``DistReplicaCollective`` runs a replica split's all-to-all and all-gather with
  ``torch.distributed`` (NCCL on GPUs, gloo on CPUs); ``ThreadReplicaCollective`` runs them
  between threads of one process that share a GPU, by device copies.
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


def chunk_sizes(P: int, processes: int):
    """Column count of every process's chunk of the averaging (column_split over P)."""
    return [column_split(P, processes, r)[1] for r in range(processes)]


class DistReplicaCollective:
    """A replica split's two collectives over torch.distributed, for one process.

    x: this process's replicas [n_local, P]; chunk_x: [n_total, P_chunk] for its chunk; rows of
    chunk_x are filled in process order, so process r's replicas must be the global replicas that
    follow those of processes 0 .. r-1.  stream: the library context's CUDA stream (None on CPU).
    ``callback`` is the COLLECTIVE_FN to pass to adpsgd_set_replica_split."""

    def __init__(self, x, chunk_x, n_locals, group=None, stream=None):
        import torch.distributed as dist
        self.dist = dist
        self.group = group
        self.x, self.chunk_x, self.stream = x, chunk_x, stream
        self.g = dist.get_world_size(group)
        self.rank = dist.get_rank(group)
        self.n_locals = list(n_locals)
        P = x.shape[1]
        self.ranges = [column_split(P, self.g, r) for r in range(self.g)]
        self.pmax = max(cols for _, cols in self.ranges)
        self.callback = abi.COLLECTIVE_FN(self._run)

    def _scatter_columns(self):
        torch = self._torch()
        n_local = self.x.shape[0]
        P_chunk = self.ranges[self.rank][1]
        send = torch.cat([self.x[:, c0:c0 + cols].reshape(-1) for c0, cols in self.ranges])
        self.dist.all_to_all_single(self.chunk_x.view(-1), send,
                                    output_split_sizes=[nl * P_chunk for nl in self.n_locals],
                                    input_split_sizes=[n_local * cols for _, cols in self.ranges], group=self.group)

    def _gather_average(self):
        torch = self._torch()
        mine = torch.zeros(self.pmax, dtype=self.x.dtype, device=self.x.device)
        P_chunk = self.ranges[self.rank][1]
        mine[:P_chunk] = self.chunk_x[0, :P_chunk]
        every = torch.empty(self.g * self.pmax, dtype=self.x.dtype, device=self.x.device)
        self.dist.all_gather_into_tensor(every, mine, group=self.group)
        for r, (c0, cols) in enumerate(self.ranges):
            self.x[:, c0:c0 + cols] = every[r * self.pmax:r * self.pmax + cols]

    @staticmethod
    def _torch():
        import torch
        return torch

    def _run(self, op, _user):
        try:
            torch = self._torch()
            if self.stream is not None:
                with torch.cuda.stream(self.stream):
                    self._dispatch(op)
            else:
                self._dispatch(op)
            return 0
        except Exception:  # reported to the caller as ADPSGD_E_PEER
            return 1

    def _dispatch(self, op):
        if op == abi.SCATTER_COLUMNS:
            self._scatter_columns()
        elif op == abi.GATHER_AVERAGE:
            self._gather_average()
        else:
            raise ValueError(op)


class ThreadReplicaCollective:
    """A replica split's two collectives between `processes` threads of one process that share a
    GPU: device copies between the threads' buffers, each thread on its own stream, with a host
    barrier on both sides of every copy so that no thread reads or overwrites a buffer another
    thread is still using.  register(r, x, chunk_x, stream) before the run; callbacks[r] is thread
    r's COLLECTIVE_FN."""

    def __init__(self, processes: int, P: int, timeout: float = 120.0):
        self.g = processes
        self.ranges = [column_split(P, processes, r) for r in range(processes)]
        self.barrier = threading.Barrier(processes, timeout=timeout)
        self.bufs = [None] * processes
        self.callbacks = [abi.COLLECTIVE_FN(self._make(r)) for r in range(processes)]

    def register(self, r, x, chunk_x, row0, stream):
        """Thread r's replicas x [n_local, P] (global rows row0 ..), its chunk buffer, its stream."""
        self.bufs[r] = (x, chunk_x, row0, stream)

    def _make(self, r):
        def collective(op, _user):
            import torch
            try:
                x, chunk_x, row0, stream = self.bufs[r]
                stream.synchronize()
                self.barrier.wait()
                with torch.cuda.stream(stream):
                    if op == abi.SCATTER_COLUMNS:
                        for c, (c0, cols) in enumerate(self.ranges):
                            dst = self.bufs[c][1]
                            dst[row0:row0 + x.shape[0], :cols].copy_(x[:, c0:c0 + cols])
                    else:
                        for c, (c0, cols) in enumerate(self.ranges):
                            x[:, c0:c0 + cols].copy_(self.bufs[c][1][0:1, :cols].expand(x.shape[0], cols))
                stream.synchronize()
                self.barrier.wait()
                return 0
            except threading.BrokenBarrierError:
                return 1
        return collective
