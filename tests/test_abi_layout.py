"""Host checks of the boundary's data layout and of the bench's bookkeeping (no GPU).

- Every struct the binding declares with ctypes has the size and field offsets that a C compiler
  gives the same struct from include/adpsgd.h: a field added or reordered on one side only is an
  ABI break that no GPU test would name.
- The source digests the bench uses to match committed ncu traffic to the current kernels can be
  computed for every kernel (their markers are present in the sources).
"""
import ctypes
import os
import shutil
import subprocess
import sys

import pytest

from paper_2007_06134_gb300 import abi

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

STRUCTS = {
    "adpsgd_config": abi.Config,
    "adpsgd_schedule": abi.Schedule,
    "adpsgd_state": abi.State,
    "adpsgd_trace": abi.Trace,
    "adpsgd_stats": abi.Stats,
    "adpsgd_kernel_timing": abi.KernelTiming,
    "adpsgd_shard": abi.Shard,
    "adpsgd_replica_split": abi.ReplicaSplit,
}


def test_ctypes_structs_match_the_c_header(tmp_path):
    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        pytest.skip("no C compiler")
    lines = ['#include <stddef.h>', '#include <stdio.h>', '#include "adpsgd.h"', "int main(void) {"]
    for cname, cls in STRUCTS.items():
        lines.append(f'    printf("{cname} size %zu\\n", sizeof({cname}));')
        for field, _ in cls._fields_:
            lines.append(f'    printf("{cname} {field} %zu\\n", offsetof({cname}, {field}));')
    lines += ["    return 0;", "}"]
    src = tmp_path / "layout.c"
    src.write_text("\n".join(lines) + "\n")
    exe = tmp_path / "layout"
    subprocess.run([cc, "-std=c99", "-I", os.path.join(ROOT, "include"), str(src), "-o", str(exe)], check=True)
    out = subprocess.run([str(exe)], check=True, capture_output=True, text=True).stdout.split("\n")
    c_side = {}
    for line in out:
        if line:
            name, field, value = line.split()
            c_side[(name, field)] = int(value)
    for cname, cls in STRUCTS.items():
        assert c_side[(cname, "size")] == ctypes.sizeof(cls), cname
        for field, _ in cls._fields_:
            assert c_side[(cname, field)] == getattr(cls, field).offset, (cname, field)


def test_bench_source_digests_compute():
    sys.path.insert(0, ROOT)
    try:
        import bench
    finally:
        sys.path.remove(ROOT)
    for kernel in bench.KERNEL_SOURCES:
        assert len(bench.kernel_source_digest(kernel)) == 16
