"""GB300 (sm_103a) data-parallel hot path of ADPSGD (Jiang & Agrawal, arXiv 2007.06134).

n replicas of a P-parameter model live on one GPU as an [n, P] fp32 tensor.  The CUDA
library ``libadpsgd.so`` (C ABI in include/adpsgd.h) runs the fused local step and the
fused average + variance; its host runtime applies the period rule of Algorithm 2.
``abi`` is the thin ctypes binding with the C names; ``inputs`` draws the seeded synthetic
workloads.  Importing the package does not load CUDA; the binding builds and loads the
library on first use and raises if it cannot.
"""
from . import inputs  # noqa: F401  (no CUDA)


def __getattr__(name):
    if name.startswith("adpsgd_") or name in ("Config", "Schedule", "State", "Stats", "TraceBuffers",
                                              "Context", "AdpsgdError", "make_config", "make_schedule"):
        from . import abi
        return getattr(abi, name)
    raise AttributeError(name)
