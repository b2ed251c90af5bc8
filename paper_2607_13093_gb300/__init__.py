"""Split-head vocabulary projection for GB300 (sm_103a).

The compute path lives in the C-ABI library built from csrc/ (declared in
include/sph.h); `paper_2607_13093_gb300.sph` is its thin ctypes binding.
`workloads` generates seeded synthetic inputs.  Submodules are imported on
first use so that input generation works without the built library.
"""
import importlib

__all__ = ["sph", "workloads"]


def __getattr__(name):
    if name in __all__:
        return importlib.import_module("." + name, __name__)
    raise AttributeError(name)
