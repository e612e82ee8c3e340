import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

# NumPy asks for transparent huge pages on large arrays; on a host whose
# memory is fragmented each such fault compacts memory synchronously, which
# made the float64 oracle runs of whole networks several times slower
# (VGG-16: 24 s -> 126 s, almost all of it system time)
os.environ.setdefault("NUMPY_MADVISE_HUGEPAGE", "0")
try:
    import numpy as _np
    _core = getattr(_np, "_core", None) or getattr(_np, "core", None)
    _core.multiarray._set_madvise_hugepage(False)
except Exception:
    pass


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a)")
    config.addinivalue_line("markers", "slow: long-running CPU test")


def has_gpu():
    try:
        import torch
        return torch.cuda.is_available()
    except Exception:
        return False


def pytest_collection_modifyitems(config, items):
    if has_gpu():
        return
    skip = pytest.mark.skip(reason="no CUDA device")
    for it in items:
        if "gpu" in it.keywords:
            it.add_marker(skip)
