"""Block-swapped DNN inference under a device-memory budget on one GB300
(SwapNet, arXiv 2401.16757), as a C-ABI library (libswapnet.so, declared in
include/swapnet.h) with a thin ctypes binding.

    from paper_2401_16757_gb300 import capi
    desc = capi.Desc(model)                      # layer sequence -> C descriptor
    plan = capi.Plan.partition(desc, budget)     # Sec. 6.2.2 partition
    eng = capi.Engine(plan, capi.HostWeights(w)) # pin + map weights, skeleton
    eng.infer(d_in, d_out, stream)               # swapped inference
"""
from . import _capi as capi  # noqa: F401
