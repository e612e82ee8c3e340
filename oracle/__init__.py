"""CPU oracle for block-swapped inference — TEST INFRASTRUCTURE ONLY.

Plain, slow, float64 restatements of what the swapped GPU path computes:

  forward.py  the layer-by-layer forward pass of a workload.  Swapping is
              lossless (the paper's Overview, "Design Scope": parameters and
              architecture are unchanged), so whatever the partition, the
              swapped result is the plain forward pass of the model.
  plan.py     the partitioner as an exhaustive search over cut vectors with
              the delay abstractions of Sec. 6.1, the block-count rule and
              objective of Sec. 6.2.2 (Eq. 2-4), the liveness-based
              activation workspace, and the multi-DNN budget split (Eq. 1).

Only tests/, __graft_entry__.smoke() and bench.py's CPU-baseline leg may
import this package.  The library under paper_2401_16757_gb300/ never does,
and nothing here imports that library.
"""
