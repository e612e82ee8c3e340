"""Synthetic workloads: layer-sequence descriptions and seeded generators.

Shared input for the CUDA path and the CPU oracle; holds none of the
swapping method's arithmetic.
"""
from . import arch, gen  # noqa: F401
