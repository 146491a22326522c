"""Shared seeded input generator (workload shapes + synthetic Q/K/V).

Holds no arithmetic of the HeadKV method; both the CPU oracle and the CUDA
path take their inputs from here.
"""
from . import configs, gen  # noqa: F401
