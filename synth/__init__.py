"""Seeded synthetic workloads shared by the tests, the benchmark and the smoke run.

This package only draws inputs (attention weights, start vectors, per-step weight
perturbations).  It contains none of the method's arithmetic: no power iteration,
no spectral norm, no scale formula.  Both the CUDA library and the float64 oracle
consume the tensors it returns, byte for byte.
"""

from .configs import WORKLOADS, Workload, get_workload  # noqa: F401
from .gen import (  # noqa: F401
    make_start_vectors,
    make_weights,
    TransientWeights,
)
