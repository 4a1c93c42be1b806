"""Seeded synthetic inputs shared by the CPU oracle and the CUDA path.

This package only draws random numbers and lays out shapes. It holds none of
the method's arithmetic (no projection, normalisation, rotation or attention),
so that neither side of a parity check can inherit a mistake from it.
"""

from .workloads import (  # noqa: F401
    Geometry,
    Workload,
    WORKLOADS,
    make_workload,
    make_custom,
    make_kv_weights,
    layout,
)
