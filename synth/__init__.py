"""Seeded synthetic inputs shared by the CPU oracle, the tests and the benchmark.

This module only draws samples and lays out grids; it holds none of the
reservation-cost arithmetic, so the oracle and the CUDA path can both take
their inputs from it without sharing any of the method's code.
"""

from .workloads import (  # noqa: F401
    Workload,
    WORKLOADS,
    lognormal_workload_k3_n1e3,
    lognormal_workload_k8_n1e5,
    heavy_tail_workload_k16_n1e6,
    regime_sweep_workload_k8_n2e5,
    drift_loop_workload_k32_n1e6,
    random_case,
    slice_workload,
)
from .bcd_instances import CONFIGS, SCALABILITY_SIZES, bcd_instance  # noqa: F401
