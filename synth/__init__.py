"""Seeded synthetic inputs for AWSRC workloads.

This module only draws inputs (weights, the RTN-INT4 backbone reconstruction
W0 = Q(W) of Eq. 1, activation and Fisher statistics); it holds none of the
codec's arithmetic. Both the CUDA path and the oracle consume the arrays it
produces.
"""
from .workloads import (  # noqa: F401
    MODULE_ORDER,
    WORKLOADS,
    Workload,
    layer_shapes,
    make_layer,
    make_module,
    rtn_int4_g128,
)
