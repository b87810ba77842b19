"""Seeded synthetic inputs for the stale-synchronous MF-SGD clock.

This package produces inputs only: observed ratings (i, j, D), the initial
factor tables, the data partition across workers and the minibatch label of
each rating.  It holds none of the method's arithmetic (no residuals, no
gradients, no schedule), so both the fp64 oracle and the CUDA library can
consume its arrays without sharing any logic.
"""
from .synth import (  # noqa: F401
    GOLDEN,
    ctr_u64,
    mix64,
    MFData,
    make_mf_data,
    shard_users,
    minibatch_labels,
)
from .workloads import WORKLOADS, Workload, workload  # noqa: F401
