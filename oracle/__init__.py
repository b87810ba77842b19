"""fp64 CPU oracle for stale-synchronous MF-SGD (test infrastructure only).

Only the test suite, the smoke check and the benchmark's CPU baseline may
import this package.  It shares no code with the CUDA library.
"""
from .oracle import Oracle, OracleConfig, build, ctr_u64, essp_thresholds, schedule_rule  # noqa: F401
