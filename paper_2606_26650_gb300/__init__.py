"""CAT-Q soft-ternary calibration hot path for GB300 (sm_103a).

The compute lives in libcatq.so (include/catq.h); `catq` is its Python binding and
`synthetic` the seeded workload generators.
"""
from . import catq, synthetic  # noqa: F401
