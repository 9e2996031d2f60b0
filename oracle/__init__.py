"""fp64 CPU oracle of the CAT-Q soft-ternary hot path (test infrastructure only).

Only tests/, __graft_entry__.smoke() and bench.py's CPU-baseline leg may import this
package.  It shares no code with the CUDA path.
"""
from . import catq_oracle  # noqa: F401
