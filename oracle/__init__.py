"""CPU oracle of the RPS scoring path: test infrastructure only.

Only the test-suite, ``__graft_entry__.smoke()`` and the benchmark's CPU-baseline
leg may import this package. The CUDA library never does.
"""
from .oracle import Oracle, RowStats, default  # noqa: F401
