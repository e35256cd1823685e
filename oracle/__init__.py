"""CPU oracle for the C2KV compose + suffix-attention path (test infrastructure only).

Only the tests, ``__graft_entry__.smoke()`` and the benchmark's CPU-baseline / reference
leg may import this package.  The product path never does.
"""
from . import c2kv_oracle  # noqa: F401
