"""fp64 CPU oracle for the adapter fine-tuning step (test infrastructure only).

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s cpu-baseline / reference
leg may import this package.  The product path never does, and the two share no code.
"""
from . import ringada_oracle  # noqa: F401
