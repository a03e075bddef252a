"""CPU oracle for the EOGP hot path: test infrastructure, not product code.

Only tests/, __graft_entry__.smoke() and bench.py's CPU-baseline / reference
arm may import this package.
"""
from . import eogp_oracle  # noqa: F401
