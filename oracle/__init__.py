"""CPU oracle for the Omega-QVLA W4A4 linear -- test infrastructure only.

Only tests/, __graft_entry__.smoke() and bench.py's CPU-baseline / reference leg may
import this package.  The product (paper_2605_28803_gb300) never imports it.
"""
from . import qvla_oracle  # noqa: F401
