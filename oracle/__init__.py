"""Float64 CPU oracle for L_JAB (test infrastructure only).

Only tests/, __graft_entry__.smoke() and bench.py's CPU-baseline / reference legs may import
this package. The product path never imports it, and it never imports the product path.
"""
from .jab_oracle import *  # noqa: F401,F403
from .jab_oracle import __all__  # noqa: F401
