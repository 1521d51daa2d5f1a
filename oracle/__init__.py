"""fp64 CPU oracle for the CoLA auto-encoder layer (test infrastructure only).

Only tests/, __graft_entry__.smoke() and bench.py's cpu_baseline / reference
legs may import this package.  It shares no code with the CUDA path.
"""
from .oracle import *  # noqa: F401,F403
