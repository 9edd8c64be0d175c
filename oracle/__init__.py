"""CPU oracle for distributed sign momentum with local steps (arXiv 2411.17866).

TEST INFRASTRUCTURE: only tests/, __graft_entry__.smoke() and bench.py's
cpu_baseline / reference arms may import this package.  It shares no code
with the CUDA library and never imports it.
"""
from .dsm_oracle import *  # noqa: F401,F403
