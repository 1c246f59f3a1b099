"""CPU oracle of the pruned DiT block (test infrastructure only).

Only tests/, __graft_entry__.smoke() and bench.py's cpu_baseline / reference leg may
import this package.  It shares no code with the CUDA library and never calls it.
"""
from .dfs_oracle import *  # noqa: F401,F403
