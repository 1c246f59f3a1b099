"""GB300 (sm_103a) engine for step-specific pruned video-DiT blocks.

The compute lives in the CUDA library behind include/dfs.h; ``dfs`` is its ctypes
binding (same entry-point names) and ``host`` moves synthetic problems between numpy
and device memory with torch.
"""
from . import build  # noqa: F401
