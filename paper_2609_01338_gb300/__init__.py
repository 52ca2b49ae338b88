"""GB300-native restoration-overlapped prefill over a partially evicted LLM
memory state (mzCache's TTFT path), as a C-ABI CUDA library plus this thin
ctypes binding.

Every step of the path runs in libmzc's sm_103a kernels; this package only
marshals arguments.  Importing it does not need a GPU; calling a compute
entry point without the built library raises instead of falling back.
"""
from .mzc import *  # noqa: F401,F403
from .mzc import load, lib_path  # noqa: F401
