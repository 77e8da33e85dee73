"""Chameleon format-adaptive quantized linear layer on GB300 (sm_103a).

The compute path is libchameleon.so (CUDA kernels behind the C ABI of include/chameleon.h); this
package holds its sources (csrc/), the in-tree build script (build.py), the ctypes binding
(_binding.py) and the seeded synthetic workload generators (workloads.py).  Importing the package
does not load the library; the first binding call does, and raises if it has not been built.
"""
from . import _binding as chameleon  # noqa: F401
from ._binding import *  # noqa: F401,F403
