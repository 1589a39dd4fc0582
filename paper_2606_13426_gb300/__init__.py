"""GB300-native (sm_103a) verification step of speculative diffusion sampling.

Layout:
  csrc/       CUDA kernels and the C-ABI (libspecdiff.so, declared in include/specdiff.h)
  buildlib.py nvcc build of libspecdiff.so (in-tree, lib/)
  binding.py  ctypes binding, one Python function per C entry point, same names
  api.py      torch-facing helpers (allocation + pointer passing only), including the
              end-to-end sampler's calls (the round loop itself runs in csrc/sdv_sampler.cu)

Nothing here computes on the CPU: when the library is missing every call raises.
"""
from .buildlib import build, lib_path  # noqa: F401

__all__ = ["build", "lib_path"]
