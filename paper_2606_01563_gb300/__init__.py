"""MomentKV hot path on one GB300 (sm_103a): compress, corrected decode and
moment-informed eviction as hand-written CUDA kernels behind a C ABI.

`mkv` is the ctypes binding of include/mkv.h (loaded lazily, fails loudly if
libmkv.so has not been built); `inputs` draws the seeded synthetic tensors;
`build` compiles the library.
"""
from . import inputs  # noqa: F401
