"""GB300-native training of parareal neural networks (Lee, Lee & Park).

The compute path is libpnn.so (CUDA kernels for sm_103a behind the C ABI of
include/pnn.h); `pnn` is its Python binding.  Build with `build.build()`."""
from . import build  # noqa: F401

__all__ = ["build", "pnn"]
