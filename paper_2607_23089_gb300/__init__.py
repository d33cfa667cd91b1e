"""librowop for GB300: row-wise reduce-then-normalise operators (softmax,
log-softmax, LayerNorm, RMSNorm; dense and ragged) as hand-written sm_103a
CUDA kernels behind a C ABI (``include/rowop.h``).

``build.build()`` compiles the library in-tree; ``rowop`` is the ctypes
binding (C-named functions plus torch tensor helpers)."""
from . import build, rowop  # noqa: F401

__all__ = ["build", "rowop"]
