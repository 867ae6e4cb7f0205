"""JIT-tuned dense MatMul / BatchMatMul for one GB300 (sm_103a).

The compute path lives in libnnjit.so (CUDA kernels + C ABI, include/nnjit.h); this
package is its Python binding.  ``build()`` compiles the library in-tree.
"""
from .nnjit import *  # noqa: F401,F403
from .nnjit import load_library, LIB_PATH, Plan, NnjitError, make_desc  # noqa: F401


def build(force: bool = False, verbose: bool = False) -> str:
    from .build_lib import build as _build
    return _build(force=force, verbose=verbose)
