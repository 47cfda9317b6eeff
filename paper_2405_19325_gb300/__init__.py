"""GB300 (sm_103a) kNN-LM step of Nearest Neighbor Speculative Decoding.

The path (search, Eq. 2, Eq. 3 / Eq. 4) runs in hand-written CUDA kernels
behind the C ABI of include/nest.h; ``nest.Datastore`` is the Python binding.
"""
from .nest import BF16, F32, LIB_PATH, Datastore, NestError, load_library, plan_offline  # noqa: F401

__all__ = ["Datastore", "NestError", "load_library", "plan_offline", "LIB_PATH", "F32", "BF16"]
