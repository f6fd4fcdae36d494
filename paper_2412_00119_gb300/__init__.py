"""GB300 (sm_103a) implementation of the fully binary BMLP training rule of
arXiv 2412.00119 (Alg. 1-3): a C-ABI CUDA library (``libbmlp.so``, declared in
``include/bmlp.h``) and its ctypes binding.  See ``bmlp`` for the API."""
from .bmlp import *  # noqa: F401,F403
from .bmlp import BMLP, BmlpError, lib, library_path  # noqa: F401
from ._build import build  # noqa: F401
