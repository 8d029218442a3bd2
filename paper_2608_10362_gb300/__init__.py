"""GB300-native (sm_103a) draft-then-verify speculative decoding step.

The compute path is libmemspec.so (hand-written CUDA behind the C ABI in
include/memspec.h); this package is its Python binding.  Importing the package
does not load the library; the first call does, and fails loudly if it was not
built (python -m paper_2608_10362_gb300.build).
"""
from ._lib import MemSpecError, load  # noqa: F401
from .engine import (Engine, fill_blob, kv_bytes, model_cfg, op_linear, pack_matrix,  # noqa: F401
                     int4_pack, op_linear_int4, op_linear_noalloc, op_sample, weights_bytes)
from .sched import DraftScheduler  # noqa: F401
