"""ctypes declarations of the C ABI in include/memspec.h and include/memspec_ops.h.

Loading fails loudly when libmemspec.so is missing: there is no fallback path.
"""
from __future__ import annotations

import ctypes as C
import os

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libmemspec.so")

# status codes (memspec_status)
OK, ERR_INVALID_ARG, ERR_CUDA, ERR_BUDGET, ERR_NOT_RESIDENT, ERR_BUSY, ERR_TIMEOUT, \
    ERR_DEVICE_STATUS, ERR_UNSUPPORTED = range(9)
STATUS_NAMES = ["OK", "INVALID_ARG", "CUDA", "BUDGET", "NOT_RESIDENT", "BUSY", "TIMEOUT",
                "DEVICE_STATUS", "UNSUPPORTED"]

# tensor ids (memspec_tensor)
T_TOK_EMB, T_ATTN_NORM, T_WQKV, T_WO, T_FFN_NORM, T_WGATE, T_WUP, T_WDOWN, T_FINAL_NORM, \
    T_LM_HEAD = range(10)

# buffer ids (memspec_buffer)
BUF_TARGET_LOGITS, BUF_DRAFT_LOGITS, BUF_DRAFT_TOKENS, BUF_TOKENS, BUF_SEQ_STATE, \
    BUF_ACCEPT_DEBUG, BUF_RESIDUAL, BUF_PASS_TRACE, BUF_SEEDS, BUF_TREE_LOGITS = range(10)

# launch modes (memspec_init_params.launch_mode)
LAUNCH_PER_OP, LAUNCH_PASS = 0, 1
# draft-step kernels (memspec_init_params.draft_kernel)
DRAFT_KERNEL_AUTO, DRAFT_KERNEL_PER_OP, DRAFT_KERNEL_FUSED = 0, 1, 2
PASS_TRACE_OPS = 2048

DEV_TIMEOUT, DEV_BAD_TOKEN, DEV_BAD_LENGTH = 0x1, 0x2, 0x4

# memspec_query_info ids
INFO_DRAFT_LAUNCHES, INFO_VERIFY_LAUNCHES, INFO_ACCEPT_LAUNCHES, INFO_DRAFT_FUSED = range(4)


class ModelCfg(C.Structure):
    _fields_ = [("n_layers", C.c_int32), ("d_model", C.c_int32), ("n_heads", C.c_int32),
                ("n_kv_heads", C.c_int32), ("head_dim", C.c_int32), ("d_ffn", C.c_int32),
                ("vocab", C.c_int32), ("tied_embeddings", C.c_int32), ("rope_base", C.c_float),
                ("norm_eps", C.c_float)]


class InitParams(C.Structure):
    _fields_ = [("target", ModelCfg), ("target_weights_dev", C.c_void_p),
                ("target_kv_dev", C.c_void_p), ("max_batch", C.c_int32), ("max_seq", C.c_int32),
                ("max_k", C.c_int32), ("max_drafts", C.c_int32), ("draft_shape_max", ModelCfg),
                ("draft_arena_dev", C.c_void_p), ("draft_budget_bytes", C.c_size_t),
                ("stream_main", C.c_void_p), ("stream_side", C.c_void_p),
                ("use_graphs", C.c_int32), ("launch_mode", C.c_int32), ("trace", C.c_int32),
                ("draft_kernel", C.c_int32)]


# draft scheduling (memspec_sched.h)
POLICY_MEMSPEC, POLICY_MAB_ASYNC, POLICY_STATIC = 0, 1, 2
SCHED_MAX_DRAFTS = 16
STATE_FN = C.CFUNCTYPE(C.c_int32, C.c_void_p, C.c_int32, C.POINTER(C.c_int32))
DRAFT_FN = C.CFUNCTYPE(C.c_int32, C.c_void_p, C.c_int32)


class Residency(C.Structure):
    _fields_ = [("user", C.c_void_p), ("state", STATE_FN), ("load", DRAFT_FN), ("evict", DRAFT_FN),
                ("set_active", DRAFT_FN)]


class SchedParams(C.Structure):
    _fields_ = [("n_drafts", C.c_int32), ("capacity", C.c_int32), ("policy", C.c_int32),
                ("ucb_c", C.c_float), ("k_draft", C.c_int32)]


class SchedDecision(C.Structure):
    _fields_ = [("active", C.c_int32), ("desired", C.c_int32), ("fallback", C.c_int32),
                ("n_evicted", C.c_int32), ("n_prefetched", C.c_int32),
                ("evicted", C.c_int32 * SCHED_MAX_DRAFTS),
                ("prefetched", C.c_int32 * SCHED_MAX_DRAFTS)]


class SchedStats(C.Structure):
    _fields_ = [("points", C.c_int64), ("desired_intervals", C.c_int64),
                ("fallback_intervals", C.c_int64), ("loads", C.c_int64), ("evictions", C.c_int64),
                ("refusals", C.c_int64), ("switches", C.c_int64), ("desired_s", C.c_double),
                ("fallback_s", C.c_double), ("policy_s", C.c_double)]


EXPORTS = {
    # name: (restype, argtypes)
    "memspec_weights_bytes": (C.c_int, [C.POINTER(ModelCfg), C.POINTER(C.c_size_t)]),
    "memspec_weights_offset": (C.c_int, [C.POINTER(ModelCfg), C.c_int32, C.c_int32,
                                         C.POINTER(C.c_size_t), C.POINTER(C.c_size_t)]),
    "memspec_kv_bytes": (C.c_int, [C.POINTER(ModelCfg), C.c_int32, C.c_int32,
                                   C.POINTER(C.c_size_t)]),
    "memspec_workspace_bytes": (C.c_int, [C.POINTER(InitParams), C.POINTER(C.c_size_t)]),
    "memspec_init": (C.c_int, [C.POINTER(InitParams), C.c_void_p, C.POINTER(C.c_void_p)]),
    "memspec_destroy": (None, [C.c_void_p]),
    "memspec_last_error": (C.c_char_p, [C.c_void_p]),
    "memspec_register_draft": (C.c_int, [C.c_void_p, C.c_int32, C.POINTER(ModelCfg), C.c_void_p,
                                         C.c_void_p]),
    "memspec_load_draft_async": (C.c_int, [C.c_void_p, C.c_int32, C.POINTER(C.c_size_t)]),
    "memspec_query_draft": (C.c_int, [C.c_void_p, C.c_int32, C.POINTER(C.c_int32)]),
    "memspec_evict_draft": (C.c_int, [C.c_void_p, C.c_int32]),
    "memspec_set_active_draft": (C.c_int, [C.c_void_p, C.c_int32]),
    "memspec_prefill": (C.c_int, [C.c_void_p, C.c_int32, C.POINTER(C.c_int32), C.c_int32,
                                  C.c_uint64]),
    "memspec_set_batch": (C.c_int, [C.c_void_p, C.c_int32]),
    "memspec_draft_step": (C.c_int, [C.c_void_p, C.c_int32, C.c_float]),
    "memspec_verify_step": (C.c_int, [C.c_void_p, C.c_int32]),
    "memspec_tree_step": (C.c_int, [C.c_void_p, C.c_int32, C.c_void_p, C.c_void_p, C.c_float, C.c_void_p]),
    "memspec_accept_commit": (C.c_int, [C.c_void_p, C.c_int32, C.c_float, C.c_void_p]),
    "memspec_sync": (C.c_int, [C.c_void_p, C.c_int32, C.POINTER(C.c_uint32)]),
    "memspec_read_buffer": (C.c_int, [C.c_void_p, C.c_int32, C.c_void_p, C.c_size_t]),
    "memspec_query_info": (C.c_int, [C.c_void_p, C.c_int32, C.POINTER(C.c_int64)]),
    "memspec_write_buffer": (C.c_int, [C.c_void_p, C.c_int32, C.c_void_p, C.c_size_t]),
    "memspec_op_linear_scratch_bytes": (C.c_int, [C.c_int32, C.c_int32, C.c_int32,
                                                  C.POINTER(C.c_size_t)]),
    "memspec_op_linear": (C.c_int, [C.c_void_p, C.c_void_p, C.c_void_p, C.c_int32, C.c_int32,
                                    C.c_int32, C.c_void_p, C.c_size_t, C.c_void_p, C.c_void_p]),
    "memspec_op_linear_noalloc": (C.c_int, [C.c_void_p, C.c_void_p, C.c_void_p, C.c_int32,
                                            C.c_int32, C.c_int32, C.c_void_p, C.c_void_p]),
    "memspec_int4_packed_bytes": (C.c_int64, [C.c_int32, C.c_int32]),
    "memspec_int4_pack": (C.c_int, [C.c_void_p, C.c_void_p, C.c_void_p, C.c_int32, C.c_int32, C.c_void_p,
                                    C.c_void_p]),
    "memspec_op_linear_int4": (C.c_int, [C.c_void_p, C.c_void_p, C.c_void_p, C.c_int32, C.c_int32, C.c_int32,
                                         C.c_void_p, C.c_void_p]),
    "memspec_op_sample": (C.c_int, [C.c_void_p, C.c_int32, C.c_int32, C.c_float, C.c_void_p,
                                    C.c_void_p, C.c_void_p]),
    "memspec_op_last_error": (C.c_char_p, []),
    "memspec_pack_matrix": (C.c_int, [C.c_void_p, C.c_void_p, C.c_int32, C.c_int32, C.c_void_p,
                                      C.c_size_t, C.c_void_p]),
    "memspec_sched_create": (C.c_int, [C.POINTER(SchedParams), C.POINTER(Residency), C.c_void_p,
                                       C.POINTER(C.c_void_p)]),
    "memspec_sched_destroy": (None, [C.c_void_p]),
    "memspec_sched_start": (C.c_int, [C.c_void_p, C.c_void_p, C.POINTER(SchedDecision)]),
    "memspec_sched_point": (C.c_int, [C.c_void_p, C.c_void_p, C.POINTER(SchedDecision)]),
    "memspec_sched_feedback": (C.c_int, [C.c_void_p, C.c_int32, C.c_int32, C.c_double]),
    "memspec_sched_get_stats": (C.c_int, [C.c_void_p, C.POINTER(SchedStats)]),
}

_lib = None


def load() -> C.CDLL:
    """Load libmemspec.so and declare every exported entry point."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise RuntimeError(
            f"{LIB_PATH} is missing: build it first (python -m paper_2608_10362_gb300.build). "
            "The speculative decoding path has no CPU fallback.")
    lib = C.CDLL(LIB_PATH)
    for name, (res, args) in EXPORTS.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    _lib = lib
    return lib


class MemSpecError(RuntimeError):
    def __init__(self, status: int, msg: str):
        name = STATUS_NAMES[status] if 0 <= status < len(STATUS_NAMES) else str(status)
        super().__init__(f"memspec {name}: {msg}")
        self.status = status
