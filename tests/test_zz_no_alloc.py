"""The GEMM entry point that allocates nothing (memspec_op_linear_noalloc).

It exists for callers that cannot allocate device memory (code running under
CUDA-graph capture, plug-ins whose host owns all device memory, fixed-budget
deployments): its split-K scratch is a fixed device array inside the library.
These tests check that it gives the same results as memspec_op_linear, on two
calls in a row (the array keeps the previous call's contents), and that sizes
beyond its fixed scratch are refused before anything runs.  This file is
collected last on purpose.
"""
import ctypes as C

import numpy as np
import pytest
import torch

from seeded_inputs import bf16_round


def _pair(seed, rows, n_out, k):
    rng = np.random.default_rng([seed, rows, n_out, k])
    x = bf16_round(rng.standard_normal((rows, k), dtype=np.float32))
    w = bf16_round((rng.standard_normal((n_out, k), dtype=np.float32) * 0.02).astype(np.float32))
    return x, w


@pytest.mark.gpu
@pytest.mark.parametrize("rows,n_out,k", [(1, 256, 128), (5, 4096, 4096), (16, 688, 256),
                                          (9, 32000, 768), (3, 2560, 2048)])
def test_noalloc_linear_matches_op_linear_twice(rows, n_out, k):
    from paper_2608_10362_gb300 import op_linear, op_linear_noalloc
    x, w = _pair(7, rows, n_out, k)
    xt = torch.from_numpy(x).to(torch.bfloat16).cuda()
    wt = torch.from_numpy(w).to(torch.bfloat16).cuda()
    ref = op_linear(xt, wt).cpu().numpy().astype(np.float64)
    bound = np.abs(x).astype(np.float64) @ np.abs(w).astype(np.float64).T
    for _ in range(2):
        y = op_linear_noalloc(xt, wt).cpu().numpy().astype(np.float64)
        assert np.all(np.abs(y - ref) <= 1e-4 * bound + 1e-6), np.abs(y - ref).max()


def test_noalloc_linear_refuses_sizes_beyond_its_scratch():
    from paper_2608_10362_gb300 import _lib
    lib = _lib.load()
    buf = C.create_string_buffer(64)
    p = C.cast(buf, C.c_void_p)
    # 17 rows exceed the fixed scratch: refused on the host, nothing enqueued
    assert lib.memspec_op_linear_noalloc(p, p, p, 17, 256, 256, None, None) == _lib.ERR_INVALID_ARG
    assert b"rows must be in 1..16" in lib.memspec_op_last_error()
    assert lib.memspec_op_linear_noalloc(p, p, p, 4, 131073, 256, None, None) == _lib.ERR_INVALID_ARG
    assert lib.memspec_op_linear_noalloc(p, p, p, 4, 256, 12, None, None) == _lib.ERR_INVALID_ARG
