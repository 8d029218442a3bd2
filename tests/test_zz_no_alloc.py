"""The GEMM entry point that allocates nothing (memspec_op_linear_noalloc).

Some callers cannot allocate device memory: plug-ins whose host application
owns all of it, fixed-budget deployments that allocate only at start-up, and
latency-critical loops that cannot afford cudaMalloc.  For them the library
keeps this GEMM's split-K scratch in a fixed device array of its own.  These
tests check, through the C ABI, that two calls in a row (the array keeps the
previous call's contents) give y = x . w^T within the GEMM tolerance of the
fp64 matmul of the same bf16 inputs, agree with memspec_op_linear within that
tolerance, leave the error word at zero, and that sizes beyond the fixed
scratch are refused before anything runs.  This file is collected last on
purpose.
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
                                          (9, 32000, 768), (3, 2560, 2048), (2, 130, 72)])
def test_noalloc_linear_matches_fp64_matmul_twice(rows, n_out, k):
    from paper_2608_10362_gb300 import op_linear, op_linear_noalloc
    x, w = _pair(7, rows, n_out, k)
    xt = torch.from_numpy(x).to(torch.bfloat16).cuda()
    wt = torch.from_numpy(w).to(torch.bfloat16).cuda()
    ref = x.astype(np.float64) @ w.astype(np.float64).T
    # fp32 accumulation of exact bf16 products: |y - ref| <= 1e-4 * sum_k |x_k w_k|
    bound = np.abs(x).astype(np.float64) @ np.abs(w).astype(np.float64).T
    other = op_linear(xt, wt).cpu().numpy().astype(np.float64)
    assert np.all(np.abs(other - ref) <= 1e-4 * bound + 1e-6)
    y = torch.empty(rows, n_out, dtype=torch.float32, device="cuda")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    for call in range(2):
        y.fill_(float("nan"))                 # every output element must be written
        op_linear_noalloc(xt, wt, y=y, status=status)
        torch.cuda.synchronize()
        assert int(status.item()) == 0, f"call {call}: device error bits {int(status.item()):#x}"
        got = y.cpu().numpy().astype(np.float64)
        assert np.all(np.isfinite(got)), call
        assert np.all(np.abs(got - ref) <= 1e-4 * bound + 1e-6), (call, np.abs(got - ref).max())
        assert np.all(np.abs(got - other) <= 2e-4 * bound + 2e-6), call


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
