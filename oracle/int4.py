"""Group-wise INT4 weight-only linear layer (oracle side).

Test infrastructure only (see ``oracle/__init__``).

MemSpec's targets are GPTQ INT4 models (Section 4.1; Section 2.1 evaluates a
GPTQ INT4 LLaMA-2 7B): each weight is a 4-bit code q in 0..15, and every group of
g consecutive inputs of an output row shares a scale s and a zero point z, so the
weight the layer multiplies by is w = (q - z) * s.  The layer is then the plain
product y = x W^T.

Storage (the CUDA path reads the same bytes):
* qweight uint8 [n][k/2]: byte j of row r holds q[r][2j] in its low nibble and
  q[r][2j+1] in its high nibble;
* scales [n][k/g] (bf16 values), zeros uint8 [n][k/g] (0..15).
"""
from __future__ import annotations

import numpy as np


def unpack(qweight: np.ndarray) -> np.ndarray:
    """uint8 [n][k/2] -> int64 codes [n][k] (low nibble first)."""
    qb = np.asarray(qweight, dtype=np.uint8)
    n, half = qb.shape
    q = np.empty((n, 2 * half), dtype=np.int64)
    q[:, 0::2] = qb & 0x0F
    q[:, 1::2] = qb >> 4
    return q


def dequant(qweight, scales, zeros, group: int) -> np.ndarray:
    """w[r][c] = (q[r][c] - z[r][c // g]) * s[r][c // g], float64 [n][k]."""
    q = unpack(qweight)
    s = np.repeat(np.asarray(scales, dtype=np.float64), group, axis=1)
    z = np.repeat(np.asarray(zeros, dtype=np.int64), group, axis=1)
    return (q - z).astype(np.float64) * s


def linear_int4(x, qweight, scales, zeros, group: int) -> np.ndarray:
    """y[m][r] = sum_c x[m][c] w[r][c] in float64."""
    return np.asarray(x, dtype=np.float64) @ dequant(qweight, scales, zeros, group).T
