"""Group-wise INT4 weight-only linear layer (the paper's GPTQ INT4 targets,
Section 4.1) through the C ABI: memspec_int4_pack's layout byte for byte
against a NumPy restatement of the documented record layout, and
memspec_op_linear_int4 against the oracle's fp64 dequantise-then-matmul
(oracle.int4.linear_int4) on seeded GPTQ-style weights.

Tolerance.  The kernel feeds each code to the MMA as the exact bf16 value
128 + q, so a group's fp32 accumulator sums 128 exact products
x_c (128 + q_c); the zero point is folded out afterwards with the group sum of
x.  fp32 summation of 128 terms errs by at most 128 u sum|terms| (u = 2^-24),
so per output
    |y - y_ref| <= 128 u sum_c s_c |x_c| (128 + q_c + 128 + z_c) + 8 u sum_c |x_c w_c|,
the second term covering the epilogue's few roundings over the groups."""
import ctypes as C

import numpy as np
import pytest
import torch

from oracle.int4 import dequant, linear_int4, unpack
from seeded_inputs import bf16_round, gen_int4_weights

U = 2.0 ** -24
REC = 1072


def _bound(x, qweight, scales, zeros):
    q = unpack(qweight).astype(np.float64)
    s = np.repeat(scales.astype(np.float64), 128, axis=1)
    z = np.repeat(zeros.astype(np.float64), 128, axis=1)
    ax = np.abs(x.astype(np.float64))
    bias = ax @ (s * (256.0 + q + z)).T
    absw = ax @ np.abs(dequant(qweight, scales, zeros, 128)).T
    return 128 * U * bias + 8 * U * absw + 1e-30


def _device(qweight, scales, zeros):
    return (torch.from_numpy(qweight).cuda(), torch.from_numpy(scales).to(torch.bfloat16).cuda(),
            torch.from_numpy(zeros).cuda())


def _x(seed, rows, k):
    rng = np.random.default_rng([seed, rows, k])
    return bf16_round(rng.standard_normal((rows, k), dtype=np.float32))


def _pack_reference(qweight, scales, zeros):
    """The record layout written out from its definition (16-row tiles x
    128-column groups, tile-major; lane L = 4 r + t holds the words at column
    offsets 32 j + 8 t of rows r and r + 8, each word's codes of columns
    e = 0..7 moved to nibble positions 0 4 1 5 2 6 3 7; then the (s[r], s[r+8])
    bf16 pairs and the (z[r], z[r+8]) byte pairs)."""
    n, half = qweight.shape
    k = 2 * half
    G, tiles = k // 128, (n + 15) // 16
    qw = np.zeros((tiles * 16, half), np.uint8)
    qw[:n] = qweight
    sb = np.zeros((tiles * 16, G), np.uint16)
    sb[:n] = (scales.astype(np.float32).view(np.uint32) >> 16).astype(np.uint16)
    zb = np.zeros((tiles * 16, G), np.uint8)
    zb[:n] = zeros
    out = np.zeros((tiles, G, REC), np.uint8)
    for T in range(tiles):
        for g in range(G):
            rec = out[T, g]
            for h in range(2):
                for lane in range(32):
                    r, t = divmod(lane, 4)
                    row = T * 16 + 8 * h + r
                    for j in range(4):
                        o = g * 64 + 16 * j + 4 * t
                        word = int.from_bytes(qw[row, o:o + 4].tobytes(), "little")
                        moved = 0
                        for e in range(8):
                            moved |= ((word >> (4 * e)) & 15) << (4 * [0, 4, 1, 5, 2, 6, 3, 7][e])
                        rec[h * 512 + lane * 16 + 4 * j: h * 512 + lane * 16 + 4 * j + 4] = \
                            np.frombuffer(moved.to_bytes(4, "little"), np.uint8)
            pairs = np.stack([sb[T * 16:T * 16 + 8, g], sb[T * 16 + 8:T * 16 + 16, g]], axis=1)
            rec[1024:1056] = np.frombuffer(pairs.astype("<u2").tobytes(), np.uint8)
            zp = np.stack([zb[T * 16:T * 16 + 8, g], zb[T * 16 + 8:T * 16 + 16, g]], axis=1)
            rec[1056:1072] = zp.reshape(-1)
    return out.reshape(-1)


@pytest.mark.gpu
@pytest.mark.parametrize("n,k", [(16, 128), (40, 384), (33, 256), (70, 640)])
def test_pack_layout_byte_for_byte(n, k):
    from paper_2608_10362_gb300 import int4_pack
    qw, sc, zs = gen_int4_weights(1, n, k)
    got = int4_pack(*_device(qw, sc, zs)).cpu().numpy()
    assert np.array_equal(got, _pack_reference(qw, sc, zs))


@pytest.mark.gpu
@pytest.mark.parametrize("rows,n,k", [(1, 16, 128), (5, 40, 384), (11, 33, 256), (3, 70, 640), (16, 520, 1024),
                                      (8, 1000, 2048), (9, 4096, 512), (5, 4096, 4096), (1, 4096, 4096),
                                      (5, 1024, 11008), (2, 3, 128)])
def test_int4_linear_matches_oracle(rows, n, k):
    from paper_2608_10362_gb300 import int4_pack, op_linear_int4
    qw, sc, zs = gen_int4_weights(2, n, k)
    x = _x(3, rows, k)
    packed = int4_pack(*_device(qw, sc, zs))
    xt = torch.from_numpy(x).to(torch.bfloat16).cuda()
    y = torch.full((rows, n), float("nan"), device="cuda")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    op_linear_int4(xt, packed, n, y=y, status=status)
    assert int(status.item()) == 0
    got = y.cpu().numpy().astype(np.float64)
    ref = linear_int4(x, qw, sc, zs, 128)
    bound = _bound(x, qw, sc, zs)
    assert np.all(np.isfinite(got))
    err = np.abs(got - ref)
    assert np.all(err <= bound), (err.max(), (err / bound).max())
    # the same call again: bit-identical (fixed summation orders)
    y2 = op_linear_int4(xt, packed, n)
    assert torch.equal(y, y2)


@pytest.mark.gpu
@pytest.mark.parametrize("rows,n,k", [(5, 12288, 4096), (5, 22016, 4096), (5, 4096, 11008), (16, 32000, 4096)])
def test_int4_linear_full_size_sampled_rows(rows, n, k):
    """7B-sized projections (and an LM-head-sized one at 16 rows): every output
    finite, and the outputs of 256 sampled weight rows against the oracle."""
    from paper_2608_10362_gb300 import int4_pack, op_linear_int4
    qw, sc, zs = gen_int4_weights(4, n, k)
    x = _x(5, rows, k)
    got = op_linear_int4(torch.from_numpy(x).to(torch.bfloat16).cuda(), int4_pack(*_device(qw, sc, zs)), n)
    got = got.cpu().numpy().astype(np.float64)
    assert np.all(np.isfinite(got))
    idx = np.unique(np.concatenate([np.random.default_rng(6).choice(n, 250, replace=False),
                                    [0, 15, 16, n - 17, n - 16, n - 1]]))
    ref = linear_int4(x, qw[idx], sc[idx], zs[idx], 128)
    bound = _bound(x, qw[idx], sc[idx], zs[idx])
    assert np.all(np.abs(got[:, idx] - ref) <= bound)


@pytest.mark.gpu
def test_int4_integer_case_is_exact():
    """Scale 1, small integer activations: every product and partial sum is an
    integer below 2^24, so the result is exact."""
    from paper_2608_10362_gb300 import int4_pack, op_linear_int4
    rows, n, k = 5, 96, 512
    qw, _, zs = gen_int4_weights(8, n, k)
    sc = np.ones((n, k // 128), np.float32)
    x = np.random.default_rng(9).integers(-3, 4, size=(rows, k)).astype(np.float32)
    got = op_linear_int4(torch.from_numpy(x).to(torch.bfloat16).cuda(), int4_pack(*_device(qw, sc, zs)), n)
    ref = linear_int4(x, qw, sc, zs, 128)
    assert np.array_equal(got.cpu().numpy().astype(np.float64), ref)


def test_int4_entry_points_refuse_bad_arguments():
    """Checked before anything is enqueued (no GPU needed)."""
    from paper_2608_10362_gb300 import _lib
    lib = _lib.load()
    buf = C.create_string_buffer(4096 + 16)
    base = (C.addressof(buf) + 15) & ~15
    p = C.c_void_p(base)
    assert lib.memspec_int4_packed_bytes(16, 100) == -1
    assert lib.memspec_int4_packed_bytes(0, 128) == -1
    assert lib.memspec_int4_packed_bytes(17, 256) == 2 * 2 * REC
    bad = [(p, p, p, 0, 128, 128), (p, p, p, 17, 128, 128), (p, p, p, 1, 128, 100), (p, p, p, 1, 0, 128),
           (C.c_void_p(base + 8), p, p, 1, 128, 128), (None, p, p, 1, 128, 128)]
    for x, w, y, rows, n, k in bad:
        assert lib.memspec_op_linear_int4(x, w, y, rows, n, k, None, None) == _lib.ERR_INVALID_ARG
    # 16 rows of k = 8192 need more shared memory than the kernel may use
    assert lib.memspec_op_linear_int4(p, p, p, 16, 128, 8192, None, None) == _lib.ERR_UNSUPPORTED
    assert lib.memspec_int4_pack(p, p, p, 16, 100, p, None) == _lib.ERR_INVALID_ARG
    assert lib.memspec_int4_pack(p, p, p, 16, 128, C.c_void_p(base + 4), None) == _lib.ERR_INVALID_ARG
