"""The INT4 oracle pinned to what the format and the arithmetic fix: a packed
byte worked by hand, the dequantisation of hand-picked codes, the special case
where it reduces to integer matrix arithmetic, and the linear map against an
independent dense product of the dequantised weights."""
import numpy as np

from oracle.int4 import dequant, linear_int4, unpack
from seeded_inputs import gen_int4_weights


def test_unpack_low_nibble_first():
    qb = np.array([[0x21, 0xF0], [0x0E, 0x7B]], dtype=np.uint8)
    np.testing.assert_array_equal(unpack(qb), [[1, 2, 0, 15], [14, 0, 11, 7]])


def test_dequant_by_hand():
    # one row, k = 8, group 4: codes 0..7, scales (0.5, 2), zeros (3, 5)
    q = np.arange(8)
    qb = (q[0::2] | (q[1::2] << 4)).astype(np.uint8)[None, :]
    w = dequant(qb, np.array([[0.5, 2.0]]), np.array([[3, 5]], dtype=np.uint8), 4)
    np.testing.assert_array_equal(w, [[-1.5, -1.0, -0.5, 0.0, -2.0, 0.0, 2.0, 4.0]])


def test_unit_scales_reduce_to_integer_matmul():
    packed, _, zeros = gen_int4_weights(3, 16, 256, 128)
    q = unpack(packed)
    z = np.repeat(zeros.astype(np.int64), 128, axis=1)
    x = np.random.default_rng(4).integers(-20, 20, size=(3, 256))
    y = linear_int4(x, packed, np.ones((16, 2)), zeros, 128)
    np.testing.assert_array_equal(y, (x @ (q - z).T).astype(np.float64))


def test_linear_matches_a_dense_product_elementwise():
    packed, scales, zeros = gen_int4_weights(5, 24, 384, 128)
    x = np.random.default_rng(6).standard_normal((2, 384))
    w = np.empty((24, 384))
    q = unpack(packed)
    for r in range(24):
        for c in range(384):
            w[r, c] = (q[r, c] - int(zeros[r, c // 128])) * float(scales[r, c // 128])
    ref = np.einsum("mc,rc->mr", x, w)
    np.testing.assert_allclose(linear_int4(x, packed, scales, zeros, 128), ref, rtol=1e-12, atol=1e-12)
