"""Pins for the oracle's Philox4x32-10 and its uniform mapping (CPU only)."""
import os

import numpy as np
from scipy import stats

from oracle.philox import philox4x32_10, step_uniforms, uniform, word_to_uniform

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "philox4x32_10_kat.txt")


def _kat_rows():
    rows = []
    with open(GOLDEN) as f:
        for line in f:
            if line.startswith("#") or not line.strip():
                continue
            w = [int(t, 16) for t in line.split()]
            rows.append((w[0:4], w[4:6], w[6:10]))
    return rows


def test_philox_known_answer_vectors():
    rows = _kat_rows()
    assert len(rows) == 3
    for ctr, key, expect in rows:
        assert list(philox4x32_10(ctr, key)) == expect


def test_uniform_is_exact_in_float32_and_open_interval():
    for w in (0, 1, 511, 512, 0xFFFFFFFF, 0x80000000, 0x12345678):
        u = word_to_uniform(w)
        assert 0.0 < u < 1.0
        assert float(np.float32(u)) == u          # exactly representable in float32
    assert word_to_uniform(0) == 2.0 ** -24
    assert word_to_uniform(0xFFFFFFFF) == 1.0 - 2.0 ** -24


def test_uniform_chi_square_and_independence_of_slots():
    # 64 equiprobable bins over 20000 draws spread over requests/steps/slots
    us = np.array([uniform(7, r, s, k) for r in range(4) for s in range(250) for k in range(20)])
    counts, _ = np.histogram(us, bins=64, range=(0.0, 1.0))
    chi2 = ((counts - len(us) / 64) ** 2 / (len(us) / 64)).sum()
    assert chi2 < stats.chi2.ppf(1 - 1e-3, 63)
    # distinct (request, step, slot) counters give distinct streams
    assert len(set(us.tolist())) > 0.99 * len(us)


def test_step_uniform_slots():
    d, a, f = step_uniforms(3, 1, 5, 4)
    assert len(d) == 4 and len(a) == 4
    assert d[2] == uniform(3, 1, 5, 2)
    assert a[0] == uniform(3, 1, 5, 4)
    assert f == uniform(3, 1, 5, 8)
    # the 64-bit seed and step are split into two 32-bit words
    assert uniform(1 << 32, 0, 0, 0) != uniform(0, 0, 0, 0)
    assert uniform(0, 0, 1 << 32, 0) != uniform(0, 0, 0, 0)
