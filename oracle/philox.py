"""Philox4x32-10 and the uniforms the speculative step draws (oracle side).

Test infrastructure only (see ``oracle/__init__``).

Philox4x32 follows Salmon et al., SC'11, Section 5: a 4 x 32-bit counter and a
2 x 32-bit key; each round multiplies two counter words by fixed constants,
mixes the high halves with the other words and the key, and the key is bumped
by the Weyl constants between rounds; ten rounds.

Uniform assignment (the speculative step draws K + K + 1 uniforms per request
per iteration):

* key     = (lo32(seed), hi32(seed))
* counter = (request, lo32(step), hi32(step), slot)
* slot j-1       -> draft sample x_j        (j = 1..K)
* slot K + i - 1 -> acceptance test of x_i  (i = 1..K)
* slot 2K        -> the resampled / bonus token
* u = (2 * (word0 >> 9) + 1) * 2^-24, an odd multiple of 2^-24 in (0, 1) that
  float32 and float64 both hold exactly.
"""
from __future__ import annotations

MASK32 = 0xFFFFFFFF
PHILOX_M0 = 0xD2511F53
PHILOX_M1 = 0xCD9E8D57
PHILOX_W0 = 0x9E3779B9
PHILOX_W1 = 0xBB67AE85


def _mulhilo(a: int, b: int):
    prod = (a * b) & 0xFFFFFFFFFFFFFFFF
    return prod >> 32, prod & MASK32


def philox4x32_10(counter, key):
    """Return the 4 output words of Philox4x32 with 10 rounds."""
    c0, c1, c2, c3 = (int(x) & MASK32 for x in counter)
    k0, k1 = (int(x) & MASK32 for x in key)
    for rnd in range(10):
        if rnd > 0:
            k0 = (k0 + PHILOX_W0) & MASK32
            k1 = (k1 + PHILOX_W1) & MASK32
        hi0, lo0 = _mulhilo(PHILOX_M0, c0)
        hi1, lo1 = _mulhilo(PHILOX_M1, c2)
        c0, c1, c2, c3 = hi1 ^ c1 ^ k0, lo1, hi0 ^ c3 ^ k1, lo0
    return c0, c1, c2, c3


def word_to_uniform(w: int) -> float:
    return float(2 * ((int(w) & MASK32) >> 9) + 1) * 2.0 ** -24


def uniform(seed: int, request: int, step: int, slot: int) -> float:
    key = (seed & MASK32, (seed >> 32) & MASK32)
    ctr = (request, step & MASK32, (step >> 32) & MASK32, slot)
    return word_to_uniform(philox4x32_10(ctr, key)[0])


def step_uniforms(seed: int, request: int, step: int, K: int):
    """(draft uniforms [K], acceptance uniforms [K], final-token uniform)."""
    u = [uniform(seed, request, step, s) for s in range(2 * K + 1)]
    return u[:K], u[K:2 * K], u[2 * K]
