"""Pins for the oracle's speculative-sampling step (CPU only).

The pins are properties that the speculative sampling papers prove and that a
plausible slip (wrong residual, wrong comparison, missing bonus token, wrong
rollback length) breaks: greedy speculative decoding reproduces greedy target
decoding token for token; a draft equal to the target is always accepted;
emitted tokens follow the target distribution (chi-square); the acceptance
probability is sum_x min(p, q) and the tokens per iteration follow
(1 - a^(K+1)) / (1 - a).
"""
import numpy as np
import pytest
from scipy import stats

from oracle.llama import LlamaOracle
from oracle.speculative import (SpecDecoder, accept, greedy_generate, sample_inverse_cdf,
                                softmax_t, speculative_generate)
from seeded_inputs import SHAPES, gen_prompt, gen_weights

CHI2_CRIT_63 = stats.chi2.ppf(1 - 1e-3, 63)      # 103.44


@pytest.fixture(scope="module")
def tiny_pair():
    t, d = SHAPES["tiny_target"], SHAPES["tiny_draft"]
    return LlamaOracle(t, gen_weights(t, 0)), LlamaOracle(d, gen_weights(d, 1))


def test_inverse_cdf_sampler():
    w = np.array([0.0, 2.0, 0.0, 1.0, 1.0])
    assert sample_inverse_cdf(w, 1e-9) == 1          # zero-mass ids are skipped
    assert sample_inverse_cdf(w, 0.4999) == 1
    assert sample_inverse_cdf(w, 0.5) == 3           # boundary belongs to the next id
    assert sample_inverse_cdf(w, 1 - 1e-9) == 4
    rng = np.random.default_rng(0)
    p = rng.dirichlet(np.ones(64))
    draws = [sample_inverse_cdf(p * 3.7, u) for u in rng.random(50000)]   # unnormalised weights
    counts = np.bincount(draws, minlength=64)
    chi2 = ((counts - 50000 * p) ** 2 / (50000 * p)).sum()
    assert chi2 < CHI2_CRIT_63


@pytest.mark.parametrize("K", [1, 3, 4])
def test_greedy_speculative_equals_greedy_target(tiny_pair, K):
    target, draft = tiny_pair
    prompt = gen_prompt(2, 128, 2048)
    spec, recs = speculative_generate(target, draft, prompt, 24, K, 0.0)
    assert spec == greedy_generate(target, prompt, 24)
    assert all(0 <= r.result.n_accepted <= K for r in recs)


def test_draft_equal_to_target_accepts_everything(tiny_pair):
    target, _ = tiny_pair
    prompt = gen_prompt(3, 40, 2048)
    for T in (1.0, 0.0):
        _, recs = speculative_generate(target, target, prompt, 20, 4, T, seed=5)
        assert all(r.result.n_accepted == 4 for r in recs)


def test_rollback_lengths(tiny_pair):
    target, draft = tiny_pair
    sd = SpecDecoder(target, draft, gen_prompt(4, 30, 2048), 80)
    for step in range(6):
        L = sd.L
        rec = sd.step(4, 1.0, 9, 0, step)
        n = rec.result.n_accepted
        assert sd.L == L + n + 1
        assert sd.tc.length == sd.L - 1
        assert sd.dc.length == (sd.L - 1 if n < 4 else sd.L - 2)


def _context_free_run(p, q, K, n_trials, rng, n_tokens):
    """SD with position-independent target p and draft q (a context-free model):
    the first n_tokens emitted tokens of each trial."""
    V = len(p)
    zt = np.log(np.tile(p, (K + 1, 1)))
    zd = np.log(np.tile(q, (K, 1)))
    out = np.zeros((n_trials, n_tokens), dtype=np.int64)
    iters = 0
    for t in range(n_trials):
        toks = []
        while len(toks) < n_tokens:
            x = [sample_inverse_cdf(q, u) for u in rng.random(K)]
            r = accept(zt, zd, x, 1.0, rng.random(K), rng.random())
            toks += x[:r.n_accepted] + [r.token]
            iters += 1
        out[t] = toks[:n_tokens]
    return out, iters


def test_emitted_tokens_follow_target_distribution():
    rng = np.random.default_rng(12)
    V = 64
    p = rng.dirichlet(np.full(V, 0.7))
    q = rng.dirichlet(np.full(V, 0.7))
    toks, _ = _context_free_run(p, q, 3, 100000, rng, 2)
    for col in range(2):        # first token (accept / resample) and second (incl. bonus)
        counts = np.bincount(toks[:, col], minlength=V)
        exp = 100000 * p
        chi2 = ((counts - exp) ** 2 / exp).sum()
        assert chi2 < CHI2_CRIT_63, (col, chi2)


def test_emitted_pairs_are_independent_draws_from_target():
    rng = np.random.default_rng(13)
    V = 8
    p = rng.dirichlet(np.ones(V))
    q = rng.dirichlet(np.ones(V))
    toks, _ = _context_free_run(p, q, 2, 100000, rng, 2)
    counts = np.bincount(toks[:, 0] * V + toks[:, 1], minlength=V * V)
    exp = 100000 * np.outer(p, p).ravel()
    chi2 = ((counts - exp) ** 2 / exp).sum()
    assert chi2 < CHI2_CRIT_63


def test_acceptance_rate_and_tokens_per_iteration_closed_forms():
    rng = np.random.default_rng(14)
    V, K, N = 32, 4, 20000
    p = rng.dirichlet(np.ones(V))
    q = rng.dirichlet(np.ones(V))
    alpha = np.minimum(p, q).sum()
    zt = np.log(np.tile(p, (K + 1, 1)))
    zd = np.log(np.tile(q, (K, 1)))
    acc1, total = 0, 0
    for _ in range(N):
        x = [sample_inverse_cdf(q, u) for u in rng.random(K)]
        r = accept(zt, zd, x, 1.0, rng.random(K), rng.random())
        acc1 += r.n_accepted >= 1
        total += r.n_accepted + 1
    se = np.sqrt(alpha * (1 - alpha) / N)
    assert abs(acc1 / N - alpha) < 5 * se
    expect = (1 - alpha ** (K + 1)) / (1 - alpha)
    assert abs(total / N - expect) < 5 * 1.5 / np.sqrt(N)


def test_zero_residual_falls_back_to_target():
    p = np.array([0.5, 0.25, 0.25])
    z = np.log(np.stack([p, p]))
    # u > 1 cannot happen with real uniforms; it forces the rejection branch
    r = accept(z, z[:1], [0], 1.0, [1.5], 0.6)
    assert r.n_accepted == 0 and r.residual_mass == 0.0
    assert r.token == sample_inverse_cdf(p, 0.6)


def test_greedy_acceptance_rule():
    zt = np.array([[0.0, 3.0, 1.0], [2.0, 2.0, 0.0], [0.0, 0.0, 5.0]])
    r = accept(zt, np.zeros((2, 3)), [1, 0], 0.0, None, None)
    assert (r.n_accepted, r.token) == (2, 2)          # ties go to the lowest id
    r = accept(zt, np.zeros((2, 3)), [1, 1], 0.0, None, None)
    assert (r.n_accepted, r.token) == (1, 0)
    r = accept(zt, np.zeros((2, 3)), [2, 1], 0.0, None, None)
    assert (r.n_accepted, r.token) == (0, 1)


def test_temperature_scales_both_models():
    z = np.array([[1.0, 2.0, 3.0]])
    np.testing.assert_allclose(softmax_t(z, 0.5), softmax_t(2 * z, 1.0), rtol=1e-15)
