"""Draft-then-verify speculative decoding step, float64 (oracle side).

Test infrastructure only (see ``oracle/__init__``).

MemSpec runs the standard draft-and-verify iteration (Section 3.5) and models
throughput as E[A] / L_iter (Section 2.1, Eq. 1).  The acceptance rule is the
one of the speculative sampling papers it cites (Leviathan et al., ICML 2023,
Algorithm 1; Chen et al. 2023, Algorithm 2):

1. the draft proposes x_1..x_K, x_i ~ q_i, autoregressively;
2. the target scores the K+1 positions [t_{L-1}, x_1..x_K] in one pass,
   giving p_1..p_{K+1};
3. for i = 1..K, with u_i ~ U(0,1): x_i is accepted iff u_i <= p_i(x_i) / q_i(x_i)
   (evaluated as u_i * q_i(x_i) <= p_i(x_i)); stop at the first rejection; n =
   number accepted;
4. if n < K, one token is drawn from norm(max(0, p_{n+1} - q_{n+1})); if n = K,
   one token is drawn from p_{K+1};
5. the committed sequence grows by x_1..x_n and that token; KV entries of the
   rejected positions are dropped (rollback).

Temperature T > 0 applies to both models: p = softmax(z_target / T),
q = softmax(z_draft / T).  T = 0 is greedy: x_i = argmax q_i, x_i is accepted
iff it equals argmax p_i, the final token is argmax p_{n+1}.  Ties in argmax go
to the lowest token id.  Sampling from a categorical distribution w (not
necessarily normalised) with uniform u takes the smallest id j with
sum_{k<=j} w_k > u * sum_k w_k.  If the residual max(0, p - q) has zero mass
(possible only when p == q up to rounding), the final token is drawn from p.
"""
from __future__ import annotations

import dataclasses

import numpy as np

from .philox import step_uniforms


def softmax_t(z: np.ndarray, T: float) -> np.ndarray:
    """softmax(z / T) along the last axis, float64."""
    z = np.asarray(z, dtype=np.float64) / T
    e = np.exp(z - z.max(axis=-1, keepdims=True))
    return e / e.sum(axis=-1, keepdims=True)


def argmax_first(z: np.ndarray) -> int:
    """Index of the maximum, lowest index on ties (numpy's argmax already is)."""
    return int(np.argmax(np.asarray(z)))


def sample_inverse_cdf(w: np.ndarray, u: float) -> int:
    """Smallest j with cumsum(w)[j] > u * sum(w)."""
    w = np.asarray(w, dtype=np.float64)
    c = np.cumsum(w)
    j = int(np.searchsorted(c, u * c[-1], side="right"))
    return min(j, len(w) - 1)


def draft_token(z_draft_row: np.ndarray, T: float, u: float) -> int:
    if T == 0.0:
        return argmax_first(z_draft_row)
    return sample_inverse_cdf(softmax_t(z_draft_row, T), u)


@dataclasses.dataclass
class AcceptResult:
    n_accepted: int
    token: int                # correction (n < K) or bonus (n == K) token
    p_of_x: np.ndarray        # p_i(x_i), i = 1..K (T > 0), else empty
    q_of_x: np.ndarray        # q_i(x_i)
    residual_mass: float      # sum max(0, p_{n+1} - q_{n+1}) (1.0 when n == K)


def accept(z_target: np.ndarray, z_draft: np.ndarray, x, T: float,
           u_accept, u_final: float) -> AcceptResult:
    """Speculative-sampling acceptance for one request.

    z_target: [K+1, V] target logits for positions L .. L+K (rows 1..K+1)
    z_draft:  [K, V] draft logits that x_1..x_K were drawn from
    x:        K draft tokens
    """
    x = [int(t) for t in x]
    K = len(x)
    if T == 0.0:
        n = 0
        while n < K and x[n] == argmax_first(z_target[n]):
            n += 1
        return AcceptResult(n, argmax_first(z_target[n]), np.zeros(0), np.zeros(0), 1.0)
    p = softmax_t(z_target, T)
    q = softmax_t(z_draft, T)
    px = np.array([p[i, x[i]] for i in range(K)])
    qx = np.array([q[i, x[i]] for i in range(K)])
    n = 0
    while n < K and u_accept[n] * qx[n] <= px[n]:
        n += 1
    if n == K:
        return AcceptResult(n, sample_inverse_cdf(p[K], u_final), px, qx, 1.0)
    r = np.maximum(p[n] - q[n], 0.0)
    mass = float(r.sum())
    if mass <= 0.0:
        return AcceptResult(n, sample_inverse_cdf(p[n], u_final), px, qx, 0.0)
    return AcceptResult(n, sample_inverse_cdf(r, u_final), px, qx, mass)


@dataclasses.dataclass
class StepRecord:
    L: int                    # committed length before the step
    draft_tokens: list
    z_draft: np.ndarray       # [K, V]
    z_target: np.ndarray      # [K+1, V]
    result: AcceptResult


class SpecDecoder:
    """Target + draft with their KV caches and the committed token sequence."""

    def __init__(self, target, draft, prompt, capacity: int):
        self.target, self.draft = target, draft
        self.tokens = [int(t) for t in prompt]
        self.tc = target.new_cache(capacity)
        self.dc = draft.new_cache(capacity)
        # every committed token except the last one is processed by both models
        target.forward(self.tc, self.tokens[:-1], want_logits=False)
        draft.forward(self.dc, self.tokens[:-1], want_logits=False)

    @property
    def L(self) -> int:
        return len(self.tokens)

    def propose(self, K: int, T: float, u_draft, forced=None):
        """Draft x_1..x_K.  ``forced`` (optional) overrides the drafted tokens
        one by one (used to follow another implementation's choices)."""
        L = self.L
        feed = self.tokens[self.dc.length:L]          # 1 token, or 2 after full acceptance
        xs, zs = [], []
        for j in range(K):
            z = self.draft.forward(self.dc, feed)[-1]
            xj = draft_token(z, T, u_draft[j] if T > 0 else 0.0)
            if forced is not None:
                xj = int(forced[j])
            xs.append(xj)
            zs.append(z)
            feed = [xj]
        # x_K is never fed: the draft cache now ends at position L+K-2
        return xs, np.stack(zs)

    def verify(self, xs):
        """Target logits for positions L..L+K from one pass over [t_{L-1}, x_1..x_K]."""
        return self.target.forward(self.tc, [self.tokens[-1]] + list(xs))

    def commit(self, xs, n: int, token: int):
        """Append x_1..x_n and the final token; roll back rejected KV entries."""
        L, K = self.L, len(xs)
        self.tc.truncate(L + n)                       # t_{L-1}, x_1..x_n stay
        self.dc.truncate(min(L + n, L + K - 1))
        self.tokens += [int(t) for t in xs[:n]] + [int(token)]

    def step(self, K: int, T: float, seed: int, request: int, step: int) -> StepRecord:
        u_d, u_a, u_f = step_uniforms(seed, request, step, K)
        L = self.L
        xs, zd = self.propose(K, T, u_d)
        zt = self.verify(xs)
        res = accept(zt, zd, xs, T, u_a, u_f)
        self.commit(xs, res.n_accepted, res.token)
        return StepRecord(L, xs, zd, zt, res)


def speculative_generate(target, draft, prompt, n_new: int, K: int, T: float,
                         seed: int = 0, request: int = 0):
    """Run iterations until at least n_new tokens are committed.

    Returns (generated tokens truncated to n_new, list of StepRecord)."""
    sd = SpecDecoder(target, draft, prompt, len(prompt) + n_new + K + 2)
    records = []
    step = 0
    while sd.L - len(prompt) < n_new:
        records.append(sd.step(K, T, seed, request, step))
        step += 1
    return sd.tokens[len(prompt):len(prompt) + n_new], records


def greedy_generate(model, prompt, n_new: int):
    """Plain greedy autoregressive decoding with one model."""
    cache = model.new_cache(len(prompt) + n_new + 1)
    z = model.forward(cache, prompt)[-1]
    out = []
    for _ in range(n_new):
        t = argmax_first(z)
        out.append(t)
        z = model.forward(cache, [t])[-1]
    return out
