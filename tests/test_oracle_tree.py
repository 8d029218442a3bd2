"""Pins for the oracle's tree verification (oracle/tree.py), CPU only.

* The per-path definition of the tree rows against an independent
  formulation: one pass over all nodes with a tree attention mask (each node
  sees the prefix, its ancestors and itself), built from torch's
  scaled_dot_product_attention with an explicit boolean mask and the
  node's own RoPE position.
* The walk against hand-worked greedy cases, against the target distribution
  (chi-square on the first emitted token and on the second one given each
  accepted child), and against the closed form of E[accepted nodes] (sum
  over nodes of the product of the target probabilities along the path).
"""
import math

import numpy as np
import pytest
import torch
import torch.nn.functional as F

from oracle.llama import LlamaOracle, apply_rope, rmsnorm, silu
from oracle.speculative import softmax_t
from oracle.tree import (accept_tree, children, path_tokens, reach_probabilities, tree_depths,
                         tree_logits)
from seeded_inputs import ModelShape, gen_weights

SHAPE = ModelShape(2, 64, 4, 2, 16, 96, 53)
#          0   1  2  3  4  5  6   (node)
TREE_P = [-1, -1, 0, 0, 2, 1, 4]
TREE_X = [5, 9, 7, 11, 3, 5, 8]


def test_depths_paths_and_children_by_hand():
    assert tree_depths(TREE_P) == [0, 0, 1, 1, 2, 1, 3]
    assert path_tokens(TREE_X, TREE_P, 6) == [5, 7, 3, 8]
    assert path_tokens(TREE_X, TREE_P, 5) == [9, 5]
    assert children(TREE_P, 0) == [0, 1]          # row 0 = the root
    assert children(TREE_P, 1) == [2, 3]          # row 1 = node 0
    assert children(TREE_P, 7) == []              # node 6 is a leaf
    with pytest.raises(ValueError):
        tree_depths([-1, 1])                      # a parent must precede its child
    with pytest.raises(ValueError):
        tree_depths([-2])


def _masked_tree_pass(model, shape, prompt, root, tokens, parents):
    """All tree rows in one pass: prefix K/V from a plain forward, then the
    root and the nodes together with a tree mask (torch SDPA)."""
    w = model.w
    cache = model.new_cache(len(prompt) + len(tokens) + 2)
    model.forward(cache, prompt, want_logits=False)
    L0 = cache.length
    depths = tree_depths(parents)
    rows_tok = [root] + list(tokens)
    pos = np.array([L0] + [L0 + 1 + d for d in depths])
    n = len(rows_tok)
    vis = np.zeros((n, n), dtype=bool)             # row -> rows it sees
    for r in range(n):
        vis[r, 0] = True
        vis[r, r] = True
        i = r - 1
        while i >= 0:
            vis[r, i + 1] = True
            i = parents[i]
    mask = np.concatenate([np.ones((n, L0), dtype=bool), vis], axis=1)
    h = w[("tok_emb", -1)][np.array(rows_tok)].astype(np.float64)
    g = shape.n_heads // shape.n_kv_heads
    for li in range(shape.n_layers):
        a = rmsnorm(h, w[("attn_norm", li)], shape.norm_eps)
        q = (a @ w[("wq", li)].astype(np.float64).T).reshape(n, shape.n_heads, shape.head_dim)
        k = (a @ w[("wk", li)].astype(np.float64).T).reshape(n, shape.n_kv_heads, shape.head_dim)
        v = (a @ w[("wv", li)].astype(np.float64).T).reshape(n, shape.n_kv_heads, shape.head_dim)
        q = apply_rope(q, pos, shape.rope_base)
        k = apply_rope(k, pos, shape.rope_base)
        # the cache holds bf16 K / V (as the oracle's layer stores them)
        kk = np.concatenate([cache.k[li, :L0], _bf16(k)], axis=0)
        vv = np.concatenate([cache.v[li, :L0], _bf16(v)], axis=0)
        qt = torch.from_numpy(q).permute(1, 0, 2)
        kt = torch.from_numpy(kk).repeat_interleave(g, dim=1).permute(1, 0, 2)
        vt = torch.from_numpy(vv).repeat_interleave(g, dim=1).permute(1, 0, 2)
        o = F.scaled_dot_product_attention(qt, kt, vt, attn_mask=torch.from_numpy(mask))
        o = o.permute(1, 0, 2).reshape(n, shape.q_dim).numpy()
        h = h + o @ w[("wo", li)].astype(np.float64).T
        m = rmsnorm(h, w[("ffn_norm", li)], shape.norm_eps)
        act = silu(m @ w[("w_gate", li)].astype(np.float64).T) * (m @ w[("w_up", li)].astype(np.float64).T)
        h = h + act @ w[("w_down", li)].astype(np.float64).T
    return model.logits(h)


def _bf16(x):
    from oracle.llama import bf16
    return bf16(x)


def test_tree_rows_equal_one_tree_masked_pass():
    weights = gen_weights(SHAPE, 3)
    model = LlamaOracle(SHAPE, weights, keep_f64=True)
    prompt = [1, 4, 9, 16, 25, 36, 2, 3, 7]
    cache = model.new_cache(64)
    model.forward(cache, prompt, want_logits=False)
    rows = tree_logits(model, cache, 44, TREE_X, TREE_P)
    assert cache.length == len(prompt)            # every path was cut back
    ref = _masked_tree_pass(model, SHAPE, prompt, 44, TREE_X, TREE_P)
    np.testing.assert_allclose(rows, ref, rtol=1e-10, atol=1e-10)


def test_chain_tree_rows_equal_one_forward():
    weights = gen_weights(SHAPE, 4)
    model = LlamaOracle(SHAPE, weights, keep_f64=True)
    prompt = [3, 1, 4, 1, 5]
    chain_x, chain_p = [9, 2, 6, 5], [-1, 0, 1, 2]
    cache = model.new_cache(32)
    model.forward(cache, prompt, want_logits=False)
    rows = tree_logits(model, cache, 8, chain_x, chain_p)
    full = model.forward(cache, [8] + chain_x)
    np.testing.assert_allclose(rows, full, rtol=1e-12, atol=1e-12)


def _onehot_rows(n, V, best):
    z = np.zeros((n, V))
    for r, b in enumerate(best):
        z[r, b] = 5.0
    return z


def test_greedy_walks_by_hand():
    V = 16
    # root -> 9 (node 1) -> 5 (node 5, a leaf) -> final token from node 5's row
    z = _onehot_rows(8, V, [9, 0, 5, 0, 0, 0, 12, 0])   # rows: root, node 1, node 5
    r = accept_tree(z, TREE_X, TREE_P, 0.0, None)
    assert r.accepted == [1, 5] and r.emitted == [9, 5, 12]
    # root's argmax 4 is no child: nothing accepted, the token is the final one
    z = _onehot_rows(8, V, [4] * 8)
    r = accept_tree(z, TREE_X, TREE_P, 0.0, None)
    assert r.accepted == [] and r.emitted == [4]
    # the deepest path 0 -> 2 -> 4 -> 6 and then the leaf's row
    z = _onehot_rows(8, V, [5, 7, 0, 3, 0, 8, 0, 1])
    r = accept_tree(z, TREE_X, TREE_P, 0.0, None)
    assert r.accepted == [0, 2, 4, 6] and r.emitted == [5, 7, 3, 8, 1]


def test_duplicate_siblings_take_the_lowest_index():
    V = 12
    parents, tokens = [-1, -1, 0, 1], [3, 3, 4, 5]
    z = _onehot_rows(5, V, [3, 4, 5, 0, 0])
    r = accept_tree(z, tokens, parents, 0.0, None)
    assert r.accepted == [0, 2]
    reach = reach_probabilities(np.log(np.full((5, V), 1.0 / V)), tokens, parents, 1.0)
    assert reach[1] == 0.0 and reach[3] == 0.0 and reach[0] > 0


def _chi2_ok(counts, probs, n):
    mask = probs * n >= 5
    exp = probs[mask] * n
    obs = counts[mask]
    chi2 = float(((obs - exp) ** 2 / exp).sum()) + 0.0
    dof = int(mask.sum()) - 1
    # 1e-4 two-sided-ish bound via Wilson-Hilferty
    z = 3.72
    bound = dof * (1 - 2 / (9 * dof) + z * math.sqrt(2 / (9 * dof))) ** 3
    return chi2 < bound, chi2, bound


def test_walk_draws_every_token_from_the_target():
    rng = np.random.default_rng(11)
    V, T = 8, 0.9
    parents, tokens = [-1, -1, -1, 0, 0, 2, 3], [1, 2, 5, 0, 6, 6, 3]
    z = rng.standard_normal((len(tokens) + 1, V)) * 1.5
    p = softmax_t(z, T)
    n = 60000
    first = np.zeros(V)
    second = {c: np.zeros(V) for c in children(parents, 0)}
    acc_len = 0
    for _ in range(n):
        r = accept_tree(z, tokens, parents, T, rng.random(len(tokens) + 1))
        first[r.emitted[0]] += 1
        acc_len += len(r.accepted)
        if r.accepted:
            second[r.accepted[0]][r.emitted[1]] += 1
    ok, chi2, b = _chi2_ok(first, p[0], n)
    assert ok, (chi2, b)
    for c, cnt in second.items():
        m = int(cnt.sum())
        assert abs(m / n - p[0, tokens[c]]) < 4 * math.sqrt(p[0, tokens[c]] / n)
        ok, chi2, b = _chi2_ok(cnt, p[c + 1], m)
        assert ok, (c, chi2, b)
    # E[accepted] = sum over nodes of P(reached)
    reach = reach_probabilities(z, tokens, parents, T)
    mean = acc_len / n
    assert abs(mean - reach.sum()) < 0.02, (mean, reach.sum())
    # closed form by hand for node 3 (root -> 1 -> 0): p_root(1) p_node0(0)
    assert reach[3] == pytest.approx(p[0, 1] * p[1, 0], rel=1e-12)
