"""Pins for the oracle's decoder forward pass (CPU only).

Each check compares the oracle with something other than itself: PyTorch
library routines (scaled_dot_product_attention, rms_norm, silu, linear),
closed forms of RoPE, and invariants that any correct KV-cached decoder has
(incremental == full recomputation, causality).
"""
import dataclasses

import numpy as np
import pytest
import torch
import torch.nn.functional as F

from oracle.llama import LlamaOracle, apply_rope, attention, rmsnorm, silu
from seeded_inputs import SHAPES, ModelShape, gen_weights

GQA = ModelShape(2, 128, 4, 2, 32, 160, 97)        # 2 query heads per KV head, odd vocab


def _t(x):
    return torch.from_numpy(np.asarray(x, dtype=np.float64))


def test_attention_matches_torch_sdpa_gqa_causal_offset():
    rng = np.random.default_rng(0)
    H, Hkv, hd, S, M = 6, 2, 16, 11, 4
    q = rng.standard_normal((M, H, hd))
    k = rng.standard_normal((S, Hkv, hd))
    v = rng.standard_normal((S, Hkv, hd))
    positions = np.arange(S - M, S)                 # the last M positions (verify-like)
    o = attention(q, k, v, positions)
    kk = _t(k).repeat_interleave(H // Hkv, dim=1).permute(1, 0, 2)      # [H, S, hd]
    vv = _t(v).repeat_interleave(H // Hkv, dim=1).permute(1, 0, 2)
    qq = _t(q).permute(1, 0, 2)                                         # [H, M, hd]
    mask = torch.arange(S)[None, :] <= torch.from_numpy(positions)[:, None]
    ref = F.scaled_dot_product_attention(qq, kk, vv, attn_mask=mask).permute(1, 0, 2)
    np.testing.assert_allclose(o, ref.numpy(), rtol=1e-12, atol=1e-12)


def test_attention_special_cases():
    rng = np.random.default_rng(1)
    q = rng.standard_normal((1, 2, 8))
    k = rng.standard_normal((5, 1, 8))
    v = rng.standard_normal((5, 1, 8))
    # one visible key -> output is exactly that value row
    o = attention(q, k, v, [0])
    np.testing.assert_allclose(o[0, 0], v[0, 0], rtol=0, atol=1e-15)
    # identical keys -> uniform weights -> mean of the visible values
    k2 = np.repeat(k[:1], 5, axis=0)
    o = attention(q, k2, v, [3])
    np.testing.assert_allclose(o[0, 1], v[:4, 0].mean(axis=0), rtol=1e-13)


def test_rmsnorm_and_silu_match_torch():
    rng = np.random.default_rng(2)
    x = rng.standard_normal((3, 64)) * 5
    g = rng.standard_normal(64)
    ref = F.rms_norm(_t(x), (64,), weight=_t(g), eps=1e-5).numpy()
    np.testing.assert_allclose(rmsnorm(x, g, 1e-5), ref, rtol=1e-13)
    np.testing.assert_allclose(silu(x), F.silu(_t(x)).numpy(), rtol=1e-13)
    # closed form: a constant row c*1 with unit gain normalises to sign(c)*1 (eps -> 0)
    np.testing.assert_allclose(rmsnorm(np.full((1, 8), -3.0), np.ones(8), 0.0), -np.ones((1, 8)))


def test_rope_closed_forms():
    hd, base = 16, 10000.0
    rng = np.random.default_rng(3)
    x = rng.standard_normal((5, 3, hd))
    # position 0 is the identity
    np.testing.assert_allclose(apply_rope(x[:1], [0], base), x[:1], rtol=0, atol=0)
    # a unit vector on dim i (i < hd/2) rotates into span{e_i, e_{i+hd/2}}
    i, p = 3, 7
    e = np.zeros((1, 1, hd))
    e[0, 0, i] = 1.0
    r = apply_rope(e, [p], base)[0, 0]
    ang = p * base ** (-2.0 * i / hd)
    expect = np.zeros(hd)
    expect[i], expect[i + hd // 2] = np.cos(ang), np.sin(ang)
    np.testing.assert_allclose(r, expect, atol=1e-15)
    # norms are preserved, and q.k depends only on the position difference
    pos = np.array([0, 3, 10, 11, 40])
    xr = apply_rope(x, pos, base)
    np.testing.assert_allclose(np.linalg.norm(xr, axis=-1), np.linalg.norm(x, axis=-1), rtol=1e-13)
    q = rng.standard_normal((1, 1, hd))
    k = rng.standard_normal((1, 1, hd))
    d1 = (apply_rope(q, [9], base) * apply_rope(k, [4], base)).sum()
    d2 = (apply_rope(q, [105], base) * apply_rope(k, [100], base)).sum()
    np.testing.assert_allclose(d1, d2, rtol=1e-12)


def _torch_layer(shape, w, li, h, positions):
    """The same decoder layer assembled from PyTorch library routines (fp64)."""
    s = shape
    W = lambda n: _t(w[(n, li)])
    h = _t(h)
    M = h.shape[0]
    a = F.rms_norm(h, (s.d_model,), weight=W("attn_norm"), eps=s.norm_eps)
    q = F.linear(a, W("wq")).view(M, s.n_heads, s.head_dim)
    k = F.linear(a, W("wk")).view(M, s.n_kv_heads, s.head_dim)
    v = F.linear(a, W("wv")).view(M, s.n_kv_heads, s.head_dim)
    half = s.head_dim // 2
    inv = s.rope_base ** (-torch.arange(half, dtype=torch.float64) * 2 / s.head_dim)
    ang = torch.from_numpy(np.asarray(positions, dtype=np.float64))[:, None] * inv[None, :]
    cos, sin = torch.cos(ang)[:, None, :], torch.sin(ang)[:, None, :]
    rot = lambda x: torch.cat([x[..., :half] * cos - x[..., half:] * sin,
                               x[..., :half] * sin + x[..., half:] * cos], dim=-1)
    q, k = rot(q), rot(k)
    # the KV cache holds bf16 values: PyTorch's own conversion
    k = k.to(torch.bfloat16).to(torch.float64)
    v = v.to(torch.bfloat16).to(torch.float64)
    g = s.n_heads // s.n_kv_heads
    kk = k.repeat_interleave(g, dim=1).permute(1, 0, 2)
    vv = v.repeat_interleave(g, dim=1).permute(1, 0, 2)
    o = F.scaled_dot_product_attention(q.permute(1, 0, 2), kk, vv, is_causal=True)
    h = h + F.linear(o.permute(1, 0, 2).reshape(M, -1), W("wo"))
    m = F.rms_norm(h, (s.d_model,), weight=W("ffn_norm"), eps=s.norm_eps)
    return (h + F.linear(F.silu(F.linear(m, W("w_gate"))) * F.linear(m, W("w_up")), W("w_down"))).numpy()


def test_bf16_rounding_of_the_kv_cache():
    from oracle.llama import bf16
    # values on the bf16 grid are kept; halfway cases go to the even neighbour
    grid = np.array([0.0, 1.0, -1.0, 1.0 + 2.0 ** -7, 3.0 * 2.0 ** -20, -255.0 * 2.0 ** 10])
    np.testing.assert_array_equal(bf16(grid), grid)
    ties = np.array([1.0 + 2.0 ** -8, 1.0 + 3.0 * 2.0 ** -8, -(2.0 + 2.0 ** -7), 0.5 + 2.0 ** -10])
    np.testing.assert_array_equal(bf16(ties), [1.0, 1.0 + 2.0 ** -6, -2.0, 0.5])
    np.testing.assert_array_equal(bf16(1.0 + 2.0 ** -8 + 2.0 ** -30), 1.0 + 2.0 ** -7)
    # PyTorch's conversion agrees on values float32 holds exactly
    x = np.random.default_rng(2).standard_normal(20000).astype(np.float32).astype(np.float64) * 3.0
    ref = torch.from_numpy(x).to(torch.bfloat16).to(torch.float64).numpy()
    np.testing.assert_array_equal(bf16(x), ref)
    # the rounding error is at most half a quantum: 2^-8 relative (unit roundoff)
    assert np.all(np.abs(bf16(x) - x) <= np.abs(x) * 2.0 ** -8)


@pytest.mark.parametrize("shape", [GQA, SHAPES["tiny_draft"]])
def test_layer_matches_torch_library_assembly(shape):
    w = gen_weights(shape, seed=11)
    # non-trivial norm gains so a dropped gain would show
    rng = np.random.default_rng(4)
    for li in range(shape.n_layers):
        for n in ("attn_norm", "ffn_norm"):
            w[(n, li)] = (1.0 + 0.1 * rng.standard_normal(shape.d_model)).astype(np.float32)
    model = LlamaOracle(shape, w)
    M = 9
    h = rng.standard_normal((M, shape.d_model))
    cache = model.new_cache(M)
    out = model.layer(0, h, cache, np.arange(M))
    ref = _torch_layer(shape, w, 0, h, np.arange(M))
    np.testing.assert_allclose(out, ref, rtol=1e-10, atol=1e-10)


@pytest.mark.parametrize("shape", [GQA, SHAPES["tiny_draft"]])
def test_kv_cached_decoding_equals_full_recomputation(shape):
    w = gen_weights(shape, seed=5)
    model = LlamaOracle(shape, w)
    toks = np.random.default_rng(6).integers(0, shape.vocab, 12)
    full = model.forward(model.new_cache(12), toks)
    c = model.new_cache(12)
    inc = np.concatenate([model.forward(c, toks[:5]), model.forward(c, toks[5:6]),
                          model.forward(c, toks[6:9]), model.forward(c, toks[9:])])
    np.testing.assert_allclose(inc, full, rtol=1e-11, atol=1e-11)
    # rollback: truncate, re-feed different tokens, equals a fresh run on the new prefix
    c.truncate(7)
    alt = np.array([1, 2, 3])
    z = model.forward(c, alt)
    ref = model.forward(model.new_cache(10), np.concatenate([toks[:7], alt]))[7:]
    np.testing.assert_allclose(z, ref, rtol=1e-11, atol=1e-11)


def test_causality():
    shape = GQA
    model = LlamaOracle(shape, gen_weights(shape, seed=8))
    a = np.array([5, 9, 13, 2, 7, 1])
    b = a.copy()
    b[4:] = [60, 61]
    za = model.forward(model.new_cache(6), a)
    zb = model.forward(model.new_cache(6), b)
    np.testing.assert_array_equal(za[:4], zb[:4])
    assert np.abs(za[4:] - zb[4:]).max() > 1e-3


def test_zero_residual_branches_reduce_to_embedding_logits():
    # with Wo = 0 and Wdown = 0 the layers add nothing: logits = RMSNorm(E[t]) Wlm^T
    shape = GQA
    w = gen_weights(shape, seed=9)
    for li in range(shape.n_layers):
        w[("wo", li)] = np.zeros_like(w[("wo", li)])
        w[("w_down", li)] = np.zeros_like(w[("w_down", li)])
    model = LlamaOracle(shape, w)
    toks = np.array([3, 50, 96])
    z = model.forward(model.new_cache(3), toks)
    e = w[("tok_emb", -1)][toks].astype(np.float64)
    e = e / np.sqrt((e * e).mean(axis=1, keepdims=True) + shape.norm_eps)
    np.testing.assert_allclose(z, e @ w[("lm_head", -1)].astype(np.float64).T, rtol=1e-12)


def test_tied_lm_head_uses_embedding():
    shape = dataclasses.replace(GQA, tied=True)
    w = gen_weights(shape, seed=10)
    assert ("lm_head", -1) not in w
    model = LlamaOracle(shape, w)
    z = model.forward(model.new_cache(2), [4, 8])
    assert z.shape == (2, shape.vocab)
    for li in range(shape.n_layers):
        w[("wo", li)] = np.zeros_like(w[("wo", li)])
        w[("w_down", li)] = np.zeros_like(w[("w_down", li)])
    z = LlamaOracle(shape, w).forward(model.new_cache(1), [4])
    e = w[("tok_emb", -1)][4].astype(np.float64)
    e = e / np.sqrt((e * e).mean() + shape.norm_eps)
    np.testing.assert_allclose(z[0], w[("tok_emb", -1)].astype(np.float64) @ e, rtol=1e-12)
