"""Llama-style decoder forward pass with a KV cache, in float64 (oracle side).

Test infrastructure only (see ``oracle/__init__``).

MemSpec (Section 4.1) runs LLaMA-2-7B / Qwen2.5-7B targets with small drafts;
the step it builds on feeds the target the K+1 positions [last committed token,
x_1..x_K] against the target's KV cache (Section 2.1, Eq. 1 context; Section
3.5).  The layer is the LLaMA-2 decoder layer:

    a = RMSNorm(h) * g_attn
    q, k, v = a Wq^T, a Wk^T, a Wv^T            (per head, head_dim hd)
    q, k = RoPE(q, pos), RoPE(k, pos)          (pairs (i, i + hd/2), theta_i = base^(-2i/hd))
    o_h = softmax(q_h K_{g(h)}^T / sqrt(hd) + causal mask) V_{g(h)}   (GQA: g(h) = h // (H/Hkv))
    h = h + o Wo^T
    m = RMSNorm(h) * g_ffn
    h = h + (silu(m Wgate^T) * (m Wup^T)) Wdown^T
    logits = (RMSNorm(h) * g_final) Wlm^T

Weights arrive as float32 arrays holding bf16 values (exactly representable) and
are used in float64.  All arithmetic is float64; the one rounding step is the
KV cache, which stores K and V as bf16 values (the workload fixes bf16 weights
and KV cache), so every attention reads bf16 keys and values, the rows just
appended included.
"""
from __future__ import annotations

import numpy as np

LAYER_TENSORS = ("attn_norm", "wq", "wk", "wv", "wo", "ffn_norm", "w_gate", "w_up", "w_down")


def bf16(x: np.ndarray) -> np.ndarray:
    """Round to the nearest bfloat16 value (8 significant bits, ties to even),
    float64 in and out: with x = m 2^e, 0.5 <= |m| < 1, the quantum is 2^(e-8)."""
    x = np.asarray(x, dtype=np.float64)
    _, e = np.frexp(x)
    q = np.ldexp(1.0, e - 8)
    return np.round(x / q) * q          # numpy rounds halves to even


def rmsnorm(x: np.ndarray, gain: np.ndarray, eps: float) -> np.ndarray:
    """x / sqrt(mean(x^2) + eps) * gain, over the last axis."""
    x = np.asarray(x, dtype=np.float64)
    ms = np.mean(x * x, axis=-1, keepdims=True)
    return x / np.sqrt(ms + eps) * np.asarray(gain, dtype=np.float64)


def silu(x: np.ndarray) -> np.ndarray:
    return x / (1.0 + np.exp(-x))


def rope_angles(positions, head_dim: int, base: float) -> np.ndarray:
    """angle[p, i] = pos_p * base^(-2i/hd), i < hd/2."""
    i = np.arange(head_dim // 2, dtype=np.float64)
    theta = base ** (-2.0 * i / head_dim)
    return np.asarray(positions, dtype=np.float64)[:, None] * theta[None, :]


def apply_rope(x: np.ndarray, positions, base: float) -> np.ndarray:
    """Rotate pairs (i, i + hd/2) of x[..., pos, head, hd] by pos * theta_i.

    x has shape [M, heads, hd]; positions has length M.
    """
    hd = x.shape[-1]
    half = hd // 2
    ang = rope_angles(positions, hd, base)[:, None, :]          # [M, 1, half]
    c, s = np.cos(ang), np.sin(ang)
    x1, x2 = x[..., :half], x[..., half:]
    return np.concatenate([x1 * c - x2 * s, x1 * s + x2 * c], axis=-1)


def attention(q: np.ndarray, k_cache: np.ndarray, v_cache: np.ndarray,
              positions) -> np.ndarray:
    """Causal grouped-query attention of M query rows against a KV cache.

    q:        [M, H, hd]   (already rotated)
    k_cache:  [S, Hkv, hd] (rotated keys for positions 0..S-1)
    v_cache:  [S, Hkv, hd]
    positions[i] is the position of query row i; it sees keys 0..positions[i].
    Returns o [M, H, hd].
    """
    M, H, hd = q.shape
    Hkv = k_cache.shape[1]
    group = H // Hkv
    o = np.zeros_like(q)
    for i in range(M):
        n = int(positions[i]) + 1
        for h in range(H):
            g = h // group
            scores = k_cache[:n, g, :] @ q[i, h, :] / np.sqrt(hd)
            w = np.exp(scores - scores.max())
            w /= w.sum()
            o[i, h, :] = w @ v_cache[:n, g, :]
    return o


class KVCache:
    """Per-layer K and V for positions 0..length-1 (rotated keys), bf16 values
    held in float64."""

    def __init__(self, n_layers: int, n_kv_heads: int, head_dim: int, capacity: int):
        self.k = np.zeros((n_layers, capacity, n_kv_heads, head_dim))
        self.v = np.zeros((n_layers, capacity, n_kv_heads, head_dim))
        self.length = 0

    def truncate(self, length: int):
        """Roll back to the first ``length`` positions (rejected drafts)."""
        assert 0 <= length <= self.length
        self.length = length


class LlamaOracle:
    """One model (target or draft).  ``weights`` maps (name, layer) -> array."""

    def __init__(self, shape, weights: dict, keep_f64: bool = False):
        """keep_f64: hold every matrix in float64 (memory for speed); otherwise
        the matrices of the most recently used layer are kept converted."""
        self.shape = shape
        self.w = weights
        lm = ("tok_emb", -1) if shape.tied else ("lm_head", -1)
        self.lm_key = lm
        self.keep_f64 = keep_f64
        self._f64 = {}
        self._f64_layer = None

    def new_cache(self, capacity: int) -> KVCache:
        s = self.shape
        return KVCache(s.n_layers, s.n_kv_heads, s.head_dim, capacity)

    def _w64(self, name: str, layer: int) -> np.ndarray:
        key = (name, layer)
        if not self.keep_f64 and layer != self._f64_layer:
            self._f64 = {}
            self._f64_layer = layer
        if key not in self._f64:
            self._f64[key] = self.w[key].astype(np.float64)
        return self._f64[key]

    def _lin(self, x: np.ndarray, name: str, layer: int) -> np.ndarray:
        # x [M, in] float64; W [out, in] float32 holding bf16 values -> x W^T in float64
        return x @ self._w64(name, layer).T

    def layer(self, li: int, h: np.ndarray, cache: KVCache, positions) -> np.ndarray:
        """One decoder layer over rows h [M, d]; appends their K, V to the cache."""
        s = self.shape
        M = h.shape[0]
        a = rmsnorm(h, self.w[("attn_norm", li)], s.norm_eps)
        q = self._lin(a, "wq", li).reshape(M, s.n_heads, s.head_dim)
        k = self._lin(a, "wk", li).reshape(M, s.n_kv_heads, s.head_dim)
        v = self._lin(a, "wv", li).reshape(M, s.n_kv_heads, s.head_dim)
        q = apply_rope(q, positions, s.rope_base)
        k = apply_rope(k, positions, s.rope_base)
        start = int(positions[0])
        cache.k[li, start:start + M] = bf16(k)
        cache.v[li, start:start + M] = bf16(v)
        end = start + M
        o = attention(q, cache.k[li, :end], cache.v[li, :end], positions)
        h = h + self._lin(o.reshape(M, s.q_dim), "wo", li)
        m = rmsnorm(h, self.w[("ffn_norm", li)], s.norm_eps)
        act = silu(self._lin(m, "w_gate", li)) * self._lin(m, "w_up", li)
        return h + self._lin(act, "w_down", li)

    def embed(self, tokens) -> np.ndarray:
        return self.w[("tok_emb", -1)][np.asarray(tokens, dtype=np.int64)].astype(np.float64)

    def logits(self, h: np.ndarray) -> np.ndarray:
        s = self.shape
        hf = rmsnorm(h, self.w[("final_norm", -1)], s.norm_eps)
        return hf @ self._w64(*self.lm_key).T

    def forward(self, cache: KVCache, tokens, want_logits: bool = True):
        """Feed ``tokens`` at positions cache.length .. cache.length+M-1.

        Returns logits [M, vocab] (float64) or None.
        """
        tokens = np.asarray(tokens, dtype=np.int64)
        M = len(tokens)
        if M == 0:
            return np.zeros((0, self.shape.vocab)) if want_logits else None
        positions = np.arange(cache.length, cache.length + M)
        h = self.embed(tokens)
        for li in range(self.shape.n_layers):
            h = self.layer(li, h, cache, positions)
        cache.length += M
        return self.logits(h) if want_logits else None
