"""Seeded synthetic inputs for the speculative decoding step.

This module is the ONE source of input data shared by the CUDA path and the
oracle.  It draws random numbers and nothing else: it holds no step of the
method (no forward pass, no softmax, no acceptance rule).  Everything it
returns is a pure function of the seed, whatever the thread count.

Workload shapes follow the evaluation set-up of the MemSpec paper (Section 4.1:
LLaMA-2-7B-class targets, small drafts, greedy/sampled decoding at batch 1) as
fixed in the build's configuration table: a tiny pair, an edge-class pair
(1.1B target / 68M draft), a 7B-shape target with a 160M draft, and an 8B-shape
target with a 1.1B draft for batched verification.  The paper's trained
checkpoints and its datasets (Alpaca, LiveCodeBench, Omni-MATH, MMLU) are not
available; random-init weights N(0, 0.02^2) rounded to bf16 and uniform-random
prompt ids stand in for them.
"""
from __future__ import annotations

import dataclasses
from concurrent.futures import ThreadPoolExecutor
import os

import numpy as np

__all__ = [
    "ModelShape", "SHAPES", "tensor_names", "tensor_shape", "gen_tensor",
    "iter_weights", "gen_weights", "gen_prompt", "gen_logits", "gen_kv",
    "bf16_round", "gen_score_stream", "gen_int4_weights",
]


@dataclasses.dataclass(frozen=True)
class ModelShape:
    """Llama-style decoder hyper-parameters (RMSNorm, RoPE, SwiGLU, GQA)."""
    n_layers: int
    d_model: int
    n_heads: int
    n_kv_heads: int
    head_dim: int
    d_ffn: int
    vocab: int
    tied: bool = False          # LM head shares the token embedding
    rope_base: float = 10000.0
    norm_eps: float = 1e-5

    @property
    def q_dim(self) -> int:
        return self.n_heads * self.head_dim

    @property
    def kv_dim(self) -> int:
        return self.n_kv_heads * self.head_dim

    def n_params(self) -> int:
        d, f, v = self.d_model, self.d_ffn, self.vocab
        per_layer = 2 * d + (self.q_dim + 2 * self.kv_dim) * d + d * self.q_dim + 3 * f * d
        return v * d * (1 if self.tied else 2) + self.n_layers * per_layer + d


SHAPES = {
    # tiny pair (oracle-sized): 4-layer target d=256, 2-layer draft d=128, vocab 2048
    "tiny_target": ModelShape(4, 256, 4, 4, 64, 688, 2048),
    "tiny_draft": ModelShape(2, 128, 2, 2, 64, 352, 2048),
    # edge-class pair: 1.1B target (GQA 32q/4kv), 68M draft
    "target_1b1": ModelShape(22, 2048, 32, 4, 64, 5632, 32000),
    "draft_68m": ModelShape(2, 768, 12, 12, 64, 3072, 32000),
    # 7B-shape target (MHA) with a 160M draft
    "target_7b": ModelShape(32, 4096, 32, 32, 128, 11008, 32000),
    "draft_160m": ModelShape(12, 768, 12, 12, 64, 3072, 32000),
    # 1.1B draft with tied embedding / LM head (fits a 2 GiB draft budget alone)
    "draft_1b1_tied": ModelShape(22, 2048, 32, 4, 64, 5632, 32000, tied=True),
    # batched verification: 8B-shape target (GQA 32q/8kv), 1.1B draft, vocab 128256
    "target_8b": ModelShape(32, 4096, 32, 8, 128, 14336, 128256),
    "draft_1b1_v128k": ModelShape(22, 2048, 32, 4, 64, 5632, 128256),
}

_LAYER_TENSORS = ("attn_norm", "wq", "wk", "wv", "wo", "ffn_norm", "w_gate", "w_up", "w_down")
_STD = 0.02
_BLOCK = 1 << 22            # elements per independently seeded block


def tensor_names(shape: ModelShape):
    """(name, layer) pairs in the fixed order that also numbers their seeds."""
    out = [("tok_emb", -1)]
    for layer in range(shape.n_layers):
        out += [(n, layer) for n in _LAYER_TENSORS]
    out.append(("final_norm", -1))
    if not shape.tied:
        out.append(("lm_head", -1))
    return out


def tensor_shape(shape: ModelShape, name: str):
    d, f = shape.d_model, shape.d_ffn
    return {
        "tok_emb": (shape.vocab, d), "lm_head": (shape.vocab, d),
        "attn_norm": (d,), "ffn_norm": (d,), "final_norm": (d,),
        "wq": (shape.q_dim, d), "wk": (shape.kv_dim, d), "wv": (shape.kv_dim, d),
        "wo": (d, shape.q_dim),
        "w_gate": (f, d), "w_up": (f, d), "w_down": (d, f),
    }[name]


def bf16_round(x: np.ndarray) -> np.ndarray:
    """Round float32 values to the nearest bfloat16 (ties to even); float32 out."""
    b = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    lsb = (b >> np.uint32(16)) & np.uint32(1)
    r = (b + (np.uint32(0x7FFF) + lsb)) & np.uint32(0xFFFF0000)
    return r.view(np.float32)


def _normal_block(seed: int, index: int, block: int, n: int) -> np.ndarray:
    rng = np.random.default_rng([seed, index, block])
    return rng.standard_normal(n, dtype=np.float32)


def gen_tensor(shape: ModelShape, seed: int, name: str, layer: int = -1,
               pool: ThreadPoolExecutor | None = None) -> np.ndarray:
    """One weight tensor: N(0, 0.02^2) rounded to bf16 (norm gains are 1.0).

    The tensor is split into blocks of 2^22 elements; block b of tensor i is
    drawn from numpy's PCG64 seeded with [seed, i, b], so the values do not
    depend on how many threads produce them.
    """
    shp = tensor_shape(shape, name)
    if name.endswith("norm"):
        return np.ones(shp, dtype=np.float32)
    index = tensor_names(shape).index((name, layer))
    n = int(np.prod(shp))
    nblk = (n + _BLOCK - 1) // _BLOCK
    sizes = [min(_BLOCK, n - b * _BLOCK) for b in range(nblk)]

    def work(b):
        return bf16_round(_normal_block(seed, index, b, sizes[b]) * np.float32(_STD))

    if pool is None or nblk == 1:
        parts = [work(b) for b in range(nblk)]
    else:
        parts = list(pool.map(work, range(nblk)))
    return np.concatenate(parts).reshape(shp)


def iter_weights(shape: ModelShape, seed: int, threads: int | None = None):
    """Yield (name, layer, float32 array) for every tensor, in seed order."""
    threads = threads or min(32, os.cpu_count() or 1)
    with ThreadPoolExecutor(threads) as pool:
        for name, layer in tensor_names(shape):
            yield name, layer, gen_tensor(shape, seed, name, layer, pool)


def gen_weights(shape: ModelShape, seed: int, threads: int | None = None) -> dict:
    """All tensors as {(name, layer): float32 array holding bf16 values}."""
    return {(n, l): a for n, l, a in iter_weights(shape, seed, threads)}


def gen_prompt(seed: int, length: int, vocab: int, request: int = 0) -> np.ndarray:
    """Uniform-random token ids in [0, vocab) standing in for a dataset prompt."""
    rng = np.random.default_rng([seed, 0x70726F6D, request])
    return rng.integers(0, vocab, size=length, dtype=np.int64).astype(np.int32)


def gen_prompt_lengths(seed: int, batch: int, lo: int, hi: int) -> np.ndarray:
    """Per-request prefix lengths uniform in [lo, hi] (batched verification)."""
    rng = np.random.default_rng([seed, 0x6C656E73])
    return rng.integers(lo, hi + 1, size=batch, dtype=np.int64).astype(np.int32)


def gen_logits(seed: int, rows: int, vocab: int, scale: float = 1.0) -> np.ndarray:
    """float32 logits N(0, scale^2) for exercising the sampling kernels alone."""
    rng = np.random.default_rng([seed, 0x6C6F6769])
    return (rng.standard_normal((rows, vocab), dtype=np.float32) * np.float32(scale))


def gen_kv(seed: int, shape_tuple, scale: float = 1.0) -> np.ndarray:
    """bf16-valued float32 array of N(0, scale^2) entries (synthetic KV cache)."""
    rng = np.random.default_rng([seed, 0x6B76])
    return bf16_round(rng.standard_normal(int(np.prod(shape_tuple)), dtype=np.float32)
                      * np.float32(scale)).reshape(shape_tuple)


def gen_score_stream(seed: int, points: int, n_drafts: int, phase: int = 4,
                     noise: float = 0.15) -> np.ndarray:
    """float32 [points][n_drafts] per-draft scores standing in for a draft
    predictor's output at successive scheduling points: a seeded "best draft"
    that changes every ``phase`` points (random phase boundaries), scored 1.0,
    the others uniform in [0, 0.8), plus N(0, noise^2) jitter."""
    rng = np.random.default_rng([seed, 0x73636F72])
    out = np.empty((points, n_drafts), dtype=np.float32)
    best = int(rng.integers(0, n_drafts))
    for i in range(points):
        if i % phase == 0 and rng.random() < 0.8:
            best = int(rng.integers(0, n_drafts))
        row = rng.random(n_drafts) * 0.8
        row[best] = 1.0
        out[i] = (row + rng.standard_normal(n_drafts) * noise).astype(np.float32)
    return out


def gen_int4_weights(seed: int, n: int, k: int, group: int = 128, scale: float = 0.004):
    """Random group-wise INT4 weights: packed codes uint8 [n][k/2] (two 4-bit codes
    per byte, low nibble first), scales [n][k/group] as bf16-valued float32 (about
    `scale` in size), zero points uint8 [n][k/group] in 0..15."""
    rng = np.random.default_rng([seed, 0x696E7434, n, k])
    codes = rng.integers(0, 16, size=(n, k), dtype=np.int64)
    packed = (codes[:, 0::2] | (codes[:, 1::2] << 4)).astype(np.uint8)
    scales = bf16_round((rng.random((n, k // group)) * 1.5 + 0.5).astype(np.float32) * np.float32(scale))
    zeros = rng.integers(0, 16, size=(n, k // group), dtype=np.int64).astype(np.uint8)
    return packed, scales, zeros
