"""Tree-based verification, float64 (oracle side).

Test infrastructure only (see ``oracle/__init__``).

MemSpec is built on a speculative-decoding engine that verifies draft trees
(Section 3.5, "System Implementation": the engine of SpecExec, Svirschevski et
al., NeurIPS 2024); MemSpec's own experiments use a chain.  The paper does not
restate the tree procedure, so this module follows SpecExec's verification as
read from that engine's description (the reading is listed with the others):

1. A draft tree hangs below the root, the last committed token t_{L-1}.  Node
   i (0-based, in an order where a parent precedes its children) carries a
   token and a parent: -1 for a child of the root, else a smaller node index.
   depth(i) = 0 for a child of the root, depth(parent) + 1 otherwise.
2. The target scores the root and every node in one pass.  The row of a node
   is the target's next-token distribution after the committed prefix, the
   root and the tokens on the path from the root to that node, i.e. exactly
   what a plain forward pass over that path gives (Definition of the row used
   below).  Positions: the root sits at L - 1, node i at L + depth(i).
3. Acceptance walks down from the root: at the current row v, one token x is
   drawn from the target's distribution p_v (inverse CDF with the uniform of
   emitted-token index e, Philox slot 64 + e; greedy: argmax).  If x is the
   token of a child of v, that child is accepted and the walk continues from
   it; otherwise x is the step's final token and the walk stops.  A leaf that
   is reached draws its final token the same way.  Every emitted token is a
   draw from the target's own conditional distribution, so the output
   distribution is the target's, for any tree.
4. The step commits the accepted nodes' tokens and the final token; the KV
   entries of the root and of the accepted nodes stay (moved to consecutive
   positions), all other nodes' entries are dropped.

Siblings with the same token: the child of lowest index is taken.
"""
from __future__ import annotations

import dataclasses

import numpy as np

from .philox import uniform
from .speculative import argmax_first, sample_inverse_cdf, softmax_t

TREE_SLOT0 = 64          # Philox slot of emitted token e: TREE_SLOT0 + e
MAX_TREE_NODES = 31      # root + 31 nodes = 32 rows of one pass


def tree_depths(parents) -> list[int]:
    """depth(i): 0 below the root, depth(parent) + 1 otherwise."""
    d = []
    for i, p in enumerate(parents):
        p = int(p)
        if not -1 <= p < i:
            raise ValueError(f"node {i}: parent {p} must be -1 or a smaller node index")
        d.append(0 if p < 0 else d[p] + 1)
    return d


def path_tokens(tokens, parents, i: int) -> list[int]:
    """Tokens on the path from the root's first child down to node i."""
    out = []
    while i >= 0:
        out.append(int(tokens[i]))
        i = int(parents[i])
    return out[::-1]


def children(parents, v: int) -> list[int]:
    """Nodes whose parent is row v (row 0 = the root, row i + 1 = node i), in
    index order."""
    return [i for i, p in enumerate(parents) if int(p) + 1 == v]


def tree_logits(model, cache, root: int, tokens, parents) -> np.ndarray:
    """Rows [N + 1, V]: row 0 after the root, row i + 1 after node i.

    Definition written out: the path root, x_.., x_i is fed as a plain
    sequence at positions cache.length .. on the committed cache, its last row
    kept, and the cache cut back (KVCache.truncate) before the next path."""
    L0 = cache.length
    rows = [model.forward(cache, [int(root)])[-1]]
    cache.truncate(L0)
    for i in range(len(tokens)):
        seq = [int(root)] + path_tokens(tokens, parents, i)
        rows.append(model.forward(cache, seq)[-1])
        cache.truncate(L0)
    return np.stack(rows)


def tree_uniforms(seed: int, request: int, step: int, n: int) -> list[float]:
    """Uniforms of emitted tokens 0..n-1 of one tree step."""
    return [uniform(seed, request, step, TREE_SLOT0 + e) for e in range(n)]


@dataclasses.dataclass
class TreeAcceptResult:
    accepted: list[int]      # node indices along the accepted path
    emitted: list[int]       # accepted tokens, then the final token
    p_path: list[float]      # p_v(x) of each emitted token (T > 0)


def accept_tree(z_rows: np.ndarray, tokens, parents, T: float, u) -> TreeAcceptResult:
    """The walk of step 3 over rows z_rows [N + 1, V] (row 0 = the root)."""
    v, accepted, emitted, probs = 0, [], [], []
    for e in range(len(tokens) + 1):
        z = z_rows[v]
        if T == 0.0:
            x = argmax_first(z)
            probs.append(1.0)
        else:
            p = softmax_t(z, T)
            x = sample_inverse_cdf(p, u[e])
            probs.append(float(p[x]))
        emitted.append(x)
        nxt = next((c for c in children(parents, v) if int(tokens[c]) == x), None)
        if nxt is None:
            break
        accepted.append(nxt)
        v = nxt + 1
    return TreeAcceptResult(accepted, emitted, probs)


def reach_probabilities(z_rows: np.ndarray, tokens, parents, T: float) -> np.ndarray:
    """P(node i is accepted) = product of p_parent(token) along its path (the
    walk draws each step from the target); used for E[accepted] pins."""
    p = softmax_t(z_rows, T)
    out = np.zeros(len(tokens))
    for i in range(len(tokens)):
        par = int(parents[i])
        prev = 1.0 if par < 0 else out[par]
        # siblings with the same token: only the lowest index can be taken
        first = min(c for c in children(parents, par + 1) if int(tokens[c]) == int(tokens[i]))
        out[i] = prev * p[par + 1, int(tokens[i])] if first == i else 0.0
    return out
