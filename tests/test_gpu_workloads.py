"""Parity at the workload sizes (GPU), in the launch configuration bench.py uses
(captured CUDA graphs):

* edge pair (1.1B GQA target, 68M draft, prefix 512, K=5): lock-step against the
  oracle, greedy and T = 0.8;
* 7B-shape target, verify pass at context 2048 with a seeded KV cache, K=4:
  logits of all K+1 rows and the K/V appended at the new positions;
* 8B-shape target, batched verify (B=16, K=8, vocab 128256, per-request
  contexts uniform in [512, 4096]): logits of three sampled requests;
* draft switching under a byte budget: load / query / evict rules, and lock-step
  parity after switching the active draft mid-generation.
"""
import dataclasses

import numpy as np
import pytest
import torch

from lockstep import LOGIT_TOL, LockstepReport, check_step
from oracle.llama import LlamaOracle
from oracle.speculative import SpecDecoder, argmax_first
from seeded_inputs import SHAPES, gen_kv, gen_prompt, gen_prompt_lengths, gen_weights

pytestmark = pytest.mark.gpu


def _kv_view(eng, shape):
    """bf16 view [layer][K|V][request][kv_head][pos][hd] of the engine's KV cache."""
    return eng.kv.view(torch.bfloat16).view(shape.n_layers, 2, eng.max_batch, shape.n_kv_heads,
                                            eng.max_seq, shape.head_dim)


def _fill_kv(eng, shape, req, ctx, seed, oracle_cache=None):
    """Seeded N(0,1) bf16 K/V for positions < ctx of one request (GPU and oracle)."""
    kv = gen_kv(seed, (shape.n_layers, 2, ctx, shape.n_kv_heads, shape.head_dim))
    view = _kv_view(eng, shape)
    t = torch.from_numpy(kv).to(torch.bfloat16)          # exact: values are bf16
    view[:, :, req, :, :ctx, :] = t.permute(0, 1, 3, 2, 4).cuda()
    if oracle_cache is not None:
        oracle_cache.k[:, :ctx] = kv[:, 0].astype(np.float64)
        oracle_cache.v[:, :ctx] = kv[:, 1].astype(np.float64)
        oracle_cache.length = ctx
    return kv


def _set_verify_state(eng, ctxs, K, tokens_last, drafts):
    from paper_2608_10362_gb300 import _lib
    B = len(ctxs)
    state = np.zeros((eng.max_batch, 4), dtype=np.int32)
    toks = np.zeros((eng.max_batch, eng.max_seq), dtype=np.int32)
    dt = np.zeros((eng.max_batch, eng.max_k), dtype=np.int32)
    for b, ctx in enumerate(ctxs):
        state[b] = (ctx + 1, ctx, 0, 0)
        toks[b, ctx] = tokens_last[b]
        dt[b, :K] = drafts[b]
    eng.write_buffer(_lib.BUF_TOKENS, toks)
    eng.write_buffer(_lib.BUF_SEQ_STATE, state)
    eng.write_buffer(_lib.BUF_DRAFT_TOKENS, dt)
    eng.set_batch(B)


# ---------------------------------------------------------------------- edge pair
@pytest.fixture(scope="module")
def edge():
    from paper_2608_10362_gb300 import Engine
    t, d = SHAPES["target_1b1"], SHAPES["draft_68m"]
    wt, wd = gen_weights(t, 0), gen_weights(d, 1)
    eng = Engine(t, wt, max_batch=1, max_seq=1024, max_k=5, max_drafts=1, draft_shape_max=d,
                 draft_budget_bytes=256 << 20, use_graphs=True)
    eng.register_draft(0, d, wd)
    eng.load_draft_async(0)
    eng.set_active_draft(0)
    yield eng, LlamaOracle(t, wt, keep_f64=True), LlamaOracle(d, wd, keep_f64=True)
    eng.close()


@pytest.mark.parametrize("T", [0.0, 0.8])
def test_edge_pair_lockstep(edge, T):
    eng, to, do = edge
    prompt = gen_prompt(21, 512, 32000)
    K, steps = 5, 6
    eng.prefill(0, prompt, seed=9)
    sd = SpecDecoder(to, do, prompt, len(prompt) + steps * (K + 1) + 4)
    rep = LockstepReport()
    for step in range(steps):
        eng.step(K, T, eng.results_host)
        check_step(eng, sd, K, T, 9, step, rep)
    print(f"edge T={T}: tokens {rep.tokens_committed} flags {rep.flags}/{rep.decisions} "
          f"max logit err {rep.max_logit_err_frac:.2e}")
    # every mismatch was checked against the band its own measured logit error allows;
    # the count only guards against a degenerate (very wide) band
    assert rep.flags <= max(2, rep.decisions // 3)


# ---------------------------------------------------------------------- 7B verify at ctx 2048
def test_7b_verify_pass_full_size():
    from paper_2608_10362_gb300 import Engine
    t = SHAPES["target_7b"]
    K, ctx = 4, 2048
    w = gen_weights(t, 0)
    eng = Engine(t, w, max_batch=1, max_seq=ctx + 64, max_k=K, max_drafts=0, use_graphs=True)
    oracle = LlamaOracle(t, w)
    cache = oracle.new_cache(ctx + K + 1)
    _fill_kv(eng, t, 0, ctx, 77, cache)
    rng = np.random.default_rng(5)
    last, drafts = int(rng.integers(0, t.vocab)), rng.integers(0, t.vocab, K).astype(np.int32)
    _set_verify_state(eng, [ctx], K, [last], [drafts])
    eng.verify_step(K)
    assert eng.sync() == 0
    zg = eng.target_logits(1, K)[0]
    kv_new = _kv_view(eng, t)[:, :, 0, :, ctx:ctx + K + 1, :].float().cpu().numpy()
    zo = oracle.forward(cache, [last] + list(drafts))
    for i in range(K + 1):
        err = np.abs(zg[i] - zo[i]).max() / np.abs(zo[i]).max()
        print(f"7B verify row {i}: logit err {err:.2e} of max")
        assert err <= LOGIT_TOL
        a, b = argmax_first(zo[i]), int(np.argmax(zg[i]))
        assert a == b or zo[i][a] - zo[i][b] <= 2 * np.abs(zg[i] - zo[i]).max()
    # K/V appended at positions ctx..ctx+K (bf16 storage of the rotated keys / values)
    ko = cache.k[:, ctx:ctx + K + 1].transpose(0, 2, 1, 3)     # [layer][kvh][pos][hd]
    vo = cache.v[:, ctx:ctx + K + 1].transpose(0, 2, 1, 3)
    for got, ref in ((kv_new[:, 0], ko), (kv_new[:, 1], vo)):
        scale = np.abs(ref).max(axis=(1, 2, 3), keepdims=True)
        assert np.all(np.abs(got - ref) <= 0.03 * scale)
    eng.close()


# ---------------------------------------------------------------------- batched 8B verify
def test_8b_batched_verify_sampled_requests():
    from paper_2608_10362_gb300 import Engine
    t = SHAPES["target_8b"]
    B, K = 16, 8
    ctxs = [int(c) for c in gen_prompt_lengths(11, B, 512, 4096)]
    w = gen_weights(t, 0)
    eng = Engine(t, w, max_batch=B, max_seq=4096 + 64, max_k=K, max_drafts=0, use_graphs=True)
    oracle = LlamaOracle(t, w)
    checked = [0, 7, 15]
    caches = {}
    for b in range(B):
        if b in checked:
            caches[b] = oracle.new_cache(ctxs[b] + K + 1)
            _fill_kv(eng, t, b, ctxs[b], 100 + b, caches[b])
    rng = np.random.default_rng(6)
    last = rng.integers(0, t.vocab, B)
    drafts = rng.integers(0, t.vocab, (B, K)).astype(np.int32)
    _set_verify_state(eng, ctxs, K, last, drafts)
    eng.verify_step(K)
    assert eng.sync() == 0
    zg = eng.target_logits(B, K)
    eng.close()
    # the checked requests advance together, layer by layer (each matrix is converted once)
    hs = {b: oracle.embed([int(last[b])] + list(drafts[b])) for b in checked}
    pos = {b: np.arange(ctxs[b], ctxs[b] + K + 1) for b in checked}
    for li in range(t.n_layers):
        for b in checked:
            hs[b] = oracle.layer(li, hs[b], caches[b], pos[b])
    for b in checked:
        zo = oracle.logits(hs[b])
        err = max(np.abs(zg[b, i] - zo[i]).max() / np.abs(zo[i]).max() for i in range(K + 1))
        print(f"8B batched request {b} (ctx {ctxs[b]}): max logit err {err:.2e} of max")
        assert err <= LOGIT_TOL


# ---------------------------------------------------------------------- draft switching
def test_draft_switching_under_budget():
    from paper_2608_10362_gb300 import Engine, MemSpecError, _lib, weights_bytes
    t = SHAPES["tiny_target"]
    d0 = SHAPES["tiny_draft"]
    d1 = dataclasses.replace(d0, n_layers=3)
    d2 = dataclasses.replace(d0, n_layers=1)
    ws = {0: gen_weights(d0, 1), 1: gen_weights(d1, 2), 2: gen_weights(d2, 3)}
    shapes = {0: d0, 1: d1, 2: d2}
    sizes = {i: weights_bytes(s) for i, s in shapes.items()}
    budget = sizes[0] + sizes[1] + 1024            # fits drafts 0 and 1, not all three
    wt = gen_weights(t, 0)
    eng = Engine(t, wt, max_batch=1, max_seq=512, max_k=4, max_drafts=3, draft_shape_max=d1,
                 draft_budget_bytes=budget, use_graphs=True)
    for i in range(3):
        eng.register_draft(i, shapes[i], ws[i])
        assert eng.query_draft(i) == 0
    eng.load_draft_async(0)
    eng.load_draft_async(1)
    with pytest.raises(MemSpecError) as ex:
        eng.load_draft_async(2)                     # over budget: refused, nothing changes
    assert ex.value.status == _lib.ERR_BUDGET
    eng.set_active_draft(0)
    assert eng.query_draft(0) == 1
    with pytest.raises(MemSpecError) as ex:
        eng.evict_draft(0)                          # the active draft is never evicted
    assert ex.value.status == _lib.ERR_BUSY
    prompt = gen_prompt(31, 100, 2048)
    eng.prefill(0, prompt, seed=4)
    to = LlamaOracle(t, wt, keep_f64=True)
    K, T = 4, 1.0
    sd = SpecDecoder(to, LlamaOracle(d0, ws[0], keep_f64=True), prompt, 400)
    rep = LockstepReport()
    step = 0
    for _ in range(3):
        eng.step(K, T, eng.results_host)
        check_step(eng, sd, K, T, 4, step, rep)
        step += 1
    # switch: evict draft 1 to make room for draft 2, load it, make it active
    eng.evict_draft(1)
    assert eng.query_draft(1) == 0
    eng.load_draft_async(2)
    eng.set_active_draft(2)                         # waits for the copy on the GPU, catches up
    assert eng.query_draft(2) == 1
    do2 = LlamaOracle(d2, ws[2], keep_f64=True)
    sd.draft = do2
    sd.dc = do2.new_cache(400)
    do2.forward(sd.dc, sd.tokens[:-1], want_logits=False)   # the new draft's catch-up
    for _ in range(3):
        eng.step(K, T, eng.results_host)
        check_step(eng, sd, K, T, 4, step, rep)
        step += 1
    # draft 0 is still resident and becomes active again: it catches up from its old length
    eng.set_active_draft(0)
    sd.draft = LlamaOracle(d0, ws[0], keep_f64=True)
    sd.dc = sd.draft.new_cache(400)
    sd.draft.forward(sd.dc, sd.tokens[:-1], want_logits=False)
    for _ in range(2):
        eng.step(K, T, eng.results_host)
        check_step(eng, sd, K, T, 4, step, rep)
        step += 1
    print(f"switching: steps {rep.steps} flags {rep.flags}/{rep.decisions}")
    assert rep.flags <= 2
    eng.close()
