"""End-to-end parity of the draft-then-verify step on the GPU against the oracle,
in lock step (tests/lockstep.py), on the tiny pair: every launch mode at T = 0
and T = 1, a batch of four requests, the greedy stream against greedy
target-only decoding, and prompt edge cases."""
import numpy as np
import pytest

from lockstep import LOGIT_TOL, RECORDS, LockstepReport, check_step
from oracle.llama import LlamaOracle
from oracle.speculative import SpecDecoder, argmax_first, greedy_generate
from seeded_inputs import SHAPES, gen_prompt, gen_weights

pytestmark = pytest.mark.gpu


def _run_lockstep(eng, target_o, draft_o, prompt, K, T, seed, steps):
    eng.prefill(0, prompt, seed=seed)
    sd = SpecDecoder(target_o, draft_o, prompt, len(prompt) + steps * (K + 1) + 4)
    rep = LockstepReport()
    for step in range(steps):
        eng.step(K, T, eng.results_host)
        check_step(eng, sd, K, T, seed, step, rep)
    return rep, sd


# (CUDA graphs, launch mode): per-op launches with and without graphs, and the
# persistent pass kernel
MODES = [(False, "per_op"), (True, "per_op"), (True, "pass"), (False, "pass")]


def _engine(t, wt, d, wd, graphs, launch, max_batch=1, draft_kernel="auto"):
    from paper_2608_10362_gb300 import Engine
    eng = Engine(t, wt, max_batch=max_batch, max_seq=512, max_k=8, max_drafts=1,
                 draft_shape_max=d, draft_budget_bytes=32 << 20, use_graphs=graphs,
                 launch_mode=launch, draft_kernel=draft_kernel)
    eng.register_draft(0, d, wd)
    eng.load_draft_async(0)
    eng.set_active_draft(0)
    return eng


@pytest.fixture(scope="module")
def tiny():
    t, d = SHAPES["tiny_target"], SHAPES["tiny_draft"]
    wt, wd = gen_weights(t, 0), gen_weights(d, 1)
    engines = {mode: _engine(t, wt, d, wd, *mode) for mode in MODES}
    yield engines, LlamaOracle(t, wt), LlamaOracle(d, wd), (t, wt, d, wd)
    for e in engines.values():
        e.close()


@pytest.mark.parametrize("mode", MODES, ids=lambda m: f"graphs{int(m[0])}-{m[1]}")
@pytest.mark.parametrize("T", [0.0, 1.0])
def test_tiny_pair_lockstep(tiny, T, mode):
    engines, to, do, _ = tiny
    eng = engines[mode]
    prompt = gen_prompt(7, 128, 2048)
    rep, sd = _run_lockstep(eng, to, do, prompt, 4, T, seed=3, steps=16)
    line = rep.record(f"tiny T={T} graphs={int(mode[0])} {mode[1]}")
    assert rep.band_flags == 0, line
    assert list(eng.committed_tokens(0)) == sd.tokens


def test_tiny_pair_lockstep_per_op_draft_path(tiny):
    """The draft step through the per-op kernels (the path larger drafts take),
    T = 1."""
    _, to, do, (t, wt, d, wd) = tiny
    eng = _engine(t, wt, d, wd, True, "per_op", draft_kernel="per_op")
    prompt = gen_prompt(17, 128, 2048)
    rep, sd = _run_lockstep(eng, to, do, prompt, 4, 1.0, seed=13, steps=12)
    line = rep.record("tiny T=1.0 per-op draft kernels")
    eng.close()
    assert rep.band_flags == 0, line


@pytest.mark.parametrize("T", [0.0, 1.0])
@pytest.mark.parametrize("launch", ["per_op", "pass"])
def test_tiny_pair_lockstep_batch4(tiny, T, launch):
    """Four requests stepped together (per-request lengths, Philox keys and
    KV caches): draft step, verify pass and acceptance at B = 4."""
    _, to, do, (t, wt, d, wd) = tiny
    B, K, steps = 4, 4, 8
    eng = _engine(t, wt, d, wd, True, launch, max_batch=B)
    lens = [128, 61, 130, 97]
    seeds = [21, 22, 23, 24]
    sds = []
    for b in range(B):
        prompt = gen_prompt(40 + b, lens[b], 2048)
        eng.prefill(b, prompt, seed=seeds[b])
        sds.append(SpecDecoder(to, do, prompt, len(prompt) + steps * (K + 1) + 4))
    eng.set_batch(B)
    rep = LockstepReport()
    for step in range(steps):
        eng.step(K, T, eng.results_host)
        bits = eng.sync()
        for b in range(B):
            check_step(eng, sds[b], K, T, seeds[b], step, rep, req=b, batch=B, bits=bits)
        res = eng.results_host.numpy()[:B * (K + 2)].reshape(B, K + 2)
        for b in range(B):      # the pinned result rows agree with the committed tokens
            n = int(res[b, 0])
            assert list(res[b, 1:n + 2]) == sds[b].tokens[-(n + 1):]
    line = rep.record(f"tiny B=4 T={T} {launch}")
    for b in range(B):
        assert list(eng.committed_tokens(b)) == sds[b].tokens
    eng.close()
    assert rep.band_flags == 0, line


def test_tiny_greedy_stream_equals_oracle_target_greedy(tiny):
    """Greedy speculative output == greedy target-only output, token for token,
    over the whole stream.  A divergence is allowed only where the oracle's two
    candidates are closer than the logit tolerance (0.03 max|z|); it is
    counted, the GPU is resynchronised to the oracle's token (prefill of the
    prompt plus the oracle's tokens so far) and the comparison continues."""
    engines, to, do, _ = tiny
    eng = engines[(True, "per_op")]
    n_new = 40
    flagged = []
    for seed in (8, 9, 10):
        prompt = [int(x) for x in gen_prompt(seed, 128, 2048)]
        ref = greedy_generate(to, prompt, n_new)
        i = 0
        while i < n_new:
            ctx = prompt + ref[:i]
            eng.prefill(0, ctx, seed=0)
            while int(eng.seq_state()[0, 0]) < len(ctx) + (n_new - i):
                eng.step(4, 0.0, eng.results_host)
                assert eng.sync() == 0
            got = [int(t) for t in eng.committed_tokens(0)[len(ctx):len(ctx) + n_new - i]]
            j = next((k for k in range(len(got)) if got[k] != ref[i + k]), None)
            if j is None:
                break
            pos = i + j
            z = to.forward(to.new_cache(len(prompt) + pos + 1), prompt + ref[:pos])[-1]
            gap = float(z[ref[pos]] - z[got[j]])
            assert ref[pos] == argmax_first(z)
            assert 0 <= gap < LOGIT_TOL * np.abs(z).max(), (seed, pos, gap)
            flagged.append((seed, pos, f"{gap / np.abs(z).max():.2e}"))
            i = pos + 1                        # resync on the oracle's token
    RECORDS.append(f"tiny greedy streams (3 x {n_new} tokens): tolerance-flags {len(flagged)} "
                   f"{flagged}")


def test_tiny_prompt_edge_cases(tiny):
    """Prompt of one token (nothing to prefill) and a prompt crossing the
    128-row prefill chunk boundary by one."""
    engines, to, do, _ = tiny
    eng = engines[(False, "per_op")]
    for n in (1, 129):
        prompt = gen_prompt(9 + n, n, 2048)
        rep, sd = _run_lockstep(eng, to, do, prompt, 3, 1.0, seed=5, steps=4)
        rep.record(f"tiny prompt length {n}")
        assert rep.steps == 4
        assert rep.band_flags == 0
