"""Device-side error reporting (GPU, through the C ABI).

The kernels never trap: a token id outside the vocabulary is clamped to id 0 and
reported, a position beyond max_seq is skipped and reported, and memspec_sync
returns MEMSPEC_ERR_DEVICE_STATUS with the status bits, then clears them so the
context stays usable.  The faults are planted on the host (buffer writes), and
every access stays in bounds.  A host-side wait that runs out returns
MEMSPEC_ERR_TIMEOUT while the stream keeps running a finite kernel.
"""
import ctypes as C

import numpy as np
import pytest
import torch

from lockstep import LockstepReport, check_step
from oracle.llama import LlamaOracle
from oracle.speculative import SpecDecoder
from seeded_inputs import SHAPES, gen_prompt, gen_weights

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def tiny_engine():
    from paper_2608_10362_gb300 import Engine
    t, d = SHAPES["tiny_target"], SHAPES["tiny_draft"]
    wt, wd = gen_weights(t, 0), gen_weights(d, 1)
    eng = Engine(t, wt, max_batch=1, max_seq=256, max_k=4, max_drafts=1, draft_shape_max=d,
                 draft_budget_bytes=16 << 20, use_graphs=True)
    eng.register_draft(0, d, wd)
    eng.load_draft_async(0)
    eng.set_active_draft(0)
    yield eng, LlamaOracle(t, wt), LlamaOracle(d, wd)
    eng.close()


def _sync_bits(eng, timeout_ms=-1):
    from paper_2608_10362_gb300 import _lib
    bits = C.c_uint32()
    st = eng.lib.memspec_sync(eng.ctx, timeout_ms, C.byref(bits))
    return st, bits.value


def _clean_step_after(eng, to, do, seed):
    """A fresh request steps cleanly and matches the oracle after an error."""
    prompt = gen_prompt(seed, 40, 2048)
    eng.prefill(0, prompt, seed=seed)
    sd = SpecDecoder(to, do, prompt, 64)
    rep = LockstepReport()
    eng.step(4, 1.0, eng.results_host)
    check_step(eng, sd, 4, 1.0, seed, 0, rep)
    assert rep.band_flags == 0


def test_out_of_range_token_is_reported(tiny_engine):
    from paper_2608_10362_gb300 import _lib
    eng, to, do = tiny_engine
    eng.prefill(0, gen_prompt(3, 40, 2048), seed=1)
    assert eng.sync() == 0
    dt = np.zeros((1, eng.max_k), dtype=np.int32)
    dt[0, :4] = [5, 2048 + 7, -3, 11]                 # two ids outside [0, vocab)
    eng.write_buffer(_lib.BUF_DRAFT_TOKENS, dt)
    eng.verify_step(4)                                # embeds [t_{L-1}, x_1..x_4]
    st, bits = _sync_bits(eng)
    assert st == _lib.ERR_DEVICE_STATUS
    assert bits & _lib.DEV_BAD_TOKEN
    assert not bits & _lib.DEV_TIMEOUT
    st, bits = _sync_bits(eng)                        # the word was cleared
    assert st == _lib.OK and bits == 0
    _clean_step_after(eng, to, do, 12)


def test_sequence_beyond_max_seq_is_reported(tiny_engine):
    from paper_2608_10362_gb300 import _lib
    eng, to, do = tiny_engine
    eng.prefill(0, gen_prompt(4, 40, 2048), seed=1)
    assert eng.sync() == 0
    # committed length max_seq - 2: the verify rows sit at positions
    # max_seq - 3 .. max_seq + 1, three of them beyond the cache
    state = eng.seq_state().copy()
    L = eng.max_seq - 2
    state[0, :3] = (L, L - 1, 0)
    eng.write_buffer(_lib.BUF_SEQ_STATE, state)
    eng.verify_step(4)
    st, bits = _sync_bits(eng)
    assert st == _lib.ERR_DEVICE_STATUS
    assert bits & _lib.DEV_BAD_LENGTH
    assert not bits & _lib.DEV_TIMEOUT
    # the acceptance step refuses to commit past max_seq and reports it too
    eng.prefill(0, gen_prompt(5, 40, 2048), seed=1)
    state = eng.seq_state().copy()
    state[0, :3] = (eng.max_seq, eng.max_seq - 1, 0)     # no room for even one token
    eng.write_buffer(_lib.BUF_SEQ_STATE, state)
    eng.accept_commit(4, 1.0, None)
    st, bits = _sync_bits(eng)
    assert st == _lib.ERR_DEVICE_STATUS and bits & _lib.DEV_BAD_LENGTH
    assert int(eng.seq_state()[0, 0]) == eng.max_seq        # nothing committed
    _clean_step_after(eng, to, do, 13)


def test_sync_timeout_on_a_busy_stream(tiny_engine):
    """memspec_sync with a 1 ms limit while the main stream runs a finite
    ~0.5 s spin kernel: TIMEOUT, then an unlimited sync succeeds."""
    from paper_2608_10362_gb300 import _lib
    eng, _, _ = tiny_engine
    assert eng.sync() == 0
    with torch.cuda.stream(eng.stream):
        torch.cuda._sleep(1_000_000_000)            # clock cycles: about 0.5 s at 2 GHz
    st, _ = _sync_bits(eng, timeout_ms=1)
    assert st == _lib.ERR_TIMEOUT
    assert b"timed out" in eng.lib.memspec_last_error(eng.ctx)
    st, bits = _sync_bits(eng, timeout_ms=-1)
    assert st == _lib.OK and bits == 0
