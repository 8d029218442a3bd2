"""Draft scheduling (CPU): the oracle's restatement of MemSpec's Algorithms 2-3
and of the MAB-Async baseline pinned to hand-worked traces, invariants and
closed forms; then the native scheduler (libmemspec.so, include/memspec_sched.h)
against the oracle, decision for decision, on seeded score streams through a
fake residency mechanism."""
import math

import numpy as np
import pytest

from oracle.scheduler import MAB_ASYNC, MEMSPEC, STATIC, FakeResidency, Scheduler, ranking
from seeded_inputs import gen_score_stream


# ---------------------------------------------------------------- oracle pins
def test_ranking_ties_go_to_the_lower_id():
    assert ranking([0.2, 0.5, 0.5, 0.1]) == [1, 2, 0, 3]


def test_memspec_trace_worked_by_hand():
    """Four drafts of equal size, capacity K = 2, the trace derived by hand from
    Algorithm 2 (top-K working set; evict outside W and never the active draft)
    and Algorithm 3 (run the best resident draft)."""
    mech = FakeResidency([1, 1, 1, 1], budget=2)
    s = Scheduler(4, 2, MEMSPEC)
    d = s.start(mech, [0.1, 0.5, 0.3, 0.1])
    # d0 = argmax = 1; W = {1, 2}: 2 is prefetched beside the active draft
    assert (d.active, d.prefetched, d.evicted) == (1, [2], [])
    mech.tick()
    d = s.point(mech, [0.6, 0.1, 0.2, 0.1])
    # W = {0, 2}; the cache {1, 2} is full and 1 is active, 2 is in W: nothing to
    # evict, so 0 is not fetched; the best resident draft is 2 (0.2 > 0.1)
    assert (d.active, d.desired, d.fallback, d.evicted, d.prefetched) == (2, 0, True, [], [])
    mech.tick()
    d = s.point(mech, [0.6, 0.1, 0.2, 0.1])
    # now 1 is neither active nor in W: evicted, and 0 is prefetched; 0 is still
    # loading, so the interval runs 2 (fallback)
    assert (d.active, d.desired, d.fallback, d.evicted, d.prefetched) == (2, 0, True, [1], [0])
    mech.tick()
    d = s.point(mech, [0.6, 0.1, 0.2, 0.1])
    assert (d.active, d.desired, d.fallback, d.evicted, d.prefetched) == (0, 0, False, [], [])
    assert mech.log == [("load", 1), ("active", 1), ("load", 2), ("active", 2), ("evict", 1),
                        ("load", 0), ("active", 0)]


def test_bytes_refusal_evicts_the_next_lowest_draft():
    """Drafts of different sizes: a load that does not fit the byte budget evicts
    the next lowest-scored unprotected draft and is retried (reading 4)."""
    mech = FakeResidency([5, 1, 1, 4], budget=6)
    s = Scheduler(4, 3, MEMSPEC)
    s.start(mech, [0.1, 0.9, 0.5, 0.2])            # d0 = 1; W = {1, 2, 3}
    assert [mech.state(d) for d in range(4)] == [0, 2, 2, 2]
    mech.tick()
    d = s.point(mech, [0.8, 0.9, 0.1, 0.05])       # W = {1, 0, 2}; 0 needs 5 bytes
    # capacity: 3 occupied -> evict the lowest-scored unprotected (3); then the
    # bytes (1 + 1 + 5 > 6) still refuse 0 and no unprotected draft is left
    assert d.evicted == [3] and d.prefetched == []
    assert mech.log[-2:] == [("evict", 3), ("refuse", 0)]


def _check_invariants(s, mech, d, scores, K):
    occ = [x for x in range(s.n) if mech.state(x) != 0]
    assert len(occ) <= K
    assert mech.state(s.active) != 0 and d.active == s.active
    if s.policy == MEMSPEC:
        elig = [x for x in range(s.n) if mech.state(x) == 1 or x == s.active]
        assert s.active == min(elig, key=lambda x: (-float(scores[x]), x))
        assert set(d.prefetched) <= set(ranking(scores)[:K])
    for v in d.evicted:
        assert v != s.active


@pytest.mark.parametrize("policy", [MEMSPEC, MAB_ASYNC, STATIC])
@pytest.mark.parametrize("n,K", [(5, 2), (3, 2), (6, 3)])
def test_invariants_on_seeded_streams(policy, n, K):
    scores = gen_score_stream(3, 60, n)
    mech = FakeResidency([1] * n, budget=K)
    s = Scheduler(n, K, policy)
    d = s.start(mech, scores[0])
    rng = np.random.default_rng(1)
    for i in range(1, 60):
        mech.tick()
        s.feedback(8, int(rng.integers(8, 40)))
        d = s.point(mech, scores[i])
        _check_invariants(s, mech, d, scores[i], K)
        if policy == STATIC:
            assert d.active == d.desired == s.active


def test_unlimited_cache_always_runs_the_best_draft():
    """K >= |D|: every draft becomes resident after the first interval, so
    MemSpec reduces to running the top-ranked draft at every point."""
    n = 4
    scores = gen_score_stream(5, 30, n)
    mech = FakeResidency([1] * n, budget=n)
    s = Scheduler(n, n, MEMSPEC)
    s.start(mech, scores[0])
    mech.tick()
    for i in range(1, 30):
        d = s.point(mech, scores[i])
        assert d.active == ranking(scores[i])[0] and not d.fallback


def test_mab_explores_every_draft_once_then_ucb():
    """MAB-Async with every draft resident: draft 0, 1, 2 in turn, then the UCB
    choice computed by hand: rewards 0.2, 0.6, 0.4 (t = 3, c = 2) give
    UCB = r + 2 sqrt(ln 3) for each, so draft 1; after a reward of 0.0 for it
    (t = 4): 0.2 + 2 sqrt(ln 4), 0.3 + 2 sqrt(ln 4 / 2), 0.4 + 2 sqrt(ln 4)
    -> draft 2."""
    mech = FakeResidency([1, 1, 1], budget=3)
    for d in range(3):
        mech.load(d)
    mech.tick()
    s = Scheduler(3, 3, MAB_ASYNC, ucb_c=2.0, k_draft=4)
    assert s.start(mech, None).active == 0
    s.feedback(10, 10)                      # reward 10 / 10 / 5 = 0.2
    assert s.point(mech, None).active == 1
    s.feedback(10, 30)                      # 0.6
    assert s.point(mech, None).active == 2
    s.feedback(10, 20)                      # 0.4
    u = [r + 2 * math.sqrt(math.log(3)) for r in (0.2, 0.6, 0.4)]
    assert np.argmax(u) == 1
    assert s.point(mech, None).active == 1
    s.feedback(10, 0)
    u = [0.2 + 2 * math.sqrt(math.log(4)), 0.3 + 2 * math.sqrt(math.log(4) / 2),
         0.4 + 2 * math.sqrt(math.log(4))]
    assert np.argmax(u) == 2
    assert s.point(mech, None).active == 2


def test_mab_falls_back_while_its_pick_loads():
    mech = FakeResidency([1, 1, 1], budget=2)
    s = Scheduler(3, 2, MAB_ASYNC)
    s.start(mech, None)
    mech.tick()
    s.feedback(4, 8)
    d = s.point(mech, None)                 # wants draft 1 (unexplored): loads it, runs 0
    assert (d.active, d.desired, d.fallback, d.prefetched) == (0, 1, True, [1])
    mech.tick()
    s.feedback(4, 8)
    d = s.point(mech, None)
    assert (d.active, d.desired, d.fallback) == (1, 1, False)


# ---------------------------------------------------------------- native vs oracle
def _native(n, K, policy, mech, c=2.0, k_draft=4):
    from paper_2608_10362_gb300 import DraftScheduler
    name = {MEMSPEC: "memspec", MAB_ASYNC: "mab_async", STATIC: "static"}[policy]
    return DraftScheduler(n, K, name, ucb_c=c, k_draft=k_draft, mechanism=mech)


@pytest.mark.parametrize("policy", [MEMSPEC, MAB_ASYNC, STATIC])
@pytest.mark.parametrize("n,K,sizes,budget", [(5, 2, [1] * 5, 2), (4, 3, [5, 1, 1, 4], 6),
                                               (3, 2, [2, 3, 4], 6), (8, 3, [1, 2, 3, 1, 2, 3, 1, 2], 6)])
def test_native_scheduler_matches_oracle(policy, n, K, sizes, budget):
    scores = gen_score_stream(11 + n + K, 80, n)
    m_o, m_n = FakeResidency(sizes, budget), FakeResidency(sizes, budget)
    so = Scheduler(n, K, policy, ucb_c=float(np.float32(2.0)), k_draft=4)
    sn = _native(n, K, policy, m_n)
    # the initial draft must fit alone
    first = ranking(scores[0])[0] if policy != MAB_ASYNC else 0
    assert sizes[first] <= budget
    do, dn = so.start(m_o, scores[0]), sn.start(scores[0])
    assert (do.active, do.evicted, do.prefetched) == (dn["active"], dn["evicted"], dn["prefetched"])
    rng = np.random.default_rng(n * 10 + K)
    for i in range(1, 80):
        m_o.tick()
        m_n.tick()
        it, tok = 8, int(rng.integers(8, 41))
        so.feedback(it, tok)
        sn.feedback(it, tok, 0.01)
        do, dn = so.point(m_o, scores[i]), sn.point(scores[i])
        assert (do.active, do.desired, do.fallback, do.evicted, do.prefetched) == \
            (dn["active"], dn["desired"], dn["fallback"], dn["evicted"], dn["prefetched"]), i
    assert m_o.log == m_n.log
    st = sn.stats()
    assert st["points"] == 80
    assert st["desired_intervals"] + st["fallback_intervals"] == 79
    sn.close()


def test_native_scheduler_rejects_bad_parameters():
    from paper_2608_10362_gb300 import DraftScheduler, MemSpecError
    mech = FakeResidency([1, 1], budget=2)
    with pytest.raises(MemSpecError):
        DraftScheduler(0, 1, mechanism=mech)
    with pytest.raises(MemSpecError):
        DraftScheduler(2, 0, mechanism=mech)
    s = DraftScheduler(2, 1, mechanism=mech)
    with pytest.raises(MemSpecError):
        s.point([0.1, 0.2])                 # before start
