"""Draft scheduling policies over a resident draft cache (oracle side).

Test infrastructure only (see ``oracle/__init__``).  Plain-Python restatement of
the host-side control logic the CUDA path's C ABI is driven by:

* MemSpec (Section 3.1 design overview, Section 3.3 Algorithm 2 "Draft Model
  Cache Update", Section 3.4 Algorithm 3 "MemSpec Runtime Loop"): every N
  iterations the drafts are ranked by their predicted scores p_i(d); the target
  working set W_i is the top-K of that ranking; each draft of W_i that is
  neither resident nor being loaded is prefetched asynchronously, after
  evicting, while the cache is full, the lowest-scored resident draft outside
  W_i and other than the active draft; the next interval runs the best draft
  that is resident now (never a draft still loading).
* MAB-Async (Section 2.3, and the baseline of Section 4.1 with c = 2.0): a UCB
  bandit over the drafts that first runs every draft once, then picks
  argmax_d mean_reward(d) + c sqrt(ln t / n_d); when the pick is not resident
  its load starts asynchronously and decoding continues with the resident
  active draft.
* Static: the initial draft for the whole run.

Readings where the paper is silent (each restated in the native scheduler):

1. The capacity K counts drafts that are resident or being loaded: a prefetch
   occupies its slot from the moment it starts.
2. Ties in a ranking go to the lower draft id; the eviction victim among equal
   scores is the one ranked last (the higher id).
3. A draft still being loaded is neither eligible to run nor evictable, except
   the active draft itself (the initial draft may still be loading; the step
   then waits for its copy on the GPU).
4. A load the mechanism refuses for lack of bytes (drafts differ in size)
   evicts the next lowest-scored unprotected resident draft and is retried;
   when none is left, the prefetch is skipped for this scheduling point.
5. MAB-Async reward of an interval: committed tokens per iteration divided by
   K_draft + 1 (in [0, 1]), credited to the draft that actually ran; t counts
   the intervals run so far; the eviction victim for a MAB load is the resident,
   non-active draft of lowest UCB value.
6. Execution breakdown (Section 4.3): an interval is "desired" when the draft
   that ran is the one the policy wanted for it, else "fallback".

The residency mechanism is an object with ``state(d)`` (0 absent, 1 resident,
2 loading), ``load(d)`` (True, or False when the bytes do not fit),
``evict(d)`` and ``set_active(d)``.
"""
from __future__ import annotations

import dataclasses
import math

MEMSPEC, MAB_ASYNC, STATIC = 0, 1, 2


def ranking(scores):
    """Draft ids sorted by descending score, ties to the lower id."""
    return sorted(range(len(scores)), key=lambda d: (-float(scores[d]), d))


@dataclasses.dataclass
class Decision:
    active: int
    desired: int
    fallback: bool
    evicted: list
    prefetched: list


class Scheduler:
    def __init__(self, n_drafts: int, capacity: int, policy: int = MEMSPEC, ucb_c: float = 2.0,
                 k_draft: int = 4):
        self.n, self.K, self.policy, self.c, self.k_draft = n_drafts, capacity, policy, ucb_c, k_draft
        self.active = -1
        self.pulls = [0] * n_drafts
        self.reward_sum = [0.0] * n_drafts
        self.t = 0
        self.last_desired = -1

    # ------------------------------------------------------------ cache update
    def _occupied(self, mech):
        return [d for d in range(self.n) if mech.state(d) != 0]

    def _evict_one(self, mech, protected, key):
        """Evict the resident, unprotected draft with the lowest key (ties: the
        later in ranking order, i.e. the higher id); None if there is none."""
        cands = [d for d in range(self.n) if mech.state(d) == 1 and d not in protected]
        if not cands:
            return None
        victim = min(cands, key=lambda d: (key(d), -d))
        mech.evict(victim)
        return victim

    def update_cache(self, mech, scores):
        """Algorithm 2 with readings 1-4; returns (evicted, prefetched)."""
        R = ranking(scores)
        W = R[:self.K]
        protected = set(W) | {self.active}
        evicted, prefetched = [], []
        for d in W:
            if mech.state(d) != 0:
                continue                        # resident or being prefetched
            while len(self._occupied(mech)) >= self.K:
                v = self._evict_one(mech, protected, lambda x: float(scores[x]))
                if v is None:
                    break
                evicted.append(v)
            if len(self._occupied(mech)) < self.K:
                while not mech.load(d):
                    v = self._evict_one(mech, protected, lambda x: float(scores[x]))
                    if v is None:
                        break
                    evicted.append(v)
                if mech.state(d) != 0:
                    prefetched.append(d)
        return evicted, prefetched

    # ------------------------------------------------------------ policies
    def start(self, mech, scores):
        """Algorithm 3 lines 2-5: initial draft from the prompt's scores, loaded
        (the caller waits for it), then the cache is prepared."""
        d0 = ranking(scores)[0] if self.policy != MAB_ASYNC else 0
        if mech.state(d0) == 0:
            assert mech.load(d0), "the initial draft must fit the budget"
        self.active = d0
        mech.set_active(d0)
        ev, pf = self.update_cache(mech, scores) if self.policy == MEMSPEC else ([], [])
        self.last_desired = d0
        return Decision(d0, d0, False, ev, pf)

    def _ucb(self, d):
        if self.pulls[d] == 0:
            return math.inf
        mean = self.reward_sum[d] / self.pulls[d]
        return mean + self.c * math.sqrt(math.log(max(self.t, 1)) / self.pulls[d])

    def point(self, mech, scores):
        """A scheduling point (Algorithm 3 lines 14-18 for MemSpec)."""
        if self.policy == STATIC:
            self.last_desired = self.active
            return Decision(self.active, self.active, False, [], [])
        if self.policy == MEMSPEC:
            desired = ranking(scores)[0]
            ev, pf = self.update_cache(mech, scores)
            eligible = [d for d in range(self.n) if mech.state(d) == 1 or d == self.active]
            nxt = min(eligible, key=lambda d: (-float(scores[d]), d))
        else:
            ucb = [self._ucb(d) for d in range(self.n)]
            desired = min(range(self.n), key=lambda d: (-ucb[d], d))
            ev, pf = [], []
            if mech.state(desired) == 0:
                protected = {self.active}
                while len(self._occupied(mech)) >= self.K:
                    v = self._evict_one(mech, protected, lambda x: ucb[x])
                    if v is None:
                        break
                    ev.append(v)
                if len(self._occupied(mech)) < self.K:
                    while not mech.load(desired):
                        v = self._evict_one(mech, protected, lambda x: ucb[x])
                        if v is None:
                            break
                        ev.append(v)
                    if mech.state(desired) != 0:
                        pf.append(desired)
            nxt = desired if mech.state(desired) == 1 else self.active
        if nxt != self.active:
            self.active = nxt
            mech.set_active(nxt)
        self.last_desired = desired
        return Decision(nxt, desired, nxt != desired, ev, pf)

    def feedback(self, iterations: int, tokens: int):
        """Reward of the interval just run, credited to the active draft (MAB)."""
        if iterations <= 0:
            return
        self.t += 1
        r = tokens / iterations / (self.k_draft + 1)
        self.pulls[self.active] += 1
        self.reward_sum[self.active] += r


class FakeResidency:
    """Residency mechanism with byte sizes and a budget; loads complete when
    ``tick`` is called (the next scheduling point), as an asynchronous copy
    overlapped with one interval would."""

    def __init__(self, sizes, budget):
        self.sizes, self.budget = list(sizes), budget
        self.st = [0] * len(sizes)
        self.active = -1
        self.log = []

    def state(self, d):
        return self.st[d]

    def used(self):
        return sum(self.sizes[d] for d in range(len(self.st)) if self.st[d] != 0)

    def load(self, d):
        if self.st[d] != 0:
            return True
        if self.used() + self.sizes[d] > self.budget:
            self.log.append(("refuse", d))
            return False
        self.st[d] = 2
        self.log.append(("load", d))
        return True

    def evict(self, d):
        assert self.st[d] == 1 and d != self.active
        self.st[d] = 0
        self.log.append(("evict", d))

    def set_active(self, d):
        assert self.st[d] != 0
        self.active = d
        self.log.append(("active", d))

    def tick(self):
        self.st = [1 if s == 2 else s for s in self.st]
