"""Binding of the host-side draft scheduler (include/memspec_sched.h): MemSpec's
cache update and runtime-loop policy, the MAB-Async baseline and a static
policy, acting on an Engine's draft calls or on a caller-supplied residency
mechanism.  Argument marshalling only; the decisions are made in libmemspec.so.
"""
from __future__ import annotations

import ctypes as C

import numpy as np

from . import _lib
from ._lib import MemSpecError

POLICIES = {"memspec": _lib.POLICY_MEMSPEC, "mab_async": _lib.POLICY_MAB_ASYNC,
            "static": _lib.POLICY_STATIC}


def _decision(d: _lib.SchedDecision) -> dict:
    return {"active": d.active, "desired": d.desired, "fallback": bool(d.fallback),
            "evicted": list(d.evicted[:d.n_evicted]), "prefetched": list(d.prefetched[:d.n_prefetched])}


class DraftScheduler:
    """policy: "memspec", "mab_async" or "static".  Either ``engine`` (its ctx's
    draft calls) or ``mechanism`` (an object with state(d) -> 0/1/2, load(d) ->
    bool (False: the bytes do not fit), evict(d), set_active(d)) drives the
    residency."""

    def __init__(self, n_drafts: int, capacity: int, policy: str = "memspec", ucb_c: float = 2.0,
                 k_draft: int = 4, engine=None, mechanism=None):
        self.lib = _lib.load()
        p = _lib.SchedParams(n_drafts, capacity, POLICIES[policy], ucb_c, k_draft)
        self.n = n_drafts
        h = C.c_void_p()
        self._keep = None
        if mechanism is not None:
            def state(_u, d, out):
                out[0] = int(mechanism.state(d))
                return _lib.OK

            def load(_u, d):
                return _lib.OK if mechanism.load(d) else _lib.ERR_BUDGET

            def evict(_u, d):
                mechanism.evict(d)
                return _lib.OK

            def set_active(_u, d):
                mechanism.set_active(d)
                return _lib.OK

            mech = _lib.Residency(None, _lib.STATE_FN(state), _lib.DRAFT_FN(load),
                                  _lib.DRAFT_FN(evict), _lib.DRAFT_FN(set_active))
            self._keep = mech            # the callbacks must outlive the scheduler
            st = self.lib.memspec_sched_create(C.byref(p), C.byref(mech), None, C.byref(h))
        else:
            st = self.lib.memspec_sched_create(C.byref(p), None, engine.ctx, C.byref(h))
        if st != _lib.OK:
            raise MemSpecError(st, "memspec_sched_create")
        self.h = h

    def _scores(self, scores):
        if scores is None:
            return None, None
        arr = np.ascontiguousarray(np.asarray(scores, dtype=np.float32))
        assert arr.shape == (self.n,)
        return arr, arr.ctypes.data

    def _call(self, fn, scores):
        arr, ptr = self._scores(scores)
        d = _lib.SchedDecision()
        st = fn(self.h, ptr, C.byref(d))
        if st != _lib.OK:
            raise MemSpecError(st, fn.__name__)
        return _decision(d)

    def start(self, scores=None) -> dict:
        return self._call(self.lib.memspec_sched_start, scores)

    def point(self, scores=None) -> dict:
        return self._call(self.lib.memspec_sched_point, scores)

    def feedback(self, iterations: int, tokens: int, seconds: float = 0.0):
        st = self.lib.memspec_sched_feedback(self.h, iterations, tokens, float(seconds))
        if st != _lib.OK:
            raise MemSpecError(st, "memspec_sched_feedback")

    def stats(self) -> dict:
        s = _lib.SchedStats()
        st = self.lib.memspec_sched_get_stats(self.h, C.byref(s))
        if st != _lib.OK:
            raise MemSpecError(st, "memspec_sched_get_stats")
        return {name: getattr(s, name) for name, _ in s._fields_}

    def close(self):
        if getattr(self, "h", None):
            self.lib.memspec_sched_destroy(self.h)
            self.h = None

    def __del__(self):  # pragma: no cover
        try:
            self.close()
        except Exception:
            pass
