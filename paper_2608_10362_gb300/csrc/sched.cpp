// sched.cpp - MemSpec's draft scheduler (Algorithms 2 and 3), the MAB-Async
// baseline and a static policy, on the draft-residency calls of the C ABI.
// Host code only; the readings it follows are listed in include/memspec_sched.h.
#include <chrono>
#include <cmath>
#include <limits>
#include <vector>

#include "../../include/memspec_sched.h"

struct memspec_sched {
  memspec_sched_params p{};
  memspec_residency mech{};
  memspec_ctx* ctx = nullptr;
  bool started = false;
  int active = -1;
  int last_desired = -1;
  bool last_fallback = false;
  std::vector<int64_t> pulls;
  std::vector<double> reward_sum;
  int64_t t = 0;
  memspec_sched_stats st{};
};

namespace {

using Clock = std::chrono::steady_clock;

// ctx-backed mechanism
int32_t ctx_state(void* u, int32_t d, int32_t* s) {
  return memspec_query_draft(static_cast<memspec_ctx*>(u), d, s);
}
int32_t ctx_load(void* u, int32_t d) {
  return memspec_load_draft_async(static_cast<memspec_ctx*>(u), d, nullptr);
}
int32_t ctx_evict(void* u, int32_t d) { return memspec_evict_draft(static_cast<memspec_ctx*>(u), d); }
int32_t ctx_set_active(void* u, int32_t d) {
  return memspec_set_active_draft(static_cast<memspec_ctx*>(u), d);
}

struct Op {   // a status-carrying step
  memspec_status s = MEMSPEC_OK;
  bool ok() const { return s == MEMSPEC_OK; }
};

memspec_status state_of(memspec_sched* S, int d, int* out) {
  int32_t v = 0;
  const int32_t r = S->mech.state(S->mech.user, d, &v);
  *out = v;
  return static_cast<memspec_status>(r);
}

// Ranking: descending score, ties to the lower id.
bool ranks_before(const float* sc, int a, int b) {
  return sc[a] > sc[b] || (sc[a] == sc[b] && a < b);
}

std::vector<int> ranking(const float* sc, int n) {
  std::vector<int> r;
  for (int d = 0; d < n; ++d) {
    size_t i = 0;
    while (i < r.size() && ranks_before(sc, r[i], d)) ++i;
    r.insert(r.begin() + static_cast<long>(i), d);
  }
  return r;
}

memspec_status occupied(memspec_sched* S, int* count) {
  int c = 0;
  for (int d = 0; d < S->p.n_drafts; ++d) {
    int st = 0;
    memspec_status e = state_of(S, d, &st);
    if (e != MEMSPEC_OK) return e;
    if (st != 0) ++c;
  }
  *count = c;
  return MEMSPEC_OK;
}

// Evict the resident, unprotected draft with the lowest key (ties: the higher
// id).  *victim = -1 when there is none.
template <class Key>
memspec_status evict_one(memspec_sched* S, const std::vector<bool>& prot, Key key, int* victim,
                         memspec_sched_decision* dec) {
  int v = -1;
  double vk = 0.0;
  for (int d = 0; d < S->p.n_drafts; ++d) {
    int st = 0;
    memspec_status e = state_of(S, d, &st);
    if (e != MEMSPEC_OK) return e;
    if (st != 1 || prot[d]) continue;
    const double k = key(d);
    if (v < 0 || k < vk || (k == vk && d > v)) {
      v = d;
      vk = k;
    }
  }
  *victim = v;
  if (v < 0) return MEMSPEC_OK;
  memspec_status e = static_cast<memspec_status>(S->mech.evict(S->mech.user, v));
  if (e != MEMSPEC_OK) return e;
  ++S->st.evictions;
  if (dec->n_evicted < MEMSPEC_SCHED_MAX_DRAFTS) dec->evicted[dec->n_evicted++] = v;
  return MEMSPEC_OK;
}

// Make room for draft d (capacity K, then bytes) and start its load.
template <class Key>
memspec_status prefetch(memspec_sched* S, int d, const std::vector<bool>& prot, Key key,
                        memspec_sched_decision* dec) {
  int occ = 0, victim = 0;
  memspec_status e = occupied(S, &occ);
  if (e != MEMSPEC_OK) return e;
  while (occ >= S->p.capacity) {
    e = evict_one(S, prot, key, &victim, dec);
    if (e != MEMSPEC_OK) return e;
    if (victim < 0) break;
    --occ;
  }
  if (occ >= S->p.capacity) return MEMSPEC_OK;
  for (;;) {
    const int32_t r = S->mech.load(S->mech.user, d);
    if (r == MEMSPEC_OK) break;
    if (r != MEMSPEC_ERR_BUDGET) return static_cast<memspec_status>(r);
    ++S->st.refusals;
    e = evict_one(S, prot, key, &victim, dec);
    if (e != MEMSPEC_OK) return e;
    if (victim < 0) return MEMSPEC_OK;   // skipped at this scheduling point
  }
  int st = 0;
  e = state_of(S, d, &st);
  if (e != MEMSPEC_OK) return e;
  if (st != 0) {
    ++S->st.loads;
    if (dec->n_prefetched < MEMSPEC_SCHED_MAX_DRAFTS) dec->prefetched[dec->n_prefetched++] = d;
  }
  return MEMSPEC_OK;
}

// Algorithm 2.
memspec_status update_cache(memspec_sched* S, const float* sc, memspec_sched_decision* dec) {
  const int n = S->p.n_drafts;
  const std::vector<int> R = ranking(sc, n);
  const int top = std::min(n, S->p.capacity);
  std::vector<bool> prot(n, false);
  for (int i = 0; i < top; ++i) prot[R[i]] = true;
  if (S->active >= 0) prot[S->active] = true;
  for (int i = 0; i < top; ++i) {
    const int d = R[i];
    int st = 0;
    memspec_status e = state_of(S, d, &st);
    if (e != MEMSPEC_OK) return e;
    if (st != 0) continue;
    e = prefetch(S, d, prot, [&](int x) { return static_cast<double>(sc[x]); }, dec);
    if (e != MEMSPEC_OK) return e;
  }
  return MEMSPEC_OK;
}

double ucb(const memspec_sched* S, int d) {
  if (S->pulls[d] == 0) return std::numeric_limits<double>::infinity();
  const double mean = S->reward_sum[d] / static_cast<double>(S->pulls[d]);
  const double t = static_cast<double>(S->t > 1 ? S->t : 1);
  return mean + static_cast<double>(S->p.ucb_c) * std::sqrt(std::log(t) / static_cast<double>(S->pulls[d]));
}

memspec_status set_active(memspec_sched* S, int d) {
  if (d == S->active) return MEMSPEC_OK;
  memspec_status e = static_cast<memspec_status>(S->mech.set_active(S->mech.user, d));
  if (e != MEMSPEC_OK) return e;
  if (S->active >= 0) ++S->st.switches;
  S->active = d;
  return MEMSPEC_OK;
}

void clear(memspec_sched_decision* dec) { *dec = memspec_sched_decision{}; }

}  // namespace

extern "C" {

memspec_status memspec_sched_create(const memspec_sched_params* p, const memspec_residency* mech,
                                    memspec_ctx* ctx, memspec_sched** out) {
  if (p == nullptr || out == nullptr) return MEMSPEC_ERR_INVALID_ARG;
  *out = nullptr;
  if (p->n_drafts < 1 || p->n_drafts > MEMSPEC_SCHED_MAX_DRAFTS || p->capacity < 1 ||
      p->policy < MEMSPEC_POLICY_MEMSPEC || p->policy > MEMSPEC_POLICY_STATIC || !(p->ucb_c >= 0.f) ||
      p->k_draft < 1)
    return MEMSPEC_ERR_INVALID_ARG;
  if (mech == nullptr && ctx == nullptr) return MEMSPEC_ERR_INVALID_ARG;
  if (mech != nullptr && (mech->state == nullptr || mech->load == nullptr || mech->evict == nullptr ||
                          mech->set_active == nullptr))
    return MEMSPEC_ERR_INVALID_ARG;
  memspec_sched* S = new memspec_sched();
  S->p = *p;
  if (mech != nullptr) {
    S->mech = *mech;
  } else {
    S->ctx = ctx;
    S->mech = memspec_residency{ctx, ctx_state, ctx_load, ctx_evict, ctx_set_active};
  }
  S->pulls.assign(p->n_drafts, 0);
  S->reward_sum.assign(p->n_drafts, 0.0);
  *out = S;
  return MEMSPEC_OK;
}

void memspec_sched_destroy(memspec_sched* s) { delete s; }

memspec_status memspec_sched_start(memspec_sched* S, const float* sc, memspec_sched_decision* dec) {
  if (S == nullptr || dec == nullptr || (sc == nullptr && S->p.policy == MEMSPEC_POLICY_MEMSPEC))
    return MEMSPEC_ERR_INVALID_ARG;
  const auto t0 = Clock::now();
  clear(dec);
  const int d0 = (S->p.policy == MEMSPEC_POLICY_MAB_ASYNC || sc == nullptr) ? 0 : ranking(sc, S->p.n_drafts)[0];
  int st = 0;
  memspec_status e = state_of(S, d0, &st);
  if (e == MEMSPEC_OK && st == 0) {
    e = static_cast<memspec_status>(S->mech.load(S->mech.user, d0));
    if (e == MEMSPEC_OK) ++S->st.loads;
  }
  if (e == MEMSPEC_OK) e = set_active(S, d0);
  if (e == MEMSPEC_OK && S->p.policy == MEMSPEC_POLICY_MEMSPEC) e = update_cache(S, sc, dec);
  if (e != MEMSPEC_OK) return e;
  S->started = true;
  S->last_desired = d0;
  S->last_fallback = false;
  dec->active = d0;
  dec->desired = d0;
  dec->fallback = 0;
  ++S->st.points;
  S->st.policy_s += std::chrono::duration<double>(Clock::now() - t0).count();
  return MEMSPEC_OK;
}

memspec_status memspec_sched_point(memspec_sched* S, const float* sc, memspec_sched_decision* dec) {
  if (S == nullptr || dec == nullptr || !S->started ||
      (sc == nullptr && S->p.policy == MEMSPEC_POLICY_MEMSPEC))
    return MEMSPEC_ERR_INVALID_ARG;
  const auto t0 = Clock::now();
  clear(dec);
  const int n = S->p.n_drafts;
  int desired = S->active, next = S->active;
  memspec_status e = MEMSPEC_OK;
  if (S->p.policy == MEMSPEC_POLICY_MEMSPEC) {
    desired = ranking(sc, n)[0];
    e = update_cache(S, sc, dec);
    if (e != MEMSPEC_OK) return e;
    next = -1;
    for (int d = 0; d < n; ++d) {
      int st = 0;
      e = state_of(S, d, &st);
      if (e != MEMSPEC_OK) return e;
      if (st != 1 && d != S->active) continue;
      if (next < 0 || ranks_before(sc, d, next)) next = d;
    }
  } else if (S->p.policy == MEMSPEC_POLICY_MAB_ASYNC) {
    std::vector<double> u(n);
    for (int d = 0; d < n; ++d) u[d] = ucb(S, d);
    desired = 0;
    for (int d = 1; d < n; ++d)
      if (u[d] > u[desired]) desired = d;
    int st = 0;
    e = state_of(S, desired, &st);
    if (e != MEMSPEC_OK) return e;
    if (st == 0) {
      std::vector<bool> prot(n, false);
      prot[S->active] = true;
      e = prefetch(S, desired, prot, [&](int x) { return u[x]; }, dec);
      if (e != MEMSPEC_OK) return e;
      e = state_of(S, desired, &st);
      if (e != MEMSPEC_OK) return e;
    }
    next = st == 1 ? desired : S->active;
  }
  e = set_active(S, next);
  if (e != MEMSPEC_OK) return e;
  S->last_desired = desired;
  S->last_fallback = next != desired;
  dec->active = next;
  dec->desired = desired;
  dec->fallback = next != desired ? 1 : 0;
  ++S->st.points;
  S->st.policy_s += std::chrono::duration<double>(Clock::now() - t0).count();
  return MEMSPEC_OK;
}

memspec_status memspec_sched_feedback(memspec_sched* S, int32_t iterations, int32_t tokens,
                                      double seconds) {
  if (S == nullptr || !S->started || iterations < 0 || tokens < 0 || !(seconds >= 0.0))
    return MEMSPEC_ERR_INVALID_ARG;
  if (iterations == 0) return MEMSPEC_OK;
  if (S->last_fallback) {
    ++S->st.fallback_intervals;
    S->st.fallback_s += seconds;
  } else {
    ++S->st.desired_intervals;
    S->st.desired_s += seconds;
  }
  S->t += 1;
  const double r = static_cast<double>(tokens) / static_cast<double>(iterations) /
                   static_cast<double>(S->p.k_draft + 1);
  S->pulls[S->active] += 1;
  S->reward_sum[S->active] += r;
  return MEMSPEC_OK;
}

memspec_status memspec_sched_get_stats(const memspec_sched* S, memspec_sched_stats* out) {
  if (S == nullptr || out == nullptr) return MEMSPEC_ERR_INVALID_ARG;
  *out = S->st;
  return MEMSPEC_OK;
}

}  // extern "C"
