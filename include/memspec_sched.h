/*
 * memspec_sched.h - host-side draft scheduling over the draft-residency calls
 * of memspec.h (same library, libmemspec.so).
 *
 * MemSpec's contribution is the control logic ABOVE the draft-then-verify step
 * (arxiv 2608.10362, Section 3): every N speculative iterations a predictor
 * scores every candidate draft, the cache manager keeps the top-K of that
 * ranking resident under the memory budget (Section 3.3, Algorithm 2: prefetch
 * asynchronously, evict the lowest-scored draft outside the working set, never
 * the active draft), and the runtime controller runs the best draft that is
 * resident now instead of stalling on one that is still loading (Section 3.4,
 * Algorithm 3).  The exploration baseline the paper compares with, MAB-Async
 * (Section 2.3; Section 4.1 "Baselines", UCB with c = 2.0), and a static policy
 * are provided on the same interface.
 *
 * The scheduler holds no device memory and launches no kernel: it decides, and
 * acts through a residency mechanism - either a memspec_ctx (the library's
 * memspec_load_draft_async / memspec_query_draft / memspec_evict_draft /
 * memspec_set_active_draft) or caller-supplied functions.
 *
 * Readings of the paper used here (the paper leaves them open):
 *  1. the capacity K counts drafts resident or being loaded;
 *  2. ranking ties go to the lower draft id; among equally scored eviction
 *     candidates the higher id is evicted;
 *  3. a draft still loading is neither runnable nor evictable, except the
 *     active draft itself;
 *  4. a load refused for lack of bytes evicts the next lowest-scored
 *     unprotected resident draft and retries; with none left, it is skipped;
 *  5. MAB-Async: every draft is run once first; reward of an interval =
 *     committed tokens / iterations / (k_draft + 1), credited to the draft that
 *     ran; UCB(d) = mean(d) + c sqrt(ln t / n_d), t = intervals run; its load
 *     victim is the resident non-active draft of lowest UCB;
 *  6. an interval is "desired" when the draft that ran is the one the policy
 *     wanted for it, else "fallback" (Section 4.3 execution breakdown).
 *
 * Errors: MEMSPEC_ERR_INVALID_ARG (bad parameters; a call before start);
 * any status the residency mechanism returns is passed through.  Calls on one
 * scheduler must not overlap (one host thread at a time).
 */
#ifndef MEMSPEC_SCHED_H_
#define MEMSPEC_SCHED_H_

#include "memspec.h"

#ifdef __cplusplus
extern "C" {
#endif

enum { MEMSPEC_POLICY_MEMSPEC = 0, MEMSPEC_POLICY_MAB_ASYNC = 1, MEMSPEC_POLICY_STATIC = 2 };
#define MEMSPEC_SCHED_MAX_DRAFTS 16

/* Residency mechanism.  Every function returns a memspec_status.
 *   state:      *st = 0 absent, 1 resident, 2 loading
 *   load:       start an asynchronous load; MEMSPEC_ERR_BUDGET if the bytes do
 *               not fit (nothing changes then)
 *   evict:      drop a resident, non-active draft
 *   set_active: the draft the next steps run */
typedef struct memspec_residency {
  void* user;
  int32_t (*state)(void* user, int32_t draft, int32_t* st);
  int32_t (*load)(void* user, int32_t draft);
  int32_t (*evict)(void* user, int32_t draft);
  int32_t (*set_active)(void* user, int32_t draft);
} memspec_residency;

typedef struct memspec_sched_params {
  int32_t n_drafts;   /* |D|, 1..MEMSPEC_SCHED_MAX_DRAFTS (draft ids 0..n-1) */
  int32_t capacity;   /* K >= 1: drafts resident or loading at once */
  int32_t policy;     /* MEMSPEC_POLICY_* */
  float ucb_c;        /* MAB-Async exploration coefficient (the paper: 2.0) */
  int32_t k_draft;    /* draft length of the steps (MAB reward normalisation) */
} memspec_sched_params;

typedef struct memspec_sched_decision {
  int32_t active;     /* draft to run for the next interval */
  int32_t desired;    /* the policy's choice (top-ranked / UCB pick) */
  int32_t fallback;   /* active != desired */
  int32_t n_evicted, n_prefetched;
  int32_t evicted[MEMSPEC_SCHED_MAX_DRAFTS];
  int32_t prefetched[MEMSPEC_SCHED_MAX_DRAFTS];
} memspec_sched_decision;

typedef struct memspec_sched_stats {
  int64_t points;              /* scheduling points (start included) */
  int64_t desired_intervals, fallback_intervals;
  int64_t loads, evictions, refusals, switches;
  double desired_s, fallback_s; /* seconds reported by memspec_sched_feedback */
  double policy_s;              /* host time inside start / point */
} memspec_sched_stats;

typedef struct memspec_sched memspec_sched;

/* Create a scheduler acting through `mech` (copied), or, when mech is NULL,
 * through ctx's draft calls (draft ids are ctx draft ids).  Errors: INVALID_ARG. */
memspec_status memspec_sched_create(const memspec_sched_params* p, const memspec_residency* mech,
                                    memspec_ctx* ctx, memspec_sched** out);
void memspec_sched_destroy(memspec_sched* s);

/* Algorithm 3 lines 2-5: pick the initial draft from the prompt's scores
 * (MAB-Async: draft 0), load it if needed, make it active, prepare the cache.
 * scores: float [n_drafts] (ignored by MAB-Async and Static). */
memspec_status memspec_sched_start(memspec_sched* s, const float* scores,
                                   memspec_sched_decision* out);

/* One scheduling point (Algorithm 3 lines 14-18 / Algorithm 2): update the
 * cache from the new scores and choose the draft of the next interval. */
memspec_status memspec_sched_point(memspec_sched* s, const float* scores,
                                   memspec_sched_decision* out);

/* The interval since the last start / point ran `iterations` steps that
 * committed `tokens` tokens in `seconds`: MAB-Async's reward, and the
 * desired / fallback time of the breakdown. */
memspec_status memspec_sched_feedback(memspec_sched* s, int32_t iterations, int32_t tokens,
                                      double seconds);

memspec_status memspec_sched_get_stats(const memspec_sched* s, memspec_sched_stats* out);

#ifdef __cplusplus
}
#endif
#endif /* MEMSPEC_SCHED_H_ */
