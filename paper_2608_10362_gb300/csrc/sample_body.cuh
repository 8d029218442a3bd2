// sample_body.cuh - vocab-wide softmax statistics, categorical sampling with
// Philox uniforms, speculative-sampling acceptance, residual resampling, and the
// commit / rollback of the sequence state; templated on the block size NT and
// on the barrier used, so the sampling kernels (NT = 512) and the persistent
// pass kernel (NT = 128 worker threads) share it.
//
// Acceptance (Leviathan et al. ICML'23 Alg. 1, which MemSpec cites and runs
// unchanged, Section 3.5): with p_i = softmax(z_target,i / T) and
// q_i = softmax(z_draft,i / T), draft token x_i is accepted iff
// u_i * q_i(x_i) <= p_i(x_i); at the first rejection n, the extra token is drawn
// from norm(max(0, p_{n+1} - q_{n+1})) (from p_{n+1} if that residual has no
// mass); if all K are accepted it is drawn from p_{K+1}.  T == 0 is greedy:
// accept while x_i == argmax p_i, extra token = argmax p_{n+1}.
//
// Categorical sampling of weights w with uniform u returns the smallest id j with
// sum_{i<=j} w_i > u * sum_i w_i.  Weights are summed in a fixed order: tiles of
// 128 consecutive ids (4 per lane, lanes combined by a fixed shuffle tree),
// tile sums combined in id order.
#pragma once
#include "internal.h"
#include "ptx.cuh"

namespace memspec {
namespace smp {

constexpr int kMaxTiles = 1024;   // 128-id tiles: vocab <= 131072

// Shared scratch of one sampling block (any NT <= 512).
struct SampleSmem {
  float scr_f[32];
  int scr_i[16];
  float tiles[kMaxTiles];
  float total;
  int is_last;
  int pick;
  int n, y;
  float u;
};

struct RowStats {
  float m;     // max of z * inv_temp   (greedy: max of z)
  float s;     // sum exp(z * inv_temp - m)
  int arg;     // first index of the maximum
};

// Block-wide sum in a fixed order (warp xor-tree, then warps 0..NW-1 in order).
template <int NT, class Sync>
__device__ float block_sum(float v, float* scratch, int tid, Sync sync) {
  constexpr int NW = NT / 32;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  sync();
  if ((tid & 31) == 0) scratch[tid >> 5] = v;
  sync();
  float t = 0.f;
  for (int i = 0; i < NW; ++i) t += scratch[i];
  return t;
}

__device__ __forceinline__ void stats_update(float raw, int x, bool greedy, float inv_temp,
                                             float& m, float& s, int& arg) {
  if (raw > m) {
    if (!greedy) s = (m == -INFINITY) ? 0.f : s * __expf((m - raw) * inv_temp);
    m = raw;
    arg = x;
  }
  if (!greedy) s += __expf((raw - m) * inv_temp);
}

// max / first-argmax / rescaled exp-sum of one row, whole block.
template <int NT, class Sync>
__device__ RowStats row_stats(const float* z, int V, float inv_temp, bool greedy, SampleSmem& sm,
                              int tid, Sync sync) {
  constexpr int NW = NT / 32;
  float m = -INFINITY, s = 0.f;
  int arg = 0x7fffffff;
  if ((V & 3) == 0 && (reinterpret_cast<uintptr_t>(z) & 15) == 0) {
    const float4* z4 = reinterpret_cast<const float4*>(z);
    const int V4 = V >> 2;
#pragma unroll 4
    for (int x4 = tid; x4 < V4; x4 += NT) {
      const float4 r = __ldcg(z4 + x4);
      stats_update(r.x, 4 * x4, greedy, inv_temp, m, s, arg);
      stats_update(r.y, 4 * x4 + 1, greedy, inv_temp, m, s, arg);
      stats_update(r.z, 4 * x4 + 2, greedy, inv_temp, m, s, arg);
      stats_update(r.w, 4 * x4 + 3, greedy, inv_temp, m, s, arg);
    }
  } else {
#pragma unroll 4
    for (int x = tid; x < V; x += NT) stats_update(__ldcg(z + x), x, greedy, inv_temp, m, s, arg);
  }
  float bm = m;
  int ba = arg;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float om = __shfl_xor_sync(0xffffffffu, bm, o);
    const int oa = __shfl_xor_sync(0xffffffffu, ba, o);
    if (om > bm || (om == bm && oa < ba)) {
      bm = om;
      ba = oa;
    }
  }
  sync();
  if ((tid & 31) == 0) {
    sm.scr_f[tid >> 5] = bm;
    sm.scr_i[tid >> 5] = ba;
  }
  sync();
  float M = -INFINITY;
  int A = 0x7fffffff;
  for (int i = 0; i < NW; ++i) {
    if (sm.scr_f[i] > M || (sm.scr_f[i] == M && sm.scr_i[i] < A)) {
      M = sm.scr_f[i];
      A = sm.scr_i[i];
    }
  }
  RowStats r;
  r.m = M * (greedy ? 1.f : inv_temp);
  r.arg = A;
  r.s = 0.f;
  if (!greedy) {
    const float mine = (m == -INFINITY) ? 0.f : s * __expf((m - M) * inv_temp);
    r.s = block_sum<NT>(mine, sm.scr_f + 16, tid, sync);
  }
  return r;
}

// Smallest id j in [0, V) with sum_{i<=j} w(i) > u * sum w; whole block.
// w(i) must be >= 0.  Returns -1 if the total weight is zero.
template <int NT, class W, class Sync>
__device__ int block_sample(const W& wfun, int V, float u, SampleSmem& sm, int tid, Sync sync) {
  constexpr int NW = NT / 32;
  constexpr int kTile = 128;
  const int ntiles = (V + kTile - 1) / kTile;
  const int w = tid >> 5, lane = tid & 31;
#pragma unroll 2
  for (int tile = w; tile < ntiles; tile += NW) {
    const int x0 = tile * kTile + lane * 4;
    float own = 0.f;
#pragma unroll
    for (int q = 0; q < 4; ++q)
      if (x0 + q < V) own += wfun(x0 + q);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) own += __shfl_xor_sync(0xffffffffu, own, o);
    if (lane == 0) sm.tiles[tile] = own;
  }
  sync();
  if (w == 0) {
    // each lane owns a contiguous range of tiles
    const int tpl = (ntiles + 31) / 32;
    const int t_lo = min(lane * tpl, ntiles), t_hi = min(t_lo + tpl, ntiles);
    float ls = 0.f;
    for (int t = t_lo; t < t_hi; ++t) ls += sm.tiles[t];
    float incl = ls;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const float n = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += n;
    }
    float excl = __shfl_up_sync(0xffffffffu, incl, 1);
    if (lane == 0) excl = 0.f;
    const float total = __shfl_sync(0xffffffffu, incl, 31);
    const float target = u * total;
    int sel = -1;
    float before = 0.f;
    if (ls > 0.f && excl <= target && target < incl) {
      float c = excl;
      for (int t = t_lo; t < t_hi; ++t) {
        if (sm.tiles[t] > 0.f) {
          sel = t;
          before = c;
          if (c + sm.tiles[t] > target) break;
        }
        c += sm.tiles[t];
      }
    }
    // the claiming lane (ranges chain exactly); otherwise the last tile with mass
    const unsigned claim = __ballot_sync(0xffffffffu, sel >= 0);
    const int last_lane = 31 - __clz(__ballot_sync(0xffffffffu, ls > 0.f) | 1u);
    const int src = claim ? (__ffs(claim) - 1) : last_lane;
    if (!claim && lane == src) {
      float c = excl;
      for (int t = t_lo; t < t_hi; ++t) {
        if (sm.tiles[t] > 0.f) {
          sel = t;
          before = c;
        }
        c += sm.tiles[t];
      }
    }
    sel = __shfl_sync(0xffffffffu, sel, src);
    before = __shfl_sync(0xffffffffu, before, src);
    int pick = -1;
    if (total > 0.f && sel >= 0) {
      const float r = target - before;
      const int x0 = sel * kTile + lane * 4;
      float wv[4], own = 0.f;
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        wv[q] = (x0 + q < V) ? wfun(x0 + q) : 0.f;
        own += wv[q];
      }
      float in2 = own;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const float n = __shfl_up_sync(0xffffffffu, in2, o);
        if (lane >= o) in2 += n;
      }
      float ex2 = __shfl_up_sync(0xffffffffu, in2, 1);
      if (lane == 0) ex2 = 0.f;
      int mine = -1;
      if (own > 0.f && ex2 <= r && r < in2) {
        float c = ex2;
        for (int q = 0; q < 4; ++q) {
          c += wv[q];
          if (wv[q] > 0.f && c > r) {
            mine = x0 + q;
            break;
          }
        }
        if (mine < 0)
          for (int q = 3; q >= 0; --q)
            if (wv[q] > 0.f) {
              mine = x0 + q;
              break;
            }
      }
      const unsigned cl = __ballot_sync(0xffffffffu, mine >= 0);
      if (cl) {
        pick = __shfl_sync(0xffffffffu, mine, __ffs(cl) - 1);
      } else {   // r at/after the tile's scanned mass: its last id with mass
        int lastq = -1;
        for (int q = 3; q >= 0; --q)
          if (wv[q] > 0.f) {
            lastq = x0 + q;
            break;
          }
        const unsigned hm = __ballot_sync(0xffffffffu, lastq >= 0);
        pick = hm ? __shfl_sync(0xffffffffu, lastq, 31 - __clz(hm)) : -1;
      }
    }
    if (lane == 0) {
      sm.pick = pick;
      sm.total = total;
    }
  }
  sync();
  return sm.pick;
}

struct ExpW {  // w(x) = exp(z(x) * it - m)
  const float* z;
  float it, m;
  __device__ float operator()(int x) const { return __expf(z[x] * it - m); }
};

struct ResidualW {  // w(x) = max(0, p(x) - q(x))
  const float* zt;
  const float* zd;
  float it, mt, st_inv, md, sd_inv;
  __device__ float operator()(int x) const {
    const float p = __expf(zt[x] * it - mt) * st_inv;
    const float q = __expf(zd[x] * it - md) * sd_inv;
    return fmaxf(p - q, 0.f);
  }
};

// Draft sampler for group g: x = argmax (T == 0) or inverse-CDF sample of softmax(z/T).
template <int NT, class Sync>
__device__ void sample_group(const SampleArgs& a, int g, SampleSmem& sm, int tid, Sync sync) {
  const float* z = a.logits + g * a.row_stride;
  const RowStats st = row_stats<NT>(z, a.vocab, a.inv_temp, a.greedy != 0, sm, tid, sync);
  int tok = st.arg;
  if (!a.greedy) {
    float u;
    if (a.u_explicit != nullptr) {
      u = a.u_explicit[g];
    } else if (a.row_slots != nullptr) {   // tree step: rows of request 0
      u = philox_uniform(a.seeds[0], 0, a.seq_state[2], a.slot + a.row_slots[g]);
    } else {
      const int step = a.seq_state[g * kStateInts + 2];
      u = philox_uniform(a.seeds[g], g, step, a.slot);
    }
    ExpW wf{z, a.inv_temp, st.m};
    const int pick = block_sample<NT>(wf, a.vocab, u, sm, tid, sync);
    tok = pick >= 0 ? pick : st.arg;
  }
  if (tid == 0) a.out_tok[g * a.out_stride] = tok;
  sync();
}

// Acceptance, part 1: statistics of row rho (0..K target rows, K+1..2K draft rows)
// of group g; the block that completes a group's last row runs part 2 (decision,
// resample, commit) and returns true.
template <int NT, class Sync>
__device__ void accept_row(const AcceptArgs& a, int rho, int g, SampleSmem& sm, int tid, Sync sync) {
  const int K = a.K, V = a.vocab;
  const bool greedy = a.greedy != 0;
  const float* zrow = rho <= K ? a.zt + (static_cast<size_t>(g) * (K + 1) + rho) * V
                               : a.zd + (static_cast<size_t>(g) * K + (rho - K - 1)) * V;
  const RowStats st = row_stats<NT>(zrow, V, a.inv_temp, greedy, sm, tid, sync);
  float* part = a.part + (static_cast<size_t>(g) * (2 * K + 1) + rho) * 4;
  // thread 0 stores this row's statistics and arrives with release semantics; the
  // block completing the group acquires them all through the same atomic
  if (tid == 0) {
    part[0] = st.m;
    part[1] = st.s;
    part[2] = __int_as_float(st.arg);
    sm.is_last = (atom_add_acq_rel_gpu(&a.counters[g], 1) == 2 * K) ? 1 : 0;
  }
  sync();
  if (!sm.is_last) return;

  // ---- decision (the whole block reads the row statistics of group g)
  const float* pg = a.part + static_cast<size_t>(g) * (2 * K + 1) * 4;
  int* state = a.seq_state + g * kStateInts;
  const int L = state[0];
  const int step = state[2];
  const int* x = a.draft_tokens + g * a.max_k;
  float* dbg = a.debug + static_cast<size_t>(g) * (2 * K + 2);
  // draft position i < K is decided by thread i (all loads in flight together);
  // n = the first rejected position (K if none)
  if (tid < 32) {
    bool acc = false;
    float p = 0.f, q = 0.f;
    if (tid < K) {
      const int xi = x[tid];
      if (greedy) {
        acc = xi == __float_as_int(ld_cg_f(pg + tid * 4 + 2));
      } else {
        const float* zt = a.zt + (static_cast<size_t>(g) * (K + 1) + tid) * V;
        const float* zd = a.zd + (static_cast<size_t>(g) * K + tid) * V;
        const float* ptn = pg + tid * 4;
        const float* pdn = pg + (K + 1 + tid) * 4;
        const float zx = ld_cg_f(zt + xi), mt = ld_cg_f(ptn), st = ld_cg_f(ptn + 1);
        const float dx = ld_cg_f(zd + xi), md = ld_cg_f(pdn), sd = ld_cg_f(pdn + 1);
        p = __expf(zx * a.inv_temp - mt) / st;
        q = __expf(dx * a.inv_temp - md) / sd;
        const float u = philox_uniform(a.seeds[g], g, step, K + tid);
        acc = u * q <= p;
      }
    }
    const unsigned acc_mask = __ballot_sync(0xffffffffu, acc);
    const int n = min(__ffs(~acc_mask) - 1, K);
    if (!greedy && tid < K) {
      dbg[tid] = p;
      dbg[K + tid] = q;
    }
    if (tid == 0) {
      sm.n = n;
      sm.u = greedy ? 0.f : philox_uniform(a.seeds[g], g, step, 2 * K);
      sm.y = greedy ? __float_as_int(ld_cg_f(pg + n * 4 + 2)) : -1;
    }
  }
  sync();
  const int n = sm.n;
  int y = sm.y;
  if (!greedy) {
    const float u = sm.u;
    const float* zt = a.zt + (static_cast<size_t>(g) * (K + 1) + n) * V;
    const float mt = ld_cg_f(pg + n * 4), stn = ld_cg_f(pg + n * 4 + 1);
    float mass = 1.f;
    int pick = -1;
    if (n < K) {
      const float* zd = a.zd + (static_cast<size_t>(g) * K + n) * V;
      const float md = ld_cg_f(pg + (K + 1 + n) * 4), sdn = ld_cg_f(pg + (K + 1 + n) * 4 + 1);
      ResidualW rw{zt, zd, a.inv_temp, mt, 1.f / stn, md, 1.f / sdn};
      pick = block_sample<NT>(rw, V, u, sm, tid, sync);
      mass = sm.total;
    }
    if (pick < 0) {  // n == K (bonus), or a residual without mass: sample p_{n+1}
      ExpW wf{zt, a.inv_temp, mt};
      pick = block_sample<NT>(wf, V, u, sm, tid, sync);
      if (n < K) mass = 0.f;
    }
    y = pick >= 0 ? pick : __float_as_int(ld_cg_f(pg + n * 4 + 2));
    if (tid == 0) {
      dbg[2 * K] = mass;
      dbg[2 * K + 1] = u;
    }
  }
  // ---- commit: append x_1..x_n, y; lengths; KV rollback is the length update
  int* res = a.results + g * (K + 2);
  int* toks = a.tokens + static_cast<size_t>(g) * a.max_seq;
  const bool fits = L + n + 1 <= a.max_seq;
  if (fits && tid < K + 2) {
    // slot tid of the result row: 0 = n, 1..n = accepted drafts, n + 1 = y, then -1
    int val = -1;
    if (tid == 0) {
      val = n;
    } else if (tid <= n) {
      val = x[tid - 1];
      toks[L + tid - 1] = val;
    } else if (tid == n + 1) {
      val = y;
      toks[L + n] = y;
    }
    res[tid] = val;
  }
  if (tid == 0) {
    if (!fits) {
      res[0] = n;
      atomicOr(a.status, 0x4u);
    } else {
      state[0] = L + n + 1;                          // committed length
      state[1] = L + n;                              // target KV valid below L'-1
      a.draft_len[g] = L + (n < K - 1 ? n : K - 1);  // draft KV valid below this count
    }
    state[2] = step + 1;
    a.counters[g] = 0;
  }
  sync();
}

}  // namespace smp
}  // namespace memspec
