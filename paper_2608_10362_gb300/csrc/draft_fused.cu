// draft_fused.cu - the draft step of a small draft model as ONE launch.
//
// The draft step is K autoregressive forward passes of one position each (two
// for the first pass after a fully accepted step) plus a categorical sample per
// pass (the proposals x_1..x_K of the draft-then-verify step).  For a small
// draft (68M-160M parameters) each projection is a few MB, so with one kernel
// launch per op the step is bound by launch and tail latency, not by bytes.
// This kernel runs the whole step in one cooperative launch, one CTA per SM:
//
//  * every op of a pass (QKV + RoPE + KV append, attention, O + residual,
//    gate/up + SwiGLU, down + residual; final RMSNorm + LM head; sampling) is a
//    phase separated from the next by a grid-wide barrier (an arrival counter in
//    global memory, release / acquire, bounded waits);
//  * projection weights are split into units of 8 output rows per warp-row (8
//    rows; 8 RoPE pairs for QKV; 8 gate + 8 up rows for the SwiGLU pair),
//    assigned round-robin to CTAs; a CTA computes its units' full dot products
//    (no split-K, no partial sums) on CUDA cores, fp32 activations times bf16
//    weights, each warp owning one output row (or one row pair);
//  * one copy-issuing lane streams the CTA's weight bytes of every op of every
//    pass, in the order the compute warps consume them, into a ring of 16 KB
//    shared-memory slots, each slot one to four multi-dimensional TMA boxes over
//    the packed tiles (8 rows x 64 columns x up to 16 k tiles), signalled on
//    mbarriers.  Weights do not depend on activations, so the ring fills ahead
//    across op and pass boundaries while the compute warps wait at barriers;
//  * attention: one (request, head, key split) unit per CTA; the keys of
//    positions before the pass are prefetched into L2 while the QKV phase runs;
//    the last split of a head to finish combines the splits (m, l, o);
//  * LM head: each CTA owns a contiguous vocabulary slice and writes its
//    logits and (max, first argmax, sum exp) statistics; after the barrier every
//    CTA redoes the tiny combine and the inverse-CDF search in the owning slice
//    (same data, same order, same result), so the next pass needs no extra
//    barrier.  Sampling follows the draft sampler: T == 0 argmax (lowest id on
//    ties), else the smallest id j with sum_{i<=j} exp((z_i - M)/T) >
//    u * sum_i exp((z_i - M)/T), u = Philox(seed, request, step, j - 1).
//
// Row r = g * R + i of pass j (R = 2 for j = 1, else 1) is position pos0[g] + i
// of request g; pass 1 feeds the committed tokens the draft has not processed
// (one, or two after a fully accepted step), pass j > 1 feeds x_{j-1}.
#include <cuda_bf16.h>

#include "internal.h"
#include "ptx.cuh"

namespace memspec {
namespace {

constexpr int kCW = kDfComputeWarps;
constexpr int kCT = kCW * 32;              // compute threads
constexpr int kUR = 8;                     // output rows (or row pairs) per unit: one per warp
constexpr int kKeyBlock = kCT;             // keys per attention block (one per thread)
// attention scores (2 rows), queries (2 x hd <= 128), per-warp o partials
// [warps][2][hd <= 128]
constexpr int kDfScratchFloats = 2 * kKeyBlock + 2 * 128 + kCW * 2 * 128;

enum DfOp { OP_QKV = 0, OP_O = 1, OP_GU = 2, OP_DOWN = 3, OP_LM = 4 };

struct DfCtl {
  uint64_t full[kDfMaxSlots];
  uint64_t empty[kDfMaxSlots];
  int abort;                          // this CTA stops (a wait ran out or the grid aborted)
  int gs_ok;                          // result of the last grid barrier (written by thread 0)
  int R, rows;                        // rows per request, rows of the pass
  int valid[kDfMaxGroups], pos0[kDfMaxGroups];
  int tok[kDfMaxRows];
  int ok[kDfMaxRows];                 // row is valid and inside the cache
  int next_tok[kDfMaxGroups];         // sample of the last pass
  float red[kCW][kDfMaxRows];
  float scale[kDfMaxRows];
  float xch[kCW][kDfMaxRows];
  float stat_m[kCW][kDfMaxGroups], stat_s[kCW][kDfMaxGroups];
  int stat_a[kCW][kDfMaxGroups];
  float samp_f[4];
  int samp_i[4];
};

__device__ __forceinline__ unsigned ld_acquire_u32(const unsigned* p) {
  unsigned v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}
__device__ __forceinline__ unsigned ld_relaxed_u32(const unsigned* p) {
  unsigned v;
  asm volatile("ld.relaxed.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}
__device__ __forceinline__ void red_release_add(unsigned* p, unsigned v) {
  asm volatile("red.release.gpu.global.add.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}
__device__ __forceinline__ void prefetch_l2(const void* p, uint32_t bytes) {
  asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(p), "r"(bytes) : "memory");
}
// One TMA request per box (a request costs about as much as its bytes only from
// several KB up, measured).
__device__ __forceinline__ void tma_load_3d(void* dst, const CUtensorMap* map, int x, int y, int z,
                                            uint64_t* bar, uint64_t pol) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint"
      " [%0], [%1, {%2, %3, %4}], [%5], %6;" ::"r"(smem_addr(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(z), "r"(smem_addr(bar)), "l"(pol)
      : "memory");
}
__device__ __forceinline__ float bf_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf_hi(uint32_t w) { return __uint_as_float(w & 0xffff0000u); }
__device__ __forceinline__ float ldcg(const float* p) { return __ldcg(p); }

__device__ __forceinline__ void csync() { named_bar_sync(1, kCT); }
// Barrier over the compute warps that also ANDs a flag: the same answer in every
// thread, so that a CTA stops as a whole.
__device__ __forceinline__ bool csync_and(bool v) {
  uint32_t r;
  asm volatile(
      "{\n\t.reg .pred p, q;\n\t"
      "setp.ne.u32 p, %1, 0;\n\t"
      "bar.red.and.pred q, 1, %2, p;\n\t"
      "selp.u32 %0, 1, 0, q;\n\t}"
      : "=r"(r)
      : "r"(static_cast<uint32_t>(v)), "n"(kCT)
      : "memory");
  return r != 0;
}

// Position in the weight ring (slot index and the phase parity of its barriers).
struct Ring {
  int i = 0, S = 1;
  uint32_t ph = 0;
  __device__ void next() {
    if (++i == S) {
      i = 0;
      ph ^= 1u;
    }
  }
};

// ------------------------------------------------------------------ schedule
// Units of each weight op, and ring slots per unit.
struct Geo {
  int G, c;
  int kt_d, kt_q, kt_f;          // 64-column tiles of d, H*hd, F
  int u_qkv, u_o, u_gu, u_down, u_lm;
  int s_qkv, s_o, s_gu, s_down, s_lm;
};

__device__ __forceinline__ Geo make_geo(const DraftFusedArgs& a) {
  Geo g;
  g.G = gridDim.x;
  g.c = blockIdx.x;
  g.kt_d = a.d / 64;
  g.kt_q = a.H * a.hd / 64;
  g.kt_f = (a.F + 63) / 64;
  g.u_qkv = (a.H + 2 * a.Hkv) * a.hd / (2 * kUR);   // 8 RoPE pairs per unit
  g.u_o = a.d / kUR;
  g.u_gu = a.F / kUR;
  g.u_down = a.d / kUR;
  g.u_lm = (a.V + kUR - 1) / kUR;
  g.s_qkv = (g.kt_d + 7) / 8;
  g.s_o = (g.kt_q + 15) / 16;
  g.s_gu = (g.kt_d + 7) / 8;
  g.s_down = (g.kt_f + 15) / 16;
  g.s_lm = a.tied ? (a.d + 1023) / 1024 : (g.kt_d + 15) / 16;
  return g;
}
__device__ __forceinline__ int first_unit(const Geo& g, int off) { return ((g.c - off) % g.G + g.G) % g.G; }
__device__ __forceinline__ int lm_lo(const Geo& g, int c) {
  return static_cast<int>(static_cast<long long>(c) * g.u_lm / g.G);
}
// The two row blocks of QKV unit u: rows lo..lo+7 and their RoPE partners hi..hi+7.
__device__ __forceinline__ void qkv_rows(const DraftFusedArgs& a, int u, int* hb, int* ui, int* lo, int* hi) {
  const int per = a.hd / (2 * kUR);
  *hb = u / per;
  *ui = u - *hb * per;
  *lo = *hb * a.hd + kUR * *ui;
  *hi = *lo + a.hd / 2;
}

// Issue the TMA boxes of slot `s` of unit `u` of op `op` (layer `l`) into `dst`
// (16 KB, completing on `bar`).  Shared-memory image of a slot (128-byte rows
// exactly as packed, swizzle included):
//   O, DOWN, packed LM: [16 k tiles][8 rows][128 B]                 (one box)
//   QKV: rows lo.. then their partners hi..: 2 x [8 k tiles][8 rows][128 B]
//   GU:  gate rows then the same up rows:    2 x [8 k tiles][8 rows][128 B]
//   tied LM (row-major embedding): 4 x [8 rows][256 columns]
__device__ void issue_slot(const DraftFusedArgs& a, const Geo& g, int op, int l, int u, int s,
                           uint8_t* dst, uint64_t* bar, uint64_t pol) {
  const CUtensorMap* maps = a.maps + static_cast<size_t>(l) * 4;
  if (op == OP_QKV) {
    int hb, ui, lo, hi;
    qkv_rows(a, u, &hb, &ui, &lo, &hi);
    const int kt0 = s * 8;
    tma_load_3d(dst, maps + 0, 0, lo % 128, (lo / 128) * g.kt_d + kt0, bar, pol);
    tma_load_3d(dst + 8192, maps + 0, 0, hi % 128, (hi / 128) * g.kt_d + kt0, bar, pol);
    return;
  }
  if (op == OP_GU) {
    const int j0 = u * kUR, rt = j0 / 64, rr = j0 % 64, kt0 = s * 8;
    tma_load_3d(dst, maps + 2, 0, rr, rt * g.kt_d + kt0, bar, pol);
    tma_load_3d(dst + 8192, maps + 2, 0, 64 + rr, rt * g.kt_d + kt0, bar, pol);
    return;
  }
  if (op == OP_LM && a.tied) {   // map {d, vocab, 1}, box {256, 8, 1}
    const CUtensorMap* m = a.maps + static_cast<size_t>(a.n_layers) * 4;
#pragma unroll
    for (int q = 0; q < 4; ++q) tma_load_3d(dst + q * 4096, m, s * 1024 + q * 256, u * kUR, 0, bar, pol);
    return;
  }
  const CUtensorMap* m;
  int kt_n;
  if (op == OP_O) {
    m = maps + 1;
    kt_n = g.kt_q;
  } else if (op == OP_DOWN) {
    m = maps + 3;
    kt_n = g.kt_f;
  } else {
    m = a.maps + static_cast<size_t>(a.n_layers) * 4;
    kt_n = g.kt_d;
  }
  const int r0 = u * kUR;
  tma_load_3d(dst, m, 0, r0 % 128, (r0 / 128) * kt_n + s * 16, bar, pol);
}

// The copy-issuing lane: every slot of every unit of every op of every pass, in
// consumption order.
__device__ void producer(const DraftFusedArgs& a, DfCtl& ctl, uint8_t* ring) {
  const Geo g = make_geo(a);
  const uint64_t pol = l2_policy_evict_first();
  Ring rg;
  rg.S = a.ring_slots;
  uint32_t n = 0;
  bool ok = true;
  for (int i = 0; i <= a.n_layers * 4; ++i) tma_prefetch_desc(a.maps + i);
  auto fill = [&](int op, int l, int u, int s) {
    if (!ok) return;
    if (n >= static_cast<uint32_t>(rg.S) &&
        !mbar_wait_bounded(&ctl.empty[rg.i], rg.ph ^ 1u, &ctl.abort, a.status)) {
      ok = false;
      return;
    }
    mbar_arrive_expect_tx(&ctl.full[rg.i], kDfSlotBytes);
    issue_slot(a, g, op, l, u, s, ring + static_cast<size_t>(rg.i) * kDfSlotBytes, &ctl.full[rg.i], pol);
    rg.next();
    ++n;
  };
  for (int j = 1; j <= a.K && ok; ++j) {
    int cum = 0;
    for (int l = 0; l < a.n_layers && ok; ++l) {
      const int nu[4] = {g.u_qkv, g.u_o, g.u_gu, g.u_down};
      const int ns[4] = {g.s_qkv, g.s_o, g.s_gu, g.s_down};
      for (int op = 0; op < 4; ++op) {
        const int off = cum % g.G;
        cum += nu[op];
        for (int u = first_unit(g, off); u < nu[op]; u += g.G)
          for (int s = 0; s < ns[op]; ++s) fill(op, l, u, s);
      }
    }
    for (int u = lm_lo(g, g.c); u < lm_lo(g, g.c + 1); ++u)
      for (int s = 0; s < g.s_lm; ++s) fill(OP_LM, 0, u, s);
  }
  // tear-down: the last fill of every slot must have landed before the CTA exits
  const uint32_t first = n > static_cast<uint32_t>(rg.S) ? n - rg.S : 0;
  for (uint32_t m = first; m < n; ++m) mbar_wait_drain(&ctl.full[m % rg.S], (m / rg.S) & 1u);
}

// ------------------------------------------------------------------ helpers (compute warps)
// Grid-wide barrier over the compute warps of every CTA.  false: the grid
// aborted (the same answer in every thread of the CTA).
__device__ bool grid_sync(const DraftFusedArgs& a, DfCtl& ctl, unsigned& epoch, int tid,
                          unsigned long long& t_phase) {
  csync();
  if (tid == 0) {
    ++epoch;
    const unsigned target = epoch * gridDim.x;
    unsigned long long* tr =
        a.trace != nullptr ? a.trace + 2 + (static_cast<size_t>(epoch - 1) * gridDim.x + blockIdx.x) * 16
                           : nullptr;
    if (tr != nullptr && epoch <= static_cast<unsigned>(a.trace_phases)) {
      tr[0] = t_phase;
      tr[1] = global_ns();
    }
    int ok = *reinterpret_cast<volatile int*>(&ctl.abort) ? 0 : 1;
    if (ok) {
      // the block barrier above orders every thread's writes before this
      // thread's release, which publishes them at GPU scope (cumulativity); the
      // acquire below and the block barrier after it order the other CTAs'
      // writes before this block's next reads
      red_release_add(&a.bar[0], 1u);
      const long long t0 = clock64();
      for (unsigned it = 0; ld_acquire_u32(&a.bar[0]) < target; ++it) {
        if ((it & 31u) == 31u && ld_relaxed_u32(&a.bar[2]) != 0u) {   // the abort word, now and then
          ok = 0;
          break;
        }
        if (clock64() - t0 > kWaitBudgetCycles) {
          atomicOr(a.status, 0x1u);
          atomicExch(&a.bar[2], 1u);
          ok = 0;
          break;
        }
      }
    }
    t_phase = global_ns();
    if (tr != nullptr && epoch <= static_cast<unsigned>(a.trace_phases)) tr[13] = t_phase;
    if (!ok) *reinterpret_cast<volatile int*>(&ctl.abort) = 1;
    ctl.gs_ok = ok;
  }
  csync();
  return ctl.gs_ok != 0;
}

// Per-row block sums of v[r] (r < rows) in a fixed order; result in ctl.red[0][r].
// Starts with a barrier, so earlier readers of ctl.xch / ctl.red are done.
__device__ void block_row_sums(DfCtl& ctl, float* v, int rows, int tid) {
  const int w = tid >> 5, lane = tid & 31;
  csync();
#pragma unroll
  for (int r = 0; r < kDfMaxRows; ++r) {
    if (r >= rows) break;
    float x = v[r];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
    if (lane == 0) ctl.xch[w][r] = x;
  }
  csync();
  if (tid < rows) {
    float s = 0.f;
    for (int i = 0; i < kCW; ++i) s += ctl.xch[i][tid];
    ctl.red[0][tid] = s;
  }
  csync();
}

// act[r][0..d) = RMSNorm(x_r) * gain for the rows of the pass (LM: one row per
// request, the last valid one), in one round trip for x and the gain.  src: 0
// embedding rows of ctl.tok (and CTA 0 writes them to the residual stream), 1
// the residual stream.
__device__ void load_norm_rows(const DraftFusedArgs& a, DfCtl& ctl, float* act, int src,
                               const bf16* gain, bool lm_rows, int tid) {
  const int d = a.d, AF = a.act_floats;
  const int nrow = lm_rows ? a.B : ctl.rows;
  float ss[kDfMaxRows];
#pragma unroll
  for (int r = 0; r < kDfMaxRows; ++r) ss[r] = 0.f;
  for (int k = tid * 4; k < d; k += kCT * 4) {
    const uint2 graw = *reinterpret_cast<const uint2*>(gain + k);
    float4 x[kDfMaxRows];
#pragma unroll
    for (int r = 0; r < kDfMaxRows; ++r) {
      x[r] = make_float4(0.f, 0.f, 0.f, 0.f);
      if (r >= nrow) continue;
      const int rs = lm_rows ? r * ctl.R + ctl.valid[r] - 1 : r;
      if (!ctl.ok[rs]) continue;
      if (src == 0) {
        const uint2 raw = *reinterpret_cast<const uint2*>(a.w + a.off_emb +
                                                          (static_cast<size_t>(ctl.tok[rs]) * d + k) * 2);
        x[r] = make_float4(bf_lo(raw.x), bf_hi(raw.x), bf_lo(raw.y), bf_hi(raw.y));
        if (blockIdx.x == 0) *reinterpret_cast<float4*>(a.h + static_cast<size_t>(rs) * d + k) = x[r];
      } else {
        x[r] = __ldcg(reinterpret_cast<const float4*>(a.h + static_cast<size_t>(rs) * d + k));
      }
    }
    const float g0 = bf_lo(graw.x), g1 = bf_hi(graw.x), g2 = bf_lo(graw.y), g3 = bf_hi(graw.y);
#pragma unroll
    for (int r = 0; r < kDfMaxRows; ++r) {
      if (r >= nrow) break;
      ss[r] += x[r].x * x[r].x + x[r].y * x[r].y + x[r].z * x[r].z + x[r].w * x[r].w;
      *reinterpret_cast<float4*>(act + r * AF + k) =
          make_float4(x[r].x * g0, x[r].y * g1, x[r].z * g2, x[r].w * g3);
    }
  }
  block_row_sums(ctl, ss, nrow, tid);
  if (tid < nrow) ctl.scale[tid] = 1.f / sqrtf(ctl.red[0][tid] / static_cast<float>(d) + a.eps);
  csync();
  for (int k = tid * 4; k < d; k += kCT * 4) {
#pragma unroll
    for (int r = 0; r < kDfMaxRows; ++r) {
      if (r >= nrow) break;
      float4* p = reinterpret_cast<float4*>(act + r * AF + k);
      const float sc = ctl.scale[r];
      float4 v = *p;
      v.x *= sc;
      v.y *= sc;
      v.z *= sc;
      v.w *= sc;
      *p = v;
    }
  }
  csync();
}

// acc[m] += w(8 bf16 of `wv`) . act row m (8 floats at kidx), for m < M.
__device__ __forceinline__ void dot8(const uint4 wv, const float* act, int AF, int kidx, int M,
                                     float (&acc)[kDfMaxRows]) {
  const float w0 = bf_lo(wv.x), w1 = bf_hi(wv.x), w2 = bf_lo(wv.y), w3 = bf_hi(wv.y);
  const float w4 = bf_lo(wv.z), w5 = bf_hi(wv.z), w6 = bf_lo(wv.w), w7 = bf_hi(wv.w);
#pragma unroll
  for (int m = 0; m < kDfMaxRows; ++m) {
    if (m >= M) break;
    const float4 x0 = *reinterpret_cast<const float4*>(act + m * AF + kidx);
    const float4 x1 = *reinterpret_cast<const float4*>(act + m * AF + kidx + 4);
    float t = acc[m];
    t = fmaf(w0, x0.x, t);
    t = fmaf(w1, x0.y, t);
    t = fmaf(w2, x0.z, t);
    t = fmaf(w3, x0.w, t);
    t = fmaf(w4, x1.x, t);
    t = fmaf(w5, x1.y, t);
    t = fmaf(w6, x1.z, t);
    t = fmaf(w7, x1.w, t);
    acc[m] = t;
  }
}

// This warp's dot products for one unit: its output row (PAIR: its two rows,
// lo / hi for QKV, gate / up for GU) against the M activation rows, over the
// unit's ring slots.  Each lane handles 4 16-byte weight chunks per slot.  The
// warp releases each slot on its own; no CTA-wide step.  Every lane ends with
// the row totals.  false: a wait gave up.
template <int OPK>
__device__ bool unit_dots(const DraftFusedArgs& a, DfCtl& ctl, const uint8_t* ring, const float* act,
                          int M, int n_slots, int kt_n, int trow_lo, int trow_hi, Ring& rg,
                          float (&acc)[2][kDfMaxRows], int w, int lane) {
  constexpr bool PAIR = OPK == OP_QKV || OPK == OP_GU;
  const int AF = a.act_floats;
#pragma unroll
  for (int q = 0; q < 2; ++q)
#pragma unroll
    for (int m = 0; m < kDfMaxRows; ++m) acc[q][m] = 0.f;
  const int sw_lo = (trow_lo + w) & 7, sw_hi = (trow_hi + w) & 7;
  for (int s = 0; s < n_slots; ++s) {
    if (!mbar_wait_bounded(&ctl.full[rg.i], rg.ph, &ctl.abort, a.status)) return false;
    const uint8_t* slot = ring + static_cast<size_t>(rg.i) * kDfSlotBytes;
    if constexpr (PAIR) {
      const int kt0 = s * 8, nkt = min(8, kt_n - kt0);
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        const int q = lane + 32 * h, ktl = q >> 3, c = q & 7;
        if (ktl < nkt) {
          const int kidx = (kt0 + ktl) * 64 + c * 8;
          const uint4 wa = *reinterpret_cast<const uint4*>(slot + ktl * 1024 + w * 128 + ((c ^ sw_lo) << 4));
          const uint4 wb =
              *reinterpret_cast<const uint4*>(slot + 8192 + ktl * 1024 + w * 128 + ((c ^ sw_hi) << 4));
          dot8(wa, act, AF, kidx, M, acc[0]);
          dot8(wb, act, AF, kidx, M, acc[1]);
        }
      }
    } else if (OPK == OP_LM && a.tied) {
      const int c0 = s * 1024;
#pragma unroll
      for (int h = 0; h < 4; ++h) {
        const int q = lane + 32 * h, kidx = c0 + q * 8;
        if (kidx < a.d) {
          const uint4 wv = *reinterpret_cast<const uint4*>(slot + h * 4096 + w * 512 + (lane << 4));
          dot8(wv, act, AF, kidx, M, acc[0]);
        }
      }
    } else {
      const int kt0 = s * 16, nkt = min(16, kt_n - kt0);
#pragma unroll
      for (int h = 0; h < 4; ++h) {
        const int q = lane + 32 * h, ktl = q >> 3, c = q & 7;
        if (ktl < nkt) {
          const uint4 wv = *reinterpret_cast<const uint4*>(slot + ktl * 1024 + w * 128 + ((c ^ sw_lo) << 4));
          dot8(wv, act, AF, (kt0 + ktl) * 64 + c * 8, M, acc[0]);
        }
      }
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(&ctl.empty[rg.i]);
    rg.next();
  }
  // fixed xor tree: every lane ends with the row totals
#pragma unroll
  for (int q = 0; q < (PAIR ? 2 : 1); ++q)
#pragma unroll
    for (int m = 0; m < kDfMaxRows; ++m) {
      if (m >= M) break;
      float x = acc[q][m];
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
      acc[q][m] = x;
    }
  return true;
}

__device__ __forceinline__ float pick(const float (&v)[kDfMaxRows], int m) {
  float r = 0.f;
#pragma unroll
  for (int i = 0; i < kDfMaxRows; ++i)
    if (i == m) r = v[i];
  return r;
}

// One (request, head, key split) of attention for the rows of request g: writes
// (m, l, o) in log2 units to the partial buffer; the O phase combines the
// splits (in split order) as it loads its input.  scratch: kDfScratchFloats
// floats.
template <int HD>
__device__ void attention_unit(const DraftFusedArgs& a, DfCtl& ctl, int layer, int g, int h, int s,
                               float* scratch, int tid) {
  constexpr int KG = kCT / HD;            // key groups of the PV product
  const int R = ctl.R, S = a.n_splits;
  const int nr = ctl.valid[g];
  const int p0 = ctl.pos0[g];
  const int ctx = p0 + nr;                // keys 0..ctx-1
  const int chunk = (ctx + S - 1) / S;
  const int k0 = s * chunk, k1 = min(k0 + chunk, ctx);
  const int kvh = h / (a.H / a.Hkv);
  const size_t kbase = static_cast<size_t>(layer) * 2 * a.layer_kv +
                       (static_cast<size_t>(g) * a.Hkv + kvh) * a.max_seq * HD;
  const bf16* kc = a.kv + kbase;
  const bf16* vc = kc + a.layer_kv;
  float* sc = scratch;                    // [2][kKeyBlock] scores, then weights
  float* qs = sc + 2 * kKeyBlock;         // [2][HD]
  float* op = qs + 2 * 128;               // [warps][2][HD] o partials
  const float qscale = 1.4426950408889634f / sqrtf(static_cast<float>(HD));
  // HD 64: the first key block's K row (one per thread) does not depend on q and
  // is requested before q is read, so q and K share one round trip (an HD 128
  // row held across the q loads would not fit the registers)
  constexpr bool kEarlyK = HD <= 64;
  uint4 kr0[kEarlyK ? HD / 8 : 1];
  if constexpr (kEarlyK) {
    if (k0 + tid < k1) {
      const uint4* src = reinterpret_cast<const uint4*>(kc + static_cast<size_t>(k0 + tid) * HD);
#pragma unroll
      for (int c = 0; c < HD / 8; ++c) kr0[c] = __ldcg(src + c);
    }
  }
  for (int e = tid; e < nr * HD; e += kCT) {
    const int i = e / HD, dd = e - i * HD;
    qs[e] = ldcg(a.qb + (static_cast<size_t>(g * R + i) * a.H + h) * HD + dd) * qscale;
  }
  float m_run[2] = {-INFINITY, -INFINITY}, l_run[2] = {0.f, 0.f};
  // PV: thread (d8, kg) accumulates dims 8 d8 .. 8 d8 + 7 over keys kg, kg + KG8, ...
  constexpr int D8 = HD / 8, KG8 = kCT / D8;
  const int d8 = tid % D8, kg = tid / D8;
  float o_run[2][8];
#pragma unroll
  for (int i = 0; i < 2; ++i)
#pragma unroll
    for (int e = 0; e < 8; ++e) o_run[i][e] = 0.f;
  csync();
  for (int kb = k0; kb < k1; kb += kKeyBlock) {
    const int t = kb + tid;
    float sco[2] = {-INFINITY, -INFINITY};
    if (t < k1) {
      // the whole key row in one round trip
      uint4 kr[HD / 8];
      const uint4* src = reinterpret_cast<const uint4*>(kc + static_cast<size_t>(t) * HD);
      if (kEarlyK && kb == k0) {
#pragma unroll
        for (int c = 0; c < HD / 8; ++c) kr[c] = kr0[kEarlyK ? c : 0];
      } else {
#pragma unroll
        for (int c = 0; c < HD / 8; ++c) kr[c] = __ldcg(src + c);
      }
      float dot[2] = {0.f, 0.f};
#pragma unroll
      for (int c = 0; c < HD / 8; ++c) {
        const float kf[8] = {bf_lo(kr[c].x), bf_hi(kr[c].x), bf_lo(kr[c].y), bf_hi(kr[c].y),
                             bf_lo(kr[c].z), bf_hi(kr[c].z), bf_lo(kr[c].w), bf_hi(kr[c].w)};
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          dot[0] = fmaf(qs[c * 8 + e], kf[e], dot[0]);
          dot[1] = fmaf(qs[HD + c * 8 + e], kf[e], dot[1]);
        }
      }
#pragma unroll
      for (int i = 0; i < 2; ++i)
        if (i < nr && t <= p0 + i) sco[i] = dot[i];
    }
    // block max per row
    float mx[2];
    {
      const int w = tid >> 5, lane = tid & 31;
#pragma unroll
      for (int i = 0; i < 2; ++i) {
        float x = sco[i];
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) x = fmaxf(x, __shfl_xor_sync(0xffffffffu, x, o));
        if (lane == 0) ctl.xch[w][i] = x;
      }
      csync();
#pragma unroll
      for (int i = 0; i < 2; ++i) {
        float x = -INFINITY;
        for (int ww = 0; ww < kCW; ++ww) x = fmaxf(x, ctl.xch[ww][i]);
        mx[i] = x;
      }
    }
    float alpha[2], mnew[2], p[2];
#pragma unroll
    for (int i = 0; i < 2; ++i) {
      mnew[i] = fmaxf(m_run[i], mx[i]);
      alpha[i] = (m_run[i] == -INFINITY) ? 0.f : exp2f(m_run[i] - mnew[i]);
      p[i] = (sco[i] == -INFINITY) ? 0.f : exp2f(sco[i] - mnew[i]);
      sc[i * kKeyBlock + tid] = p[i];
    }
    float ps[kDfMaxRows];
#pragma unroll
    for (int i = 0; i < kDfMaxRows; ++i) ps[i] = i < 2 ? p[i] : 0.f;
    block_row_sums(ctl, ps, 2, tid);       // also a barrier: sc is complete
#pragma unroll
    for (int i = 0; i < 2; ++i) {
      l_run[i] = l_run[i] * alpha[i] + ctl.red[0][i];
      m_run[i] = mnew[i];
#pragma unroll
      for (int e = 0; e < 8; ++e) o_run[i][e] *= alpha[i];
    }
    const int nk = min(kKeyBlock, k1 - kb);
    const bf16* vb = vc + static_cast<size_t>(kb) * HD + d8 * 8;
    constexpr int kPer = (kKeyBlock + KG8 - 1) / KG8;       // keys per thread per block
    uint4 vv[kPer];
#pragma unroll
    for (int q = 0; q < kPer; ++q) {
      const int tt = kg + q * KG8;
      vv[q] = tt < nk ? __ldcg(reinterpret_cast<const uint4*>(vb + static_cast<size_t>(tt) * HD))
                      : make_uint4(0u, 0u, 0u, 0u);
    }
#pragma unroll
    for (int q = 0; q < kPer; ++q) {
      const int tt = kg + q * KG8;
      if (tt < nk) {
        const float vf[8] = {bf_lo(vv[q].x), bf_hi(vv[q].x), bf_lo(vv[q].y), bf_hi(vv[q].y),
                             bf_lo(vv[q].z), bf_hi(vv[q].z), bf_lo(vv[q].w), bf_hi(vv[q].w)};
        const float p0v = sc[tt], p1v = sc[kKeyBlock + tt];
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          o_run[0][e] = fmaf(p0v, vf[e], o_run[0][e]);
          o_run[1][e] = fmaf(p1v, vf[e], o_run[1][e]);
        }
      }
    }
    csync();                                // sc is rewritten by the next block
  }
  // key groups: first across the lanes of a warp that share d8 (xor tree), then
  // the warps in order through shared memory
  {
    const int w = tid >> 5, lane = tid & 31;
#pragma unroll
    for (int i = 0; i < 2; ++i)
#pragma unroll
      for (int e = 0; e < 8; ++e)
#pragma unroll
        for (int o = 16; o >= D8; o >>= 1) o_run[i][e] += __shfl_xor_sync(0xffffffffu, o_run[i][e], o);
    if (lane < D8) {
#pragma unroll
      for (int i = 0; i < 2; ++i)
#pragma unroll
        for (int e = 0; e < 8; ++e) op[(w * 2 + i) * HD + lane * 8 + e] = o_run[i][e];
    }
  }
  csync();
  const int stride = HD + 4;
  float* mine = a.att + (static_cast<size_t>(g * R) * a.H + h) * S * stride;   // row i at + i * H * S * stride
  for (int e = tid; e < nr * HD; e += kCT) {
    const int i = e / HD, d2 = e - i * HD;
    float o = 0.f;
#pragma unroll
    for (int w = 0; w < kCW; ++w) o += op[(w * 2 + i) * HD + d2];
    mine[(static_cast<size_t>(i) * a.H * S + s) * stride + 4 + d2] = o;
  }
  if (tid < nr) {
    float* hdr = mine + (static_cast<size_t>(tid) * a.H * S + s) * stride;
    hdr[0] = tid == 0 ? m_run[0] : m_run[1];
    hdr[1] = tid == 0 ? l_run[0] : l_run[1];
  }
  // the splits are combined by every CTA of the O phase as it loads its input
}

// Sample request g's token of pass j from the LM-head statistics (warp 0);
// result in ctl.next_tok[g].
__device__ void sample_group(const DraftFusedArgs& a, DfCtl& ctl, int j, int g, int lane) {
  const int G = gridDim.x;
  const float* part = a.lm_part + static_cast<size_t>(g) * G * 4;
  const int per = (G + 31) / 32;               // <= 8 (grid <= 256)
  const int c_lo = min(lane * per, G), c_hi = min(c_lo + per, G);
  float pm[8], ps[8];
  int pa[8];
#pragma unroll
  for (int q = 0; q < 8; ++q) {
    float4 v = make_float4(-INFINITY, 0.f, __int_as_float(0x7fffffff), 0.f);
    if (c_lo + q < c_hi) v = __ldcg(reinterpret_cast<const float4*>(part + (c_lo + q) * 4));
    pm[q] = v.x;
    ps[q] = v.y;
    pa[q] = __float_as_int(v.z);
  }
  // max and first argmax
  float bm = -INFINITY;
  int ba = 0x7fffffff;
#pragma unroll
  for (int q = 0; q < 8; ++q)
    if (pm[q] > bm || (pm[q] == bm && pa[q] < ba)) {
      bm = pm[q];
      ba = pa[q];
    }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float om = __shfl_xor_sync(0xffffffffu, bm, o);
    const int oa = __shfl_xor_sync(0xffffffffu, ba, o);
    if (om > bm || (om == bm && oa < ba)) {
      bm = om;
      ba = oa;
    }
  }
  int tok = ba;
  if (!a.greedy) {
    const float it = a.inv_temp, M = bm;
    // per-CTA weights in CTA (= vocabulary) order, inclusive scan over lanes
    float wq[8], ls = 0.f;
#pragma unroll
    for (int q = 0; q < 8; ++q) {
      wq[q] = ps[q] > 0.f ? ps[q] * __expf((pm[q] - M) * it) : 0.f;
      ls += wq[q];
    }
    float incl = ls;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const float nb = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += nb;
    }
    float excl = __shfl_up_sync(0xffffffffu, incl, 1);
    if (lane == 0) excl = 0.f;
    const float total = __shfl_sync(0xffffffffu, incl, 31);
    const int step = a.seq_state[g * kStateInts + 2];
    const float u = philox_uniform(a.seeds[g], g, step, j - 1);
    const float target = u * total;
    int sel = -1;
    float before = 0.f;
    if (ls > 0.f && excl <= target && target < incl) {
      float cum = excl;
      bool done = false;
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        if (!done && wq[q] > 0.f) {
          sel = c_lo + q;
          before = cum;
          if (cum + wq[q] > target) done = true;
        }
        if (!done) cum += wq[q];
      }
    }
    const unsigned claim = __ballot_sync(0xffffffffu, sel >= 0);
    const int last_lane = 31 - __clz(__ballot_sync(0xffffffffu, ls > 0.f) | 1u);
    const int src = claim ? (__ffs(claim) - 1) : last_lane;
    if (!claim && lane == src) {
      float cum = excl;
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        if (wq[q] > 0.f) {
          sel = c_lo + q;
          before = cum;
        }
        cum += wq[q];
      }
    }
    sel = __shfl_sync(0xffffffffu, sel, src);
    before = __shfl_sync(0xffffffffu, before, src);
    if (total > 0.f && sel >= 0) {
      // the owning slice, in id order: contiguous ranges per lane
      const Geo geo = make_geo(a);
      const int v0 = lm_lo(geo, sel) * kUR, v1 = min(lm_lo(geo, sel + 1) * kUR, a.V);
      const int n = v1 - v0, pl = (n + 31) / 32;   // <= 32 (slice <= 1024 ids)
      const int x0 = min(v0 + lane * pl, v1), x1 = min(x0 + pl, v1);
      const float* z = a.zd + (static_cast<size_t>(g) * a.K + (j - 1)) * a.V;
      float wv[32];
#pragma unroll
      for (int q = 0; q < 32; ++q) wv[q] = x0 + q < x1 ? ldcg(z + x0 + q) : -INFINITY;
      float own = 0.f;
#pragma unroll
      for (int q = 0; q < 32; ++q) {
        wv[q] = x0 + q < x1 ? __expf((wv[q] - M) * it) : 0.f;
        own += wv[q];
      }
      float in2 = own;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const float nb = __shfl_up_sync(0xffffffffu, in2, o);
        if (lane >= o) in2 += nb;
      }
      float ex2 = __shfl_up_sync(0xffffffffu, in2, 1);
      if (lane == 0) ex2 = 0.f;
      const float r = target - before;
      int mine = -1, lastx = -1;
      {
        float cum = ex2;
        const bool scan = own > 0.f && ex2 <= r && r < in2;
#pragma unroll
        for (int q = 0; q < 32; ++q) {
          cum += wv[q];
          if (wv[q] > 0.f) {
            lastx = x0 + q;
            if (scan && mine < 0 && cum > r) mine = x0 + q;
          }
        }
        if (scan && mine < 0) mine = lastx;
      }
      const unsigned cl = __ballot_sync(0xffffffffu, mine >= 0);
      if (cl) {
        tok = __shfl_sync(0xffffffffu, mine, __ffs(cl) - 1);
      } else {   // r at or after the slice's scanned mass: its last id with mass
        const unsigned hm = __ballot_sync(0xffffffffu, lastx >= 0);
        if (hm) tok = __shfl_sync(0xffffffffu, lastx, 31 - __clz(hm));
      }
    }
  }
  if (lane == 0) ctl.next_tok[g] = tok;
}

__global__ void __launch_bounds__(kDfThreads, 1) draft_fused_kernel(const __grid_constant__ DraftFusedArgs a) {
  __shared__ DfCtl ctl;
  extern __shared__ __align__(128) uint8_t dsm[];
  uint8_t* ring = dsm;
  float* act = reinterpret_cast<float*>(dsm + static_cast<size_t>(a.ring_slots) * kDfSlotBytes);
  float* scratch = act + static_cast<size_t>(2 * a.B) * a.act_floats;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  if (tid == 0) {
    for (int i = 0; i < a.ring_slots; ++i) {
      mbar_init(&ctl.full[i], 1);
      mbar_init(&ctl.empty[i], kCW);
    }
    ctl.abort = 0;
    fence_mbar_init();
  }
  __syncthreads();
  if (warp == kCW) {
    if (lane == 0) producer(a, ctl, ring);
  } else {
    const Geo geo = make_geo(a);
    const int G = geo.G, c = geo.c;
    Ring rg;
    rg.S = a.ring_slots;
    unsigned epoch = 0;
    unsigned long long t_phase = global_ns();
    bool run = true;
    float acc[2][kDfMaxRows];
    for (int j = 1; j <= a.K && run; ++j) {
      // ---------------- the rows of this pass (one thread per request)
      if (tid < a.B) {
        const int g = tid, R = j == 1 ? 2 : 1;
        const int L = a.seq_state[g * kStateInts + 0];
        int valid, pos0;
        if (j == 1) {
          int nv = L - a.draft_len[g];
          if (nv < 1 || nv > 2) {
            atomicOr(a.status, 0x4u);     // draft cache not caught up
            nv = nv < 1 ? 1 : 2;
          }
          valid = nv;
          pos0 = L - nv;
        } else {
          valid = 1;
          pos0 = L + j - 2;
        }
        ctl.valid[g] = valid;
        ctl.pos0[g] = pos0;
        for (int i = 0; i < R; ++i) {
          const int r = g * R + i, pos = pos0 + i;
          bool ok = i < valid;
          int tok = 0;
          if (ok && (pos < 0 || pos >= a.max_seq)) {
            atomicOr(a.status, 0x4u);
            ok = false;
          }
          if (ok) {
            tok = j == 1 ? a.tokens[static_cast<size_t>(g) * a.max_seq + pos] : ctl.next_tok[g];
            if (tok < 0 || tok >= a.V) {
              atomicOr(a.status, 0x2u);
              tok = 0;
            }
          }
          ctl.ok[r] = ok ? 1 : 0;
          ctl.tok[r] = tok;
        }
      }
      if (tid == 0) {
        ctl.R = j == 1 ? 2 : 1;
        ctl.rows = a.B * ctl.R;
      }
      csync();
      const int R = ctl.R, rows = ctl.rows;
      int cum = 0;
      for (int l = 0; l < a.n_layers && run; ++l) {
        const size_t loff = static_cast<size_t>(l) * a.lstride;
        // ---------------- QKV + RoPE + KV append
        {
          // this layer's attention units: earlier keys into L2 while QKV runs
          const int units = a.B * a.H * a.n_splits;
          if (tid == 0)
            for (int ua = c; ua < units; ua += G) {
              const int g = ua / (a.H * a.n_splits), h = (ua / a.n_splits) % a.H, s = ua % a.n_splits;
              const int ctx = ctl.pos0[g] + ctl.valid[g];
              const int chunk = (ctx + a.n_splits - 1) / a.n_splits;
              const int k0 = s * chunk, k1 = min(min(k0 + chunk, ctx), ctl.pos0[g]);
              if (k1 > k0 && ctx <= a.max_seq) {
                const int kvh = h / (a.H / a.Hkv);
                const bf16* kc = a.kv + static_cast<size_t>(l) * 2 * a.layer_kv +
                                 (static_cast<size_t>(g) * a.Hkv + kvh) * a.max_seq * a.hd;
                const uint32_t nb = static_cast<uint32_t>(k1 - k0) * a.hd * 2;
                prefetch_l2(kc + static_cast<size_t>(k0) * a.hd, nb);
                prefetch_l2(kc + a.layer_kv + static_cast<size_t>(k0) * a.hd, nb);
              }
            }
          load_norm_rows(a, ctl, act, l == 0 ? 0 : 1,
                         reinterpret_cast<const bf16*>(a.w + a.off_attn_norm + loff), false, tid);
          const int off = cum % G;
          cum += geo.u_qkv;
          bool ok = true;
          const int half = a.hd / 2;
          for (int u = first_unit(geo, off); u < geo.u_qkv && ok; u += G) {
            int hb, ui, lo, hi;
            qkv_rows(a, u, &hb, &ui, &lo, &hi);
            ok = unit_dots<OP_QKV>(a, ctl, ring, act, rows, geo.s_qkv, geo.kt_d, lo % 128, hi % 128, rg, acc,
                                   warp, lane);
            if (!ok) break;
            // this warp's pair (fi, fi + hd/2) of head block hb; lane m: row m
            const int fi = kUR * ui + warp;
            if (lane < rows && ctl.ok[lane]) {
              const int m = lane, g = m / R, pos = ctl.pos0[g] + (m - g * R);
              const float x1 = pick(acc[0], m), x2 = pick(acc[1], m);
              if (hb < a.H + a.Hkv) {
                const float cs = a.rope_cos[static_cast<size_t>(pos) * half + fi];
                const float sn = a.rope_sin[static_cast<size_t>(pos) * half + fi];
                const float y1 = x1 * cs - x2 * sn, y2 = x1 * sn + x2 * cs;
                if (hb < a.H) {
                  float* qd = a.qb + (static_cast<size_t>(m) * a.H + hb) * a.hd;
                  qd[fi] = y1;
                  qd[fi + half] = y2;
                } else {
                  bf16* kd = a.kv + static_cast<size_t>(l) * 2 * a.layer_kv +
                             ((static_cast<size_t>(g) * a.Hkv + (hb - a.H)) * a.max_seq + pos) * a.hd;
                  kd[fi] = __float2bfloat16_rn(y1);
                  kd[fi + half] = __float2bfloat16_rn(y2);
                }
              } else {
                bf16* vd = a.kv + static_cast<size_t>(l) * 2 * a.layer_kv + a.layer_kv +
                           ((static_cast<size_t>(g) * a.Hkv + (hb - a.H - a.Hkv)) * a.max_seq + pos) * a.hd;
                vd[fi] = __float2bfloat16_rn(x1);
                vd[fi + half] = __float2bfloat16_rn(x2);
              }
            }
          }
          run = csync_and(ok);
          if (run) run = grid_sync(a, ctl, epoch, tid, t_phase);
        }
        // ---------------- attention
        if (run) {
          const int units = a.B * a.H * a.n_splits;
          for (int ua = c; ua < units; ua += G) {
            const int g = ua / (a.H * a.n_splits), h = (ua / a.n_splits) % a.H, s = ua % a.n_splits;
            bool grp_ok = true;
            for (int i = 0; i < ctl.valid[g]; ++i) grp_ok = grp_ok && ctl.ok[g * R + i];
            if (grp_ok) {
              if (a.hd == 64)
                attention_unit<64>(a, ctl, l, g, h, s, scratch, tid);
              else
                attention_unit<128>(a, ctl, l, g, h, s, scratch, tid);
            }
            csync();                            // scratch and ctl are reused by the next unit
          }
          run = grid_sync(a, ctl, epoch, tid, t_phase);
        }
        // ---------------- O projection + residual
        if (run) {
          const int off = cum % G;
          cum += geo.u_o;
          const int fu = first_unit(geo, off);
          if (fu < geo.u_o) {
            // the heads' attention outputs: every split's (m, l, o) of this
            // element in one round trip, combined here in split order
            //   o = sum_s 2^(m_s - M) o_s / sum_s 2^(m_s - M) l_s,  M = max_s m_s
            // (every CTA redoes it: cheaper than one more barrier)
            // hd / 4 lanes per (row, head), four features each, so that every
            // split's loads of a pair are in flight together
            const int S = a.n_splits, stride = a.hd + 4;
            const int lpp = a.hd / 4, pairs = rows * a.H, per_pass = kCT / lpp;
            for (int p0 = 0; p0 < pairs; p0 += per_pass) {
              const int p = p0 + tid / lpp, d = (tid % lpp) * 4;
              if (tid >= per_pass * lpp || p >= pairs) continue;
              const int m = p / a.H, hh = p - m * a.H;
              float4 o = make_float4(0.f, 0.f, 0.f, 0.f);
              if (ctl.ok[m]) {
                const float* base = a.att + (static_cast<size_t>(m) * a.H + hh) * S * stride;
                float2 ml[kDfMaxSplits];
                float4 ov[kDfMaxSplits];
#pragma unroll
                for (int q = 0; q < kDfMaxSplits; ++q) {
                  ml[q] = make_float2(-INFINITY, 0.f);
                  ov[q] = make_float4(0.f, 0.f, 0.f, 0.f);
                  if (q < S) {
                    ml[q] = __ldcg(reinterpret_cast<const float2*>(base + q * stride));
                    ov[q] = __ldcg(reinterpret_cast<const float4*>(base + q * stride + 4 + d));
                  }
                }
                float M = -INFINITY;
#pragma unroll
                for (int q = 0; q < kDfMaxSplits; ++q)
                  if (ml[q].y > 0.f) M = fmaxf(M, ml[q].x);
                float L = 0.f;
#pragma unroll
                for (int q = 0; q < kDfMaxSplits; ++q) {
                  const float w = ml[q].y > 0.f ? exp2f(ml[q].x - M) : 0.f;
                  L = fmaf(w, ml[q].y, L);
                  o.x = fmaf(w, ov[q].x, o.x);
                  o.y = fmaf(w, ov[q].y, o.y);
                  o.z = fmaf(w, ov[q].z, o.z);
                  o.w = fmaf(w, ov[q].w, o.w);
                }
                const float inv = L > 0.f ? 1.f / L : 0.f;
                o = make_float4(o.x * inv, o.y * inv, o.z * inv, o.w * inv);
              }
              *reinterpret_cast<float4*>(act + m * a.act_floats + hh * a.hd + d) = o;
            }
            csync();
          }
          bool ok = true;
          for (int u = fu; u < geo.u_o && ok; u += G) {
            const int row = u * kUR + warp;
            float hold = 0.f;
            if (lane < rows && ctl.ok[lane]) hold = ldcg(a.h + static_cast<size_t>(lane) * a.d + row);
            ok = unit_dots<OP_O>(a, ctl, ring, act, rows, geo.s_o, geo.kt_q, (u * kUR) % 128, 0, rg, acc, warp,
                                 lane);
            if (ok && lane < rows && ctl.ok[lane])
              a.h[static_cast<size_t>(lane) * a.d + row] = hold + pick(acc[0], lane);
          }
          run = csync_and(ok);
          if (run) run = grid_sync(a, ctl, epoch, tid, t_phase);
        }
        // ---------------- gate/up + SwiGLU
        if (run) {
          const int off = cum % G;
          cum += geo.u_gu;
          const int fu = first_unit(geo, off);
          if (fu < geo.u_gu)
            load_norm_rows(a, ctl, act, 1, reinterpret_cast<const bf16*>(a.w + a.off_ffn_norm + loff), false,
                           tid);
          bool ok = true;
          for (int u = fu; u < geo.u_gu && ok; u += G) {
            ok = unit_dots<OP_GU>(a, ctl, ring, act, rows, geo.s_gu, geo.kt_d, (u * kUR) % 64, (u * kUR) % 64, rg,
                                  acc, warp, lane);
            if (ok && lane < rows && ctl.ok[lane]) {
              const float gt = pick(acc[0], lane), up = pick(acc[1], lane);
              const float sg = gt / (1.f + expf(-gt));
              a.act[static_cast<size_t>(lane) * a.F + u * kUR + warp] = sg * up;
            }
          }
          run = csync_and(ok);
          if (run) run = grid_sync(a, ctl, epoch, tid, t_phase);
        }
        // ---------------- down + residual
        if (run) {
          const int off = cum % G;
          cum += geo.u_down;
          const int fu = first_unit(geo, off);
          if (fu < geo.u_down) {
            const int Fp = geo.kt_f * 64, n4 = rows * Fp / 4;
            for (int e0 = tid; e0 < n4; e0 += 4 * kCT) {
              float4 v[4];
#pragma unroll
              for (int q = 0; q < 4; ++q) {
                const int e = e0 + q * kCT;
                const int m = e < n4 ? (4 * e) / Fp : 0, k = 4 * e - m * Fp;
                v[q] = (e < n4 && k < a.F && ctl.ok[m])
                           ? __ldcg(reinterpret_cast<const float4*>(a.act + static_cast<size_t>(m) * a.F + k))
                           : make_float4(0.f, 0.f, 0.f, 0.f);
              }
#pragma unroll
              for (int q = 0; q < 4; ++q) {
                const int e = e0 + q * kCT;
                if (e < n4) {
                  const int m = (4 * e) / Fp, k = 4 * e - m * Fp;
                  *reinterpret_cast<float4*>(act + m * a.act_floats + k) = v[q];
                }
              }
            }
            csync();
          }
          bool ok = true;
          for (int u = fu; u < geo.u_down && ok; u += G) {
            const int row = u * kUR + warp;
            float hold = 0.f;
            if (lane < rows && ctl.ok[lane]) hold = ldcg(a.h + static_cast<size_t>(lane) * a.d + row);
            ok = unit_dots<OP_DOWN>(a, ctl, ring, act, rows, geo.s_down, geo.kt_f, (u * kUR) % 128, 0, rg, acc,
                                    warp, lane);
            if (ok && lane < rows && ctl.ok[lane])
              a.h[static_cast<size_t>(lane) * a.d + row] = hold + pick(acc[0], lane);
          }
          run = csync_and(ok);
          if (run) run = grid_sync(a, ctl, epoch, tid, t_phase);
        }
      }
      // ---------------- final RMSNorm + LM head (this CTA's vocabulary slice)
      if (run) {
        const int B = a.B;
        const int ulo = lm_lo(geo, c), uhi = lm_lo(geo, c + 1);
        float sm_m = -INFINITY, sm_s = 0.f;
        int sm_a = 0x7fffffff;
        if (ulo < uhi)
          load_norm_rows(a, ctl, act, 1, reinterpret_cast<const bf16*>(a.w + a.off_final_norm), true, tid);
        const bool greedy = a.greedy != 0;
        const float it = a.inv_temp;
        float* zrow = a.zd + (static_cast<size_t>(lane) * a.K + (j - 1)) * a.V;
        bool ok = true;
        for (int u = ulo; u < uhi && ok; ++u) {
          ok = unit_dots<OP_LM>(a, ctl, ring, act, B, geo.s_lm, geo.kt_d, (u * kUR) % 128, 0, rg, acc, warp,
                                lane);
          const int v = u * kUR + warp;
          if (ok && lane < B && v < a.V) {
            const float z = pick(acc[0], lane);
            zrow[v] = z;
            if (z > sm_m) {
              if (!greedy) sm_s = (sm_m == -INFINITY) ? 0.f : sm_s * __expf((sm_m - z) * it);
              sm_m = z;
              sm_a = v;
            }
            if (!greedy) sm_s += __expf((z - sm_m) * it);
          }
        }
        run = csync_and(ok);
        if (run) {
          // this CTA's statistics per request: warps combined in order
          if (lane < B) {
            ctl.stat_m[warp][lane] = sm_m;
            ctl.stat_s[warp][lane] = sm_s;
            ctl.stat_a[warp][lane] = sm_a;
          }
          csync();
          if (tid < B) {
            float M = -INFINITY;
            int A = 0x7fffffff;
            for (int w = 0; w < kCW; ++w) {
              const float m = ctl.stat_m[w][tid];
              const int ar = ctl.stat_a[w][tid];
              if (m > M || (m == M && ar < A)) {
                M = m;
                A = ar;
              }
            }
            float Ssum = 0.f;
            if (!greedy)
              for (int w = 0; w < kCW; ++w) {
                const float m = ctl.stat_m[w][tid];
                if (m != -INFINITY) Ssum += ctl.stat_s[w][tid] * __expf((m - M) * it);
              }
            float* p = a.lm_part + (static_cast<size_t>(tid) * G + c) * 4;
            p[0] = M;
            p[1] = Ssum;
            p[2] = __int_as_float(A);
          }
          run = grid_sync(a, ctl, epoch, tid, t_phase);
        }
      }
      // ---------------- sampling: every CTA before the next pass, CTA 0 after the last
      if (run && (j < a.K || c == 0)) {
        if (warp == 0)
          for (int g = 0; g < a.B; ++g) sample_group(a, ctl, j, g, lane);
        csync();
        if (c == 0 && tid < a.B) a.draft_tokens[tid * a.max_k + (j - 1)] = ctl.next_tok[tid];
        csync();
      }
    }
    // a consumer that stopped early releases the copy-issuing lane and the grid
    if (!run && tid == 0) {
      *reinterpret_cast<volatile int*>(&ctl.abort) = 1;
      atomicExch(&a.bar[2], 1u);
    }
  }
  __syncthreads();
  // the last CTA to leave resets the barrier counters for the next launch
  if (tid == 0) {
    __threadfence();
    if (atomicAdd(&a.bar[1], 1u) == gridDim.x - 1) {
      atomicExch(&a.bar[0], 0u);
      atomicExch(&a.bar[2], 0u);
      __threadfence();
      atomicExch(&a.bar[1], 0u);
    }
  }
}

}  // namespace

size_t draft_fused_smem_bytes(int ring_slots, int act_rows, int act_floats) {
  return static_cast<size_t>(ring_slots) * kDfSlotBytes + static_cast<size_t>(act_rows) * act_floats * 4 +
         static_cast<size_t>(kDfScratchFloats) * 4;
}

// Static shared memory of the kernel as compiled (the control block, padded).
size_t draft_fused_static_smem() {
  cudaFuncAttributes fa{};
  if (cudaFuncGetAttributes(&fa, draft_fused_kernel) != cudaSuccess) return 4096;
  return fa.sharedSizeBytes;
}

cudaError_t draft_fused_set_max_smem() {
  return cudaFuncSetAttribute(draft_fused_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              static_cast<int>(227 * 1024 - draft_fused_static_smem()));
}

cudaError_t launch_draft_fused(const DraftFusedArgs& a, int grid, cudaStream_t s, bool cooperative) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(kDfThreads);
  cfg.dynamicSmemBytes = draft_fused_smem_bytes(a.ring_slots, 2 * a.B, a.act_floats);
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeCooperative;
  attr[0].val.cooperative = 1;
  cfg.attrs = attr;
  cfg.numAttrs = cooperative ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, draft_fused_kernel, a);
}

}  // namespace memspec
