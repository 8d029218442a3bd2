// gemm_epi.cuh - device code shared by the projection GEMM kernel and the
// persistent pass kernel: tile constants, activation-operand layouts, the fused
// epilogues, and the per-segment epilogue routine (TMEM -> registers -> either
// the epilogue or a split-K partial; the last contributor of a row tile sums
// the partials in ascending CTA order).
#pragma once
#include <cuda_bf16.h>

#include "internal.h"
#include "ptx.cuh"

namespace memspec {
namespace gemm {

constexpr int kTileM = 128;
constexpr int kTileK = 64;
constexpr int kABytes = kTileM * kTileK * 2;  // 16 KB
constexpr int kMaxStages = 12;
constexpr int kStagePitch = 17;                // epilogue staging row pitch (floats)
constexpr int kStageFloats = kTileM * kStagePitch;

// MMA layouts of the activation operand:
//   kPlain  one bf16 plane, N = n_pad
//   kWide   hi and lo planes as one operand of N = 2 n_pad (one MMA per k-step);
//           accumulator columns [0, n_pad) hold W.hi, [n_pad, 2 n_pad) W.lo
//   kTwice  hi and lo planes as two MMAs into the same accumulator (2 n_pad > 256)
enum BLayout : int { kPlain = 0, kWide = 1, kTwice = 2 };

__device__ __forceinline__ int acc_cols(const GemmArgs& a, int layout) {
  return layout == kWide ? 2 * a.n_pad : a.n_pad;
}

__device__ __forceinline__ uint32_t tmem_cols_for(int cols) {
  uint32_t need = 2u * static_cast<uint32_t>(cols);
  uint32_t c = 32;
  while (c < need) c <<= 1;
  return c;
}

__device__ __forceinline__ bool row_valid(const GemmArgs& a, int r) {
  if (r >= a.rows_total) return false;
  return a.plan == nullptr ? true : plan_row_valid(a.plan, r);
}

// Per-launch epilogue context in shared memory.  The epilogue warps fill it
// while the weights stream (epi_prologue), so that the tail of the launch - the
// split-K reduction and the epilogue - reads no row plan or RoPE table from
// global memory: each such read would be a dependent L2 round trip there.
constexpr int kCtxRopeRows = 16;   // rows whose RoPE cos/sin are staged (the first chunk)
struct EpiCtx {
  int pos[kMaxRows];               // KV slot of each row (plan rows)
  int rpos[kTreeRows];             // RoPE position of rows < 32 (differs in tree passes)
  int req[kMaxRows];               // its request
  int grp[kMaxRows];               // its group
  uint32_t valid[kMaxRows / 32];   // bit r: row r is valid
  uint32_t last[kMaxRows / 32];    // bit r: row r is the last valid row of its group
  float rc[kCtxRopeRows][64];      // EPI_QKV: cos / sin at (row, rotation pair)
  float rs[kCtxRopeRows][64];
};

__device__ __forceinline__ bool ctx_bit(const uint32_t* w, int r) { return (w[r >> 5] >> (r & 31)) & 1u; }

// Fill the context (the 128 epilogue threads, et = 0..127); ends with a barrier.
template <int EPI>
__device__ __forceinline__ void epi_prologue(const GemmArgs& a, EpiCtx* ctx, int et) {
  const RowPlan* plan = a.plan;
  const int rows_total = a.rows_total, n_pad = a.n_pad;
  const int R = plan != nullptr ? plan->rows_per_group : 1;
  for (int base = 0; base < n_pad; base += 128) {   // uniform trip count: ballots below
    const int r = base + et;
    bool valid = false, last = false;
    int g = 0, pos = 0, rpos = 0, req = 0;
    if (r < rows_total) {
      if (plan == nullptr) {
        valid = true;
      } else {
        g = r / R;
        const int i = r - g * R;
        const int nv = plan->valid[g];
        valid = i < nv;
        last = i == nv - 1;
        pos = plan->pos0[g] + i;
        rpos = (plan->tree && i < kTreeRows) ? plan->pos0[g] + plan->rope_off[i] : pos;
        req = plan->req[g];
      }
    }
    if (r < n_pad) {
      ctx->pos[r] = pos;
      if (r < kTreeRows) ctx->rpos[r] = rpos;
      ctx->req[r] = req;
      ctx->grp[r] = g;
    }
    const uint32_t vb = __ballot_sync(0xffffffffu, valid);
    const uint32_t lb = __ballot_sync(0xffffffffu, last);
    if ((et & 31) == 0 && r < kMaxRows) {
      ctx->valid[r >> 5] = vb;
      ctx->last[r >> 5] = lb;
    }
  }
  named_bar_sync(1, 128);
  if constexpr (EPI == EPI_QKV) {
    const int half = a.head_dim >> 1;
    const int nr = min(n_pad, kCtxRopeRows);
    for (int idx = et; idx < nr * half; idx += 128) {
      const int j = idx / half, ip = idx - j * half;
      const int pos = ctx->pos[j];
      const bool ok = ctx_bit(ctx->valid, j) && pos >= 0 && pos < a.max_seq;
      const size_t ri = ok ? static_cast<size_t>(j < kTreeRows ? ctx->rpos[j] : pos) * half + ip : 0;
      ctx->rc[j][ip] = a.rope_cos[ri];
      ctx->rs[j][ip] = a.rope_sin[ri];
    }
    named_bar_sync(1, 128);
  }
}

// Epilogue for one 16-row chunk of a finished 128-feature row tile.  Called by
// the 128 epilogue threads together; et = feature within the tile (= TMEM lane).
// EPI (a GemmEpi) is a template argument so that a kernel carries the code of
// one epilogue only: the tail of a launch runs this code once, cold, and every
// instruction-cache miss there sits on the critical path.
template <int EPI>
static __device__ __noinline__ void apply_epilogue(const GemmArgs& a, const EpiCtx* ctx,
                                                   float (*red)[16], float* stage,
                                                   const float* rms, int rt, int chunk, int et,
                                                   const float* vin, unsigned long long* ts,
                                                   bool dry) {
  const int ew = et >> 5, lane = et & 31;
  constexpr int epi = EPI;
  const int rows_total = a.rows_total;
  const int r0 = chunk * 16;
  float v[16];
  if (a.rms) {
#pragma unroll
    for (int j = 0; j < 16; ++j) v[j] = vin[j] * rms[r0 + j];
  } else {
#pragma unroll
    for (int j = 0; j < 16; ++j) v[j] = vin[j];
  }
  if constexpr (epi == EPI_F32) {
    const int f = rt * kTileM + et;
    const int n_out = a.n_out, out_ld = a.out_ld, last_only = a.last_only;
    const long long gstride = a.out_group_stride;
    float* out = a.out;
    if (f < n_out) {
#pragma unroll
      for (int j = 0; j < 16; ++j) {
        const int r = r0 + j;
        if (last_only) {
          if (ctx_bit(ctx->last, r) && !dry) out[ctx->grp[r] * gstride + f] = v[j];
        } else if (ctx_bit(ctx->valid, r) && !dry) {
          out[static_cast<size_t>(r) * out_ld + f] = v[j];
        }
      }
    }
    return;
  }
  if constexpr (epi == EPI_RESIDUAL) {
    const int f = rt * kTileM + et;  // n_out is a multiple of 128 (d_model)
    float* h = a.h;
    const int h_ld = a.h_ld;
    const bf16* gain_next = a.gain_next;
    bf16* xg_out = a.xg_out;
    bf16* xg_lo_out = a.xg_lo_out;
    float* ss_out = a.ss_out;
    const int ss_stride = a.ss_stride;
    const float gain = gain_next != nullptr ? __bfloat162float(gain_next[f]) : 0.f;
    float hn[16], sq[16];
#pragma unroll
    for (int j = 0; j < 16; ++j)
      hn[j] = (r0 + j < rows_total) ? h[static_cast<size_t>(r0 + j) * h_ld + f] : 0.f;
    trace_after(ts, 8, hn[0] + gain);
#pragma unroll
    for (int j = 0; j < 16; ++j) {
      hn[j] += v[j];
      sq[j] = (r0 + j < rows_total) ? hn[j] * hn[j] : 0.f;
    }
#pragma unroll
    for (int j = 0; j < 16; ++j) {
      const int r = r0 + j;
      if (r >= rows_total || dry) continue;
      const size_t o = static_cast<size_t>(r) * h_ld + f;
      h[o] = hn[j];
      if (gain_next != nullptr)
        store_split_bf16(xg_out + o, xg_lo_out != nullptr ? xg_lo_out + o : nullptr, hn[j] * gain);
    }
    trace_at(ts, 12);
    // per-row sums over the warp's 32 features, valid rows only (a decode pass
    // has 1 to a few rows of the 16)
#pragma unroll
    for (int j = 0; j < 16; ++j) {
      if (r0 + j < rows_total) {
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) sq[j] += __shfl_xor_sync(0xffffffffu, sq[j], o);
      }
    }
    trace_after(ts, 14, sq[0]);
    if (lane == 0) {
#pragma unroll
      for (int j = 0; j < 16; ++j) red[ew][j] = sq[j];
    }
    trace_at(ts, 9);
    named_bar_sync(1, 128);
    trace_at(ts, 10);
    if (et < 16) {
      const int r = r0 + et;
      if (r < rows_total && !dry) {
        const float s = ((red[0][et] + red[1][et]) + red[2][et]) + red[3][et];
        ss_out[static_cast<size_t>(rt) * ss_stride + r] = s;
      }
    }
    named_bar_sync(1, 128);
    trace_at(ts, 11);
    return;
  }
  if constexpr (epi == EPI_SWIGLU || epi == EPI_QKV) {
    // staged epilogues: make the whole 128 x 16 chunk visible to all 128 threads
#pragma unroll
    for (int j = 0; j < 16; ++j) stage[et * kStagePitch + j] = v[j];
    named_bar_sync(1, 128);
    if constexpr (epi == EPI_SWIGLU) {
      if (et < 64) {
        const int f = rt * 64 + et;
        if (f < a.n_out) {
          bf16* act = a.act;
          bf16* act_lo = a.act_lo;
          const int act_ld = a.act_ld;
          // rolled: the inputs are in shared memory, and a launch runs this once,
          // with a cold instruction cache
#pragma unroll 1
          for (int j = 0; j < 16; ++j) {
            const int r = r0 + j;
            if (r >= rows_total) break;
            const float g = stage[et * kStagePitch + j];
            const float u = stage[(et + 64) * kStagePitch + j];
            const float y = g / (1.0f + expf(-g)) * u;
            if (dry) continue;
            const size_t o = static_cast<size_t>(r) * act_ld + f;
            store_split_bf16(act + o, act_lo != nullptr ? act_lo + o : nullptr, y);
          }
        }
      }
    } else {  // EPI_QKV: RoPE on q and k, K/V appended to the cache
      const int f = rt * kTileM + et;
      const int q_dim = a.q_dim, kv_dim = a.kv_dim;
      const int hd = a.head_dim, half_hd = hd >> 1;
      const int n_kv_heads = a.n_kv_heads, max_seq = a.max_seq;
      float* q_out = a.q_out;
      const float* rope_cos = a.rope_cos;
      const float* rope_sin = a.rope_sin;
      int seg, fs;
      if (f < q_dim) {
        seg = 0;
        fs = f;
      } else if (f < q_dim + kv_dim) {
        seg = 1;
        fs = f - q_dim;
      } else {
        seg = 2;
        fs = f - q_dim - kv_dim;
      }
      const int head = fs / hd, d = fs - head * hd;
      const int ip = d < half_hd ? d : d - half_hd;   // rotation pair index
      const int e1 = et - d + ip;                     // staging index of element ip of this head
      bf16* cache = seg == 1 ? a.kcache : a.vcache;
      if (chunk == 0) {
        // rolled (see SwiGLU): every input of the first chunk is in shared memory
#pragma unroll 1
        for (int j = 0; j < 16; ++j) {
          const int r = j;
          const int pos = ctx->pos[r];
          // invalid positions were flagged by the embedding kernel: skip the row
          if (!(ctx_bit(ctx->valid, r) && pos >= 0 && pos < max_seq)) continue;
          float y = stage[et * kStagePitch + j];
          if (seg < 2) {
            const float c = ctx->rc[j][ip], sn = ctx->rs[j][ip];
            const float x1 = stage[e1 * kStagePitch + j];
            const float x2 = stage[(e1 + half_hd) * kStagePitch + j];
            y = d < half_hd ? (x1 * c - x2 * sn) : (x1 * sn + x2 * c);
          }
          if (dry) continue;
          if (seg == 0) {
            q_out[static_cast<size_t>(r) * q_dim + f] = y;
          } else {
            const size_t off =
                ((static_cast<size_t>(ctx->req[r]) * n_kv_heads + head) * max_seq + pos) * hd + d;
            cache[off] = __float2bfloat16_rn(y);
          }
        }
      } else {
        // later chunks (batched and prefill passes): the sixteen rows' cos / sin
        // are loaded together, before any store
        float y[16];
        uint32_t ok_mask = 0;
#pragma unroll
        for (int j = 0; j < 16; ++j) {
          const int r = r0 + j;
          const int pos = ctx->pos[r];
          const bool ok = ctx_bit(ctx->valid, r) && pos >= 0 && pos < max_seq;
          if (ok) ok_mask |= 1u << j;
          y[j] = stage[et * kStagePitch + j];
          if (seg < 2) {
            const size_t ri = ok ? static_cast<size_t>(r < kTreeRows ? ctx->rpos[r] : pos) * half_hd + ip : 0;
            const float c = rope_cos[ri], sn = rope_sin[ri];
            const float x1 = stage[e1 * kStagePitch + j];
            const float x2 = stage[(e1 + half_hd) * kStagePitch + j];
            y[j] = d < half_hd ? (x1 * c - x2 * sn) : (x1 * sn + x2 * c);
          }
        }
        if (dry) ok_mask = 0;
#pragma unroll
        for (int j = 0; j < 16; ++j) {
          if (!(ok_mask & (1u << j))) continue;
          const int r = r0 + j;
          if (seg == 0) {
            q_out[static_cast<size_t>(r) * q_dim + f] = y[j];
          } else {
            const size_t off =
                ((static_cast<size_t>(ctx->req[r]) * n_kv_heads + head) * max_seq + ctx->pos[r]) * hd + d;
            cache[off] = __float2bfloat16_rn(y[j]);
          }
        }
      }
    }
    named_bar_sync(1, 128);  // staging buffer is reused by the next chunk
  }
}

// Per-row RMSNorm scale from the partial sums of squares (128 epilogue threads).
__device__ __forceinline__ void rms_prologue(const GemmArgs& a, float* rms, int et) {
  for (int r = et; r < a.n_pad; r += 128) {
    float val = 0.f;
    if (r < a.rows_total) {
      float sum = 0.f;
      // partial sums added in index order; loads issued eight at a time
      for (int i0 = 0; i0 < a.ss_count; i0 += 8) {
        float t[8];
#pragma unroll
        for (int q = 0; q < 8; ++q)
          t[q] = (i0 + q < a.ss_count) ? a.ss[static_cast<size_t>(i0 + q) * a.ss_stride + r] : 0.f;
#pragma unroll
        for (int q = 0; q < 8; ++q) sum += t[q];
      }
      val = rsqrtf(sum / static_cast<float>(a.k_in) + a.eps);
    }
    rms[r] = val;
  }
  named_bar_sync(1, 128);
}

// rms_prologue for the 16 rows of one chunk only (threads et < 16, the same
// summation order, every partial sum of a row in flight at once); ends with a
// barrier over the 128 threads.
__device__ __forceinline__ void rms_chunk(const GemmArgs& a, float* rms, int chunk, int et) {
  const int r = chunk * 16 + et;
  if (et < 16 && r < a.n_pad) {
    float val = 0.f;
    if (r < a.rows_total) {
      float sum = 0.f;
      for (int i0 = 0; i0 < a.ss_count; i0 += 32) {
        float t[32];
#pragma unroll
        for (int q = 0; q < 32; ++q)
          t[q] = (i0 + q < a.ss_count) ? a.ss[static_cast<size_t>(i0 + q) * a.ss_stride + r] : 0.f;
#pragma unroll
        for (int q = 0; q < 32; ++q) sum += t[q];
      }
      val = rsqrtf(sum / static_cast<float>(a.k_in) + a.eps);
    }
    rms[r] = val;
  }
  named_bar_sync(1, 128);
}

// Sum of the split-K partials of row tile rt, chunk `chunk`, for feature et:
// contributors in ascending CTA order, four fetched at once.
__device__ __forceinline__ void reduce_partials(const GemmArgs& a, int rt, int c_first, int c_last,
                                                int chunk, int et, int T, int G, float* v) {
  const int KT = a.k_tiles;
#pragma unroll
  for (int j = 0; j < 16; ++j) v[j] = 0.f;
  for (int cc0 = c_first; cc0 <= c_last; cc0 += 4) {
    float4 tmp[4][4];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const int cc = cc0 + q;
      if (cc <= c_last) {
        const int sl = (sk_begin(cc, T, G) >= rt * KT) ? 0 : 1;
        const float* pp = a.partials + static_cast<size_t>(2 * cc + sl) * a.n_pad * kTileM +
                          (static_cast<size_t>(chunk) * kTileM + et) * 16;
#pragma unroll
        for (int e = 0; e < 4; ++e) tmp[q][e] = ld_cg_f4(pp + 4 * e);
      }
    }
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      if (cc0 + q <= c_last) {
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          v[4 * e] += tmp[q][e].x;
          v[4 * e + 1] += tmp[q][e].y;
          v[4 * e + 2] += tmp[q][e].z;
          v[4 * e + 3] += tmp[q][e].w;
        }
      }
    }
  }
}

// Synthetic context for the dry run (below): every row valid, position and
// request 0, so every address the dry run forms is in bounds.  Ends with a barrier.
__device__ __forceinline__ void epi_ctx_dry(EpiCtx* ctx, int n_pad, int et) {
  for (int r = et; r < n_pad; r += 128) {
    ctx->pos[r] = 0;
    if (r < kTreeRows) ctx->rpos[r] = 0;
    ctx->req[r] = 0;
    ctx->grp[r] = 0;
  }
  if (et < kMaxRows / 32) {
    ctx->valid[et] = 0xffffffffu;
    ctx->last[et] = 0u;
  }
  for (int i = et; i < kCtxRopeRows * 64; i += 128) {
    ctx->rc[i / 64][i % 64] = 1.f;
    ctx->rs[i / 64][i % 64] = 0.f;
  }
  named_bar_sync(1, 128);
}

// Cluster exchange, first contributor: its own accumulator plus the n_recv
// pushed partials in contributor order, then the epilogue (dry: nothing stored).
template <int EPI>
static __device__ __noinline__ void csk_reduce(const GemmArgs& a, const EpiCtx* ctx,
                                               float (*red)[16], float* stage, const float* rms,
                                               int rt, int et, const float* own, const float* recv,
                                               int n_recv, unsigned long long* ts, bool dry) {
  float sum[16];
#pragma unroll
  for (int j = 0; j < 16; ++j) sum[j] = 0.f + own[j];
  for (int k = 0; k < n_recv; ++k) {
    const float4* src = reinterpret_cast<const float4*>(recv + (static_cast<size_t>(k) * kTileM + et) * 16);
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const float4 x = src[q];
      sum[4 * q] += x.x;
      sum[4 * q + 1] += x.y;
      sum[4 * q + 2] += x.z;
      sum[4 * q + 3] += x.w;
    }
  }
  trace_after(ts, 6, sum[15]);
  apply_epilogue<EPI>(a, ctx, red, stage, rms, rt, 0, et, sum, ts, dry);
}

// Dry run of the tail - the partial reduction and the epilogue of this CTA's
// first row tile, with every global store off - by the 128 epilogue threads
// before the launch waits for its predecessor (griddepcontrol.wait): it only
// reads scratch and weights, with the synthetic context of epi_ctx_dry.  The
// tail runs once per launch; without this its instructions are fetched cold,
// one miss after another, on the critical path.  With the cluster exchange, a
// CTA that sums pushed partials warms that path instead (on whatever its
// receive slots hold; nothing is stored).
template <int EPI, bool CSK>
__device__ __forceinline__ void epilogue_warmup(const GemmArgs& a, const EpiCtx* ctx,
                                                float (*red)[16], float* stage, const float* rms,
                                                int c, int G, int et, const float* recv,
                                                bool csk_reducer) {
  const int KT = a.k_tiles, T = a.row_tiles * KT;
  float v[16];
  if constexpr (CSK) {
    if (csk_reducer) {
      const int rt = (sk_begin(c + 1, T, G) - 1) / KT;
#pragma unroll
      for (int j = 0; j < 16; ++j) v[j] = 0.f;
      csk_reduce<EPI>(a, ctx, red, stage, rms, rt, et, v, recv, a.csk - 1, nullptr, true);
      return;
    }
  }
  const int rt = sk_begin(c, T, G) / KT;
  const int c_first = sk_cta_of(rt * KT, T, G);
  const int c_last = sk_cta_of((rt + 1) * KT - 1, T, G);
  reduce_partials(a, rt, c_first, c_last, 0, et, T, G, v);
  apply_epilogue<EPI>(a, ctx, red, stage, rms, rt, 0, et, v, nullptr, true);
}

// Epilogue of one accumulated segment [k0, k1) of row tile rt, run by the 128
// epilogue threads (et = TMEM lane = tile feature).  `c` is this CTA's index and
// G the op's grid; T = row_tiles * k_tiles.  The caller has waited for the
// accumulator; this routine reads it (wide layout: adds the hi and lo halves),
// releases it via acc_empty, and writes the epilogue or a partial.
//
// Cluster exchange (CSK: a kernel launched in clusters, a.csk > 1, n_pad == 16;
// kernels without it carry none of this code): when every contributor of row tile
// rt sits in this CTA's cluster, the contributors after the first push their
// accumulator into slot (c - c_first - 1) of the first contributor's `recv`
// (st.async, completing bytes on its `recv_bar`) and are done; the first
// contributor - for which rt is the last row tile of its range, so `recv` is
// used once per launch - waits for the bytes and adds the slots to its own
// accumulator in contributor order, the order of the global-memory path.
template <int EPI, bool CSK>
__device__ __forceinline__ void epilogue_segment(const GemmArgs& a, const EpiCtx* ctx, int layout,
                                                 int acols,
                                                 uint32_t tmem_base, int buf, int seg, int c,
                                                 int G, int rt, int k0, int k1, float* stage,
                                                 const float* rms, float (*red)[16],
                                                 int* reduce_flag, uint64_t* acc_empty, int et,
                                                 int ew, int lane, float* recv, uint64_t* recv_bar,
                                                 volatile int* abort_flag,
                                                 unsigned long long* ts = nullptr) {
  const int KT = a.k_tiles;
  const int T = a.row_tiles * KT;
  const bool full = (k0 == 0 && k1 == KT);
  const int c_first = sk_cta_of(rt * KT, T, G);
  const int c_last = sk_cta_of((rt + 1) * KT - 1, T, G);
  const bool dsm = CSK && !full && c_first / a.csk == c_last / a.csk;
  const uint32_t tbase = tmem_base + (static_cast<uint32_t>(ew * 32) << 16) +
                         static_cast<uint32_t>(buf * acols);
  float v[16];
  auto load_chunk = [&](int chunk) {
    tmem_ld_32x32b_x16(tbase + chunk * 16, v);
    if (layout == kWide) {
      float lo[16];
      tmem_ld_32x32b_x16(tbase + a.n_pad + chunk * 16, lo);
#pragma unroll
      for (int j = 0; j < 16; ++j) v[j] += lo[j];
    }
  };
  if (full) {
    for (int chunk = 0; chunk < a.n_pad / 16; ++chunk) {
      load_chunk(chunk);
      apply_epilogue<EPI>(a, ctx, red, stage, rms, rt, chunk, et, v, nullptr, false);
    }
  } else if (CSK && dsm) {
    load_chunk(0);   // n_pad == 16: the whole accumulator
    if (c != c_first) {
      const uint32_t rank = static_cast<uint32_t>(c_first % a.csk);
      const uint32_t slot = smem_addr(recv + (static_cast<size_t>(c - c_first - 1) * kTileM + et) * 16);
      const uint32_t raddr = mapa_shared(slot, rank);
      const uint32_t rbar = mapa_shared(smem_addr(recv_bar), rank);
#pragma unroll
      for (int q = 0; q < 4; ++q)
        st_async_f4(raddr + 16 * q, v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3], rbar);
    }
  } else {
    // partial sums, chunk-major: the 16 rows of chunk k for feature et at
    // ((k * 128) + et) * 16 (a warp's stores, and a reader's loads, of one chunk
    // are one contiguous 2 KB run)
    const int slot = (seg == 0) ? 0 : 1;
    float* pb = a.partials + static_cast<size_t>(2 * c + slot) * a.n_pad * kTileM +
                static_cast<size_t>(et) * 16;
    for (int chunk = 0; chunk < a.n_pad / 16; ++chunk) {
      load_chunk(chunk);
      float4* dst = reinterpret_cast<float4*>(pb + static_cast<size_t>(chunk) * kTileM * 16);
#pragma unroll
      for (int q = 0; q < 4; ++q) dst[q] = make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
    }
  }
  tc_fence_before();
  __syncwarp();
  if (lane == 0) mbar_arrive(&acc_empty[buf]);
  if (full) return;
  trace_at(ts, 4);
  if (a.split_epi) return;   // the split epilogue kernel finishes this row tile
  if (CSK && dsm) {
    if (c != c_first) return;
    // one thread waits; the epilogue threads follow (or stop) together, then each
    // acquires the peers' bytes itself (the phase is complete: no wait)
    if (et == 0) *reduce_flag = mbar_wait_cluster_bounded(recv_bar, 0, abort_flag, a.status) ? 1 : 0;
    named_bar_sync(1, 128);
    const int ok = *reduce_flag;
    named_bar_sync(1, 128);
    if (!ok) return;
    mbar_wait_cluster_bounded(recv_bar, 0, nullptr, nullptr);
    trace_at(ts, 5);
    csk_reduce<EPI>(a, ctx, red, stage, rms, rt, et, v, recv, c_last - c_first, ts, false);
    trace_at(ts, 7);
    return;
  }
  // The barrier orders this CTA's partial stores before thread 0's arrival, whose
  // release (acq_rel, GPU scope) publishes them; the last contributor's acquire
  // and the second barrier order every other contributor's partials before its
  // loads (which bypass L1).
  named_bar_sync(1, 128);
  if (et == 0) {
    const int old = atom_add_acq_rel_gpu(&a.counters[rt], 1);
    *reduce_flag = (old == c_last - c_first) ? 1 : 0;
  }
  named_bar_sync(1, 128);
  trace_at(ts, 5);
  if (!*reduce_flag) return;
  for (int chunk = 0; chunk < a.n_pad / 16; ++chunk) {
    reduce_partials(a, rt, c_first, c_last, chunk, et, T, G, v);
    if (chunk == 0) trace_after(ts, 6, v[15]);
    apply_epilogue<EPI>(a, ctx, red, stage, rms, rt, chunk, et, v, ts, false);
  }
  trace_at(ts, 7);
  if (et == 0) a.counters[rt] = 0;
}

}  // namespace gemm
}  // namespace memspec
