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

// Epilogue for one 16-row chunk of a finished 128-feature row tile.  Called by
// the 128 epilogue threads together; et = feature within the tile (= TMEM lane).
static __device__ __noinline__ void apply_epilogue(const GemmArgs& a, float (*red)[16], float* stage,
                                            const float* rms, int rt, int chunk, int et,
                                            const float* vin) {
  const int ew = et >> 5, lane = et & 31;
  float v[16];
#pragma unroll
  for (int j = 0; j < 16; ++j) v[j] = a.rms ? vin[j] * rms[chunk * 16 + j] : vin[j];
  if (a.epi == EPI_F32) {
    const int f = rt * kTileM + et;
    if (f < a.n_out) {
#pragma unroll
      for (int j = 0; j < 16; ++j) {
        const int r = chunk * 16 + j;
        if (!row_valid(a, r)) continue;
        if (a.last_only) {
          const int g = r / a.plan->rows_per_group;
          const int i = r - g * a.plan->rows_per_group;
          if (i != a.plan->valid[g] - 1) continue;
          a.out[g * a.out_group_stride + f] = v[j];
        } else {
          a.out[static_cast<size_t>(r) * a.out_ld + f] = v[j];
        }
      }
    }
    return;
  }
  if (a.epi == EPI_RESIDUAL) {
    const int f = rt * kTileM + et;  // n_out is a multiple of 128 (d_model)
#pragma unroll
    for (int j = 0; j < 16; ++j) {
      const int r = chunk * 16 + j;
      float sq = 0.f;
      if (r < a.rows_total) {
        float* hp = a.h + static_cast<size_t>(r) * a.h_ld + f;
        const float hn = *hp + v[j];
        *hp = hn;
        sq = hn * hn;
        if (a.gain_next != nullptr) {
          const float xv = hn * __bfloat162float(a.gain_next[f]);
          const size_t o = static_cast<size_t>(r) * a.h_ld + f;
          if (a.xg_lo_out != nullptr) {
            split_bf16(xv, a.xg_out[o], a.xg_lo_out[o]);
          } else {
            a.xg_out[o] = __float2bfloat16_rn(xv);
          }
        }
      }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) sq += __shfl_xor_sync(0xffffffffu, sq, o);
      if (lane == 0) red[ew][j] = sq;
    }
    named_bar_sync(1, 128);
    if (et < 16) {
      const int r = chunk * 16 + et;
      if (r < a.rows_total) {
        const float s = ((red[0][et] + red[1][et]) + red[2][et]) + red[3][et];
        a.ss_out[static_cast<size_t>(rt) * a.ss_stride + r] = s;
      }
    }
    named_bar_sync(1, 128);
    return;
  }
  // staged epilogues: make the whole 128 x 16 chunk visible to all 128 threads
#pragma unroll
  for (int j = 0; j < 16; ++j) stage[et * kStagePitch + j] = v[j];
  named_bar_sync(1, 128);
  if (a.epi == EPI_SWIGLU) {
    if (et < 64) {
      const int f = rt * 64 + et;
      if (f < a.n_out) {
#pragma unroll
        for (int j = 0; j < 16; ++j) {
          const int r = chunk * 16 + j;
          if (r >= a.rows_total) continue;
          const float g = stage[et * kStagePitch + j];
          const float u = stage[(et + 64) * kStagePitch + j];
          const float sg = g / (1.0f + expf(-g));
          const size_t o = static_cast<size_t>(r) * a.act_ld + f;
          if (a.act_lo != nullptr) {
            split_bf16(sg * u, a.act[o], a.act_lo[o]);
          } else {
            a.act[o] = __float2bfloat16_rn(sg * u);
          }
        }
      }
    }
  } else {  // EPI_QKV: RoPE on q and k, K/V appended to the cache
    const int f = rt * kTileM + et;
    const int hd = a.head_dim, half = hd >> 1;
    int seg, fs;
    if (f < a.q_dim) {
      seg = 0;
      fs = f;
    } else if (f < a.q_dim + a.kv_dim) {
      seg = 1;
      fs = f - a.q_dim;
    } else {
      seg = 2;
      fs = f - a.q_dim - a.kv_dim;
    }
    const int head = fs / hd, d = fs - head * hd;
    const int ip = d < half ? d : d - half;   // rotation pair index
    const int e1 = et - d + ip;               // staging index of element ip of this head
#pragma unroll 1
    for (int j = 0; j < 16; ++j) {
      const int r = chunk * 16 + j;
      if (!row_valid(a, r)) continue;
      const int g = r / a.plan->rows_per_group;
      const int i = r - g * a.plan->rows_per_group;
      const int pos = a.plan->pos0[g] + i;
      if (pos < 0 || pos >= a.max_seq) continue;   // flagged by the embedding kernel
      float val = stage[et * kStagePitch + j];
      if (seg < 2) {
        const float x1 = stage[e1 * kStagePitch + j];
        const float x2 = stage[(e1 + half) * kStagePitch + j];
        const float c = a.rope_cos[static_cast<size_t>(pos) * half + ip];
        const float s = a.rope_sin[static_cast<size_t>(pos) * half + ip];
        val = d < half ? (x1 * c - x2 * s) : (x1 * s + x2 * c);
      }
      if (seg == 0) {
        a.q_out[static_cast<size_t>(r) * a.q_dim + f] = val;
      } else {
        const int req = a.plan->req[g];
        const size_t off =
            ((static_cast<size_t>(req) * a.n_kv_heads + head) * a.max_seq + pos) * hd + d;
        (seg == 1 ? a.kcache : a.vcache)[off] = __float2bfloat16_rn(val);
      }
    }
  }
  named_bar_sync(1, 128);  // staging buffer is reused by the next chunk
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

// Epilogue of one accumulated segment [k0, k1) of row tile rt, run by the 128
// epilogue threads (et = TMEM lane = tile feature).  `c` is this CTA's index and
// G the op's grid; T = row_tiles * k_tiles.  The caller has waited for the
// accumulator; this routine reads it (wide layout: adds the hi and lo halves),
// releases it via acc_empty, and writes the epilogue or a partial.
__device__ __forceinline__ void epilogue_segment(const GemmArgs& a, int layout, int acols,
                                                 uint32_t tmem_base, int buf, int seg, int c,
                                                 int G, int rt, int k0, int k1, float* stage,
                                                 const float* rms, float (*red)[16],
                                                 int* reduce_flag, uint64_t* acc_empty, int et,
                                                 int ew, int lane) {
  const int KT = a.k_tiles;
  const int T = a.row_tiles * KT;
  const bool full = (k0 == 0 && k1 == KT);
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
      apply_epilogue(a, red, stage, rms, rt, chunk, et, v);
    }
  } else {
    // partial sums, feature-major: thread et owns n_pad consecutive floats
    const int slot = (seg == 0) ? 0 : 1;
    float* pb = a.partials + static_cast<size_t>(2 * c + slot) * a.n_pad * kTileM +
                static_cast<size_t>(et) * a.n_pad;
    for (int chunk = 0; chunk < a.n_pad / 16; ++chunk) {
      load_chunk(chunk);
      float4* dst = reinterpret_cast<float4*>(pb + chunk * 16);
#pragma unroll
      for (int q = 0; q < 4; ++q) dst[q] = make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
    }
  }
  tc_fence_before();
  __syncwarp();
  if (lane == 0) mbar_arrive(&acc_empty[buf]);
  if (full) return;
  __threadfence();
  named_bar_sync(1, 128);
  const int c_first = sk_cta_of(rt * KT, T, G);
  const int c_last = sk_cta_of((rt + 1) * KT - 1, T, G);
  if (et == 0) {
    const int old = atomicAdd(&a.counters[rt], 1);
    *reduce_flag = (old == c_last - c_first) ? 1 : 0;
  }
  named_bar_sync(1, 128);
  if (!*reduce_flag) return;
  __threadfence();
  for (int chunk = 0; chunk < a.n_pad / 16; ++chunk) {
#pragma unroll
    for (int j = 0; j < 16; ++j) v[j] = 0.f;
    // contributors are summed in ascending CTA order; four are fetched at once
    for (int cc0 = c_first; cc0 <= c_last; cc0 += 4) {
      float4 tmp[4][4];
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const int cc = cc0 + q;
        if (cc <= c_last) {
          const int sl = (sk_begin(cc, T, G) >= rt * KT) ? 0 : 1;
          const float* pp = a.partials + static_cast<size_t>(2 * cc + sl) * a.n_pad * kTileM +
                            static_cast<size_t>(et) * a.n_pad + chunk * 16;
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
    apply_epilogue(a, red, stage, rms, rt, chunk, et, v);
  }
  if (et == 0) a.counters[rt] = 0;
}

}  // namespace gemm
}  // namespace memspec
