// embed_body.cuh - row plan + token-embedding gather that starts every forward
// pass (see embed.cu), shared by the embedding kernel and the pass kernel.
#pragma once
#include "internal.h"
#include "ptx.cuh"

namespace memspec {
namespace emb {

static __device__ void compute_group(const EmbedArgs& a, int g, int* req, int* valid, int* pos0) {
  if (a.mode == PLAN_PREFILL) {
    *req = a.prefill_req;
    *valid = a.prefill_count;
    *pos0 = a.prefill_start;
    return;
  }
  *req = g;
  const int L = a.seq_state[g * kStateInts + 0];
  if (a.mode == PLAN_VERIFY || a.mode == PLAN_TREE) {
    *valid = a.R;
    *pos0 = L - 1;
  } else if (a.mode == PLAN_DRAFT_FIRST) {
    const int ld = a.draft_len[g];
    int n = L - ld;
    if (n < 1 || n > a.R) {
      atomicOr(a.status, 0x4u);  // draft cache not caught up with the committed tokens
      n = n < 1 ? 1 : a.R;
    }
    *valid = n;
    *pos0 = L - n;
  } else {  // PLAN_DRAFT_NEXT
    *valid = 1;
    *pos0 = L + a.j - 2;
  }
}

static __device__ int row_token(const EmbedArgs& a, int req, int pos, int i) {
  const int L = a.mode == PLAN_PREFILL ? 0 : a.seq_state[req * kStateInts + 0];
  if (a.mode == PLAN_VERIFY) {
    return i == 0 ? a.tokens[static_cast<size_t>(req) * a.max_seq + L - 1]
                  : a.draft_tokens[req * a.max_k + i - 1];
  }
  if (a.mode == PLAN_TREE) return i == 0 ? a.tokens[static_cast<size_t>(req) * a.max_seq + L - 1] : a.tree->tokens[i];
  if (a.mode == PLAN_DRAFT_NEXT) return a.draft_tokens[req * a.max_k + a.j - 2];
  return a.tokens[static_cast<size_t>(req) * a.max_seq + pos];
}

// Row r of the pass (one block of NT threads; `sync` is a barrier over them):
// the plan (written by the block of row 0), the embedding row, bf16(h * gain)
// in hi + lo planes and the row's sum of squares.
template <int NT, class Sync>
__device__ void embed_row(const EmbedArgs& a, int r, float* red, int tid, Sync sync) {
  const int g = r / a.R, i = r - g * a.R;
  int req, valid, pos0;
  compute_group(a, g, &req, &valid, &pos0);
  if (r == 0 && tid < a.n_groups) {
    int rq, vl, p0;
    compute_group(a, tid, &rq, &vl, &p0);
    a.plan->req[tid] = rq;
    a.plan->valid[tid] = vl;
    a.plan->pos0[tid] = p0;
  }
  if (r == 0 && tid < kTreeRows) {   // tree passes: per-row RoPE offsets and visibility
    const bool tr = a.mode == PLAN_TREE;
    a.plan->rope_off[tid] = tr ? a.tree->rope_off[tid] : tid;
    a.plan->anc[tid] = tr ? a.tree->anc[tid] : 0u;
  }
  if (r == 0 && tid == 0) {
    a.plan->tree = a.mode == PLAN_TREE ? 1 : 0;
    a.plan->n_groups = a.n_groups;
    a.plan->rows_per_group = a.R;
    a.plan->rows_total = a.n_groups * a.R;
    int mp = 0;
    for (int gg = 0; gg < a.n_groups; ++gg) {
      int rq, vl, p0;
      compute_group(a, gg, &rq, &vl, &p0);
      mp = max(mp, p0 + vl - 1);
    }
    a.plan->max_pos = mp;
  }
  float* hr = a.h + static_cast<size_t>(r) * a.d;
  float sq = 0.f;
  const bool ok = i < valid;
  int tok = 0;
  if (ok) {
    const int pos = pos0 + i;
    if (pos < 0 || pos >= a.max_seq) {
      if (tid == 0) atomicOr(a.status, 0x4u);
    } else {
      tok = row_token(a, req, pos, i);
    }
    if (tok < 0 || tok >= a.vocab) {
      if (tid == 0) atomicOr(a.status, 0x2u);
      tok = 0;
    }
  }
  const bf16* er = a.emb + static_cast<size_t>(tok) * a.d;
  for (int c = tid * 8; c < a.d; c += NT * 8) {
    float f[8];
    if (ok) {
      const uint4 raw = *reinterpret_cast<const uint4*>(er + c);
      const __nv_bfloat16* b = reinterpret_cast<const __nv_bfloat16*>(&raw);
#pragma unroll
      for (int q = 0; q < 8; ++q) f[q] = __bfloat162float(b[q]);
    } else {
#pragma unroll
      for (int q = 0; q < 8; ++q) f[q] = 0.f;
    }
#pragma unroll
    for (int q = 0; q < 8; ++q) sq += f[q] * f[q];
    reinterpret_cast<float4*>(hr + c)[0] = make_float4(f[0], f[1], f[2], f[3]);
    reinterpret_cast<float4*>(hr + c)[1] = make_float4(f[4], f[5], f[6], f[7]);
    // bf16(h * gain): the first projection's input, its RMSNorm scale applied
    // per row in that projection's epilogue
    const uint4 graw = *reinterpret_cast<const uint4*>(a.gain + c);
    const __nv_bfloat16* gb = reinterpret_cast<const __nv_bfloat16*>(&graw);
    __nv_bfloat16 o8[8];
#pragma unroll
    for (int q = 0; q < 8; ++q) o8[q] = __float2bfloat16_rn(f[q] * __bfloat162float(gb[q]));
    *reinterpret_cast<uint4*>(a.xg + static_cast<size_t>(r) * a.d + c) =
        *reinterpret_cast<const uint4*>(o8);
    if (a.xg_lo != nullptr) {   // low-order plane: bf16(x - bf16(x))
      __nv_bfloat16 l8[8];
#pragma unroll
      for (int q = 0; q < 8; ++q)
        l8[q] = __float2bfloat16_rn(f[q] * __bfloat162float(gb[q]) - __bfloat162float(o8[q]));
      *reinterpret_cast<uint4*>(a.xg_lo + static_cast<size_t>(r) * a.d + c) =
          *reinterpret_cast<const uint4*>(l8);
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) sq += __shfl_xor_sync(0xffffffffu, sq, o);
  if ((tid & 31) == 0) red[tid >> 5] = sq;
  sync();
  if (tid == 0) {
    float s = 0.f;
    for (int w = 0; w < NT / 32; ++w) s += red[w];
    a.ss[r] = s;
  }
  sync();   // red is reused by the next row
}


}  // namespace emb
}  // namespace memspec
