// attn_body.cuh - split-KV attention CTA body, shared by the attention kernel and
// the persistent pass kernel (see attention.cu for the algorithm).
#pragma once
#include "internal.h"
#include "ptx.cuh"

namespace memspec {
namespace attn {

constexpr int kAttThreads = 128;
constexpr int kKeyTile = 64;
constexpr int kStages = 3;
constexpr int kMaxQ = 64;   // query vectors per CTA (4 m-tiles of 16)

__device__ __forceinline__ void cp_async16_zfill(void* smem_dst, const void* gsrc, bool valid) {
  const int n = valid ? 16 : 0;
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(smem_addr(smem_dst)),
               "l"(gsrc), "r"(n)
               : "memory");
}
__device__ __forceinline__ void cp_async_commit() {
  asm volatile("cp.async.commit_group;" ::: "memory");
}
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                        uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                          uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}
__device__ __forceinline__ void mma16816(float* c, const uint32_t* a, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, "
      "{%4, %5, %6, %7}, {%8, %9}, {%0, %1, %2, %3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}
__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  __nv_bfloat162 t = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&t);
}

// Byte offset of 16-byte chunk `ch` of row `row` in a [64 rows][HD] bf16 tile:
// 64-column halves one after the other, each [64 rows][128 bytes] with chunk c
// of row r at c ^ (r % 8) - the layout a TMA box {64, 64} with the 128-byte
// swizzle writes (and the cp.async path mirrors).
template <int HD>
__device__ __forceinline__ uint32_t swz(int row, int ch) {
  return static_cast<uint32_t>((ch >> 3) * (kKeyTile * 128) + row * 128 + (((ch & 7) ^ (row & 7)) << 4));
}

template <int HD>
__host__ __device__ constexpr size_t attention_body_bytes() {
  // kStages x (K tile + V tile); the merge buffers (o, (m, l), weights, (M, L)) reuse it
  return static_cast<size_t>(kStages) * 2 * kKeyTile * HD * 2 >
                 static_cast<size_t>(4) * 16 * HD * 4 + 4 * 16 * 2 * 4 + kMaxQ * 6 * 4
             ? static_cast<size_t>(kStages) * 2 * kKeyTile * HD * 2
             : static_cast<size_t>(4) * 16 * HD * 4 + 4 * 16 * 2 * 4 + kMaxQ * 6 * 4;
}
// + up to 1008 bytes to align the stages to 1024 (the swizzle's period), + a
// 16-byte flag at the end
template <int HD>
__host__ __device__ constexpr size_t attention_smem_bytes_hd() {
  return 1008 + attention_body_bytes<HD>() + 16;
}

// One CTA of split-KV attention for unit (g, kvh, rb, split), run by 128 threads
// (tid 0..127); `sync` is a barrier over exactly those threads; smem_raw is the
// CTA's attention shared memory (attention_smem_bytes).  Returns early, all
// threads together, when the unit has no work.
// dry: a run of the same code on one synthetic tile that reads only scratch and
// writes no global memory (no output, no partials, no counters): launched
// before griddepcontrol.wait, it brings this code into the instruction cache
// while the previous kernel finishes.  Callers pass g = kvh = rb = split = 0.
// wait: called once by every thread before the first read of the previous
// kernel's output (the kernel passes griddepcontrol.wait).  early: the row plan
// and the cached keys / values before the group's first new position are final
// before wait() (see AttnArgs::ctx_early): the plan is read, and the first tiles
// that hold only such keys are requested, before it.
// bars: kStages mbarriers (count 1) for the TMA path (a.tma, not dry), else nullptr.
template <int HD, class Sync, class Wait>
__device__ __forceinline__ void attention_cta(const AttnArgs& a, int g, int kvh, int rb, int split,
                                              uint8_t* smem_raw, int tid, Sync sync, Wait wait,
                                              bool early, unsigned long long* ts = nullptr,
                                              bool dry = false, uint64_t* bars = nullptr) {
  constexpr int kChunks = HD / 8;                        // 16-byte chunks per row
  constexpr int kTileBytes = kKeyTile * HD * 2;          // one K (or V) tile
  constexpr int kNT = HD / 8;                            // n8 tiles of the output
  if (!early) wait();
  const RowPlan* plan = a.plan;
  // every plan field in one round trip (g < kMaxGroups: in bounds before the check)
  int n_groups = 1, R = a.rows_per_block, req = 0, valid = a.rows_per_block, pos0 = 0, tree = 0;
  if (!dry) {
    n_groups = plan->n_groups;
    R = plan->rows_per_group;
    req = plan->req[g];
    valid = plan->valid[g];
    pos0 = plan->pos0[g];
    tree = plan->tree;
  }
  if (g >= n_groups) return;
  const int r_lo = rb * a.rows_per_block;
  const int r_hi = min(r_lo + a.rows_per_block, valid);
  if (r_lo >= r_hi) return;
  const int nr = r_hi - r_lo;
  const int gs = a.H / a.Hkv;
  const int nq = gs * nr;
  const int kmax = pos0 + r_hi - 1;
  if (pos0 < 0 || kmax >= a.max_seq || nq > kMaxQ || a.n_splits > 16) {   // reported, never read
    if (threadIdx.x == 0 && split == 0) atomicOr(a.status, 0x4u);
    return;
  }
  const int n_active = (kmax + a.chunk) / a.chunk;   // ceil((kmax + 1) / chunk)
  if (split >= n_active) return;
  const int k0 = split * a.chunk;
  const int k1 = min(k0 + a.chunk, kmax + 1);
  const int n_tiles = (k1 - k0 + kKeyTile - 1) / kKeyTile;

  const int n_mt = (nq + 15) >> 4;
  const int kg = n_mt == 1 ? 4 : (n_mt == 2 ? 2 : 1);    // warps per m-tile (key groups)
  const int warp = tid >> 5, lane = tid & 31;
  const int mt = warp / kg, kgi = warp - mt * kg;
  const bool active = mt < n_mt;

  // kStages x (K tile, V tile), 1024-byte aligned
  uint8_t* kv = smem_raw + ((1024u - (smem_addr(smem_raw) & 1023u)) & 1023u);
  const bool tma = bars != nullptr && !dry;
  int* flag = reinterpret_cast<int*>(smem_raw + attention_smem_bytes_hd<HD>() - 16);
  // Q (hi and lo planes, [64][HD] bf16 each, swizzled) is staged in the last
  // pipeline stage, which the prologue leaves empty; the fragments move to
  // registers before that stage is first filled.
  uint8_t* qs = kv + (kStages - 1) * 2 * kTileBytes;
  const size_t kv_base = (static_cast<size_t>(req) * a.Hkv + kvh) * a.max_seq;
  const bf16* kc = a.kcache + kv_base * HD;
  const bf16* vc = a.vcache + kv_base * HD;

  const int kv_row0 = (req * a.Hkv + kvh) * a.max_seq;   // first row of this head in the maps
  auto load_tile = [&](int t) {
    uint8_t* ks = kv + (t % kStages) * 2 * kTileBytes;
    uint8_t* vs = ks + kTileBytes;
    const int kt0 = k0 + t * kKeyTile;
    if (tma) {   // one thread: the K and V boxes of the tile (rows past k1 are masked / zeroed later)
      if (tid == 0) {
        uint64_t* bar = &bars[t % kStages];
        const uint64_t pol = l2_policy_evict_first();
        mbar_arrive_expect_tx(bar, 2u * kTileBytes);
#pragma unroll
        for (int hf = 0; hf < HD / 64; ++hf) {
          tma_load_2d(ks + hf * kKeyTile * 128, &a.kmap, hf * 64, kv_row0 + kt0, bar, pol);
          tma_load_2d(vs + hf * kKeyTile * 128, &a.vmap, hf * 64, kv_row0 + kt0, bar, pol);
        }
      }
      return;
    }
    for (int c = tid; c < kKeyTile * kChunks; c += kAttThreads) {
      const int row = c / kChunks, ch = c - row * kChunks;
      const bool ok = kt0 + row < k1 && !dry;   // dry: zero-fill, no global read
      const size_t off = ok ? static_cast<size_t>(kt0 + row) * HD + ch * 8 : 0;
      cp_async16_zfill(ks + swz<HD>(row, ch), kc + off, ok);
      cp_async16_zfill(vs + swz<HD>(row, ch), vc + off, ok);
    }
  };

  // prologue: start the first kStages-1 tiles (early: those below pos0 before the
  // wait), then stage Q (fp32 -> bf16, scaled)
  int s_pre = 0;
  if (early) {
    for (; s_pre < kStages - 1 && s_pre < n_tiles && k0 + (s_pre + 1) * kKeyTile <= pos0; ++s_pre) {
      load_tile(s_pre);
      cp_async_commit();
    }
    wait();
  }
  for (int s = s_pre; s < kStages - 1; ++s) {
    if (s < n_tiles) load_tile(s);
    cp_async_commit();
  }
  for (int c = tid; c < kMaxQ * kChunks; c += kAttThreads) {
    const int v = c / kChunks, ch = c - v * kChunks;
    __nv_bfloat16 e[8], el[8];
    if (v < nq && !dry) {
      const int hl = v / nr, rr = v - hl * nr;
      const int row = g * R + r_lo + rr;
      const int h = kvh * gs + hl;
      const float* src = a.q + (static_cast<size_t>(row) * a.H + h) * HD + ch * 8;
      const float4 x0 = *reinterpret_cast<const float4*>(src);
      const float4 x1 = *reinterpret_cast<const float4*>(src + 4);
      const float f[8] = {x0.x, x0.y, x0.z, x0.w, x1.x, x1.y, x1.z, x1.w};
#pragma unroll
      for (int i = 0; i < 8; ++i) split_bf16(f[i] * a.scale_log2, e[i], el[i]);
    } else {
#pragma unroll
      for (int i = 0; i < 8; ++i) e[i] = el[i] = __float2bfloat16_rn(0.f);
    }
    *reinterpret_cast<uint4*>(qs + swz<HD>(v, ch)) = *reinterpret_cast<const uint4*>(e);
    *reinterpret_cast<uint4*>(qs + kTileBytes + swz<HD>(v, ch)) = *reinterpret_cast<const uint4*>(el);
  }
  sync();
  trace_at(ts, 8);

  // Q fragments (hi and lo) of this warp's m-tile stay in registers
  uint32_t qa[HD / 16][4], ql[HD / 16][4];
  if (active) {
#pragma unroll
    for (int ks = 0; ks < HD / 16; ++ks) {
      const int row = mt * 16 + (lane & 15);
      const int ch = ks * 2 + (lane >> 4);
      ldsm_x4(smem_addr(qs) + swz<HD>(row, ch), qa[ks][0], qa[ks][1], qa[ks][2], qa[ks][3]);
      ldsm_x4(smem_addr(qs + kTileBytes) + swz<HD>(row, ch), ql[ks][0], ql[ks][1], ql[ks][2],
              ql[ks][3]);
    }
  }
  // positions of this thread's two rows (v = mt*16 + lane/4 and +8); -1: padding row
  // tree passes: beyond pos0 a row sees only the rows in its ancestor mask
  int prow[2];
  uint32_t amask[2] = {0u, 0u};
#pragma unroll
  for (int h2 = 0; h2 < 2; ++h2) {
    const int v = mt * 16 + (lane >> 2) + 8 * h2;
    prow[h2] = (active && v < nq) ? pos0 + r_lo + (v % nr) : -1;
    if (tree && prow[h2] >= 0 && r_lo + (v % nr) < kTreeRows) amask[h2] = plan->anc[r_lo + (v % nr)];
  }
  float m_run[2] = {-INFINITY, -INFINITY}, l_run[2] = {0.f, 0.f};
  float o[kNT][4];
#pragma unroll
  for (int i = 0; i < kNT; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.f;

  const int sub_per_warp = (kKeyTile / 16) / kg;          // 16-key sub-blocks per warp per tile
  int waited = 0;   // TMA: tiles whose stage completion was observed
  for (int t = 0; t < n_tiles; ++t) {
    if (tma) {
      // one thread waits (bounded); all follow its outcome
      if (tid == 0)
        *flag = mbar_wait_bounded(&bars[t % kStages], static_cast<uint32_t>(t / kStages) & 1u, nullptr, a.status)
                    ? 1
                    : 0;
      sync();
      if (!*flag) break;
      waited = t + 1;
      const int nk = min(kKeyTile, k1 - (k0 + t * kKeyTile));
      if (nk < kKeyTile) {   // V rows past the split's end hold other positions (or garbage): zero them
        uint8_t* vs = kv + (t % kStages) * 2 * kTileBytes + kTileBytes;
        for (int c = tid; c < (kKeyTile - nk) * kChunks; c += kAttThreads) {
          const int row = nk + c / kChunks, ch = c % kChunks;
          *reinterpret_cast<uint4*>(vs + swz<HD>(row, ch)) = make_uint4(0u, 0u, 0u, 0u);
        }
        sync();
      }
      // the stage refilled next was last read (ldmatrix, generic proxy) before the barrier above
      if (tid == 0) fence_proxy_async_smem();
    } else {
      cp_async_wait<kStages - 2>();
      sync();
    }
    if (t == 0) trace_at(ts, 10);
    if (t + kStages - 1 < n_tiles) load_tile(t + kStages - 1);
    cp_async_commit();
    if (!active) continue;
    const uint32_t ks_addr = smem_addr(kv + (t % kStages) * 2 * kTileBytes);
    const uint32_t vs_addr = ks_addr + kTileBytes;
    const int kt0 = k0 + t * kKeyTile;
    for (int sb = 0; sb < sub_per_warp; ++sb) {
      const int kb = (kgi * sub_per_warp + sb) * 16;      // key offset within the tile
      float s0[4] = {0.f, 0.f, 0.f, 0.f}, s1[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
      for (int ks = 0; ks < HD / 16; ++ks) {
        uint32_t b0, b1, b2, b3;
        const int row = kb + (lane & 7) + ((lane >> 4) << 3);
        const int ch = ks * 2 + ((lane >> 3) & 1);
        ldsm_x4(ks_addr + swz<HD>(row, ch), b0, b1, b2, b3);
        mma16816(s0, qa[ks], b0, b1);
        mma16816(s0, ql[ks], b0, b1);
        mma16816(s1, qa[ks], b2, b3);
        mma16816(s1, ql[ks], b2, b3);
      }
      // causal / range mask, then online softmax (base 2)
      const int key_c = kt0 + kb + ((lane & 3) << 1);
      float mx[2];
#pragma unroll
      for (int h2 = 0; h2 < 2; ++h2) {
        const int p = prow[h2];
        const int lim = min(p, k1 - 1);
        const uint32_t am = amask[h2];
        // key visible: causal (and in this split) and, in a tree pass, below
        // pos0 or an ancestor row (rows past 31 never appear in a tree pass)
        auto vis = [&](int key) {
          if (key > lim) return false;
          if (!tree) return true;
          const int rel = key - pos0;
          return rel < 0 || (rel < kTreeRows && ((am >> rel) & 1u) != 0u);
        };
        float* a0 = s0 + 2 * h2;
        float* a1 = s1 + 2 * h2;
        a0[0] = vis(key_c) ? a0[0] : -INFINITY;
        a0[1] = vis(key_c + 1) ? a0[1] : -INFINITY;
        a1[0] = vis(key_c + 8) ? a1[0] : -INFINITY;
        a1[1] = vis(key_c + 9) ? a1[1] : -INFINITY;
        mx[h2] = fmaxf(fmaxf(a0[0], a0[1]), fmaxf(a1[0], a1[1]));
        mx[h2] = fmaxf(mx[h2], __shfl_xor_sync(0xffffffffu, mx[h2], 1));
        mx[h2] = fmaxf(mx[h2], __shfl_xor_sync(0xffffffffu, mx[h2], 2));
      }
      float scale[2];
#pragma unroll
      for (int h2 = 0; h2 < 2; ++h2) {
        const float m_new = fmaxf(m_run[h2], mx[h2]);
        float* a0 = s0 + 2 * h2;
        float* a1 = s1 + 2 * h2;
        if (m_new == -INFINITY) {
          scale[h2] = 1.f;
          a0[0] = a0[1] = a1[0] = a1[1] = 0.f;
        } else {
          scale[h2] = exp2f(m_run[h2] - m_new);
          a0[0] = exp2f(a0[0] - m_new);
          a0[1] = exp2f(a0[1] - m_new);
          a1[0] = exp2f(a1[0] - m_new);
          a1[1] = exp2f(a1[1] - m_new);
        }
        float rs = (a0[0] + a0[1]) + (a1[0] + a1[1]);
        rs += __shfl_xor_sync(0xffffffffu, rs, 1);
        rs += __shfl_xor_sync(0xffffffffu, rs, 2);
        l_run[h2] = l_run[h2] * scale[h2] + rs;
        m_run[h2] = m_new;
      }
#pragma unroll
      for (int i = 0; i < kNT; ++i) {
        o[i][0] *= scale[0];
        o[i][1] *= scale[0];
        o[i][2] *= scale[1];
        o[i][3] *= scale[1];
      }
      // P as hi + lo bf16 fragments
      uint32_t pa[4], pl[4];
      {
        const float pv[8] = {s0[0], s0[1], s0[2], s0[3], s1[0], s1[1], s1[2], s1[3]};
        float lo[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) lo[i] = pv[i] - __bfloat162float(__float2bfloat16_rn(pv[i]));
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          pa[i] = pack_bf16x2(pv[2 * i], pv[2 * i + 1]);
          pl[i] = pack_bf16x2(lo[2 * i], lo[2 * i + 1]);
        }
      }
#pragma unroll
      for (int n2 = 0; n2 < HD / 16; ++n2) {
        uint32_t b0, b1, b2, b3;
        const int row = kb + (lane & 7) + (((lane >> 3) & 1) << 3);
        const int ch = n2 * 2 + (lane >> 4);
        ldsm_x4_t(vs_addr + swz<HD>(row, ch), b0, b1, b2, b3);
        mma16816(o[2 * n2], pa, b0, b1);
        mma16816(o[2 * n2], pl, b0, b1);
        mma16816(o[2 * n2 + 1], pa, b2, b3);
        mma16816(o[2 * n2 + 1], pl, b2, b3);
      }
    }
  }
  cp_async_wait<0>();
  if (tma && waited < n_tiles) {   // a wait ran out: let the copies still in flight land, then stop
    if (tid == 0)
      for (int t = waited; t < min(n_tiles, waited + kStages); ++t)
        mbar_wait_drain(&bars[t % kStages], static_cast<uint32_t>(t / kStages) & 1u);
    sync();
    return;
  }
  sync();
  trace_at(ts, 9);
  if (ts != nullptr) trace_after(ts, 12, o[0][0] + o[kNT - 1][3]);   // last MMAs retired

  // merge the key groups of each m-tile (shared memory reuses the K/V stages):
  // the query vectors' rows of o go to shared memory (padding rows are not
  // written or read), one thread per vector computes M = max_w m_w, the group
  // weights f_w = 2^(m_w - M) and L = sum_w f_w l_w, then four features per
  // thread: o = sum_w f_w o_w (groups in ascending order)
  float* mo = reinterpret_cast<float*>(kv);                 // [4 warps][16][HD]
  float* ml = mo + 4 * 16 * HD;                             // [4 warps][16][2]
  float* mf = ml + 4 * 16 * 2;                              // [kMaxQ][4] weights
  float* mml = mf + kMaxQ * 4;                              // [kMaxQ][2] M, L
  if (active) {
    const int r0 = lane >> 2, cc = (lane & 3) << 1;
    const bool lo_ok = mt * 16 + r0 < nq, hi_ok = mt * 16 + r0 + 8 < nq;
#pragma unroll
    for (int i = 0; i < kNT; ++i) {
      float* dst = mo + (warp * 16) * HD + i * 8 + cc;
      if (lo_ok) *reinterpret_cast<float2*>(dst + r0 * HD) = make_float2(o[i][0], o[i][1]);
      if (hi_ok) *reinterpret_cast<float2*>(dst + (r0 + 8) * HD) = make_float2(o[i][2], o[i][3]);
    }
    if ((lane & 3) == 0) {
      ml[(warp * 16 + r0) * 2] = m_run[0];
      ml[(warp * 16 + r0) * 2 + 1] = l_run[0];
      ml[(warp * 16 + r0 + 8) * 2] = m_run[1];
      ml[(warp * 16 + r0 + 8) * 2 + 1] = l_run[1];
    }
  }
  sync();
  for (int v = tid; v < nq; v += kAttThreads) {
    const int m_t = v >> 4, r = v & 15;
    float M = -INFINITY;
    for (int w = 0; w < kg; ++w) M = fmaxf(M, ml[((m_t * kg + w) * 16 + r) * 2]);
    float L = 0.f;
    for (int w = 0; w < kg; ++w) {
      const int ww = m_t * kg + w;
      const float mw = ml[(ww * 16 + r) * 2];
      const float f = mw == -INFINITY ? 0.f : exp2f(mw - M);
      mf[v * 4 + w] = f;
      L += f * ml[(ww * 16 + r) * 2 + 1];
    }
    mml[v * 2] = M;
    mml[v * 2 + 1] = L;
  }
  sync();
  trace_at(ts, 11);
  const int unit = (g * a.Hkv + kvh) * a.row_blocks + rb;
  const size_t pbase = (static_cast<size_t>(unit) * a.n_splits + split) * a.qmax;
  constexpr int kMV4 = HD / 4;
  for (int idx = tid; idx < nq * kMV4; idx += kAttThreads) {
    const int v = idx / kMV4, d = (idx - v * kMV4) * 4;
    const int m_t = v >> 4, r = v & 15;
    float4 O = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int w = 0; w < kg; ++w) {
      const float f = mf[v * 4 + w];
      const float4 x = *reinterpret_cast<const float4*>(mo + ((m_t * kg + w) * 16 + r) * HD + d);
      O.x += f * x.x;
      O.y += f * x.y;
      O.z += f * x.z;
      O.w += f * x.w;
    }
    if (dry) continue;
    *reinterpret_cast<float4*>(a.part_o + (pbase + v) * HD + d) = O;
    if (d == 0) *reinterpret_cast<float2*>(a.part_ml + (pbase + v) * 2) = *reinterpret_cast<const float2*>(mml + v * 2);
  }
  trace_at(ts, 4);
  // same arrival protocol as the GEMM split-K: the barrier orders this CTA's
  // partial stores before thread 0's acq_rel arrival; the last split's acquire
  // and the next barrier order every split's partials before its loads
  sync();
  int* last = flag;
  if (tid == 0)
    *last = dry ? 1 : ((atom_add_acq_rel_gpu(&a.counters[unit], 1) == n_active - 1) ? 1 : 0);
  sync();
  trace_at(ts, 5);
  if (!*last) return;
  const size_t ubase = static_cast<size_t>(unit) * a.n_splits * a.qmax;
  const int qmax = a.qmax;
  const float* part_ml = a.part_ml;
  const float* part_o = a.part_o;
  // One round trip: each thread fetches, for its query vector v and its four
  // features, every split's (m_s, l_s) (the 32 threads of a vector read the same
  // words: one transaction) together with its o_s (n_active <= 16: the geometry
  // caps the splits), then M = max m_s, weights 2^(m_s - M), L and the weighted
  // sum, all in ascending split order.
  constexpr int kV4 = HD / 4;
  bf16* out = a.out;
  bf16* out_lo = a.out_lo;
  const int H = a.H;
  for (int idx = tid; idx < nq * kV4; idx += kAttThreads) {
    const int v = idx / kV4, d = (idx - v * kV4) * 4;
    float2 mlv[16];
    float4 ov[16];
#pragma unroll
    for (int q = 0; q < 16; ++q) {
      if (q < n_active) {
        const size_t pv = ubase + static_cast<size_t>(q) * qmax + v;
        mlv[q] = ld_cg_f2(part_ml + pv * 2);
        ov[q] = ld_cg_f4(part_o + pv * HD + d);
      }
    }
    if (idx == tid) trace_after(ts, 6, mlv[0].x + ov[0].x);
    float M = -INFINITY;
#pragma unroll
    for (int q = 0; q < 16; ++q)
      if (q < n_active) M = fmaxf(M, mlv[q].x);
    float L = 0.f;
    float O[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
    for (int q = 0; q < 16; ++q) {
      if (q < n_active) {
        const float w = mlv[q].x == -INFINITY ? 0.f : exp2f(mlv[q].x - M);
        L += w * mlv[q].y;
        O[0] += w * ov[q].x;
        O[1] += w * ov[q].y;
        O[2] += w * ov[q].z;
        O[3] += w * ov[q].w;
      }
    }
    const float li = 1.f / L;
    const int hl = v / nr, rr = v - hl * nr;
    const int row = g * R + r_lo + rr;
    const int h = kvh * gs + hl;
    const size_t oi = (static_cast<size_t>(row) * H + h) * HD + d;
    if (dry) continue;
    // four features: one 8-byte store per plane (oi is a multiple of 4)
    __nv_bfloat16 hv[4], lv[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) split_bf16(O[e] * li, hv[e], lv[e]);
    *reinterpret_cast<uint2*>(out + oi) = *reinterpret_cast<const uint2*>(hv);
    if (out_lo != nullptr) *reinterpret_cast<uint2*>(out_lo + oi) = *reinterpret_cast<const uint2*>(lv);
  }
  trace_at(ts, 7);
  if (tid == 0 && !dry) a.counters[unit] = 0;
}


}  // namespace attn
}  // namespace memspec
