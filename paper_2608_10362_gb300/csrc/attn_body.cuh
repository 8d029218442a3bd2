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
// 8x8 b16 matrix held as the ldmatrix fragment (lane: row lane/4, columns
// 2(lane%4), +1) -> the same fragment of its transpose
__device__ __forceinline__ uint32_t movmatrix_trans(uint32_t x) {
  uint32_t y;
  asm volatile("movmatrix.sync.aligned.m8n8.trans.b16 %0, %1;" : "=r"(y) : "r"(x));
  return y;
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

// Pipeline stages: 3; the transposed form (at most 8 query vectors, three CTAs
// per SM) runs 2.
template <bool kTQ>
__host__ __device__ constexpr int attention_stages() {
  return kTQ ? 2 : kStages;
}

template <int HD, bool kTQ = false>
__host__ __device__ constexpr size_t attention_body_bytes() {
  // stages x (K tile + V tile); the merge buffers (o, (m, l), weights, (M, L)) reuse it
  return static_cast<size_t>(attention_stages<kTQ>()) * 2 * kKeyTile * HD * 2 >
                 static_cast<size_t>(4) * 16 * HD * 4 + 4 * 16 * 2 * 4 + kMaxQ * 6 * 4
             ? static_cast<size_t>(attention_stages<kTQ>()) * 2 * kKeyTile * HD * 2
             : static_cast<size_t>(4) * 16 * HD * 4 + 4 * 16 * 2 * 4 + kMaxQ * 6 * 4;
}
// + up to 1008 bytes to align the stages to 1024 (the swizzle's period), + a
// 16-byte flag at the end
template <int HD, bool kTQ = false>
__host__ __device__ constexpr size_t attention_smem_bytes_hd() {
  return 1008 + attention_body_bytes<HD, kTQ>() + 16;
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
// bars: attention_stages<kTQ>() mbarriers (count 1) for the TMA path (a.tma, not
// dry), else nullptr.
// kTQ: at most 8 query vectors (the launch's qmax <= 8; checked): the keys are the
// MMA's M side, S^T = K Q^T and O^T = V^T P^T with the queries as N = 8, half the
// MMAs, accumulator registers and rescaling work of the 16-row form.
template <int HD, bool kTQ = false, class Sync, class Wait>
__device__ __forceinline__ void attention_cta(const AttnArgs& a, int g, int kvh, int rb, int split,
                                              uint8_t* smem_raw, int tid, Sync sync, Wait wait,
                                              bool early, unsigned long long* ts = nullptr,
                                              bool dry = false, uint64_t* bars = nullptr) {
  constexpr int kChunks = HD / 8;                        // 16-byte chunks per row
  constexpr int kSt = attention_stages<kTQ>();           // pipeline stages
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
  if (pos0 < 0 || kmax >= a.max_seq || nq > (kTQ ? 8 : kMaxQ) || a.n_splits > 16) {   // reported, never read
    if (threadIdx.x == 0 && split == 0) atomicOr(a.status, 0x4u);
    return;
  }
  // the keys 0..kmax spread evenly over the launch's splits, whole 64-key tiles
  // each (a.chunk sizes the splits for max_seq; the context may be far shorter)
  const int chunk = ((kmax + a.n_splits) / a.n_splits + kKeyTile - 1) / kKeyTile * kKeyTile;
  const int n_active = (kmax + chunk) / chunk;   // ceil((kmax + 1) / chunk)
  if (split >= n_active) return;
  const int k0 = split * chunk;
  const int k1 = min(k0 + chunk, kmax + 1);
  const int n_tiles = (k1 - k0 + kKeyTile - 1) / kKeyTile;

  const int n_mt = (nq + 15) >> 4;
  const int kg = n_mt == 1 ? 4 : (n_mt == 2 ? 2 : 1);    // warps per m-tile (key groups)
  const int warp = tid >> 5, lane = tid & 31;
  const int mt = warp / kg, kgi = warp - mt * kg;
  const bool active = mt < n_mt;

  // kSt x (K tile, V tile), 1024-byte aligned
  uint8_t* kv = smem_raw + ((1024u - (smem_addr(smem_raw) & 1023u)) & 1023u);
  const bool tma = bars != nullptr && !dry;
  int* flag = reinterpret_cast<int*>(smem_raw + attention_smem_bytes_hd<HD, kTQ>() - 16);
  const size_t kv_base = (static_cast<size_t>(req) * a.Hkv + kvh) * a.max_seq;
  const bf16* kc = a.kcache + kv_base * HD;
  const bf16* vc = a.vcache + kv_base * HD;

  const int kv_row0 = (req * a.Hkv + kvh) * a.max_seq;   // first row of this head in the maps
  auto load_tile = [&](int t) {
    uint8_t* ks = kv + (t % kSt) * 2 * kTileBytes;
    uint8_t* vs = ks + kTileBytes;
    const int kt0 = k0 + t * kKeyTile;
    if (tma) {   // one thread: the K and V boxes of the tile (rows past k1 are masked / zeroed later)
      if (tid == 0) {
        uint64_t* bar = &bars[t % kSt];
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

  // prologue: the TMA path requests every stage (Q goes straight to registers),
  // the cp.async path the first kSt-1 tiles (one commit group per stage);
  // early: the tiles that hold only keys below pos0 go before the wait
  const int depth = tma ? kSt : kSt - 1;
  int s_pre = 0;
  if (early) {
    for (; s_pre < depth && s_pre < n_tiles && k0 + (s_pre + 1) * kKeyTile <= pos0; ++s_pre) {
      load_tile(s_pre);
      cp_async_commit();
    }
    wait();
  }
  for (int s = s_pre; s < depth; ++s) {
    if (s < n_tiles) load_tile(s);
    cp_async_commit();
  }
  int next = min(depth, n_tiles);   // tiles requested so far

  // Q fragments (hi and lo planes, pre-scaled), loaded from the fp32 rows
  // straight into registers.  16-row form: A operand of m16n8k16 for this
  // warp's m-tile, register j of k-step ks holds row lane/4 (+8 if j is odd) and
  // columns 2(lane%4), +1 (+8 if j >= 2).  kTQ: B operand, query lane/4, register
  // j of k-step ks holds columns 2(lane%4), +1 (+8 if j == 1).
  // Query vector v of the block is head v / nr of the group, row v % nr.
  auto q_row = [&](int v) {
    const int hl = v / nr, rr = v - hl * nr;
    return a.q + (static_cast<size_t>(g * R + r_lo + rr) * a.H + kvh * gs + hl) * HD + 2 * (lane & 3);
  };
  auto split2 = [&](float2 x, uint32_t& hi, uint32_t& lo) {
    __nv_bfloat16 h0, l0, h1, l1;
    split_bf16(x.x * a.scale_log2, h0, l0);
    split_bf16(x.y * a.scale_log2, h1, l1);
    hi = pack_bf16x2(__bfloat162float(h0), __bfloat162float(h1));
    lo = pack_bf16x2(__bfloat162float(l0), __bfloat162float(l1));
  };
  uint32_t qa[kTQ ? 1 : HD / 16][4], ql[kTQ ? 1 : HD / 16][4];
  uint32_t qb[kTQ ? HD / 16 : 1][2], qbl[kTQ ? HD / 16 : 1][2];
  if constexpr (kTQ) {
    const int v = lane >> 2;
    const float* src = (v < nq && !dry) ? q_row(v) : nullptr;
    float2 x[HD / 16][2];
#pragma unroll
    for (int ks = 0; ks < HD / 16; ++ks)
#pragma unroll
      for (int j = 0; j < 2; ++j)
        x[ks][j] = src != nullptr ? *reinterpret_cast<const float2*>(src + ks * 16 + j * 8) : make_float2(0.f, 0.f);
#pragma unroll
    for (int ks = 0; ks < HD / 16; ++ks)
#pragma unroll
      for (int j = 0; j < 2; ++j) split2(x[ks][j], qb[ks][j], qbl[ks][j]);
    if (ts != nullptr) trace_after(ts, 8, __uint_as_float(qb[0][0] ^ qbl[HD / 16 - 1][1]));
  } else {
    const float* qsrc[2] = {nullptr, nullptr};
#pragma unroll
    for (int h2 = 0; h2 < 2; ++h2) {
      const int v = mt * 16 + (lane >> 2) + 8 * h2;
      if (active && v < nq && !dry) qsrc[h2] = q_row(v);
    }
    float2 x[HD / 16][4];
#pragma unroll
    for (int ks = 0; ks < HD / 16; ++ks)
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const float* src = qsrc[j & 1];
        x[ks][j] = src != nullptr ? *reinterpret_cast<const float2*>(src + ks * 16 + (j >> 1) * 8)
                                  : make_float2(0.f, 0.f);
      }
#pragma unroll
    for (int ks = 0; ks < HD / 16; ++ks)
#pragma unroll
      for (int j = 0; j < 4; ++j) split2(x[ks][j], qa[ks][j], ql[ks][j]);
    if (ts != nullptr) trace_after(ts, 8, __uint_as_float(qa[0][0] ^ ql[HD / 16 - 1][3]));
  }
  // positions of this thread's two query vectors (16-row form: v = mt*16 +
  // lane/4 and +8; kTQ: v = 2(lane%4) and +1); -1: padding.  Tree passes:
  // beyond pos0 a vector sees only the rows in its ancestor mask
  int prow[2];
  uint32_t amask[2] = {0u, 0u};
#pragma unroll
  for (int h2 = 0; h2 < 2; ++h2) {
    const int v = kTQ ? 2 * (lane & 3) + h2 : mt * 16 + (lane >> 2) + 8 * h2;
    prow[h2] = (active && v < nq) ? pos0 + r_lo + (v % nr) : -1;
    if (tree && prow[h2] >= 0 && r_lo + (v % nr) < kTreeRows) amask[h2] = plan->anc[r_lo + (v % nr)];
  }
  float m_run[2] = {-INFINITY, -INFINITY}, l_run[2] = {0.f, 0.f};
  // output accumulators: 16-row form [n8 tile of features][4]; kTQ: [16-feature
  // block][4] of O^T (features lane/4 and +8, queries 2(lane%4) and +1)
  constexpr int kNO = kTQ ? HD / 16 : kNT;
  float o[kNO][4];
#pragma unroll
  for (int i = 0; i < kNO; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.f;

  const int sub_per_warp = (kKeyTile / 16) / kg;          // 16-key sub-blocks per warp per tile
  int waited = 0;   // TMA: tiles whose stage completion was observed
  for (int t = 0; t < n_tiles; ++t) {
    if (tma) {
      // one thread waits (bounded); all follow its outcome
      if (tid == 0)
        *flag = mbar_wait_bounded(&bars[t % kSt], static_cast<uint32_t>(t / kSt) & 1u, nullptr, a.status)
                    ? 1
                    : 0;
      sync();
      if (!*flag) break;
      waited = t + 1;
      const int nk = min(kKeyTile, k1 - (k0 + t * kKeyTile));
      if (nk < kKeyTile) {   // V rows past the split's end hold other positions (or garbage): zero them
        uint8_t* vs = kv + (t % kSt) * 2 * kTileBytes + kTileBytes;
        for (int c = tid; c < (kKeyTile - nk) * kChunks; c += kAttThreads) {
          const int row = nk + c / kChunks, ch = c % kChunks;
          *reinterpret_cast<uint4*>(vs + swz<HD>(row, ch)) = make_uint4(0u, 0u, 0u, 0u);
        }
        sync();
      }
      // the stage refilled next (tile t-1's) was last read (ldmatrix, generic
      // proxy) before the barrier above
      if (next < n_tiles && next < t + kSt) {
        if (tid == 0) fence_proxy_async_smem();
        load_tile(next);
        ++next;
      }
    } else {
      cp_async_wait<kSt - 2>();
      sync();
      if (t + kSt - 1 < n_tiles) load_tile(t + kSt - 1);
      cp_async_commit();
    }
    if (t == 0) trace_at(ts, 10);
    if (!active) continue;
    const uint32_t ks_addr = smem_addr(kv + (t % kSt) * 2 * kTileBytes);
    const uint32_t vs_addr = ks_addr + kTileBytes;
    const int kt0 = k0 + t * kKeyTile;
    if constexpr (kTQ) {
      for (int sb = 0; sb < sub_per_warp; ++sb) {
        const int kb = (kgi * sub_per_warp + sb) * 16;    // key offset within the tile
        // S^T (16 keys x 8 queries): A = K rows from the stage, B = Q; chains
        // per Q plane and (hd 128) k-step parity, summed at the end
        constexpr int kPar = HD >= 128 ? 2 : 1;
        float sp[2][kPar][4];
#pragma unroll
        for (int pl = 0; pl < 2; ++pl)
#pragma unroll
          for (int par = 0; par < kPar; ++par)
#pragma unroll
            for (int i = 0; i < 4; ++i) sp[pl][par][i] = 0.f;
#pragma unroll
        for (int ks = 0; ks < HD / 16; ++ks) {
          uint32_t ka[4];
          const int row = kb + (lane & 7) + (((lane >> 3) & 1) << 3);
          const int ch = ks * 2 + (lane >> 4);
          ldsm_x4(ks_addr + swz<HD>(row, ch), ka[0], ka[1], ka[2], ka[3]);
          const int par = ks % kPar;
          mma16816(sp[0][par], ka, qb[ks][0], qb[ks][1]);
          mma16816(sp[1][par], ka, qbl[ks][0], qbl[ks][1]);
        }
        // sc[0], sc[1]: key kb + lane/4, queries 2(lane%4) and +1; sc[2], sc[3]: key + 8
        float sc[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          if constexpr (kPar == 2)
            sc[i] = (sp[0][0][i] + sp[0][1][i]) + (sp[1][0][i] + sp[1][1][i]);
          else
            sc[i] = sp[0][0][i] + sp[1][0][i];
        }
        const int key_c = kt0 + kb + (lane >> 2);
        float mx[2];
#pragma unroll
        for (int h2 = 0; h2 < 2; ++h2) {
          const int p = prow[h2];
          const int lim = min(p, k1 - 1);
          const uint32_t am = amask[h2];
          auto vis = [&](int key) {
            if (key > lim) return false;
            if (!tree) return true;
            const int rel = key - pos0;
            return rel < 0 || (rel < kTreeRows && ((am >> rel) & 1u) != 0u);
          };
          sc[h2] = vis(key_c) ? sc[h2] : -INFINITY;
          sc[2 + h2] = vis(key_c + 8) ? sc[2 + h2] : -INFINITY;
          mx[h2] = fmaxf(sc[h2], sc[2 + h2]);
          mx[h2] = fmaxf(mx[h2], __shfl_xor_sync(0xffffffffu, mx[h2], 4));
          mx[h2] = fmaxf(mx[h2], __shfl_xor_sync(0xffffffffu, mx[h2], 8));
          mx[h2] = fmaxf(mx[h2], __shfl_xor_sync(0xffffffffu, mx[h2], 16));
        }
        float scale[2];
#pragma unroll
        for (int h2 = 0; h2 < 2; ++h2) {
          const float m_new = fmaxf(m_run[h2], mx[h2]);
          if (m_new == -INFINITY) {
            scale[h2] = 1.f;
            sc[h2] = sc[2 + h2] = 0.f;
          } else {
            scale[h2] = exp2f(m_run[h2] - m_new);
            sc[h2] = exp2f(sc[h2] - m_new);
            sc[2 + h2] = exp2f(sc[2 + h2] - m_new);
          }
          float rs = sc[h2] + sc[2 + h2];
          rs += __shfl_xor_sync(0xffffffffu, rs, 4);
          rs += __shfl_xor_sync(0xffffffffu, rs, 8);
          rs += __shfl_xor_sync(0xffffffffu, rs, 16);
          l_run[h2] = l_run[h2] * scale[h2] + rs;
          m_run[h2] = m_new;
        }
#pragma unroll
        for (int i = 0; i < kNO; ++i) {
          o[i][0] *= scale[0];
          o[i][1] *= scale[1];
          o[i][2] *= scale[0];
          o[i][3] *= scale[1];
        }
        // P^T as the B operand (keys x queries), hi + lo planes: the 8x8 blocks
        // [key][query] this lane holds (rows lane/4, columns 2(lane%4), +1) are
        // transposed across the warp, giving query lane/4, keys 2(lane%4), +1
        uint32_t pb[2], pbl[2];
#pragma unroll
        for (int hk = 0; hk < 2; ++hk) {
          const float x0 = sc[2 * hk], x1 = sc[2 * hk + 1];
          const float h0 = __bfloat162float(__float2bfloat16_rn(x0));
          const float h1 = __bfloat162float(__float2bfloat16_rn(x1));
          pb[hk] = movmatrix_trans(pack_bf16x2(x0, x1));
          pbl[hk] = movmatrix_trans(pack_bf16x2(x0 - h0, x1 - h1));
        }
        // O^T += V^T P^T: A = V^T (16 features x 16 keys) by transposing loads
#pragma unroll
        for (int i = 0; i < kNO; ++i) {
          uint32_t va[4];
          const int row = kb + (lane & 7) + ((lane >> 4) << 3);
          const int ch = i * 2 + ((lane >> 3) & 1);
          ldsm_x4_t(vs_addr + swz<HD>(row, ch), va[0], va[1], va[2], va[3]);
          mma16816(o[i], va, pb[0], pb[1]);
          mma16816(o[i], va, pbl[0], pbl[1]);
        }
      }
    } else {
      for (int sb = 0; sb < sub_per_warp; ++sb) {
        const int kb = (kgi * sub_per_warp + sb) * 16;      // key offset within the tile
        // independent accumulator chains (n8 tile x Q plane x, at hd 128, k-step
        // parity), summed at the end: one chain per n8 tile would serialise
        // 2 hd / 16 dependent MMAs per sub-block
        constexpr int kPar = HD >= 128 ? 2 : 1;
        float sp[2][2][kPar][4];
  #pragma unroll
        for (int n = 0; n < 2; ++n)
  #pragma unroll
          for (int pl = 0; pl < 2; ++pl)
  #pragma unroll
            for (int par = 0; par < kPar; ++par)
  #pragma unroll
              for (int i = 0; i < 4; ++i) sp[n][pl][par][i] = 0.f;
  #pragma unroll
        for (int ks = 0; ks < HD / 16; ++ks) {
          uint32_t b0, b1, b2, b3;
          const int row = kb + (lane & 7) + ((lane >> 4) << 3);
          const int ch = ks * 2 + ((lane >> 3) & 1);
          ldsm_x4(ks_addr + swz<HD>(row, ch), b0, b1, b2, b3);
          const int par = ks % kPar;
          mma16816(sp[0][0][par], qa[ks], b0, b1);
          mma16816(sp[0][1][par], ql[ks], b0, b1);
          mma16816(sp[1][0][par], qa[ks], b2, b3);
          mma16816(sp[1][1][par], ql[ks], b2, b3);
        }
        float s0[4], s1[4];
  #pragma unroll
        for (int i = 0; i < 4; ++i) {
          if constexpr (kPar == 2) {
            s0[i] = (sp[0][0][0][i] + sp[0][0][1][i]) + (sp[0][1][0][i] + sp[0][1][1][i]);
            s1[i] = (sp[1][0][0][i] + sp[1][0][1][i]) + (sp[1][1][0][i] + sp[1][1][1][i]);
          } else {
            s0[i] = sp[0][0][0][i] + sp[0][1][0][i];
            s1[i] = sp[1][0][0][i] + sp[1][1][0][i];
          }
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
  }
  cp_async_wait<0>();
  if (tma && waited < n_tiles) {   // a wait ran out: let the copies still in flight land, then stop
    if (tid == 0)
      for (int t = waited; t < next; ++t)
        mbar_wait_drain(&bars[t % kSt], static_cast<uint32_t>(t / kSt) & 1u);
    sync();
    return;
  }
  sync();
  trace_at(ts, 9);
  if (ts != nullptr) trace_after(ts, 12, o[0][0] + o[kNO - 1][3]);   // last MMAs retired

  // merge the key groups of each m-tile (shared memory reuses the K/V stages):
  // the query vectors' rows of o go to shared memory (padding rows are not
  // written or read), one thread per vector computes M = max_w m_w, the group
  // weights f_w = 2^(m_w - M) and L = sum_w f_w l_w, then four features per
  // thread: o = sum_w f_w o_w (groups in ascending order)
  float* mo = reinterpret_cast<float*>(kv);                 // [4 warps][16][HD]
  float* ml = mo + 4 * 16 * HD;                             // [4 warps][16][2]
  float* mf = ml + 4 * 16 * 2;                              // [kMaxQ][4] weights
  float* mml = mf + kMaxQ * 4;                              // [kMaxQ][2] M, L
  if (kTQ) {   // O^T fragments: features 16i + lane/4 (+8), queries 2(lane%4), +1
    const int f0 = lane >> 2;
#pragma unroll
    for (int h2 = 0; h2 < 2; ++h2) {
      const int v = 2 * (lane & 3) + h2;
      if (v >= nq) continue;
      float* dst = mo + (warp * 16 + v) * HD + f0;
#pragma unroll
      for (int i = 0; i < kNO; ++i) {
        dst[i * 16] = o[i][h2];
        dst[i * 16 + 8] = o[i][2 + h2];
      }
      if (f0 == 0) {
        ml[(warp * 16 + v) * 2] = m_run[h2];
        ml[(warp * 16 + v) * 2 + 1] = l_run[h2];
      }
    }
  } else if (active) {
    const int r0 = lane >> 2, cc = (lane & 3) << 1;
    const bool lo_ok = mt * 16 + r0 < nq, hi_ok = mt * 16 + r0 + 8 < nq;
#pragma unroll
    for (int i = 0; i < kNO; ++i) {
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
  constexpr int kV4 = HD / 4;
  bf16* out = a.out;
  bf16* out_lo = a.out_lo;
  const int H = a.H;
  // o = O / L of query vector v, features d..d+3: hi and lo planes, one 8-byte
  // store each (the index is a multiple of 4)
  auto emit = [&](int v, int d, float O0, float O1, float O2, float O3, float L) {
    const float O[4] = {O0, O1, O2, O3};
    const float li = 1.f / L;
    const int hl = v / nr, rr = v - hl * nr;
    const int row = g * R + r_lo + rr;
    const int h = kvh * gs + hl;
    const size_t oi = (static_cast<size_t>(row) * H + h) * HD + d;
    if (dry) return;
    __nv_bfloat16 hv[4], lv[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) split_bf16(O[e] * li, hv[e], lv[e]);
    *reinterpret_cast<uint2*>(out + oi) = *reinterpret_cast<const uint2*>(hv);
    if (out_lo != nullptr) *reinterpret_cast<uint2*>(out_lo + oi) = *reinterpret_cast<const uint2*>(lv);
  };
  // Both ways below compute M = max m_s, weights 2^(m_s - M), L and the weighted
  // sum of the o_s in ascending split order (identical results).
  const size_t land_o = static_cast<size_t>(n_active) * qmax * HD;   // floats
  if ((land_o + static_cast<size_t>(n_active) * qmax * 2) * 4 <= attention_body_bytes<HD, kTQ>()) {
    // every active split's o (contiguous, [split][qmax][HD]) by 16-byte cp.async
    // (L2) and its (m, l) by ld.cg land in the stages - free now: this CTA's own
    // partial went out above - in one round trip; the sums read shared memory
    float* so = reinterpret_cast<float*>(kv);
    float* sml = so + land_o;
    const float* src = part_o + ubase * HD;
    for (size_t i = tid; i < land_o / 4; i += kAttThreads) cp_async16_zfill(so + 4 * i, src + 4 * i, true);
    cp_async_commit();
    for (int i = tid; i < n_active * qmax; i += kAttThreads)
      *reinterpret_cast<float2*>(sml + 2 * i) = ld_cg_f2(part_ml + (ubase + i) * 2);
    cp_async_wait<0>();
    sync();
    trace_at(ts, 6);
    for (int idx = tid; idx < nq * kV4; idx += kAttThreads) {
      const int v = idx / kV4, d = (idx - v * kV4) * 4;
      float M = -INFINITY;
      for (int q = 0; q < n_active; ++q) M = fmaxf(M, sml[(q * qmax + v) * 2]);
      float L = 0.f;
      float O[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll 4
      for (int q = 0; q < n_active; ++q) {
        const float2 ml = *reinterpret_cast<const float2*>(sml + (q * qmax + v) * 2);
        const float4 ov = *reinterpret_cast<const float4*>(so + (static_cast<size_t>(q) * qmax + v) * HD + d);
        const float w = ml.x == -INFINITY ? 0.f : exp2f(ml.x - M);
        L += w * ml.y;
        O[0] += w * ov.x;
        O[1] += w * ov.y;
        O[2] += w * ov.z;
        O[3] += w * ov.w;
      }
      emit(v, d, O[0], O[1], O[2], O[3], L);
    }
  } else {
    // too many splits or vectors to land: each thread fetches, for its query
    // vector v and its four features, every split's (m_s, l_s) (the 32 threads
    // of a vector read the same words: one transaction) together with its o_s
    // (n_active <= 16: the geometry caps the splits), one round trip per pass
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
      emit(v, d, O[0], O[1], O[2], O[3], L);
    }
  }
  trace_at(ts, 7);
  if (tid == 0 && !dry) a.counters[unit] = 0;
}


}  // namespace attn
}  // namespace memspec
