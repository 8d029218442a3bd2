// int4.cu - group-wise INT4 weight-only linear layer for decode-sized row counts
// (the paper's targets are GPTQ INT4 models, Section 4.1).
//
// y[m][r] = sum_c x[m][c] w[r][c],  w[r][c] = (q[r][c] - z[r][g]) s[r][g],  g = c / 128,
// q 4-bit codes, s bf16 scales, z 4-bit zero points (stored one per byte).
//
// Why the tensor pipe.  At 4 bits the weights arrive at ~2 weights per byte of
// HBM traffic, i.e. ~44 weights per clock per SM at the copy bandwidth.  A
// CUDA-core kernel spends ~3 instructions per weight on unpacking plus one FMA
// per weight per activation row, which for the verify pass's K + 1 = 5 rows is
// ~1.7x more issue than an SM has.  So the kernel unpacks the codes straight
// into the A-operand registers of a register-sourced bf16 MMA (m16n8k16; the
// weights are A, 16 rows, the activation rows are the n = 8 side) and lets the
// tensor pipe do the products.  tcgen05 would need the unpacked tile written to
// shared memory or TMEM first (2 extra bytes moved per weight for 0.5 loaded);
// the contraction is far too thin (<= 16 activation rows) to need its rate.
//
// Exactness of the operands.  A code q enters the MMA as the bf16 128 + q
// (exponent of 128, q in the mantissa's low bits: one LOP3 per two codes), the
// zero point is folded out per group:
//   sum_c x (q - z) = sum_c x (128 + q) - (128 + z) sum_c x,
// with the group sums of x formed once per CTA by the tensor pipe too: MMAs with
// an all-ones A operand on the same B fragments leave sum_c x in exactly the
// accumulator layout of the products (no shuffles, no extra ALU work), kept in
// shared memory for the fold.  Products are exact; the MMAs' fp32
// accumulation is the only rounding beyond the epilogue's.
//
// Layout (memspec_int4_pack).  The kernel reads a repacked copy: one record per
// (16-row tile, group) unit, in tile-major order:
//   bytes [0, 512)     rows 0..7 :  lane L = 4 r + t holds 16 bytes = four 32-bit
//   bytes [512, 1024)  rows 8..15:  words, word j = the GPTQ bytes of row r at
//                                   column offsets g*128 + 32 j + 8 t + (0..7)
//   bytes [1024, 1056) eight bf16 pairs (s[r], s[r + 8])
//   bytes [1056, 1072) eight byte pairs (z[r], z[r + 8])
// and within each word the codes of columns e = 0..7 sit at nibble positions
// 0 4 1 5 2 6 3 7 (e = 0..7), so that masking nibbles p and p + 4 of
// (word >> 4 p) yields the bf16 pair of columns (2p, 2p + 1): exactly the
// A-fragment pair that meets the activation pair (x[2p], x[2p + 1]) in the
// natural bf16 layout.  Lane L's record bytes are its A fragments and one
// 16-byte load of x gives the B fragments of two k16 steps.
//
// Work split.  Whole 16-row tiles are dealt to CTAs, the same number to each
// (ceil(tiles / SMs); the grid shrinks to fit), so no output is shared between
// CTAs.  A CTA's units (its tiles x groups, contiguous in memory) are cut into
// 16 equal contiguous ranges, one per warp.  Each warp streams its range
// through its own ring of D = 2 record slots with cp.async, one commit group
// per record (small copies: per-request cost decides, and 1 KB bulk copies
// were slower).  Measured on GB300, rings of 4 and 8 slots were no faster
// (the load/store pipe's throughput, not the bytes in flight, is the limit)
// and took longer to issue.  The
// activations arrive as one 1-D bulk copy (TMA) per row, outside the
// load/store unit's queue.  That wait is bounded: on expiry the kernel sets
// bit 0 of the optional status word and finishes without computing.  A tile a warp covers whole is stored directly; the partial sums
// of a tile shared by several warps are added in warp order at the end.  Every
// sum has a fixed order: results are bit-reproducible.  Launched with
// programmatic stream serialisation: a CTA starts its weight copies, then
// waits for the previous kernel (whose output may be x).
#include <cuda_bf16.h>

#include "internal.h"
#include "ptx.cuh"

namespace memspec {
namespace {

constexpr int kI4Warps = 16;
constexpr int kI4Threads = kI4Warps * 32;
constexpr int kI4Depth = 2;   // record slots per warp

__device__ __forceinline__ uint32_t prmt(uint32_t a, uint32_t b, uint32_t sel) {
  uint32_t d;
  asm("prmt.b32 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(sel));
  return d;
}

// nibbles 0 and 4 of w -> bf16 pair (128 + lo, 128 + hi)
__device__ __forceinline__ uint32_t nib2(uint32_t w) {
  uint32_t d;
  asm("lop3.b32 %0, %1, 0x000F000F, 0x43004300, 0xEA;" : "=r"(d) : "r"(w));   // (a & b) | c
  return d;
}

__device__ __forceinline__ void mma_bf16(float (&c)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                         uint32_t b0, uint32_t b1) {
  asm("mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

__device__ __forceinline__ void cp16(void* dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_addr(dst)), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

// one record into a ring slot: three 16-byte copies per lane (lanes 0..2 carry
// the scale / zero-point tail)
__device__ __forceinline__ void copy_record(uint8_t* slot, const uint8_t* src, int lane) {
  cp16(slot + lane * 16, src + lane * 16);
  cp16(slot + 512 + lane * 16, src + 512 + lane * 16);
  if (lane < 3) cp16(slot + 1024 + lane * 16, src + 1024 + lane * 16);
}

// the last of `parts` equal contiguous parts of [0, total) that starts at or
// before v (never an empty part)
__device__ __forceinline__ int part_of(int v, int total, int parts) {
  return ((v + 1) * parts + total - 1) / total - 1;
}

// Bounded mbarrier wait with a warp-uniform outcome (the MMAs after it need
// every lane): true once every lane has seen the phase complete; false if the
// budget ran out or another warp gave up (then lane 0 raises the flag and the
// status bit).
__device__ __forceinline__ bool warp_wait(uint64_t* bar, uint32_t parity, volatile int* abort_flag,
                                          uint32_t* status) {
  const long long t0 = clock64();
  for (;;) {
    const bool ok = mbar_try_wait(bar, parity);
    if (__all_sync(0xffffffffu, ok)) return true;
    const bool bad = *abort_flag != 0 || clock64() - t0 > kWaitBudgetCycles;
    if (__any_sync(0xffffffffu, bad)) {
      if ((threadIdx.x & 31) == 0) {
        *abort_flag = 1;
        if (status != nullptr) atomicOr(status, 0x1u);
      }
      return false;
    }
  }
}

template <int NT, int D>
__global__ void __launch_bounds__(kI4Threads, 1) int4_linear_kernel(const __grid_constant__ Int4Args a) {
  constexpr int Mp = 8 * NT;
  extern __shared__ __align__(128) uint8_t dsm[];
  __shared__ uint64_t xbar;
  __shared__ int abort_flag;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int rq = lane >> 2, t = lane & 3;
  const int M = a.rows, k = a.k, G = k >> 7, n = a.n;
  const int P = 2 * k + 64;   // bytes per staged activation row (the pad makes the fragment loads conflict-free)
  uint8_t* xs = dsm;                                                        // [M][P]
  float* sx = reinterpret_cast<float*>(dsm + ((static_cast<size_t>(M) * P + 127) & ~static_cast<size_t>(127)));
  uint8_t* ring = reinterpret_cast<uint8_t*>(sx) + ((static_cast<size_t>(G) * Mp * 4 + 127) & ~static_cast<size_t>(127));
  uint8_t* my_ring = ring + static_cast<size_t>(warp) * D * kInt4RecordBytes;
  volatile int* abort_v = &abort_flag;

  // this CTA's tiles [T0, T1) and this warp's units [lo, hi) of them
  const int tiles = (n + 15) >> 4;
  const int T0 = min(tiles, static_cast<int>(blockIdx.x) * a.tiles_per_cta);   // CTAs past the end: no tiles
  const int T1 = min(tiles, T0 + a.tiles_per_cta);
  const int L = (T1 - T0) * G;
  const int lo = L * warp / kI4Warps, hi = L * (warp + 1) / kI4Warps;
  const int cnt = hi - lo;
  const uint8_t* src = a.packed + (static_cast<size_t>(T0) * G + lo) * kInt4RecordBytes;

  if (tid == 0) {
    mbar_init(&xbar, 1);
    abort_flag = 0;
  }
  fence_mbar_init();
  __syncthreads();

  // ---- this warp's weight stream first (it does not depend on the previous
  // kernel); one commit group per record, empty ones included
#pragma unroll
  for (int i = 0; i < D; ++i) {
    if (i < cnt) copy_record(my_ring + i * kInt4RecordBytes, src + static_cast<size_t>(i) * kInt4RecordBytes, lane);
    cp_commit();
  }

  // ---- the activations (the previous kernel's output): one bulk copy per row
  pdl_wait();
  if (tid == 0) {
    const uint64_t pol = l2_policy_evict_last();
    mbar_arrive_expect_tx(&xbar, static_cast<uint32_t>(M) * 2 * k);
    for (int m = 0; m < M; ++m)
      bulk_load(xs + static_cast<size_t>(m) * P, a.x + static_cast<size_t>(m) * k, 2 * k, &xbar, pol);
  }
  bool ok = warp_wait(&xbar, 0, abort_v, a.status);
  const uint8_t* xrow[NT];
  bool xok[NT];
#pragma unroll
  for (int j = 0; j < NT; ++j) {
    xrow[j] = xs + static_cast<size_t>(8 * j + rq) * P + 16 * t;
    xok[j] = 8 * j + rq < M;
  }
  constexpr uint32_t kOnes = 0x3F803F80u;   // bf16 pair (1, 1)
  // group sums sx[g][m] = sum of x[m][128 g .. 128 g + 127]: MMAs with an
  // all-ones A operand, one group per warp at a time (rows past M read as 0)
  if (ok) {
    for (int gg = warp; gg < G; gg += kI4Warps) {
#pragma unroll
      for (int j = 0; j < NT; ++j) {
        float c[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int w = 0; w < 4; ++w) {
          uint4 X = make_uint4(0u, 0u, 0u, 0u);
          if (xok[j]) X = *reinterpret_cast<const uint4*>(xrow[j] + gg * 256 + w * 64);
          mma_bf16(c, kOnes, kOnes, kOnes, kOnes, X.x, X.y);
          mma_bf16(c, kOnes, kOnes, kOnes, kOnes, X.z, X.w);
        }
        if (rq == 0) *reinterpret_cast<float2*>(sx + gg * Mp + 8 * j + 2 * t) = make_float2(c[0], c[1]);
      }
    }
  }
  __syncthreads();
  ok = ok && *abort_v == 0;

  // ---- main loop: unit u of the warp sits in ring slot u % D
  float o[NT][4], of[NT][4];
#pragma unroll
  for (int j = 0; j < NT; ++j)
#pragma unroll
    for (int e = 0; e < 4; ++e) o[j][e] = of[j][e] = 0.f;
  int T = T0 + lo / G, g = lo - (lo / G) * G;
  const int T_first = T;
  bool first_partial = false, last_partial = false;
  for (int base = 0; base < cnt && ok; base += D) {
#pragma unroll
    for (int i = 0; i < D; ++i) {
      const int u = base + i;
      if (u < cnt) {
        {
          cp_wait<D - 1>();   // this lane's copies of unit u have landed
          __syncwarp();       // ... and every other lane's
          const uint8_t* slot = my_ring + i * kInt4RecordBytes;
          const uint4 qa = *reinterpret_cast<const uint4*>(slot + lane * 16);
          const uint4 qb = *reinterpret_cast<const uint4*>(slot + 512 + lane * 16);
          const uint32_t sp = *reinterpret_cast<const uint32_t*>(slot + 1024 + rq * 4);
          const uint32_t zp = *reinterpret_cast<const uint16_t*>(slot + 1056 + rq * 2);
          __syncwarp();   // every lane has read the slot: refill it
          if (u + D < cnt)
            copy_record(my_ring + i * kInt4RecordBytes, src + static_cast<size_t>(u + D) * kInt4RecordBytes, lane);
          cp_commit();
          float acc0[NT][4], acc1[NT][4];
#pragma unroll
          for (int j = 0; j < NT; ++j)
#pragma unroll
            for (int e = 0; e < 4; ++e) acc0[j][e] = acc1[j][e] = 0.f;
          const uint32_t wa[4] = {qa.x, qa.y, qa.z, qa.w};
          const uint32_t wb[4] = {qb.x, qb.y, qb.z, qb.w};
#pragma unroll
          for (int w = 0; w < 4; ++w) {
            const uint32_t a0 = nib2(wa[w]), a1 = nib2(wb[w]);
            const uint32_t a2 = nib2(wa[w] >> 4), a3 = nib2(wb[w] >> 4);
            const uint32_t a4 = nib2(wa[w] >> 8), a5 = nib2(wb[w] >> 8);
            const uint32_t a6 = nib2(wa[w] >> 12), a7 = nib2(wb[w] >> 12);
#pragma unroll
            for (int j = 0; j < NT; ++j) {
              uint4 X = make_uint4(0u, 0u, 0u, 0u);
              if (xok[j]) X = *reinterpret_cast<const uint4*>(xrow[j] + g * 256 + w * 64);
              // k slots (2t, 2t+1) <- columns (0, 1) of the 8; (2t+8, 2t+9) <- (2, 3); then (4, 5), (6, 7)
              mma_bf16(acc0[j], a0, a1, a2, a3, X.x, X.y);
              mma_bf16(acc1[j], a4, a5, a6, a7, X.z, X.w);
            }
          }
          // fold the scale and zero point of this group
          const float s0 = __uint_as_float(sp << 16), s1 = __uint_as_float(sp & 0xffff0000u);
          const float z0 = 128.f + static_cast<float>(zp & 0xffu), z1 = 128.f + static_cast<float>(zp >> 8);
#pragma unroll
          for (int j = 0; j < NT; ++j) {
            const float2 sv = *reinterpret_cast<const float2*>(sx + g * Mp + 8 * j + 2 * t);
            o[j][0] = fmaf(s0, fmaf(-z0, sv.x, acc0[j][0] + acc1[j][0]), o[j][0]);
            o[j][1] = fmaf(s0, fmaf(-z0, sv.y, acc0[j][1] + acc1[j][1]), o[j][1]);
            o[j][2] = fmaf(s1, fmaf(-z1, sv.x, acc0[j][2] + acc1[j][2]), o[j][2]);
            o[j][3] = fmaf(s1, fmaf(-z1, sv.y, acc0[j][3] + acc1[j][3]), o[j][3]);
          }
          // end of a tile, or of the warp's range
          ++g;
          const bool last = u + 1 == cnt;
          if (g == G || last) {
            const bool whole = g == G && (T != T_first || lo == (T - T0) * G);
            if (whole) {
              const int r0 = T * 16 + rq, r1 = r0 + 8;
#pragma unroll
              for (int j = 0; j < NT; ++j) {
                const int m = 8 * j + 2 * t;
                if (m < M) {
                  if (r0 < n) a.y[static_cast<size_t>(m) * n + r0] = o[j][0];
                  if (r1 < n) a.y[static_cast<size_t>(m) * n + r1] = o[j][2];
                }
                if (m + 1 < M) {
                  if (r0 < n) a.y[static_cast<size_t>(m + 1) * n + r0] = o[j][1];
                  if (r1 < n) a.y[static_cast<size_t>(m + 1) * n + r1] = o[j][3];
                }
              }
            } else if (T == T_first) {
              first_partial = true;
#pragma unroll
              for (int j = 0; j < NT; ++j)
#pragma unroll
                for (int e = 0; e < 4; ++e) of[j][e] = o[j][e];
            } else {
              last_partial = true;   // the range ends inside this tile: keep o
            }
            if (!last || whole || T == T_first) {
#pragma unroll
              for (int j = 0; j < NT; ++j)
#pragma unroll
                for (int e = 0; e < 4; ++e) o[j][e] = 0.f;
            }
            if (g == G) {
              g = 0;
              ++T;
            }
          }
        }
      }
    }
  }
  pdl_launch_dependents();
  cp_wait<0>();
  if (tid == 0 && *abort_v) mbar_wait_drain(&xbar, 0);   // after a timeout: let the copies land before exit
  __syncthreads();   // the rings are free: they hold the partial sums from here on
  if (*abort_v) return;

  // ---- partial tiles: slot 0 = the warp's first tile, slot 1 = its last
  float* part = reinterpret_cast<float*>(ring);   // [warp][2][16][Mp]
  if (first_partial || last_partial) {
#pragma unroll
    for (int s2 = 0; s2 < 2; ++s2) {
      if (s2 == 0 ? !first_partial : !last_partial) continue;
      float* ps = part + (warp * 2 + s2) * 16 * Mp;
#pragma unroll
      for (int j = 0; j < NT; ++j) {
        const int m = 8 * j + 2 * t;
        const float* v = s2 == 0 ? of[j] : o[j];
        ps[rq * Mp + m] = v[0];
        ps[rq * Mp + m + 1] = v[1];
        ps[(rq + 8) * Mp + m] = v[2];
        ps[(rq + 8) * Mp + m + 1] = v[3];
      }
    }
  }
  __syncthreads();
  // one (tile, row, column) output per thread and pass; warps w_lo..w_hi
  // share the tile, added in warp order
  const int outs = (T1 - T0) * 16 * Mp;
  for (int idx = tid; idx < outs; idx += kI4Threads) {
    const int tl = idx / (16 * Mp), rc = idx - tl * 16 * Mp;
    const int v0 = tl * G, v1 = v0 + G - 1;
    const int w_lo = part_of(v0, L, kI4Warps), w_hi = part_of(v1, L, kI4Warps);
    if (w_lo == w_hi) continue;   // stored by that warp
    float v = 0.f;
    for (int w = w_lo; w <= w_hi; ++w) {
      const int wlo = L * w / kI4Warps, whi = L * (w + 1) / kI4Warps;
      if (wlo == whi) continue;
      v += part[(w * 2 + (wlo >= v0 ? 0 : 1)) * 16 * Mp + rc];
    }
    const int r = (T0 + tl) * 16 + rc / Mp, m = rc % Mp;
    if (m < M && r < n) a.y[static_cast<size_t>(m) * n + r] = v;
  }
}

// code of column e (nibble e of the GPTQ word) -> nibble position (e >> 1) + 4 (e & 1)
__device__ __forceinline__ uint32_t interleave_nibbles(uint32_t w) {
  uint32_t r = 0;
#pragma unroll
  for (int e = 0; e < 8; ++e) r |= ((w >> (4 * e)) & 0xFu) << (4 * ((e >> 1) + 4 * (e & 1)));
  return r;
}

// One thread per 16-byte code block (64 per unit) plus one per unit tail.
__global__ void int4_pack_kernel(const uint8_t* __restrict__ qweight, const bf16* __restrict__ scales,
                                 const uint8_t* __restrict__ zeros, uint8_t* __restrict__ out, int n, int k,
                                 long long units) {
  const int G = k >> 7;
  const long long i = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (i >= units * 65) return;
  const long long u = i / 65;
  const int b = static_cast<int>(i - u * 65);
  const long long T = u / G;
  const int g = static_cast<int>(u - T * G);
  uint8_t* rec = out + u * kInt4RecordBytes;
  if (b < 64) {
    const int half = b >> 5, lane = b & 31, r = lane >> 2, t = lane & 3;
    const long long row = T * 16 + half * 8 + r;
    uint32_t w4[4] = {0u, 0u, 0u, 0u};
    if (row < n) {
      const uint8_t* src = qweight + row * (k / 2) + g * 64 + 4 * t;
#pragma unroll
      for (int j = 0; j < 4; ++j) w4[j] = interleave_nibbles(*reinterpret_cast<const uint32_t*>(src + 16 * j));
    }
    *reinterpret_cast<uint4*>(rec + half * 512 + lane * 16) = make_uint4(w4[0], w4[1], w4[2], w4[3]);
  } else {
    uint32_t sw[8];
    uint16_t zw[8];
    for (int r = 0; r < 8; ++r) {
      const long long r0 = T * 16 + r, r1 = r0 + 8;
      uint16_t s0 = 0, s1 = 0, z0 = 0, z1 = 0;
      if (r0 < n) {
        s0 = __bfloat16_as_ushort(scales[r0 * G + g]);
        z0 = zeros[r0 * G + g];
      }
      if (r1 < n) {
        s1 = __bfloat16_as_ushort(scales[r1 * G + g]);
        z1 = zeros[r1 * G + g];
      }
      sw[r] = static_cast<uint32_t>(s0) | (static_cast<uint32_t>(s1) << 16);
      zw[r] = static_cast<uint16_t>(z0 | (z1 << 8));
    }
    uint4* d = reinterpret_cast<uint4*>(rec + 1024);
    d[0] = make_uint4(sw[0], sw[1], sw[2], sw[3]);
    d[1] = make_uint4(sw[4], sw[5], sw[6], sw[7]);
    d[2] = make_uint4(zw[0] | (static_cast<uint32_t>(zw[1]) << 16), zw[2] | (static_cast<uint32_t>(zw[3]) << 16),
                      zw[4] | (static_cast<uint32_t>(zw[5]) << 16), zw[6] | (static_cast<uint32_t>(zw[7]) << 16));
  }
}

}  // namespace

size_t int4_packed_bytes(long long n, int k) {
  return static_cast<size_t>((n + 15) / 16) * static_cast<size_t>(k / 128) * kInt4RecordBytes;
}

static size_t int4_smem_for(int rows, int k, int depth) {
  const int Mp = rows <= 8 ? 8 : 16;
  const size_t xs = (static_cast<size_t>(rows) * (2 * k + 64) + 127) & ~static_cast<size_t>(127);
  const size_t sxb = (static_cast<size_t>(k / 128) * Mp * 4 + 127) & ~static_cast<size_t>(127);
  size_t ring = static_cast<size_t>(kI4Warps) * depth * kInt4RecordBytes;
  const size_t part = static_cast<size_t>(kI4Warps) * 2 * 16 * Mp * 4;
  if (ring < part) ring = part;
  return xs + sxb + ring;
}

int int4_pick_depth(int rows, int k) {
  return int4_smem_for(rows, k, kI4Depth) <= static_cast<size_t>(kInt4MaxSmem) ? kI4Depth : 0;
}

cudaError_t int4_set_max_smem() {
  const void* fns[] = {reinterpret_cast<const void*>(int4_linear_kernel<1, kI4Depth>),
                       reinterpret_cast<const void*>(int4_linear_kernel<2, kI4Depth>)};
  for (const void* f : fns) {
    cudaError_t e = cudaFuncSetAttribute(f, cudaFuncAttributeMaxDynamicSharedMemorySize, kInt4MaxSmem);
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

Int4Plan int4_plan(int rows, int n, int k, int sms) {
  Int4Plan p{};
  p.depth = int4_pick_depth(rows, k);
  if (p.depth == 0) return p;
  const int tiles = (n + 15) / 16;
  p.tiles_per_cta = (tiles + sms - 1) / sms;
  p.grid = (tiles + p.tiles_per_cta - 1) / p.tiles_per_cta;
  return p;
}

cudaError_t launch_int4_linear(const Int4Args& a, const Int4Plan& p, cudaStream_t s) {
  if (p.depth == 0) return cudaErrorInvalidValue;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(p.grid);
  cfg.blockDim = dim3(kI4Threads);
  cfg.dynamicSmemBytes = int4_smem_for(a.rows, a.k, p.depth);
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return a.rows > 8 ? cudaLaunchKernelEx(&cfg, int4_linear_kernel<2, kI4Depth>, a)
                    : cudaLaunchKernelEx(&cfg, int4_linear_kernel<1, kI4Depth>, a);
}

cudaError_t launch_int4_pack(const uint8_t* qweight, const bf16* scales, const uint8_t* zeros, uint8_t* out,
                             int n, int k, cudaStream_t s) {
  const long long units = static_cast<long long>((n + 15) / 16) * (k / 128);
  const long long threads = units * 65;
  const int block = 256;
  const long long grid = (threads + block - 1) / block;
  int4_pack_kernel<<<static_cast<unsigned>(grid), block, 0, s>>>(qweight, scales, zeros, out, n, k, units);
  return cudaGetLastError();
}

}  // namespace memspec
