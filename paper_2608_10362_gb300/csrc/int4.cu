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
// with sum_c x over the group (sx) formed once per CTA.  Products are exact;
// the MMA's fp32 accumulation of the biased terms is the only rounding beyond
// the epilogue's.
//
// Layout (memspec_int4_pack).  The kernel reads a repacked copy: one record per
// (16-row tile, group) unit, in tile-major order:
//   bytes [0, 512)     rows 0..7 :  lane L = 4 r + t holds 16 bytes = four 32-bit
//   bytes [512, 1024)  rows 8..15:  words, word j = the GPTQ bytes of row r at
//                                   column offsets g*128 + 32 j + 8 t + (0..7)
//   bytes [1024, 1056) eight bf16 pairs (s[r], s[r + 8])
//   bytes [1056, 1072) eight byte pairs (z[r], z[r + 8])
// so a warp copies a record with three 16-byte-per-lane copies and lane L reads
// exactly its MMA fragment.  Word j's 8 nibbles e = 0..7 become the k slots
// {2t, 2t+1, 2t+8, 2t+9} of two k16 steps as pairs (e, e+4); the activations
// are staged in shared memory with each 16-byte vector permuted the same way,
// so one 16-byte load gives both steps' B fragments and each step contracts
// matching columns.
//
// Work split.  Whole 16-row tiles are dealt to CTAs, the same number to each
// (ceil(tiles / SMs); the grid shrinks to fit), so no output is shared between
// CTAs.  A CTA's units (its tiles x groups, contiguous in memory) are cut into
// 16 equal contiguous ranges, one per warp.  Each warp streams its range
// through its own ring of D record slots with cp.async (D = 8, 4 or 2, the most
// that fits beside the activations), so D records per warp are in flight while
// it computes.  A tile a warp covers whole is stored directly; the partial sums
// of a tile shared by several warps are added in warp order at the end.  Every
// sum has a fixed order: results are bit-reproducible.  Launched with
// programmatic stream serialisation: a CTA starts its weight copies, then
// waits for the previous kernel (whose output may be x).
#include <cuda_bf16.h>

#include "internal.h"

namespace memspec {
namespace {

constexpr int kI4Warps = 16;
constexpr int kI4Threads = kI4Warps * 32;

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

__device__ __forceinline__ uint32_t saddr(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ void cp16(void* dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(saddr(dst)), "l"(src) : "memory");
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

template <int NT, int D>
__global__ void __launch_bounds__(kI4Threads, 1) int4_linear_kernel(const __grid_constant__ Int4Args a) {
  constexpr int Mp = 8 * NT;
  extern __shared__ __align__(128) uint8_t dsm[];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int rq = lane >> 2, t = lane & 3;
  const int M = a.rows, k = a.k, G = k >> 7, n = a.n;
  const int P = 2 * k + 64;   // bytes per staged activation row (the pad makes the fragment loads conflict-free)
  uint8_t* xs = dsm;                                                        // [M][P]
  float* sx = reinterpret_cast<float*>(dsm + ((static_cast<size_t>(M) * P + 15) & ~static_cast<size_t>(15)));
  uint8_t* ring = reinterpret_cast<uint8_t*>(sx) + ((static_cast<size_t>(G) * Mp * 4 + 127) & ~static_cast<size_t>(127));
  uint8_t* my_ring = ring + static_cast<size_t>(warp) * D * kInt4RecordBytes;

  // this CTA's tiles [T0, T1) and this warp's units [lo, hi) of them
  const int tiles = (n + 15) >> 4;
  const int T0 = blockIdx.x * a.tiles_per_cta;
  const int T1 = min(tiles, T0 + a.tiles_per_cta);
  const int L = (T1 - T0) * G;
  const int lo = L * warp / kI4Warps, hi = L * (warp + 1) / kI4Warps;
  const int cnt = hi - lo;
  const uint8_t* src = a.packed + (static_cast<size_t>(T0) * G + lo) * kInt4RecordBytes;

  // ---- start this warp's weight stream first (it does not depend on the
  // previous kernel); one commit group per unit, empty ones included
#pragma unroll
  for (int i = 0; i < D; ++i) {
    if (i < cnt) copy_record(my_ring + i * kInt4RecordBytes, src + static_cast<size_t>(i) * kInt4RecordBytes, lane);
    cp_commit();
  }

  // the activations are the previous kernel's output
  asm volatile("griddepcontrol.wait;" ::: "memory");

  // ---- activations into shared memory, each 16-byte vector (8 columns e) in
  // the order (e0,e4)(e1,e5)(e2,e6)(e3,e7) of the B fragments; and their
  // per-group sums sx[g][m]: half a warp covers one group of one row (16
  // vectors), summed by a fixed xor tree
  {
    const int per_row = k >> 3;
    const int total = M * per_row;
    constexpr int kBatch = 4;
    for (int base = warp * 32; base < total; base += kBatch * kI4Threads) {
      uint4 xv[kBatch];
#pragma unroll
      for (int b = 0; b < kBatch; ++b) {
        const int idx = base + b * kI4Threads + lane;
        xv[b] = idx < total ? __ldg(reinterpret_cast<const uint4*>(a.x) + idx) : make_uint4(0u, 0u, 0u, 0u);
      }
#pragma unroll
      for (int b = 0; b < kBatch; ++b) {
        const int idx = base + b * kI4Threads + lane;
        const uint4 X = xv[b];
        float sum = 0.f;
        const uint32_t w4[4] = {X.x, X.y, X.z, X.w};
#pragma unroll
        for (int e = 0; e < 4; ++e) sum += __uint_as_float(w4[e] << 16) + __uint_as_float(w4[e] & 0xffff0000u);
#pragma unroll
        for (int o = 8; o > 0; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
        if (idx < total) {
          const int m = idx / per_row, v = idx - m * per_row;
          *reinterpret_cast<uint4*>(xs + static_cast<size_t>(m) * P + v * 16) =
              make_uint4(prmt(X.x, X.z, 0x5410), prmt(X.x, X.z, 0x7632), prmt(X.y, X.w, 0x5410),
                         prmt(X.y, X.w, 0x7632));
          if ((lane & 15) == 0) sx[(v >> 4) * Mp + m] = sum;
        }
      }
    }
    for (int i = tid; i < (Mp - M) * G; i += kI4Threads) {   // padding rows: zero sums
      const int g = i / (Mp - M), m = M + i % (Mp - M);
      sx[g * Mp + m] = 0.f;
    }
  }
  __syncthreads();

  // ---- main loop: unit j of the warp sits in ring slot j % D
  float o[NT][4], of[NT][4];
#pragma unroll
  for (int j = 0; j < NT; ++j)
#pragma unroll
    for (int e = 0; e < 4; ++e) o[j][e] = of[j][e] = 0.f;
  int T = T0 + lo / G, g = lo - (lo / G) * G;
  const int T_first = T;
  bool first_partial = false, last_partial = false;
  const uint8_t* xrow[NT];
  bool xok[NT];
#pragma unroll
  for (int j = 0; j < NT; ++j) {
    xrow[j] = xs + static_cast<size_t>(8 * j + rq) * P + 16 * t;
    xok[j] = 8 * j + rq < M;
  }

  for (int base = 0; base < cnt; base += D) {
#pragma unroll
    for (int i = 0; i < D; ++i) {
      const int u = base + i;
      if (u < cnt) {
        cp_wait<D - 1>();
        __syncwarp();
        const uint8_t* slot = my_ring + i * kInt4RecordBytes;
        const uint4 qa = *reinterpret_cast<const uint4*>(slot + lane * 16);
        const uint4 qb = *reinterpret_cast<const uint4*>(slot + 512 + lane * 16);
        const uint32_t sp = *reinterpret_cast<const uint32_t*>(slot + 1024 + rq * 4);
        const uint32_t zp = *reinterpret_cast<const uint16_t*>(slot + 1056 + rq * 2);
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
            // k slots (2t, 2t+1) <- columns (e, e + 4); (2t+8, 2t+9) <- (e+1, e+5)
            mma_bf16(acc0[j], a0, a1, a2, a3, X.x, X.y);
            mma_bf16(acc1[j], a4, a5, a6, a7, X.z, X.w);
          }
        }
        __syncwarp();   // every lane has read the slot: refill it
        if (u + D < cnt)
          copy_record(my_ring + i * kInt4RecordBytes, src + static_cast<size_t>(u + D) * kInt4RecordBytes, lane);
        cp_commit();
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
  asm volatile("griddepcontrol.launch_dependents;");
  cp_wait<0>();
  __syncthreads();   // the rings are free: they hold the partial sums from here on

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
      for (int j = 0; j < 4; ++j) w4[j] = *reinterpret_cast<const uint32_t*>(src + 16 * j);
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
  const size_t xs = (static_cast<size_t>(rows) * (2 * k + 64) + 15) & ~static_cast<size_t>(15);
  const size_t sxb = (static_cast<size_t>(k / 128) * Mp * 4 + 127) & ~static_cast<size_t>(127);
  size_t ring = static_cast<size_t>(kI4Warps) * depth * kInt4RecordBytes;
  const size_t part = static_cast<size_t>(kI4Warps) * 2 * 16 * Mp * 4;
  if (ring < part) ring = part;
  return xs + sxb + ring;
}

int int4_pick_depth(int rows, int k) {
  for (int d : {8, 4, 2})
    if (int4_smem_for(rows, k, d) <= static_cast<size_t>(kInt4MaxSmem)) return d;
  return 0;
}

size_t int4_smem_bytes(int rows, int k) {
  const int d = int4_pick_depth(rows, k);
  return int4_smem_for(rows, k, d == 0 ? 2 : d);
}

cudaError_t int4_set_max_smem() {
  const void* fns[] = {reinterpret_cast<const void*>(int4_linear_kernel<1, 8>),
                       reinterpret_cast<const void*>(int4_linear_kernel<1, 4>),
                       reinterpret_cast<const void*>(int4_linear_kernel<1, 2>),
                       reinterpret_cast<const void*>(int4_linear_kernel<2, 8>),
                       reinterpret_cast<const void*>(int4_linear_kernel<2, 4>),
                       reinterpret_cast<const void*>(int4_linear_kernel<2, 2>)};
  for (const void* f : fns) {
    cudaError_t e = cudaFuncSetAttribute(f, cudaFuncAttributeMaxDynamicSharedMemorySize, kInt4MaxSmem);
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

cudaError_t launch_int4_linear(const Int4Args& a, int grid, cudaStream_t s) {
  const int d = int4_pick_depth(a.rows, a.k);
  if (d == 0) return cudaErrorInvalidValue;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(kI4Threads);
  cfg.dynamicSmemBytes = int4_smem_for(a.rows, a.k, d);
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  const bool wide = a.rows > 8;
  if (d == 8) return wide ? cudaLaunchKernelEx(&cfg, int4_linear_kernel<2, 8>, a)
                          : cudaLaunchKernelEx(&cfg, int4_linear_kernel<1, 8>, a);
  if (d == 4) return wide ? cudaLaunchKernelEx(&cfg, int4_linear_kernel<2, 4>, a)
                          : cudaLaunchKernelEx(&cfg, int4_linear_kernel<1, 4>, a);
  return wide ? cudaLaunchKernelEx(&cfg, int4_linear_kernel<2, 2>, a)
              : cudaLaunchKernelEx(&cfg, int4_linear_kernel<1, 2>, a);
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
