// gemm.cu - weight-streaming projection GEMM for the verify and draft passes.
//
// Y[rows][n_out] = X[rows][k] . W[n_out][k]^T with rows <= 256 (K+1 verify rows,
// 1-2 draft rows, up to 128 prefill rows).  At these row counts every projection
// of the decoder (QKV, O, gate/up, down, LM head) reads each weight exactly once
// and is bound by HBM bandwidth, so the kernel is organised around streaming
// weights:
//
//  * swap-AB: the weight tile is the MMA's M=128 operand, the activation rows
//    are its N (16..256) operand; tcgen05.mma.kind::f16 (bf16 in, fp32 out)
//    accumulates in TMEM;
//  * weight tiles [128 rows x 64 k] arrive by TMA (128-byte swizzle) into a
//    multi-stage mbarrier ring; they are independent of earlier kernels, so the
//    producer starts streaming before griddepcontrol.wait (programmatic
//    dependent launch hides the previous kernel's tail);
//  * activation tiles [n_pad rows x 64 k] arrive by TMA on the same barrier,
//    issued only after griddepcontrol.wait (they are the previous kernel's
//    output); RMSNorm is folded in: the previous epilogue wrote bf16(h * gain)
//    and per-row-tile sums of squares, and this kernel's epilogue scales each
//    output row by rsqrt(mean(h^2) + eps) (exact: the scale is per row);
//  * stream-K: the (row-tile, k-tile) space is cut into one contiguous range
//    per CTA, one CTA per SM; a row tile split over several CTAs is reduced by
//    the last-arriving CTA in ascending CTA order (deterministic, no float
//    atomics) from an fp32 partial buffer;
//  * fused epilogues: fp32 logits; residual add (+ the row sums of squares
//    the next RMSNorm needs); SwiGLU of interleaved gate/up tiles; RoPE on q/k
//    with K/V appended to the KV cache at each row's position.
#include <cuda_bf16.h>

#include <cstdlib>

#include "gemm_epi.cuh"
#include "internal.h"
#include "ptx.cuh"

namespace memspec {

namespace {

using namespace gemm;

constexpr int kThreads = 192;   // warp 0 TMA, warp 1 MMA, warps 2-5 epilogue

struct SmemCtl {
  uint64_t full[kMaxStages];
  uint64_t empty[kMaxStages];
  uint64_t acc_full[2];
  uint64_t acc_empty[2];
  uint64_t drain;
  uint32_t tmem_base;
  int abort_flag;
  int reduce_flag;
  int wait_ok;
  float red[4][16];
  uint64_t recv;        // cluster exchange: partials pushed by peers (one phase)
  int recv_pending;     // this CTA expects pushed partials it has not yet consumed
};

// CSK: launched in clusters of a.csk CTAs with the cluster exchange of split row
// tiles (epilogue_segment); the plain kernel carries none of that code.
template <int EPI, bool CSK>
__global__ void __launch_bounds__(kThreads, 1) gemm_stream_kernel(const __grid_constant__ GemmArgs a) {
  __shared__ SmemCtl ctl;
  extern __shared__ uint8_t dsmem_raw[];
  uint8_t* dsmem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(dsmem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  const int S = a.stages;
  const int plane_bytes = a.n_pad * 128;              // one [n_pad][64] bf16 activation plane
  const int b_bytes = plane_bytes * (a.split ? 2 : 1);
  const uint32_t stage_tx = static_cast<uint32_t>(kABytes + b_bytes);
  uint8_t* smem_a = dsmem;
  uint8_t* smem_b = dsmem + static_cast<size_t>(S) * kABytes;
  float* stage = reinterpret_cast<float*>(smem_b + static_cast<size_t>(S) * b_bytes);
  float* rms = stage + kStageFloats;
  EpiCtx* ectx = reinterpret_cast<EpiCtx*>(rms + kMaxRows);
  float* recv = reinterpret_cast<float*>(
      (reinterpret_cast<uintptr_t>(ectx + 1) + 15) & ~static_cast<uintptr_t>(15));

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int T = a.row_tiles * a.k_tiles;
  const int G = gridDim.x, c = blockIdx.x;
  const int t_begin = sk_begin(c, T, G), t_end = sk_begin(c + 1, T, G);
  const int KT = a.k_tiles;
  const int layout = !a.split ? kPlain : (2 * a.n_pad <= 256 ? kWide : kTwice);
  const int acols = acc_cols(a, layout);                 // accumulator columns per buffer
  const uint32_t tmem_cols = tmem_cols_for(acols);

  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(&ctl.full[s], 1);
      mbar_init(&ctl.empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&ctl.acc_full[b], 1);
      mbar_init(&ctl.acc_empty[b], 4);
    }
    mbar_init(&ctl.drain, 1);
    if constexpr (CSK) {
      mbar_init(&ctl.recv, 1);
      ctl.recv_pending = 0;
    }
    ctl.abort_flag = 0;
    ctl.reduce_flag = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    __syncwarp();
    tmem_alloc(&ctl.tmem_base, tmem_cols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  // cluster exchange: the barriers above are initialised before any peer pushes
  // (every thread arrives here; a thread waits before its first push)
  if constexpr (CSK) cluster_arrive_release();
  pdl_launch_dependents();
  const uint32_t tmem_base = ctl.tmem_base;
  // optional trace (16 slots per CTA): 0 entry, 13 dependency released,
  // 2 activation loads issued, 3 first MMA, 4..11 epilogue, 1 exit
  unsigned long long* trace = a.trace != nullptr ? a.trace + blockIdx.x * 16 : nullptr;
  if (threadIdx.x == 64) trace_at(trace, 0);
  volatile int* abort_flag = &ctl.abort_flag;

  if (warp == 0) {
    // ------------------------------------------------ TMA producer
    // Weight tiles do not depend on earlier kernels: the first S of them are
    // requested before griddepcontrol.wait.  Activation tiles are requested after.
    if (lane == 0) {
      if (a.a_packed == nullptr) {
        tma_prefetch_desc(&a.map_a);
        if (a.pair) tma_prefetch_desc(&a.map_a2);
      }
      tma_prefetch_desc(&a.map_b);
      if (a.split) tma_prefetch_desc(&a.map_b2);
      const uint64_t pol = a.l2_hint == L2_EVICT_FIRST  ? l2_policy_evict_first()
                           : a.l2_hint == L2_EVICT_LAST ? l2_policy_evict_last()
                                                        : l2_policy_evict_normal();
      const uint64_t pol_b = l2_policy_evict_last();   // activations are re-read by every CTA
      uint32_t issued_mask = 0, last_par = 0;
      bool ok = true;
      const int n_pre = min(S, t_end - t_begin);
      // One thread issues every copy, so the loop is lean: the ring position and
      // the tile coordinates advance incrementally (no division per tile).
      const uint8_t* wsrc = a.a_packed != nullptr
                                ? a.a_packed + static_cast<size_t>(t_begin) * kABytes : nullptr;
      int rt = t_begin / KT, kt = t_begin - rt * KT;
      auto load_a = [&](int slot) {
        uint8_t* dst = smem_a + static_cast<size_t>(slot) * kABytes;
        if (wsrc != nullptr) {
          bulk_load(dst, wsrc, kABytes, &ctl.full[slot], pol);
          wsrc += kABytes;
        } else if (a.pair) {
          tma_load_2d(dst, &a.map_a, kt * kTileK, rt * 64, &ctl.full[slot], pol);
          tma_load_2d(dst + kABytes / 2, &a.map_a2, kt * kTileK, rt * 64, &ctl.full[slot], pol);
        } else {
          tma_load_2d(dst, &a.map_a, kt * kTileK, rt * kTileM, &ctl.full[slot], pol);
        }
      };
      auto load_b = [&](int slot, int k_tile) {
        uint8_t* dst = smem_b + static_cast<size_t>(slot) * b_bytes;
        tma_load_2d(dst, &a.map_b, k_tile * kTileK, 0, &ctl.full[slot], pol_b);
        if (a.split) tma_load_2d(dst + plane_bytes, &a.map_b2, k_tile * kTileK, 0, &ctl.full[slot], pol_b);
      };
      // weights of the first n_pre tiles (the ring is empty: no wait needed)
      const int kt_first = kt;
      for (int p = 0; p < n_pre; ++p) {
        mbar_arrive_expect_tx(&ctl.full[p], stage_tx);
        load_a(p);
        issued_mask |= 1u << p;
        if (++kt == KT) {
          kt = 0;
          ++rt;
        }
      }
      pdl_wait();
      trace_at(trace, 2);
      {
        int k2 = kt_first;
        for (int p = 0; p < n_pre; ++p) {
          load_b(p, k2);
          if (++k2 == KT) k2 = 0;
        }
      }
      int s = n_pre == S ? 0 : n_pre;
      uint32_t ph = n_pre == S ? 1u : 0u;   // phase of the fill the next wait is for
      for (int t = t_begin + n_pre; t < t_end; ++t) {
        if (!mbar_wait_bounded(&ctl.empty[s], ph ^ 1u, abort_flag, a.status)) {
          ok = false;
          break;
        }
        mbar_arrive_expect_tx(&ctl.full[s], stage_tx);
        load_a(s);
        load_b(s, kt);
        issued_mask |= 1u << s;
        last_par = (last_par & ~(1u << s)) | (ph << s);
        if (++kt == KT) {
          kt = 0;
          ++rt;
        }
        if (++s == S) {
          s = 0;
          ph ^= 1u;
        }
      }
      if (!ok) {  // tear-down: let every copy still in flight land before exit
        for (int s = 0; s < S; ++s)
          if (issued_mask & (1u << s)) mbar_wait_drain(&ctl.full[s], (last_par >> s) & 1u);
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------ MMA issuer
    if (lane == 0) {
      const uint32_t idesc = make_idesc_bf16_f32(kTileM, layout == kWide ? 2 * a.n_pad : a.n_pad);
      // descriptors of stage 0; a stage's (and a k-step's) are offsets in the
      // start-address field (address >> 4, 14 bits: shared memory < 256 KB)
      const uint64_t adesc0 = make_smem_desc_sw128(smem_addr(smem_a));
      const uint64_t bdesc0 = make_smem_desc_sw128(smem_addr(smem_b));
      const uint32_t a_step = kABytes >> 4, b_step = static_cast<uint32_t>(b_bytes) >> 4;
      const uint32_t p_step = static_cast<uint32_t>(plane_bytes) >> 4;
      int s = 0, seg = 0;
      uint32_t ph = 0;
      bool ok = true, first = true;
      for (int t = t_begin; t < t_end && ok; ++seg) {
        const int rt = t / KT;
        const int seg_end = min(t_end, (rt + 1) * KT);
        const int buf = seg & 1;
        if (seg >= 2 &&
            !mbar_wait_bounded(&ctl.acc_empty[buf], static_cast<uint32_t>((seg >> 1) - 1) & 1u,
                               abort_flag, a.status)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + static_cast<uint32_t>(buf * acols);
        for (int tt = t; tt < seg_end; ++tt) {
          if (!mbar_wait_bounded(&ctl.full[s], ph, abort_flag, a.status)) {
            ok = false;
            break;
          }
          if (first) {
            trace_at(trace, 3);
            first = false;
          }
          tc_fence_after();
          const uint64_t ad = adesc0 + static_cast<uint32_t>(s) * a_step;
          const uint64_t bd = bdesc0 + static_cast<uint32_t>(s) * b_step;
          const uint32_t acc0 = tt > t ? 1u : 0u;
          if (layout != kTwice) {   // one MMA per k-step (N = n_pad or 2 n_pad)
#pragma unroll
            for (int kk = 0; kk < kTileK / 16; ++kk)
              tc_mma_bf16(d_tmem, ad + 2 * kk, bd + 2 * kk, idesc, kk > 0 ? 1u : acc0);
          } else {                  // hi then lo plane into the same accumulator
#pragma unroll
            for (int kk = 0; kk < kTileK / 16; ++kk) {
              tc_mma_bf16(d_tmem, ad + 2 * kk, bd + 2 * kk, idesc, kk > 0 ? 1u : acc0);
              tc_mma_bf16(d_tmem, ad + 2 * kk, bd + p_step + 2 * kk, idesc, 1u);
            }
          }
          tc_commit(&ctl.empty[s]);
          if (++s == S) {
            s = 0;
            ph ^= 1u;
          }
        }
        if (!ok) break;
        tc_commit(&ctl.acc_full[buf]);
        t = seg_end;
      }
      if (!ok) {  // tear-down: wait for every MMA already issued
        tc_commit(&ctl.drain);
        mbar_wait_drain(&ctl.drain, 0);
      }
    }
  } else {
    // ------------------------------------------------ epilogue (warps 2-5)
    // a warp may only read TMEM lanes 32*(warp % 4) .. +31: that is its feature block
    const int ew = warp & 3;
    const int et = ew * 32 + lane;  // tile feature == TMEM lane
    // cluster exchange: the first contributor of the row tile this range ends in
    // expects its peers' partials (arrival count 1: this arrive; bytes may land first)
    bool csk_reducer = false;
    if (CSK && t_end > t_begin) {
      const int rt_last = (t_end - 1) / KT;
      const int cf = sk_cta_of(rt_last * KT, T, G), cl = sk_cta_of((rt_last + 1) * KT - 1, T, G);
      csk_reducer = cf == c && cl > c && cf / a.csk == cl / a.csk;
      if (csk_reducer && threadIdx.x == 64) {
        mbar_arrive_expect_tx(&ctl.recv, static_cast<uint32_t>((cl - cf) * kTileM * 16 * 4));
        ctl.recv_pending = 1;
      }
    }
    // the dry run overlaps the previous launch's tail; the real context follows
    // (ctx_early: the row plan is final before the wait, so the real context is
    // built there and the dry run uses it)
    if (a.ctx_early) {
      epi_prologue<EPI>(a, ectx, et);
      if (a.warm) epilogue_warmup<EPI, CSK>(a, ectx, ctl.red, stage, rms, c, G, et, recv, csk_reducer);
    } else if (a.warm) {
      epi_ctx_dry(ectx, a.n_pad, et);
      epilogue_warmup<EPI, CSK>(a, ectx, ctl.red, stage, rms, c, G, et, recv, csk_reducer);
    }
    pdl_wait();
    if constexpr (CSK) cluster_wait_acquire();
    if (threadIdx.x == 64) trace_at(trace, 13);
    if (a.rms) rms_prologue(a, rms, et);
    if (!a.ctx_early) epi_prologue<EPI>(a, ectx, et);
    int seg = 0;
    for (int t = t_begin; t < t_end; ++seg) {
      const int rt = t / KT;
      const int k0 = t - rt * KT;
      const int seg_end = min(t_end, (rt + 1) * KT);
      const int k1 = seg_end - rt * KT;
      const int buf = seg & 1;
      // one thread waits; the four epilogue warps follow (or stop) together
      if (threadIdx.x == 64)
        ctl.wait_ok = mbar_wait_bounded(&ctl.acc_full[buf], static_cast<uint32_t>(seg >> 1) & 1u,
                                        abort_flag, a.status)
                          ? 1
                          : 0;
      named_bar_sync(1, 128);
      const int ok = ctl.wait_ok;
      named_bar_sync(1, 128);
      if (!ok) break;
      tc_fence_after();
      epilogue_segment<EPI, CSK>(a, ectx, layout, acols, tmem_base, buf, seg, c, G, rt, k0, k1, stage, rms,
                       ctl.red, &ctl.reduce_flag, ctl.acc_empty, et, ew, lane, recv, &ctl.recv,
                       abort_flag, threadIdx.x == 64 ? trace : nullptr);
      t = seg_end;
    }
  }

  // a CTA that expects pushed partials leaves only after they landed (they do at
  // once unless a peer stopped early; the wait is bounded)
  if constexpr (CSK) {
    if (threadIdx.x == 64 && ctl.recv_pending) mbar_wait_drain(&ctl.recv, 0);
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem_base, tmem_cols);
  }
  if (threadIdx.x == 64) trace_at(trace, 1);
}

// The epilogue of the split row tiles of a GEMM launched with split_epi (at
// least 64 rows: one CTA folding every 16-row chunk of a tile in turn would
// hold the launch for tens of microseconds).  CTA (rt, chunk), 128 threads
// (thread = feature within the tile): if row tile rt had several contributors,
// sum their partials in ascending CTA order (the order of the in-kernel
// reduction) and run the epilogue for the chunk's 16 rows; row tiles owned by
// one CTA were finished by it.  gemm_grid: the GEMM's grid (its stream-K split).
template <int EPI>
__global__ void __launch_bounds__(128) gemm_split_epi_kernel(const __grid_constant__ GemmArgs a,
                                                             int gemm_grid) {
  __shared__ EpiCtx ectx;
  __shared__ float stage[kStageFloats];
  __shared__ float rms[kMaxRows];
  __shared__ float red[4][16];
  const int rt = blockIdx.x, chunk = blockIdx.y, et = threadIdx.x;
  const int KT = a.k_tiles, T = a.row_tiles * KT, G = gemm_grid;
  const int c_first = sk_cta_of(rt * KT, T, G), c_last = sk_cta_of((rt + 1) * KT - 1, T, G);
  // optional trace (a.trace: 16 slots per CTA, CTAs in launch order up to the
  // row's width): 0 entry, 13 dependency released, 2 partials summed, 3 context
  // built, 1 done
  const int lin = blockIdx.y * gridDim.x + blockIdx.x;
  unsigned long long* ts = (a.trace != nullptr && et == 0 && lin < a.trace_ctas) ? a.trace + lin * 16 : nullptr;
  trace_at(ts, 0);
  pdl_launch_dependents();
  if (c_first == c_last) return;
  pdl_wait();
  trace_at(ts, 13);
  float v[16];
  reduce_partials(a, rt, c_first, c_last, chunk, et, T, G, v);
  if (ts != nullptr) trace_after(ts, 2, v[0] + v[15]);
  if (a.rms) rms_chunk(a, rms, chunk, et);
  epi_prologue<EPI>(a, &ectx, et);
  trace_at(ts, 3);
  apply_epilogue<EPI>(a, &ectx, red, stage, rms, rt, chunk, et, v, nullptr, false);
  trace_at(ts, 1);
}

}  // namespace

// Shared-memory budget of the stage ring.  A deep ring keeps more weight bytes
// in flight per SM; a budget under ~110 KB lets the next kernel's CTA start on
// the same SM early (programmatic dependent launch).  MEMSPEC_GEMM_SMEM_KB
// overrides the default (for measurement).
static int gemm_budget_bytes(int n_pad) {
  static int env_kb = -1;
  if (env_kb < 0) {
    const char* e = std::getenv("MEMSPEC_GEMM_SMEM_KB");
    env_kb = e != nullptr ? std::atoi(e) : 0;
  }
  if (env_kb > 0) return env_kb * 1024;
  return n_pad <= 32 ? 200 * 1024 : 200 * 1024;
}

// Shared memory that receives the partials pushed by cluster peers: csk - 1
// slots of one 128 x 16 fp32 accumulator each.
static int csk_recv_bytes(int csk) { return csk > 1 ? (csk - 1) * kTileM * 16 * 4 + 16 : 0; }

int gemm_pick_stages(int n_pad, int planes, int csk) {
  const int stage = kABytes + n_pad * 128 * planes;
  const int budget = gemm_budget_bytes(n_pad);
  const int fixed = kTileM * kStagePitch * 4 + kMaxRows * 4 + static_cast<int>(sizeof(EpiCtx)) + 1024 +
                    csk_recv_bytes(csk);
  int s = (budget - fixed) / stage;
  if (s > kMaxStages) s = kMaxStages;
  if (s < 2) s = 2;
  return s;
}

size_t gemm_smem_bytes(int n_pad, int stages, int planes, int csk) {
  return static_cast<size_t>(stages) * (kABytes + n_pad * 128 * planes) + kTileM * kStagePitch * 4 +
         kMaxRows * 4 + sizeof(EpiCtx) + 1024 + csk_recv_bytes(csk);
}

cudaError_t gemm_set_max_smem() {
  // 227 KB per block minus the kernel's static shared memory
  const void* fns[8] = {reinterpret_cast<const void*>(gemm_stream_kernel<EPI_F32, false>),
                        reinterpret_cast<const void*>(gemm_stream_kernel<EPI_RESIDUAL, false>),
                        reinterpret_cast<const void*>(gemm_stream_kernel<EPI_SWIGLU, false>),
                        reinterpret_cast<const void*>(gemm_stream_kernel<EPI_QKV, false>),
                        reinterpret_cast<const void*>(gemm_stream_kernel<EPI_F32, true>),
                        reinterpret_cast<const void*>(gemm_stream_kernel<EPI_RESIDUAL, true>),
                        reinterpret_cast<const void*>(gemm_stream_kernel<EPI_SWIGLU, true>),
                        reinterpret_cast<const void*>(gemm_stream_kernel<EPI_QKV, true>)};
  for (const void* f : fns) {
    cudaError_t e = cudaFuncSetAttribute(f, cudaFuncAttributeMaxDynamicSharedMemorySize, 220 * 1024);
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

template <bool CSK>
static const void* gemm_kernel_for(int epi) {
  switch (epi) {
    case EPI_F32: return reinterpret_cast<const void*>(gemm_stream_kernel<EPI_F32, CSK>);
    case EPI_RESIDUAL: return reinterpret_cast<const void*>(gemm_stream_kernel<EPI_RESIDUAL, CSK>);
    case EPI_SWIGLU: return reinterpret_cast<const void*>(gemm_stream_kernel<EPI_SWIGLU, CSK>);
    case EPI_QKV: return reinterpret_cast<const void*>(gemm_stream_kernel<EPI_QKV, CSK>);
    default: return nullptr;
  }
}

int gemm_max_active_clusters(int epi, int csk, size_t smem) {
  const void* fn = gemm_kernel_for<true>(epi);
  if (fn == nullptr || csk < 2 || csk > 8) return 0;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(csk);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = smem;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = csk;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, fn, &cfg) != cudaSuccess) {
    (void)cudaGetLastError();
    return 0;
  }
  return n;
}

cudaError_t launch_gemm(const GemmArgs& a, int grid, size_t smem, cudaStream_t s, bool pdl) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  int n_attr = 0;
  if (pdl) {
    attr[n_attr].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[n_attr].val.programmaticStreamSerializationAllowed = 1;
    ++n_attr;
  }
  if (a.csk > 1) {
    if (a.csk > 8 || grid % a.csk != 0 || a.n_pad != 16) return cudaErrorInvalidValue;
    attr[n_attr].id = cudaLaunchAttributeClusterDimension;
    attr[n_attr].val.clusterDim.x = a.csk;
    attr[n_attr].val.clusterDim.y = 1;
    attr[n_attr].val.clusterDim.z = 1;
    ++n_attr;
  }
  cfg.attrs = attr;
  cfg.numAttrs = n_attr;
  if (a.csk > 1) {
    switch (a.epi) {
      case EPI_F32: return cudaLaunchKernelEx(&cfg, gemm_stream_kernel<EPI_F32, true>, a);
      case EPI_RESIDUAL: return cudaLaunchKernelEx(&cfg, gemm_stream_kernel<EPI_RESIDUAL, true>, a);
      case EPI_SWIGLU: return cudaLaunchKernelEx(&cfg, gemm_stream_kernel<EPI_SWIGLU, true>, a);
      case EPI_QKV: return cudaLaunchKernelEx(&cfg, gemm_stream_kernel<EPI_QKV, true>, a);
      default: return cudaErrorInvalidValue;
    }
  }
  switch (a.epi) {
    case EPI_F32: return cudaLaunchKernelEx(&cfg, gemm_stream_kernel<EPI_F32, false>, a);
    case EPI_RESIDUAL: return cudaLaunchKernelEx(&cfg, gemm_stream_kernel<EPI_RESIDUAL, false>, a);
    case EPI_SWIGLU: return cudaLaunchKernelEx(&cfg, gemm_stream_kernel<EPI_SWIGLU, false>, a);
    case EPI_QKV: return cudaLaunchKernelEx(&cfg, gemm_stream_kernel<EPI_QKV, false>, a);
    default: return cudaErrorInvalidValue;
  }
}

cudaError_t launch_gemm_split_epi(const GemmArgs& a, int gemm_grid, cudaStream_t s, bool pdl) {
  if (a.n_pad % 16 != 0 || a.n_pad > kMaxRows) return cudaErrorInvalidValue;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(a.row_tiles, a.n_pad / 16);
  cfg.blockDim = dim3(128);
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  switch (a.epi) {
    case EPI_F32: return cudaLaunchKernelEx(&cfg, gemm_split_epi_kernel<EPI_F32>, a, gemm_grid);
    case EPI_RESIDUAL: return cudaLaunchKernelEx(&cfg, gemm_split_epi_kernel<EPI_RESIDUAL>, a, gemm_grid);
    case EPI_SWIGLU: return cudaLaunchKernelEx(&cfg, gemm_split_epi_kernel<EPI_SWIGLU>, a, gemm_grid);
    case EPI_QKV: return cudaLaunchKernelEx(&cfg, gemm_split_epi_kernel<EPI_QKV>, a, gemm_grid);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace memspec
