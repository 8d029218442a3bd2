// pass.cu - persistent kernel that runs a whole forward pass (the verify pass,
// or all K passes of a draft step) as one launch.
//
// At batch 1 every op of a pass is short (a 33 MB projection streams in ~5 us)
// and separate launches pay a launch, a pipeline fill and a split-K tail each.
// Here one CTA per SM walks the op list of the pass in order:
//
//   warp 0      weight producer: TMA loads of weight tiles into the stage ring.
//               Weights never depend on earlier ops, so it runs ahead across op
//               boundaries and through attention, limited only by free stages;
//   warp 6      activation producer: TMA loads of activation tiles, issued
//               once the op that writes them has completed on every CTA;
//   warp 1      MMA issuer (tcgen05.mma into double-buffered TMEM accumulators);
//   warps 2-5   workers: GEMM epilogues (and split-K reductions), attention,
//               embedding, sampling, acceptance.
//
// Completion of op n is a counter done[n] that every CTA increments once it has
// finished its share of op n (all of its epilogue writes); consumers wait until
// it reaches the grid size.  All CTAs are co-resident (one per SM, cooperative
// launch), every wait is bounded, and the last CTA to leave resets the counters
// for the next launch.
#include "attn_body.cuh"
#include "embed_body.cuh"
#include "gemm_epi.cuh"
#include "internal.h"
#include "pass.h"
#include "ptx.cuh"
#include "sample_body.cuh"

namespace memspec {

namespace {

using namespace gemm;

constexpr int kThreads = 224;
constexpr int kWorkerBar = 1;   // named barrier of the 128 worker threads

struct PassCtl {
  uint64_t full_a[kMaxStages];
  uint64_t full_b[kMaxStages];
  uint64_t empty[kMaxStages];
  uint64_t acc_full[2];
  uint64_t acc_empty[2];
  uint64_t drain;
  uint32_t tmem_base;
  int abort_flag;
  int reduce_flag;
  int wait_ok;
  int ops_ready;     // highest op whose inputs are complete (workers -> producer)
  float red[4][16];
  float red8[8];
};

// Completion counters are polled with relaxed loads (they read L2 and leave the
// SM's L1 alone); one acquire fence follows the successful poll.
__device__ __forceinline__ int ld_relaxed(const int* p) {
  int v;
  asm volatile("ld.relaxed.gpu.global.s32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

// Bounded wait until done[n] reaches `target`; false on timeout or abort.
__device__ bool wait_done(const int* done, int n, int target, volatile int* abort_flag,
                          uint32_t* status) {
  if (ld_relaxed(done + n) < target) {
    const long long t0 = clock64();
    while (ld_relaxed(done + n) < target) {
      if (*abort_flag) return false;
      if (clock64() - t0 > kWaitBudgetCycles) {
        *abort_flag = 1;
        atomicOr(status, 0x1u);
        return false;
      }
      __nanosleep(32);
    }
  }
  asm volatile("fence.acq_rel.gpu;" ::: "memory");
  return true;
}

// The worker group tells the activation producer of its own CTA that op n may
// start (ops_ready = n) once it has observed done[n - 1]: one poller per CTA.
__device__ __forceinline__ void publish_ready(volatile int* ops_ready, int n) {
  __threadfence_block();
  *ops_ready = n;
}

// Bounded wait of the activation producer until ops_ready >= n.
__device__ bool wait_ready(volatile int* ops_ready, int n, volatile int* abort_flag,
                           uint32_t* status) {
  if (*ops_ready < n) {
    const long long t0 = clock64();
    while (*ops_ready < n) {
      if (*abort_flag) return false;
      if (clock64() - t0 > kWaitBudgetCycles) {
        *abort_flag = 1;
        atomicOr(status, 0x1u);
        return false;
      }
      __nanosleep(32);
    }
  }
  __threadfence_block();
  return true;
}

// Trace slot of (op n, this CTA, event e), or nullptr when tracing is off.
__device__ __forceinline__ unsigned long long* trace_slot(const PassArgs& p, int n, int e) {
  if (p.trace == nullptr || n >= kPassTraceOps) return nullptr;
  return p.trace + 2 + (static_cast<size_t>(n) * gridDim.x + blockIdx.x) * kPassTraceSlots + e;
}

__device__ __forceinline__ void fence_proxy_async_global() {
  asm volatile("fence.proxy.async.global;" ::: "memory");
}

__device__ __forceinline__ int op_layout(const GemmArgs& a) {
  return !a.split ? kPlain : (2 * a.n_pad <= 256 ? kWide : kTwice);
}

__global__ void __launch_bounds__(kThreads, 1) pass_kernel(const __grid_constant__ PassArgs p) {
  __shared__ PassCtl ctl;
  extern __shared__ uint8_t dsmem_raw[];
  uint8_t* dsmem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(dsmem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  const int S = p.stages;
  uint8_t* ring_a = dsmem;
  uint8_t* ring_b = ring_a + static_cast<size_t>(S) * kABytes;
  uint8_t* attn_smem = ring_b + static_cast<size_t>(S) * p.b_stage_bytes;
  float* stage = reinterpret_cast<float*>(attn_smem + p.attn_bytes);
  float* rms = stage + kStageFloats;
  EpiCtx* ectx = reinterpret_cast<EpiCtx*>(rms + kMaxRows);
  smp::SampleSmem* ssm = reinterpret_cast<smp::SampleSmem*>(ectx + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int G = gridDim.x, c = blockIdx.x;
  volatile int* abort_flag = &ctl.abort_flag;

  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(&ctl.full_a[s], 1);
      mbar_init(&ctl.full_b[s], 1);
      mbar_init(&ctl.empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&ctl.acc_full[b], 1);
      mbar_init(&ctl.acc_empty[b], 4);
    }
    mbar_init(&ctl.drain, 1);
    ctl.abort_flag = 0;
    ctl.reduce_flag = 0;
    ctl.ops_ready = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    __syncwarp();
    tmem_alloc(&ctl.tmem_base, p.tmem_cols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = ctl.tmem_base;

  if (warp == 0 || warp == 6) {
    // ---------------------------------------------------- TMA producers
    if (lane == 0) {
      const bool weights = warp == 0;
      const uint64_t pol_w = l2_policy_evict_first();
      const uint64_t pol_b = l2_policy_evict_last();
      uint32_t issued = 0, last_par = 0;
      int s = 0;                // ring position of the next tile (incremental: no division)
      uint32_t ph = 0;
      bool ok = true;
      for (int n = 0; n < p.n_ops && ok; ++n) {
        const PassOp& op = p.ops[n];
        if (op.type != OP_GEMM) continue;
        const GemmArgs& a = op.u.g;
        const int Gn = op.grid;
        if (c >= Gn) continue;
        const int T = a.row_tiles * a.k_tiles, KT = a.k_tiles;
        const int t_begin = sk_begin(c, T, Gn), t_end = sk_begin(c + 1, T, Gn);
        const int plane_bytes = a.n_pad * 128;
        int rt = t_begin / KT, kt = t_begin - rt * KT;
        if (!weights) {
          // activations are written by op n-1 (and earlier): wait until it completed
          if (n > 0 && !wait_ready(&ctl.ops_ready, n, abort_flag, p.status)) {
            ok = false;
            break;
          }
          fence_proxy_async_global();
          if (unsigned long long* ts = trace_slot(p, n, 2)) *ts = global_ns();
        }
        for (int t = t_begin; t < t_end; ++t) {
          if (!mbar_wait_bounded(&ctl.empty[s], ph ^ 1u, abort_flag, p.status)) {
            ok = false;
            break;
          }
          if (weights) {
            uint8_t* dst = ring_a + static_cast<size_t>(s) * kABytes;
            mbar_arrive_expect_tx(&ctl.full_a[s], kABytes);
            if (a.a_packed != nullptr) {
              bulk_load(dst, a.a_packed + static_cast<size_t>(t) * kABytes, kABytes, &ctl.full_a[s],
                        pol_w);
            } else if (a.pair) {
              tma_load_2d(dst, &a.map_a, kt * kTileK, rt * 64, &ctl.full_a[s], pol_w);
              tma_load_2d(dst + kABytes / 2, &a.map_a2, kt * kTileK, rt * 64, &ctl.full_a[s], pol_w);
            } else {
              tma_load_2d(dst, &a.map_a, kt * kTileK, rt * kTileM, &ctl.full_a[s], pol_w);
            }
          } else {
            uint8_t* dst = ring_b + static_cast<size_t>(s) * p.b_stage_bytes;
            mbar_arrive_expect_tx(&ctl.full_b[s], plane_bytes * (a.split ? 2 : 1));
            tma_load_2d(dst, &a.map_b, kt * kTileK, 0, &ctl.full_b[s], pol_b);
            if (a.split) tma_load_2d(dst + plane_bytes, &a.map_b2, kt * kTileK, 0, &ctl.full_b[s], pol_b);
          }
          issued |= 1u << s;
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
      }
      if (!ok) {   // tear-down: let the copies in flight land before exit
        for (int s = 0; s < S; ++s)
          if (issued & (1u << s))
            mbar_wait_drain(weights ? &ctl.full_a[s] : &ctl.full_b[s], (last_par >> s) & 1u);
      }
    }
  } else if (warp == 1) {
    // ---------------------------------------------------- MMA issuer
    if (lane == 0) {
      int seg = 0, s = 0;
      uint32_t ph = 0;
      bool ok = true;
      const uint64_t adesc0 = make_smem_desc_sw128(smem_addr(ring_a));
      const uint64_t bdesc0 = make_smem_desc_sw128(smem_addr(ring_b));
      const uint32_t a_step = kABytes >> 4, b_step = static_cast<uint32_t>(p.b_stage_bytes) >> 4;
      for (int n = 0; n < p.n_ops && ok; ++n) {
        const PassOp& op = p.ops[n];
        if (op.type != OP_GEMM) continue;
        const GemmArgs& a = op.u.g;
        const int Gn = op.grid;
        if (c >= Gn) continue;
        const int T = a.row_tiles * a.k_tiles, KT = a.k_tiles;
        const int t_begin = sk_begin(c, T, Gn), t_end = sk_begin(c + 1, T, Gn);
        const int layout = op_layout(a);
        const int acols = acc_cols(a, layout);
        const int plane_bytes = a.n_pad * 128;
        const uint32_t idesc = make_idesc_bf16_f32(kTileM, layout == kWide ? 2 * a.n_pad : a.n_pad);
        unsigned long long* ts_mma = trace_slot(p, n, 3);
        for (int t = t_begin; t < t_end && ok; ++seg) {
          const int rt = t / KT;
          const int seg_end = min(t_end, (rt + 1) * KT);
          const int buf = seg & 1;
          if (seg >= 2 &&
              !mbar_wait_bounded(&ctl.acc_empty[buf], static_cast<uint32_t>((seg >> 1) - 1) & 1u,
                                 abort_flag, p.status)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t d_tmem = tmem_base + static_cast<uint32_t>(buf * acols);
          const uint32_t p_step = static_cast<uint32_t>(plane_bytes) >> 4;
          for (int tt = t; tt < seg_end; ++tt) {
            if (!mbar_wait_bounded(&ctl.full_a[s], ph, abort_flag, p.status) ||
                !mbar_wait_bounded(&ctl.full_b[s], ph, abort_flag, p.status)) {
              ok = false;
              break;
            }
            if (ts_mma != nullptr) {
              *ts_mma = global_ns();
              ts_mma = nullptr;
            }
            tc_fence_after();
            const uint64_t ad = adesc0 + static_cast<uint32_t>(s) * a_step;
            const uint64_t bd = bdesc0 + static_cast<uint32_t>(s) * b_step;
            const uint32_t acc0 = tt > t ? 1u : 0u;
            if (layout != kTwice) {
#pragma unroll
              for (int kk = 0; kk < kTileK / 16; ++kk)
                tc_mma_bf16(d_tmem, ad + 2 * kk, bd + 2 * kk, idesc, kk > 0 ? 1u : acc0);
            } else {
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
      }
      if (!ok) {
        tc_commit(&ctl.drain);
        mbar_wait_drain(&ctl.drain, 0);
      }
    }
  } else {
    // ---------------------------------------------------- workers (warps 2-5)
    const int ew = warp & 3;
    const int et = ew * 32 + lane;        // GEMM: tile feature == TMEM lane
    const int tid = threadIdx.x - 64;     // 0..127 for the other bodies
    auto wsync = [] { named_bar_sync(kWorkerBar, 128); };
    int seg = 0;
    bool ok = true;
    for (int n = 0; n < p.n_ops && ok; ++n) {
      const PassOp& op = p.ops[n];
      if (n > 0) {   // everything this op reads was written by op n-1 or earlier
        if (tid == 0) {
          const bool ok_n = wait_done(p.done, n - 1, G, abort_flag, p.status);
          ctl.wait_ok = ok_n ? 1 : 0;
          if (ok_n) publish_ready(&ctl.ops_ready, n);
        }
        wsync();
        const int wok = ctl.wait_ok;
        wsync();
        if (!wok) {
          ok = false;
          break;
        }
      }
      if (tid == 0)
        if (unsigned long long* ts = trace_slot(p, n, 0)) *ts = global_ns();
      if (op.type == OP_EMBED) {
        for (int r = c; r < op.n_units; r += G) emb::embed_row<128>(op.u.e, r, ctl.red8, tid, wsync);
      } else if (op.type == OP_GEMM) {
        const GemmArgs& a = op.u.g;
        const int Gn = op.grid;
        if (c < Gn) {
          const int T = a.row_tiles * a.k_tiles, KT = a.k_tiles;
          const int t_begin = sk_begin(c, T, Gn), t_end = sk_begin(c + 1, T, Gn);
          const int layout = op_layout(a);
          const int acols = acc_cols(a, layout);
          if (a.rms) rms_prologue(a, rms, et);
          switch (a.epi) {
            case EPI_F32: epi_prologue<EPI_F32>(a, ectx, et); break;
            case EPI_RESIDUAL: epi_prologue<EPI_RESIDUAL>(a, ectx, et); break;
            case EPI_SWIGLU: epi_prologue<EPI_SWIGLU>(a, ectx, et); break;
            default: epi_prologue<EPI_QKV>(a, ectx, et); break;
          }
          int lseg = 0;   // segment index within this op (partial slot choice)
          for (int t = t_begin; t < t_end; ++seg, ++lseg) {
            const int rt = t / KT;
            const int k0 = t - rt * KT;
            const int seg_end = min(t_end, (rt + 1) * KT);
            const int k1 = seg_end - rt * KT;
            const int buf = seg & 1;
            // one thread waits; the four warps follow (or stop) together
            if (tid == 0)
              ctl.wait_ok = mbar_wait_bounded(&ctl.acc_full[buf], static_cast<uint32_t>(seg >> 1) & 1u,
                                              abort_flag, p.status)
                                ? 1
                                : 0;
            wsync();
            const int wok = ctl.wait_ok;
            wsync();
            if (!wok) {
              ok = false;
              break;
            }
            tc_fence_after();
            unsigned long long* ts = tid == 0 ? trace_slot(p, n, 0) : nullptr;
#define MEMSPEC_PASS_EPI(E)                                                                  \
  epilogue_segment<E, false>(a, ectx, layout, acols, tmem_base, buf, lseg, c, Gn, rt, k0, k1, stage, rms, \
                      ctl.red, &ctl.reduce_flag, ctl.acc_empty, et, ew, lane, nullptr, nullptr, \
                      nullptr, ts)
            switch (a.epi) {
              case EPI_F32: MEMSPEC_PASS_EPI(EPI_F32); break;
              case EPI_RESIDUAL: MEMSPEC_PASS_EPI(EPI_RESIDUAL); break;
              case EPI_SWIGLU: MEMSPEC_PASS_EPI(EPI_SWIGLU); break;
              default: MEMSPEC_PASS_EPI(EPI_QKV); break;
            }
#undef MEMSPEC_PASS_EPI
            t = seg_end;
          }
        }
      } else if (op.type == OP_ATTN) {
        const AttnArgs& at = op.u.at;
        const int per_group = at.n_splits * at.Hkv * at.row_blocks;
        for (int u = c; u < op.n_units; u += G) {
          const int g = u / per_group;
          const int rem = u - g * per_group;
          const int kr = rem / at.n_splits, split = rem - kr * at.n_splits;
          const int kvh = kr / at.row_blocks, rb = kr - kvh * at.row_blocks;
          if (at.hd == 64)
            attn::attention_cta<64>(at, g, kvh, rb, split, attn_smem, tid, wsync, [] {}, false,
                                    tid == 0 ? trace_slot(p, n, 0) : nullptr);
          else
            attn::attention_cta<128>(at, g, kvh, rb, split, attn_smem, tid, wsync, [] {}, false,
                                     tid == 0 ? trace_slot(p, n, 0) : nullptr);
          wsync();
        }
      } else if (op.type == OP_SAMPLE) {
        for (int g = c; g < op.n_units; g += G) smp::sample_group<128>(op.u.s, g, *ssm, tid, wsync);
      } else if (op.type == OP_ACCEPT) {
        const int rows = 2 * op.u.acc.K + 1;
        for (int u = c; u < op.n_units; u += G)
          smp::accept_row<128>(op.u.acc, u % rows, u / rows, *ssm, tid, wsync);
      }
      wsync();
      if (!ok) break;
      if (tid == 0) {
        if (unsigned long long* ts = trace_slot(p, n, 1)) *ts = global_ns();
        __threadfence();
        atomicAdd(p.done + n, 1);
      }
    }
  }

  // ---------------------------------------------------- exit
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem_base, p.tmem_cols);
  }
  if (threadIdx.x == 0) {
    __threadfence();
    // every CTA has finished all of its waits once it gets here: the last one
    // resets the completion counters for the next launch
    if (atomicAdd(p.exit_cnt, 1) == G - 1) {
      if (p.trace != nullptr) {
        p.trace[0] = static_cast<unsigned long long>(p.n_ops);
        p.trace[1] = static_cast<unsigned long long>(G);
      }
      for (int n = 0; n < p.n_ops; ++n) p.done[n] = 0;
      __threadfence();
      *p.exit_cnt = 0;
    }
  }
}

}  // namespace

size_t pass_smem_bytes(const PassArgs& p) {
  return static_cast<size_t>(p.stages) * (kABytes + p.b_stage_bytes) + p.attn_bytes +
         kStageFloats * 4 + kMaxRows * 4 + sizeof(EpiCtx) + sizeof(smp::SampleSmem) + 1024;
}

int pass_pick_stages(int b_stage_bytes, int attn_bytes) {
  const int budget = 226 * 1024 - attn_bytes - kStageFloats * 4 - kMaxRows * 4 -
                     static_cast<int>(sizeof(EpiCtx)) -
                     static_cast<int>(sizeof(smp::SampleSmem)) - 1024 - 1024;
  int s = budget / (kABytes + b_stage_bytes);
  if (s > kMaxStages) s = kMaxStages;
  return s;
}

size_t pass_attn_bytes(int hd) {
  return hd == 64 ? attn::attention_smem_bytes_hd<64>() : attn::attention_smem_bytes_hd<128>();
}

cudaError_t pass_set_max_smem() {
  return cudaFuncSetAttribute(pass_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, 226 * 1024);
}

cudaError_t launch_pass(const PassArgs& p, int grid, cudaStream_t s, bool cooperative) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = pass_smem_bytes(p);
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeCooperative;
  attr[0].val.cooperative = 1;
  cfg.attrs = attr;
  cfg.numAttrs = cooperative ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, pass_kernel, p);
}

}  // namespace memspec
