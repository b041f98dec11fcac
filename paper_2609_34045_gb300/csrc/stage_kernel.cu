// Persistent stage kernel: a whole decode step of a stage (every block's Q/K/V, attention, O,
// gate/up and down, then lm_head) in one cooperative launch of one CTA per SM.
//
// A stage's cost is the time to stream its weights once (Kafila, section V-A, Eq. 2).  Split
// into one kernel per operation, every boundary drains the memory pipe: the launch, the ramp of
// the next kernel and the tail of the previous one.  Here the weights of every phase stream back
// to back through one TMA ring per SM, and only the consumers synchronise between phases:
//
//   warps 0-7  consumers: GEMV tiles, epilogues and attention units of each phase in turn; a
//              grid barrier (counter in global memory) separates a phase from its inputs
//   warp 8     weight producer: the tiles of every GEMV phase of this CTA, in order, into the
//              ring (cp.async.bulk), limited only by free stages, never by a grid barrier
//   warp 9     activation producer: after the grid barrier that makes a phase's input ready,
//              the matching activation chunks into the stages the weight producer armed
//
// While the consumers wait at a barrier or run attention, the weight producer keeps filling the
// ring with the next phase's tiles, so HBM stays busy across phase boundaries.  Every wait is
// bounded; a timeout sets the error word and a global abort flag that ends every other wait, so
// the kernel always returns.
#include "attn_core.cuh"
#include "gemv_core.cuh"

namespace kfl {

constexpr int MK_WARPS = CONSUMER_WARPS + 2;
constexpr int MK_THREADS = MK_WARPS * 32;

__device__ __forceinline__ unsigned ld_acquire(const unsigned *p) {
  unsigned v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

// Wait until the grid-barrier counter reaches `target` (bounded; false on timeout or abort).
__device__ bool grid_wait(const StageKernelParams &kp, unsigned target, volatile int *s_abort) {
  for (uint32_t i = 0; i < WAIT_LIMIT; ++i) {
    if (ld_acquire(kp.bar) >= target) return true;
    if (i >= 64) {
      if (*s_abort || *reinterpret_cast<volatile int *>(kp.abort_flag)) {
        *s_abort = 1;
        return false;
      }
      __nanosleep(i < 4096 ? 32 : 256);
    }
  }
  *s_abort = 1;
  atomicExch(kp.abort_flag, 1);
  atomicOr(kp.err, ERR_TIMEOUT);
  return false;
}

// Tile range of CTA c in a GEMV phase: stream-K over min(T, grid) CTAs; the rest get none.
__device__ __forceinline__ void phase_range(const GemvParams &g, int c, int grid, long long &T, int &G,
                                            long long &t0, int &n) {
  T = (long long)g.n_rb * g.n_kt;
  G = T < grid ? static_cast<int>(T) : grid;
  if (c >= G) {
    t0 = 0;
    n = 0;
    return;
  }
  t0 = (long long)c * T / G;
  n = static_cast<int>((long long)(c + 1) * T / G - t0);
}

// Phase bodies as separate (not inlined) functions: each gets its own register allocation, so
// the widest one does not raise the pressure of the rest of the kernel.
template <int B, int EPI, int FMT>
__device__ __noinline__ void gemv_phase(const GemvParams &g, uint8_t *ring, uint64_t *full, uint64_t *empty, int S,
                                        int &s, uint32_t &phase, long long t0, int n, long long T, int G, int c,
                                        float *red, float *scr, const float *inv, int *s_last, volatile int *abort_flag,
                                        int tid) {
  gemv_consume<B, EPI, FMT>(g, ring, full, empty, S, s, phase, t0, n, T, G, c, red, scr, inv, s_last, abort_flag,
                            tid);
}

template <int HD>
__device__ __noinline__ void attn_phase_unit(const AttnParams &a, int b, int kvh, int ch, int nc, uint8_t *att,
                                             int *s_last, int tid) {
  attn_unit<HD>(a, b, kvh, ch, nc, att, s_last, tid);
}

template <int B, int FMT>
__global__ void __maxnreg__(200) stage_kernel(const __grid_constant__ StageKernelParams kp) {
  extern __shared__ __align__(1024) uint8_t smem[];
  const int S = kp.stages;
  uint8_t *ring = smem;
  uint8_t *att = smem + (size_t)S * STAGE_BYTES;
  uint64_t *full = reinterpret_cast<uint64_t *>(att + kp.attn_bytes);
  uint64_t *empty = full + S;
  float *red = reinterpret_cast<float *>(empty + S);  // [RB][MAXB]
  float *scr = red + RB * MAXB;                       // 2 * CONSUMER_WARPS words
  volatile int *armed = reinterpret_cast<volatile int *>(scr + 2 * CONSUMER_WARPS);  // [S]
  __shared__ GemvParams s_gp;
  __shared__ AttnParams s_ap;
  __shared__ float s_inv[MAXB];
  __shared__ int s_last;
  __shared__ volatile int s_abort;
  __shared__ volatile int s_issued;

  constexpr int KTILE = FMT == 0 ? KT : KT4;
  constexpr uint32_t WBYTES = FMT == 0 ? TILE_BYTES : TILE4_BYTES;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int c = blockIdx.x, grid = gridDim.x;

  if (tid == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(smem_addr(&full[s]), 1);
      mbar_init(smem_addr(&empty[s]), CONSUMER_WARPS);
      armed[s] = -1;
    }
    s_abort = 0;
    s_issued = 0;
    fence_mbar_init();
  }
  __syncthreads();

  if (warp == CONSUMER_WARPS) {
    // -------------------------------------------------------------- weight producer
    if (lane == 0) {
      const uint64_t pol = policy_evict_first();
      const uint32_t bytes = WBYTES + B * (KTILE * 4);
      int s = 0, round = 0, gi = 0;
      for (int k = 0; k < kp.n_phases && !s_abort; ++k) {
        const Phase *ph = kp.phases + k;
        if (ph->kind != PH_GEMV) continue;
        long long T, t0;
        int G, n;
        phase_range(ph->g, c, grid, T, G, t0, n);
        const uint8_t *w = ph->g.w;
        for (int i = 0; i < n; ++i) {
          if (round > 0 && !consumer_wait(smem_addr(&empty[s]), (round & 1) ^ 1, &s_abort, kp.err)) break;
          const uint32_t fb = smem_addr(&full[s]);
          mbar_arrive_expect_tx(fb, bytes);
          bulk_g2s(smem_addr(ring + (size_t)s * STAGE_BYTES), w + (size_t)(t0 + i) * WBYTES, WBYTES, fb, pol);
          armed[s] = gi;
          s_issued = gi + 1;
          ++gi;
          if (++s == S) {
            s = 0;
            ++round;
          }
        }
      }
    }
    return;
  }
  if (warp == CONSUMER_WARPS + 1) {
    // ---------------------------------------------------------- activation producer
    if (lane == 0) {
      const uint64_t pol = policy_evict_last();
      int s = 0, gi = 0;
      for (int k = 0; k < kp.n_phases && !s_abort; ++k) {
        const Phase *ph = kp.phases + k;
        if (ph->kind != PH_GEMV) continue;
        long long T, t0;
        int G, n;
        phase_range(ph->g, c, grid, T, G, t0, n);
        if (n == 0) continue;
        if (k > 0) {
          if (!grid_wait(kp, (unsigned)k * grid, &s_abort)) break;
          // the activations were written by other CTAs' generic stores; order them before
          // this thread's bulk (async-proxy) reads
          asm volatile("fence.proxy.async.global;" ::: "memory");
        }
        const float *x = ph->g.x;
        const int ldx = ph->g.ldx, n_kt = ph->g.n_kt;
        int kt = static_cast<int>(t0 % n_kt);
        for (int i = 0; i < n; ++i) {
          bool ok = false;
          for (uint32_t it = 0; it < WAIT_LIMIT; ++it) {
            if (armed[s] == gi) {
              ok = true;
              break;
            }
            if (s_abort) break;
            if (it >= WAIT_FAST_SPINS) __nanosleep(64);
          }
          if (!ok) {
            if (!s_abort) {
              s_abort = 1;
              atomicExch(kp.abort_flag, 1);
              atomicOr(kp.err, ERR_TIMEOUT);
            }
            break;
          }
          const uint32_t fb = smem_addr(&full[s]);
          const uint32_t dst = smem_addr(ring + (size_t)s * STAGE_BYTES + WBYTES);
#pragma unroll
          for (int b = 0; b < B; ++b)
            bulk_g2s(dst + b * (KTILE * 4), x + (size_t)b * ldx + (size_t)kt * KTILE, KTILE * 4, fb, pol);
          ++gi;
          if (++s == S) s = 0;
          if (++kt == n_kt) kt = 0;
        }
      }
    }
    return;
  }

  // ------------------------------------------------------------------- consumers
  int s = 0;
  uint32_t phase = 0;
  for (int k = 0; k < kp.n_phases; ++k) {
    const Phase *ph = kp.phases + k;
    const int kind = ph->kind;
    if (tid == 0) {
      // the phase table is read-only: copy this phase's parameters before waiting
      if (kind == PH_GEMV)
        s_gp = ph->g;
      else
        s_ap = ph->a;
      if (k > 0) grid_wait(kp, (unsigned)k * grid, &s_abort);
    }
    consumer_sync();
    if (kind == PH_GEMV) {
      const GemvParams &g = s_gp;
      norm_scale<B>(g, s_inv, tid);
      consumer_sync();
      long long T, t0;
      int G, n;
      phase_range(g, c, grid, T, G, t0, n);
      switch (ph->epi) {
        case EPI_QKV:
          gemv_phase<B, EPI_QKV, FMT>(g, ring, full, empty, S, s, phase, t0, n, T, G, c, red, scr, s_inv, &s_last,
                                        &s_abort, tid);
          break;
        case EPI_RESID:
          gemv_phase<B, EPI_RESID, FMT>(g, ring, full, empty, S, s, phase, t0, n, T, G, c, red, scr, s_inv,
                                          &s_last, &s_abort, tid);
          break;
        case EPI_SWIGLU:
          gemv_phase<B, EPI_SWIGLU, FMT>(g, ring, full, empty, S, s, phase, t0, n, T, G, c, red, scr, s_inv,
                                           &s_last, &s_abort, tid);
          break;
        case EPI_ARGMAX:
          gemv_phase<B, EPI_ARGMAX, FMT>(g, ring, full, empty, S, s, phase, t0, n, T, G, c, red, scr, s_inv,
                                           &s_last, &s_abort, tid);
          break;
        default:
          gemv_phase<B, EPI_STORE, FMT>(g, ring, full, empty, S, s, phase, t0, n, T, G, c, red, scr, s_inv,
                                          &s_last, &s_abort, tid);
          break;
      }
    } else {
      const AttnParams &a = s_ap;
      // units (user, KV head, chunk), users in order; user b has n_kv_heads * nc_b units
      const int nc0 = attn_chunks(a, 0);
      const int nc1 = a.batch > 1 ? attn_chunks(a, 1) : 0;
      const int nc2 = a.batch > 2 ? attn_chunks(a, 2) : 0;
      const int nc3 = a.batch > 3 ? attn_chunks(a, 3) : 0;
      const int hk = a.n_kv_heads;
      const int units = (nc0 + nc1 + nc2 + nc3) * hk;
      for (int u = c; u < units; u += grid) {
        int rem = u, b = 0, ncb = nc0;
        if (rem >= nc0 * hk) {
          rem -= nc0 * hk;
          b = 1;
          ncb = nc1;
          if (rem >= nc1 * hk) {
            rem -= nc1 * hk;
            b = 2;
            ncb = nc2;
            if (rem >= nc2 * hk) {
              rem -= nc2 * hk;
              b = 3;
              ncb = nc3;
            }
          }
        }
        const int kvh = rem / ncb, ch = rem % ncb;
        if (kp.head_dim == 128)
          attn_phase_unit<128>(a, b, kvh, ch, ncb, att, &s_last, tid);
        else
          attn_phase_unit<64>(a, b, kvh, ch, ncb, att, &s_last, tid);
        consumer_sync();
      }
    }
    // this CTA's part of phase k is written: arrive at the grid barrier
    consumer_sync();
    if (tid == 0) {
      __threadfence();
      atomicAdd(kp.bar, 1u);
    }
  }

  if (s_abort && tid == 0) {
    // drain copies still in flight before the CTA's shared memory goes away (bounded)
    const int issued = s_issued;
    for (int i = (issued > S ? issued - S : 0); i < issued; ++i) mbar_wait(smem_addr(&full[i % S]), (i / S) & 1);
  }
}

// ------------------------------------------------------------------------------- launch
size_t stage_kernel_smem(int stages, int head_dim) {
  const size_t att = head_dim == 128 ? AttnLayout<128>::BYTES : AttnLayout<64>::BYTES;
  return (size_t)stages * STAGE_BYTES + att + 2 * stages * sizeof(uint64_t) +
         (RB * MAXB + 2 * CONSUMER_WARPS) * sizeof(float) + stages * sizeof(int);
}

int stage_kernel_attn_bytes(int head_dim) { return head_dim == 128 ? AttnLayout<128>::BYTES : AttnLayout<64>::BYTES; }

template <int B, int FMT>
static cudaError_t prepare_one_stage(size_t smem) {
  return cudaFuncSetAttribute(stage_kernel<B, FMT>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
}

cudaError_t prepare_stage_kernel(size_t smem) {
  cudaError_t e;
  if ((e = prepare_one_stage<1, 0>(smem)) != cudaSuccess) return e;
  if ((e = prepare_one_stage<2, 0>(smem)) != cudaSuccess) return e;
  if ((e = prepare_one_stage<3, 0>(smem)) != cudaSuccess) return e;
  if ((e = prepare_one_stage<4, 0>(smem)) != cudaSuccess) return e;
  if ((e = prepare_one_stage<1, 1>(smem)) != cudaSuccess) return e;
  if ((e = prepare_one_stage<2, 1>(smem)) != cudaSuccess) return e;
  if ((e = prepare_one_stage<3, 1>(smem)) != cudaSuccess) return e;
  return prepare_one_stage<4, 1>(smem);
}

template <int B, int FMT>
static cudaError_t launch_stage_one(const StageKernelParams &kp, int grid, size_t smem, cudaStream_t s) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(MK_THREADS);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeCooperative;
  attr[0].val.cooperative = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, stage_kernel<B, FMT>, kp);
}

cudaError_t launch_stage_kernel(const StageKernelParams &kp, int batch, int fmt, int grid, size_t smem,
                                cudaStream_t s) {
  if (kp.stages < 2 || kp.stages > MAX_STAGES) return cudaErrorInvalidValue;
  if (fmt == 0) {
    switch (batch) {
      case 1: return launch_stage_one<1, 0>(kp, grid, smem, s);
      case 2: return launch_stage_one<2, 0>(kp, grid, smem, s);
      case 3: return launch_stage_one<3, 0>(kp, grid, smem, s);
      case 4: return launch_stage_one<4, 0>(kp, grid, smem, s);
    }
  } else {
    switch (batch) {
      case 1: return launch_stage_one<1, 1>(kp, grid, smem, s);
      case 2: return launch_stage_one<2, 1>(kp, grid, smem, s);
      case 3: return launch_stage_one<3, 1>(kp, grid, smem, s);
      case 4: return launch_stage_one<4, 1>(kp, grid, smem, s);
    }
  }
  return cudaErrorInvalidValue;
}

}  // namespace kfl
