// Persistent stage kernel: a whole decode step of a stage (every block's Q/K/V, attention, O,
// gate/up and down, then lm_head) in one cooperative launch of one CTA per SM.
//
// A stage's cost is the time to stream its weights once (Kafila, section V-A, Eq. 2).  Split
// into one kernel per operation, every boundary drains the memory pipe: the launch, the ramp of
// the next kernel and the tail of the previous one.  Here the weights of every phase stream back
// to back through one TMA ring per SM, and phases overlap as far as the data allows:
//
//   warps 0-7  consumers: GEMV tiles, epilogues and attention units of each phase in turn;
//              every finished piece of output is published on a readiness counter in global
//              memory (release), per activation chunk, per KV head, and per phase
//   warp 8     weight producer (one thread): the weight tiles of every GEMV phase of this CTA,
//              in order, into the ring (cp.async.bulk) as soon as a stage is free; weights
//              never wait for data, so HBM keeps streaming while the consumers wait
//   warp 9     activation producer: for each tile, once the counters of its activation chunk
//              say the producing phase has written it (polled a warp at a time, 32 chunks per
//              L2 round trip), the chunk into the stage the weight producer armed
//
// There is no grid-wide barrier: a CTA starts the next phase's tiles as soon as their inputs
// exist, so the tail of one phase overlaps the start of the next.  Every wait is bounded; a
// timeout sets the error word and a global abort flag that ends every other wait, so the kernel
// always returns.
#include "attn_core.cuh"
#include "gemv_core.cuh"

namespace kfl {

constexpr int MK_WARPS = CONSUMER_WARPS + 3;  // consumers, weight producer, activation producer, epilogue
constexpr int MK_THREADS = MK_WARPS * 32;

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

// Is activation chunk kt of a GEMV phase written?  (acquire loads of the producers' counters)
__device__ __forceinline__ bool chunk_ready(const GemvParams &g, int kt) {
  if (g.in_kind == 1) {
    const int kk = tile_k(g.fmt);
    const int len = min(kk, g.in_len - kt * kk);
    const unsigned need = (unsigned)((len + g.in_unit - 1) / g.in_unit);
    return ld_acquire_gpu(g.in_ready + kt) >= need;
  }
  if (g.in_kind == 2) {
    const int kk = tile_k(g.fmt);
    const int h0 = (kt * kk) / g.in_head_dim;
    const int h1 = min(((kt + 1) * kk - 1) / g.in_head_dim, g.in_len / g.in_head_dim - 1);
    for (int kvh = h0 / g.in_group; kvh <= h1 / g.in_group; ++kvh)
      if (ld_acquire_gpu(g.in_ready + kvh) < (unsigned)g.in_need) return false;
    return true;
  }
  return true;
}

// Phase bodies as separate (not inlined) functions get their own register allocation, so the
// widest one does not raise the pressure of the rest of the kernel.
template <int B, int FMT>
__device__ __noinline__ void gemv_consume_call(int n_kt, uint8_t *ring, uint64_t *full, uint64_t *empty, int S,
                                               int &s, uint32_t &phase, long long t0, int n, const SegRing &sr,
                                               int &segc, volatile int *abort_flag, unsigned *err, int tid,
                                               bool xsplit) {
  gemv_consume<B, FMT>(n_kt, ring, full, empty, S, s, phase, t0, n, sr, segc, abort_flag, err, tid, xsplit);
}

template <int B>
__device__ __noinline__ void gemv_epilogues_call(int epi, const GemvParams &p, long long t0, int n, long long T, int G,
                                                 int c, const SegRing &sr, int &segc, float *inv, bool &inv_ready,
                                                 volatile int *abort_flag, int lane) {
  gemv_epilogues_any<B>(epi, p, t0, n, T, G, c, sr, segc, inv, inv_ready, abort_flag, lane);
}

template <int HD>
__device__ __noinline__ void attn_phase_unit(const AttnParams &a, int b, int kvh, int ch, int nc, uint8_t *att,
                                             int *s_last, int tid, int prefetched) {
  attn_unit<HD, 1>(a, b, kvh, ch, nc, att, s_last, tid, prefetched);
}

template <int B, int FMT>
__global__ void __launch_bounds__(MK_THREADS, 1) stage_kernel(const __grid_constant__ StageKernelParams kp) {
  extern __shared__ __align__(1024) uint8_t smem[];
  constexpr int SB = stage_bytes(B, FMT);
  const int S = kp.stages;
  uint8_t *ring = smem;
  uint8_t *att = smem + (size_t)S * SB;
  uint64_t *full = reinterpret_cast<uint64_t *>(att + kp.attn_bytes);
  uint64_t *empty = full + S;
  uint64_t *armed = empty + S;                        // weight tile issued (for the x producer)
  uint64_t *seg_full = armed + S;                     // staged segments (consumers -> epilogue)
  uint64_t *seg_empty = seg_full + NSLOT;
  // staging slots (SegRing: seg_floats(FMT) floats), 128-byte aligned (read as float4)
  float *red = reinterpret_cast<float *>((reinterpret_cast<uintptr_t>(seg_empty + NSLOT) + 127) & ~uintptr_t(127));
  __shared__ GemvParams s_egp;  // the epilogue warp's copy of the current GEMV's parameters
  __shared__ AttnParams s_ap;
  __shared__ float s_inv[MAXB];
  __shared__ int s_last;
  __shared__ volatile int s_abort;
  __shared__ volatile int s_issued;
  __shared__ int s_pos[MAXB];                           // this step's positions
  __shared__ float s_cos[MAXB * 64], s_sin[MAXB * 64];  // their RoPE rows

  constexpr int KTILE = FMT == 0 ? KT : KT4;
  constexpr uint32_t WBYTES = FMT == 0 ? TILE_BYTES : TILE4_BYTES;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int c = blockIdx.x, grid = gridDim.x;
  const SegRing sr = {red, seg_full, seg_empty, seg_slots(FMT), seg_subs(FMT)};
  auto stamp = [&](int k, int slot) {
    if (kp.trace) kp.trace[((size_t)k * grid + c) * TRACE_SLOTS + slot] = global_ns();
  };

  if (tid == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(smem_addr(&full[s]), 1);
      mbar_init(smem_addr(&empty[s]), ring_empty_count(FMT));
      mbar_init(smem_addr(&armed[s]), 1);
    }
    for (int s = 0; s < NSLOT; ++s) {
      mbar_init(smem_addr(&seg_full[s]), CONSUMER_WARPS);
      mbar_init(smem_addr(&seg_empty[s]), 1);
    }
    s_abort = 0;
    s_issued = 0;
    fence_mbar_init();
  }
  {
    // positions never change during the step: keep them and their RoPE rows in shared memory
    const int half = kp.head_dim / 2;
    for (int e = tid; e < B * half; e += MK_THREADS) {
      const int b = e / half, i = e % half;
      int pos = kp.positions[b];
      if (pos < 0 || pos >= kp.max_ctx) pos = 0;
      s_cos[e] = kp.rope_cos[(size_t)pos * half + i];
      s_sin[e] = kp.rope_sin[(size_t)pos * half + i];
    }
    if (tid < MAXB) s_pos[tid] = tid < B ? kp.positions[tid] : 0;
  }
  for (int e = tid; e < seg_floats(FMT); e += MK_THREADS) red[e] = 0.f;  // int4 tiles add into it
  __syncthreads();

  if (warp == CONSUMER_WARPS + 2) {
    // ------------------------------------------------------------- epilogue warp
    int segc = 0;
    for (int k = 0; k < kp.n_phases && !s_abort; ++k) {
      const Phase *ph = kp.phases + k;
      if (ph->kind != PH_GEMV) continue;
      long long T, t0;
      int G, n;
      phase_range(ph->g, c, grid, T, G, t0, n);
      if (n == 0) continue;
      if (lane == 0) {
        s_egp = ph->g;
        s_egp.positions = s_pos;
        if (s_egp.rope_cos) {
          s_egp.rope_cos = s_cos;
          s_egp.rope_sin = s_sin;
          s_egp.rope_per_user = 1;
        }
      }
      __syncwarp();
      bool inv_ready = false;
      gemv_epilogues_call<B>(ph->epi, s_egp, t0, n, T, G, c, sr, segc, s_inv, inv_ready, &s_abort, lane);
      __syncwarp();
      if (lane == 0) stamp(k, TR_CONS_DONE);
    }
    return;
  }
  if (warp == CONSUMER_WARPS) {
    // ---------------------------------------------------------- weight producer
    // Two cursors over this CTA's weight tiles of every GEMV phase, in order: the ring cursor
    // loads a tile into a free stage; the L2 cursor, l2_ahead tiles in front of it, prefetches
    // tiles into L2, so HBM keeps streaming while the consumers wait on data (phase tails,
    // attention) and the ring loads then hit L2.
    if (lane == 0) {
      const uint64_t pol_ring = policy_evict_first();
      const uint64_t pol_l2 = policy_evict_normal();
      struct Cursor {
        int k, i, n;
        long long t0;
        const uint8_t *w;
        uint32_t bytes;  // a stage's copies: the tile and its activations
      };
      auto seek = [&](Cursor &cu, int from) {
        for (int k = from; k < kp.n_phases; ++k) {
          const Phase *ph = kp.phases + k;
          if (ph->kind != PH_GEMV) continue;
          long long T, t0;
          int G, n;
          phase_range(ph->g, c, grid, T, G, t0, n);
          if (n == 0) continue;
          cu.k = k;
          cu.i = 0;
          cu.n = n;
          cu.t0 = t0;
          cu.w = ph->g.w;
          cu.bytes = WBYTES + (FMT == 0 ? B * (KTILE * 4) : act16_copy_bytes(B, ph->g.xsplit));
          return;
        }
        cu.k = kp.n_phases;
      };
      Cursor cr, cp;
      seek(cr, 0);
      cp = cr;
      int ahead = 0;  // tiles the L2 cursor is in front of the ring cursor
      auto prefetch_up_to = [&](int want) {
        while (ahead < want && cp.k < kp.n_phases) {
          bulk_prefetch_l2(cp.w + (size_t)(cp.t0 + cp.i) * WBYTES, WBYTES, pol_l2);
          ++ahead;
          if (++cp.i == cp.n) seek(cp, cp.k + 1);
        }
      };
      prefetch_up_to(kp.l2_ahead);
      int s = 0, round = 0, gi = 0;
      int last_k = -1;
      while (cr.k < kp.n_phases && !s_abort) {
        if (cr.k != last_k) {
          stamp(cr.k, TR_W_FIRST);
          last_k = cr.k;
        }
        if (round > 0 && !consumer_wait(smem_addr(&empty[s]), (round & 1) ^ 1, &s_abort, kp.err)) break;
        const uint32_t fb = smem_addr(&full[s]);
        mbar_arrive_expect_tx(fb, cr.bytes);
        bulk_g2s(smem_addr(ring + (size_t)s * SB), cr.w + (size_t)(cr.t0 + cr.i) * WBYTES, WBYTES, fb, pol_ring);
        mbar_arrive(smem_addr(&armed[s]));
        s_issued = ++gi;
        if (++s == S) {
          s = 0;
          ++round;
        }
        if (ahead > 0) --ahead;
        if (++cr.i == cr.n) {
          stamp(cr.k, TR_W_LAST);
          seek(cr, cr.k + 1);
        }
        prefetch_up_to(kp.l2_ahead);
      }
    }
    return;
  }
  if (warp == CONSUMER_WARPS + 1) {
    // ------------------------------------------------------- activation producer
    // The whole warp polls the readiness of the next 32 tiles' chunks at once; lane 0 then
    // issues the copies of the ready prefix, in order, into the armed stages.
    const uint64_t pol = policy_evict_last();
    int s = 0;
    uint32_t aph = 0;
    for (int k = 0; k < kp.n_phases && !s_abort; ++k) {
      const Phase *ph = kp.phases + k;
      if (ph->kind != PH_GEMV) continue;
      const GemvParams &g = ph->g;
      long long T, t0;
      int G, n;
      phase_range(g, c, grid, T, G, t0, n);
      if (n == 0) continue;
      const float *x = g.x;
      const int ldx = g.ldx, n_kt = g.n_kt;
      int kt = static_cast<int>(t0 % n_kt);
      int i = 0;
      uint32_t idle = 0;
      bool first = true;
      while (i < n && !s_abort) {
        const int my_kt = (kt + lane) % n_kt;
        const bool ok = (i + lane >= n) || chunk_ready(g, my_kt);
        const unsigned ready = __ballot_sync(0xffffffffu, ok);
        // every lane's acquire happens before lane 0's copies (__syncwarp orders memory among
        // the participating threads)
        __syncwarp();
        const int run = min(n - i, (int)__ffs(~ready) - 1 < 0 ? 32 : (int)__ffs(~ready) - 1);
        if (run <= 0) {
          if (++idle > WAIT_LIMIT) {
            if (lane == 0) {
              s_abort = 1;
              atomicExch(kp.abort_flag, 1);
              atomicOr(kp.err, ERR_TIMEOUT);
            }
            break;
          }
          if ((idle & 63) == 0 && *reinterpret_cast<volatile int *>(kp.abort_flag)) {
            if (lane == 0) s_abort = 1;
            break;
          }
          continue;
        }
        idle = 0;
        if (lane == 0) {
          // the chunks were written by other CTAs' generic stores: order them before this
          // thread's bulk (async-proxy) reads
          asm volatile("fence.proxy.async.global;" ::: "memory");
          if (first) stamp(k, TR_X_GO);
          for (int j = 0; j < run; ++j) {
            if (!consumer_wait(smem_addr(&armed[s]), aph, &s_abort, kp.err)) break;
            const uint32_t fb = smem_addr(&full[s]);
            const uint32_t dst = smem_addr(ring + (size_t)s * SB + WBYTES);
            const int ktj = (kt + j) % n_kt;
            if constexpr (FMT == 0) {
#pragma unroll
              for (int b = 0; b < B; ++b)
                bulk_g2s(dst + b * (KTILE * 4), x + (size_t)b * ldx + (size_t)ktj * KTILE, KTILE * 4, fb, pol);
            } else {
              bulk_g2s(dst, act16_tile(g.xin, ktj), act16_copy_bytes(B, g.xsplit), fb, pol);
            }
            if (++s == S) {
              s = 0;
              aph ^= 1u;
            }
          }
        }
        s = __shfl_sync(0xffffffffu, s, 0);
        aph = __shfl_sync(0xffffffffu, aph, 0);
        first = false;
        i += run;
        kt = (kt + run) % n_kt;
      }
      if (lane == 0) stamp(k, TR_X_LAST);
    }
    return;
  }

  // ------------------------------------------------------------------- consumers
  int s = 0, segc = 0;
  uint32_t phase = 0;
  for (int k = 0; k < kp.n_phases; ++k) {
    const Phase *ph = kp.phases + k;
    const int kind = ph->kind;
    if (kind == PH_GEMV) {
      long long T, t0;
      int G, n;
      phase_range(ph->g, c, grid, T, G, t0, n);
      if (tid == 0) stamp(k, TR_CONS_GO);
      if (B <= 2)
        gemv_consume<B, FMT>(ph->g.n_kt, ring, full, empty, S, s, phase, t0, n, sr, segc, &s_abort, kp.err, tid,
                             ph->g.xsplit != 0);
      else
        gemv_consume_call<B, FMT>(ph->g.n_kt, ring, full, empty, S, s, phase, t0, n, sr, segc, &s_abort, kp.err,
                                  tid, ph->g.xsplit != 0);
    } else {
      if (tid == 0) {
        stamp(k, TR_CONS_ENTER);
        s_ap = ph->a;
        s_ap.positions = s_pos;
        s_ap.chunk = attn_chunk_size(s_ap);
      }
      consumer_sync();
      const AttnParams &a = s_ap;
      const int nc0 = attn_chunks(a, 0);
      const int nc1 = a.batch > 1 ? attn_chunks(a, 1) : 0;
      const int nc2 = a.batch > 2 ? attn_chunks(a, 2) : 0;
      const int nc3 = a.batch > 3 ? attn_chunks(a, 3) : 0;
      const int units = (nc0 + nc1 + nc2 + nc3) * a.n_kv_heads;
      for (int u = c; u < units; u += grid) {
        int b, kvh, ch, ncb;
        attn_unit_coords(u, a.n_kv_heads, nc0, nc1, nc2, nc3, b, kvh, ch, ncb);
        // the cached K/V rows do not depend on this step: load them while the Q/K/V rows of
        // this KV head are still being produced
        if (kp.head_dim == 128)
          attn_prefetch<128, 1>(a, b, kvh, ch, att, tid);
        else
          attn_prefetch<64, 1>(a, b, kvh, ch, att, tid);
        if (tid == 0) {
          if (u == c) stamp(k, TR_CONS_GO);
          if (a.in_ready) wait_counter(a.in_ready + kvh, (unsigned)a.in_need, &s_abort, kp.err);
        }
        consumer_sync();
        if (kp.head_dim == 128)
          attn_phase_unit<128>(a, b, kvh, ch, ncb, att, &s_last, tid, 1);
        else
          attn_phase_unit<64>(a, b, kvh, ch, ncb, att, &s_last, tid, 1);
        consumer_sync();
      }
      if (tid == 0) stamp(k, TR_CONS_DONE);
      consumer_sync();
    }
  }

  consumer_sync();
  if (s_abort && tid == 0) {
    // drain copies still in flight before the CTA's shared memory goes away (bounded)
    const int issued = s_issued;
    for (int i = (issued > S ? issued - S : 0); i < issued; ++i) mbar_wait(smem_addr(&full[i % S]), (i / S) & 1);
  }
}

// ------------------------------------------------------------------------------- launch
size_t stage_kernel_smem(int stages, int head_dim, int batch, int fmt) {
  // + 128: the staging buffer is aligned up to 128 bytes after the barriers
  return (size_t)stages * stage_bytes(batch, fmt) + stage_kernel_attn_bytes(head_dim) +
         (3 * stages + 2 * NSLOT) * sizeof(uint64_t) + 128 + seg_floats(fmt) * sizeof(float);
}

int stage_kernel_attn_bytes(int head_dim) {
  return head_dim == 128 ? AttnLayout<128, 1>::BYTES : AttnLayout<64, 1>::BYTES;
}

template <int B, int FMT>
static cudaError_t prepare_one_stage(size_t smem) {
  return cudaFuncSetAttribute(stage_kernel<B, FMT>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
}

cudaError_t prepare_stage_kernel(size_t smem) {
  // every instantiation may use up to `smem` bytes of dynamic shared memory
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
  if (kp.stages < 2 || kp.stages > MAX_STAGES || kp.stages != ring_depth(fmt, kp.stages)) return cudaErrorInvalidValue;
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
