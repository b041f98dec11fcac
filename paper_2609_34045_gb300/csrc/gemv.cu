// Weight-streaming GEMV y[b] = W . x[b] for batch 1..4 on sm_103a.
//
// Decode at batch one is memory-bandwidth bound: a stage reads each of its weights once per
// token and does two flops per weight (Kafila, section V-A, Eq. 2).  So the kernel is built
// around one thing, keeping HBM busy:
//
//   * weights are pre-tiled at load time ([N/64][K/128][64][128] bf16), so each 16 KiB tile is
//     one contiguous HBM chunk;
//   * the grid is persistent (one CTA per SM) and split "stream-K" style: CTA c streams the
//     contiguous tile range [c*T/G, (c+1)*T/G) of the flattened tile sequence, so every SM
//     moves the same number of bytes whatever the matrix shape;
//   * one producer thread per CTA feeds a ring of shared-memory stages with 1-D TMA bulk
//     copies (cp.async.bulk + mbarrier complete_tx); eight consumer warps read tiles and the
//     matching fp32 activation chunks from shared memory and accumulate in fp32;
//   * under programmatic dependent launch the producer starts streaming weights, which do not
//     depend on the previous kernel, before griddepcontrol.wait, hiding launch and tail gaps;
//   * row blocks split between CTAs are combined deterministically: each CTA writes its partial
//     sums, the last to arrive (atomic ticket, no spin) adds them in CTA order;
//   * epilogues are fused: RoPE + KV append, residual add + next RMSNorm input + sum of squares,
//     SwiGLU, greedy argmax.
#include "gemv_core.cuh"

namespace kfl {

constexpr int GEMV_MAX_STAGES = 13;  // 13 x 16.9 KiB (batch 1) still fits one CTA's shared memory
constexpr int GEMV_STATIC_SMEM = 3072;  // allowance for the kernel's own __shared__ variables

// ---------------------------------------------------------------------------- the kernel
// FMT 0: bf16 tiles [RB][KT].  FMT 1: int4 tiles, codes [RB][KT4/8] uint32 + RB x KT4/64 scales.
// Warps 0-7 consume tiles, warp 8 is the TMA producer, warp 9 the epilogue warp.
template <int B, int EPI, int FMT>
__global__ void __launch_bounds__(GEMV_THREADS, 2) gemv_kernel(const __grid_constant__ GemvParams p) {
  extern __shared__ __align__(1024) uint8_t smem[];
  constexpr int SB = stage_bytes(B, FMT);
  const int S = p.stages;
  uint64_t *full = reinterpret_cast<uint64_t *>(smem + (size_t)S * SB);
  uint64_t *empty = full + S;
  uint64_t *seg_full = empty + S;
  uint64_t *seg_empty = seg_full + NSLOT;
  // staging slots (SegRing: seg_floats(FMT) floats), 128-byte aligned (read as float4)
  float *red = reinterpret_cast<float *>((reinterpret_cast<uintptr_t>(seg_empty + NSLOT) + 127) & ~uintptr_t(127));
  __shared__ float s_inv[MAXB];
  __shared__ volatile int s_abort;
  __shared__ volatile int s_issued;
  __shared__ __align__(8) uint64_t s_rx_bar;  // cluster: rank 0 waits here for the other ranks' partials
  // cluster: [cluster - 1][RB][MAXB] partials of ranks 1.., after the staging slots
  float *rx = red + seg_floats(FMT);

  constexpr int KTILE = FMT == 0 ? KT : KT4;
  constexpr uint32_t WBYTES = FMT == 0 ? TILE_BYTES : TILE4_BYTES;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const long long T = (long long)p.n_rb * p.n_kt;
  const int G = gridDim.x, c = blockIdx.x;
  const long long t0 = (long long)c * T / G, t1 = (long long)(c + 1) * T / G;
  const int n = static_cast<int>(t1 - t0);
  const SegRing sr = {red, seg_full, seg_empty, seg_slots(FMT), seg_subs(FMT)};

  if (tid == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(smem_addr(&full[s]), 1);
      mbar_init(smem_addr(&empty[s]), ring_empty_count(FMT));
    }
    for (int s = 0; s < NSLOT; ++s) {
      mbar_init(smem_addr(&seg_full[s]), CONSUMER_WARPS);
      mbar_init(smem_addr(&seg_empty[s]), 1);
    }
    if (p.cluster > 1) mbar_init(smem_addr(&s_rx_bar), p.cluster - 1);
    s_abort = 0;
    s_issued = 0;
    fence_mbar_init();
  }
  for (int e = tid; e < seg_floats(FMT); e += GEMV_THREADS) red[e] = 0.f;  // int4 tiles add into it
  __syncthreads();
  if (p.cluster > 1) cluster_sync_all();  // the other ranks write rx / arrive on s_rx_bar only after this
  // The next kernel may launch (its CTAs start streaming their weights as SMs free up): bf16
  // GEMVs at once; int4 GEMVs once their last tile is issued, so that the next kernel's streams
  // do not contend with this one's last tiles and row-block tails (72B int4 b=4: -1.4% per step;
  // bf16: no gain)
  if constexpr (FMT == 0) pdl_launch_dependents();
  auto stamp = [&](int slot) {
    if (p.trace) p.trace[(size_t)c * TRACE_SLOTS + slot] = global_ns();
  };
  if (tid == 0) stamp(TR_CONS_GO);

  if (warp == CONSUMER_WARPS) {
    // ------------------------------------------------------------------ producer
    if (lane == 0) {
      const uint64_t pol_w = policy_evict_first();
      const uint64_t pol_x = policy_evict_last();
      // int4: the K tile's block of the Act16 input, one contiguous copy
      const uint32_t xbytes = FMT == 0 ? B * (KTILE * 4) : act16_copy_bytes(B, p.xsplit);
      const int pre = n < S ? n : S;
      stamp(TR_W_FIRST);
      for (int i = 0; i < pre; ++i) {
        const uint32_t fb = smem_addr(&full[i]);
        mbar_arrive_expect_tx(fb, WBYTES + xbytes);
        bulk_g2s(smem_addr(smem + (size_t)i * SB), p.w + (size_t)(t0 + i) * WBYTES, WBYTES, fb, pol_w);
        s_issued = i + 1;
      }
      pdl_wait();
      stamp(TR_X_GO);
      auto issue_x = [&](int kt, int s) {
        const uint32_t fb = smem_addr(&full[s]);
        const uint32_t dst = smem_addr(smem + (size_t)s * SB + WBYTES);
        if constexpr (FMT == 0) {
#pragma unroll
          for (int b = 0; b < B; ++b)
            bulk_g2s(dst + b * (KTILE * 4), p.x + (size_t)b * p.ldx + (size_t)kt * KTILE, KTILE * 4, fb, pol_x);
        } else {
          bulk_g2s(dst, act16_tile(p.xin, kt), xbytes, fb, pol_x);
        }
      };
      int kt_x = static_cast<int>(t0 % p.n_kt);
      for (int i = 0; i < pre; ++i) {
        issue_x(kt_x, i);
        if (++kt_x == p.n_kt) kt_x = 0;
      }
      int s = 0;
      uint32_t eph = 0;
      for (int i = pre; i < n; ++i) {
        if (!consumer_wait(smem_addr(&empty[s]), eph, &s_abort, p.err)) break;
        const uint32_t fb = smem_addr(&full[s]);
        mbar_arrive_expect_tx(fb, WBYTES + xbytes);
        bulk_g2s(smem_addr(smem + (size_t)s * SB), p.w + (size_t)(t0 + i) * WBYTES, WBYTES, fb, pol_w);
        issue_x(kt_x, s);
        s_issued = i + 1;
        if (++kt_x == p.n_kt) kt_x = 0;
        if (++s == S) {
          s = 0;
          eph ^= 1u;
        }
      }
      stamp(TR_W_LAST);
      if constexpr (FMT == 1) pdl_launch_dependents();
    }
    return;
  }
  if (warp == CONSUMER_WARPS + 1) {
    // -------------------------------------------------------------- epilogue warp
    pdl_wait();
    norm_scale_warp<B>(p, s_inv, lane);
    bool inv_ready = true;
    int segc = 0;
    gemv_epilogues<B, EPI>(p, t0, n, T, G, c, sr, segc, s_inv, inv_ready, &s_abort, lane,
                           p.cluster > 1 ? rx : nullptr, &s_rx_bar);
    if (lane == 0) stamp(TR_CONS_DONE);
    return;
  }

  // -------------------------------------------------------------------- consumers
  int s = 0, segc = 0;
  uint32_t phase = 0;
  if constexpr (FMT == 1) {
    // only the Q/K/V projection multiplies its input's rests (GemvParams::xsplit)
    gemv_consume_int4<B, EPI == EPI_QKV>(p.n_kt, smem, full, empty, S, s, phase, t0, n, sr, segc, &s_abort, p.err,
                                         tid);
  } else {
    gemv_consume<B, FMT>(p.n_kt, smem, full, empty, S, s, phase, t0, n, sr, segc, &s_abort, p.err, tid, false);
  }

  consumer_sync();
  if (tid == 0) stamp(TR_CONS_ENTER);
  if (s_abort && tid == 0) {
    // drain copies still in flight before the CTA's shared memory goes away (bounded)
    const int issued = s_issued;
    for (int i = (issued > S ? issued - S : 0); i < issued; ++i)
      mbar_wait(smem_addr(&full[i % S]), (i / S) & 1);
  }
}

// ---------------------------------------------------------------------------- launch
static size_t gemv_smem_bytes(int stages, int batch, int fmt, int cluster = 1) {
  return (size_t)stages * stage_bytes(batch, fmt) + (2 * stages + 2 * NSLOT) * sizeof(uint64_t) + 128 +
         (seg_floats(fmt) + (cluster > 1 ? cluster - 1 : 0) * RB * MAXB) * sizeof(float);
}

static int g_smem_optin = 0, g_smem_per_sm = 0, g_n_sm = 0;

// Dynamic shared memory of a launch.  Stream-K gives every CTA an equal share of the tiles, so a
// grid of at most one CTA per SM assumes each CTA has its SM's issue slots to itself.  Where two
// rings fit one SM (int4 tiles at batch 1), the block scheduler may place two CTAs of one GEMV on
// an SM that frees up early while other SMs still hold the previous kernel's CTAs; those two then
// share the SM and the whole GEMV waits for them.  Asking for more than half of the SM's shared
// memory keeps such a grid at one CTA per SM.
static size_t gemv_launch_smem(size_t need, int grid) {
  if (grid > g_n_sm) return need;
  const size_t half = (size_t)g_smem_per_sm / 2;
  const size_t cap = (size_t)g_smem_optin - GEMV_STATIC_SMEM;
  return need >= half ? need : (half < cap ? half : cap);
}

template <int B, int EPI, int FMT>
static cudaError_t launch_one(const GemvParams &p, int grid, cudaStream_t s, bool pdl) {
  cudaLaunchConfig_t cfg = {};
  const size_t smem = gemv_launch_smem(gemv_smem_bytes(p.stages, B, FMT, p.cluster), grid);
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(GEMV_THREADS);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  int na = 0;
  if (pdl) {
    attr[na].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[na].val.programmaticStreamSerializationAllowed = 1;
    ++na;
  }
  if (p.cluster > 1) {
    attr[na].id = cudaLaunchAttributeClusterDimension;
    attr[na].val.clusterDim.x = p.cluster;
    attr[na].val.clusterDim.y = 1;
    attr[na].val.clusterDim.z = 1;
    ++na;
  }
  cfg.attrs = attr;
  cfg.numAttrs = na;
  return cudaLaunchKernelEx(&cfg, gemv_kernel<B, EPI, FMT>, p);
}

template <int EPI, int FMT>
static cudaError_t launch_b(const GemvParams &p, int grid, cudaStream_t s, bool pdl) {
  switch (p.batch) {
    case 1: return launch_one<1, EPI, FMT>(p, grid, s, pdl);
    case 2: return launch_one<2, EPI, FMT>(p, grid, s, pdl);
    case 3: return launch_one<3, EPI, FMT>(p, grid, s, pdl);
    case 4: return launch_one<4, EPI, FMT>(p, grid, s, pdl);
    default: return cudaErrorInvalidValue;
  }
}

template <int FMT>
static cudaError_t launch_f(const GemvParams &p, int epi, int grid, cudaStream_t s, bool pdl) {
  switch (epi) {
    case EPI_STORE: return launch_b<EPI_STORE, FMT>(p, grid, s, pdl);
    case EPI_QKV: return launch_b<EPI_QKV, FMT>(p, grid, s, pdl);
    case EPI_RESID: return launch_b<EPI_RESID, FMT>(p, grid, s, pdl);
    case EPI_SWIGLU: return launch_b<EPI_SWIGLU, FMT>(p, grid, s, pdl);
    case EPI_ARGMAX: return launch_b<EPI_ARGMAX, FMT>(p, grid, s, pdl);
    default: return cudaErrorInvalidValue;
  }
}

// The deepest ring of this batch size and format that fits a CTA's shared memory.
// The deepest ring such that `per_sm` CTAs of a GEMV with this cluster size fit one SM's shared
// memory (each also holds its static shared memory and the per-CTA reservation).
int gemv_stages_for(int batch, int fmt, int cluster, int per_sm) {
  int s = GEMV_MAX_STAGES;
  auto fits = [&](int st) {
    const size_t cta = gemv_smem_bytes(st, batch, fmt, cluster) + GEMV_STATIC_SMEM;
    return cta <= (size_t)g_smem_optin && (size_t)per_sm * (cta + 1024) <= (size_t)g_smem_per_sm;
  };
  while (s > 2 && !fits(s)) --s;
  return ring_depth(fmt, s);
}

int gemv_max_stages(int batch, int fmt, int smem_optin) {
  int s = GEMV_MAX_STAGES;
  while (s > 2 && gemv_smem_bytes(s, batch, fmt) + GEMV_STATIC_SMEM > (size_t)smem_optin) --s;
  return ring_depth(fmt, s);
}

template <int B, int EPI, int FMT>
static cudaError_t prepare_one() {
  // every launch asks for at most this (a deepest ring, or a cluster's partials with a shallower one)
  return cudaFuncSetAttribute(gemv_kernel<B, EPI, FMT>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              g_smem_optin - GEMV_STATIC_SMEM);
}

template <int EPI, int FMT>
static cudaError_t prepare_b() {
  cudaError_t e;
  if ((e = prepare_one<1, EPI, FMT>()) != cudaSuccess) return e;
  if ((e = prepare_one<2, EPI, FMT>()) != cudaSuccess) return e;
  if ((e = prepare_one<3, EPI, FMT>()) != cudaSuccess) return e;
  return prepare_one<4, EPI, FMT>();
}

template <int FMT>
static cudaError_t prepare_f() {
  cudaError_t e;
  if ((e = prepare_b<EPI_STORE, FMT>()) != cudaSuccess) return e;
  if ((e = prepare_b<EPI_QKV, FMT>()) != cudaSuccess) return e;
  if ((e = prepare_b<EPI_RESID, FMT>()) != cudaSuccess) return e;
  if ((e = prepare_b<EPI_SWIGLU, FMT>()) != cudaSuccess) return e;
  return prepare_b<EPI_ARGMAX, FMT>();
}

// Raise the dynamic shared-memory limit of every GEMV instantiation (once per device, before
// any launch or stream capture).
cudaError_t prepare_gemv() {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&g_smem_optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
  if (e == cudaSuccess)
    e = cudaDeviceGetAttribute(&g_smem_per_sm, cudaDevAttrMaxSharedMemoryPerMultiprocessor, dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&g_n_sm, cudaDevAttrMultiProcessorCount, dev);
  if (e != cudaSuccess) return e;
  e = prepare_f<0>();
  return e != cudaSuccess ? e : prepare_f<1>();
}

cudaError_t launch_gemv(const GemvParams &p, int epi, int grid, cudaStream_t s, bool pdl) {
  if (p.stages < 2 || p.stages > gemv_max_stages(p.batch, p.fmt, g_smem_optin)) return cudaErrorInvalidValue;
  if (p.stages != ring_depth(p.fmt, p.stages)) return cudaErrorInvalidValue;  // int4: an even ring
  // clusters: each CTA exactly 1/cluster of the K range of one row block
  if (p.cluster > 1 && (p.cluster > MAX_CLUSTER || grid != p.cluster * p.n_rb || p.n_kt < p.cluster))
    return cudaErrorInvalidValue;
  if (gemv_smem_bytes(p.stages, p.batch, p.fmt, p.cluster) + GEMV_STATIC_SMEM > (size_t)g_smem_optin)
    return cudaErrorInvalidValue;
  // the int4 consumers take the rests exactly when the Q/K/V projection runs (a template choice)
  if (p.fmt == 1 && (p.xsplit != 0) != (epi == EPI_QKV)) return cudaErrorInvalidValue;
  return p.fmt == 0 ? launch_f<0>(p, epi, grid, s, pdl) : launch_f<1>(p, epi, grid, s, pdl);
}

}  // namespace kfl
