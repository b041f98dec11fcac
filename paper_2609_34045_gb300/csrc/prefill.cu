// Dense prompt prefill kernels (sm_103a): the tcgen05 GEMM with its fused epilogues, causal
// attention of the prompt's tokens over the user's KV cache, row RMSNorm, the prompt's input rows
// and the greedy argmax over the column tiles.
//
// The prefill computes what one decode step per prompt token computes (section III: a stage
// applies its block range to every token; the head's sampler is greedy), with the tokens of a
// pass as the rows of dense matrix products instead of one weight pass per token.
#include <cudaTypedefs.h>

#include <algorithm>
#include <cmath>

#include "../../include/kafila_gemm.h"
#include "prefill.cuh"

namespace kfl {

// ---------------------------------------------------------------------------- tcgen05 / TMA
namespace {

__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

// Tensor-memory allocation by one whole warp; the base address is written to shared memory.
__device__ __forceinline__ void tmem_alloc(uint32_t dst_smem, uint32_t cols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(dst_smem), "r"(cols)
               : "memory");
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t cols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(cols) : "memory");
}

// Shared-memory matrix descriptor of a K-major operand in the 128-byte swizzled layout: rows of
// 128 bytes (64 bf16 of K), groups of 8 rows 1024 bytes apart (the stride byte offset); the
// leading byte offset is unused in this layout (1 by convention); descriptor version 1; swizzle
// mode 2 (128 bytes).  A slice of 16 K values starts 32 bytes further within the row.
__device__ __forceinline__ uint64_t sdesc_k_sw128(uint32_t addr) {
  uint64_t d = 0;
  d |= (uint64_t)((addr & 0x3FFFFu) >> 4);
  d |= (uint64_t)1 << 16;
  d |= (uint64_t)(1024 >> 4) << 32;
  d |= (uint64_t)1 << 46;
  d |= (uint64_t)2 << 61;
  return d;
}

// Instruction descriptor of kind::f16: fp32 accumulator (bits 4-5 = 1), A and B both bf16 (bits
// 7-9 and 10-12 = 1) or both fp16 (0), both K-major (bits 15, 16 = 0), N >> 3 in bits 17-22,
// M >> 4 in bits 24-28.
__host__ __device__ constexpr uint32_t idesc_kind_f16(int m, int n, bool bf16) {
  return (1u << 4) | ((bf16 ? 1u : 0u) << 7) | ((bf16 ? 1u : 0u) << 10) | ((uint32_t)(n >> 3) << 17) |
         ((uint32_t)(m >> 4) << 24);
}

__device__ __forceinline__ void mma_bf16_ss(uint32_t d_tmem, uint64_t da, uint64_t db, uint32_t idesc,
                                            uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(da), "l"(db), "r"(idesc), "r"(accumulate)
      : "memory");
}

// Arrive on an mbarrier of this CTA once every MMA this thread issued before has completed.
__device__ __forceinline__ void mma_commit(uint32_t bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
               : "memory");
}

// 32 consecutive fp32 columns of this thread's tensor-memory lane (warp w reads lanes 32 w ..).
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
      "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
        "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
        "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap *map, int c0, int c1, uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::"r"(
          dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(bar)
      : "memory");
}

__device__ __forceinline__ void tma_load_4d(uint32_t dst, const CUtensorMap *map, int c0, int c1, int c2, int c3,
                                            uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.4d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3, %4, %5}], "
      "[%6];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(c2), "r"(c3), "r"(bar)
      : "memory");
}

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  return (uint32_t)f32_to_bf16_rne(lo) | ((uint32_t)f32_to_bf16_rne(hi) << 16);
}

// x as two bf16 terms: hi = bf16(x), lo = bf16(x - hi) (the difference is exact in fp32).
__device__ __forceinline__ void split_bf16(float x, uint16_t &hi, uint16_t &lo) {
  hi = f32_to_bf16_rne(x);
  lo = f32_to_bf16_rne(x - bf16_to_f32(hi));
}
// The same with fp16 terms (about 2^-22 relative left; |x| must stay below 65504).
__device__ __forceinline__ void split_f16(float x, uint16_t &hi, uint16_t &lo) {
  hi = f32_to_f16_rn(x);
  lo = f32_to_f16_rn(x - f16_to_f32(hi));
}
__device__ __forceinline__ void split_term(float x, uint16_t &hi, uint16_t &lo, int f16) {
  if (f16)
    split_f16(x, hi, lo);
  else
    split_bf16(x, hi, lo);
}
// Two values as packed pairs of their hi and lo terms.  fp16 terms of a value that fp16 cannot
// hold (|x| >= 65520 rounds to infinity, or not finite) set ERR_F16_RANGE in *err.
__device__ __forceinline__ void split_pack(float x0, float x1, uint32_t &hi, uint32_t &lo, int f16 = 0,
                                           unsigned *err = nullptr) {
  if (f16 && err && !(fabsf(x0) < 65520.f && fabsf(x1) < 65520.f)) atomicOr(err, ERR_F16_RANGE);
  uint16_t h0, l0, h1, l1;
  split_term(x0, h0, l0, f16);
  split_term(x1, h1, l1, f16);
  hi = (uint32_t)h0 | ((uint32_t)h1 << 16);
  lo = (uint32_t)l0 | ((uint32_t)l1 << 16);
}

// ---------------------------------------------------------------------------- GEMM epilogues
// Thread = one token t of the tile (its tensor-memory lane); v[j] = Y[t][n + j], j < 32.

template <int MODE>
struct EpiState {
  float best = -INFINITY;
  int bidx = 0x7FFFFFFF;
};

template <int MODE>
__device__ __forceinline__ void epilogue32(const PrefillEpiParams &ep, int t, int n, const uint32_t (&r)[32],
                                           EpiState<MODE> &st) {
  float v[32];
#pragma unroll
  for (int j = 0; j < 32; ++j) v[j] = __uint_as_float(r[j]);
  if constexpr (MODE == PE_STORE || MODE == PE_RESID) {
    float *row = ep.out + (size_t)t * ep.ldo + n;
    if (n + 32 <= ep.N) {
#pragma unroll
      for (int j = 0; j < 32; j += 4) {
        float4 y = make_float4(v[j], v[j + 1], v[j + 2], v[j + 3]);
        if constexpr (MODE == PE_RESID) {
          const float4 h = *reinterpret_cast<const float4 *>(row + j);
          y.x += h.x;
          y.y += h.y;
          y.z += h.z;
          y.w += h.w;
        }
        *reinterpret_cast<float4 *>(row + j) = y;
      }
    } else {
#pragma unroll
      for (int j = 0; j < 32; ++j)
        if (n + j < ep.N) row[j] = (MODE == PE_RESID ? row[j] : 0.f) + v[j];
    }
  } else if constexpr (MODE == PE_SWIGLU) {
    // 16 outputs j0 .. j0 + 15, as hi and lo terms
    const int j0 = n >> 1;
    uint32_t w[8], wl[8];
#pragma unroll
    for (int i = 0; i < 16; i += 2) {
      const float g0 = v[2 * i], u0 = v[2 * i + 1], g1 = v[2 * i + 2], u1 = v[2 * i + 3];
      split_pack(g0 / (1.0f + expf(-g0)) * u0, g1 / (1.0f + expf(-g1)) * u1, w[i / 2], wl[i / 2], ep.f16, ep.err);
    }
    uint16_t *row = ep.out16 + (size_t)t * ep.ldo16 + j0;
    uint16_t *rlo = ep.out16lo + (size_t)t * ep.ldo16 + j0;
    if (n + 32 <= ep.N) {
      reinterpret_cast<uint4 *>(row)[0] = make_uint4(w[0], w[1], w[2], w[3]);
      reinterpret_cast<uint4 *>(row)[1] = make_uint4(w[4], w[5], w[6], w[7]);
      reinterpret_cast<uint4 *>(rlo)[0] = make_uint4(wl[0], wl[1], wl[2], wl[3]);
      reinterpret_cast<uint4 *>(rlo)[1] = make_uint4(wl[4], wl[5], wl[6], wl[7]);
    } else {
#pragma unroll
      for (int i = 0; i < 16; ++i)
        if (n + 2 * i + 1 < ep.N) {
          row[i] = (uint16_t)(w[i / 2] >> (16 * (i & 1)));
          rlo[i] = (uint16_t)(wl[i / 2] >> (16 * (i & 1)));
        }
    }
  } else if constexpr (MODE == PE_QKV) {
    const int pos = ep.positions[t];
    if (pos < 0) return;
    const int half = ep.hd / 2;
    if (n < ep.qdim + ep.kvdim) {
      // 16 RoPE pairs (i, i + hd/2) of one head
      const bool is_q = n < ep.qdim;
      const int r0 = is_q ? n : n - ep.qdim;
      const int head = r0 / ep.hd, i0 = (r0 % ep.hd) / 2;
      // the 16 factors of each kind are 64 contiguous, 64-byte aligned bytes
      const float4 *cs = reinterpret_cast<const float4 *>(ep.rope_cos + (size_t)pos * half + i0);
      const float4 *sn = reinterpret_cast<const float4 *>(ep.rope_sin + (size_t)pos * half + i0);
      float c[16], sv[16];
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const float4 a = cs[j], b = sn[j];
        c[4 * j] = a.x, c[4 * j + 1] = a.y, c[4 * j + 2] = a.z, c[4 * j + 3] = a.w;
        sv[4 * j] = b.x, sv[4 * j + 1] = b.y, sv[4 * j + 2] = b.z, sv[4 * j + 3] = b.w;
      }
      uint16_t *dst;
      if (is_q) {
        dst = ep.out16 + (size_t)t * ep.ldo16 + (size_t)head * ep.hd;
      } else {
        dst = ep.kcache + (((size_t)ep.slot * ep.hkv + head) * ep.max_ctx + pos) * ep.hd;
      }
      // rotated first halves -> dst[i0 ..], second halves -> dst[i0 + hd/2 ..]: 32 bytes each
      uint32_t w1[8], w2[8];
#pragma unroll
      for (int i = 0; i < 16; i += 2) {
        const float a1 = v[2 * i], a2 = v[2 * i + 1], b1 = v[2 * i + 2], b2 = v[2 * i + 3];
        w1[i / 2] = pack_bf16(a1 * c[i] - a2 * sv[i], b1 * c[i + 1] - b2 * sv[i + 1]);
        w2[i / 2] = pack_bf16(a2 * c[i] + a1 * sv[i], b2 * c[i + 1] + b1 * sv[i + 1]);
      }
      uint4 *d1 = reinterpret_cast<uint4 *>(dst + i0), *d2 = reinterpret_cast<uint4 *>(dst + i0 + half);
      d1[0] = make_uint4(w1[0], w1[1], w1[2], w1[3]);
      d1[1] = make_uint4(w1[4], w1[5], w1[6], w1[7]);
      d2[0] = make_uint4(w2[0], w2[1], w2[2], w2[3]);
      d2[1] = make_uint4(w2[4], w2[5], w2[6], w2[7]);
    } else {
      const int r0 = n - ep.qdim - ep.kvdim;
      const int head = r0 / ep.hd, j0 = r0 % ep.hd;
      uint16_t *dst = ep.vcache + (((size_t)ep.slot * ep.hkv + head) * ep.max_ctx + pos) * ep.hd + j0;
      uint32_t w[16];
#pragma unroll
      for (int i = 0; i < 16; ++i) w[i] = pack_bf16(v[2 * i], v[2 * i + 1]);
#pragma unroll
      for (int i = 0; i < 16; i += 4) reinterpret_cast<uint4 *>(dst)[i / 4] = make_uint4(w[i], w[i + 1], w[i + 2], w[i + 3]);
    }
  } else if constexpr (MODE == PE_ARGMAX) {
#pragma unroll
    for (int j = 0; j < 32; ++j)
      if (n + j < ep.N && v[j] > st.best) {
        st.best = v[j];
        st.bidx = n + j;
      }
  }
}

// ---------------------------------------------------------------------------- GEMM kernel
// Split-K: the launch is a cluster of ep.splits (2, 4 or 8) CTAs per output tile (blockIdx.z =
// rank); unsplit GEMMs run prefill_gemm_persistent.
template <int MODE>
__global__ void __launch_bounds__(PG_THREADS, 1)
    prefill_gemm_kernel(const __grid_constant__ CUtensorMap tm_a, const __grid_constant__ CUtensorMap tm_a2,
                        const __grid_constant__ CUtensorMap tm_b, int n_kblocks, PrefillEpiParams ep) {
  static_assert(MODE != PE_ARGMAX, "the argmax partials are per whole tile: lm_head is never split");
  extern __shared__ uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t s_full[PG_STAGES], s_empty[PG_STAGES], s_accum;
  __shared__ uint32_t s_tmem;
  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  const int t0 = blockIdx.x * PG_M, n0 = blockIdx.y * PG_N;
  // split-K: split blockIdx.z of ep.splits takes K blocks [kb0, kb1)
  const int kb0 = (int)((long long)blockIdx.z * n_kblocks / ep.splits);
  const int kb1 = (int)((long long)(blockIdx.z + 1) * n_kblocks / ep.splits);
  const int nkb = kb1 - kb0;
  // the swizzled tiles start on a 1024-byte boundary
  const uint32_t raw = smem_addr(smem_raw);
  const uint32_t sa = (raw + 1023u) & ~1023u;      // [stage][hi, lo] activation tiles
  const uint32_t sb = sa + PG_STAGES * 2 * PG_A_BYTES;

  if (threadIdx.x == 0) {
    for (int s = 0; s < PG_STAGES; ++s) {
      mbar_init(smem_addr(&s_full[s]), 1);
      mbar_init(smem_addr(&s_empty[s]), 1);
    }
    mbar_init(smem_addr(&s_accum), 1);
    fence_mbar_init();
  }
  __syncwarp();
  if (warp == 0) tmem_alloc(smem_addr(&s_tmem), PG_TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = s_tmem;

  if (threadIdx.x == 0) {
    // ---- TMA producer
    int issued[PG_STAGES] = {};
    bool ok = true;
    for (int j = 0; j < nkb; ++j) {
      const int s = j % PG_STAGES, kb = kb0 + j;
      const uint32_t use = j / PG_STAGES;
      if (use > 0 && !mbar_wait(smem_addr(&s_empty[s]), (use - 1) & 1)) {
        ok = false;
        break;
      }
      const uint32_t full = smem_addr(&s_full[s]);
      mbar_arrive_expect_tx(full, 2 * PG_A_BYTES + PG_B_BYTES);
      tma_load_2d(sa + s * 2 * PG_A_BYTES, &tm_a, kb * PG_K, t0, full);
      tma_load_2d(sa + s * 2 * PG_A_BYTES + PG_A_BYTES, &tm_a2, kb * PG_K, t0, full);
      // weight tiles: (column within the K tile, row within the row block, K tile, row block)
      tma_load_4d(sb + s * PG_B_BYTES, &tm_b, (kb & 1) * PG_K, 0, kb >> 1, n0 / RB, full);
      ++issued[s];
    }
    if (!ok) {
      atomicOr(ep.err, ERR_TIMEOUT);
      // let the copies in flight land before the CTA's shared memory is released
      for (int s = 0; s < PG_STAGES; ++s)
        if (issued[s] > 0) mbar_wait(smem_addr(&s_full[s]), (issued[s] - 1) & 1);
    }
  } else if (threadIdx.x == 32) {
    // ---- MMA issuer
    // A and B always share one type: both bf16, or (int4 stages) both fp16
    const uint32_t idesc = ep.f16 ? idesc_kind_f16(PG_M, PG_N, false) : idesc_kind_f16(PG_M, PG_N, true);
    for (int j = 0; j < nkb; ++j) {
      const int s = j % PG_STAGES;
      if (!mbar_wait(smem_addr(&s_full[s]), (j / PG_STAGES) & 1)) {
        atomicOr(ep.err, ERR_TIMEOUT);
        break;
      }
      tc_fence_after();
      const uint32_t a = sa + s * 2 * PG_A_BYTES, b = sb + s * PG_B_BYTES;
#pragma unroll
      for (int k = 0; k < PG_K / 16; ++k) {
        const uint64_t db = sdesc_k_sw128(b + 32 * k);
        mma_bf16_ss(tmem, sdesc_k_sw128(a + 32 * k), db, idesc, (j | k) != 0);
        mma_bf16_ss(tmem, sdesc_k_sw128(a + PG_A_BYTES + 32 * k), db, idesc, 1);
      }
      mma_commit(smem_addr(&s_empty[s]));  // the stage is free once these MMAs have read it
    }
    mma_commit(smem_addr(&s_accum));  // the accumulator is complete (or, after a timeout, idle)
  }
  __syncwarp();

  // ---- epilogue: warp w holds tokens t0 + 32 w + lane
  // block-uniform: the split path synchronises the whole block
  const bool ready = __syncthreads_and(mbar_wait(smem_addr(&s_accum), 0)) != 0;
  if (!ready && threadIdx.x == 0) atomicOr(ep.err, ERR_TIMEOUT);
  tc_fence_after();
  const int row = warp * 32 + lane, t = t0 + row;
  EpiState<MODE> st;
  {
    // split-K over a cluster of S = ep.splits CTAs (rank = blockIdx.z).  Column chunk c (32
    // columns) of the tile belongs to rank c / (8 / S).  Every CTA pushes each chunk of its fp32
    // accumulator into the owner's shared memory (posted remote stores; the pipeline buffers are
    // idle now), at [own rank][row][chunk within the owner's share]; after the cluster barrier
    // each owner sums its chunks over the ranks in rank order (deterministic) from its own shared
    // memory and runs the epilogue.  The first barrier keeps a CTA from writing into a peer whose
    // pipeline still uses that memory.  Both barriers are reached by every CTA, whatever its
    // pipeline did.
    const int S = ep.splits, per = (PG_N / 32) / S, ld = per * 32 + 4;
    float *red = reinterpret_cast<float *>(smem_raw + (sa - raw));  // [S][PG_M][ld]
    cluster_sync_all();
    if (ready) {
      for (int c = 0; c < PG_N / 32; ++c) {
        if (n0 + 32 * c >= ep.N) break;
        uint32_t r[32];
        tmem_ld32(tmem + ((uint32_t)(warp * 32) << 16) + 32 * c, r);
        const int owner = c / per;
        const uint32_t dst = map_to_rank(smem_addr(red + ((size_t)blockIdx.z * PG_M + row) * ld + (c % per) * 32),
                                         owner);
#pragma unroll
        for (int j = 0; j < 8; ++j)
          st_cluster_f4(dst + 16 * j, make_float4(__uint_as_float(r[4 * j]), __uint_as_float(r[4 * j + 1]),
                                                  __uint_as_float(r[4 * j + 2]), __uint_as_float(r[4 * j + 3])));
      }
    }
    cluster_sync_all();
    if (ready) {
      for (int cc = 0; cc < per; ++cc) {
        const int n = n0 + 32 * (blockIdx.z * per + cc);
        if (n >= ep.N) break;
        float acc[32];
#pragma unroll
        for (int j = 0; j < 32; ++j) acc[j] = 0.f;
        for (int q = 0; q < S; ++q) {
          const float4 *src = reinterpret_cast<const float4 *>(red + ((size_t)q * PG_M + row) * ld + cc * 32);
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            const float4 v4 = src[j];
            acc[4 * j] += v4.x;
            acc[4 * j + 1] += v4.y;
            acc[4 * j + 2] += v4.z;
            acc[4 * j + 3] += v4.w;
          }
        }
        uint32_t r[32];
#pragma unroll
        for (int j = 0; j < 32; ++j) r[j] = __float_as_uint(acc[j]);
        if (t < ep.T) epilogue32<MODE>(ep, t, n, r, st);
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem, PG_TMEM_COLS);
  }
}

// ---------------------------------------------------------------------------- persistent GEMM
// The unsplit GEMM as a persistent kernel: one CTA per SM takes tiles c, c + grid, ...  The TMA
// ring runs on across tile boundaries, and two accumulators (all 512 TMEM columns) let the MMAs of
// the next tile proceed while four epilogue warps drain the previous one.  Warp 0 lane 0 issues
// TMA, warp 1 lane 0 issues MMAs, warps 2-5 run the epilogue (warp w reads TMEM lanes
// 32 (w % 4) ..).  Every wait is bounded; a CTA that gives up sets ERR_TIMEOUT, lets its copies
// and MMAs in flight complete (bounded), frees its TMEM and returns.
constexpr int PP_THREADS = 192;
constexpr int PP_TMEM_COLS = 2 * PG_N;

template <int MODE>
__global__ void __launch_bounds__(PP_THREADS, 1)
    prefill_gemm_persistent(const __grid_constant__ CUtensorMap tm_a, const __grid_constant__ CUtensorMap tm_a2,
                            const __grid_constant__ CUtensorMap tm_b, int n_kblocks, PrefillEpiParams ep) {
  extern __shared__ uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t s_full[PG_STAGES], s_empty[PG_STAGES], s_acc_full[2], s_acc_empty[2], s_drain;
  __shared__ uint32_t s_tmem;
  __shared__ int s_abort;
  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  const int t_tiles = (ep.T + PG_M - 1) / PG_M, n_tiles = (ep.N + PG_N - 1) / PG_N;
  const int tiles = t_tiles * n_tiles;
  const uint32_t raw = smem_addr(smem_raw);
  const uint32_t sa = (raw + 1023u) & ~1023u;  // [stage][hi, lo] activation tiles
  const uint32_t sb = sa + PG_STAGES * 2 * PG_A_BYTES;
  if (threadIdx.x == 0) {
    for (int s = 0; s < PG_STAGES; ++s) {
      mbar_init(smem_addr(&s_full[s]), 1);
      mbar_init(smem_addr(&s_empty[s]), 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(smem_addr(&s_acc_full[b]), 1);
      mbar_init(smem_addr(&s_acc_empty[b]), 4);  // one arrival per epilogue warp
    }
    mbar_init(smem_addr(&s_drain), 1);
    s_abort = 0;
    fence_mbar_init();
  }
  __syncwarp();
  if (warp == 0) tmem_alloc(smem_addr(&s_tmem), PP_TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = s_tmem;
  volatile int *abort_flag = &s_abort;

  if (warp == 0) {
    if (lane == 0) {
      // ---- TMA producer: k-block it of the CTA's sequence uses stage it % S
      int issued[PG_STAGES] = {};
      long long it = 0;
      bool ok = true;
      for (int tile = blockIdx.x; tile < tiles && ok; tile += gridDim.x) {
        const int t0 = (tile % t_tiles) * PG_M, n0 = (tile / t_tiles) * PG_N;
        for (int kb = 0; kb < n_kblocks; ++kb, ++it) {
          const int s = (int)(it % PG_STAGES);
          const uint32_t use = (uint32_t)(it / PG_STAGES);
          if (*abort_flag || (use > 0 && !mbar_wait(smem_addr(&s_empty[s]), (use - 1) & 1))) {
            ok = false;
            break;
          }
          const uint32_t full = smem_addr(&s_full[s]);
          mbar_arrive_expect_tx(full, 2 * PG_A_BYTES + PG_B_BYTES);
          tma_load_2d(sa + s * 2 * PG_A_BYTES, &tm_a, kb * PG_K, t0, full);
          tma_load_2d(sa + s * 2 * PG_A_BYTES + PG_A_BYTES, &tm_a2, kb * PG_K, t0, full);
          tma_load_4d(sb + s * PG_B_BYTES, &tm_b, (kb & 1) * PG_K, 0, kb >> 1, n0 / RB, full);
          ++issued[s];
        }
      }
      if (!ok) {
        *abort_flag = 1;
        atomicOr(ep.err, ERR_TIMEOUT);
        for (int s = 0; s < PG_STAGES; ++s)
          if (issued[s] > 0) mbar_wait(smem_addr(&s_full[s]), (issued[s] - 1) & 1);
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    if (lane == 0) {
      // ---- MMA issuer: tile i of this CTA accumulates into TMEM columns (i % 2) * PG_N
      const uint32_t idesc = ep.f16 ? idesc_kind_f16(PG_M, PG_N, false) : idesc_kind_f16(PG_M, PG_N, true);
      long long it = 0;
      int i = 0;
      bool ok = true;
      for (int tile = blockIdx.x; tile < tiles && ok; tile += gridDim.x, ++i) {
        const int buf = i & 1;
        if (i >= 2 && !mbar_wait(smem_addr(&s_acc_empty[buf]), ((i >> 1) - 1) & 1)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d = tmem + (uint32_t)(buf * PG_N);
        for (int kb = 0; kb < n_kblocks; ++kb, ++it) {
          const int s = (int)(it % PG_STAGES);
          if (*abort_flag || !mbar_wait(smem_addr(&s_full[s]), (uint32_t)(it / PG_STAGES) & 1)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t a = sa + s * 2 * PG_A_BYTES, b = sb + s * PG_B_BYTES;
#pragma unroll
          for (int k = 0; k < PG_K / 16; ++k) {
            const uint64_t db = sdesc_k_sw128(b + 32 * k);
            mma_bf16_ss(d, sdesc_k_sw128(a + 32 * k), db, idesc, (kb | k) != 0);
            mma_bf16_ss(d, sdesc_k_sw128(a + PG_A_BYTES + 32 * k), db, idesc, 1);
          }
          mma_commit(smem_addr(&s_empty[s]));
        }
        if (ok) mma_commit(smem_addr(&s_acc_full[buf]));
      }
      if (!ok) {
        *abort_flag = 1;
        atomicOr(ep.err, ERR_TIMEOUT);
      }
      // every MMA issued has completed before TMEM can be freed
      mma_commit(smem_addr(&s_drain));
      mbar_wait(smem_addr(&s_drain), 0);
    }
    __syncwarp();
  } else {
    // ---- epilogue warps 2..5: TMEM lanes 32 q .. 32 q + 31 (q = warp % 4) are tokens t0 + 32 q + lane
    const int q = warp & 3, row = 32 * q + lane;
    int i = 0;
    for (int tile = blockIdx.x; tile < tiles; tile += gridDim.x, ++i) {
      const int buf = i & 1;
      const bool ready = __all_sync(0xffffffffu, !*abort_flag && mbar_wait(smem_addr(&s_acc_full[buf]), (i >> 1) & 1));
      if (!ready) {
        if (lane == 0) {
          *abort_flag = 1;
          atomicOr(ep.err, ERR_TIMEOUT);
        }
        break;
      }
      tc_fence_after();
      const int t_tile = tile % t_tiles, n_tile = tile / t_tiles;
      const int t = t_tile * PG_M + row, n0 = n_tile * PG_N;
      EpiState<MODE> st;
      for (int c = 0; c < PG_N / 32; ++c) {
        const int n = n0 + 32 * c;
        if (n >= ep.N) break;  // uniform across the warp
        uint32_t r[32];
        tmem_ld32(tmem + ((uint32_t)(32 * q) << 16) + (uint32_t)(buf * PG_N + 32 * c), r);
        if (t < ep.T) epilogue32<MODE>(ep, t, n, r, st);
      }
      if constexpr (MODE == PE_ARGMAX) {
        if (t < ep.T) {
          ep.amax[(size_t)t * ep.n_tiles + n_tile] = st.best;
          ep.aidx[(size_t)t * ep.n_tiles + n_tile] = st.bidx;
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_addr(&s_acc_empty[buf]));
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem, PP_TMEM_COLS);
  }
}

// ---------------------------------------------------------------------------- attention
// Causal attention of a block of 64 prompt tokens (4 warps x 16) for one query head over the
// user's cache rows [0, position]: S = Q K^T and O = P V on bf16 m16n8k16 MMAs, softmax online
// over key blocks of 64 rows double-buffered in shared memory (rows padded by 16 bytes so the
// matrix loads are free of bank conflicts).

constexpr int PA_ROWS = 64;
constexpr int PA_THREADS = 128;

__device__ __forceinline__ void mma16816(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                         uint32_t b0, uint32_t b1) {
  asm("mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

__device__ __forceinline__ void ldsm_x4(uint32_t &r0, uint32_t &r1, uint32_t &r2, uint32_t &r3, uint32_t addr) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr)
               : "memory");
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t &r0, uint32_t &r1, uint32_t &r2, uint32_t &r3, uint32_t addr) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr)
               : "memory");
}

__device__ __forceinline__ void cp_async16(uint32_t dst, const void *src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(dst), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
__device__ __forceinline__ void cp_async_wait_all() { asm volatile("cp.async.wait_group 0;" ::: "memory"); }

template <int HD>
struct PaLayout {
  static constexpr int ROW = (HD + 8) * 2;  // bytes per padded row
  static constexpr int TILE = PA_ROWS * ROW;
  static constexpr int Q_OFF = 0;
  static constexpr int K_OFF = TILE;          // 2 buffers
  static constexpr int V_OFF = 3 * TILE;      // 2 buffers
  static constexpr int POS_OFF = 5 * TILE;    // int [64]
  static constexpr int BYTES = POS_OFF + PA_ROWS * 4;
};

// Rows [r0, r0 + 64) of a [rows][HD] bf16 matrix (row stride ld elements) into a padded tile;
// rows at or above `limit` are zero.
template <int HD>
__device__ __forceinline__ void pa_load_tile(uint8_t *tile, const uint16_t *src, size_t ld, int r0, int limit) {
  constexpr int CH = HD / 8;
  for (int e = threadIdx.x; e < PA_ROWS * CH; e += PA_THREADS) {
    const int r = e / CH, ch = e % CH;
    uint8_t *dst = tile + r * PaLayout<HD>::ROW + ch * 16;
    if (r0 + r < limit)
      cp_async16(smem_addr(dst), src + (size_t)(r0 + r) * ld + ch * 8);
    else
      *reinterpret_cast<uint4 *>(dst) = make_uint4(0, 0, 0, 0);
  }
}

template <int HD>
__global__ void __launch_bounds__(PA_THREADS) prefill_attn_kernel(PrefillAttnParams p) {
  using L = PaLayout<HD>;
  extern __shared__ __align__(16) uint8_t sm[];
  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  const int g = lane / 4, c = lane % 4;
  // the longest blocks (latest tokens) first
  const int qb = gridDim.x - 1 - blockIdx.x;
  const int h = blockIdx.y, kvh = h / (p.n_heads / p.n_kv_heads);
  const int t0 = qb * PA_ROWS;
  int *s_pos = reinterpret_cast<int *>(sm + L::POS_OFF);
  if (threadIdx.x < PA_ROWS) s_pos[threadIdx.x] = t0 + threadIdx.x < p.T ? p.positions[t0 + threadIdx.x] : -1;
  pa_load_tile<HD>(sm + L::Q_OFF, p.q + h * HD, p.ldq, t0, p.T);
  cp_async_commit();
  __syncthreads();
  int max_pos = -1;
  for (int i = 0; i < PA_ROWS; ++i) max_pos = max(max_pos, s_pos[i]);
  const int n_kb = (max_pos + PA_ROWS) / PA_ROWS;  // key blocks covering [0, max_pos]
  const int kv_limit = min(max_pos + 1, p.max_ctx);
  const size_t head_base = ((size_t)p.slot * p.n_kv_heads + kvh) * p.max_ctx * HD;
  const uint16_t *kg = p.kcache + head_base, *vg = p.vcache + head_base;
  if (n_kb > 0) {
    pa_load_tile<HD>(sm + L::K_OFF, kg, HD, 0, kv_limit);
    pa_load_tile<HD>(sm + L::V_OFF, vg, HD, 0, kv_limit);
  }
  cp_async_commit();
  const int qp0 = s_pos[16 * warp + g], qp1 = s_pos[16 * warp + g + 8];
  cp_async_wait_all();
  __syncthreads();
  // Q fragments of this warp's 16 rows
  uint32_t qf[HD / 16][4];
  {
    const uint32_t qbase = smem_addr(sm + L::Q_OFF) + (16 * warp + (lane % 16)) * L::ROW + (lane / 16) * 16;
#pragma unroll
    for (int kk = 0; kk < HD / 16; ++kk) ldsm_x4(qf[kk][0], qf[kk][1], qf[kk][2], qf[kk][3], qbase + kk * 32);
  }
  float oacc[HD / 8][4] = {};
  float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;
  for (int kb = 0; kb < n_kb; ++kb) {
    const int buf = kb & 1;
    if (kb + 1 < n_kb) {  // the next block loads while this one is used
      pa_load_tile<HD>(sm + L::K_OFF + (buf ^ 1) * L::TILE, kg, HD, (kb + 1) * PA_ROWS, kv_limit);
      pa_load_tile<HD>(sm + L::V_OFF + (buf ^ 1) * L::TILE, vg, HD, (kb + 1) * PA_ROWS, kv_limit);
    }
    cp_async_commit();
    const uint32_t kbase = smem_addr(sm + L::K_OFF + buf * L::TILE);
    const uint32_t vbase = smem_addr(sm + L::V_OFF + buf * L::TILE);
    // S = Q K^T: 8 key tiles of 8
    float s[8][4];
#pragma unroll
    for (int nt = 0; nt < 8; ++nt) {
      s[nt][0] = s[nt][1] = s[nt][2] = s[nt][3] = 0.f;
#pragma unroll
      for (int kk = 0; kk < HD / 16; kk += 2) {
        uint32_t b0, b1, b2, b3;
        ldsm_x4(b0, b1, b2, b3, kbase + (nt * 8 + (lane % 8)) * L::ROW + kk * 32 + (lane / 8) * 16);
        mma16816(s[nt], qf[kk][0], qf[kk][1], qf[kk][2], qf[kk][3], b0, b1);
        mma16816(s[nt], qf[kk + 1][0], qf[kk + 1][1], qf[kk + 1][2], qf[kk + 1][3], b2, b3);
      }
    }
    // scale, causal mask, online softmax (rows g and g + 8 of the warp)
    float mx0 = -INFINITY, mx1 = -INFINITY;
#pragma unroll
    for (int nt = 0; nt < 8; ++nt) {
      const int kp = kb * PA_ROWS + nt * 8 + 2 * c;
      s[nt][0] = kp <= qp0 ? s[nt][0] * p.scale_log2 : -INFINITY;
      s[nt][1] = kp + 1 <= qp0 ? s[nt][1] * p.scale_log2 : -INFINITY;
      s[nt][2] = kp <= qp1 ? s[nt][2] * p.scale_log2 : -INFINITY;
      s[nt][3] = kp + 1 <= qp1 ? s[nt][3] * p.scale_log2 : -INFINITY;
      mx0 = fmaxf(mx0, fmaxf(s[nt][0], s[nt][1]));
      mx1 = fmaxf(mx1, fmaxf(s[nt][2], s[nt][3]));
    }
    mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 1));
    mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 2));
    mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 1));
    mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 2));
    const float mn0 = fmaxf(m0, mx0), mn1 = fmaxf(m1, mx1);
    // rows with no visible key yet keep m = -inf; their factors stay 0 / 1
    const float base0 = mn0 == -INFINITY ? 0.f : mn0, base1 = mn1 == -INFINITY ? 0.f : mn1;
    const float corr0 = exp2f(m0 - base0), corr1 = exp2f(m1 - base1);
    m0 = mn0;
    m1 = mn1;
    float rs0 = 0.f, rs1 = 0.f;
#pragma unroll
    for (int nt = 0; nt < 8; ++nt) {
      s[nt][0] = exp2f(s[nt][0] - base0);
      s[nt][1] = exp2f(s[nt][1] - base0);
      s[nt][2] = exp2f(s[nt][2] - base1);
      s[nt][3] = exp2f(s[nt][3] - base1);
      rs0 += s[nt][0] + s[nt][1];
      rs1 += s[nt][2] + s[nt][3];
    }
    l0 = l0 * corr0 + rs0;
    l1 = l1 * corr1 + rs1;
#pragma unroll
    for (int dt = 0; dt < HD / 8; ++dt) {
      oacc[dt][0] *= corr0;
      oacc[dt][1] *= corr0;
      oacc[dt][2] *= corr1;
      oacc[dt][3] *= corr1;
    }
    // O += P V: 4 key steps of 16; V fragments by transposed matrix loads
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const uint32_t a0 = pack_bf16(s[2 * j][0], s[2 * j][1]), a1 = pack_bf16(s[2 * j][2], s[2 * j][3]);
      const uint32_t a2 = pack_bf16(s[2 * j + 1][0], s[2 * j + 1][1]), a3 = pack_bf16(s[2 * j + 1][2], s[2 * j + 1][3]);
#pragma unroll
      for (int dt = 0; dt < HD / 8; dt += 2) {
        uint32_t b0, b1, b2, b3;
        ldsm_x4_t(b0, b1, b2, b3,
                  vbase + (j * 16 + (lane % 8) + ((lane / 8) & 1) * 8) * L::ROW + (dt + lane / 16) * 16);
        mma16816(oacc[dt], a0, a1, a2, a3, b0, b1);
        mma16816(oacc[dt + 1], a0, a1, a2, a3, b2, b3);
      }
    }
    cp_async_wait_all();
    __syncthreads();
  }
  // row sums over the quad, normalize, store bf16
  l0 += __shfl_xor_sync(0xffffffffu, l0, 1);
  l0 += __shfl_xor_sync(0xffffffffu, l0, 2);
  l1 += __shfl_xor_sync(0xffffffffu, l1, 1);
  l1 += __shfl_xor_sync(0xffffffffu, l1, 2);
  const float inv0 = l0 > 0.f ? 1.f / l0 : 0.f, inv1 = l1 > 0.f ? 1.f / l1 : 0.f;
  const int ta = t0 + 16 * warp + g, tb = ta + 8;
#pragma unroll
  for (int dt = 0; dt < HD / 8; ++dt) {
    const int col = h * HD + dt * 8 + 2 * c;
    uint32_t hi, lo;
    if (ta < p.T) {
      split_pack(oacc[dt][0] * inv0, oacc[dt][1] * inv0, hi, lo, p.f16, p.err);
      *reinterpret_cast<uint32_t *>(p.o + (size_t)ta * p.ldo + col) = hi;
      *reinterpret_cast<uint32_t *>(p.o_lo + (size_t)ta * p.ldo + col) = lo;
    }
    if (tb < p.T) {
      split_pack(oacc[dt][2] * inv1, oacc[dt][3] * inv1, hi, lo, p.f16, p.err);
      *reinterpret_cast<uint32_t *>(p.o + (size_t)tb * p.ldo + col) = hi;
      *reinterpret_cast<uint32_t *>(p.o_lo + (size_t)tb * p.ldo + col) = lo;
    }
  }
}

// ---------------------------------------------------------------------------- small kernels
// One block per prompt token: its input row (embedding row or given hidden state) and its
// position, refused (-1, ERR_POSITION) outside [0, max_ctx) or when an earlier token of the pass
// holds the same position.
__global__ void prefill_input_kernel(const int *ids, const float *hidden_in, const int *positions_in, int T,
                                     const uint16_t *embed, int vocab, int d, int ldh, float *h, int *positions,
                                     int max_ctx, unsigned *err) {
  const int t = blockIdx.x;
  __shared__ int s_bad;
  if (threadIdx.x == 0) s_bad = 0;
  __syncthreads();
  const int pos = positions_in[t];
  for (int j = threadIdx.x; j < t; j += blockDim.x)
    if (positions_in[j] == pos) s_bad = 1;
  __syncthreads();
  if (threadIdx.x == 0) {
    const bool ok = pos >= 0 && pos < max_ctx && !s_bad;
    if (!ok) atomicOr(err, ERR_POSITION);
    positions[t] = ok ? pos : -1;
  }
  int id = 0;
  if (embed) {
    id = ids[t];
    if (id < 0 || id >= vocab) {
      if (threadIdx.x == 0) atomicOr(err, ERR_TOKEN);
      id = 0;
    }
  }
  for (int i = threadIdx.x; i < d; i += blockDim.x)
    h[(size_t)t * ldh + i] = embed ? bf16_to_f32(embed[(size_t)id * d + i]) : hidden_in[(size_t)t * d + i];
}

// x[t] = h[t] / rms(h[t]) * g as hi and lo 16-bit terms, one block per token, four elements per
// thread step (d a multiple of 8; h, g and x rows 16-byte aligned).
__global__ void prefill_rmsnorm_kernel(const float *h, int ldh, int d, const float *g, float eps, uint16_t *x,
                                       uint16_t *x_lo, int ldx, int f16, unsigned *err) {
  const int t = blockIdx.x, d4 = d / 4;
  const float4 *row = reinterpret_cast<const float4 *>(h + (size_t)t * ldh);
  float ss = 0.f;
  for (int i = threadIdx.x; i < d4; i += blockDim.x) {
    const float4 v = row[i];
    ss += v.x * v.x + v.y * v.y + v.z * v.z + v.w * v.w;
  }
  __shared__ float red[32];
  for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
  if (threadIdx.x % 32 == 0) red[threadIdx.x / 32] = ss;
  __syncthreads();
  if (threadIdx.x < 32) {
    float v = threadIdx.x < blockDim.x / 32 ? red[threadIdx.x] : 0.f;
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    if (threadIdx.x == 0) red[0] = v;
  }
  __syncthreads();
  const float inv = rsqrtf(red[0] / d + eps);
  const float4 *g4 = reinterpret_cast<const float4 *>(g);
  uint2 *xh = reinterpret_cast<uint2 *>(x + (size_t)t * ldx), *xl = reinterpret_cast<uint2 *>(x_lo + (size_t)t * ldx);
  for (int i = threadIdx.x; i < d4; i += blockDim.x) {
    const float4 v = row[i], gg = g4[i];
    uint2 hi, lo;
    split_pack(v.x * inv * gg.x, v.y * inv * gg.y, hi.x, lo.x, f16, err);
    split_pack(v.z * inv * gg.z, v.w * inv * gg.w, hi.y, lo.y, f16, err);
    xh[i] = hi;
    xl[i] = lo;
  }
}

// One thread per 8 consecutive outputs of one row (16 bytes): the int4 tile stores the nibble of
// (row rb*64 + r16*16 + gid + 8 ((i >> 1) & 1), column kt*256 + 128 h + 16 (4 q + j) + 2 tig +
// 8 (i & 1) + ((i >> 2) & 1)) as nibble i of word j + 4 lane + 128 q + 256 r16 + 1024 h
// (lane = 4 gid + tig), and the row's group scales after the codes; so the 8 columns
// 16 m + 8 e .. + 7 of a row come from lanes tig = 0..3, nibbles i with i & 1 = e.
__global__ void dequant_int4_f16_kernel(const uint8_t *tiles4, int n_rb, int n_kt, uint16_t *dst) {
  const long long total = (long long)n_rb * n_kt * RB * (KT4 / 8);
  for (long long e = blockIdx.x * (long long)blockDim.x + threadIdx.x; e < total;
       e += (long long)gridDim.x * blockDim.x) {
    const int c8 = (int)(e % (KT4 / 8));      // 8-column chunk within the int4 tile (0..31)
    const long long rt = e / (KT4 / 8);
    const int r = (int)(rt % RB);              // row within the row block
    const long long t = rt / RB;               // int4 tile index rb * n_kt + kt
    const int col0 = c8 * 8;                   // 0..248
    const int h = col0 >> 7, m = (col0 >> 4) & 7, ebit = (col0 >> 3) & 1;
    const int q = m >> 2, j = m & 3, r16 = r >> 4, gid = r & 7, rhalf = (r >> 3) & 1;
    const uint8_t *tile = tiles4 + (size_t)t * TILE4_BYTES;
    const uint32_t *words = reinterpret_cast<const uint32_t *>(tile);
    const float sc = bf16_to_f32(reinterpret_cast<const uint16_t *>(tile + TILE4_CODE_BYTES)[tile4_scale_index(r, col0 >> 6)]);
    uint16_t out[8];
#pragma unroll
    for (int tig = 0; tig < 4; ++tig) {
      const uint32_t w = words[j + 4 * (4 * gid + tig) + 128 * q + 256 * r16 + 1024 * h];
#pragma unroll
      for (int b = 0; b < 2; ++b) {
        const int i = ebit | (rhalf << 1) | (b << 2);
        const int nib = (int)((w >> (4 * i)) & 0xFu);
        out[2 * tig + b] = f32_to_f16_rn((float)(nib >= 8 ? nib - 16 : nib) * sc);
      }
    }
    // fp16 tile (rb, 2 kt + h): row r, columns (col0 & 127) ..
    const long long rb = t / n_kt, kt = t % n_kt;
    uint16_t *d = dst + ((size_t)(rb * 2 * n_kt + 2 * kt + h) * RB + r) * KT + (col0 & 127);
    *reinterpret_cast<uint4 *>(d) = make_uint4(out[0] | (uint32_t)out[1] << 16, out[2] | (uint32_t)out[3] << 16,
                                               out[4] | (uint32_t)out[5] << 16, out[6] | (uint32_t)out[7] << 16);
  }
}

// fp32 rows [T][K] (stride ldx) -> hi and lo bf16 terms (stride ld).
__global__ void split_rows_kernel(const float *x, int K, int ldx, uint16_t *hi, uint16_t *lo, int ld) {
  const int t = blockIdx.x;
  for (int i = threadIdx.x; i < K; i += blockDim.x)
    split_bf16(x[(size_t)t * ldx + i], hi[(size_t)t * ld + i], lo[(size_t)t * ld + i]);
}

// next_ids[t]: the lowest index among the largest logits, over the column tiles' partial maxima;
// one warp per token (each lane scans every 32nd tile, then the warp keeps the largest value and,
// among equal values, the lowest index).
__global__ void prefill_argmax_kernel(const float *amax, const int *aidx, int n_tiles, int T, int *next_ids) {
  const int t = blockIdx.x * (blockDim.x / 32) + threadIdx.x / 32, lane = threadIdx.x % 32;
  if (t >= T) return;  // uniform per warp
  float best = -INFINITY;
  int bi = 0x7FFFFFFF;
  for (int j = lane; j < n_tiles; j += 32) {
    const float v = amax[(size_t)t * n_tiles + j];
    const int i = aidx[(size_t)t * n_tiles + j];
    if (v > best || (v == best && i < bi)) {
      best = v;
      bi = i;
    }
  }
  for (int o = 16; o > 0; o >>= 1) {
    const float ov = __shfl_xor_sync(0xffffffffu, best, o);
    const int oi = __shfl_xor_sync(0xffffffffu, bi, o);
    if (ov > best || (ov == best && oi < bi)) {
      best = ov;
      bi = oi;
    }
  }
  if (lane == 0) next_ids[t] = bi == 0x7FFFFFFF ? 0 : bi;
}

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (!fn) {
    void *p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    else
      cudaGetLastError();
  }
  return fn;
}

}  // namespace

// ---------------------------------------------------------------------------- host side
// Activation rows [rows][K] bf16 at row stride ld (a multiple of 8): boxes of 64 columns x PG_M
// rows; columns >= K and rows >= rows read as zero.
int encode_act_map(CUtensorMap *map, const uint16_t *base, int K, int rows, int ld) {
  auto fn = encode_fn();
  if (!fn || ld % 8 != 0 || (reinterpret_cast<uintptr_t>(base) & 15) != 0) return -1;
  const cuuint64_t dims[2] = {(cuuint64_t)K, (cuuint64_t)rows};
  const cuuint64_t strides[1] = {(cuuint64_t)ld * 2};
  const cuuint32_t box[2] = {PG_K, PG_M};
  const cuuint32_t estr[2] = {1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<uint16_t *>(base), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS
             ? 0
             : -1;
}

// Weight tiles [n_rb][n_kt][RB][KT] bf16 as a 4-D tensor (column, row, K tile, row block):
// boxes of 64 columns x RB rows x 1 K tile x PG_N / RB row blocks; row blocks >= n_rb read as zero.
int encode_tiles_map(CUtensorMap *map, const uint8_t *tiles, int n_kt, int n_rb) {
  auto fn = encode_fn();
  if (!fn) return -1;
  const cuuint64_t dims[4] = {(cuuint64_t)KT, (cuuint64_t)RB, (cuuint64_t)n_kt, (cuuint64_t)n_rb};
  const cuuint64_t strides[3] = {(cuuint64_t)KT * 2, (cuuint64_t)TILE_BYTES, (cuuint64_t)TILE_BYTES * n_kt};
  const cuuint32_t box[4] = {PG_K, RB, 1, PG_N / RB};
  const cuuint32_t estr[4] = {1, 1, 1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<uint8_t *>(tiles), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS
             ? 0
             : -1;
}

template <int MODE>
static cudaError_t launch_mode(const CUtensorMap &a, const CUtensorMap &a2, const CUtensorMap &b, int n_kt,
                               const PrefillEpiParams &ep, cudaStream_t s) {
  static bool smem_set = false;
  if (!smem_set) {
    cudaError_t e = cudaFuncSetAttribute(prefill_gemm_persistent<MODE>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)PG_SMEM);
    if constexpr (MODE != PE_ARGMAX)
      if (e == cudaSuccess)
        e = cudaFuncSetAttribute(prefill_gemm_kernel<MODE>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)PG_SMEM);
    if (e != cudaSuccess) return e;
    smem_set = true;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.blockDim = dim3(PG_THREADS);
  cfg.dynamicSmemBytes = PG_SMEM;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 1;
  attr[0].val.clusterDim.y = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  PrefillEpiParams e = ep;
  if constexpr (MODE != PE_ARGMAX) {
    // the largest split count not above the chosen one whose cluster fits on the device
    static int fits[9] = {};  // 0 unknown, 1 yes, -1 no
    while (e.splits > 1) {
      if (fits[e.splits] == 0) {
        attr[0].val.clusterDim.z = e.splits;
        cfg.gridDim = dim3(1, 1, e.splits);
        int n = 0;
        fits[e.splits] =
            cudaOccupancyMaxActiveClusters(&n, prefill_gemm_kernel<MODE>, &cfg) == cudaSuccess && n > 0 ? 1 : -1;
        cudaGetLastError();
      }
      if (fits[e.splits] > 0) break;
      e.splits /= 2;
    }
    if (e.splits > 1) {
      cfg.gridDim = dim3((e.T + PG_M - 1) / PG_M, (e.N + PG_N - 1) / PG_N, e.splits);
      attr[0].val.clusterDim.z = e.splits;
      return cudaLaunchKernelEx(&cfg, prefill_gemm_kernel<MODE>, a, a2, b, 2 * n_kt, e);
    }
  }
  // one persistent CTA per SM (fewer if there are fewer tiles)
  static int n_sm = 0;
  if (!n_sm) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&n_sm, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
      return cudaErrorInvalidDevice;
  }
  const long long tiles = (long long)((e.T + PG_M - 1) / PG_M) * ((e.N + PG_N - 1) / PG_N);
  cfg.gridDim = dim3((unsigned)std::min<long long>(tiles, n_sm));
  cfg.blockDim = dim3(PP_THREADS);
  cfg.numAttrs = 0;
  return cudaLaunchKernelEx(&cfg, prefill_gemm_persistent<MODE>, a, a2, b, 2 * n_kt, e);
}

int prefill_splits(int T, int N, int n_kt, int n_sm) {
  const long long base = (long long)((T + PG_M - 1) / PG_M) * ((N + PG_N - 1) / PG_N);
  const int n_kb = 2 * n_kt;
  // waves x (K blocks per split + a fixed cost per CTA of about 6 K blocks: pipeline fill and
  // epilogue; 1.5 more for the cluster reduction), over the split counts 1, 2, 4, 8 that keep
  // at least 4 K blocks each
  int best = 1;
  double best_t = 1e30;
  for (int S = 1; S <= 8 && n_kb / S >= 4; S *= 2) {
    const double waves = (double)((base * S + n_sm - 1) / n_sm);
    const double t = waves * ((double)n_kb / S + 6.0 + (S > 1 ? 1.5 : 0.0));
    if (t < best_t - 1e-9) {
      best_t = t;
      best = S;
    }
  }
  return best;
}

cudaError_t launch_prefill_gemm(int mode, const CUtensorMap &a, const CUtensorMap &a2, const CUtensorMap &b,
                                int n_kt, const PrefillEpiParams &ep, cudaStream_t s) {
  if (ep.T <= 0 || ep.N <= 0) return cudaSuccess;
  if (ep.splits != 1 && ep.splits != 2 && ep.splits != 4 && ep.splits != 8) return cudaErrorInvalidValue;
  if (mode == PE_ARGMAX && ep.splits != 1) return cudaErrorInvalidValue;  // partial maxima are per tile
  switch (mode) {
    case PE_STORE: return launch_mode<PE_STORE>(a, a2, b, n_kt, ep, s);
    case PE_RESID: return launch_mode<PE_RESID>(a, a2, b, n_kt, ep, s);
    case PE_SWIGLU: return launch_mode<PE_SWIGLU>(a, a2, b, n_kt, ep, s);
    case PE_QKV: return launch_mode<PE_QKV>(a, a2, b, n_kt, ep, s);
    case PE_ARGMAX: return launch_mode<PE_ARGMAX>(a, a2, b, n_kt, ep, s);
    default: return cudaErrorInvalidValue;
  }
}

template <int HD>
static cudaError_t launch_attn_hd(const PrefillAttnParams &p, cudaStream_t s) {
  static bool attr = false;
  const int bytes = PaLayout<HD>::BYTES;
  if (!attr) {
    cudaError_t e = cudaFuncSetAttribute(prefill_attn_kernel<HD>, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
    if (e != cudaSuccess) return e;
    attr = true;
  }
  const dim3 grid((p.T + PA_ROWS - 1) / PA_ROWS, p.n_heads);
  prefill_attn_kernel<HD><<<grid, PA_THREADS, bytes, s>>>(p);
  return cudaGetLastError();
}

cudaError_t launch_prefill_attention(const PrefillAttnParams &p, int hd, cudaStream_t s) {
  if (p.T <= 0) return cudaSuccess;
  return hd == 128 ? launch_attn_hd<128>(p, s) : launch_attn_hd<64>(p, s);
}

cudaError_t launch_prefill_input(const int *ids, const float *hidden_in, const int *positions_in, int T,
                                 const uint16_t *embed, int vocab, int d, int ldh, float *h, int *positions,
                                 int max_ctx, unsigned *err, cudaStream_t s) {
  prefill_input_kernel<<<T, 256, 0, s>>>(ids, hidden_in, positions_in, T, embed, vocab, d, ldh, h, positions,
                                         max_ctx, err);
  return cudaGetLastError();
}

cudaError_t launch_prefill_rmsnorm(const float *h, int ldh, int T, int d, const float *g, float eps, uint16_t *x,
                                   uint16_t *x_lo, int ldx, int f16, unsigned *err, cudaStream_t s) {
  prefill_rmsnorm_kernel<<<T, 256, 0, s>>>(h, ldh, d, g, eps, x, x_lo, ldx, f16, err);
  return cudaGetLastError();
}

cudaError_t launch_dequant_int4_f16(const uint8_t *tiles4, int n_rb, int n_kt, uint16_t *dst, cudaStream_t s) {
  dequant_int4_f16_kernel<<<8 * 152, 256, 0, s>>>(tiles4, n_rb, n_kt, dst);
  return cudaGetLastError();
}

cudaError_t launch_split_bf16(const float *x, int T, int K, int ldx, uint16_t *hi, uint16_t *lo, int ld,
                              cudaStream_t s) {
  split_rows_kernel<<<T, 256, 0, s>>>(x, K, ldx, hi, lo, ld);
  return cudaGetLastError();
}

cudaError_t launch_prefill_argmax(const float *amax, const int *aidx, int n_tiles, int T, int *next_ids,
                                  cudaStream_t s) {
  prefill_argmax_kernel<<<(T + 3) / 4, 128, 0, s>>>(amax, aidx, n_tiles, T, next_ids);
  return cudaGetLastError();
}

}  // namespace kfl

// ---------------------------------------------------------------------------- C ABI
extern "C" int kfl_matmul_bf16w(const float *x, int T, int K, int ldx, const uint16_t *w, int N, float *y, int ldy,
                                void *cuda_stream) {
  using namespace kfl;
  if (!x || !w || !y || T < 1 || K < 1 || N < 1 || ldx < K || ldy < N || ldy % 4 != 0 ||
      (reinterpret_cast<uintptr_t>(y) & 15) != 0)
    return KFL_ERR_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(cuda_stream);
  const int n_rb = (N + RB - 1) / RB, n_kt = (K + KT - 1) / KT, ld = (K + 63) / 64 * 64;
  int dev = 0, n_sm = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&n_sm, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) {
    cudaGetLastError();
    return KFL_ERR_CUDA;
  }
  const int splits = prefill_splits(T, N, n_kt, n_sm);
  void *mem = nullptr;
  const size_t tile_bytes = (size_t)n_rb * n_kt * TILE_BYTES, x_bytes = (size_t)T * ld * 2;
  if (cudaMalloc(&mem, tile_bytes + 2 * x_bytes + 16) != cudaSuccess) {
    cudaGetLastError();
    return KFL_ERR_OOM;
  }
  uint8_t *tiles = static_cast<uint8_t *>(mem);
  uint16_t *xhi = reinterpret_cast<uint16_t *>(tiles + tile_bytes);
  uint16_t *xlo = xhi + (size_t)T * ld;
  unsigned *err = reinterpret_cast<unsigned *>(xlo + (size_t)T * ld);
  int rc = KFL_OK;
  CUtensorMap mh, ml, mb;
  if (cudaMemsetAsync(err, 0, 4, s) != cudaSuccess ||
      launch_split_bf16(x, T, K, ldx, xhi, xlo, ld, s) != cudaSuccess ||
      launch_repack_bf16(w, N, K, nullptr, N, n_rb, n_kt, tiles, s) != cudaSuccess) {
    rc = KFL_ERR_CUDA;
  } else if (encode_act_map(&mh, xhi, K, T, ld) || encode_act_map(&ml, xlo, K, T, ld) ||
             encode_tiles_map(&mb, tiles, n_kt, n_rb)) {
    rc = KFL_ERR_CUDA;
  } else {
    PrefillEpiParams e = {};
    e.T = T;
    e.N = N;
    e.out = y;
    e.ldo = ldy;
    e.err = err;
    e.splits = splits;
    unsigned h_err = 0;
    if (launch_prefill_gemm(PE_STORE, mh, ml, mb, n_kt, e, s) != cudaSuccess || cudaStreamSynchronize(s) != cudaSuccess ||
        cudaMemcpy(&h_err, err, 4, cudaMemcpyDeviceToHost) != cudaSuccess)
      rc = KFL_ERR_CUDA;
    else if (h_err & ERR_TIMEOUT)
      rc = KFL_ERR_TIMEOUT;
  }
  cudaStreamSynchronize(s);
  cudaFree(mem);
  cudaGetLastError();
  return rc;
}
