// Grouped-query decode attention, split along the cached positions (flash-decoding).
//
// User b's new token at position P_b attends to its cached slots [0, P_b] (its own K/V were
// appended by the QKV epilogue).  A CTA handles one (chunk of positions, KV head, user): it
// loads the chunk's K and V rows once for all G = Hq/Hkv query heads that share the KV head,
// keeps an online-softmax state (running max m, running sum l, weighted V sum) per head, and
// writes (m, l, acc) for its chunk.  The last CTA of a (user, KV head) to finish (atomic
// ticket, no spin) merges the chunks in chunk order, so the result does not depend on
// scheduling.  Scores are kept in the log2 domain (q is pre-scaled by log2(e)/sqrt(hd)).
#include "common.cuh"

#include <math.h>

namespace kfl {

constexpr int ATT_THREADS = 128;
constexpr int ATT_SUB = 64;  // positions per shared-memory sub-tile
constexpr int ATT_MAXG = 8;
constexpr int ATT_MERGE_MAX = 2048;  // chunks x heads merged in shared memory (fits the K buffers)

__device__ __forceinline__ void cp_async16(void *dst, const void *src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_addr(dst)), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

template <int HD>
struct AttnSmem {
  static constexpr int KROW = HD * 2 + 16;  // padded K row (bytes): conflict-free row-per-lane reads
  static constexpr int VROW = HD * 2;
  static constexpr int K_OFF = 0;
  static constexpr int V_OFF = K_OFF + 2 * ATT_SUB * KROW;
  static constexpr int Q_OFF = V_OFF + 2 * ATT_SUB * VROW;
  static constexpr int S_OFF = Q_OFF + ATT_MAXG * HD * 4;
  static constexpr int M_OFF = S_OFF + ATT_MAXG * ATT_SUB * 4;
  static constexpr int BYTES = M_OFF + 3 * ATT_MAXG * 4;
};

template <int HD>
__global__ void __launch_bounds__(ATT_THREADS) attn_kernel(const __grid_constant__ AttnParams p) {
  using L = AttnSmem<HD>;
  extern __shared__ __align__(128) uint8_t sm[];
  uint8_t *sk = sm + L::K_OFF;
  uint8_t *sv = sm + L::V_OFF;
  float *sq = reinterpret_cast<float *>(sm + L::Q_OFF);
  float *ss = reinterpret_cast<float *>(sm + L::S_OFF);
  float *s_m = reinterpret_cast<float *>(sm + L::M_OFF);
  float *s_l = s_m + ATT_MAXG;
  float *s_alpha = s_l + ATT_MAXG;
  __shared__ int s_last;

  const int c = blockIdx.x, kvh = blockIdx.y, b = blockIdx.z;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int G = p.n_heads / p.n_kv_heads;

  pdl_launch_dependents();
  pdl_wait();

  const int P = p.positions[b];
  if (P < 0 || P >= p.max_ctx) {
    // the input kernel flagged the position; leave a defined (zero) output
    if (c == 0)
      for (int e = tid; e < G * HD; e += ATT_THREADS) p.o[(size_t)b * p.ldo + kvh * G * HD + e] = 0.f;
    return;
  }
  const int ntok = P + 1;
  const int nc = (ntok + p.chunk - 1) / p.chunk;
  if (c >= nc) return;
  const int start = c * p.chunk;
  const int end = min(ntok, start + p.chunk);

  const size_t head_base = ((size_t)b * p.n_kv_heads + kvh) * p.max_ctx;
  const uint16_t *kg = p.kcache + head_base * HD;
  const uint16_t *vg = p.vcache + head_base * HD;

  for (int e = tid; e < G * HD; e += ATT_THREADS)
    sq[e] = p.q[(size_t)b * p.n_heads * HD + kvh * G * HD + e] * p.scale_log2;
  if (tid < ATT_MAXG) {
    s_m[tid] = -INFINITY;
    s_l[tid] = 0.f;
  }

  auto load_sub = [&](int sub, int buf) {
    const int p0 = start + sub * ATT_SUB;
    const int cnt = min(ATT_SUB, end - p0);
    constexpr int CH = HD / 8;  // 16-byte chunks per row
    for (int e = tid; e < cnt * CH; e += ATT_THREADS) {
      const int r = e / CH, ch = e % CH;
      cp_async16(sk + buf * ATT_SUB * L::KROW + r * L::KROW + ch * 16, kg + (size_t)(p0 + r) * HD + ch * 8);
      cp_async16(sv + buf * ATT_SUB * L::VROW + r * L::VROW + ch * 16, vg + (size_t)(p0 + r) * HD + ch * 8);
    }
    cp_async_commit();
  };

  // PV mapping: HD=128 -> thread owns dim tid, all heads; HD=64 -> dim tid&63, heads of parity tid>>6
  constexpr int DSPLIT = (HD == 128) ? 1 : 2;
  const int d = tid % HD;
  const int gpar = tid / HD;
  float acc[ATT_MAXG];
#pragma unroll
  for (int g = 0; g < ATT_MAXG; ++g) acc[g] = 0.f;

  const int nsub = (end - start + ATT_SUB - 1) / ATT_SUB;
  load_sub(0, 0);
  for (int it = 0; it < nsub; ++it) {
    const int buf = it & 1;
    if (it + 1 < nsub) {
      load_sub(it + 1, buf ^ 1);
      cp_async_wait<1>();
    } else {
      cp_async_wait<0>();
    }
    __syncthreads();
    const int p0 = start + it * ATT_SUB;
    const int cnt = min(ATT_SUB, end - p0);
    const uint8_t *kb = sk + buf * ATT_SUB * L::KROW;
    const uint8_t *vb = sv + buf * ATT_SUB * L::VROW;

    // scores: thread -> position tid & 63, heads of parity tid >> 6
    {
      const int pp = tid & (ATT_SUB - 1), half = tid >> 6;
      float dot[ATT_MAXG / 2];
#pragma unroll
      for (int k = 0; k < ATT_MAXG / 2; ++k) dot[k] = 0.f;
      if (pp < cnt) {
        const uint4 *kr = reinterpret_cast<const uint4 *>(kb + pp * L::KROW);
#pragma unroll 4
        for (int ch = 0; ch < HD / 8; ++ch) {
          const uint4 k4 = kr[ch];
          float kv[8];
          kv[0] = bf16_lo(k4.x); kv[1] = bf16_hi(k4.x); kv[2] = bf16_lo(k4.y); kv[3] = bf16_hi(k4.y);
          kv[4] = bf16_lo(k4.z); kv[5] = bf16_hi(k4.z); kv[6] = bf16_lo(k4.w); kv[7] = bf16_hi(k4.w);
#pragma unroll
          for (int k = 0; k < ATT_MAXG / 2; ++k) {
            const int g = half + 2 * k;
            if (g < G) {
              const float4 q0 = reinterpret_cast<const float4 *>(sq + g * HD)[ch * 2];
              const float4 q1 = reinterpret_cast<const float4 *>(sq + g * HD)[ch * 2 + 1];
              dot[k] = fmaf(kv[0], q0.x, dot[k]); dot[k] = fmaf(kv[1], q0.y, dot[k]);
              dot[k] = fmaf(kv[2], q0.z, dot[k]); dot[k] = fmaf(kv[3], q0.w, dot[k]);
              dot[k] = fmaf(kv[4], q1.x, dot[k]); dot[k] = fmaf(kv[5], q1.y, dot[k]);
              dot[k] = fmaf(kv[6], q1.z, dot[k]); dot[k] = fmaf(kv[7], q1.w, dot[k]);
            }
          }
        }
      }
#pragma unroll
      for (int k = 0; k < ATT_MAXG / 2; ++k) {
        const int g = half + 2 * k;
        if (g < G) ss[g * ATT_SUB + pp] = (pp < cnt) ? dot[k] : -INFINITY;
      }
    }
    __syncthreads();
    // online softmax update: warp w owns heads w, w + 4
    for (int g = warp; g < G; g += ATT_THREADS / 32) {
      const float a0 = ss[g * ATT_SUB + lane], a1 = ss[g * ATT_SUB + lane + 32];
      float mx = fmaxf(a0, a1);
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, off));
      const float m_old = s_m[g];
      const float m_new = fmaxf(m_old, mx);
      const float e0 = exp2f(a0 - m_new), e1 = exp2f(a1 - m_new);
      float sum = e0 + e1;
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, off);
      ss[g * ATT_SUB + lane] = e0;
      ss[g * ATT_SUB + lane + 32] = e1;
      __syncwarp();
      if (lane == 0) {
        const float alpha = exp2f(m_old - m_new);
        s_alpha[g] = alpha;
        s_l[g] = s_l[g] * alpha + sum;
        s_m[g] = m_new;
      }
    }
    __syncthreads();
    // acc = acc * alpha + P . V
#pragma unroll
    for (int k = 0; k < ATT_MAXG / DSPLIT; ++k) {
      const int g = gpar + DSPLIT * k;
      if (g < G) acc[k] *= s_alpha[g];
    }
    for (int pp = 0; pp < cnt; ++pp) {
      const float v = bf16_to_f32(reinterpret_cast<const uint16_t *>(vb + pp * L::VROW)[d]);
#pragma unroll
      for (int k = 0; k < ATT_MAXG / DSPLIT; ++k) {
        const int g = gpar + DSPLIT * k;
        if (g < G) acc[k] = fmaf(ss[g * ATT_SUB + pp], v, acc[k]);
      }
    }
    __syncthreads();
  }

  float *o = p.o + (size_t)b * p.ldo + kvh * G * HD;
  if (nc == 1) {
#pragma unroll
    for (int k = 0; k < ATT_MAXG / DSPLIT; ++k) {
      const int g = gpar + DSPLIT * k;
      if (g < G) o[g * HD + d] = acc[k] / s_l[g];
    }
    return;
  }
  const int pstride = HD + 2;
  float *part = p.partial + (((size_t)b * p.n_kv_heads + kvh) * p.n_chunks + c) * (ATT_MAXG * pstride);
#pragma unroll
  for (int k = 0; k < ATT_MAXG / DSPLIT; ++k) {
    const int g = gpar + DSPLIT * k;
    if (g < G) part[g * pstride + d] = acc[k];
  }
  if (tid < G) {
    part[tid * pstride + HD] = s_m[tid];
    part[tid * pstride + HD + 1] = s_l[tid];
  }
  __threadfence();
  __syncthreads();
  if (tid == 0) {
    int *tk = p.tickets + b * p.n_kv_heads + kvh;
    const int prev = atomicAdd(tk, 1);
    s_last = (prev == nc - 1);
    if (s_last) atomicExch(tk, 0);
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  // merge: stage every chunk's (m, l) in shared memory (the K buffers are free now), turn them
  // into per-chunk weights 2^(m_c - M) / L once per head, then each thread sums its outputs
  // over the chunks with independent loads
  const float *base = p.partial + (((size_t)b * p.n_kv_heads + kvh) * p.n_chunks) * (ATT_MAXG * pstride);
  float *wm = reinterpret_cast<float *>(sk);  // [nc][G] weights (host keeps nc * G <= ATT_MERGE_MAX)
  float *wl = wm + ATT_MERGE_MAX;             // [nc][G] l values
  for (int e = tid; e < nc * G; e += ATT_THREADS) {
    const int cc = e / G, g = e % G;
    const float *pc = base + (size_t)cc * ATT_MAXG * pstride + g * pstride;
    wm[e] = __ldcg(pc + HD);
    wl[e] = __ldcg(pc + HD + 1);
  }
  __syncthreads();
  for (int g = warp; g < G; g += ATT_THREADS / 32) {
    float M = -INFINITY;
    for (int cc = lane; cc < nc; cc += 32) M = fmaxf(M, wm[cc * G + g]);
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, off));
    float Lsum = 0.f;
    for (int cc = lane; cc < nc; cc += 32) Lsum += wl[cc * G + g] * exp2f(wm[cc * G + g] - M);
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) Lsum += __shfl_xor_sync(0xffffffffu, Lsum, off);
    __syncwarp();
    const float invL = 1.0f / Lsum;
    for (int cc = lane; cc < nc; cc += 32) wm[cc * G + g] = exp2f(wm[cc * G + g] - M) * invL;
  }
  __syncthreads();
#pragma unroll 1
  for (int k = 0; k < ATT_MAXG / DSPLIT; ++k) {
    const int g = gpar + DSPLIT * k;
    if (g >= G) continue;
    const float *pg = base + g * pstride + d;
    float O0 = 0.f, O1 = 0.f, O2 = 0.f, O3 = 0.f;
    int cc = 0;
    for (; cc + 4 <= nc; cc += 4) {
      const float a0 = __ldcg(pg + (size_t)cc * ATT_MAXG * pstride);
      const float a1 = __ldcg(pg + (size_t)(cc + 1) * ATT_MAXG * pstride);
      const float a2 = __ldcg(pg + (size_t)(cc + 2) * ATT_MAXG * pstride);
      const float a3 = __ldcg(pg + (size_t)(cc + 3) * ATT_MAXG * pstride);
      O0 = fmaf(wm[cc * G + g], a0, O0);
      O1 = fmaf(wm[(cc + 1) * G + g], a1, O1);
      O2 = fmaf(wm[(cc + 2) * G + g], a2, O2);
      O3 = fmaf(wm[(cc + 3) * G + g], a3, O3);
    }
    for (; cc < nc; ++cc) O0 = fmaf(wm[cc * G + g], __ldcg(pg + (size_t)cc * ATT_MAXG * pstride), O0);
    o[g * HD + d] = (O0 + O1) + (O2 + O3);
  }
}

cudaError_t prepare_attention() {
  cudaError_t e = cudaFuncSetAttribute(attn_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       AttnSmem<128>::BYTES);
  if (e != cudaSuccess) return e;
  return cudaFuncSetAttribute(attn_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize, AttnSmem<64>::BYTES);
}

template <int HD>
static cudaError_t launch_hd(const AttnParams &p, cudaStream_t s, bool pdl) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(p.n_chunks, p.n_kv_heads, p.batch);
  cfg.blockDim = dim3(ATT_THREADS);
  cfg.dynamicSmemBytes = AttnSmem<HD>::BYTES;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, attn_kernel<HD>, p);
}

cudaError_t launch_attention(const AttnParams &p, int head_dim, cudaStream_t s, bool pdl) {
  if (p.n_heads % p.n_kv_heads != 0 || p.n_heads / p.n_kv_heads > ATT_MAXG) return cudaErrorInvalidValue;
  if (p.n_chunks * (p.n_heads / p.n_kv_heads) > ATT_MERGE_MAX) return cudaErrorInvalidValue;
  if (head_dim == 128) return launch_hd<128>(p, s, pdl);
  if (head_dim == 64) return launch_hd<64>(p, s, pdl);
  return cudaErrorInvalidValue;
}

}  // namespace kfl
