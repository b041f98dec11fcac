// Decode attention, one thread-block cluster per (user, KV head), for the one-kernel-per-phase
// mode (the persistent stage kernel runs attn_unit of attn_core.cuh instead).
//
// User b's token at position P_b attends to its cached slots [0, P_b] (its own K/V were appended
// before this kernel), query head h reading KV head h / G.  The cluster's C CTAs split the
// positions in whole 64-position sub-tiles: CTA r takes sub-tiles [r n / C, (r + 1) n / C) of the
// n = ceil((P_b + 1) / 64).  Each keeps an online-softmax state (running max m, running sum l,
// unnormalised weighted sum of V) per head; the C partial states then meet through distributed
// shared memory: CTA r merges its share of the output's 32-element chunks, reading every CTA's
// (m, l) and partial sums in CTA order (deterministic), and writes them (int4 stages: also in
// the O projection's input form).  No global partial buffer, ticket or last-unit merge.
//
// Scores S = q K^T and the weighted sum P V run as bf16 m16n8k16 MMAs with fp32 accumulation.
// q and P enter as bf16 pairs (rounded value, bf16 of the rest: about 2^-17 relative): rows
// 0..7 of the MMA's A operand hold the heads' rounded parts and rows 8..15 their rests, so one
// MMA yields both products and the head's value is the sum of accumulator rows g and g + 8,
// which the same lane holds.  K and V are the cache's bf16 values, exact.  Scores: warp w takes
// positions 8w..8w+7; P V: warp w takes head dimensions hd/8 * w onwards; softmax: warp g takes
// head g.  Scores are in the log2 domain (q pre-scaled by log2(e)/sqrt(hd)).
#include "attn_core.cuh"

namespace kfl {

template <int HD>
__global__ void __launch_bounds__(ATT_THREADS) attn_cluster_kernel(const __grid_constant__ AttnParams p) {
  using L = AttnLayout<HD, 2>;
  extern __shared__ __align__(128) uint8_t sm[];
  __shared__ float s_w[MAX_CLUSTER_ATT][ATT_MAXG];  // merge: (m, then weight) of each CTA and head
  __shared__ float s_lw[MAX_CLUSTER_ATT][ATT_MAXG];
  pdl_launch_dependents();
  const int C = p.cluster;
  const int pair = blockIdx.x / C, r = blockIdx.x % C;  // r: the CTA's rank in its cluster
  const int b = pair / p.n_kv_heads, kvh = pair % p.n_kv_heads;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int G = p.n_heads / p.n_kv_heads;
  const int gid = lane >> 2, tig = lane & 3;
  const bool hrow = gid < G;
  auto stamp = [&](int slot) {
    if (p.trace && (int)blockIdx.x < p.trace_grid && tid == 0)
      p.trace[(size_t)blockIdx.x * TRACE_SLOTS + slot] = global_ns();
  };
  stamp(TR_CONS_GO);
  uint8_t *sk = sm + L::K_OFF;
  uint8_t *sv = sm + L::V_OFF;
  float *ss = reinterpret_cast<float *>(sm + L::S_OFF);
  float *s_m = reinterpret_cast<float *>(sm + L::M_OFF);
  float *s_l = s_m + ATT_MAXG;
  float *s_alpha = s_l + ATT_MAXG;
  uint4 *qf = reinterpret_cast<uint4 *>(sm + L::QF_OFF);
  uint4 *pf = reinterpret_cast<uint4 *>(sm + L::PF_OFF);

  const int P = p.positions[b];
  const bool valid = P >= 0 && P < p.max_ctx;
  int start = 0, end = 0;
  if (valid) {
    const int nsub = (P + ATT_SUB) / ATT_SUB;
    start = static_cast<int>((long long)r * nsub / C) * ATT_SUB;
    end = min(P + 1, static_cast<int>((long long)(r + 1) * nsub / C) * ATT_SUB);
  }
  const int nsub = end > start ? (end - start + ATT_SUB - 1) / ATT_SUB : 0;
  // the cached rows [0, lo) were written by earlier steps: the first two sub-tiles' copies of
  // them go out while the Q/K/V projection may still run; rows from lo (written by this step)
  // after the wait
  const int lo = valid ? attn_step_lo(p, b) : 0;
  for (int sub = 0; sub < 2 && sub < nsub; ++sub) {
    const int p0 = start + sub * ATT_SUB;
    attn_load_rows<HD, 2>(p, b, kvh, p0, min(ATT_SUB, end - p0), sub, 1, lo, P, sm, tid);
  }
  pdl_wait();
  stamp(TR_X_GO);
  for (int sub = 0; sub < 2 && sub < nsub; ++sub) {
    const int p0 = start + sub * ATT_SUB;
    attn_load_rows<HD, 2>(p, b, kvh, p0, min(ATT_SUB, end - p0), sub, 2, lo, P, sm, tid);
  }

  constexpr int KS = HD / 16;  // K steps of the scores
  constexpr int NT = HD / 64;  // P V n-tiles (8 dimensions) per warp: warp w owns dims NT*8*w ...
  const int n_base = warp * NT * 8;
  {
    // q (scaled to log2 units) as the scores' A fragments: entry (step, lane) = registers a0..a3:
    // rows gid (the heads' rounded parts) and gid + 8 (their rests), columns 2 tig, 2 tig + 1
    // (a0, a1) and + 8 (a2, a3); rows of heads >= G are zero
    if (tid < KS * 32) {
      const int st = tid >> 5, l = tid & 31, g = l >> 2, t = l & 3;
      uint4 f = make_uint4(0u, 0u, 0u, 0u);
      if (valid && g < G) {
        const float *qg = p.q + (size_t)b * p.n_heads * HD + (size_t)(kvh * G + g) * HD + 16 * st + 2 * t;
        const float2 x0 = __ldcg(reinterpret_cast<const float2 *>(qg));
        const float2 x1 = __ldcg(reinterpret_cast<const float2 *>(qg + 8));
        const float v[4] = {x0.x * p.scale_log2, x0.y * p.scale_log2, x1.x * p.scale_log2, x1.y * p.scale_log2};
        uint16_t hi[4], lo_[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          hi[i] = f32_to_bf16_rne(v[i]);
          lo_[i] = f32_to_bf16_rne(v[i] - bf16_to_f32(hi[i]));
        }
        f = make_uint4(hi[0] | ((uint32_t)hi[1] << 16), lo_[0] | ((uint32_t)lo_[1] << 16),
                       hi[2] | ((uint32_t)hi[3] << 16), lo_[2] | ((uint32_t)lo_[3] << 16));
      }
      qf[tid] = f;
    }
    // P fragments of rows of heads >= G stay zero
    if (tid < (ATT_SUB / 16) * 32 && ((tid & 31) >> 2) >= G) pf[tid] = make_uint4(0u, 0u, 0u, 0u);
  }
  if (tid < ATT_MAXG) {
    s_m[tid] = -INFINITY;
    s_l[tid] = 0.f;
  }
  float acc[NT][4];  // rows gid (P's rounded parts) and gid + 8 (rests): both head gid's
#pragma unroll
  for (int nt = 0; nt < NT; ++nt) acc[nt][0] = acc[nt][1] = acc[nt][2] = acc[nt][3] = 0.f;

  for (int it = 0; it < nsub; ++it) {
    const int buf = it & 1;
    if (it + 1 < nsub) {
      // sub-tiles 0 and 1 were issued above; from sub-tile 2 on, each goes out one step ahead.
      // Every copy group but the newest is then complete, this sub-tile's among them
      if (it >= 1) {
        const int p0 = start + (it + 1) * ATT_SUB;
        attn_load_rows<HD, 2>(p, b, kvh, p0, min(ATT_SUB, end - p0), buf ^ 1, 0, 0, -1, sm, tid);
      }
      cp_async_wait<1>();
    } else {
      cp_async_wait<0>();
    }
    att_sync();
    const int p0 = start + it * ATT_SUB;
    const int cnt = min(ATT_SUB, end - p0);
    const uint8_t *kb = sk + buf * ATT_SUB * L::KROW;
    uint8_t *vb = sv + buf * ATT_SUB * L::VROW;
    // rows past the sub-tile's positions take part in P V with weight 0: make them finite
    if (cnt < ATT_SUB)
      for (int e = tid; e < (ATT_SUB - cnt) * (HD / 8); e += ATT_THREADS)
        *reinterpret_cast<uint4 *>(vb + (cnt + e / (HD / 8)) * L::VROW + (e % (HD / 8)) * 16) = make_uint4(0u, 0u, 0u, 0u);
    {
      // scores of positions 8w .. 8w + 7 (MMA columns) for every head: one MMA per K step (two
      // accumulator chains by K-step parity); head gid's score = rows gid + gid + 8
      float sp[2][4] = {};
      const uint8_t *krow = kb + (8 * warp + gid) * L::KROW + 4 * tig;
#pragma unroll
      for (int s16 = 0; s16 < KS; ++s16) {
        const uint4 f = qf[s16 * 32 + lane];
        const uint32_t k0 = *reinterpret_cast<const uint32_t *>(krow + 32 * s16);
        const uint32_t k1 = *reinterpret_cast<const uint32_t *>(krow + 32 * s16 + 16);
        mma_bf16_full(sp[s16 & 1], f, k0, k1);
      }
      if (hrow) {
        const float s0 = (sp[0][0] + sp[1][0]) + (sp[0][2] + sp[1][2]);
        const float s1 = (sp[0][1] + sp[1][1]) + (sp[0][3] + sp[1][3]);
        const int pp = 8 * warp + 2 * tig;
        *reinterpret_cast<float2 *>(ss + gid * L::SS + pp) =
            make_float2(pp < cnt ? s0 : -INFINITY, pp + 1 < cnt ? s1 : -INFINITY);
      }
    }
    att_sync();
    // online softmax update: warp g owns head g; its weights go to the P fragments as bf16
    // pairs (rounded part in rows g, rest in rows g + 8)
    if (warp < G) {
      const int g = warp;
      const float a0 = ss[g * L::SS + lane], a1 = ss[g * L::SS + lane + 32];
      float mx = fmaxf(a0, a1);
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, off));
      const float m_old = s_m[g];
      const float m_new = fmaxf(m_old, mx);
      const float e0 = exp2f(a0 - m_new), e1 = exp2f(a1 - m_new);
      float sum = e0 + e1;
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, off);
      // position pp of the sub-tile: step pp / 16, lane 4 g + ((pp & 7) >> 1), register a0 / a1
      // (columns 2 tig, 2 tig + 1) or a2 / a3 (pp & 8), half pp & 1
      auto put = [&](int pp, float e) {
        uint16_t *f = reinterpret_cast<uint16_t *>(pf + (pp >> 4) * 32 + 4 * g + ((pp & 7) >> 1));
        const uint16_t hi = f32_to_bf16_rne(e);
        const int reg = (pp & 8) ? 2 : 0;
        f[2 * reg + (pp & 1)] = hi;
        f[2 * (reg + 1) + (pp & 1)] = f32_to_bf16_rne(e - bf16_to_f32(hi));
      };
      put(lane, e0);
      put(lane + 32, e1);
      if (lane == 0) {
        const float alpha = exp2f(m_old - m_new);
        s_alpha[g] = alpha;
        s_l[g] = s_l[g] * alpha + sum;
        s_m[g] = m_new;
      }
    }
    att_sync();
    // acc = acc * alpha + P V over the sub-tile: P fragments from shared memory, V fragments by
    // transposing loads (ldmatrix .trans: 8 x 8 blocks of positions x dimensions)
    {
      const float al = hrow ? s_alpha[gid] : 0.f;
#pragma unroll
      for (int nt = 0; nt < NT; ++nt)
#pragma unroll
        for (int i = 0; i < 4; ++i) acc[nt][i] *= al;
      float pv[NT][2][4] = {};
      const int mi = lane >> 3;  // the 8 x 8 block whose row this lane addresses
      const uint8_t *vrow = vb + (8 * (mi & 1) + (lane & 7)) * L::VROW + 2 * (n_base + 8 * (mi >> 1));
#pragma unroll
      for (int s16 = 0; s16 < ATT_SUB / 16; ++s16) {
        const uint4 f = pf[s16 * 32 + lane];
        if constexpr (NT == 2) {
          uint32_t v0, v1, v2, v3;
          ldsm_x4_trans(v0, v1, v2, v3, vrow + 16 * s16 * L::VROW);
          mma_bf16_full(pv[0][s16 & 1], f, v0, v1);
          mma_bf16_full(pv[1][s16 & 1], f, v2, v3);
        } else {
          uint32_t v0, v1;
          ldsm_x2_trans(v0, v1, vrow + 16 * s16 * L::VROW);
          mma_bf16_full(pv[0][s16 & 1], f, v0, v1);
        }
      }
#pragma unroll
      for (int nt = 0; nt < NT; ++nt)
#pragma unroll
        for (int i = 0; i < 4; ++i) acc[nt][i] += pv[nt][0][i] + pv[nt][1][i];
    }
    att_sync();
  }
  stamp(TR_W_FIRST);

  // this CTA's partial state into its own shared memory (the K buffers): sums [G][HD], and the
  // (m, l) of each head, read by the cluster after the barrier
  float *part = reinterpret_cast<float *>(sk);
  if (hrow) {
#pragma unroll
    for (int nt = 0; nt < NT; ++nt)
      *reinterpret_cast<float2 *>(part + gid * HD + n_base + 8 * nt + 2 * tig) =
          make_float2(acc[nt][0] + acc[nt][2], acc[nt][1] + acc[nt][3]);
  }
  cluster_sync_all();
  stamp(TR_W_LAST);

  // merge: CTA r takes chunks [r nch / C, (r + 1) nch / C) of the pair's G x HD outputs
  const int nch = G * HD / XCHUNK;
  const int c0 = static_cast<int>((long long)r * nch / C), c1 = static_cast<int>((long long)(r + 1) * nch / C);
  if (valid) {
    // every CTA's (m, l) per head, then each head's weights 2^(m_q - M) / L in CTA order
    if (tid < C * G) {
      const int q = tid / G, g = tid % G;
      s_w[q][g] = ld_cluster_f32(map_to_rank(smem_addr(s_m + g), q));
      s_lw[q][g] = ld_cluster_f32(map_to_rank(smem_addr(s_l + g), q));
    }
    __syncthreads();
    if (tid < G) {
      const int g = tid;
      float M = -INFINITY;
      for (int q = 0; q < C; ++q) M = fmaxf(M, s_w[q][g]);
      float Ls = 0.f;
      for (int q = 0; q < C; ++q) Ls += s_lw[q][g] * exp2f(s_w[q][g] - M);
      const float inv = 1.0f / Ls;
      for (int q = 0; q < C; ++q) s_w[q][g] = exp2f(s_w[q][g] - M) * inv;
    }
    __syncthreads();
  }
  {
    // lane groups of 8 take one chunk each (4 elements per lane): warp w chunks c0 + 4w .. + 3
    const int jj = c0 + warp * 4 + (lane >> 3);
    const bool mine = jj < c1;
    const int jc = mine ? jj : c0;
    const int g = jc / (HD / XCHUNK), d0 = (jc % (HD / XCHUNK)) * XCHUNK + 4 * (lane & 7);
    float4 O = make_float4(0.f, 0.f, 0.f, 0.f);
    if (valid && mine) {
      // the CTAs' sums are loaded four at a time before any is used, so that the distributed
      // shared memory round trips overlap; then added in CTA order
      const uint32_t src = smem_addr(part + g * HD + d0);
      for (int q0 = 0; q0 < C; q0 += 4) {
        float4 v[4];
#pragma unroll
        for (int j = 0; j < 4; ++j) v[j] = q0 + j < C ? ld_cluster_f4(map_to_rank(src, q0 + j)) : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          if (q0 + j < C) {
            const float w = s_w[q0 + j][g];
            O.x = fmaf(w, v[j].x, O.x);
            O.y = fmaf(w, v[j].y, O.y);
            O.z = fmaf(w, v[j].z, O.z);
            O.w = fmaf(w, v[j].w, O.w);
          }
        }
      }
    }
    float *o = p.o + (size_t)b * p.ldo + (size_t)kvh * G * HD;
    if (mine) *reinterpret_cast<float4 *>(o + g * HD + d0) = O;
    if (p.o16.base && (warp * 4 < c1 - c0))  // the whole warp calls it; `mine` selects the lanes that store
      act16_put_quad(p.o16, b, ((kvh * G + g) * HD + d0) / XCHUNK, O, lane, mine);
  }
  // no CTA leaves while another may still read its shared memory
  cluster_sync_all();
  stamp(TR_CONS_DONE);
}

cudaError_t prepare_attention_cluster() {
  cudaError_t e;
  if ((e = cudaFuncSetAttribute(attn_cluster_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                AttnLayout<128, 2>::BYTES)) != cudaSuccess)
    return e;
  if ((e = cudaFuncSetAttribute(attn_cluster_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                AttnLayout<64, 2>::BYTES)) != cudaSuccess)
    return e;
  if ((e = cudaFuncSetAttribute(attn_cluster_kernel<128>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1)) !=
      cudaSuccess)
    return e;
  return cudaFuncSetAttribute(attn_cluster_kernel<64>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
}

// The largest cluster size up to `want` (a power of two) that the device schedules for this
// kernel, or 0 if none.
int attention_cluster_size(int head_dim, int want) {
  for (int c = want; c >= 2; c >>= 1) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(c);
    cfg.blockDim = dim3(ATT_THREADS);
    cfg.dynamicSmemBytes = head_dim == 128 ? AttnLayout<128, 2>::BYTES : AttnLayout<64, 2>::BYTES;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = c;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int n = 0;
    const cudaError_t e = head_dim == 128 ? cudaOccupancyMaxActiveClusters(&n, attn_cluster_kernel<128>, &cfg)
                                          : cudaOccupancyMaxActiveClusters(&n, attn_cluster_kernel<64>, &cfg);
    if (e != cudaSuccess) {
      cudaGetLastError();
      continue;
    }
    if (n >= 1) return c;
  }
  return 0;
}

template <int HD>
static cudaError_t launch_cluster_hd(const AttnParams &p, cudaStream_t s, bool pdl) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(p.batch * p.n_kv_heads * p.cluster);
  cfg.blockDim = dim3(ATT_THREADS);
  cfg.dynamicSmemBytes = AttnLayout<HD, 2>::BYTES;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  int na = 0;
  attr[na].id = cudaLaunchAttributeClusterDimension;
  attr[na].val.clusterDim.x = p.cluster;
  attr[na].val.clusterDim.y = 1;
  attr[na].val.clusterDim.z = 1;
  ++na;
  if (pdl) {
    attr[na].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[na].val.programmaticStreamSerializationAllowed = 1;
    ++na;
  }
  cfg.attrs = attr;
  cfg.numAttrs = na;
  return cudaLaunchKernelEx(&cfg, attn_cluster_kernel<HD>, p);
}

cudaError_t launch_attention_cluster(const AttnParams &p, int head_dim, cudaStream_t s, bool pdl) {
  if (p.n_heads % p.n_kv_heads != 0 || p.n_heads / p.n_kv_heads > ATT_MAXG || p.cluster < 1 ||
      p.cluster > MAX_CLUSTER_ATT)
    return cudaErrorInvalidValue;
  if (head_dim == 128) return launch_cluster_hd<128>(p, s, pdl);
  if (head_dim == 64) return launch_cluster_hd<64>(p, s, pdl);
  return cudaErrorInvalidValue;
}

}  // namespace kfl
