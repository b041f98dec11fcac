// Grouped-query decode attention over one chunk of cached positions (flash-decoding unit),
// shared by the standalone attention kernel (attention.cu) and the persistent stage kernel.
//
// User b's token at position P_b attends to its cached slots [0, P_b] (its own K/V were
// appended by the QKV epilogue), query head h reading KV head h / G.  A unit is one (user, KV
// head, chunk of positions): the chunk's K and V rows are loaded once (cp.async, 64-position
// sub-tiles, double buffered) for all G query heads that share the KV head; an online-softmax
// state (running max m, running sum l, weighted sum of V) is kept per head.  A single-chunk
// unit writes its output directly; otherwise each unit writes (m, l, acc) and the last unit of
// its (user, KV head) to finish (atomic ticket, no spin) merges the chunks in chunk order.
// Scores are in the log2 domain (q pre-scaled by log2(e)/sqrt(hd)).
//
// 256 threads.  Scores S = q K^T and the weighted sum P V are small dense products (at most 8
// heads x 64 positions x hd): both run on the tensor cores as warp-level bf16 m16n8k16 MMAs with
// fp32 accumulation.  q and P enter as bf16 pairs (rounded value and the bf16 rounding of the
// rest: about 2^-17 relative), the rounded parts in the A operand's rows 0..7 (the heads) and the
// rests in rows 8..15, so one MMA gives both products; K and V are the cache's bf16 values,
// exact.  Scores: warp w takes positions
// 8w..8w+7; P V: warp w takes head dimensions hd/8 * w onwards.
#pragma once

#include <math.h>

#include "common.cuh"

namespace kfl {

constexpr int ATT_THREADS = 256;
constexpr int ATT_SUB = 64;          // positions per shared-memory sub-tile
constexpr int ATT_MAXG = 8;          // query heads per KV head
constexpr int ATT_MERGE_MAX = 1024;  // chunks x heads merged in shared memory (fits the K buffers)
constexpr int ATT_BAR = 2;           // named barrier of the attention threads

__device__ __forceinline__ void att_sync() { named_bar_sync(ATT_BAR, ATT_THREADS); }

__device__ __forceinline__ void cp_async16(void *dst, const void *src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_addr(dst)), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

template <int HD, int NBUF>
struct AttnLayout {
  // K and V rows padded by 16 bytes (4 banks) so that the MMA fragments (and the transposing
  // loads) of 8 consecutive rows fall in distinct banks; score rows padded by 4 floats
  static constexpr int KROW = HD * 2 + 16;
  static constexpr int VROW = HD * 2 + 16;
  static constexpr int SS = ATT_SUB + 4;
  static constexpr int K_OFF = 0;
  static constexpr int V_OFF = K_OFF + NBUF * ATT_SUB * KROW;
  static constexpr int S_OFF = V_OFF + NBUF * ATT_SUB * VROW;
  static constexpr int M_OFF = S_OFF + ATT_MAXG * SS * 4;
  // q and P as MMA A fragments: [K step][lane] x (rounded a0, a2, rest a0, a2)
  static constexpr int QF_OFF = M_OFF + 4 * ATT_MAXG * 4;
  static constexpr int PF_OFF = QF_OFF + (HD / 16) * 32 * 16;
  static constexpr int BYTES = PF_OFF + (ATT_SUB / 16) * 32 * 16;
  static constexpr int MERGE_MAX = (NBUF * ATT_SUB * KROW) / 8;  // chunks x heads in the K buffers
  static_assert(MERGE_MAX >= 1024, "merge scratch too small");
};

__host__ __device__ constexpr int attn_pstride(int hd) { return hd + 4; }

// Number of chunks of user b (1 for an invalid position: that unit writes zeros).  The
// positions are never written while a step runs, so they need no L2-coherent load.
__device__ __forceinline__ int attn_chunks(const AttnParams &p, int b) {
  const int P = p.positions[b];
  if (P < 0 || P >= p.max_ctx) return 1;
  return (P + 1 + p.chunk - 1) / p.chunk;
}

// (user, KV head, chunk) of attention unit u: users in order, n_kv_heads * nc_b units each.
__device__ __forceinline__ void attn_unit_coords(int u, int hk, int nc0, int nc1, int nc2, int nc3, int &b, int &kvh,
                                                 int &ch, int &ncb) {
  int rem = u;
  b = 0;
  ncb = nc0;
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
  kvh = rem / ncb;
  ch = rem % ncb;
}

// Positions per unit for this step: about target_units units over the users' actual contexts
// (a multiple of 64, at least 64), and few enough chunks per (user, KV head) for the merge to
// take (chunks x heads <= ATT_MERGE_MAX).  Every CTA of a launch computes the same value.
__device__ __forceinline__ int attn_chunk_size(const AttnParams &p) {
  long long total = 0;
  int maxp1 = 1;
  for (int b = 0; b < p.batch; ++b) {
    const int P = p.positions[b];
    const int n = (P < 0 || P >= p.max_ctx) ? 1 : P + 1;
    total += n;
    maxp1 = max(maxp1, n);
  }
  const long long work = total * p.n_kv_heads;
  const long long want = (work + p.target_units - 1) / max(1, p.target_units);
  int chunk = static_cast<int>(max((long long)p.chunk, (want + 63) / 64 * 64));  // p.chunk: the smallest
  const int G = p.n_heads / p.n_kv_heads;
  const int need = (maxp1 * G + ATT_MERGE_MAX - 1) / ATT_MERGE_MAX;
  return max(chunk, (need + 63) / 64 * 64);
}

// Rows [p0, p0 + cnt) of user b / KV head kvh into K/V buffer `buf`: mode 0 all of them, mode 1
// those outside [new_lo, new_hi] (the rows this step writes), mode 2 those inside; one cp.async
// group.
template <int HD, int NBUF>
__device__ __forceinline__ void attn_load_rows(const AttnParams &p, int b, int kvh, int p0, int cnt, int buf,
                                               int mode, int new_lo, int new_hi, uint8_t *sm, int tid) {
  using L = AttnLayout<HD, NBUF>;
  const size_t head_base = ((size_t)p.slots[b] * p.n_kv_heads + kvh) * p.max_ctx;
  const uint16_t *kg = p.kcache + head_base * HD;
  const uint16_t *vg = p.vcache + head_base * HD;
  uint8_t *sk = sm + L::K_OFF + buf * ATT_SUB * L::KROW;
  uint8_t *sv = sm + L::V_OFF + buf * ATT_SUB * L::VROW;
  constexpr int CH = HD / 8;   // 16-byte chunks per row
  for (int e = tid; e < cnt * CH; e += ATT_THREADS) {
    const int r = e / CH, ch = e % CH;
    const int row = p0 + r;
    const bool fresh = row >= new_lo && row <= new_hi;
    if ((mode == 1 && fresh) || (mode == 2 && !fresh)) continue;
    cp_async16(sk + r * L::KROW + ch * 16, kg + (size_t)row * HD + ch * 8);
    cp_async16(sv + r * L::VROW + ch * 16, vg + (size_t)row * HD + ch * 8);
  }
  cp_async_commit();
}

// The lowest position of user b's KV slot that this step writes: its own position, or an
// earlier one of another batch row on the same slot (several of a user's tokens in one step, as
// in a prefill).  Rows from there to its own position are written by this step's Q/K/V phase.
__device__ __forceinline__ int attn_step_lo(const AttnParams &p, int b) {
  const int P = p.positions[b], sl = p.slots[b];
  int lo = P;
  for (int j = 0; j < p.batch; ++j) {
    const int q = p.positions[j];
    if (p.slots[j] == sl && q >= 0 && q < lo) lo = q;
  }
  return lo;
}

// Issue the loads of a unit's first sub-tile that do not depend on the current step: every row
// before the step's first new one (attn_step_lo).  The unit then runs with prefetched = 1.
// Positions and slots are final before the step's kernels start.
template <int HD, int NBUF>
__device__ __forceinline__ void attn_prefetch(const AttnParams &p, int b, int kvh, int c, uint8_t *sm, int tid) {
  const int P = p.positions[b];
  if (P < 0 || P >= p.max_ctx) return;
  const int start = c * p.chunk;
  const int end = min(P + 1, start + p.chunk);
  attn_load_rows<HD, NBUF>(p, b, kvh, start, min(ATT_SUB, end - start), 0, 1, attn_step_lo(p, b), P, sm, tid);
}

// The (user, KV head) output is written: publish it (persistent kernel; the bar.sync orders every
// thread's stores before the release).
__device__ __forceinline__ void attn_publish(const AttnParams &p, int kvh, int tid) {
  if (!p.out_ready) return;
  att_sync();
  if (tid == 0) red_add_release(p.out_ready + kvh, 1u);
}

// d += a b for one m16n8k16 bf16 tile (a: 16x16 row-major, b: 16x8 column-major, fp32
// accumulate).  Rows 0..7 of a hold the heads' rounded parts and rows 8..15 their rests (bf16
// pairs of q or P), so accumulator rows g and g + 8, which one lane holds, add up to head g's.
__device__ __forceinline__ void mma_bf16_full(float (&d)[4], const uint4 &a, uint32_t b0, uint32_t b1) {
  asm("mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a.x), "r"(a.y), "r"(a.z), "r"(a.w), "r"(b0), "r"(b1));
}

// Four (two) 8 x 8 blocks of 16-bit values, transposed: lanes 8 i .. 8 i + 7 address the rows of
// block i (16-byte aligned); a lane receives elements (2 (lane % 4), lane / 4) and
// (2 (lane % 4) + 1, lane / 4) of each block, the B fragment layout of the MMA.
__device__ __forceinline__ void ldsm_x4_trans(uint32_t &r0, uint32_t &r1, uint32_t &r2, uint32_t &r3, const void *p) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(smem_addr(p))
               : "memory");
}
__device__ __forceinline__ void ldsm_x2_trans(uint32_t &r0, uint32_t &r1, const void *p) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x2.trans.shared.b16 {%0,%1}, [%2];"
               : "=r"(r0), "=r"(r1)
               : "r"(smem_addr(p))
               : "memory");
}

// int4 stages: the output of heads (kvh, og), dimensions od .. od + 3, also in the O
// projection's input form (8 lanes hold a 32-dimension chunk); every thread of the unit calls it.
template <int HD>
__device__ __forceinline__ void attn_out16(const AttnParams &p, int b, int kvh, int G, int og, int od, float4 v,
                                           bool owns, int lane) {
  if (!p.o16.base) return;
  act16_put_quad(p.o16, b, ((kvh * G + og) * HD + od) / XCHUNK, v, lane, owns);
}

template <int HD, int NBUF>
__device__ void attn_unit(const AttnParams &p, int b, int kvh, int c, int nc, uint8_t *sm, int *s_last, int tid,
                          int prefetched, unsigned long long *tr = nullptr) {
  // tr: this CTA's trace slots (tuning aid): 4 K/V in shared memory, 5 output or partial
  // computed, 6 the merge starts (the last unit of its user and KV head)
  auto stamp = [&](int slot) {
    if (tr && tid == 0) tr[slot] = global_ns();
  };
  using L = AttnLayout<HD, NBUF>;
  uint8_t *sk = sm + L::K_OFF;
  uint8_t *sv = sm + L::V_OFF;
  float *ss = reinterpret_cast<float *>(sm + L::S_OFF);
  float *s_m = reinterpret_cast<float *>(sm + L::M_OFF);
  float *s_l = s_m + ATT_MAXG;
  float *s_alpha = s_l + ATT_MAXG;
  const int warp = tid >> 5, lane = tid & 31;
  const int G = p.n_heads / p.n_kv_heads;
  // P.V / output mapping: head og, dimensions od .. od + 3
  const int og = (HD == 128) ? warp : 2 * warp + (lane >> 4);
  const int od = 4 * ((HD == 128) ? lane : (lane & 15));
  const bool owns = og < G;
  float *o = p.o + (size_t)b * p.ldo + (size_t)kvh * G * HD;

  const int P = p.positions[b];
  if (P < 0 || P >= p.max_ctx) {
    // the stage input flagged the position; leave a defined (zero) output
    if (owns) *reinterpret_cast<float4 *>(o + og * HD + od) = make_float4(0.f, 0.f, 0.f, 0.f);
    attn_out16<HD>(p, b, kvh, G, og, od, make_float4(0.f, 0.f, 0.f, 0.f), owns, lane);
    attn_publish(p, kvh, tid);
    return;
  }
  const int ntok = P + 1;
  const int start = c * p.chunk;
  const int end = min(ntok, start + p.chunk);

  auto load_sub = [&](int sub, int buf) {
    const int p0 = start + sub * ATT_SUB;
    attn_load_rows<HD, NBUF>(p, b, kvh, p0, min(ATT_SUB, end - p0), buf, 0, 0, -1, sm, tid);
  };
  // the first sub-tile's copies go out first, so that their latency overlaps the q loads
  if (prefetched)  // only the rows this step wrote (attn_step_lo .. P) are still to load
    attn_load_rows<HD, NBUF>(p, b, kvh, start, min(ATT_SUB, end - start), 0, 2, attn_step_lo(p, b), P, sm, tid);
  else
    load_sub(0, 0);

  // MMA fragment coordinates: lane = 4 * gid + tig; accumulator rows gid are heads (gid < G)
  const int gid = lane >> 2, tig = lane & 3;
  const bool hrow = gid < G;
  constexpr int KS = HD / 16;   // K steps of the scores
  constexpr int NT = HD / 64;   // P V n-tiles (8 dimensions) per warp: warp w owns dims NT*8*w ...
  const int n_base = warp * NT * 8;
  uint4 *qf = reinterpret_cast<uint4 *>(sm + L::QF_OFF);
  uint4 *pf = reinterpret_cast<uint4 *>(sm + L::PF_OFF);
  {
    // q (scaled to log2 units) as the scores' A fragments, a bf16 pair each (rounded, rest:
    // about 2^-17 relative, for the softmax turns a relative error e of a score s into an error
    // of about |s| e of its weight): entry (step s, lane) = registers a0..a3, rows gid the
    // heads' rounded parts and rows gid + 8 their rests; rows of heads >= G are zero
    if (tid < KS * 32) {
      const int st = tid >> 5, l = tid & 31, g = l >> 2, t = l & 3;
      uint4 f = make_uint4(0u, 0u, 0u, 0u);
      if (g < G) {
        const float *qg = p.q + (size_t)b * p.n_heads * HD + (size_t)(kvh * G + g) * HD + 16 * st + 2 * t;
        const float2 x0 = __ldcg(reinterpret_cast<const float2 *>(qg));
        const float2 x1 = __ldcg(reinterpret_cast<const float2 *>(qg + 8));
        const float v[4] = {x0.x * p.scale_log2, x0.y * p.scale_log2, x1.x * p.scale_log2, x1.y * p.scale_log2};
        uint16_t hi[4], lo[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          hi[i] = f32_to_bf16_rne(v[i]);
          lo[i] = f32_to_bf16_rne(v[i] - bf16_to_f32(hi[i]));
        }
        f = make_uint4(hi[0] | ((uint32_t)hi[1] << 16), lo[0] | ((uint32_t)lo[1] << 16),
                       hi[2] | ((uint32_t)hi[3] << 16), lo[2] | ((uint32_t)lo[3] << 16));
      }
      qf[tid] = f;
    }
    // P fragments of rows gid >= G stay zero for the whole unit
    if (tid < (ATT_SUB / 16) * 32 && ((tid & 31) >> 2) >= G) pf[tid] = make_uint4(0u, 0u, 0u, 0u);
  }
  if (tid < ATT_MAXG) {
    s_m[tid] = -INFINITY;
    s_l[tid] = 0.f;
  }
  float acc[NT][4];
#pragma unroll
  for (int nt = 0; nt < NT; ++nt) acc[nt][0] = acc[nt][1] = acc[nt][2] = acc[nt][3] = 0.f;

  const int nsub = (end - start + ATT_SUB - 1) / ATT_SUB;
  for (int it = 0; it < nsub; ++it) {
    const int buf = NBUF == 2 ? (it & 1) : 0;
    if (NBUF == 2 && it + 1 < nsub) {
      load_sub(it + 1, buf ^ 1);
      cp_async_wait<1>();
    } else {
      if (NBUF == 1 && it > 0) load_sub(it, 0);
      cp_async_wait<0>();
    }
    att_sync();
    if (it == 0) stamp(TR_X_LAST);
    const int p0 = start + it * ATT_SUB;
    const int cnt = min(ATT_SUB, end - p0);
    const uint8_t *kb = sk + buf * ATT_SUB * L::KROW;
    uint8_t *vb = sv + buf * ATT_SUB * L::VROW;
    // rows past the sub-tile's positions take part in P V with weight 0: make them finite
    if (cnt < ATT_SUB)
      for (int e = tid; e < (ATT_SUB - cnt) * (HD / 8); e += ATT_THREADS)
        *reinterpret_cast<uint4 *>(vb + (cnt + e / (HD / 8)) * L::VROW + (e % (HD / 8)) * 16) = make_uint4(0u, 0u, 0u, 0u);

    // scores of positions 8w .. 8w + 7 (MMA columns) for every head (rows gid, rests gid + 8):
    // bf16 m16n8k16 MMAs, K rows as the B fragments (two 32-bit loads per step); two
    // independent accumulator chains (K steps modulo 2) so that the MMAs overlap
    {
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
    // online softmax update: warp g owns head g; its weights go to the P fragments as bf16 pairs
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
      // position pp of the sub-tile: step pp / 16, lane 4 g + ((pp & 7) >> 1), registers a0
      // (rounded part) and a1 (rest) or, for pp & 8, a2 and a3; half pp & 1
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
      // rows gid (P's rounded parts) and gid + 8 (rests) are both head gid's
      const float al = hrow ? s_alpha[gid] : 0.f;
#pragma unroll
      for (int nt = 0; nt < NT; ++nt)
#pragma unroll
        for (int i = 0; i < 4; ++i) acc[nt][i] *= al;
      // this sub-tile's P V in two chains per n-tile (K steps modulo 2), then into acc
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
  if (nc == 1) {
    if (!p.o16.base) {
      if (hrow) {
        const float il = 1.0f / s_l[gid];
#pragma unroll
        for (int nt = 0; nt < NT; ++nt)
          *reinterpret_cast<float2 *>(o + gid * HD + n_base + 8 * nt + 2 * tig) =
              make_float2((acc[nt][0] + acc[nt][2]) * il, (acc[nt][1] + acc[nt][3]) * il);
      }
    } else {
      // through shared memory (the K buffers) into the output mapping of the merge
      float *so = reinterpret_cast<float *>(sk);
      if (hrow) {
        const float il = 1.0f / s_l[gid];
#pragma unroll
        for (int nt = 0; nt < NT; ++nt)
          *reinterpret_cast<float2 *>(so + gid * HD + n_base + 8 * nt + 2 * tig) =
              make_float2((acc[nt][0] + acc[nt][2]) * il, (acc[nt][1] + acc[nt][3]) * il);
      }
      att_sync();
      const float4 v = owns ? *reinterpret_cast<const float4 *>(so + og * HD + od) : make_float4(0.f, 0.f, 0.f, 0.f);
      if (owns) *reinterpret_cast<float4 *>(o + og * HD + od) = v;
      attn_out16<HD>(p, b, kvh, G, og, od, v, owns, lane);
    }
    attn_publish(p, kvh, tid);
    return;
  }
  constexpr int PS = attn_pstride(HD);
  const size_t unit_base = ((size_t)b * p.n_kv_heads + kvh) * p.n_chunks;
  float *part = p.partial + (unit_base + c) * (ATT_MAXG * PS);
  if (hrow) {
#pragma unroll
    for (int nt = 0; nt < NT; ++nt)
      *reinterpret_cast<float2 *>(part + gid * PS + n_base + 8 * nt + 2 * tig) =
          make_float2(acc[nt][0] + acc[nt][2], acc[nt][1] + acc[nt][3]);
  }
  if (tid < G) {
    part[tid * PS + HD] = s_m[tid];
    part[tid * PS + HD + 1] = s_l[tid];
  }
  att_sync();
  if (tid == 0) {
    int *tk = p.tickets + b * p.n_kv_heads + kvh;
    const unsigned prev = atom_add_acq_rel(reinterpret_cast<unsigned *>(tk), 1u);
    *s_last = (prev == (unsigned)(nc - 1));
    if (*s_last) atomicExch(tk, 0);
  }
  att_sync();
  if (!*s_last) return;
  stamp(TR_W_LAST);
  // merge: per-chunk weights 2^(m_c - M) / L staged in shared memory (the K buffers), then each
  // thread sums its 4 outputs over the chunks.  The chunk outputs are loaded MB at a time, the
  // first MB before the weights are computed, so that few L2 round trips are in series (MB 8
  // inside the persistent stage kernel, whose register budget is shared with its other roles).
  constexpr int MB = NBUF == 2 ? 16 : 8;
  const float *base = p.partial + unit_base * (ATT_MAXG * PS);
  const float *pg = base + og * PS + od;
  float4 a[MB];
  auto load_batch = [&](int c0) {
#pragma unroll
    for (int j = 0; j < MB; ++j)
      a[j] = owns && c0 + j < nc ? __ldcg(reinterpret_cast<const float4 *>(pg + (size_t)(c0 + j) * ATT_MAXG * PS))
                                 : make_float4(0.f, 0.f, 0.f, 0.f);
  };
  load_batch(0);
  float *wm = reinterpret_cast<float *>(sk);
  float *wl = wm + L::MERGE_MAX;
  for (int e = tid; e < nc * G; e += ATT_THREADS) {
    const int cc = e / G, g = e % G;
    const float *pc = base + (size_t)cc * ATT_MAXG * PS + g * PS;
    wm[e] = __ldcg(pc + HD);
    wl[e] = __ldcg(pc + HD + 1);
  }
  att_sync();
  if (warp < G) {
    const int g = warp;
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
  att_sync();
  float4 O = make_float4(0.f, 0.f, 0.f, 0.f);
  if (owns) {
    for (int c0 = 0; c0 < nc; c0 += MB) {
      if (c0 > 0) load_batch(c0);
#pragma unroll
      for (int j = 0; j < MB; ++j) {
        if (c0 + j < nc) {
          const float w = wm[(c0 + j) * G + og];
          O.x = fmaf(w, a[j].x, O.x);
          O.y = fmaf(w, a[j].y, O.y);
          O.z = fmaf(w, a[j].z, O.z);
          O.w = fmaf(w, a[j].w, O.w);
        }
      }
    }
    *reinterpret_cast<float4 *>(o + og * HD + od) = O;
  }
  attn_out16<HD>(p, b, kvh, G, og, od, O, owns, lane);
  attn_publish(p, kvh, tid);
}

}  // namespace kfl
