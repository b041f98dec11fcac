// Decode attention, one thread-block cluster per (user, KV head), for the one-kernel-per-phase
// mode (the persistent stage kernel runs attn_unit of attn_core.cuh instead).
//
// User b's token at position P_b attends to its cached slots [0, P_b] (its own K/V were appended
// before this kernel), query head h reading KV head h / G.  The cluster's C CTAs split the
// positions in whole 64-position sub-tiles: CTA r takes sub-tiles [ceil(r n / C), ceil((r + 1) n / C))
// of the n = ceil((P_b + 1) / 64).
//
// Inside a CTA one producer warp streams the sub-tiles' K and V rows into a ring of shared-memory
// stages with 2-D TMA copies (boxes of 64 positions x 64 dimensions, 128-byte swizzle: the
// fragment loads of 8 consecutive rows fall in distinct banks without padding), and four consumer
// warps each take 16 positions of every stage.  A consumer warp keeps its own online-softmax state
// (running max m, running sum l, unnormalised weighted sum of V) per head and needs no block
// barrier in its loop: the scores of its 16 positions (two m16n8k16 accumulator tiles) are, after
// the softmax, exactly the A fragments of its P V product, so P never leaves the registers.
// After the loop the four warp states merge into the CTA's (in shared memory), and the C CTA
// states meet in distributed shared memory: every CTA sends its (m, l) per head to all CTAs of
// the cluster and its sums of each 32-element output chunk to the CTA that merges that chunk, with
// asynchronous stores whose bytes complete on the receiver's mbarrier (no round trip, no cluster
// barrier between sending and merging); CTA r then adds its chunks' sums in CTA order
// (deterministic) and writes them (int4 stages: also in the O projection's input form).
//
// Scores S = q K^T and P V run as bf16 m16n8k16 MMAs with fp32 accumulation.  q and P enter as
// bf16 pairs (rounded value, bf16 of the rest: about 2^-17 relative): rows 0..7 of the MMA's A
// operand hold the heads' rounded parts and rows 8..15 their rests, so one MMA yields both
// products and the head's value is the sum of accumulator rows g and g + 8, which the same lane
// holds.  K and V are the cache's bf16 values, exact.  Scores are in the log2 domain (q
// pre-scaled by log2(e)/sqrt(hd)).
#include <cuda.h>  // CUtensorMap
#include <cudaTypedefs.h>  // the type of cuTensorMapEncodeTiled

#include "attn_core.cuh"

namespace kfl {

constexpr int ATC_WARPS = 4;                       // consumer warps, 16 positions of a stage each
constexpr int ATC_THREADS = (ATC_WARPS + 1) * 32;  // + the producer warp

// Shared memory of a CTA with a ring of S stages: the stages, q's A fragments, the barriers.
template <int HD>
struct AtcLayout {
  static constexpr int BOXES = HD / 64;                  // 64-dimension boxes of a row
  static constexpr int BOX_BYTES = ATT_SUB * 128;        // 64 positions x 64 bf16, swizzled
  static constexpr int KV_BYTES = BOXES * BOX_BYTES;     // the K (or V) rows of one stage
  static constexpr int STAGE_BYTES = 2 * KV_BYTES;
  static constexpr int QF_BYTES = (HD / 16) * 32 * 16;   // q as A fragments [HD / 16][32] uint4
  __host__ __device__ static constexpr int qf_off(int S) { return S * STAGE_BYTES; }
  __host__ __device__ static constexpr int bar_off(int S) { return qf_off(S) + QF_BYTES; }
  // + 1024: the alignment of the swizzled boxes
  __host__ __device__ static constexpr int smem(int S) { return bar_off(S) + 2 * S * 8 + 1024; }
  // after the loop, in the stage buffers: the warps' sums [ATC_WARPS][ATT_MAXG][HD]
  static_assert(ATC_WARPS * ATT_MAXG * HD * 4 <= STAGE_BYTES, "merge scratch");
};

// Byte offset of 16-byte chunk c of row r in a box of 128-byte rows written with the 128-byte
// swizzle (the chunk index is XORed with the row's index modulo 8).
__device__ __forceinline__ uint32_t swz128(int r, int c) { return static_cast<uint32_t>(r * 128 + ((c ^ (r & 7)) << 4)); }

__device__ __forceinline__ void atc_tma_load(uint32_t dst, const CUtensorMap *map, int c0, int c1, uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::"r"(
          dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(bar)
      : "memory");
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

__device__ __forceinline__ void mma_bf16(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                         uint32_t b0, uint32_t b1) {
  asm("mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// Asynchronous stores into another CTA of the cluster that count their bytes on that CTA's
// mbarrier (complete_tx): the receiver learns that every store has landed from the barrier alone.
__device__ __forceinline__ void st_async_f4(uint32_t addr, float4 v, uint32_t bar) {
  asm volatile("st.async.shared::cluster.mbarrier::complete_tx::bytes.v4.f32 [%0], {%1, %2, %3, %4}, [%5];" ::"r"(addr),
               "f"(v.x), "f"(v.y), "f"(v.z), "f"(v.w), "r"(bar)
               : "memory");
}
__device__ __forceinline__ void st_async_f2(uint32_t addr, float a, float b, uint32_t bar) {
  asm volatile("st.async.shared::cluster.mbarrier::complete_tx::bytes.v2.f32 [%0], {%1, %2}, [%3];" ::"r"(addr),
               "f"(a), "f"(b), "r"(bar)
               : "memory");
}
// The cluster barrier in two halves, so that a CTA does other work between its arrival and its wait.
__device__ __forceinline__ void cluster_arrive_release() {
  asm volatile("barrier.cluster.arrive.release.aligned;" ::: "memory");
}
__device__ __forceinline__ void cluster_arrive_relaxed() {
  asm volatile("barrier.cluster.arrive.relaxed.aligned;" ::: "memory");
}
__device__ __forceinline__ void cluster_wait_acquire() {
  asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory");
}

// (rounded, rest) bf16 pairs of two weights as the packed registers of one A-fragment row pair
__device__ __forceinline__ void bf16_pair2(float x0, float x1, uint32_t &hi, uint32_t &lo) {
  const uint16_t h0 = f32_to_bf16_rne(x0), h1 = f32_to_bf16_rne(x1);
  hi = (uint32_t)h0 | ((uint32_t)h1 << 16);
  lo = (uint32_t)f32_to_bf16_rne(x0 - bf16_to_f32(h0)) | ((uint32_t)f32_to_bf16_rne(x1 - bf16_to_f32(h1)) << 16);
}

template <int HD>
__global__ void __launch_bounds__(ATC_THREADS, 2) attn_cluster_kernel(const __grid_constant__ AttnParams p,
                                                                   const __grid_constant__ CUtensorMap kmap,
                                                                   const __grid_constant__ CUtensorMap vmap) {
  using L = AtcLayout<HD>;
  extern __shared__ uint8_t sm_raw[];
  uint8_t *sm = sm_raw + ((1024u - (smem_addr(sm_raw) & 1023u)) & 1023u);
  // the cluster merge: what every CTA of the cluster sends this one (its (m, l) per head, and its
  // sums of this CTA's output chunks, [source CTA][chunk - c0][XCHUNK]), the barrier that counts
  // those bytes, and each source CTA's weight per head
  __shared__ __align__(16) float s_recv[(ATT_MAXG * 128 / XCHUNK + MAX_CLUSTER_ATT) * XCHUNK];
  __shared__ __align__(8) float2 s_rml[MAX_CLUSTER_ATT][ATT_MAXG];
  __shared__ __align__(8) uint64_t s_rbar;
  __shared__ float s_w[MAX_CLUSTER_ATT][ATT_MAXG];
  __shared__ float s_wm[ATC_WARPS][ATT_MAXG];       // each consumer warp's (m, then weight) per head
  __shared__ float s_wl[ATC_WARPS][ATT_MAXG];
  __shared__ float s_m[ATT_MAXG], s_l[ATT_MAXG];     // this CTA's state, read by the cluster
  __shared__ volatile int s_abort;
  if (p.launch_at == 0) pdl_launch_dependents();
  const int C = p.cluster;
  const int pair = blockIdx.x / C, r = blockIdx.x % C;  // r: the CTA's rank in its cluster
  const int b = pair / p.n_kv_heads, kvh = pair % p.n_kv_heads;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int G = p.n_heads / p.n_kv_heads;
  const int gid = lane >> 2, tig = lane & 3;
  // trace slots of an attention CTA: go (start), enter (consumers past the wait on Q/K/V), x_go
  // (q's fragments built), x_last (first stage landed), kind (warp 0 done with the first stage),
  // seg (warp 0 done with its stages), ticket
  // (every consumer warp done), summed (producer past its wait on Q/K/V), w_last (producer issued
  // its first sub-tile), w_first (before the cluster barrier), epi (cluster weights computed), done
  // (end)
  auto stamp_by = [&](bool who, int slot) {
    if (p.trace && (int)blockIdx.x < p.trace_grid && who) p.trace[(size_t)blockIdx.x * TRACE_SLOTS + slot] = global_ns();
  };
  auto stamp = [&](int slot) { stamp_by(tid == 0, slot); };
  stamp(TR_CONS_GO);
  const int S = p.stages;  // ring depth
  uint64_t *full = reinterpret_cast<uint64_t *>(sm + L::bar_off(S));
  uint64_t *empty = full + S;
  uint4 *qf = reinterpret_cast<uint4 *>(sm + L::qf_off(S));
  const uint32_t sm0 = smem_addr(sm);

  // the step's positions and KV slots: the producer loads every user's at once (it needs the
  // lowest row this step writes into its user's slot, attn_step_lo), the others this user's
  // position; the tensor maps' descriptors are fetched meanwhile
  int P = -1, slot = 0, lo = 0;
  if (warp == ATC_WARPS && lane == 0) {
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&kmap)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&vmap)) : "memory");
    int pj[MAXB], sj[MAXB];
#pragma unroll
    for (int j = 0; j < MAXB; ++j) {
      pj[j] = j < p.batch ? p.positions[j] : -1;
      sj[j] = j < p.batch ? p.slots[j] : -1;
    }
#pragma unroll
    for (int j = 0; j < MAXB; ++j)
      if (j == b) {
        P = pj[j];
        slot = sj[j];
      }
    lo = P;
#pragma unroll
    for (int j = 0; j < MAXB; ++j)
      if (sj[j] == slot && pj[j] >= 0 && pj[j] < lo) lo = pj[j];
  } else {
    P = p.positions[b];
  }
  const bool valid = P >= 0 && P < p.max_ctx;
  int start = 0, end = 0;
  if (valid) {
    const int nsub_all = (P + ATT_SUB) / ATT_SUB;
    // rounded up: the larger shares go to the first CTAs, so that the last one, which holds the
    // rows this step writes and loads them only after the wait on Q/K/V, has the fewest
    start = static_cast<int>(((long long)r * nsub_all + C - 1) / C) * ATT_SUB;
    end = min(P + 1, static_cast<int>(((long long)(r + 1) * nsub_all + C - 1) / C) * ATT_SUB);
  }
  const int nsub = end > start ? (end - start + ATT_SUB - 1) / ATT_SUB : 0;
  // output chunks of XCHUNK elements of the pair's G x HD: CTA r merges [c0, c1)
  const int nch = G * HD / XCHUNK;
  const int c0 = static_cast<int>((long long)r * nch / C), c1 = static_cast<int>((long long)(r + 1) * nch / C);
  const int own = (nch + C - 1) / C;  // rows of s_recv per source CTA
  const uint32_t rbar = smem_addr(&s_rbar);
  if (tid == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(smem_addr(&full[s]), 1);
      mbar_init(smem_addr(&empty[s]), ATC_WARPS * 32);
    }
    // every CTA of the cluster sends its (m, l) of the G heads and its sums of chunks [c0, c1)
    mbar_init(rbar, 1);
    mbar_arrive_expect_tx(rbar, static_cast<uint32_t>(C * (G * 8 + (c1 - c0) * XCHUNK * 4)));
    s_abort = 0;
    fence_mbar_init();
  }
  __syncthreads();
  // the other CTAs send into this one's shared memory only after its barrier is initialised: they
  // wait on the cluster barrier after the loop (this arrival makes the initialisation visible)
  cluster_arrive_release();

  constexpr int KS = HD / 16;  // K steps of the scores
  constexpr int NT = HD / 8;   // n-tiles (8 dimensions) of P V
  if (warp == ATC_WARPS) {
    // ------------------------------------------------------------------ producer
    // The cached rows [0, lo) were written by earlier steps: sub-tiles below lo go out while the
    // Q/K/V projection may still run, the rest after the wait on it.
    if (lane == 0 && nsub > 0) {
      const int row0 = (slot * p.n_kv_heads + kvh) * p.max_ctx;
      bool waited = false;
      int issued = 0;
      for (int t = 0; t < nsub; ++t) {
        const int s = t % S;
        if (t >= S && !mbar_wait(smem_addr(&empty[s]), ((t / S) - 1) & 1)) {
          s_abort = 1;
          atomicOr(p.err, ERR_TIMEOUT);
          break;
        }
        if (s_abort) break;
        const int p0 = start + t * ATT_SUB;
        if (!waited && p0 + ATT_SUB > lo) {
          pdl_wait();
          waited = true;
          stamp_by(true, TR_E_SUMMED);
        }
        const uint32_t fb = smem_addr(&full[s]);
        mbar_arrive_expect_tx(fb, L::STAGE_BYTES);
        const uint32_t kd = sm0 + s * L::STAGE_BYTES, vd = kd + L::KV_BYTES;
#pragma unroll
        for (int hb = 0; hb < L::BOXES; ++hb) {
          atc_tma_load(kd + hb * L::BOX_BYTES, &kmap, 64 * hb, row0 + p0, fb);
          atc_tma_load(vd + hb * L::BOX_BYTES, &vmap, 64 * hb, row0 + p0, fb);
        }
        ++issued;
        if (t == 0) stamp_by(true, TR_W_LAST);
      }
      if (p.launch_at == 1) pdl_launch_dependents();
      // copies still in flight land before the shared memory is reused (bounded)
      for (int t = issued > S ? issued - S : 0; t < issued; ++t) mbar_wait(smem_addr(&full[t % S]), (t / S) & 1);
    }
  } else {
    // ------------------------------------------------------------------ consumers
    pdl_wait();  // q and this step's K/V rows come from the Q/K/V projection
    stamp(TR_CONS_ENTER);
    // q (scaled to log2 units) as the scores' A fragments: entry (step, lane) = registers a0..a3:
    // rows gid (the heads' rounded parts) and gid + 8 (their rests), columns 2 tig, 2 tig + 1
    // (a0, a1) and + 8 (a2, a3); rows of heads >= G are zero
    // (every load is issued before any is used: one round trip to L2)
    constexpr int QPT = KS / ATC_WARPS;  // entries per consumer thread
    static_assert(QPT * ATC_WARPS == KS, "q fragments per thread");
    float2 xq[QPT][2];
#pragma unroll
    for (int i = 0; i < QPT; ++i) {
      const int e = tid + i * ATC_WARPS * 32;
      const int st = e >> 5, l = e & 31, g = l >> 2, t = l & 3;
      xq[i][0] = xq[i][1] = make_float2(0.f, 0.f);
      if (valid && g < G) {
        const float *qg = p.q + (size_t)b * p.n_heads * HD + (size_t)(kvh * G + g) * HD + 16 * st + 2 * t;
        xq[i][0] = __ldcg(reinterpret_cast<const float2 *>(qg));
        xq[i][1] = __ldcg(reinterpret_cast<const float2 *>(qg + 8));
      }
    }
#pragma unroll
    for (int i = 0; i < QPT; ++i) {
      uint4 f;
      bf16_pair2(xq[i][0].x * p.scale_log2, xq[i][0].y * p.scale_log2, f.x, f.y);
      bf16_pair2(xq[i][1].x * p.scale_log2, xq[i][1].y * p.scale_log2, f.z, f.w);
      qf[tid + i * ATC_WARPS * 32] = f;
    }
    named_bar_sync(ATT_BAR, ATC_WARPS * 32);
    stamp(TR_X_GO);

    // q's A fragments stay in registers for the whole loop
    uint4 qr[KS];
#pragma unroll
    for (int k = 0; k < KS; ++k) qr[k] = qf[k * 32 + lane];
    const int w0 = warp * 16;  // this warp's positions within a stage
    float m_run = -INFINITY, l_run = 0.f;  // head gid
    float acc[NT][4];  // rows gid (P's rounded parts) and gid + 8 (rests): both head gid's
#pragma unroll
    for (int d = 0; d < NT; ++d) acc[d][0] = acc[d][1] = acc[d][2] = acc[d][3] = 0.f;
    for (int t = 0; t < nsub; ++t) {
      const int s = t % S;
      if (s_abort) break;
      if (!mbar_wait(smem_addr(&full[s]), (t / S) & 1)) {
        s_abort = 1;
        atomicOr(p.err, ERR_TIMEOUT);
        break;
      }
      if (t == 0) stamp(TR_X_LAST);
      const int nv = min(ATT_SUB, end - (start + t * ATT_SUB)) - w0;  // valid positions of this warp
      const uint32_t kb = sm0 + s * L::STAGE_BYTES, vb = kb + L::KV_BYTES;
      if (nv > 0) {
        if (nv < 16) {
          // rows past the last position take part in P V with weight 0: make them finite
          uint8_t *vg = sm + s * L::STAGE_BYTES + L::KV_BYTES;
          for (int e = lane; e < (16 - nv) * 8 * L::BOXES; e += 32) {
            const int row = w0 + nv + e / (8 * L::BOXES), rest = e % (8 * L::BOXES);
            *reinterpret_cast<uint4 *>(vg + (rest >> 3) * L::BOX_BYTES + row * 128 + (rest & 7) * 16) =
                make_uint4(0u, 0u, 0u, 0u);
          }
          // these stores come before the stage's next TMA write (another proxy) in every order
          asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
          __syncwarp();
        }
        // scores of positions w0 + 8 j + (2 tig, 2 tig + 1), n-tile j = 0, 1, for head gid: two
        // accumulator chains per n-tile (K-step parity); every K fragment is loaded first (one
        // round of shared-memory latency per stage, not one per K step)
        const int mi = lane >> 3, rr = lane & 7;
        uint32_t kf[KS / 2][2][4];
#pragma unroll
        for (int k2 = 0; k2 < KS / 2; ++k2) {
          const int ch = 4 * k2 + mi;  // the 16-byte chunk of dimensions this lane addresses
#pragma unroll
          for (int j = 0; j < 2; ++j)
            ldsm_x4(kf[k2][j][0], kf[k2][j][1], kf[k2][j][2], kf[k2][j][3],
                    kb + (ch >> 3) * L::BOX_BYTES + swz128(w0 + 8 * j + rr, ch & 7));
        }
        float sc[2][2][4] = {};
#pragma unroll
        for (int k2 = 0; k2 < KS / 2; ++k2) {
          const uint4 qa = qr[2 * k2], qb = qr[2 * k2 + 1];
#pragma unroll
          for (int j = 0; j < 2; ++j) {
            mma_bf16(sc[j][0], qa.x, qa.y, qa.z, qa.w, kf[k2][j][0], kf[k2][j][1]);
            mma_bf16(sc[j][1], qb.x, qb.y, qb.z, qb.w, kf[k2][j][2], kf[k2][j][3]);
          }
        }
        // V's fragments (8 x 8 blocks of positions x dimensions, by transposing loads), in flight
        // during the softmax
        uint32_t vf[NT / 2][4];
        {
          const int vrow = w0 + 8 * (mi & 1) + rr;
#pragma unroll
          for (int d2 = 0; d2 < NT / 2; ++d2) {
            const int ch = 2 * d2 + (mi >> 1);
            ldsm_x4_t(vf[d2][0], vf[d2][1], vf[d2][2], vf[d2][3], vb + (ch >> 3) * L::BOX_BYTES + swz128(vrow, ch & 7));
          }
        }
        float sv[2][2];
        float mx = -INFINITY;
#pragma unroll
        for (int j = 0; j < 2; ++j)
#pragma unroll
          for (int e = 0; e < 2; ++e) {
            const float v = (sc[j][0][e] + sc[j][1][e]) + (sc[j][0][e + 2] + sc[j][1][e + 2]);
            sv[j][e] = 8 * j + 2 * tig + e < nv ? v : -INFINITY;
            mx = fmaxf(mx, sv[j][e]);
          }
        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 2));
        const float m_new = fmaxf(m_run, mx);
        // a head with no finite score yet keeps weight 0 and scale 1
        const float alpha = m_new == -INFINITY ? 1.f : exp2f(m_run - m_new);
        float pr[2][2], lsum = 0.f;
#pragma unroll
        for (int j = 0; j < 2; ++j)
#pragma unroll
          for (int e = 0; e < 2; ++e) {
            pr[j][e] = m_new == -INFINITY ? 0.f : exp2f(sv[j][e] - m_new);
            lsum += pr[j][e];
          }
        lsum += __shfl_xor_sync(0xffffffffu, lsum, 1);
        lsum += __shfl_xor_sync(0xffffffffu, lsum, 2);
        l_run = l_run * alpha + lsum;
        m_run = m_new;
        if (__any_sync(0xffffffffu, alpha != 1.f)) {
#pragma unroll
          for (int d = 0; d < NT; ++d)
#pragma unroll
            for (int i = 0; i < 4; ++i) acc[d][i] *= alpha;
        }
        // P as the A fragment of P V over the warp's 16 positions: a0 / a2 the rounded parts of
        // positions (2 tig, 2 tig + 1) and (8 + 2 tig, 9 + 2 tig), a1 / a3 their rests
        uint32_t a0, a1, a2, a3;
        bf16_pair2(pr[0][0], pr[0][1], a0, a1);
        bf16_pair2(pr[1][0], pr[1][1], a2, a3);
        // acc += P V
#pragma unroll
        for (int d2 = 0; d2 < NT / 2; ++d2) {
          mma_bf16(acc[2 * d2], a0, a1, a2, a3, vf[d2][0], vf[d2][1]);
          mma_bf16(acc[2 * d2 + 1], a0, a1, a2, a3, vf[d2][2], vf[d2][3]);
        }
      }
      mbar_arrive(smem_addr(&empty[s]));
      if (t == 0) stamp(TR_E_KIND);
    }
    stamp(TR_E_SEG);
    if (p.launch_at == 2) pdl_launch_dependents();
    // this warp's state: (m, l) per head, sums [warp][head][HD] (rounded + rest rows) in the
    // stage buffers, once every consumer warp has read its last stage (the copies have all landed:
    // each was awaited)
    named_bar_sync(ATT_BAR, ATC_WARPS * 32);
    stamp(TR_E_TICKET);
    if (tig == 0 && gid < G) {
      s_wm[warp][gid] = m_run;
      s_wl[warp][gid] = l_run;
    }
    float *ws = reinterpret_cast<float *>(sm) + (size_t)warp * ATT_MAXG * HD;
    if (gid < G) {
#pragma unroll
      for (int d = 0; d < NT; ++d)
        *reinterpret_cast<float2 *>(ws + gid * HD + 8 * d + 2 * tig) =
            make_float2(acc[d][0] + acc[d][2], acc[d][1] + acc[d][3]);
    }
  }
  __syncthreads();
  // the CTA's state: per head M = max of the warps' m, each warp's weight 2^(m_w - M), l and the
  // sums combined in warp order (unnormalised, relative to M)
  if (tid < G) {
    const int g = tid;
    float M = -INFINITY;
    for (int w = 0; w < ATC_WARPS; ++w) M = fmaxf(M, s_wm[w][g]);
    float Ls = 0.f;
    for (int w = 0; w < ATC_WARPS; ++w) {
      const float e = M == -INFINITY ? 0.f : exp2f(s_wm[w][g] - M);
      s_wm[w][g] = e;
      Ls += s_wl[w][g] * e;
    }
    s_m[g] = M;
    s_l[g] = Ls;
  }
  __syncthreads();
  stamp(TR_W_FIRST);
  // every CTA's receive barrier is initialised
  __syncwarp();
  cluster_wait_acquire();
  // send: this CTA's (m, l) of every head to every CTA of the cluster, and its sums (the warps'
  // sums weighted in warp order) of each output chunk to the CTA that merges the chunk, the
  // largest o with o nch / C <= j
  if (tid < C * G) {
    const int q = tid / G, g = tid % G;
    st_async_f2(map_to_rank(smem_addr(&s_rml[r][g]), q), s_m[g], s_l[g], map_to_rank(rbar, q));
  }
  {
    const float *wsum = reinterpret_cast<const float *>(sm);
    for (int e4 = tid; e4 < G * HD / 4; e4 += ATC_THREADS) {
      const int e = 4 * e4, g = e / HD;
      float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
      for (int w = 0; w < ATC_WARPS; ++w) {
        const float sw = s_wm[w][g];
        const float4 x = *reinterpret_cast<const float4 *>(wsum + (size_t)w * ATT_MAXG * HD + e);
        v.x = fmaf(sw, x.x, v.x);
        v.y = fmaf(sw, x.y, v.y);
        v.z = fmaf(sw, x.z, v.z);
        v.w = fmaf(sw, x.w, v.w);
      }
      const int j = e / XCHUNK;
      const int o = ((j + 1) * C - 1) / nch;
      const int jl = j - static_cast<int>((long long)o * nch / C);
      st_async_f4(map_to_rank(smem_addr(s_recv + ((size_t)r * own + jl) * XCHUNK + e % XCHUNK), o), v,
                  map_to_rank(rbar, o));
    }
  }
  // no CTA leaves while another may still send to it (its wait at the end)
  __syncwarp();
  cluster_arrive_relaxed();

  // receive: every CTA's (m, l) and sums of chunks [c0, c1) have landed (bounded)
  if (!mbar_wait_cluster(rbar, 0)) {
    if (tid == 0) atomicOr(p.err, ERR_TIMEOUT);
  }
  // each CTA's weight per head, 2^(m_q - M) / L with M the largest m and L = sum of l_q 2^(m_q - M)
  // (one warp per head, lane q holding CTA q; a head no CTA has seen gets weight 0)
  for (int g = warp; g < G; g += ATC_WARPS + 1) {
    const float2 ml = lane < C ? s_rml[lane][g] : make_float2(-INFINITY, 0.f);
    float M = ml.x;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, off));
    const float e = ml.x == -INFINITY ? 0.f : exp2f(ml.x - M);
    float Ls = ml.y * e;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) Ls += __shfl_xor_sync(0xffffffffu, Ls, off);
    if (lane < C) s_w[lane][g] = Ls > 0.f ? e * (1.0f / Ls) : 0.f;
  }
  __syncthreads();
  stamp(TR_E_DONE);
  // lane groups of 8 take one chunk each (4 elements per lane); the warps walk the CTA's chunks
  // in groups of 4 per warp (every warp calls act16_put_quad as a whole); the CTAs' sums are
  // added in CTA order
  for (int cb = c0 + warp * 4; cb < c1; cb += (ATC_WARPS + 1) * 4) {
    const int jj = cb + (lane >> 3);
    const bool mine = jj < c1;
    const int jc = mine ? jj : c0;
    const int g = jc / (HD / XCHUNK), d0 = (jc % (HD / XCHUNK)) * XCHUNK + 4 * (lane & 7);
    float4 O = make_float4(0.f, 0.f, 0.f, 0.f);
    if (valid && mine) {
      const float *src = s_recv + (size_t)(jc - c0) * XCHUNK + 4 * (lane & 7);
      for (int q = 0; q < C; ++q) {
        const float4 v = *reinterpret_cast<const float4 *>(src + (size_t)q * own * XCHUNK);
        const float w = s_w[q][g];
        O.x = fmaf(w, v.x, O.x);
        O.y = fmaf(w, v.y, O.y);
        O.z = fmaf(w, v.z, O.z);
        O.w = fmaf(w, v.w, O.w);
      }
    }
    float *o = p.o + (size_t)b * p.ldo + (size_t)kvh * G * HD;
    if (mine) *reinterpret_cast<float4 *>(o + g * HD + d0) = O;
    if (p.o16.base) act16_put_quad(p.o16, b, ((kvh * G + g) * HD + d0) / XCHUNK, O, lane, mine);
  }
  __syncwarp();
  cluster_wait_acquire();
  stamp(TR_CONS_DONE);
}

cudaError_t prepare_attention_cluster() {
  cudaError_t e;
  if ((e = cudaFuncSetAttribute(attn_cluster_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                AtcLayout<128>::smem(ATT_RING_MAX))) != cudaSuccess)
    return e;
  if ((e = cudaFuncSetAttribute(attn_cluster_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                AtcLayout<64>::smem(ATT_RING_MAX))) != cudaSuccess)
    return e;
  if ((e = cudaFuncSetAttribute(attn_cluster_kernel<128>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1)) !=
      cudaSuccess)
    return e;
  return cudaFuncSetAttribute(attn_cluster_kernel<64>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
}

// The largest cluster size up to `want` that the device schedules for this kernel with a ring of
// `stages` sub-tiles, or 0 if none.
int attention_cluster_size(int head_dim, int want, int stages) {
  for (int c = want; c >= 2; --c) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(c);
    cfg.blockDim = dim3(ATC_THREADS);
    cfg.dynamicSmemBytes = head_dim == 128 ? AtcLayout<128>::smem(stages) : AtcLayout<64>::smem(stages);
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
static cudaError_t launch_cluster_hd(const AttnParams &p, const CUtensorMap &km, const CUtensorMap &vm,
                                     cudaStream_t s, bool pdl) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(p.batch * p.n_kv_heads * p.cluster);
  cfg.blockDim = dim3(ATC_THREADS);
  cfg.dynamicSmemBytes = AtcLayout<HD>::smem(p.stages);
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
  return cudaLaunchKernelEx(&cfg, attn_cluster_kernel<HD>, p, km, vm);
}

cudaError_t launch_attention_cluster(const AttnParams &p, const CUtensorMap &km, const CUtensorMap &vm, int head_dim,
                                     cudaStream_t s, bool pdl) {
  if (p.batch < 1 || p.batch > MAXB || p.n_heads % p.n_kv_heads != 0 || p.n_heads / p.n_kv_heads > ATT_MAXG || p.cluster < 1 ||
      p.cluster > MAX_CLUSTER_ATT || p.stages < 2 || p.stages > ATT_RING_MAX)
    return cudaErrorInvalidValue;
  if (head_dim == 128) return launch_cluster_hd<128>(p, km, vm, s, pdl);
  if (head_dim == 64) return launch_cluster_hd<64>(p, km, vm, s, pdl);
  return cudaErrorInvalidValue;
}

// The K (or V) cache of one layer, [max_batch][n_kv_heads][max_ctx][head_dim] bf16, as a 2-D
// tensor of head_dim columns and max_batch * n_kv_heads * max_ctx rows, read in boxes of 64
// positions x 64 dimensions with the 128-byte swizzle; rows past the end read as zero.
int encode_kv_map(CUtensorMap *map, const uint16_t *base, int head_dim, long long rows) {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (!fn) {
    void *f = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault, &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess) {
      cudaGetLastError();
      return -1;
    }
    fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(f);
  }
  if ((head_dim != 64 && head_dim != 128) || (reinterpret_cast<uintptr_t>(base) & 15) != 0 || rows < 1 ||
      rows > 0x7FFFFFFFLL)
    return -1;
  const cuuint64_t dims[2] = {(cuuint64_t)head_dim, (cuuint64_t)rows};
  const cuuint64_t strides[1] = {(cuuint64_t)head_dim * 2};
  const cuuint32_t box[2] = {64, (cuuint32_t)ATT_SUB};
  const cuuint32_t estr[2] = {1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<uint16_t *>(base), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS
             ? 0
             : -1;
}

}  // namespace kfl
