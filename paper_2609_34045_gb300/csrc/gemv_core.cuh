// Device-side building blocks of the weight-streaming GEMV, shared by the standalone GEMV
// kernel (gemv.cu) and the persistent stage kernel (stage_kernel.cu).
//
// Tile layout: a matrix [N][K] is stored as tiles [N/64][K/KT][64][KT]; a consumer CTA has 8
// warps; lane `kc = lane & 15` owns a K chunk (8 bf16 or 16 int4 codes) of the rows
// warp*8 + (lane >> 4) + 2j, j < 4, so each warp-wide shared-memory load reads two whole tile
// rows (conflict-free) and the activation chunk is reused over four rows.
//
// Every global read of data written by other CTAs goes through L2 (ld.global.cg): inside the
// persistent kernel a CTA's L1 may hold lines from an earlier phase.
#pragma once

#include <math.h>

#include "common.cuh"

namespace kfl {

constexpr int CONSUMER_THREADS = CONSUMER_WARPS * 32;
constexpr int CONSUMER_BAR = 1;  // named barrier of the consumer warps

__device__ __forceinline__ void consumer_sync() { named_bar_sync(CONSUMER_BAR, CONSUMER_THREADS); }

// (a0, a1) += (w0, w1) * (x0, x1) with one packed fp32x2 FMA (sm_100+)
__device__ __forceinline__ void ffma2(float &a0, float &a1, float w0, float w1, float x0, float x1) {
  asm("{\n\t.reg .b64 a, w, x;\n\t"
      "mov.b64 a, {%0, %1};\n\tmov.b64 w, {%2, %3};\n\tmov.b64 x, {%4, %5};\n\t"
      "fma.rn.f32x2 a, w, x, a;\n\tmov.b64 {%0, %1}, a;\n\t}"
      : "+f"(a0), "+f"(a1)
      : "f"(w0), "f"(w1), "f"(x0), "f"(x1));
}

// Signed 4-bit code j of a word as an exact float: the offset-binary nibble (code ^ 8) is
// placed in the mantissa of 2^23, and 2^23 + 8 is subtracted.
__device__ __forceinline__ float int4_code(uint32_t word, int j) {
  return __uint_as_float(((word >> (4 * j)) & 0xFu) ^ 0x4B000008u) - 8388616.0f;
}

__device__ __forceinline__ int cta_of_tile(long long t, long long T, int G) {
  // the largest c with floor(c*T/G) <= t
  return static_cast<int>(((t + 1) * G - 1) / T);
}

__device__ __forceinline__ bool consumer_wait(uint32_t bar, uint32_t parity, volatile int *abort_flag,
                                              unsigned *err) {
  if (*abort_flag) return false;
  for (uint32_t i = 0; i < WAIT_LIMIT; ++i) {
    if (mbar_try_wait(bar, parity)) return true;
    if (i >= WAIT_FAST_SPINS) {
      if (*abort_flag) return false;
      __nanosleep(64);
    }
  }
  *abort_flag = 1;
  atomicOr(err, ERR_TIMEOUT);
  return false;
}

// ---------------------------------------------------------------------------- epilogues
// red[r * MAXB + b] holds the finished dot product of row rb*RB + r for user b (before the
// RMSNorm scale inv[b]).  Called by the 256 consumer threads; every thread reaches every
// barrier.
template <int B, int EPI>
__device__ __forceinline__ void epilogue(const GemvParams &p, int rb, const float *red, const float *inv,
                                         float *scr, int tid) {
  const int warp = tid >> 5, lane = tid & 31;
  if constexpr (EPI == EPI_STORE) {
    if (tid < RB * B) {
      const int b = tid / RB, r = tid % RB, n = rb * RB + r;
      if (n < p.n_rows) p.out[(size_t)b * p.ldo + n] = red[r * MAXB + b] * inv[b];
    }
  } else if constexpr (EPI == EPI_RESID) {
    float sq = 0.f;
    if (tid < RB * B) {
      const int b = tid >> 6, r = tid & 63, n = rb * RB + r;
      if (n < p.n_rows) {
        const size_t o = (size_t)b * p.ldh + n;
        const float hn = __ldcg(p.h + o) + red[r * MAXB + b] * inv[b];
        p.h[o] = hn;
        if (p.g_next) p.xn[o] = hn * p.g_next[n];
        if (p.capture) p.capture[(size_t)b * p.n_rows + n] = hn;
        sq = hn * hn;
      }
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) sq += __shfl_xor_sync(0xffffffffu, sq, off);
    if (lane == 0) scr[warp] = sq;
    named_bar_sync(1, CONSUMER_WARPS * 32);
    if (tid < B) p.sumsq_out[rb * MAXB + tid] = scr[2 * tid] + scr[2 * tid + 1];
  } else if constexpr (EPI == EPI_SWIGLU) {
    if (tid < 32 * B) {
      const int b = tid >> 5, pr = tid & 31, j = rb * (RB / 2) + pr;
      if (2 * j < p.n_rows) {
        const float g = red[(2 * pr) * MAXB + b] * inv[b];
        const float u = red[(2 * pr + 1) * MAXB + b] * inv[b];
        p.out[(size_t)b * p.ldo + j] = g / (1.0f + expf(-g)) * u;
      }
    }
  } else if constexpr (EPI == EPI_QKV) {
    if (tid < 32 * B) {
      const int b = tid >> 5, pr = tid & 31, r0 = rb * RB + 2 * pr;
      int pos = p.positions[b];
      const bool ok = pos >= 0 && pos < p.max_ctx;
      if (!ok) pos = 0;
      if (r0 < p.n_rows) {
        const int hd = p.head_dim, half = hd >> 1;
        const float v1 = red[(2 * pr) * MAXB + b] * inv[b];
        const float v2 = red[(2 * pr + 1) * MAXB + b] * inv[b];
        if (r0 < p.n_q_rows + p.n_kv_rows) {
          const bool is_q = r0 < p.n_q_rows;
          const int rr = is_q ? r0 : r0 - p.n_q_rows;
          const int head = rr / hd, i = (rr % hd) >> 1;
          const size_t ri = (size_t)(p.rope_per_user ? b : pos) * half + i;
          const float cs = p.rope_cos[ri];
          const float sn = p.rope_sin[ri];
          const float a = v1 * cs - v2 * sn;
          const float c = v2 * cs + v1 * sn;
          if (is_q) {
            float *qd = p.q + (size_t)b * p.n_q_rows + head * hd;
            qd[i] = a;
            qd[i + half] = c;
          } else if (ok) {
            uint16_t *kd = p.kcache + (((size_t)b * p.n_kv_heads + head) * p.max_ctx + pos) * hd;
            kd[i] = f32_to_bf16_rne(a);
            kd[i + half] = f32_to_bf16_rne(c);
          }
        } else if (ok) {
          const int rr = r0 - p.n_q_rows - p.n_kv_rows;
          const int head = rr / hd, j = rr % hd;
          uint16_t *vd = p.vcache + (((size_t)b * p.n_kv_heads + head) * p.max_ctx + pos) * hd;
          vd[j] = f32_to_bf16_rne(v1);
          vd[j + 1] = f32_to_bf16_rne(v2);
        }
      }
    }
  } else if constexpr (EPI == EPI_ARGMAX) {
    int *scri = reinterpret_cast<int *>(scr + CONSUMER_WARPS);
    __shared__ int s_last_am;
    float v = -INFINITY;
    int idx = 0x7fffffff;
    if (tid < RB * B) {
      const int b = tid >> 6, r = tid & 63, n = rb * RB + r;
      if (n < p.n_rows) {
        v = red[r * MAXB + b] * inv[b];
        idx = n;
      }
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      const float ov = __shfl_xor_sync(0xffffffffu, v, off);
      const int oi = __shfl_xor_sync(0xffffffffu, idx, off);
      if (ov > v || (ov == v && oi < idx)) { v = ov; idx = oi; }
    }
    if (lane == 0) { scr[warp] = v; scri[warp] = idx; }
    named_bar_sync(1, CONSUMER_WARPS * 32);
    if (tid < B) {
      float bv = scr[2 * tid];
      int bi = scri[2 * tid];
      const float ov = scr[2 * tid + 1];
      const int oi = scri[2 * tid + 1];
      if (ov > bv || (ov == bv && oi < bi)) { bv = ov; bi = oi; }
      p.cand_val[rb * MAXB + tid] = bv;
      p.cand_idx[rb * MAXB + tid] = bi;
    }
    named_bar_sync(1, CONSUMER_WARPS * 32);
    if (tid == 0) {
      const unsigned prev = atom_add_acq_rel(reinterpret_cast<unsigned *>(p.argmax_ticket), 1u);
      s_last_am = (prev == (unsigned)(p.n_rb - 1));
      if (s_last_am) atomicExch(p.argmax_ticket, 0);
    }
    named_bar_sync(1, CONSUMER_WARPS * 32);
    if (s_last_am) {
      for (int b = 0; b < B; ++b) {
        float bv = -INFINITY;
        int bi = 0x7fffffff;
        for (int r = tid; r < p.n_rb; r += CONSUMER_WARPS * 32) {
          const float ov = __ldcg(p.cand_val + r * MAXB + b);
          const int oi = __ldcg(p.cand_idx + r * MAXB + b);
          if (ov > bv || (ov == bv && oi < bi)) { bv = ov; bi = oi; }
        }
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) {
          const float ov = __shfl_xor_sync(0xffffffffu, bv, off);
          const int oi = __shfl_xor_sync(0xffffffffu, bi, off);
          if (ov > bv || (ov == bv && oi < bi)) { bv = ov; bi = oi; }
        }
        named_bar_sync(1, CONSUMER_WARPS * 32);
        if (lane == 0) { scr[warp] = bv; scri[warp] = bi; }
        named_bar_sync(1, CONSUMER_WARPS * 32);
        if (tid == 0) {
          bv = scr[0];
          bi = scri[0];
          for (int w = 1; w < CONSUMER_WARPS; ++w) {
            if (scr[w] > bv || (scr[w] == bv && scri[w] < bi)) { bv = scr[w]; bi = scri[w]; }
          }
          p.next_ids[b] = (bi == 0x7fffffff) ? 0 : bi;
        }
      }
    }
  }
}


// Accumulate one tile (in shared memory at `st`, activations after the weights) into acc.
template <int B, int FMT>
__device__ __forceinline__ void tile_compute(const uint8_t *st, int warp, int lane, float (&acc)[B][4][2]) {
  const int kc = lane & 15, rsub = lane >> 4;
  if constexpr (FMT == 0) {
    float xv[B][8];
    const float4 *xp = reinterpret_cast<const float4 *>(st + TILE_BYTES) + kc * 2;
#pragma unroll
    for (int b = 0; b < B; ++b) {
      const float4 a0 = xp[b * (KT / 4)], a1 = xp[b * (KT / 4) + 1];
      xv[b][0] = a0.x; xv[b][1] = a0.y; xv[b][2] = a0.z; xv[b][3] = a0.w;
      xv[b][4] = a1.x; xv[b][5] = a1.y; xv[b][6] = a1.z; xv[b][7] = a1.w;
    }
    const uint4 *wp = reinterpret_cast<const uint4 *>(st) + (warp * 8 + rsub) * (KT / 8) + kc;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const uint4 w4 = wp[j * 2 * (KT / 8)];
      const uint32_t wu[4] = {w4.x, w4.y, w4.z, w4.w};
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const float wl = bf16_lo(wu[e]), wh = bf16_hi(wu[e]);
#pragma unroll
        for (int b = 0; b < B; ++b) ffma2(acc[b][j][0], acc[b][j][1], wl, wh, xv[b][2 * e], xv[b][2 * e + 1]);
      }
    }
  } else {
    // int4 tile: codes [RB][KT4/8] uint32 (32 words = 128 B per row), scales [RB][4] bf16.
    // The lane's 16 codes of a row (two words, one scale group) are taken a word at a time so
    // that only 8 activations per user are live.
    const float4 *xp = reinterpret_cast<const float4 *>(st + TILE4_BYTES) + kc * 4;
    const uint2 *cp = reinterpret_cast<const uint2 *>(st) + (warp * 8 + rsub) * (KT4 / 16) + kc;
    const uint16_t *sp = reinterpret_cast<const uint16_t *>(st + TILE4_CODE_BYTES);
    uint2 cw[4];
    float sc[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      cw[j] = cp[j * 2 * (KT4 / 16)];
      sc[j] = bf16_to_f32(sp[(warp * 8 + rsub + 2 * j) * (KT4 / 64) + (kc >> 2)]);
    }
#pragma unroll
    for (int hw = 0; hw < 2; ++hw) {
      float xv[B][8];
#pragma unroll
      for (int b = 0; b < B; ++b) {
        const float4 a0 = xp[b * (KT4 / 4) + 2 * hw], a1 = xp[b * (KT4 / 4) + 2 * hw + 1];
        xv[b][0] = a0.x; xv[b][1] = a0.y; xv[b][2] = a0.z; xv[b][3] = a0.w;
        xv[b][4] = a1.x; xv[b][5] = a1.y; xv[b][6] = a1.z; xv[b][7] = a1.w;
      }
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const uint32_t word = hw ? cw[j].y : cw[j].x;
        float part[B][2];
#pragma unroll
        for (int b = 0; b < B; ++b) part[b][0] = part[b][1] = 0.f;
#pragma unroll
        for (int e = 0; e < 8; e += 2) {
          const float q0 = int4_code(word, e), q1 = int4_code(word, e + 1);
#pragma unroll
          for (int b = 0; b < B; ++b) ffma2(part[b][0], part[b][1], q0, q1, xv[b][e], xv[b][e + 1]);
        }
#pragma unroll
        for (int b = 0; b < B; ++b) ffma2(acc[b][j][0], acc[b][j][1], sc[j], sc[j], part[b][0], part[b][1]);
      }
    }
  }
}

// RMSNorm scale of the GEMV input (1 without a norm): warp b sums the per-row-block sums of
// squares of user b's h (lane j takes parts j, j+32, ... in order, then a fixed butterfly), so
// the loads are independent and the order is the same on every call.  Writes inv[0..B).
template <int B>
__device__ __forceinline__ void norm_scale(const GemvParams &p, float *inv, int tid) {
  const int warp = tid >> 5, lane = tid & 31;
  if (warp < B) {
    float v = 1.0f;
    if (p.sumsq) {
      float s = 0.f;
      for (int i = lane; i < p.n_parts; i += 32) s += __ldcg(p.sumsq + i * MAXB + warp);
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) s += __shfl_xor_sync(0xffffffffu, s, off);
      v = 1.0f / sqrtf(s / static_cast<float>(p.d_norm) + p.eps);
    }
    if (lane == 0) inv[warp] = v;
  }
}

// End of a row-block segment [seg_kt0, kt] of tile row block rb in CTA c (of G) whose tile range
// starts at t0: reduce the lanes of each row, combine with the neighbouring CTAs that share the
// row block (partials + atomic ticket; the last to arrive sums them in CTA order), and run the
// epilogue once per row block.  All consumer threads call it.
// Wait (one thread, bounded) until a counter written by other CTAs reaches `need`.
__device__ __forceinline__ bool wait_counter(const unsigned *ctr, unsigned need, volatile int *abort_flag,
                                             unsigned *err) {
  for (uint32_t i = 0; i < 64u * WAIT_LIMIT; ++i) {
    if (ld_acquire_gpu(ctr) >= need) return true;
    if ((i & 255) == 255 && *abort_flag) return false;
  }
  *abort_flag = 1;
  atomicOr(err, ERR_TIMEOUT);
  return false;
}

template <int B, int EPI>
__device__ __forceinline__ void segment_end(const GemvParams &p, int rb, int kt, int seg_kt0, long long t0,
                                            long long T, int G, int c, float (&acc)[B][4][2], float *red,
                                            float *scr, float *inv, int *inv_ready, int *s_last,
                                            volatile int *abort_flag, int tid) {
  const int warp = tid >> 5, lane = tid & 31, kc = lane & 15, rsub = lane >> 4;
  float tot[B][4];
#pragma unroll
  for (int b = 0; b < B; ++b)
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      float v = acc[b][j][0] + acc[b][j][1];
      v += __shfl_xor_sync(0xffffffffu, v, 8);
      v += __shfl_xor_sync(0xffffffffu, v, 4);
      v += __shfl_xor_sync(0xffffffffu, v, 2);
      v += __shfl_xor_sync(0xffffffffu, v, 1);
      tot[b][j] = v;
    }
  if (kc == 0) {
#pragma unroll
    for (int j = 0; j < 4; ++j)
#pragma unroll
      for (int b = 0; b < B; ++b) red[(warp * 8 + rsub + 2 * j) * MAXB + b] = tot[b][j];
  }
  consumer_sync();
  bool do_epi = true;
  if (!(seg_kt0 == 0 && kt == p.n_kt - 1)) {
    // this row block is shared with neighbouring CTAs
    const int first_rb = static_cast<int>(t0 / p.n_kt);
    const int slot = (rb == first_rb) ? 0 : 1;
    float *mine = p.partial + (size_t)(c * 2 + slot) * (RB * MAXB);
    for (int e = tid; e < RB * MAXB; e += CONSUMER_THREADS) mine[e] = red[e];
    consumer_sync();
    const int c_lo = cta_of_tile((long long)rb * p.n_kt, T, G);
    const int c_hi = cta_of_tile((long long)(rb + 1) * p.n_kt - 1, T, G);
    if (tid == 0) {
      // release this CTA's partials; the last to arrive acquires everyone's
      const unsigned prev = atom_add_acq_rel(reinterpret_cast<unsigned *>(p.tickets + rb), 1u);
      *s_last = (prev == (unsigned)(c_hi - c_lo));
      if (*s_last) atomicExch(p.tickets + rb, 0);
    }
    consumer_sync();
    do_epi = *s_last != 0;
    if (do_epi) {
      // issue every partial's load first (independent), then add them in CTA order
      constexpr int MAXPART = 8;
      for (int e = tid; e < RB * MAXB; e += CONSUMER_THREADS) {
        float sum = 0.f;
        for (int c0 = c_lo; c0 <= c_hi; c0 += MAXPART) {
          float v[MAXPART];
#pragma unroll
          for (int j = 0; j < MAXPART; ++j) {
            const int cc = c0 + j;
            v[j] = 0.f;
            if (cc <= c_hi) {
              const int frb = static_cast<int>(((long long)cc * T / G) / p.n_kt);
              const int sl = (rb == frb) ? 0 : 1;
              v[j] = __ldcg(p.partial + (size_t)(cc * 2 + sl) * (RB * MAXB) + e);
            }
          }
#pragma unroll
          for (int j = 0; j < MAXPART; ++j)
            if (c0 + j <= c_hi) sum += v[j];
        }
        red[e] = sum;
      }
      consumer_sync();
    }
  }
  if (do_epi && !*inv_ready) {
    // the RMSNorm scale needs every row block of h: in the persistent kernel wait for the
    // phase that produces h to complete them
    if (tid == 0 && p.norm_done) wait_counter(p.norm_done, (unsigned)p.norm_need, abort_flag, p.err);
    consumer_sync();
    norm_scale<B>(p, inv, tid);
    consumer_sync();
    if (tid == 0) *inv_ready = 1;
  }
  if (do_epi) epilogue<B, EPI>(p, rb, red, inv, scr, tid);
  consumer_sync();
  if (do_epi && tid == 0) {
    // publish this row block (the bar.sync above ordered every consumer's stores before it)
    if (p.out_ready) {
      int idx;
      if constexpr (EPI == EPI_QKV) {
        const int r0 = rb * RB, hd = p.head_dim;
        const int group = p.n_q_rows / p.n_kv_rows;
        if (r0 < p.n_q_rows)
          idx = (r0 / hd) / group;
        else if (r0 < p.n_q_rows + p.n_kv_rows)
          idx = (r0 - p.n_q_rows) / hd;
        else
          idx = (r0 - p.n_q_rows - p.n_kv_rows) / hd;
      } else {
        idx = (rb * p.out_unit) / p.out_kt;
      }
      red_add_release(p.out_ready + idx, 1u);
    }
    if (p.out_done) red_add_release(p.out_done, 1u);
  }
}

// Consumer side of one GEMV over this CTA's tile range [t0, t0 + n): wait for each tile's ring
// stage, accumulate, release the stage, finish segments.  (s, phase) is the ring position,
// carried across calls when consecutive GEMVs share one ring.
template <int B, int EPI, int FMT>
__device__ __forceinline__ void gemv_consume(const GemvParams &p, uint8_t *ring, uint64_t *full, uint64_t *empty,
                                             int S, int &s, uint32_t &phase, long long t0, int n, long long T,
                                             int G, int c, float *red, float *scr, float *inv, int *inv_ready,
                                             int *s_last, volatile int *abort_flag, int tid) {
  const int warp = tid >> 5, lane = tid & 31;
  float acc[B][4][2];
  int seg_kt0 = 0;
  int rb = static_cast<int>(t0 / p.n_kt);
  int kt = static_cast<int>(t0 - (long long)rb * p.n_kt);
  for (int i = 0; i < n; ++i) {
    if (i == 0 || kt == 0) {
#pragma unroll
      for (int b = 0; b < B; ++b)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[b][j][0] = acc[b][j][1] = 0.f;
      seg_kt0 = kt;
    }
    consumer_wait(smem_addr(&full[s]), phase, abort_flag, p.err);
    tile_compute<B, FMT>(ring + (size_t)s * stage_bytes(B, FMT), warp, lane, acc);
    __syncwarp();
    if (lane == 0) mbar_arrive(smem_addr(&empty[s]));
    if (kt == p.n_kt - 1 || i == n - 1)
      segment_end<B, EPI>(p, rb, kt, seg_kt0, t0, T, G, c, acc, red, scr, inv, inv_ready, s_last, abort_flag, tid);
    if (++kt == p.n_kt) {
      kt = 0;
      ++rb;
    }
    if (++s == S) {
      s = 0;
      phase ^= 1u;
    }
  }
}

}  // namespace kfl
