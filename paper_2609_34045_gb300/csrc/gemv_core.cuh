// Device-side building blocks of the weight-streaming GEMV, shared by the standalone GEMV
// kernel (gemv.cu) and the persistent stage kernel (stage_kernel.cu).
//
// Tile layout: a matrix [N][K] is stored as tiles [N/64][K/KT][64][KT]; the 8 consumer warps of
// a CTA each own 8 rows of every tile: lane `kc = lane & 15` takes a K chunk (8 bf16 or 16 int4
// codes) of rows warp*8 + (lane >> 4) + 2j, j < 4, so a warp-wide shared-memory load reads two
// whole tile rows (conflict-free) and the activation chunk is reused over four rows.
//
// The consumer warps never stop for an epilogue: at the end of a row-block segment each warp
// reduces its rows into a staging slot and goes on with the next tile.  One epilogue warp takes
// the slots in the same order and does everything with latency: the partial sums of row blocks
// shared with neighbouring CTAs (written to global memory; the last CTA to arrive on an atomic
// ticket adds them in CTA order), the RMSNorm scale, the fused epilogue, and (persistent kernel)
// the readiness counters.  Memory in flight therefore never drains at a segment end.
//
// Every global read of data written by other CTAs goes through L2 (ld.global.cg): inside the
// persistent kernel a CTA's L1 may hold lines from an earlier phase.
#pragma once

#include <math.h>

#include "common.cuh"

namespace kfl {

constexpr int CONSUMER_THREADS = CONSUMER_WARPS * 32;
constexpr int CONSUMER_BAR = 1;  // named barrier of the consumer warps
constexpr int NSLOT = 4;         // staging slots between the consumer warps and the epilogue warp

__device__ __forceinline__ void consumer_sync() { named_bar_sync(CONSUMER_BAR, CONSUMER_THREADS); }

// (a0, a1) += (w0, w1) * (x0, x1) with one packed fp32x2 FMA (sm_100+)
__device__ __forceinline__ void ffma2(float &a0, float &a1, float w0, float w1, float x0, float x1) {
  asm("{\n\t.reg .b64 a, w, x;\n\t"
      "mov.b64 a, {%0, %1};\n\tmov.b64 w, {%2, %3};\n\tmov.b64 x, {%4, %5};\n\t"
      "fma.rn.f32x2 a, w, x, a;\n\tmov.b64 {%0, %1}, a;\n\t}"
      : "+f"(a0), "+f"(a1)
      : "f"(w0), "f"(w1), "f"(x0), "f"(x1));
}

// (d0, d1) = (a0, a1) * (b0, b1) with one packed fp32x2 multiply (sm_100+)
__device__ __forceinline__ void fmul2(float &d0, float &d1, float a0, float a1, float b0, float b1) {
  asm("{\n\t.reg .b64 d, a, b;\n\t"
      "mov.b64 a, {%2, %3};\n\tmov.b64 b, {%4, %5};\n\t"
      "mul.rn.f32x2 d, a, b;\n\tmov.b64 {%0, %1}, d;\n\t}"
      : "=f"(d0), "=f"(d1)
      : "f"(a0), "f"(a1), "f"(b0), "f"(b1));
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

// Bounded wait on an mbarrier phase that also ends when the CTA aborts.
// The first poll comes before the abort flag is read: in a running ring the phase is usually
// complete already, and then the wait costs one poll.
__device__ __forceinline__ bool consumer_wait(uint32_t bar, uint32_t parity, volatile int *abort_flag,
                                              unsigned *err) {
  if (mbar_try_wait(bar, parity)) return true;
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

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
  return v;
}

// (value, index) maximum with the lowest index on ties
__device__ __forceinline__ void argmax_merge(float &v, int &i, float ov, int oi) {
  if (ov > v || (ov == v && oi < i)) {
    v = ov;
    i = oi;
  }
}

__device__ __forceinline__ void warp_argmax(float &v, int &i) {
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    const float ov = __shfl_xor_sync(0xffffffffu, v, off);
    const int oi = __shfl_xor_sync(0xffffffffu, i, off);
    argmax_merge(v, i, ov, oi);
  }
}

// ---------------------------------------------------------------------------- consumers
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
  }
}

// d += a b for one m16n8k16 fp16 tile (a: 16x16 row-major, b: 16x8 column-major, fp32 accumulate)
__device__ __forceinline__ void mma_f16_16816(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                               uint32_t b0, uint32_t b1) {
  asm(
      "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// The A fragment of one m16n8k16 MMA from one 32-bit word of 8 offset-binary codes u = code + 8
// (repack_int4_kernel): the nibble pairs at bits (0, 16) and (8, 24) become the fp16 pairs
// 1024 + u (registers a0, a1: K elements 0..7 of the step), those at (4, 20) and (12, 28)
// become 1024 + 16 u (a2, a3: elements 8..15, whose activations are stored divided by 16), each
// with one lop3 ((w & mask) | 0x6400 in each half, with the code's top bit flipped: the stored
// nibble is the two's-complement code).  The offsets 1032 x and 1152 x / 16 that this adds to
// the product are taken off with the activations' offset sums (Act16).
__device__ __forceinline__ void int4_frag_f16(uint32_t w, uint32_t &a0, uint32_t &a1, uint32_t &a2, uint32_t &a3) {
  const uint32_t w8 = w >> 8;
  asm("lop3.b32 %0, %1, %2, %3, 0x6A;" : "=r"(a0) : "r"(w), "r"(0x000F000Fu), "r"(0x64086408u));   // (w & m) ^ c
  asm("lop3.b32 %0, %1, %2, %3, 0x6A;" : "=r"(a1) : "r"(w8), "r"(0x000F000Fu), "r"(0x64086408u));
  asm("lop3.b32 %0, %1, %2, %3, 0x6A;" : "=r"(a2) : "r"(w), "r"(0x00F000F0u), "r"(0x64806480u));
  asm("lop3.b32 %0, %1, %2, %3, 0x6A;" : "=r"(a3) : "r"(w8), "r"(0x00F000F0u), "r"(0x64806480u));
}

// d = a b + c for one m16n8k16 fp16 tile, the accumulator seeded from c
__device__ __forceinline__ void mma_f16_16816_seed(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                                    uint32_t b0, uint32_t b1, float4 c) {
  asm(
      "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%10,%11,%12,%13};"
      : "=f"(d[0]), "=f"(d[1]), "=f"(d[2]), "=f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1), "f"(c.x), "f"(c.y), "f"(c.z), "f"(c.w));
}

// int4 tile (FMT 1) on the tensor cores.  The consumer warps form two teams of four: team
// w / 4 takes every other tile of the CTA's range, and warp w takes weight group g4 = w % 4 (64
// of the tile's 256 K) of all four row groups (64 rows).  Per K step of 16, one m16n8k16 MMA
// (fp16, fp32 accumulate) of the decoded codes against eight columns of activations; so every
// B fragment, seed and multiplier a warp loads from shared memory serves four MMAs, one per row
// group (a warp per row group would load them four times over, and shared-memory wavefronts,
// not instructions, would bound the kernel).  Column j is source row j % B (the users' rounded
// parts); with XSPLIT, columns 4..7 are the rests (source rows MAXB + (j - 4) % B).  Columns past
// the users carry copies and are dropped at the end.  A chunk's first MMA seeds the accumulator
// with minus the columns' offset sums, so that after its two MMAs it holds the product of the
// codes with the scaled activations; the group's two chunks are multiplied back by their
// multipliers and summed (packed fp32x2), then scaled by the rows' group scale into acc.
// acc[r16][0..1]: row r16*16 + gid, columns 2 tig, 2 tig + 1; acc[r16][2..3]: row + 8.

// Byte offsets, within a ring stage, of one consumer lane's operands (fixed for the whole GEMV).
struct Int4Lane {
  uint32_t cw;  // code words of row group 0 (uint4: the group's four K steps); row group r16 at + 1024 r16
  uint32_t sc;  // scales of rows gid and gid + 8 of the four row groups (tile4_scale_index), 16 bytes
  uint32_t xb;  // B fragments of the group's first chunk (its second at + 64)
  uint32_t xc;  // the group's constants: seed a, seed b (+ 64), multipliers (+ 128)
};

template <int B, bool XSPLIT>
__device__ __forceinline__ Int4Lane int4_lane(int warp, int lane) {
  const int g4 = warp & 3, h = g4 >> 1, q = g4 & 1, gid = lane >> 2, tig = lane & 3;
  const int src = XSPLIT ? (gid < 4 ? gid % B : MAXB + (gid - 4) % B) : gid % B;
  Int4Lane L;
  L.cw = static_cast<uint32_t>(((h * 8 + q) * 32 + lane) * 16);
  L.sc = static_cast<uint32_t>(TILE4_CODE_BYTES + 2 * tile4_scale_index(gid, g4));
  L.xb = static_cast<uint32_t>(TILE4_BYTES + XC_TILE_BYTES + src * X16_SRC_STRIDE + g4 * 128 + tig * 16);
  L.xc = static_cast<uint32_t>(TILE4_BYTES + g4 * XC_GROUP_BYTES + tig * 16);
  return L;
}

template <int B, bool XSPLIT>
__device__ __forceinline__ void tile_compute_int4(const uint8_t *st, const Int4Lane &L, float (&acc)[4][4]) {
  uint4 w[4];
#pragma unroll
  for (int r16 = 0; r16 < 4; ++r16) w[r16] = *reinterpret_cast<const uint4 *>(st + L.cw + r16 * 1024);
  const uint4 sc = *reinterpret_cast<const uint4 *>(st + L.sc);  // row groups 0..3: (row gid, row gid + 8)
  const uint4 ba = *reinterpret_cast<const uint4 *>(st + L.xb);
  const uint4 bb = *reinterpret_cast<const uint4 *>(st + L.xb + 64);
  const float4 seed_a = *reinterpret_cast<const float4 *>(st + L.xc);
  const float4 seed_b = *reinterpret_cast<const float4 *>(st + L.xc + 64);
  const float4 mq = *reinterpret_cast<const float4 *>(st + L.xc + 128);  // (m_a, m_b) of the two columns
  const float2 ma = make_float2(mq.x, mq.y), mb = make_float2(mq.z, mq.w);
#pragma unroll
  for (int r16 = 0; r16 < 4; ++r16) {
    uint32_t a0, a1, a2, a3;
    float ca[4], cb[4];
    int4_frag_f16(w[r16].x, a0, a1, a2, a3);
    mma_f16_16816_seed(ca, a0, a1, a2, a3, ba.x, ba.y, seed_a);
    int4_frag_f16(w[r16].z, a0, a1, a2, a3);
    mma_f16_16816_seed(cb, a0, a1, a2, a3, bb.x, bb.y, seed_b);
    int4_frag_f16(w[r16].y, a0, a1, a2, a3);
    mma_f16_16816(ca, a0, a1, a2, a3, ba.z, ba.w);
    int4_frag_f16(w[r16].w, a0, a1, a2, a3);
    mma_f16_16816(cb, a0, a1, a2, a3, bb.z, bb.w);
    float2 g0 = __fmul2_rn(ma, make_float2(ca[0], ca[1]));
    float2 g1 = __fmul2_rn(ma, make_float2(ca[2], ca[3]));
    g0 = __ffma2_rn(mb, make_float2(cb[0], cb[1]), g0);
    g1 = __ffma2_rn(mb, make_float2(cb[2], cb[3]), g1);
    const uint32_t sw = r16 == 0 ? sc.x : r16 == 1 ? sc.y : r16 == 2 ? sc.z : sc.w;
    const float sc0 = bf16_lo(sw), sc1 = bf16_hi(sw);
    acc[r16][0] = fmaf(sc0, g0.x, acc[r16][0]);
    acc[r16][1] = fmaf(sc0, g0.y, acc[r16][1]);
    acc[r16][2] = fmaf(sc1, g1.x, acc[r16][2]);
    acc[r16][3] = fmaf(sc1, g1.y, acc[r16][3]);
  }
}

// Staging ring between the consumer warps and the epilogue warp: nslot slots of nsub sub-slots
// of [RB][MAXB] sums.  bf16 tiles: 4 slots of one sub-slot, each value written by one lane.  int4
// tiles: 2 slots of 4 sub-slots, sub-slot g4 receiving exactly two additions (one per team) onto
// zero, so that the order does not change the sum; the epilogue warp adds the sub-slots in order.
struct SegRing {
  float *red;      // [nslot][nsub][RB][MAXB]
  uint64_t *full;  // [nslot], count CONSUMER_WARPS
  uint64_t *empty; // [nslot], count 1
  int nslot, nsub;
};
__host__ __device__ constexpr int seg_slots(int fmt) { return fmt == 0 ? NSLOT : 2; }
__host__ __device__ constexpr int seg_subs(int fmt) { return fmt == 0 ? 1 : 4; }
__host__ __device__ constexpr int seg_floats(int fmt) { return seg_slots(fmt) * seg_subs(fmt) * RB * MAXB; }

// Arrivals that release a weight-ring stage: one per consumer warp (bf16 tiles, lane 0 after a
// __syncwarp) or one per thread of the team that consumed it (int4 tiles: no warp barrier in the
// tile loop).
__host__ __device__ constexpr int ring_empty_count(int fmt) { return fmt == 0 ? CONSUMER_WARPS : CONSUMER_THREADS / 2; }

// int4 consumer side of one GEMV over this CTA's tile range [t0, t0 + n).  The ring depth S is
// even and ring stage r belongs to team r % 2: tile i of the range, in stage (s + i) % S, is
// team (s + i) % 2's.  (Were a stage used by both teams in turn, a warp could come back to it for
// the use after next while the other team's use is still landing, and a parity wait cannot tell
// those two phases apart.)  Per segment (the tiles of one row block) a warp waits for each of its
// team's tiles, computes its weight group of it and releases it with every lane, then adds the
// segment's sums into its sub-slot of the next staging slot.  (s, phase), the ring position of
// the range's first tile, comes back advanced by n, as the persistent kernel carries it across
// GEMVs that share the ring.
template <int B, bool XSPLIT>
__device__ __forceinline__ void gemv_consume_int4(int n_kt, uint8_t *ring, uint64_t *full, uint64_t *empty, int S,
                                                  int &s, uint32_t &phase, long long t0, int n, const SegRing &sr,
                                                  int &segc, volatile int *abort_flag, unsigned *err, int tid) {
  constexpr uint32_t SB = stage_bytes(B, 1);
  const int warp = tid >> 5, lane = tid & 31, team = warp >> 2;
  const Int4Lane L = int4_lane<B, XSPLIT>(warp, lane);
  const uint32_t full0 = smem_addr(full), empty0 = smem_addr(empty);
  // this team's ring position: its first tile of the range, (team ^ s) & 1
  const int par = (team ^ s) & 1;  // tile i is this team's when (i & 1) == par
  int ms = s + par;
  uint32_t mph = phase;
  if (ms >= S) {
    ms -= S;
    mph ^= 1u;
  }
  int kt = static_cast<int>(t0 % n_kt);
  int i = 0;
  while (i < n) {
    const int seg = min(n_kt - kt, n - i);
    float acc[4][4] = {};
    for (int j = (par ^ i) & 1; j < seg; j += 2) {
      consumer_wait(full0 + 8u * ms, mph, abort_flag, err);
      tile_compute_int4<B, XSPLIT>(ring + (size_t)ms * SB, L, acc);
      mbar_arrive(empty0 + 8u * ms);
      ms += 2;
      if (ms >= S) {
        ms -= S;
        mph ^= 1u;
      }
    }
    i += seg;
    kt = 0;
    const int slot = segc % sr.nslot, use = segc / sr.nslot;
    float *rd = sr.red + (slot * sr.nsub + (warp & 3)) * RB * MAXB;
    if (XSPLIT) {
      // rounded part (columns 0-3, lanes tig < 2) + rest (columns 4-7, lanes tig + 2)
#pragma unroll
      for (int r16 = 0; r16 < 4; ++r16)
#pragma unroll
        for (int v = 0; v < 4; ++v) acc[r16][v] += __shfl_down_sync(0xffffffffu, acc[r16][v], 2);
    }
    if (use > 0) consumer_wait(smem_addr(&sr.empty[slot]), (use - 1) & 1, abort_flag, err);
    const int gid = lane >> 2, tig = lane & 3;
#pragma unroll
    for (int r16 = 0; r16 < 4; ++r16) {
      const int r0 = r16 * 16 + gid;
      if (2 * tig < B) {
        atomicAdd(rd + r0 * MAXB + 2 * tig, acc[r16][0]);
        atomicAdd(rd + (r0 + 8) * MAXB + 2 * tig, acc[r16][2]);
      }
      if (2 * tig + 1 < B) {
        atomicAdd(rd + r0 * MAXB + 2 * tig + 1, acc[r16][1]);
        atomicAdd(rd + (r0 + 8) * MAXB + 2 * tig + 1, acc[r16][3]);
      }
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(smem_addr(&sr.full[slot]));
    ++segc;
  }
  const int adv = s + n;
  s = adv % S;
  phase ^= static_cast<uint32_t>((adv / S) & 1);
}

// Consumer side of one GEMV over this CTA's tile range [t0, t0 + n): wait for each tile's ring
// stage, accumulate, release the stage; at each segment end reduce the rows of this warp into the
// next staging slot.  (s, phase) is the ring position and segc the staging count, both carried
// across calls when consecutive GEMVs share the rings.
template <int B, int FMT>
__device__ __forceinline__ void gemv_consume(int n_kt, uint8_t *ring, uint64_t *full, uint64_t *empty, int S, int &s,
                                             uint32_t &phase, long long t0, int n, const SegRing &sr, int &segc,
                                             volatile int *abort_flag, unsigned *err, int tid, bool xsplit) {
  if constexpr (FMT == 1) {
    if (xsplit)
      gemv_consume_int4<B, true>(n_kt, ring, full, empty, S, s, phase, t0, n, sr, segc, abort_flag, err, tid);
    else
      gemv_consume_int4<B, false>(n_kt, ring, full, empty, S, s, phase, t0, n, sr, segc, abort_flag, err, tid);
  } else {
    const int warp = tid >> 5, lane = tid & 31, kc = lane & 15, rsub = lane >> 4;
    float acc[B][4][2];  // rows warp*8 + rsub + 2j, this lane's K chunk
    int kt = static_cast<int>(t0 % n_kt);
    for (int i = 0; i < n; ++i) {
      if (i == 0 || kt == 0) {
#pragma unroll
        for (int b = 0; b < B; ++b)
#pragma unroll
          for (int j = 0; j < 4; ++j) acc[b][j][0] = acc[b][j][1] = 0.f;
      }
      consumer_wait(smem_addr(&full[s]), phase, abort_flag, err);
      tile_compute<B, FMT>(ring + (size_t)s * stage_bytes(B, FMT), warp, lane, acc);
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_addr(&empty[s]));
      if (kt == n_kt - 1 || i == n - 1) {
        const int slot = segc % sr.nslot, use = segc / sr.nslot;
        float *rd = sr.red + slot * RB * MAXB;
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
        if (use > 0) consumer_wait(smem_addr(&sr.empty[slot]), (use - 1) & 1, abort_flag, err);
        if (kc == 0) {
#pragma unroll
          for (int j = 0; j < 4; ++j)
#pragma unroll
            for (int b = 0; b < B; ++b) rd[(warp * 8 + rsub + 2 * j) * MAXB + b] = tot[b][j];
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(smem_addr(&sr.full[slot]));
        ++segc;
      }
      if (++kt == n_kt) kt = 0;
      if (++s == S) {
        s = 0;
        phase ^= 1u;
      }
    }
  }
}


// ---------------------------------------------------------------------------- epilogue warp
// RMSNorm scale of the GEMV input (1 without a norm): user b's scale from the per-row-block sums
// of squares of h, the lanes taking parts j, j+32, ... in order, then a fixed butterfly, so the
// result is the same on every call.
template <int B>
__device__ __forceinline__ void norm_scale_warp(const GemvParams &p, float *inv, int lane) {
#pragma unroll
  for (int b = 0; b < B; ++b) {
    float v = 1.0f;
    if (p.sumsq) {
      float s = 0.f;
      for (int i = lane; i < p.n_parts; i += 32) s += __ldcg(p.sumsq + i * MAXB + b);
      s = warp_sum(s);
      v = 1.0f / sqrtf(s / static_cast<float>(p.d_norm) + p.eps);
    }
    inv[b] = v;
  }
}

// Values the epilogue of a row block reads from global memory, loaded before the row block's
// partial sums are combined so that their latency overlaps the combine (RESID: the residual rows
// and the next RMSNorm gain).  Loaded after the segment's staging slot is full, which orders them
// after the writes of earlier phases.
struct EpiPre {
  float h[MAXB][2];
  float g[2];
  float cs[MAXB], sn[MAXB];  // QKV: the RoPE cos / sin of this lane's row pair, per user
  int pos[MAXB], slot[MAXB]; // QKV: each user's position (-1 if invalid) and KV slot
};

template <int B, int EPI>
__device__ __forceinline__ void epilogue_prefetch(const GemvParams &p, int rb, int lane, EpiPre &e) {
  if constexpr (EPI == EPI_QKV) {
    // lane = row pair (RB / 2 = 32 of them), one user per pass (as in epilogue_warp)
    const int hd = p.head_dim, half = hd >> 1, r0 = rb * RB + 2 * lane;
    const bool rot = r0 < p.n_rows && r0 < p.n_q_rows + p.n_kv_rows;
    const int rr = r0 < p.n_q_rows ? r0 : r0 - p.n_q_rows;
    const int i = (rr % hd) >> 1;
#pragma unroll
    for (int b = 0; b < B; ++b) {
      const int pv = p.positions[b];
      const bool ok = pv >= 0 && pv < p.max_ctx;
      e.pos[b] = ok ? pv : -1;
      e.slot[b] = p.slots[b];
      const size_t ri = (size_t)(p.rope_per_user ? b : (ok ? pv : 0)) * half + i;
      e.cs[b] = rot ? p.rope_cos[ri] : 0.f;
      e.sn[b] = rot ? p.rope_sin[ri] : 0.f;
    }
  } else if constexpr (EPI == EPI_RESID) {
#pragma unroll
    for (int h2 = 0; h2 < 2; ++h2) {
      const int n = rb * RB + lane + 32 * h2;
      const bool ok = n < p.n_rows;
#pragma unroll
      for (int b = 0; b < B; ++b) e.h[b][h2] = ok ? __ldcg(p.h + (size_t)b * p.ldh + n) : 0.f;
      e.g[h2] = ok && p.g_next ? p.g_next[n] : 0.f;
    }
  }
}

// The fused epilogue of row block rb: red[r * MAXB + b] is the dot product of row rb*RB + r for
// user b, before the RMSNorm scale inv[b].  One warp.
template <int B, int EPI>
__device__ __forceinline__ void epilogue_warp(const GemvParams &p, int rb, float *red, const float *inv,
                                              const EpiPre &pre, int lane) {
  if constexpr (EPI == EPI_STORE) {
    for (int e = lane; e < RB * B; e += 32) {
      const int b = e / RB, r = e % RB, n = rb * RB + r;
      if (n < p.n_rows) p.out[(size_t)b * p.ldo + n] = red[r * MAXB + b] * inv[b];
    }
  } else if constexpr (EPI == EPI_RESID) {
    // the new h of every user first, in place of the sums (each lane its own elements), then one
    // user at a time through a loop that is not unrolled: the users' stores and conversions run
    // the same instructions, which a CTA fetches once (the epilogue runs once per row block, so
    // unrolled over the users its code would be fetched cold four times over)
#pragma unroll
    for (int b = 0; b < B; ++b)
#pragma unroll
      for (int h2 = 0; h2 < 2; ++h2) {
        const int r = lane + 32 * h2;
        red[r * MAXB + b] = rb * RB + r < p.n_rows ? pre.h[b][h2] + red[r * MAXB + b] * inv[b] : 0.f;
      }
#pragma unroll 1
    for (int b = 0; b < B; ++b) {
      float sq = 0.f;
#pragma unroll
      for (int h2 = 0; h2 < 2; ++h2) {
        const int r = lane + 32 * h2, n = rb * RB + r;
        const bool ok = n < p.n_rows;
        const size_t o = (size_t)b * p.ldh + n;
        const float hn = red[r * MAXB + b];
        const float xv = hn * pre.g[h2];
        // int4 stage: xn in the tensor-core input form, chunk rb * 2 + h2
        if (p.xout.base && p.g_next) act16_put_warp(p.xout, b, rb * 2 + h2, xv, lane);
        if (ok) {
          p.h[o] = hn;
          if (p.g_next && !p.xout.base) p.xn[o] = xv;
          if (p.capture) p.capture[(size_t)b * p.n_rows + n] = hn;
          sq = fmaf(hn, hn, sq);
        }
      }
      sq = warp_sum(sq);
      if (lane == 0) p.sumsq_out[rb * MAXB + b] = sq;
    }
  } else if constexpr (EPI == EPI_SWIGLU) {
    // lane = output (RB / 2 = 32 of them per row block), one user per pass of a loop that is not
    // unrolled (as in RESID)
#pragma unroll 1
    for (int b = 0; b < B; ++b) {
      const int pr = lane, j = rb * (RB / 2) + pr;
      const bool ok = 2 * j < p.n_rows;
      float a = 0.f;
      if (ok) {
        const float g = red[(2 * lane) * MAXB + b] * inv[b];
        const float u = red[(2 * lane + 1) * MAXB + b] * inv[b];
        a = g / (1.0f + expf(-g)) * u;
      }
      if (p.xout.base)
        act16_put_warp(p.xout, b, rb, a, lane);  // int4 stage: the row block's 32 outputs, one chunk
      else if (ok)
        p.out[(size_t)b * p.ldo + j] = a;
    }
  } else if constexpr (EPI == EPI_QKV) {
    const int hd = p.head_dim, half = hd >> 1;
    // every read before the first store (the compiler cannot tell the stores from these reads)
    float rv1[B], rv2[B], iv[B];
#pragma unroll
    for (int b = 0; b < B; ++b) {
      rv1[b] = red[(2 * lane) * MAXB + b];
      rv2[b] = red[(2 * lane + 1) * MAXB + b];
      iv[b] = inv[b];
    }
#pragma unroll
    for (int b = 0; b < B; ++b) {
      const int pr = lane, r0 = rb * RB + 2 * pr;
      const bool ok = pre.pos[b] >= 0;
      const int pos = ok ? pre.pos[b] : 0;
      if (r0 >= p.n_rows) continue;
      const float v1 = rv1[b] * iv[b];
      const float v2 = rv2[b] * iv[b];
      if (p.qk_raw) {  // QK-norm stage: the kernel after this one rotates and appends
        float *rw = p.qk_raw + (size_t)b * p.ld_raw + r0;
        rw[0] = v1;
        rw[1] = v2;
        continue;
      }
      if (r0 < p.n_q_rows + p.n_kv_rows) {
        const bool is_q = r0 < p.n_q_rows;
        const int rr = is_q ? r0 : r0 - p.n_q_rows;
        const int head = rr / hd, i = (rr % hd) >> 1;
        const float cs = pre.cs[b];
        const float sn = pre.sn[b];
        const float a = v1 * cs - v2 * sn;
        const float c2 = v2 * cs + v1 * sn;
        if (is_q) {
          float *qd = p.q + (size_t)b * p.n_q_rows + head * hd;
          qd[i] = a;
          qd[i + half] = c2;
        } else if (ok) {
          uint16_t *kd = p.kcache + (((size_t)pre.slot[b] * p.n_kv_heads + head) * p.max_ctx + pos) * hd;
          kd[i] = f32_to_bf16_rne(a);
          kd[i + half] = f32_to_bf16_rne(c2);
        }
      } else if (ok) {
        const int rr = r0 - p.n_q_rows - p.n_kv_rows;
        const int head = rr / hd, j = rr % hd;
        uint16_t *vd = p.vcache + (((size_t)pre.slot[b] * p.n_kv_heads + head) * p.max_ctx + pos) * hd;
        vd[j] = f32_to_bf16_rne(v1);
        vd[j + 1] = f32_to_bf16_rne(v2);
      }
    }
  } else if constexpr (EPI == EPI_ARGMAX) {
    // per row block: each user's best row; the last row block to finish (global ticket) reduces
    // the candidates of all row blocks
#pragma unroll
    for (int b = 0; b < B; ++b) {
      float v = -INFINITY;
      int idx = 0x7fffffff;
#pragma unroll
      for (int h2 = 0; h2 < 2; ++h2) {
        const int r = lane + 32 * h2, n = rb * RB + r;
        if (n < p.n_rows) argmax_merge(v, idx, red[r * MAXB + b] * inv[b], n);
      }
      warp_argmax(v, idx);
      if (lane == 0) {
        p.cand_val[rb * MAXB + b] = v;
        p.cand_idx[rb * MAXB + b] = idx;
      }
    }
    __syncwarp();
    unsigned prev = 0;
    if (lane == 0) prev = atom_add_acq_rel(reinterpret_cast<unsigned *>(p.argmax_ticket), 1u);
    prev = __shfl_sync(0xffffffffu, prev, 0);
    if (prev == (unsigned)(p.n_rb - 1)) {
      if (lane == 0) atomicExch(p.argmax_ticket, 0);
      __syncwarp();
#pragma unroll
      for (int b = 0; b < B; ++b) {
        float bv = -INFINITY;
        int bi = 0x7fffffff;
        for (int r = lane; r < p.n_rb; r += 32)
          argmax_merge(bv, bi, __ldcg(p.cand_val + r * MAXB + b), __ldcg(p.cand_idx + r * MAXB + b));
        warp_argmax(bv, bi);
        if (lane == 0) p.next_ids[b] = (bi == 0x7fffffff) ? 0 : bi;
      }
    }
  }
}

// Epilogue warp side of one GEMV over this CTA's tile range [t0, t0 + n): takes the staged
// segments in order; a row block shared with neighbouring CTAs is combined (partials in global
// memory, atomic ticket, the last to arrive sums them in CTA order); each finished row block gets
// its epilogue and (persistent kernel) is published on the readiness counters.
// inv / inv_ready: the RMSNorm scale of this GEMV, computed once, when first needed.
template <int B, int EPI>
__device__ __forceinline__ void gemv_epilogues(const GemvParams &p, long long t0, int n, long long T, int G, int c,
                                               const SegRing &sr, int &segc, float *inv, bool &inv_ready,
                                               volatile int *abort_flag, int lane, float *rx = nullptr,
                                               uint64_t *rx_bar = nullptr) {
  int i = 0;
  while (i < n) {
    const long long t = t0 + i;
    const int rb = static_cast<int>(t / p.n_kt);
    const int kt0 = static_cast<int>(t - (long long)rb * p.n_kt);
    const int len = min(p.n_kt - kt0, n - i);
    i += len;
    const int slot = segc % sr.nslot, use = segc / sr.nslot;
    ++segc;
    consumer_wait(smem_addr(&sr.full[slot]), use & 1, abort_flag, p.err);
    unsigned long long *tr = p.trace && lane == 0 ? p.trace + (size_t)c * TRACE_SLOTS : nullptr;
    if (tr) {
      tr[TR_E_SEG] = global_ns();
      tr[TR_E_KIND] = 0;
    }
    float *red = sr.red + slot * sr.nsub * RB * MAXB;
    if (sr.nsub > 1) {
      // int4 tiles: the sub-slots' sums in sub-slot order into the first, the others back to zero
      float4 *r4 = reinterpret_cast<float4 *>(red);
      for (int e = lane; e < RB * MAXB / 4; e += 32) {
        float4 a = r4[e];
        for (int j = 1; j < sr.nsub; ++j) {
          const float4 v = r4[j * (RB * MAXB / 4) + e];
          a = make_float4(a.x + v.x, a.y + v.y, a.z + v.z, a.w + v.w);
          r4[j * (RB * MAXB / 4) + e] = make_float4(0.f, 0.f, 0.f, 0.f);
        }
        r4[e] = a;
      }
      __syncwarp();
    }
    EpiPre pre;
    epilogue_prefetch<B, EPI>(p, rb, lane, pre);
    bool do_epi = true;
    if (!(kt0 == 0 && len == p.n_kt) && rx) {
      // a cluster of p.cluster CTAs splits this row block's K range: ranks 1.. write their
      // partials into rank 0's shared memory (slot rank - 1) and arrive on its barrier; rank 0
      // adds them to its own in rank order (K order, as the ticket path sums in CTA order)
      const uint32_t rank = cluster_ctarank();
      if (rank != 0) {
        const uint32_t dst = map_to_rank(smem_addr(rx + (rank - 1) * (RB * MAXB)), 0);
        const float4 *r4 = reinterpret_cast<const float4 *>(red);
        for (int e = lane; e < RB * MAXB / 4; e += 32) st_cluster_f4(dst + e * 16, r4[e]);
        __syncwarp();
        if (lane == 0) mbar_arrive_remote(map_to_rank(smem_addr(rx_bar), 0));
        do_epi = false;
      } else {
        int ok = 1;
        if (lane == 0) {
          ok = mbar_wait_cluster(smem_addr(rx_bar), 0) ? 1 : 0;
          if (!ok) {
            *abort_flag = 1;
            atomicOr(p.err, ERR_TIMEOUT);
          }
        }
        ok = __shfl_sync(0xffffffffu, ok, 0);
        __syncwarp();
        if (ok) {
          float4 *r4 = reinterpret_cast<float4 *>(red);
          const float4 *x4 = reinterpret_cast<const float4 *>(rx);
          for (int e = lane; e < RB * MAXB / 4; e += 32) {
            float4 a = r4[e];
            for (int j = 0; j + 1 < p.cluster; ++j) {
              const float4 b = x4[j * (RB * MAXB / 4) + e];
              a = make_float4(a.x + b.x, a.y + b.y, a.z + b.z, a.w + b.w);
            }
            r4[e] = a;
          }
          __syncwarp();
        }
        do_epi = ok != 0;
      }
      if (tr) tr[TR_E_KIND] = do_epi ? 2 : 1;
    } else if (!(kt0 == 0 && len == p.n_kt)) {
      // this row block is shared with neighbouring CTAs: the ticket counts the CTAs that have
      // published their partial; the one that finds all the others there sums every partial
      const int c_lo = cta_of_tile((long long)rb * p.n_kt, T, G);
      const int c_hi = cta_of_tile((long long)(rb + 1) * p.n_kt - 1, T, G);
      const unsigned others = static_cast<unsigned>(c_hi - c_lo);
      unsigned *ticket = reinterpret_cast<unsigned *>(p.tickets + rb);
      unsigned seen = 0;
      if (lane == 0) seen = ld_acquire_gpu(ticket);
      seen = __shfl_sync(0xffffffffu, seen, 0);
      __syncwarp();
      do_epi = seen == others;
      if (!do_epi) {
        const int first_rb = static_cast<int>(t0 / p.n_kt);
        const int myslot = (rb == first_rb) ? 0 : 1;
        float4 *mine = reinterpret_cast<float4 *>(p.partial + (size_t)(c * 2 + myslot) * (RB * MAXB));
        const float4 *r4 = reinterpret_cast<const float4 *>(red);
        for (int e = lane; e < RB * MAXB / 4; e += 32) mine[e] = r4[e];
        __syncwarp();
        unsigned prev = 0;
        // release this CTA's partial; the last to arrive acquires everyone's
        if (lane == 0) prev = atom_add_acq_rel(ticket, 1u);
        prev = __shfl_sync(0xffffffffu, prev, 0);
        __syncwarp();
        do_epi = prev == others;
      }
      if (tr) {
        tr[TR_E_TICKET] = global_ns();
        tr[TR_E_KIND] = do_epi ? 2 : 1;
      }
      if (do_epi) {
        if (lane == 0) atomicExch(ticket, 0u);  // ready for the next use
        // every partial in CTA order (this CTA's own from shared memory): each lane's loads of a
        // group of four CTAs are issued together, then added
        static_assert(RB * MAXB / 4 == 64, "two float4 per lane");
        float4 sum[2] = {make_float4(0.f, 0.f, 0.f, 0.f), make_float4(0.f, 0.f, 0.f, 0.f)};
        for (int c0 = c_lo; c0 <= c_hi; c0 += 4) {
          float4 v[2][4];
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            const int cc = c0 + j;
            const int frb = static_cast<int>(((long long)cc * T / G) / p.n_kt);
            const float4 *src = reinterpret_cast<const float4 *>(p.partial + (size_t)(cc * 2 + (rb == frb ? 0 : 1)) * (RB * MAXB));
#pragma unroll
            for (int k = 0; k < 2; ++k) {
              const int e = lane + 32 * k;
              v[k][j] = cc > c_hi ? make_float4(0.f, 0.f, 0.f, 0.f)
                        : cc == c ? reinterpret_cast<const float4 *>(red)[e] : __ldcg(src + e);
            }
          }
#pragma unroll
          for (int j = 0; j < 4; ++j)
            if (c0 + j <= c_hi) {
#pragma unroll
              for (int k = 0; k < 2; ++k) {
                sum[k].x += v[k][j].x;
                sum[k].y += v[k][j].y;
                sum[k].z += v[k][j].z;
                sum[k].w += v[k][j].w;
              }
            }
        }
#pragma unroll
        for (int k = 0; k < 2; ++k) reinterpret_cast<float4 *>(red)[lane + 32 * k] = sum[k];
        __syncwarp();
        if (tr) tr[TR_E_SUMMED] = global_ns();
      }
    }
    if (do_epi) {
      if (!inv_ready) {
        // the RMSNorm scale needs every row block of h: in the persistent kernel wait for the
        // phase that produces h to complete them
        if (lane == 0 && p.norm_done) wait_counter(p.norm_done, (unsigned)p.norm_need, abort_flag, p.err);
        __syncwarp();
        norm_scale_warp<B>(p, inv, lane);
        inv_ready = true;
      }
      epilogue_warp<B, EPI>(p, rb, red, inv, pre, lane);
      __syncwarp();
      if (lane == 0) {
        // publish this row block (the __syncwarp above ordered every lane's stores before it)
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
    if (tr) tr[TR_E_DONE] = global_ns();
    __syncwarp();
    // leave the slot at zero: int4 tiles add into it
    for (int e = lane; e < RB * MAXB / 4; e += 32) reinterpret_cast<float4 *>(red)[e] = make_float4(0.f, 0.f, 0.f, 0.f);
    __syncwarp();
    if (lane == 0) mbar_arrive(smem_addr(&sr.empty[slot]));
  }
}

template <int B>
__device__ __forceinline__ void gemv_epilogues_any(int epi, const GemvParams &p, long long t0, int n, long long T,
                                                   int G, int c, const SegRing &sr, int &segc, float *inv,
                                                   bool &inv_ready, volatile int *abort_flag, int lane) {
  switch (epi) {
    case EPI_QKV: gemv_epilogues<B, EPI_QKV>(p, t0, n, T, G, c, sr, segc, inv, inv_ready, abort_flag, lane); break;
    case EPI_RESID: gemv_epilogues<B, EPI_RESID>(p, t0, n, T, G, c, sr, segc, inv, inv_ready, abort_flag, lane); break;
    case EPI_SWIGLU:
      gemv_epilogues<B, EPI_SWIGLU>(p, t0, n, T, G, c, sr, segc, inv, inv_ready, abort_flag, lane);
      break;
    case EPI_ARGMAX:
      gemv_epilogues<B, EPI_ARGMAX>(p, t0, n, T, G, c, sr, segc, inv, inv_ready, abort_flag, lane);
      break;
    default: gemv_epilogues<B, EPI_STORE>(p, t0, n, T, G, c, sr, segc, inv, inv_ready, abort_flag, lane); break;
  }
}

}  // namespace kfl
