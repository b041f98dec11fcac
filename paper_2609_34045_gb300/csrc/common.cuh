// Internal definitions shared by the stage-decode kernels and the runtime (sm_103a only).
#pragma once

#include <cuda.h>  // CUtensorMap (the type only; maps are encoded through the runtime's entry point)
#include <cuda_runtime.h>
#include <stdint.h>

#if defined(__CUDA_ARCH__) && (__CUDA_ARCH__ < 1000)
#error "this library targets sm_103a (Blackwell) only"
#endif

namespace kfl {

// ---- tiling of the weight-streaming GEMV ------------------------------------------------
// A matrix [N][K] is stored as tiles [N/RB][K/KT][RB][KT] (zero-padded), each tile one
// contiguous 16 KiB chunk of HBM, so a CTA streams its share of the matrix with 1-D bulk
// copies and every warp reads a whole tile row from shared memory without bank conflicts.
constexpr int RB = 64;            // rows per row block (and per tile)
constexpr int KT = 128;           // K per bf16 tile
constexpr int TILE_BYTES = RB * KT * 2;
constexpr int MAXB = 4;           // users per step
constexpr int CONSUMER_WARPS = 8;
constexpr int GEMV_THREADS = (CONSUMER_WARPS + 2) * 32;  // consumers, producer, epilogue warp
constexpr int MAX_STAGES = 12;
constexpr int MAX_CLUSTER = 8;  // CTAs of a split-K GEMV cluster (the portable cluster size)
constexpr int MAX_CLUSTER_ATT = 16;  // CTAs of an attention cluster (non-portable above 8)

// int4 group-64 tiles: [N/RB][K/KT4], each 64 x 256 codes (8 KiB, in the order of the
// tensor-core MMA fragments, see repack_int4_kernel) then RB x KT4/64 bf16 scales (in the order of
// tile4_scale_index)
constexpr int KT4 = 256;
constexpr int TILE4_CODE_BYTES = RB * KT4 / 2;     // 8 KiB
constexpr int TILE4_SCALE_BYTES = RB * (KT4 / 64) * 2;  // 512 B
constexpr int TILE4_BYTES = TILE4_CODE_BYTES + TILE4_SCALE_BYTES;

// Position (in bf16 units, after the codes) of the scale of row r (0..63) and weight group g4
// (0..3) of an int4 tile: grouped by the consumer warp that reads them (weight group g4), then by
// the lane's row gid = r % 8, so that one 16-byte load gives a lane the scales of rows gid and
// gid + 8 of all four row groups r / 16 of its group.
__host__ __device__ constexpr int tile4_scale_index(int r, int g4) {
  return ((g4 * 8 + (r & 7)) * 4 + (r >> 4)) * 2 + ((r >> 3) & 1);
}
// A weight-ring depth usable by this format: int4 rings have an even number of stages (each stage
// then belongs to one of the two consumer teams, gemv_consume_int4).
__host__ __device__ constexpr int ring_depth(int fmt, int stages) { return fmt == 0 ? stages : (stages & ~1); }
__host__ __device__ constexpr int tile_k(int fmt) { return fmt == 0 ? KT : KT4; }
__host__ __device__ constexpr int tile_bytes(int fmt) { return fmt == 0 ? TILE_BYTES : TILE4_BYTES; }
// A ring stage holds one weight tile and the activations of its K range: bf16 tiles, the B
// users' fp32 values; int4 tiles, one K tile's block of its Act16 input (below): the chunk
// constants, then fp16 source rows at a padded stride.
constexpr int XCHUNK = 32;                          // elements per scale chunk of an int4 input
constexpr int X16_SRC_BYTES = KT4 * 2;              // 512
// 576: the sources start on different halves of the banks, so that the 16-byte B-fragment loads of
// one quarter warp (two sources) fall in distinct banks
constexpr int X16_SRC_STRIDE = X16_SRC_BYTES + 64;
constexpr int XC_GROUP_BYTES = 192;                 // per weight group (two chunks): 3 x [4 lane quads][4]
constexpr int XC_TILE_BYTES = (KT4 / (2 * XCHUNK)) * XC_GROUP_BYTES;  // 768
// Bytes of one K tile's block of an Act16 (rest: with the rests' rows), and the part of it a
// GEMV at batch B copies into a ring stage: the constants and the rounded parts of users
// 0..B-1, or (xsplit) all MAXB rounded parts and the rests of users 0..B-1.
__host__ __device__ constexpr int act16_tile_bytes(int rest) {
  return XC_TILE_BYTES + (rest ? 2 : 1) * MAXB * X16_SRC_STRIDE;
}
__host__ __device__ constexpr int act16_copy_bytes(int batch, int xsplit) {
  return XC_TILE_BYTES + (xsplit ? MAXB + batch : batch) * X16_SRC_STRIDE;
}
__host__ __device__ constexpr int stage_bytes(int batch, int fmt) {
  return fmt == 0 ? (TILE_BYTES + batch * KT * 4 + 127) / 128 * 128
                  : (TILE4_BYTES + act16_copy_bytes(batch, 1) + 127) / 128 * 128;
}
constexpr int STAGE_BYTES_MAX = stage_bytes(MAXB, 0);

// A GEMV input of an int4 stage, in the form the tensor-core tile loop reads (tile_compute_int4).
// Per user b: x divided by a power of two per XCHUNK elements (m, the multiplier that undoes it,
// brings the chunk's largest value into [2^14, 2^15)) and rounded to fp16; in each 16-element
// block, elements 8..15 are also divided by 16 (the decoder makes their weights 16 x larger);
// each 32-element chunk is stored in the order of the MMA's B fragments of its two 16-element K
// steps (act16_index).  The Q/K/V projection's input also keeps what rounding to fp16 left
// over (the rest), in fp16.
// Layout, tile-major so that a ring stage's activations are one contiguous copy: per K tile of
// KT4 elements a block of act16_tile_bytes(rest) bytes, holding
//   [0, XC_TILE_BYTES): the chunk constants, per weight group of two chunks (a, b) three blocks
//     [t][0..3] for MMA columns 2t, 2t+1: chunk a's seed, chunk b's seed, then the multipliers
//     (m_a(2t), m_a(2t+1), m_b(2t), m_b(2t+1)); a seed is minus the columns' offset sums twice over
//     (the MMA's accumulator quad of rows gid and gid + 8); column u < 4 is user u's rounded part and
//     column u + 4 its rest, and a column's offset sum is the sum over the chunk of its fp16
//     values times 1032 (block elements 0..7) or 1152 (8..15): what the decoder's offsets add
//     to the MMA's product;
//   then source rows of X16_SRC_STRIDE bytes: rows 0..MAXB-1 the users' rounded parts, rows
//     MAXB..2 MAXB-1 their rests (rest only).
struct Act16 {
  uint8_t *base;  // NULL: the stage has no int4 input of this kind
  int ld;         // elements per user row, a multiple of KT4
  int rest;       // 1: the rests are stored
};

// Position of element k of a user's row in Act16 order: within a 32-element chunk, lane quad t
// of a warp reads the 16 bytes at 16 t: elements 2t, 2t+1 (B fragment register b0) and 2t+8,
// 2t+9 (b1) of the chunk's first 16-element block, then the same of its second block.
__host__ __device__ constexpr int act16_index(int k) {
  return (k & ~31) + ((k & 7) >> 1) * 8 + ((k >> 4) & 1) * 4 + ((k & 15) < 8 ? 0 : 2) + (k & 1);
}

__host__ __device__ inline uint8_t *act16_tile(const Act16 &a, int kt) {
  return a.base + (size_t)kt * act16_tile_bytes(a.rest);
}
// Element k of source row r (r < MAXB: user r's rounded part; MAXB + u: user u's rest).
__host__ __device__ inline uint16_t *act16_elem(const Act16 &a, int r, int k) {
  return reinterpret_cast<uint16_t *>(act16_tile(a, k / KT4) + XC_TILE_BYTES + r * X16_SRC_STRIDE) +
         act16_index(k % KT4);
}
// The constants block of the weight group holding chunk ch.
__host__ __device__ inline float *act16_consts(const Act16 &a, int ch) {
  return reinterpret_cast<float *>(act16_tile(a, ch / (KT4 / XCHUNK)) + ((ch % (KT4 / XCHUNK)) >> 1) * XC_GROUP_BYTES);
}

// ---- device error word bits ---------------------------------------------------------------
constexpr unsigned ERR_POSITION = 1u;
constexpr unsigned ERR_TOKEN = 2u;
constexpr unsigned ERR_TIMEOUT = 4u;
constexpr unsigned ERR_F16_RANGE = 8u;  // an int4 prefill activation beyond the fp16 range

// bounded waits: spins before backing off, total polls before giving up (~1-2 s)
constexpr uint32_t WAIT_FAST_SPINS = 1024;
constexpr uint32_t WAIT_LIMIT = 1u << 24;

enum Epilogue : int {
  EPI_STORE = 0,   // out[b][n] = y
  EPI_QKV = 1,     // RoPE on q/k row pairs, q to fp32, k/v appended to the bf16 cache
  EPI_RESID = 2,   // h[b][n] += y; xn = h * g_next; per-row-block sum of squares
  EPI_SWIGLU = 3,  // rows (2j, 2j+1) = (gate_j, up_j) -> a[b][j] = silu(gate) * up
  EPI_ARGMAX = 4,  // greedy argmax over rows, lowest index on ties
};

struct GemvParams {
  const uint8_t *w;  // tiled weights
  int fmt;           // 0 bf16, 1 int4
  int n_rows;        // valid rows N
  int n_rb, n_kt;    // row blocks, K tiles
  int tile_bytes;
  int kt;            // K per tile
  const float *x;    // activations [batch][ldx]
  int ldx;
  int batch;
  int stages;
  // RMSNorm folded into the GEMV: y = inv_rms[b] * (W . x) with x = h * g precomputed by the
  // producer of h; inv_rms from the per-row-block sums of squares of h
  const float *sumsq;  // [n_parts][MAXB] or NULL
  int n_parts;
  int d_norm;
  float eps;
  // EPI_STORE / EPI_SWIGLU
  float *out;
  int ldo;
  // EPI_RESID
  float *h;
  float *xn;
  const float *g_next;
  float *sumsq_out;
  float *capture;  // [MAXB? no: batch rows][ldh] per-layer hidden, or NULL
  int ldh;
  // EPI_QKV
  float *q;
  uint16_t *kcache, *vcache;  // this layer's [max_batch][Hkv][max_ctx][hd]
  const int *positions;       // [batch]; never written while a step runs
  const int *slots;           // [batch]: the KV-cache user slot of each batch row
  const float *rope_cos, *rope_sin;  // [max_ctx][hd/2], or [batch][hd/2] when rope_per_user
  int rope_per_user;
  int n_q_rows, n_kv_rows, head_dim, max_ctx, n_kv_heads;
  // stages with QK-norm: the projection (rows in GEMV order, after the RMSNorm scale) goes to
  // qk_raw[b * ld_raw + n] instead, and qknorm_rope_kernel normalises, rotates and appends it
  float *qk_raw;
  int ld_raw;
  // int4 weights: the GEMV multiplies fp16 activations on the tensor cores
  Act16 xin;          // this GEMV's input (int4 stages; x and ldx are then unused)
  Act16 xout;         // RESID / SWIGLU: the output in the same form (int4 stages; base NULL else)
  int xsplit;         // the input's rests are multiplied too (Q/K/V projection)
  // one kernel per phase, cluster > 1: launched as clusters of `cluster` CTAs (at most
  // MAX_CLUSTER), grid cluster x n_rb, each CTA 1/cluster of the K range of one row block; ranks
  // 1.. hand their partials to rank 0 through distributed shared memory instead of global
  // memory and a ticket
  int cluster;
  // EPI_ARGMAX
  float *cand_val;
  int *cand_idx;
  int *argmax_ticket;
  int *next_ids;
  // stream-K bookkeeping
  float *partial;  // [grid][2][RB][MAXB]
  int *tickets;    // [n_rb], zero between launches
  unsigned *err;
  // dataflow (persistent stage kernel only; all NULL / 0 otherwise)
  int in_kind;                // 0 inputs complete at launch, 1 per-chunk counters, 2 per-KV-head counters
  const unsigned *in_ready;   // counters of the producing phase
  int in_len;                 // kind 1: length of the input vector (elements)
  int in_unit;                // kind 1: input elements one producing row block completes
  int in_group;               // kind 2: query heads per KV head
  int in_head_dim;            // kind 2
  int in_need;                // kind 2: completions per KV head (the batch)
  const unsigned *norm_done;  // row blocks of h completed by the phase producing h (NULL: ready)
  int norm_need;
  unsigned *out_ready;        // per consumer chunk (RESID, SWIGLU) or per KV head (QKV)
  int out_unit;               // output elements per row block (RESID 64, SWIGLU 32)
  int out_kt;                 // the consumer's tile K
  unsigned *out_done;         // row blocks completed
  unsigned long long *trace;  // one-kernel-per-phase mode: this launch's [grid][TRACE_SLOTS]
                              // %globaltimer stamps, or NULL
};

struct AttnParams {
  const float *q;            // [batch][Hq*hd] (RoPE applied)
  const uint16_t *kcache;    // this layer's [max_batch][Hkv][max_ctx][hd]
  const uint16_t *vcache;
  const int *positions;
  const int *slots;          // [batch]: the KV-cache user slot of each batch row
  float *o;                  // [batch][ldo]
  int ldo;
  Act16 o16;                 // int4 stages: o also in the O projection's input form (base NULL else)
  float *partial;            // [batch][Hkv][n_chunks][G][hd + 2]
  int *tickets;              // [batch][Hkv]
  int batch, n_heads, n_kv_heads, max_ctx;
  // positions per unit: set on the device at each launch from the step's positions
  // (attn_chunk_size), so that a step has about target_units units; the partial buffer holds
  // n_chunks (= max_ctx / 64, rounded up) chunks per (user, KV head)
  int chunk, n_chunks, target_units;
  // one kernel per phase: > 0 runs attn_cluster_kernel, one thread-block cluster of `cluster`
  // CTAs per (user, KV head) that split its positions and merge through distributed shared
  // memory (partial, tickets, chunk and target_units are then unused), each with a ring of
  // `stages` sub-tiles (three: two CTAs fit an SM; two: three)
  int cluster;
  int stages;
  int launch_at;             // the next kernel may launch: 0 at once, 1 when every sub-tile is issued, 2 after the loop
  float scale_log2;          // log2(e) / sqrt(hd)
  unsigned *err;
  // dataflow (persistent stage kernel only)
  const unsigned *in_ready;  // per KV head: Q/K/V row blocks completed
  int in_need;
  unsigned *out_ready;       // per KV head: (user, KV head) outputs completed
  unsigned long long *trace;  // one-kernel-per-phase mode: this launch's [grid][TRACE_SLOTS], or NULL
  int trace_grid;
};

// QK-norm (per-head RMSNorm of q and k over head_dim, then RoPE, then the KV append) of the
// Q/K/V projection of stages with qk_norm, between the projection and attention.
struct QkNormParams {
  const float *raw;                  // [batch][ld_raw]: q, k, v rows in GEMV order (RoPE pairs adjacent)
  int ld_raw;
  const float *g_q, *g_k;            // [hd] gains
  float *q;                          // [batch][Hq * hd]: normalised, rotated q
  uint16_t *kcache, *vcache;         // this layer's [max_batch][Hkv][max_ctx][hd]
  const int *positions, *slots;      // [batch] (a position of -1: the row is invalid)
  const float *rope_cos, *rope_sin;  // [max_ctx][hd/2]
  int batch, n_heads, n_kv_heads, head_dim, max_ctx;
  float eps;
};

// One phase of a step: a GEMV (with its epilogue) or an attention pass (preceded, in stages with
// QK-norm, by the QK-norm kernel: qn.raw non-NULL).
enum PhaseKind : int { PH_GEMV = 0, PH_ATTN = 1 };

struct Phase {
  int kind;
  int epi;
  GemvParams g;
  AttnParams a;
  QkNormParams qn;
};

struct StageKernelParams {
  const Phase *phases;  // device array
  int n_phases;
  int stages;      // ring stages
  int head_dim;
  int attn_bytes;  // shared memory of the attention unit
  unsigned *bar;   // [1] is the abort flag, zeroed by the stage input kernel
  int *abort_flag; // set when any wait gives up; zeroed by the stage input kernel
  unsigned *err;
  unsigned long long *trace;  // [n_phases][grid][TRACE_SLOTS] globaltimer stamps, or NULL
  const int *positions;       // [batch] (static during the step)
  const float *rope_cos, *rope_sin;  // [max_ctx][hd/2]
  int max_ctx;
  int l2_ahead;               // weight tiles prefetched into L2 ahead of the ring, per CTA
};

// phase trace slots (ns, %globaltimer)
constexpr int TRACE_SLOTS = 12;
constexpr int TR_CONS_ENTER = 0;   // consumers reach the phase
constexpr int TR_CONS_GO = 1;      // consumers start its work
constexpr int TR_CONS_DONE = 2;    // consumers finished the phase
constexpr int TR_X_GO = 3;         // activation producer issued the phase's first chunk
constexpr int TR_X_LAST = 4;       // activation producer issued the phase's last chunk
constexpr int TR_W_FIRST = 5;      // weight producer issued the phase's first tile
constexpr int TR_W_LAST = 6;       // weight producer issued the phase's last tile
// GEMV epilogue warp, last row-block segment of the CTA (one kernel per phase)
constexpr int TR_E_SEG = 7;        // the consumers' sums of the segment are staged
constexpr int TR_E_TICKET = 8;     // shared row block: this CTA's partial published, ticket taken
constexpr int TR_E_SUMMED = 9;     // last arriver: every partial of the row block summed
constexpr int TR_E_DONE = 10;      // fused epilogue of the segment done
constexpr int TR_E_KIND = 11;      // 0 row block of this CTA alone, 1 shared (not last), 2 shared, last

__device__ __forceinline__ unsigned long long global_ns() {
  unsigned long long t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

// ---- PTX helpers --------------------------------------------------------------------------
__device__ __forceinline__ uint32_t smem_addr(const void *p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}

__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

// ---- thread-block clusters (distributed shared memory) ----
__device__ __forceinline__ uint32_t cluster_ctarank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
// Every thread of every CTA of the cluster (shared memory written before is visible after).
__device__ __forceinline__ void cluster_sync_all() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}
// The address of the same shared-memory location in cluster CTA `rank`.
__device__ __forceinline__ uint32_t map_to_rank(uint32_t addr, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(addr), "r"(rank));
  return r;
}
__device__ __forceinline__ void st_cluster_f4(uint32_t addr, float4 v) {
  asm volatile("st.shared::cluster.v4.f32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "f"(v.x), "f"(v.y), "f"(v.z),
               "f"(v.w)
               : "memory");
}
// Arrive (release, cluster scope) on an mbarrier of another CTA of the cluster.
__device__ __forceinline__ void mbar_arrive_remote(uint32_t cluster_addr) {
  asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(cluster_addr) : "memory");
}
// Bounded wait (acquire, cluster scope) on a local mbarrier phase; false after WAIT_LIMIT polls.
__device__ __forceinline__ bool mbar_wait_cluster(uint32_t bar, uint32_t parity) {
  for (uint32_t i = 0; i < WAIT_LIMIT; ++i) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    if (ok) return true;
    if (i >= WAIT_FAST_SPINS) __nanosleep(64);
  }
  return false;
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes)
               : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}

// Non-blocking test of an mbarrier phase.
__device__ __forceinline__ bool mbar_test_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}

__device__ __forceinline__ int ld_acquire_cta_shared(const volatile int *p) {
  int v;
  asm volatile("ld.acquire.cta.shared.b32 %0, [%1];" : "=r"(v) : "r"(smem_addr((const void *)p)) : "memory");
  return v;
}

__device__ __forceinline__ void st_release_cta_shared(volatile int *p, int v) {
  asm volatile("st.release.cta.shared.b32 [%0], %1;" ::"r"(smem_addr((const void *)p)), "r"(v) : "memory");
}

// Bounded wait on an mbarrier phase; false after WAIT_LIMIT polls.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity) {
  for (uint32_t i = 0; i < WAIT_LIMIT; ++i) {
    if (mbar_try_wait(bar, parity)) return true;
    if (i >= WAIT_FAST_SPINS) __nanosleep(64);
  }
  return false;
}

__device__ __forceinline__ uint64_t policy_evict_first() {
  uint64_t pol;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol));
  return pol;
}

__device__ __forceinline__ uint64_t policy_evict_last() {
  uint64_t pol;
  asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(pol));
  return pol;
}

// 1-D bulk copy global -> shared (TMA), completion counted in bytes on `bar`.
// dst, src 16-byte aligned; bytes a multiple of 16.
__device__ __forceinline__ void bulk_g2s(uint32_t dst, const void *src, uint32_t bytes, uint32_t bar,
                                         uint64_t policy) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint"
      " [%0], [%1], %2, [%3], %4;" ::"r"(dst),
      "l"(src), "r"(bytes), "r"(bar), "l"(policy)
      : "memory");
}

// 1-D bulk prefetch global -> L2 (no completion tracking); 16-byte aligned, size multiple of 16.
__device__ __forceinline__ void bulk_prefetch_l2(const void *src, uint32_t bytes, uint64_t policy) {
  asm volatile("cp.async.bulk.prefetch.L2.global.L2::cache_hint [%0], %1, %2;" ::"l"(src), "r"(bytes), "l"(policy)
               : "memory");
}

__device__ __forceinline__ uint64_t policy_evict_normal() {
  uint64_t pol;
  asm volatile("createpolicy.fractional.L2::evict_normal.b64 %0, 1.0;" : "=l"(pol));
  return pol;
}

// Programmatic dependent launch (PDL)
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_launch_dependents() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

__device__ __forceinline__ void named_bar_sync(int id, int n) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(n) : "memory");
}

__device__ __forceinline__ float bf16_lo(uint32_t u) { return __uint_as_float(u << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t u) { return __uint_as_float(u & 0xFFFF0000u); }
__device__ __forceinline__ float bf16_to_f32(uint16_t b) { return __uint_as_float(uint32_t(b) << 16); }

// fp32 -> bf16, round to nearest even (NaN -> quiet NaN)
__device__ __forceinline__ uint16_t f32_to_bf16_rne(float f) {
  uint32_t u = __float_as_uint(f);
  if ((u & 0x7FFFFFFFu) > 0x7F800000u) return 0x7FC0;
  u += 0x7FFFu + ((u >> 16) & 1u);
  return static_cast<uint16_t>(u >> 16);
}

__device__ __forceinline__ float ld_cg(const float *p) { return __ldcg(p); }

// gpu-scope atomics with release / acquire-release semantics: the writes a CTA made before a
// bar.sync become visible with the atomic, without a separate membar
__device__ __forceinline__ unsigned atom_add_acq_rel(unsigned *p, unsigned v) {
  unsigned old;
  asm volatile("atom.acq_rel.gpu.global.add.u32 %0, [%1], %2;" : "=r"(old) : "l"(p), "r"(v) : "memory");
  return old;
}
__device__ __forceinline__ void red_add_release(unsigned *p, unsigned v) {
  asm volatile("red.release.gpu.global.add.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}
// The power of two 2^e that a chunk of values with largest magnitude m is divided by so that it
// fits fp16 with its largest value in [2^14, 2^15) (exact: a power of two); *inv = 2^-e.  A chunk
// of zeros gets 1.
__device__ __forceinline__ float xchunk_scale(float m, float *inv) {
  int e = 0;
  if (m > 0.f) e = static_cast<int>((__float_as_uint(m) >> 23) & 0xFF) - 127 - 14;
  e = max(-100, min(100, e));
  *inv = __uint_as_float(static_cast<uint32_t>(127 - e) << 23);
  return __uint_as_float(static_cast<uint32_t>(127 + e) << 23);
}

__device__ __forceinline__ unsigned ld_acquire_gpu(const unsigned *p) {
  unsigned v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

__device__ __forceinline__ uint16_t f32_to_f16_rn(float x) {
  uint16_t h;
  asm("cvt.rn.f16.f32 %0, %1;" : "=h"(h) : "f"(x));
  return h;
}
__device__ __forceinline__ float f16_to_f32(uint16_t h) {
  float f;
  asm("cvt.f32.f16 %0, %1;" : "=f"(f) : "h"(h));
  return f;
}

// Chunk ch's constants for user b (column b: rounded part, column b + 4: rest).
__device__ __forceinline__ void act16_put_consts(const Act16 &a, int b, int ch, float m, float off_hi, float off_lo) {
  float *g = act16_consts(a, ch);
  float *seed = g + (ch & 1) * 16, *mult = g + 32 + (ch & 1) * 2;
  const int t = b >> 1, j = b & 1;
  seed[t * 4 + j] = seed[t * 4 + 2 + j] = -off_hi;
  seed[(t + 2) * 4 + j] = seed[(t + 2) * 4 + 2 + j] = -off_lo;
  mult[t * 4 + j] = mult[(t + 2) * 4 + j] = m;
}

// Chunk ch of user b of an Act16, one element per lane (x = 0 past the vector's end); the whole
// warp calls it.
__device__ __forceinline__ void act16_put_warp(const Act16 &a, int b, int ch, float x, int lane) {
  float mx = fabsf(x);
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, off));
  float iv;
  const float m = xchunk_scale(mx, &iv);
  const bool upper = (lane & 15) >= 8;
  const float y = x * iv * (upper ? 0.0625f : 1.0f);
  const float wgt = upper ? 1152.0f : 1032.0f;
  const uint16_t h = f32_to_f16_rn(y);
  const float yh = f16_to_f32(h);
  const int k = ch * XCHUNK + lane;
  *act16_elem(a, b, k) = h;
  float oh = yh * wgt, ol = 0.f;
  if (a.rest) {
    const uint16_t l = f32_to_f16_rn(y - yh);
    *act16_elem(a, MAXB + b, k) = l;
    ol = f16_to_f32(l) * wgt;
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    oh += __shfl_xor_sync(0xffffffffu, oh, off);
    ol += __shfl_xor_sync(0xffffffffu, ol, off);
  }
  if (lane == 0) act16_put_consts(a, b, ch, m, oh, ol);
}

// The same, with the chunk held by 8 consecutive lanes, 4 consecutive elements each (lane & 7
// holds elements 4 (lane & 7) .. + 3); the whole warp calls it, `write` selects the lanes that
// store.
__device__ __forceinline__ void act16_put_quad(const Act16 &a, int b, int ch, float4 v, int lane, bool write) {
  float mx = fmaxf(fmaxf(fabsf(v.x), fabsf(v.y)), fmaxf(fabsf(v.z), fabsf(v.w)));
#pragma unroll
  for (int off = 4; off > 0; off >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, off));
  float iv;
  const float m = xchunk_scale(mx, &iv);
  const int sub = lane & 7;
  const bool upper = (sub & 2) != 0;  // elements 4 sub .. + 3 lie in one half of a 16-block
  const float sc = iv * (upper ? 0.0625f : 1.0f), wgt = upper ? 1152.0f : 1032.0f;
  const float y[4] = {v.x * sc, v.y * sc, v.z * sc, v.w * sc};
  uint16_t h[4], l[4];
  float oh = 0.f, ol = 0.f;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    h[i] = f32_to_f16_rn(y[i]);
    const float yh = f16_to_f32(h[i]);
    l[i] = f32_to_f16_rn(y[i] - yh);
    oh += yh * wgt;
    ol += f16_to_f32(l[i]) * wgt;
  }
  if (!a.rest) ol = 0.f;
#pragma unroll
  for (int off = 4; off > 0; off >>= 1) {
    oh += __shfl_xor_sync(0xffffffffu, oh, off);
    ol += __shfl_xor_sync(0xffffffffu, ol, off);
  }
  if (write) {
    const int k0 = ch * XCHUNK + 4 * sub;
    *reinterpret_cast<uint32_t *>(act16_elem(a, b, k0)) = (uint32_t)h[0] | ((uint32_t)h[1] << 16);
    *reinterpret_cast<uint32_t *>(act16_elem(a, b, k0 + 2)) = (uint32_t)h[2] | ((uint32_t)h[3] << 16);
    if (a.rest) {
      *reinterpret_cast<uint32_t *>(act16_elem(a, MAXB + b, k0)) = (uint32_t)l[0] | ((uint32_t)l[1] << 16);
      *reinterpret_cast<uint32_t *>(act16_elem(a, MAXB + b, k0 + 2)) = (uint32_t)l[2] | ((uint32_t)l[3] << 16);
    }
    if (sub == 0) act16_put_consts(a, b, ch, m, oh, ol);
  }
}

}  // namespace kfl

// Kernel launchers (defined in the .cu files; used by the runtime).
namespace kfl {
cudaError_t prepare_gemv();
cudaError_t prepare_attention();
cudaError_t launch_gemv(const GemvParams &p, int epi, int grid, cudaStream_t s, bool pdl);
int gemv_max_stages(int batch, int fmt, int smem_optin);  // valid after prepare_gemv
int gemv_stages_for(int batch, int fmt, int cluster, int per_sm);  // valid after prepare_gemv
cudaError_t launch_attention(const AttnParams &p, int head_dim, cudaStream_t s, bool pdl);
cudaError_t launch_qknorm(const QkNormParams &p, cudaStream_t s, bool pdl);
cudaError_t prepare_attention_cluster();
constexpr int ATT_RING_MAX = 3;  // attention clusters: the deepest ring (sub-tiles); two CTAs fit an SM
int attention_cluster_size(int head_dim, int want, int stages);  // valid after prepare_attention_cluster
cudaError_t launch_attention_cluster(const AttnParams &p, const CUtensorMap &kmap, const CUtensorMap &vmap,
                                     int head_dim, cudaStream_t s, bool pdl);
int encode_kv_map(CUtensorMap *map, const uint16_t *base, int head_dim, long long rows);
cudaError_t launch_stage_input(const int *ids, const float *hidden_in, const int *positions_in,
                               int batch, const uint16_t *embed, int vocab, int d, int ldh,
                               const float *g_next, float *h, float *xn, float *sumsq,
                               int *positions, int max_ctx, unsigned *err, unsigned *bar, Act16 xn16,
                               const int *users, int user_all, int max_batch, int *slots,
                               cudaStream_t s);
size_t stage_kernel_smem(int stages, int head_dim, int batch, int fmt);
int stage_kernel_attn_bytes(int head_dim);
cudaError_t prepare_stage_kernel(size_t smem);
cudaError_t launch_stage_kernel(const StageKernelParams &kp, int batch, int fmt, int grid, size_t smem,
                                cudaStream_t s);
cudaError_t launch_stage_output(const float *h, int ldh, int d, int batch, float *hidden_out,
                                const int *next_in, int *next_ids, cudaStream_t s, bool pdl);
cudaError_t launch_repack_bf16(const uint16_t *src, int n_src_rows, int k, const int *row_map,
                               int n_rows_out, int n_rb, int n_kt, uint8_t *dst, cudaStream_t s);
cudaError_t launch_repack_int4(const uint32_t *words, const uint16_t *scales, int n_src_rows, int k,
                               const int *row_map, int n_rows_out, int n_rb, int n_kt, uint8_t *dst,
                               cudaStream_t s);
cudaError_t launch_bf16_to_f32(const uint16_t *src, float *dst, int n, cudaStream_t s);
}  // namespace kfl
