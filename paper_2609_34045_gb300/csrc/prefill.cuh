// Internal definitions of the dense prompt prefill (sm_103a only): a tcgen05 GEMM over the
// prompt's tokens with fused epilogues, causal attention over the cache, row RMSNorm.
#pragma once

#include <cuda.h>  // CUtensorMap (the type only; maps are encoded through the runtime's entry point)

#include "common.cuh"

namespace kfl {

// ---- the prefill GEMM: Y[T][N] = X[T][K] W[N][K]^T ------------------------------------------
// X is fp32 in meaning and given as two bf16 terms, X = Xhi + Xlo (Xhi = bf16(X), Xlo =
// bf16(X - Xhi), about 2^-16 relative error left), so that the products keep the accuracy of the
// decode path's fp32 activations; W is bf16 as stored (int4 stages: fp16 tiles dequantized from
// the int4 ones, with fp16 terms of X).  An output tile is PG_M tokens x PG_N weight rows,
// computed with tcgen05.mma (M = PG_M, N = PG_N, K = 16 per instruction; each K slice once with
// Xhi and once with Xlo against the same W slice), the fp32 accumulator in tensor memory: by a
// persistent CTA per SM with two accumulators (prefill_gemm_persistent), or, split over K, by a
// cluster of 2, 4 or 8 CTAs that reduce through distributed shared memory (prefill_gemm_kernel).  Operands reach shared memory by TMA with the 128-byte swizzle, PG_K = 64 bf16 (one
// swizzle row) per pipeline stage: Xhi and Xlo through 2-D maps of the activation rows, W through
// a 4-D map of the decode path's weight tiles [N/RB][K/KT][RB][KT] (one box = PG_N / RB row
// blocks x 64 columns of one K tile), so the prefill streams the weights from where the decode
// step reads them.
constexpr int PG_M = 128;
constexpr int PG_N = 256;
constexpr int PG_K = 64;
constexpr int PG_STAGES = 3;
constexpr int PG_A_BYTES = PG_M * PG_K * 2;  // 16 KiB per term
constexpr int PG_B_BYTES = PG_N * PG_K * 2;  // 32 KiB
constexpr int PG_THREADS = 128;              // split kernel: TMA (thread 0), MMA (thread 32); all: epilogue
constexpr int PG_TMEM_COLS = PG_N;           // split kernel: fp32 accumulator columns
constexpr size_t PG_SMEM = (size_t)PG_STAGES * (2 * PG_A_BYTES + PG_B_BYTES) + 1024;  // + alignment slack

enum PrefillEpi : int {
  PE_STORE = 0,   // out[t][n] = y
  PE_RESID = 1,   // out[t][n] += y (the residual stream)
  PE_SWIGLU = 2,  // columns (2j, 2j+1) = (gate j, up j): silu(g) u as hi/lo terms -> out16, out16lo
  PE_QKV = 3,     // Q/K/V rows in the decode path's order: RoPE, q -> out16, k and v -> KV cache
  PE_ARGMAX = 4,  // per (token, column tile): the largest y and its lowest index
};

struct PrefillEpiParams {
  int T, N;                // valid tokens and columns
  int f16;                 // operands are fp16 (int4 stages: weights dequantized to fp16), else bf16
  float *out;              // PE_STORE / PE_RESID: fp32 [T][ldo]
  int ldo;
  uint16_t *out16;         // PE_SWIGLU: hi term, bf16 [T][ldo16] (N / 2 columns); PE_QKV: q, bf16 [T][ldo16]
  uint16_t *out16lo;       // PE_SWIGLU: lo term, same layout
  int ldo16;
  // PE_QKV: rows [0, qdim) q, [qdim, qdim + kvdim) k (pairs (i, i + hd/2) adjacent per head, as
  // the weights were loaded), then v in natural order; K/V stored at the token's position of
  // KV slot `slot` of this layer's caches [max_batch][Hkv][max_ctx][hd]
  uint16_t *kcache, *vcache;
  const int *positions;    // [T], -1 for a refused token (nothing of it is stored)
  int slot, hd, hkv, qdim, kvdim, max_ctx;
  const float *rope_cos, *rope_sin;  // [max_ctx][hd / 2]
  // PE_ARGMAX: [T][n_tiles] partial maxima and their indices
  float *amax;
  int *aidx;
  int n_tiles;
  // split-K: 1, 2, 4 or 8 CTAs per output tile, launched as a cluster that reduces through
  // distributed shared memory (PE_ARGMAX: 1)
  int splits;
  unsigned *err;           // ERR_TIMEOUT if a pipeline wait gave up; ERR_F16_RANGE (PE_SWIGLU, fp16
                           // terms) if a value is beyond the fp16 range
};

struct PrefillAttnParams {
  const uint16_t *q;       // [T][ldq] bf16, RoPE applied, heads in natural order
  int ldq;
  uint16_t *o, *o_lo;      // [T][ldo]: the output as hi and lo terms (fp16 if f16, else bf16)
  int ldo, f16;
  const uint16_t *kcache, *vcache;  // this layer's [max_batch][Hkv][max_ctx][hd]
  const int *positions;    // [T], -1: refused (output 0)
  int slot, T, n_heads, n_kv_heads, max_ctx;
  float scale_log2;        // log2(e) / sqrt(hd)
  unsigned *err;           // ERR_F16_RANGE if an fp16 output term cannot hold its value
};

// Host side (prefill.cu).
int encode_act_map(CUtensorMap *map, const uint16_t *base, int K, int rows, int ld);
int encode_tiles_map(CUtensorMap *map, const uint8_t *tiles, int n_kt, int n_rb);
// Splits of K (1, 2, 4 or 8) for a GEMM of T tokens x N rows (n_kt K tiles) on n_sm SMs: the
// count that minimises an estimate of waves x work per CTA.
int prefill_splits(int T, int N, int n_kt, int n_sm);
cudaError_t launch_prefill_gemm(int mode, const CUtensorMap &a_hi, const CUtensorMap &a_lo, const CUtensorMap &b,
                                int n_kt, const PrefillEpiParams &ep, cudaStream_t s);
cudaError_t launch_prefill_attention(const PrefillAttnParams &p, int hd, cudaStream_t s);
cudaError_t launch_prefill_input(const int *ids, const float *hidden_in, const int *positions_in, int T,
                                 const uint16_t *embed, int vocab, int d, int ldh, float *h, int *positions,
                                 int max_ctx, unsigned *err, cudaStream_t s);
cudaError_t launch_prefill_rmsnorm(const float *h, int ldh, int T, int d, const float *g, float eps, uint16_t *x,
                                   uint16_t *x_lo, int ldx, int f16, unsigned *err, cudaStream_t s);
// int4 group-64 tiles [n_rb][n_kt][TILE4_BYTES] -> fp16 tiles [n_rb][2 n_kt][RB][KT] of code x scale.
cudaError_t launch_dequant_int4_f16(const uint8_t *tiles4, int n_rb, int n_kt, uint16_t *dst, cudaStream_t s);
cudaError_t launch_split_bf16(const float *x, int T, int K, int ldx, uint16_t *hi, uint16_t *lo, int ld,
                              cudaStream_t s);
cudaError_t launch_prefill_argmax(const float *amax, const int *aidx, int n_tiles, int T, int *next_ids,
                                  cudaStream_t s);

}  // namespace kfl
