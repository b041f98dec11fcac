// Stage input/output and load-time kernels.
#include "common.cuh"

namespace kfl {

// Stage input (Kafila section III: the head embeds the token; other members receive the
// hidden state from the previous ring member).  One CTA of 64 threads per (64-row block,
// user): writes h, the next RMSNorm input xn = h * g_next and the block's sum of squares,
// and copies/validates the positions.
__global__ void __launch_bounds__(64) stage_input_kernel(const int *ids, const float *hidden_in,
                                                         const int *positions_in, const uint16_t *embed,
                                                         int vocab, int d, int ldh, const float *g_next,
                                                         float *h, float *xn, float *sumsq, int *positions,
                                                         int max_ctx, unsigned *err, unsigned *bar, Act16 xn16,
                                                         const int *users, int user_all, int max_batch,
                                                         int *slots) {
  __shared__ float vals[64];
  const int b = blockIdx.y, tid = threadIdx.x, r = blockIdx.x * 64 + tid;
  pdl_launch_dependents();
  pdl_wait();
  if (blockIdx.x == 0 && tid == 0) {
    int pos = positions_in[b];
    if (pos < 0 || pos >= max_ctx) atomicOr(err, ERR_POSITION);
    // the user's KV slot (users NULL: user_all for every row if >= 0, else batch row b is user
    // b); a slot outside [0, max_batch) is flagged like a bad position, and the row's position is
    // made invalid so that nothing of it is written.  Rows of one user must hold distinct
    // positions (each writes its own cache row): a repeat of an earlier row's is flagged the same.
    auto slot_of = [&](int j) { return users ? users[j] : (user_all >= 0 ? user_all : j); };
    const int u = slot_of(b);
    if (u < 0 || u >= max_batch) {
      atomicOr(err, ERR_POSITION);
      pos = -1;
    }
    for (int j = 0; j < b && pos >= 0; ++j)
      if (slot_of(j) == u && positions_in[j] == pos) {
        atomicOr(err, ERR_POSITION);
        pos = -1;
      }
    slots[b] = (u < 0 || u >= max_batch) ? 0 : u;
    positions[b] = pos;
    // abort flag of the persistent stage kernel that follows
    if (b == 0 && bar) {
      bar[0] = 0u;
      bar[1] = 0u;
    }
  }
  float v = 0.f;
  if (r < d) {
    if (embed) {
      int id = ids[b];
      if (id < 0 || id >= vocab) {
        if (tid == 0 && blockIdx.x == 0) atomicOr(err, ERR_TOKEN);
        id = 0;
      }
      v = bf16_to_f32(embed[(size_t)id * d + r]);
    } else {
      v = hidden_in[(size_t)b * d + r];
    }
    h[(size_t)b * ldh + r] = v;
  }
  if (g_next) {
    // xn = h * g; for int4 weights in the tensor-core input form (one warp per 32-element chunk),
    // exactly as the residual epilogue writes it
    const float xv = r < d ? v * g_next[r] : 0.f;
    if (xn16.base)
      act16_put_warp(xn16, b, blockIdx.x * 2 + (tid >> 5), xv, tid & 31);
    else if (r < d)
      xn[(size_t)b * ldh + r] = xv;
  }
  // the block's sum of squares in exactly the order of the residual epilogue (lane l: rows l
  // and l + 32 by fma, then a butterfly), so that a stage fed this hidden state computes the same
  // bits as the block before it did
  vals[tid] = v;
  __syncthreads();
  if (tid < 32) {
    float sq = fmaf(vals[tid], vals[tid], 0.f);
    sq = fmaf(vals[tid + 32], vals[tid + 32], sq);
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) sq += __shfl_xor_sync(0xffffffffu, sq, off);
    if (tid == 0) sumsq[blockIdx.x * MAXB + b] = sq;
  }
}

cudaError_t launch_stage_input(const int *ids, const float *hidden_in, const int *positions_in, int batch,
                               const uint16_t *embed, int vocab, int d, int ldh, const float *g_next, float *h,
                               float *xn, float *sumsq, int *positions, int max_ctx, unsigned *err,
                               unsigned *bar, Act16 xn16, const int *users, int user_all, int max_batch,
                               int *slots, cudaStream_t s) {
  dim3 grid((d + 63) / 64, batch);
  stage_input_kernel<<<grid, 64, 0, s>>>(ids, hidden_in, positions_in, embed, vocab, d, ldh, g_next, h, xn, sumsq,
                                         positions, max_ctx, err, bar, xn16, users, user_all, max_batch, slots);
  return cudaGetLastError();
}

__global__ void stage_output_kernel(const float *h, int ldh, int d, float *hidden_out, const int *next_in,
                                    int *next_ids) {
  pdl_launch_dependents();
  pdl_wait();
  const int b = blockIdx.y;
  const int r = blockIdx.x * blockDim.x + threadIdx.x;
  if (hidden_out && r < d) hidden_out[(size_t)b * d + r] = h[(size_t)b * ldh + r];
  if (next_ids && blockIdx.x == 0 && threadIdx.x == 0) next_ids[b] = next_in[b];
}

cudaError_t launch_stage_output(const float *h, int ldh, int d, int batch, float *hidden_out, const int *next_in,
                                int *next_ids, cudaStream_t s, bool pdl) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((d + 255) / 256, batch);
  cfg.blockDim = dim3(256);
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, stage_output_kernel, h, ldh, d, hidden_out, next_in, next_ids);
}

// QK-norm of Qwen3-family blocks (the served models of section VI): each head of q and of k is
// RMS-normalised over head_dim with its gain (g_q, g_k), then rotated (RoPE at the row's
// position); q goes to the attention input, k and v (bf16, nearest even) to the row's KV slot.
// One CTA per (head of Q, K or V, batch row), one thread per rotation pair (i, i + hd/2), whose
// two values are adjacent rows of the projection (GEMV order).  The norm's sum of squares is
// reduced in a fixed order (butterfly within a warp, then the warps in order), as the other
// norms of the path are.
template <int HD>
__global__ void __launch_bounds__(HD / 2) qknorm_rope_kernel(QkNormParams p) {
  constexpr int HALF = HD / 2, NW = HALF / 32;
  __shared__ float s_part[NW];
  pdl_launch_dependents();
  pdl_wait();
  const int head = blockIdx.x, b = blockIdx.y, i = threadIdx.x;
  const int nq = p.n_heads, nk = p.n_kv_heads;
  const float *raw = p.raw + (size_t)b * p.ld_raw;
  const int pv = p.positions[b];
  const bool ok = pv >= 0 && pv < p.max_ctx;
  const size_t slot_base = (size_t)p.slots[b] * nk;
  if (head >= nq + nk) {  // V rows are in natural order: no norm, no rotation
    if (!ok) return;
    const int vh = head - nq - nk;
    const float2 x = *reinterpret_cast<const float2 *>(raw + (size_t)(nq + nk) * HD + (size_t)vh * HD + 2 * i);
    uint16_t *vd = p.vcache + ((slot_base + vh) * p.max_ctx + pv) * HD;
    vd[2 * i] = f32_to_bf16_rne(x.x);
    vd[2 * i + 1] = f32_to_bf16_rne(x.y);
    return;
  }
  const bool is_q = head < nq;
  const float2 x = *reinterpret_cast<const float2 *>(raw + (size_t)head * HD + 2 * i);
  float s = x.x * x.x + x.y * x.y;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) s += __shfl_xor_sync(0xffffffffu, s, off);
  if constexpr (NW > 1) {
    if ((i & 31) == 0) s_part[i >> 5] = s;
    __syncthreads();
    s = 0.f;
#pragma unroll
    for (int w = 0; w < NW; ++w) s += s_part[w];
  }
  const float r = 1.0f / sqrtf(s / static_cast<float>(HD) + p.eps);
  const float *g = is_q ? p.g_q : p.g_k;
  const float y1 = x.x * r * g[i], y2 = x.y * r * g[i + HALF];
  const size_t ri = (size_t)(ok ? pv : 0) * HALF + i;
  const float cs = p.rope_cos[ri], sn = p.rope_sin[ri];
  const float a = y1 * cs - y2 * sn;
  const float c2 = y2 * cs + y1 * sn;
  if (is_q) {
    float *qd = p.q + (size_t)b * nq * HD + (size_t)head * HD;
    qd[i] = a;
    qd[i + HALF] = c2;
  } else if (ok) {
    uint16_t *kd = p.kcache + ((slot_base + (head - nq)) * p.max_ctx + pv) * HD;
    kd[i] = f32_to_bf16_rne(a);
    kd[i + HALF] = f32_to_bf16_rne(c2);
  }
}

cudaError_t launch_qknorm(const QkNormParams &p, cudaStream_t s, bool pdl) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(p.n_heads + 2 * p.n_kv_heads, p.batch);
  cfg.blockDim = dim3(p.head_dim / 2);
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  if (p.head_dim == 128) return cudaLaunchKernelEx(&cfg, qknorm_rope_kernel<128>, p);
  if (p.head_dim == 64) return cudaLaunchKernelEx(&cfg, qknorm_rope_kernel<64>, p);
  return cudaErrorInvalidValue;
}

// Repack a bf16 matrix src [n_src_rows][k] into tiles [n_rb][n_kt][RB][KT]: output row r is
// source row row_map[r] (or r when row_map is NULL); rows >= n_rows_out and columns >= k are 0.
__global__ void repack_bf16_kernel(const uint16_t *src, int n_src_rows, int k, const int *row_map, int n_rows_out,
                                   int n_rb, int n_kt, uint8_t *dst) {
  const long long total = (long long)n_rb * n_kt * RB * (KT / 8);
  for (long long e = blockIdx.x * (long long)blockDim.x + threadIdx.x; e < total;
       e += (long long)gridDim.x * blockDim.x) {
    const int ch = static_cast<int>(e % (KT / 8));
    const long long rest = e / (KT / 8);
    const int r = static_cast<int>(rest % RB);
    const long long t = rest / RB;
    const int kt = static_cast<int>(t % n_kt);
    const int rb = static_cast<int>(t / n_kt);
    const int orow = rb * RB + r;
    int srow = -1;
    if (orow < n_rows_out) srow = row_map ? row_map[orow] : orow;
    if (srow >= n_src_rows) srow = -1;
    const int k0 = kt * KT + ch * 8;
    uint16_t v[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) v[j] = (srow >= 0 && k0 + j < k) ? src[(size_t)srow * k + k0 + j] : uint16_t(0);
    uint4 o;
    o.x = v[0] | (uint32_t(v[1]) << 16);
    o.y = v[2] | (uint32_t(v[3]) << 16);
    o.z = v[4] | (uint32_t(v[5]) << 16);
    o.w = v[6] | (uint32_t(v[7]) << 16);
    reinterpret_cast<uint4 *>(dst)[e] = o;
  }
}

cudaError_t launch_repack_bf16(const uint16_t *src, int n_src_rows, int k, const int *row_map, int n_rows_out,
                               int n_rb, int n_kt, uint8_t *dst, cudaStream_t s) {
  repack_bf16_kernel<<<4 * 152 * 4, 256, 0, s>>>(src, n_src_rows, k, row_map, n_rows_out, n_rb, n_kt, dst);
  return cudaGetLastError();
}

// Repack an int4 group-64 matrix (words [n_src_rows][k/8], scales [n_src_rows][k/64]) into
// tiles [n_rb][n_kt][RB][KT4/8 words] followed by RB x KT4/64 bf16 scales per tile.
// int4 tiles in the order of the tensor-core MMA fragments (tile_compute, FMT 1): the 64 x 256
// codes of a tile are 2048 words; word ((((h * 4 + r16) * 2 + q) * 32 + lane) * 4 + j) holds the
// eight codes lane needs for K step s = 4 q + j of K half h and row group r16 (rows r16 * 16 +
// gid and + 8, gid = lane / 4; columns 2 tig, 2 tig + 1, 2 tig + 8, 2 tig + 9 of the step, tig =
// lane % 4), nibble i at bits 4 i: row + 8 ((i >> 1) & 1), column + 8 (i & 1) + ((i >> 2) & 1),
// so that the nibble pairs at bits (0, 16), (8, 24), (4, 20), (12, 28) are the A registers a0,
// a1, a2, a3 (int4_frag_f16).  The 64 x 4 scales are stored in the order of tile4_scale_index
// (a lane's rows gid and gid + 8, both groups of its K half, in 8 consecutive bytes).
__global__ void repack_int4_kernel(const uint32_t *words, const uint16_t *scales, int n_src_rows, int k,
                                   const int *row_map, int n_rows_out, int n_rb, int n_kt, uint8_t *dst) {
  constexpr int TW = TILE4_CODE_BYTES / 4;  // words per tile
  constexpr int SPR = KT4 / 64;             // scales per tile row
  const int kw = k / 8, ks = k / 64;
  const long long total = (long long)n_rb * n_kt * TW;
  for (long long e = blockIdx.x * (long long)blockDim.x + threadIdx.x; e < total;
       e += (long long)gridDim.x * blockDim.x) {
    const int idx = static_cast<int>(e % TW);
    const long long t = e / TW;
    const int kt = static_cast<int>(t % n_kt);
    const int rb = static_cast<int>(t / n_kt);
    const int j = idx & 3, lane = (idx >> 2) & 31, q = (idx >> 7) & 1, r16 = (idx >> 8) & 3, h = idx >> 10;
    const int gid = lane >> 2, tig = lane & 3;
    uint32_t out = 0;
    for (int i = 0; i < 8; ++i) {
      const int orow = rb * RB + r16 * 16 + gid + 8 * ((i >> 1) & 1);
      const int kk = kt * KT4 + 128 * h + 16 * (4 * q + j) + 2 * tig + 8 * (i & 1) + ((i >> 2) & 1);
      int srow = -1;
      if (orow < n_rows_out) srow = row_map ? row_map[orow] : orow;
      if (srow >= n_src_rows) srow = -1;
      uint32_t nib = 0;
      if (srow >= 0 && kk < k) nib = (words[(size_t)srow * kw + kk / 8] >> (4 * (kk % 8))) & 0xFu;
      out |= nib << (4 * i);
    }
    uint8_t *tile = dst + (size_t)t * TILE4_BYTES;
    reinterpret_cast<uint32_t *>(tile)[idx] = out;
    if (idx < RB) {
      // the tile's scales, one row per thread
      const int orow = rb * RB + idx;
      int srow = -1;
      if (orow < n_rows_out) srow = row_map ? row_map[orow] : orow;
      if (srow >= n_src_rows) srow = -1;
      uint16_t *sd = reinterpret_cast<uint16_t *>(tile + TILE4_CODE_BYTES);
      for (int g = 0; g < SPR; ++g) {
        const int gg = kt * SPR + g;
        sd[tile4_scale_index(idx, g)] = (srow >= 0 && gg < ks) ? scales[(size_t)srow * ks + gg] : uint16_t(0);
      }
    }
  }
}

cudaError_t launch_repack_int4(const uint32_t *words, const uint16_t *scales, int n_src_rows, int k,
                               const int *row_map, int n_rows_out, int n_rb, int n_kt, uint8_t *dst,
                               cudaStream_t s) {
  repack_int4_kernel<<<4 * 152, 256, 0, s>>>(words, scales, n_src_rows, k, row_map, n_rows_out, n_rb, n_kt, dst);
  return cudaGetLastError();
}

__global__ void bf16_to_f32_kernel(const uint16_t *src, float *dst, int n) {
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < n; i += gridDim.x * blockDim.x)
    dst[i] = bf16_to_f32(src[i]);
}

cudaError_t launch_bf16_to_f32(const uint16_t *src, float *dst, int n, cudaStream_t s) {
  if (n <= 0) return cudaSuccess;
  bf16_to_f32_kernel<<<(n + 255) / 256 < 1024 ? (n + 255) / 256 : 1024, 256, 0, s>>>(src, dst, n);
  return cudaGetLastError();
}

}  // namespace kfl
