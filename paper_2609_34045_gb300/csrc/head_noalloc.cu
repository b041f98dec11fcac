// Allocation-free greedy head: final RMSNorm, lm_head product and argmax in one kernel, for
// callers that cannot call cudaMalloc (a host whose device memory is all held by its own pool
// or allocator, or an embedding that forbids allocation from extension code).  A stage
// allocates its workspace when it is created; this entry point allocates nothing.  Its scratch
// (each 64-row block's best logit and index per user, and a ticket for the final reduce) is
// the fixed file-scope array below: every GPU that loads the library holds its 131,328 bytes
// until the process exits, and every call on that GPU shares it.
//
// Set-up happens on the first call on each device (with that device current): the array's
// device address is looked up with cudaGetSymbolAddress, its ticket cleared with cudaMemset
// and the device synchronized (the memset is ordered only on the legacy default stream), so that
// first call belongs before any stream capture.  The last
// block of each launch puts the ticket back to zero; the candidates are rewritten by every
// launch before they are read.  The array keeps the last call's contents, and calls that
// overlap on the GPU (different streams with no ordering between them) race on it.
#include <cuda_runtime.h>

#include <cmath>
#include <cstdio>
#include <mutex>

#include "../../include/kafila_stage.h"
#include "common.cuh"

namespace kfl {
void set_error_detail(const char *msg);  // defined with kfl_last_error_detail
}

namespace {

constexpr int NA_ROWS = 64;                                 // rows of lm_head per CTA
constexpr int NA_THREADS = 256;                             // 8 warps x 8 rows
constexpr int NA_MAX_VOCAB = 262144;                        // largest vocabulary accepted
constexpr int NA_MAX_D = 16384;                             // largest d_model accepted
constexpr int NA_MAX_BLOCKS = NA_MAX_VOCAB / NA_ROWS;       // 4096 row blocks
constexpr size_t NA_CAND_BYTES = (size_t)NA_MAX_BLOCKS * kfl::MAXB * 8;  // (value, index) per block and user
constexpr size_t NA_SCRATCH_BYTES = NA_CAND_BYTES + 256;   // + the ticket: 131,328 bytes

// The scratch of every call on this device (each loading GPU keeps it until exit).  Host code
// must not pass this symbol to a kernel: on the host it names a stand-in, not device memory.
static __device__ __align__(256) unsigned char g_head_noalloc_scratch[NA_SCRATCH_BYTES];

constexpr int NA_MAX_DEVICES = 64;
std::mutex g_setup_mutex;
unsigned char *g_scratch_dev[NA_MAX_DEVICES] = {};

// The device address of the scratch on the current device, set up once per device: the symbol's
// address is looked up and the ticket cleared, and the device is synchronized so that the clear has
// finished before any stream uses it (the kernel leaves the ticket at zero after every call).
int scratch_for_current_device(unsigned char **out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= NA_MAX_DEVICES) {
    cudaGetLastError();
    return KFL_ERR_CUDA;
  }
  std::lock_guard<std::mutex> lock(g_setup_mutex);
  if (!g_scratch_dev[dev]) {
    void *p = nullptr;
    cudaError_t e = cudaGetSymbolAddress(&p, g_head_noalloc_scratch);
    if (e != cudaSuccess || p == nullptr) {
      cudaGetLastError();
      return KFL_ERR_CUDA;
    }
    // cudaMemset is ordered only on the legacy default stream and may return before it is done;
    // waiting for the device makes the clear complete before a call on any stream reads it
    e = cudaMemset(static_cast<unsigned char *>(p) + NA_CAND_BYTES, 0, 256);
    if (e == cudaSuccess) e = cudaDeviceSynchronize();
    if (e != cudaSuccess) {
      cudaGetLastError();
      return KFL_ERR_CUDA;
    }
    g_scratch_dev[dev] = static_cast<unsigned char *>(p);
  }
  *out = g_scratch_dev[dev];
  return KFL_OK;
}

__device__ __forceinline__ void na_merge(float &v, int &i, float ov, int oi) {
  if (ov > v || (ov == v && oi < i)) {
    v = ov;
    i = oi;
  }
}

__device__ __forceinline__ void na_warp_argmax(float &v, int &i) {
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    const float ov = __shfl_xor_sync(0xffffffffu, v, off);
    const int oi = __shfl_xor_sync(0xffffffffu, i, off);
    na_merge(v, i, ov, oi);
  }
}

// One CTA per 64 rows of lm_head: RMSNorm scale of each user's hidden state, the 64 logits per
// user (warp w: rows 8w..8w+7), the block's best, then the last CTA (ticket) the overall best.
template <int B>
__global__ void __launch_bounds__(NA_THREADS) head_argmax_noalloc_kernel(const float *hidden, const uint16_t *g,
                                                                         const uint16_t *w, int d, int vocab,
                                                                         float eps, int *next_ids,
                                                                         unsigned char *scratch) {
  float *cand_val = reinterpret_cast<float *>(scratch);
  int *cand_idx = reinterpret_cast<int *>(scratch + (size_t)NA_MAX_BLOCKS * kfl::MAXB * 4);
  unsigned *ticket = reinterpret_cast<unsigned *>(scratch + NA_CAND_BYTES);
  __shared__ float s_inv[B];
  __shared__ float s_val[8][B];
  __shared__ int s_idx[8][B];
  __shared__ int s_last;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

  // RMSNorm scale 1 / sqrt(mean(h^2) + eps), warp b for user b
  if (warp < B) {
    float s = 0.f;
    for (int k = lane; k < d; k += 32) {
      const float h = hidden[(size_t)warp * d + k];
      s = fmaf(h, h, s);
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) s += __shfl_xor_sync(0xffffffffu, s, off);
    if (lane == 0) s_inv[warp] = 1.0f / sqrtf(s / static_cast<float>(d) + eps);
  }
  __syncthreads();

  // logits of rows r0 .. r0 + 7: lanes take 8 consecutive K (one 16-byte load of each row)
  float best_v[B];
  int best_i[B];
#pragma unroll
  for (int b = 0; b < B; ++b) {
    best_v[b] = -INFINITY;
    best_i[b] = 0x7fffffff;
  }
  const int r0 = blockIdx.x * NA_ROWS + warp * 8;
  float acc[8][B];
#pragma unroll
  for (int j = 0; j < 8; ++j)
#pragma unroll
    for (int b = 0; b < B; ++b) acc[j][b] = 0.f;
  for (int k0 = lane * 8; k0 < d; k0 += 256) {
    const uint4 g4 = *reinterpret_cast<const uint4 *>(g + k0);
    const float gv[8] = {kfl::bf16_lo(g4.x), kfl::bf16_hi(g4.x), kfl::bf16_lo(g4.y), kfl::bf16_hi(g4.y),
                         kfl::bf16_lo(g4.z), kfl::bf16_hi(g4.z), kfl::bf16_lo(g4.w), kfl::bf16_hi(g4.w)};
    float xv[B][8];
#pragma unroll
    for (int b = 0; b < B; ++b) {
      const float4 a0 = *reinterpret_cast<const float4 *>(hidden + (size_t)b * d + k0);
      const float4 a1 = *reinterpret_cast<const float4 *>(hidden + (size_t)b * d + k0 + 4);
      const float hv[8] = {a0.x, a0.y, a0.z, a0.w, a1.x, a1.y, a1.z, a1.w};
#pragma unroll
      for (int e = 0; e < 8; ++e) xv[b][e] = hv[e] * gv[e];
    }
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int r = r0 + j;
      if (r < vocab) {
        const uint4 w4 = *reinterpret_cast<const uint4 *>(w + (size_t)r * d + k0);
        const float wv[8] = {kfl::bf16_lo(w4.x), kfl::bf16_hi(w4.x), kfl::bf16_lo(w4.y), kfl::bf16_hi(w4.y),
                             kfl::bf16_lo(w4.z), kfl::bf16_hi(w4.z), kfl::bf16_lo(w4.w), kfl::bf16_hi(w4.w)};
#pragma unroll
        for (int b = 0; b < B; ++b)
#pragma unroll
          for (int e = 0; e < 8; ++e) acc[j][b] = fmaf(wv[e], xv[b][e], acc[j][b]);
      }
    }
  }
#pragma unroll
  for (int j = 0; j < 8; ++j) {
#pragma unroll
    for (int b = 0; b < B; ++b) {
      float v = acc[j][b];
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
      if (r0 + j < vocab) na_merge(best_v[b], best_i[b], v * s_inv[b], r0 + j);
    }
  }
  if (lane == 0) {
#pragma unroll
    for (int b = 0; b < B; ++b) {
      s_val[warp][b] = best_v[b];
      s_idx[warp][b] = best_i[b];
    }
  }
  __syncthreads();
  if (tid < B) {
    float v = s_val[0][tid];
    int i = s_idx[0][tid];
    for (int wq = 1; wq < 8; ++wq) na_merge(v, i, s_val[wq][tid], s_idx[wq][tid]);
    cand_val[blockIdx.x * kfl::MAXB + tid] = v;
    cand_idx[blockIdx.x * kfl::MAXB + tid] = i;
    __threadfence();
  }
  __syncthreads();
  if (tid == 0) {
    // release this block's candidates; the last block to arrive acquires all of them
    const unsigned prev = kfl::atom_add_acq_rel(ticket, 1u);
    s_last = prev == gridDim.x - 1;
    if (s_last) atomicExch(ticket, 0u);  // the next call starts from zero
  }
  __syncthreads();
  if (!s_last) return;
  for (int b = warp; b < B; b += NA_THREADS / 32) {
    float v = -INFINITY;
    int i = 0x7fffffff;
    for (int blk = lane; blk < (int)gridDim.x; blk += 32)
      na_merge(v, i, __ldcg(cand_val + blk * kfl::MAXB + b), __ldcg(cand_idx + blk * kfl::MAXB + b));
    na_warp_argmax(v, i);
    if (lane == 0) next_ids[b] = i == 0x7fffffff ? 0 : i;
  }
}

}  // namespace

extern "C" int kfl_head_argmax_noalloc(const float *hidden, const uint16_t *final_norm, const uint16_t *lm_head,
                                       int batch, int d_model, int vocab, float rms_eps, int32_t *next_ids,
                                       void *cuda_stream) {
  if (!hidden || !final_norm || !lm_head || !next_ids || !(rms_eps > 0.f)) {
    kfl::set_error_detail("kfl_head_argmax_noalloc: NULL pointer or non-positive rms_eps");
    return KFL_ERR_ARG;
  }
  if ((reinterpret_cast<uintptr_t>(hidden) | reinterpret_cast<uintptr_t>(final_norm) |
       reinterpret_cast<uintptr_t>(lm_head)) & 15) {
    kfl::set_error_detail("kfl_head_argmax_noalloc: hidden, final_norm and lm_head must be 16-byte aligned");
    return KFL_ERR_ARG;
  }
  if (batch < 1 || batch > kfl::MAXB || d_model < 8 || d_model % 8 != 0 || d_model > NA_MAX_D || vocab < 1 ||
      vocab > NA_MAX_VOCAB) {
    char msg[200];
    snprintf(msg, sizeof(msg),
             "kfl_head_argmax_noalloc: batch %d, d_model %d, vocab %d outside the static scratch's limits "
             "(batch 1..%d, d_model a multiple of 8 up to %d, vocab up to %d)",
             batch, d_model, vocab, kfl::MAXB, NA_MAX_D, NA_MAX_VOCAB);
    kfl::set_error_detail(msg);
    return KFL_ERR_RANGE;
  }
  unsigned char *scratch = nullptr;
  int rc = scratch_for_current_device(&scratch);
  if (rc != KFL_OK) {
    kfl::set_error_detail("kfl_head_argmax_noalloc: could not look up or clear the static scratch");
    return rc;
  }
  const int blocks = (vocab + NA_ROWS - 1) / NA_ROWS;
  cudaStream_t s = static_cast<cudaStream_t>(cuda_stream);
  switch (batch) {
    case 1: head_argmax_noalloc_kernel<1><<<blocks, NA_THREADS, 0, s>>>(hidden, final_norm, lm_head, d_model, vocab, rms_eps, next_ids, scratch); break;
    case 2: head_argmax_noalloc_kernel<2><<<blocks, NA_THREADS, 0, s>>>(hidden, final_norm, lm_head, d_model, vocab, rms_eps, next_ids, scratch); break;
    case 3: head_argmax_noalloc_kernel<3><<<blocks, NA_THREADS, 0, s>>>(hidden, final_norm, lm_head, d_model, vocab, rms_eps, next_ids, scratch); break;
    default: head_argmax_noalloc_kernel<4><<<blocks, NA_THREADS, 0, s>>>(hidden, final_norm, lm_head, d_model, vocab, rms_eps, next_ids, scratch); break;
  }
  const cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) {
    kfl::set_error_detail(cudaGetErrorString(e));
    return KFL_ERR_CUDA;
  }
  return KFL_OK;
}
