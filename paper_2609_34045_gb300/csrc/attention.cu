// Standalone launch of the decode-attention unit (attn_core.cuh): one CTA per (chunk, KV head,
// user); CTAs beyond a user's chunk count exit at once.  Used when the stage runs one kernel per
// phase; the persistent stage kernel runs the same units itself.
#include "attn_core.cuh"

namespace kfl {

template <int HD>
__global__ void __launch_bounds__(ATT_THREADS) attn_kernel(const __grid_constant__ AttnParams p) {
  extern __shared__ __align__(128) uint8_t sm[];
  __shared__ int s_last;
  const int c = blockIdx.x, kvh = blockIdx.y, b = blockIdx.z;
  pdl_launch_dependents();
  const int lin = c + gridDim.x * (kvh + gridDim.y * b);
  auto stamp = [&](int slot) {
    if (p.trace && lin < p.trace_grid && threadIdx.x == 0) p.trace[(size_t)lin * TRACE_SLOTS + slot] = global_ns();
  };
  stamp(TR_CONS_GO);
  // the positions were written before the step and the cached rows [0, P) in earlier steps:
  // load the unit's first sub-tile (all but the new row, which the Q/K/V kernel writes) while
  // that kernel is still running
  const int nc = attn_chunks(p, b);
  if (c >= nc) {
    pdl_wait();
    return;
  }
  attn_prefetch<HD, 2>(p, b, kvh, c, sm, threadIdx.x);
  pdl_wait();
  stamp(TR_X_GO);
  attn_unit<HD, 2>(p, b, kvh, c, nc, sm, &s_last, threadIdx.x, 1,
                   p.trace && lin < p.trace_grid ? p.trace + (size_t)lin * TRACE_SLOTS : nullptr);
  stamp(TR_CONS_DONE);
}

cudaError_t prepare_attention() {
  cudaError_t e = cudaFuncSetAttribute(attn_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       AttnLayout<128, 2>::BYTES);
  if (e != cudaSuccess) return e;
  return cudaFuncSetAttribute(attn_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize, AttnLayout<64, 2>::BYTES);
}

template <int HD>
static cudaError_t launch_hd(const AttnParams &p, cudaStream_t s, bool pdl) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(p.n_chunks, p.n_kv_heads, p.batch);
  cfg.blockDim = dim3(ATT_THREADS);
  cfg.dynamicSmemBytes = AttnLayout<HD, 2>::BYTES;
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
  static_assert(AttnLayout<64, 1>::MERGE_MAX >= ATT_MERGE_MAX, "merge scratch");
  if (head_dim == 128) return launch_hd<128>(p, s, pdl);
  if (head_dim == 64) return launch_hd<64>(p, s, pdl);
  return cudaErrorInvalidValue;
}

}  // namespace kfl
