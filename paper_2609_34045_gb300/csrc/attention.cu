// Standalone launch of the decode-attention unit (attn_core.cuh): one CTA per (chunk, KV head,
// user); CTAs beyond a user's chunk count exit at once.  Used when the stage runs one kernel per
// phase; the persistent stage kernel runs the same units itself.
#include "attn_core.cuh"

namespace kfl {

template <int HD>
__global__ void __launch_bounds__(ATT_THREADS) attn_kernel(const __grid_constant__ AttnParams p0) {
  extern __shared__ __align__(128) uint8_t sm[];
  __shared__ int s_last;
  pdl_launch_dependents();
  // the positions were written before the step: the chunk size and the units follow from them
  AttnParams p = p0;
  p.chunk = attn_chunk_size(p0);
  const int nc0 = attn_chunks(p, 0);
  const int nc1 = p.batch > 1 ? attn_chunks(p, 1) : 0;
  const int nc2 = p.batch > 2 ? attn_chunks(p, 2) : 0;
  const int nc3 = p.batch > 3 ? attn_chunks(p, 3) : 0;
  const int units = (nc0 + nc1 + nc2 + nc3) * p.n_kv_heads;
  const int lin = blockIdx.x;
  auto stamp = [&](int slot) {
    if (p.trace && lin < p.trace_grid && threadIdx.x == 0) p.trace[(size_t)lin * TRACE_SLOTS + slot] = global_ns();
  };
  stamp(TR_CONS_GO);
  bool waited = false;
  for (int u = blockIdx.x; u < units; u += gridDim.x) {
    int b, kvh, ch, ncb;
    attn_unit_coords(u, p.n_kv_heads, nc0, nc1, nc2, nc3, b, kvh, ch, ncb);
    // the cached rows [0, P) were written in earlier steps: the unit's first sub-tile (all but the
    // new row, which the Q/K/V kernel writes) loads while that kernel may still run
    attn_prefetch<HD, 2>(p, b, kvh, ch, sm, threadIdx.x);
    if (!waited) {
      pdl_wait();
      stamp(TR_X_GO);
      waited = true;
    }
    attn_unit<HD, 2>(p, b, kvh, ch, ncb, sm, &s_last, threadIdx.x, 1,
                     p.trace && lin < p.trace_grid && u == (int)blockIdx.x ? p.trace + (size_t)lin * TRACE_SLOTS
                                                                           : nullptr);
    __syncthreads();  // the next unit reuses the shared memory
  }
  if (!waited) pdl_wait();
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
  // every unit of the step, whatever the positions: about target_units, plus one partly filled
  // chunk per (user, KV head); a CTA takes further units if there are more
  cfg.gridDim = dim3(p.target_units + p.batch * p.n_kv_heads);
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
  if (p.n_heads % p.n_kv_heads != 0 || p.n_heads / p.n_kv_heads > ATT_MAXG || p.target_units < 1)
    return cudaErrorInvalidValue;
  static_assert(AttnLayout<64, 1>::MERGE_MAX >= ATT_MERGE_MAX, "merge scratch");
  if (head_dim == 128) return launch_hd<128>(p, s, pdl);
  if (head_dim == 64) return launch_hd<64>(p, s, pdl);
  return cudaErrorInvalidValue;
}

}  // namespace kfl
