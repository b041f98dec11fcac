// Device twin of the seeded synthetic-input generator (harness support, not the method).
// Definition in kafila_synth.h; every float step is one IEEE fp32 operation written with an
// explicit rounding intrinsic so that no multiply-add contraction changes a bit, and the
// values match the numpy implementation exactly.
#include "../../include/kafila_stage.h"
#include "../../include/kafila_synth.h"
#include "common.cuh"

namespace {

constexpr uint64_t GAMMA = 0x9E3779B97F4A7C15ull;
constexpr uint64_t TAGMUL = 0xD1B54A32D192ED03ull;

__host__ __device__ __forceinline__ uint64_t mix64(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

__device__ __forceinline__ uint16_t bf16_rne_bits(float f) {
  uint32_t u = __float_as_uint(f);
  if ((u & 0x7FFFFFFFu) > 0x7F800000u) return 0x7FC0;
  return static_cast<uint16_t>((u + 0x7FFFu + ((u >> 16) & 1u)) >> 16);
}

__global__ void synth_kernel(void *dst, long long n, uint64_t key, int kind, float c, float mean, long long start) {
  for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < n;
       i += (long long)gridDim.x * blockDim.x) {
    const uint64_t d = mix64(key + (static_cast<uint64_t>(start + i) + 1ull) * GAMMA);
    if (kind == KFL_SYNTH_NORMAL_BF16) {
      const uint32_t s = static_cast<uint32_t>(d & 0xFFFF) + static_cast<uint32_t>((d >> 16) & 0xFFFF) +
                         static_cast<uint32_t>((d >> 32) & 0xFFFF) + static_cast<uint32_t>(d >> 48);
      float z = __fmul_rn(static_cast<float>(static_cast<int>(s) - 131070), c);
      if (mean != 0.0f) z = __fadd_rn(mean, z);
      static_cast<uint16_t *>(dst)[i] = bf16_rne_bits(z);
    } else if (kind == KFL_SYNTH_INT4_WORDS) {
      static_cast<uint32_t *>(dst)[i] = static_cast<uint32_t>(d & 0xFFFFFFFFull);
    } else {
      const float u = __fmul_rn(static_cast<float>(static_cast<uint32_t>(d >> 40)), 5.9604644775390625e-08f);
      static_cast<uint16_t *>(dst)[i] = bf16_rne_bits(__fmul_rn(c, __fadd_rn(0.5f, u)));
    }
  }
}

}  // namespace

extern "C" uint64_t kfl_synth_key(uint64_t seed, uint64_t tag) { return mix64(seed ^ (tag * TAGMUL)); }

extern "C" int kfl_synth_fill(void *dst, int64_t n, uint64_t seed, uint64_t tag, int kind, float c, float mean,
                              int64_t start, void *cuda_stream) {
  if (n < 0 || start < 0 || (n > 0 && dst == nullptr)) return KFL_ERR_ARG;
  if (kind != KFL_SYNTH_NORMAL_BF16 && kind != KFL_SYNTH_INT4_WORDS && kind != KFL_SYNTH_INT4_SCALES_BF16)
    return KFL_ERR_ARG;
  if (n == 0) return KFL_OK;
  const long long blocks_needed = (n + 255) / 256;
  const int blocks = blocks_needed < 152 * 32 ? static_cast<int>(blocks_needed) : 152 * 32;
  synth_kernel<<<blocks, 256, 0, static_cast<cudaStream_t>(cuda_stream)>>>(dst, n, kfl_synth_key(seed, tag), kind, c,
                                                                          mean, start);
  return cudaGetLastError() == cudaSuccess ? KFL_OK : KFL_ERR_CUDA;
}
