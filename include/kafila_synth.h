/*
 * kafila_synth.h -- device twin of the seeded synthetic-input generator.
 *
 * Harness support, not part of the method: the paper fixes no inputs, so the workloads are
 * synthetic and seeded.  One definition of the generator is implemented twice, here on the
 * GPU and in paper_2609_34045_gb300/workload.py with numpy, so that multi-gigabyte weights
 * can be made directly in device memory while the CPU oracle draws bit-identical values.
 *
 *   key(seed, tag) = mix64(seed ^ (tag * 0xD1B54A32D192ED03))
 *   draw(key, i)   = mix64(key + (i + 1) * 0x9E3779B97F4A7C15)        (mod 2^64)
 *   mix64          = the SplitMix64 output function (Steele, Lea, Flood, OOPSLA 2014)
 */
#ifndef KAFILA_SYNTH_H
#define KAFILA_SYNTH_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define KFL_SYNTH_NORMAL_BF16 0      /* uint16_t bf16: mean + c * (S - 131070), S = Irwin-Hall of the
                                        four 16-bit fields of a draw; mean added only if != 0 */
#define KFL_SYNTH_INT4_WORDS 1       /* uint32_t: low 32 bits of a draw */
#define KFL_SYNTH_INT4_SCALES_BF16 2 /* uint16_t bf16: c * (0.5 + (draw >> 40) * 2^-24) */

/* The key of stream (seed, tag). */
uint64_t kfl_synth_key(uint64_t seed, uint64_t tag);

/* Write n values of `kind`, draw indices [start, start + n), into device memory dst,
 * enqueued on cuda_stream.  c and mean are the fp32 constants of the kind.
 * Returns 0 or KFL_ERR_ARG / KFL_ERR_CUDA (kafila_stage.h). */
int kfl_synth_fill(void *dst, int64_t n, uint64_t seed, uint64_t tag, int kind, float c, float mean,
                   int64_t start, void *cuda_stream);

#ifdef __cplusplus
}
#endif
#endif /* KAFILA_SYNTH_H */
