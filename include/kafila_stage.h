/*
 * kafila_stage.h -- C ABI of the GB300 (sm_103a) stage-decode engine.
 *
 * One call of kfl_stage_decode runs one decode step of one pipeline stage: the contiguous
 * range of decoder blocks [l0, l1) that a ring member holds (Kafila, section III: a token
 * leaves the head, passes through each member's block range in turn and returns to the
 * head), plus, for the head, the embedding gather before the blocks and the final RMSNorm,
 * unembedding and greedy sampler after them (section III: the head holds the embedding, the
 * unembedding and the sampler).  Its cost is the stage compute c_i of the paper's cost model
 * (section V-A, Eq. 2): every weight of the stage read once per token.
 *
 * Conventions shared by every call:
 *   - Return value: KFL_OK (0) or a negative KFL_ERR_* code; kfl_strerror names it.
 *   - "device" pointers are CUDA device pointers of the current device (for example
 *     torch.Tensor.data_ptr() of a CUDA tensor); "host" pointers are ordinary CPU memory.
 *   - The caller owns every buffer it passes; the stage owns its weights (repacked copies),
 *     KV cache and workspace, all allocated by kfl_stage_create and freed by
 *     kfl_stage_destroy.
 *   - Matrices are given row-major [out][in] (the nn.Linear convention).  bf16 values are
 *     passed as their 16-bit patterns (uint16_t).
 *   - A stage is not thread-safe: calls on one stage must not overlap on the host.
 */
#ifndef KAFILA_STAGE_H
#define KAFILA_STAGE_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* ---- error codes ---------------------------------------------------------------------- */
#define KFL_OK 0
#define KFL_ERR_ARG (-1)     /* a NULL pointer, a bad size or flag, inconsistent config */
#define KFL_ERR_RANGE (-2)   /* batch > max_batch, a position outside [0, max_ctx), a token id
                                outside [0, vocab), a layer or user index out of range */
#define KFL_ERR_OOM (-3)     /* a device allocation failed; nothing stays allocated */
#define KFL_ERR_CUDA (-4)    /* a CUDA runtime call failed (no device, launch failure, ...) */
#define KFL_ERR_STATE (-5)   /* decode before the weights were loaded, or a destroyed stage */
#define KFL_ERR_TIMEOUT (-6) /* a bounded device-side wait gave up (reported by kfl_stage_status) */
#define KFL_ERR_OVERFLOW (-8) /* an int4 stage's dense prefill met an activation fp16 cannot hold
                                 (|x| >= 65520 or not finite); that prefill's outputs and cache
                                 rows are not valid (reported by kfl_stage_status) */

/* ---- weight formats and stage flags --------------------------------------------------- */
#define KFL_BF16 0     /* bf16 matrices */
#define KFL_INT4_G64 1 /* symmetric int4, group 64 along K, bf16 scales (see kfl_matrix) */

#define KFL_EMBED_IN 1   /* the stage starts from token ids through the embedding (head) */
#define KFL_LOGITS_OUT 2 /* the stage ends with final RMSNorm, lm_head and greedy argmax (head) */
#define KFL_IS_HEAD (KFL_EMBED_IN | KFL_LOGITS_OUT)

/* Model shape (a Qwen-family pre-norm decoder).  rms_eps and rope_theta are the RMSNorm
 * epsilon and the RoPE base.  max_ctx is the number of KV slots reserved per user and
 * max_batch the number of users (batch slots); together they are the session's declared
 * context and concurrency, at which the cache is reserved (section V-C, the block limit
 * lim(i); section V-D, admission).  qk_norm: 0, or 1 for Qwen3-family blocks (the models served
 * in section VI): each head of q and of k is RMS-normalised over head_dim with its own gain (the
 * layer's q_norm, k_norm; epsilon rms_eps) before RoPE.  A qk_norm stage runs one kernel per
 * phase (KFL_PERSISTENT is ignored) and prefills through decode steps. */
typedef struct {
  int n_layers_total, d_model, n_heads, n_kv_heads, head_dim, ffn, vocab;
  float rms_eps, rope_theta;
  int weight_fmt, max_ctx, max_batch, qk_norm;
} kfl_model_cfg;

/* One weight matrix [out][in].  KFL_BF16: w = uint16_t[out][in] bf16 patterns, scales unused.
 * KFL_INT4_G64: w = uint32_t[out][in/8], code j of a word is bits [4j, 4j+4) (low nibble
 * first along K), read as a two's-complement 4-bit integer; scales = uint16_t[out][in/64]
 * bf16; value = code * scale[row][k/64]. */
typedef struct {
  const void *w;
  const void *scales;
} kfl_matrix;

/* One decoder block's weights: RMSNorm gains (bf16 [d_model]), Q/K/V/O and gate/up/down, and
 * with qk_norm the per-head Q and K RMSNorm gains (bf16 [head_dim]; ignored without qk_norm). */
typedef struct {
  const uint16_t *attn_norm, *ffn_norm;
  kfl_matrix wq, wk, wv, wo, wg, wu, wd;
  const uint16_t *q_norm, *k_norm;
} kfl_layer_weights;

/* A stage's weights.  layers[i] is global block l0 + i (n_layers = l1 - l0 entries).  embed
 * (bf16 [vocab][d_model]) is needed with KFL_EMBED_IN; final_norm (bf16 [d_model]) and lm_head
 * ([vocab][d_model], in weight_fmt) with KFL_LOGITS_OUT.  on_device selects whether every
 * pointer is a device (1) or host (0) pointer. */
typedef struct {
  int n_layers;
  int on_device;
  const kfl_layer_weights *layers;
  const uint16_t *embed;
  const uint16_t *final_norm;
  kfl_matrix lm_head;
} kfl_weights;

typedef struct kfl_stage kfl_stage;

/* Bytes of device memory kfl_stage_create would allocate for this stage (weights, KV cache
 * reserved at max_ctx x max_batch, workspace): the per-device block limit lim(i) and the
 * admission check of the paper's planner need exactly this number (section V-C, V-D).
 * Needs no GPU.  Errors: KFL_ERR_ARG. */
int kfl_stage_memory_bytes(const kfl_model_cfg *cfg, int l0, int l1, int flags, size_t *out);

/* Create a stage holding blocks [l0, l1) (0 <= l0 <= l1 <= n_layers_total; l0 == l1 is a pure
 * head tail) with flags KFL_EMBED_IN / KFL_LOGITS_OUT, on the current CUDA device.  Allocates
 * everything up front; the KV cache starts zeroed.  *out receives the stage, or NULL on error.
 * Errors: KFL_ERR_ARG (bad config), KFL_ERR_OOM (an allocation failed; everything allocated so
 * far is freed), KFL_ERR_CUDA. */
int kfl_stage_create(const kfl_model_cfg *cfg, int l0, int l1, int flags, kfl_stage **out);

/* Load every weight of the stage (copies and repacks them; the caller's buffers may be freed
 * afterwards).  Synchronous.  Errors: KFL_ERR_ARG, KFL_ERR_CUDA. */
int kfl_stage_load_weights(kfl_stage *st, const kfl_weights *w);

/* Load one block (local index 0 <= local < l1 - l0) or the head parts; kfl_stage_load_weights
 * is these calls in turn.  The stage counts as loaded once every block and needed head part
 * has been loaded once.  Synchronous. */
int kfl_stage_load_layer(kfl_stage *st, int local, const kfl_layer_weights *w, int on_device);
int kfl_stage_load_head(kfl_stage *st, const uint16_t *embed, const uint16_t *final_norm,
                        const kfl_matrix *lm_head, int on_device);

/* One decode step for users 0..batch-1 (1 <= batch <= max_batch), enqueued on cuda_stream
 * (a cudaStream_t; NULL = the legacy default stream); returns without waiting.
 *   token_ids  device int32[batch]: the token of each user (KFL_EMBED_IN), else ignored
 *   hidden_in  device fp32[batch][d_model]: the stage input (without KFL_EMBED_IN)
 *   positions  device int32[batch]: user b's token position P_b; it attends to its cached
 *              slots [0, P_b] and its K/V are stored at slot P_b (users may differ: ragged)
 *   hidden_out device fp32[batch][d_model]: the stage output (needed without KFL_LOGITS_OUT,
 *              optional with it)
 *   next_ids   device int32[batch]: greedy token of each user (KFL_LOGITS_OUT): the lowest
 *              index among the largest logits
 * A position outside [0, max_ctx) or a token id outside [0, vocab) is found on the device: that
 * user's cache is not written, and kfl_stage_status reports KFL_ERR_RANGE afterwards.
 * Errors returned here: KFL_ERR_ARG, KFL_ERR_RANGE (batch), KFL_ERR_STATE, KFL_ERR_CUDA. */
int kfl_stage_decode(kfl_stage *st, const int32_t *token_ids, const float *hidden_in,
                     const int32_t *positions, int batch, float *hidden_out, int32_t *next_ids,
                     void *cuda_stream);

/* kfl_stage_decode for chosen users: batch row b serves user users[b] (device int32[batch],
 * values in [0, max_batch)), whose KV cache slot it reads and appends to; positions, token_ids,
 * hidden_in/out and next_ids stay indexed by batch row.  A user may fill several rows (several
 * of its tokens in one step) at distinct positions: each row attends to the slot's rows
 * [0, P_b], the ones this step writes included.  A row repeating an earlier row's user and
 * position is treated like a bad position.  This is how one stage of a
 * ring serves one user's token at a time while other users' tokens are elsewhere in the ring
 * (Section VII, "Serving several users at once").  A user outside [0, max_batch) is found on the
 * device and treated like a bad position (nothing of that row is written, kfl_stage_status then
 * reports KFL_ERR_RANGE).  Errors returned here: those of kfl_stage_decode, and KFL_ERR_ARG for
 * users == NULL. */
int kfl_stage_decode_users(kfl_stage *st, const int32_t *token_ids, const float *hidden_in,
                           const int32_t *positions, const int32_t *users, int batch, float *hidden_out,
                           int32_t *next_ids, void *cuda_stream);

/* Prefill: run n_tokens tokens of one user's prompt through the stage, filling the user's KV
 * cache slot at the given positions; each token attends to the slot's rows up to its own
 * position, earlier tokens of the same call included (time to first token is the prefill plus
 * one decode step, Section VI, instrumentation paragraph).  From KFL_PREFILL_DENSE_MIN tokens
 * (environment, default 16) the prompt runs densely: passes of up to 2048 tokens through
 * tensor-core matrix products (tcgen05) and causal attention, each activation carried as two
 * 16-bit terms (bf16 with bf16 weights; fp16 with int4 weights, dequantized to fp16 tiles in
 * device memory the stage allocates at its first dense prefill).  Shorter prompts, and every
 * prompt of a qk_norm stage, go as steps of up to max_batch rows, in order, every row of a step
 * addressing the user's slot (the decode step's kernels).  Enqueued on cuda_stream, returns
 * without waiting.
 *   token_ids  device int32[n_tokens] (KFL_EMBED_IN), else ignored
 *   hidden_in  device fp32[n_tokens][d_model] (without KFL_EMBED_IN)
 *   positions  device int32[n_tokens]: token t's position, distinct, normally start + t; the
 *              slot's rows below a token's position must be cached before the call or be
 *              earlier tokens of it (rows never written read as whatever the slot holds)
 *   user       the KV cache slot, in [0, max_batch)
 *   hidden_out device fp32[n_tokens][d_model] (needed without KFL_LOGITS_OUT)
 *   next_ids   device int32[n_tokens]: the greedy token after each prompt token
 *              (KFL_LOGITS_OUT; the last one starts the decode)
 * Bad positions and token ids are found on the device as in kfl_stage_decode.  In an int4
 * stage's dense prefill an activation beyond the fp16 range (|x| >= 65520, or not finite) is
 * found on the device too: kfl_stage_status then reports KFL_ERR_OVERFLOW and the call's
 * outputs and cache rows are not valid.
 * Errors returned here: KFL_ERR_ARG, KFL_ERR_RANGE (user), KFL_ERR_STATE, KFL_ERR_CUDA. */
int kfl_stage_prefill(kfl_stage *st, const int32_t *token_ids, const float *hidden_in,
                      const int32_t *positions, int user, int n_tokens, float *hidden_out,
                      int32_t *next_ids, void *cuda_stream);

/* kfl_stage_decode with HOST buffers of the same shapes: copies the inputs to the device,
 * runs the step and copies the outputs back, then waits for cuda_stream.  Pinned host memory
 * makes the copies asynchronous to the host; pageable memory works too. */
int kfl_stage_decode_host(kfl_stage *st, const int32_t *token_ids, const float *hidden_in,
                          const int32_t *positions, int batch, float *hidden_out,
                          int32_t *next_ids, void *cuda_stream);

/* Zero the KV cache of one user (0 <= user < max_batch) or of all users (user = -1) in every
 * block of the stage.  Synchronous. */
int kfl_kv_reset(kfl_stage *st, int user);

/* Fill slots [0, len) of one user (or all users, user = -1) in every block of the stage with
 * the seeded synthetic values of the workload generator (bf16, mean 0, standard deviation 1;
 * stream tag depends on the global block index, so stage splits see the same cache).
 * Test/benchmark harness only.  Synchronous. */
int kfl_kv_fill_seeded(kfl_stage *st, int user, int len, uint64_t seed);

/* Copy K and V (bf16 [n_kv_heads][len][head_dim]) into slots [0, len) of one user in block
 * `local`, or read back all slots (bf16 [n_kv_heads][max_ctx][head_dim]).  on_device selects
 * device or host pointers.  Synchronous (the device is synchronised first). */
int kfl_kv_write(kfl_stage *st, int local, int user, const uint16_t *k, const uint16_t *v, int len,
                 int on_device);
int kfl_kv_read(kfl_stage *st, int local, int user, uint16_t *k, uint16_t *v, int on_device);

/* Parity aid: when per_layer_hidden (device fp32 [l1-l0][max_batch][d_model]) is not NULL,
 * every later decode also writes the hidden state after each block there; NULL turns it off.
 * Changing it rebuilds the stage's CUDA graphs on the next decode. */
int kfl_stage_debug_capture(kfl_stage *st, float *per_layer_hidden);

/* Phase trace (tuning aid).  When buf (device uint64 [n_phases][grid][slots], shape from
 * kfl_stage_trace_shape) is not NULL, every later decode writes %globaltimer stamps (ns) per
 * phase and CTA.  Slots: 0 the consumers reach an attention phase / finish a GEMV's tiles,
 * 1 the phase starts on the CTA, 2 the CTA finishes it (epilogues included), 3 its activation
 * input is available (first chunk copied; one-kernel-per-phase: past griddepcontrol.wait),
 * 4 the last activation chunk is copied (persistent kernel), 5/6 the first/last weight tile is
 * issued; one kernel per phase, a GEMV CTA's last row-block segment: 7 its sums are staged,
 * 8 (row block shared with other CTAs) its partial is published and the ticket taken, 9 (last
 * arriver) every partial is summed, 10 the fused epilogue is done, 11 the kind of segment (0 the
 * CTA's alone, 1 shared, 2 shared and last).  Slots of events that do not happen are left as
 * they were.  NULL turns it off.
 * Changing it rebuilds the stage's CUDA graphs on the next decode. */
int kfl_stage_trace(kfl_stage *st, uint64_t *buf);
int kfl_stage_trace_shape(kfl_stage *st, int batch, int *n_phases, int *grid, int *slots);

/* Sticky device-side error word of the stage: waits for the device, then returns KFL_OK,
 * KFL_ERR_TIMEOUT (a bounded wait gave up), KFL_ERR_RANGE (a bad position or token id was
 * seen) or KFL_ERR_OVERFLOW (an int4 dense prefill met an activation fp16 cannot hold), in this
 * order of precedence, and clears it. */
int kfl_stage_status(kfl_stage *st);

/* Per-kernel timing: with enable = 1 later decodes run their kernels one by one (no CUDA
 * graph) with CUDA events around each, accumulating the time of each kernel kind; 0 returns
 * to graph replay.  kfl_stage_profile_read waits for the device and writes, for each kind
 * k < n (KFL_KERNEL_* below), the total milliseconds and the number of launches, then clears
 * the totals.  Returns the number of kinds. */
#define KFL_KERNEL_INPUT 0
#define KFL_KERNEL_QKV 1
#define KFL_KERNEL_ATTN 2
#define KFL_KERNEL_OPROJ 3
#define KFL_KERNEL_GATEUP 4
#define KFL_KERNEL_DOWN 5
#define KFL_KERNEL_LMHEAD 6
#define KFL_KERNEL_OUTPUT 7
#define KFL_KERNEL_KINDS 8
int kfl_stage_profile(kfl_stage *st, int enable);
int kfl_stage_profile_read(kfl_stage *st, double *ms, int64_t *launches, int n);

/* Kernels one decode of this stage launches at this batch (for launch accounting). */
int kfl_stage_launches_per_step(kfl_stage *st, int batch);

void kfl_stage_destroy(kfl_stage *st);
const char *kfl_strerror(int code);

/* Text of the last CUDA runtime error behind a KFL_ERR_CUDA on this thread (the failing call
 * and its error string), or "" if none.  The pointer stays valid until the next failing call. */
const char *kfl_last_error_detail(void);

/* Greedy next token from a head's final hidden state WITHOUT allocating any device memory: the
 * final RMSNorm, the lm_head product and the argmax of a KFL_LOGITS_OUT stage, as one kernel on
 * the caller's buffers.  The paper has no counterpart; this is for callers that cannot call
 * cudaMalloc, such as a host whose device memory is all held by its own pool or allocator, or
 * an embedding that forbids allocation from extension code, and that keep their lm_head
 * themselves.  Enqueued on cuda_stream (a cudaStream_t; NULL = the legacy default stream);
 * returns without waiting.
 *   hidden     device fp32[batch][d_model], 16-byte aligned: the stage output before the norm
 *   final_norm device bf16[d_model], 16-byte aligned: the final RMSNorm gain
 *   lm_head    device bf16[vocab][d_model], row-major, 16-byte aligned (not a stage's tiles)
 *   next_ids   device int32[batch]: the lowest index among the largest logits of each user
 * Limits (the size of its static scratch): 1 <= batch <= 4, d_model a multiple of 8 up to
 * 16384, vocab up to 262144; larger sizes return KFL_ERR_RANGE with the limits in
 * kfl_last_error_detail.  Its scratch is one fixed array of 131,328 bytes of device memory per
 * GPU that loads this library, held until the process exits.  The first call on a device looks
 * the array up, clears its ticket with cudaMemset and waits for the device (cudaDeviceSynchronize),
 * so make that first call before any stream capture.  Every call on a device shares the array and leaves its contents
 * behind; calls that overlap on the GPU (other streams, no ordering) race and give wrong ids.
 * Errors: KFL_ERR_ARG (NULL, misaligned or rms_eps <= 0), KFL_ERR_RANGE, KFL_ERR_CUDA. */
int kfl_head_argmax_noalloc(const float *hidden, const uint16_t *final_norm, const uint16_t *lm_head,
                            int batch, int d_model, int vocab, float rms_eps, int32_t *next_ids,
                            void *cuda_stream);

#ifdef __cplusplus
}
#endif
#endif /* KAFILA_STAGE_H */
