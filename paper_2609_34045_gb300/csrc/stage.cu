// Stage runtime and C ABI (kafila_stage.h).
//
// A stage owns its repacked weights, its KV cache (reserved at max_ctx x max_batch, the
// declared context and concurrency of Kafila section V-C/V-D) and a small workspace.  A decode
// step is: stage input kernel -> one CUDA graph of the block kernels (captured once per batch
// size, kernels chained with programmatic dependent launch) -> stage output kernel.
#include <cuda_runtime.h>

#include <cmath>
#include <algorithm>
#include <cstdlib>
#include <cstdio>
#include <cstring>
#include <vector>

#include "../../include/kafila_plan.h"
#include "../../include/kafila_stage.h"
#include "../../include/kafila_synth.h"
#include "common.cuh"
#include "prefill.cuh"

using namespace kfl;

namespace {

int round_up(int x, int m) { return (x + m - 1) / m * m; }

struct Mat {
  uint8_t *tiles = nullptr;
  int N = 0, K = 0, n_rb = 0, n_kt = 0, fmt = 0;
  size_t bytes = 0;
};

Mat mat_shape(int N, int K, int fmt) {
  Mat m;
  m.N = N;
  m.K = K;
  m.fmt = fmt;
  m.n_rb = (N + RB - 1) / RB;
  const int kt = fmt == KFL_BF16 ? KT : KT4;
  m.n_kt = (K + kt - 1) / kt;
  m.bytes = (size_t)m.n_rb * m.n_kt * (fmt == KFL_BF16 ? TILE_BYTES : TILE4_BYTES);
  return m;
}

struct LayerDev {
  Mat qkv, o, gu, down;
  float *g_attn = nullptr, *g_ffn = nullptr;
  float *g_q = nullptr, *g_k = nullptr;  // QK-norm gains [hd] (qk_norm stages)
  bool loaded = false;
};

// Every size the stage allocates, computed once for kfl_stage_memory_bytes and create.
struct Plan {
  int d, hq, hkv, hd, F, V, qdim, kvdim, nl;
  int ldh, ldq, lda;  // activation row strides, multiples of 256 floats
  int ld_raw;         // QK-norm stages: row stride of the raw Q/K/V projection (else 0)
  Mat qkv, o, gu, down, lm;
  size_t kv_elems_per_layer;  // per cache (K or V)
  int n_sm, ctas_per_sm, stages, gemv_grid_max, n_rb_max, n_parts, attn_nchunks_max;
  int small_gemv_tiles, small_gemv_stages;  // GEMVs of at most this many tiles: one CTA per SM
  int cluster;                              // small GEMVs run as clusters of this many CTAs (see enqueue_body)
  int n_phases, ctr_stride;  // persistent kernel: phases per step, readiness counters per phase
  int attn_units;            // attention units a step aims at (the kernels size chunks to it)
  int attn_cluster_max;      // one kernel per phase: the largest attention cluster (0: unit kernel)
  int attn_stages;           // attention clusters: ring depth (sub-tiles) of a CTA
  int attn_cluster_sub;      // clusters are taken up to this many 64-position sub-tiles per CTA
  int attn_launch_at;        // AttnParams::launch_at, for O projections of at most attn_late_max_mb MiB
  int attn_late_max_mb;
  int down_cluster;          // the down projection as clusters of this many CTAs per row block (0: stream-K)
  size_t bytes_weights, bytes_kv, bytes_ws;
};

// Bytes of one int4 GEMV input (Act16) of row length ld: MAXB fp16 rows (and their rests), and
// the per-chunk constants.
size_t act16_bytes(int ld, bool with_rest) { return (size_t)(ld / KT4) * act16_tile_bytes(with_rest ? 1 : 0); }

int env_int(const char *name, int dflt) {
  const char *v = std::getenv(name);
  return (v && *v) ? std::atoi(v) : dflt;
}

int validate_cfg(const kfl_model_cfg *c, int l0, int l1, int flags) {
  if (!c) return KFL_ERR_ARG;
  if (c->n_layers_total <= 0 || c->d_model <= 0 || c->n_heads <= 0 || c->n_kv_heads <= 0 || c->head_dim <= 0 ||
      c->ffn <= 0 || c->vocab <= 0)
    return KFL_ERR_ARG;
  if (c->n_heads % c->n_kv_heads != 0 || c->n_heads / c->n_kv_heads > 8) return KFL_ERR_ARG;
  if (c->head_dim != 64 && c->head_dim != 128) return KFL_ERR_ARG;
  if (c->d_model % 8 != 0 || c->ffn % 8 != 0) return KFL_ERR_ARG;
  if (c->weight_fmt != KFL_BF16 && c->weight_fmt != KFL_INT4_G64) return KFL_ERR_ARG;
  if (c->weight_fmt == KFL_INT4_G64 &&
      (c->d_model % 64 != 0 || c->ffn % 64 != 0 || (c->n_heads * c->head_dim) % 64 != 0))
    return KFL_ERR_ARG;
  if (c->max_ctx <= 0 || c->max_batch <= 0 || c->max_batch > MAXB) return KFL_ERR_ARG;
  if (c->max_ctx > (1 << 20)) return KFL_ERR_ARG;
  if (c->qk_norm != 0 && c->qk_norm != 1) return KFL_ERR_ARG;
  if (!(c->rms_eps > 0.f) || !(c->rope_theta > 0.f)) return KFL_ERR_ARG;
  if (l0 < 0 || l1 < l0 || l1 > c->n_layers_total) return KFL_ERR_ARG;
  if (flags & ~KFL_IS_HEAD) return KFL_ERR_ARG;
  if (l0 == l1 && !(flags & KFL_LOGITS_OUT) && !(flags & KFL_EMBED_IN)) return KFL_ERR_ARG;
  return KFL_OK;
}

void make_plan(const kfl_model_cfg *c, int l0, int l1, int flags, int n_sm, Plan *p) {
  p->d = c->d_model;
  p->hq = c->n_heads;
  p->hkv = c->n_kv_heads;
  p->hd = c->head_dim;
  p->F = c->ffn;
  p->V = c->vocab;
  p->qdim = p->hq * p->hd;
  p->kvdim = p->hkv * p->hd;
  p->nl = l1 - l0;
  p->ldh = round_up(p->d, 256);
  p->ldq = round_up(p->qdim, 256);
  p->lda = round_up(p->F, 256);
  p->ld_raw = c->qk_norm ? round_up(p->qdim + 2 * p->kvdim, 256) : 0;
  const int f = c->weight_fmt;
  p->qkv = mat_shape(p->qdim + 2 * p->kvdim, p->d, f);
  p->o = mat_shape(p->d, p->qdim, f);
  p->gu = mat_shape(2 * p->F, p->d, f);
  p->down = mat_shape(p->d, p->F, f);
  p->lm = mat_shape(p->V, p->d, f);
  p->kv_elems_per_layer = (size_t)c->max_batch * p->hkv * c->max_ctx * p->hd;
  p->n_sm = n_sm;
  // Two CTAs per SM: a single CTA's consumer warps (8) leave the tile loop bound by instruction
  // latency (int4 decoding; bf16 at batch 4), two give every SM twice the warps to hide it.  The
  // rings are sized so that two fit an SM at every batch size: 5 bf16 stages (at most 90 KiB);
  // int4 rings take the deepest even depth up to 8 that fits (8 at batch 1, 6 at batch 4, with
  // its staging slots): 70-100 KiB of weights in flight per SM.
  const bool i4 = f == KFL_INT4_G64;
  p->ctas_per_sm = env_int("KFL_GEMV_CTAS_PER_SM", 2);
  if (p->ctas_per_sm < 1 || p->ctas_per_sm > 2) p->ctas_per_sm = 2;
  p->stages = env_int("KFL_GEMV_STAGES", i4 ? 8 : 5);
  if (p->stages < 2 || p->stages > 13) p->stages = i4 ? 8 : 5;
  p->gemv_grid_max = n_sm * p->ctas_per_sm;
  // bf16 GEMVs of 2 x SMs to 4096 tiles (the 7B Q/K/V and O: 28 tiles per row block) run one
  // CTA per SM with 6 stages: half the CTAs share each row block, so their combine ends sooner
  // (7B b=1: -1.4% per step); int4 ones keep two CTAs per SM, which their decoding needs, and
  // GEMVs of fewer tiles keep one tile per CTA
  p->small_gemv_tiles = env_int("KFL_SMALL_GEMV_TILES", i4 ? 0 : 4096);
  p->small_gemv_stages = env_int("KFL_SMALL_GEMV_STAGES", 6);
  p->cluster = env_int("KFL_GEMV_CLUSTER", 3);
  if (p->cluster > MAX_CLUSTER) p->cluster = MAX_CLUSTER;
  int nrb = 1;
  if (p->nl > 0) {
    nrb = p->qkv.n_rb;
    if (p->o.n_rb > nrb) nrb = p->o.n_rb;
    if (p->gu.n_rb > nrb) nrb = p->gu.n_rb;
    if (p->down.n_rb > nrb) nrb = p->down.n_rb;
  }
  if ((flags & KFL_LOGITS_OUT) && p->lm.n_rb > nrb) nrb = p->lm.n_rb;
  p->n_rb_max = nrb;
  p->n_parts = (p->d + RB - 1) / RB;
  // two attention CTAs fit an SM: about two units per SM over the step's actual contexts
  p->attn_units = n_sm * std::max(1, env_int("KFL_ATTN_UNITS_PER_SM", 2));
  p->attn_cluster_sub = env_int("KFL_ATTN_CLUSTER_SUB", 1 << 20);
  // a small O projection's CTAs launch once the attention CTAs have left their loop: earlier,
  // their weight prefetch (most of the matrix) delays the attention's own loads (7B b=1, 26 MB:
  // -2.7% per step; 72B int4, 36 MB: -0.7%); a larger one's prefetch is worth starting at once
  // (32B, 52 MB: +0.7% late; 72B bf16, 134 MB: +1.1%)
  p->attn_launch_at = env_int("KFL_ATTN_LAUNCH", 2);
  p->attn_late_max_mb = env_int("KFL_ATTN_LATE_MAX_MB", 48);
  // a bf16 down projection over few row blocks (every row block shared by four or more CTAs in
  // the stream-K split) runs as clusters of 3 or 4 CTAs per row block, which combine through
  // distributed shared memory instead of the ticket's partial sums in global memory (the last
  // arriver's loads, round trips of about a microsecond each while the next kernel streams):
  // 7B b=1 -2.2% per step (4), 32B -0.6% (3); clusters of 2 (72B bf16, int4) measured slower, as
  // did clusters of 5 (56 clusters of 5 do not all fit the SMs at once); some slots are left for
  // the packing of clusters into the GPCs
  {
    int N = std::min(4, (2 * n_sm - 32) / std::max(1, p->down.n_rb));
    if (f != KFL_BF16 || N < 3 || p->down.n_kt < N) N = 0;
    p->down_cluster = std::min(MAX_CLUSTER, env_int("KFL_DOWN_CLUSTER", N));
  }
  p->attn_nchunks_max = (c->max_ctx + 63) / 64;
  p->n_phases = 5 * p->nl + ((flags & KFL_LOGITS_OUT) ? 1 : 0);
  {
    const int kk = tile_k(f);
    int m = p->hkv;
    const int lens[3] = {p->d, p->qdim, p->F};
    for (int i = 0; i < 3; ++i) m = std::max(m, (lens[i] + kk - 1) / kk);
    p->ctr_stride = round_up(m + 2, 32);
  }

  size_t w = 0;
  if (p->nl > 0)
    w += (size_t)p->nl * (p->qkv.bytes + p->o.bytes + p->gu.bytes + p->down.bytes + 2 * (size_t)p->d * 4 +
                          (c->qk_norm ? 2 * (size_t)p->hd * 4 : 0));
  if (flags & KFL_EMBED_IN) w += (size_t)p->V * p->d * 2;
  if (flags & KFL_LOGITS_OUT) w += p->lm.bytes + (size_t)p->d * 4;
  p->bytes_weights = w;
  p->bytes_kv = 2 * (size_t)p->nl * p->kv_elems_per_layer * 2;
  size_t ws = 0;
  ws += (size_t)c->max_ctx * (p->hd / 2) * 4 * 2;                      // rope tables
  ws += (size_t)MAXB * (2 * p->ldh + 2 * p->ldq + p->lda + p->ld_raw) * 4;  // h, xn, q, o, a, raw Q/K/V
  ws += act16_bytes(p->ldh, true) + act16_bytes(p->ldq, false) + act16_bytes(p->lda, false);  // int4 inputs
  ws += (size_t)p->n_parts * MAXB * 4;                                 // sum of squares
  ws += 3 * MAXB * 4;                                                  // positions, KV slots, next ids
  ws += (size_t)4 * p->gemv_grid_max * 2 * RB * MAXB * 4;              // stream-K partials (x4)
  ws += (size_t)(4 * p->n_rb_max + 1) * 4;                             // tickets (x4) + argmax ticket
  ws += (size_t)std::max(1, p->n_phases) * p->ctr_stride * 4;          // readiness counters
  ws += (size_t)p->n_rb_max * MAXB * 8;                                // argmax candidates
  ws += (size_t)MAXB * p->hkv * p->attn_nchunks_max * 8 * (p->hd + 4) * 4;  // attention partials
  ws += (size_t)MAXB * p->hkv * 4;                                     // attention tickets
  ws += 16;                                                            // error word
  ws += (size_t)MAXB * (2 + p->d) * 4;                                 // host-decode staging
  ws += 16;                                                            // grid barrier
  p->bytes_ws = ws;
}

}  // namespace

struct kfl_stage {
  kfl_model_cfg cfg;
  int l0 = 0, l1 = 0, flags = 0;
  int dev = 0;
  Plan P;
  std::vector<LayerDev> layers;
  Mat lm;
  uint16_t *embed = nullptr;
  float *g_final = nullptr;
  bool head_loaded = false;
  uint16_t *kc = nullptr, *vc = nullptr;
  float *rope_cos = nullptr, *rope_sin = nullptr;
  float *h = nullptr, *xn = nullptr, *q = nullptr, *o = nullptr, *a = nullptr, *sumsq = nullptr;
  float *qk_raw = nullptr;  // QK-norm stages: the Q/K/V projection before the norm and RoPE
  // int4 stages: the GEMV inputs in the tensor cores' fp16 form (xn with its rests, for Q/K/V)
  Act16 xn16 = {}, a16 = {}, o16 = {};
  int *pos = nullptr, *next_int = nullptr;
  int *slots = nullptr;  // [MAXB] KV-cache user slot of each batch row (this step)
  int *io_pos = nullptr, *io_ids = nullptr;  // host-buffer decode staging
  float *io_hin = nullptr;
  float *gemv_partial = nullptr;
  int *tickets = nullptr, *am_ticket = nullptr;
  float *cand_val = nullptr;
  int *cand_idx = nullptr;
  float *attn_partial = nullptr;
  int *attn_tickets = nullptr;
  unsigned *counters = nullptr;  // persistent kernel readiness counters [n_phases][ctr_stride]
  unsigned *err = nullptr;
  float *capture = nullptr;
  unsigned long long *trace = nullptr;
  std::vector<void *> allocs;
  int alloc_count = 0, fault_at = 0;
  cudaStream_t cap_stream = nullptr;
  int smem_optin = 0;  // shared memory a block may opt in to
  cudaGraphExec_t graph[MAXB + 1] = {};
  // persistent stage kernel
  bool persistent = true;
  int mk_stages[MAXB + 1] = {};
  size_t mk_smem[MAXB + 1] = {};
  unsigned *bar = nullptr;  // [0] grid-barrier counter, [1] abort flag
  Phase *phases_dev[MAXB + 1] = {};
  int n_phases = 0;
  bool profile = false;
  std::vector<cudaEvent_t> ev;
  double prof_ms[KFL_KERNEL_KINDS] = {};
  int64_t prof_n[KFL_KERNEL_KINDS] = {};
  // dense prefill (bf16 stages): the workspace of one pass of up to pf_cap tokens, allocated at
  // the first dense prefill, and the tensor maps of the weight tiles (per layer: Q/K/V, O,
  // gate/up, down; then lm_head)
  int pf_cap = 0;
  float *pf_h = nullptr;
  uint16_t *pf_q = nullptr;
  uint16_t *pf_x[2] = {}, *pf_o[2] = {}, *pf_a[2] = {};  // GEMM inputs as hi and lo bf16 terms
  int *pf_pos = nullptr, *pf_aidx = nullptr;
  float *pf_amax = nullptr;
  std::vector<void *> pf_allocs;
  // bf16 stages: the maps of every layer's weight tiles [4 l + j] (Q/K/V, O, gate/up, down), then
  // lm_head.  int4 stages: one map per matrix kind [j] (then lm_head) over pf_w16, the fp16 tiles
  // of the matrix being multiplied (dequantized just before its GEMM)
  std::vector<CUtensorMap> pf_maps;  // int4: [buffer * 5 + kind]
  std::vector<CUtensorMap> kv_maps;  // attention clusters: layer l's K cache [2 l] and V cache [2 l + 1]
  uint16_t *pf_w16[2] = {};
  // int4: matrix g + 1 of a pass is dequantized on pf_side into buffer (g + 1) % 2 while GEMM g
  // reads buffer g % 2; pf_deq[b] marks a buffer filled, pf_used[b] its GEMM done
  cudaStream_t pf_side = nullptr;
  cudaEvent_t pf_deq[2] = {}, pf_used[2] = {};
  int pf_seq = 0;  // GEMMs of the current pass issued so far
  int magic = 0x4B464C53;

  int alloc(void **p, size_t bytes) {
    ++alloc_count;
    if (fault_at > 0 && alloc_count == fault_at) return KFL_ERR_OOM;
    if (bytes == 0) bytes = 16;
    if (cudaMalloc(p, bytes) != cudaSuccess) {
      cudaGetLastError();
      *p = nullptr;
      return KFL_ERR_OOM;
    }
    allocs.push_back(*p);
    return KFL_OK;
  }
  bool loaded() const {
    for (const auto &l : layers)
      if (!l.loaded) return false;
    if ((flags & (KFL_EMBED_IN | KFL_LOGITS_OUT)) && !head_loaded) return false;
    return true;
  }
  void drop_graphs() {
    for (auto &g : graph)
      if (g) {
        cudaGraphExecDestroy(g);
        g = nullptr;
      }
    for (auto &p : phases_dev)
      if (p) {
        cudaFree(p);
        p = nullptr;
      }
  }
};

namespace {

bool valid(const kfl_stage *st) { return st && st->magic == 0x4B464C53; }

thread_local char g_last_error[512] = "";

int record_cuda_error(cudaError_t e, const char *what, int line) {
  snprintf(g_last_error, sizeof(g_last_error), "%s (%s) at stage.cu:%d", cudaGetErrorString(e), what, line);
  cudaGetLastError();
  return KFL_ERR_CUDA;
}

#define CK(x)                                                   \
  do {                                                          \
    cudaError_t _e = (x);                                       \
    if (_e != cudaSuccess) return record_cuda_error(_e, #x, __LINE__); \
  } while (0)


GemvParams base_gemv(kfl_stage *st, const Mat &m, const float *x, int ldx, int batch) {
  GemvParams g = {};
  g.w = m.tiles;
  g.fmt = m.fmt;
  g.n_rows = m.N;
  g.n_rb = m.n_rb;
  g.n_kt = m.n_kt;
  g.tile_bytes = m.fmt == KFL_BF16 ? TILE_BYTES : TILE4_BYTES;
  g.kt = m.fmt == KFL_BF16 ? KT : KT4;
  g.x = x;
  g.ldx = ldx;
  g.batch = batch;
  g.stages = ring_depth(m.fmt, std::min(st->P.stages, gemv_stages_for(batch, m.fmt, 1, st->P.ctas_per_sm)));
  g.rope_per_user = 0;
  g.partial = st->gemv_partial;
  g.tickets = st->tickets;
  g.err = st->err;
  return g;
}


// The phases of one decode step of the stage at this batch size: for every block Q/K/V (+RoPE,
// KV append), attention, O (+residual), gate/up (+SwiGLU), down (+residual); then lm_head
// (+argmax) for the head.  Both execution modes run exactly these.
std::vector<Phase> build_phases(kfl_stage *st, int batch, bool dataflow = false) {
  const Plan &P = st->P;
  const kfl_model_cfg &c = st->cfg;
  const bool i4 = c.weight_fmt == KFL_INT4_G64;
  std::vector<Phase> ph;
  auto gemv = [&](int epi, const GemvParams &g) {
    Phase x = {};
    x.kind = PH_GEMV;
    x.epi = epi;
    x.g = g;
    // stream-K partials and tickets rotate over four buffers, so a phase never reuses those
    // of the three before it (in the persistent kernel phases overlap)
    const int r = (int)ph.size() % 4;
    x.g.partial = st->gemv_partial + (size_t)r * P.gemv_grid_max * 2 * RB * MAXB;
    // int4: the Q/K/V projection carries its activations as an fp16 pair (its errors are
    // amplified by the attention softmax)
    x.g.xsplit = (g.fmt == KFL_INT4_G64 && epi == EPI_QKV) ? 1 : 0;
    x.g.tickets = st->tickets + (size_t)r * P.n_rb_max;
    ph.push_back(x);
  };
  for (int l = 0; l < P.nl; ++l) {
    const LayerDev &L = st->layers[l];
    uint16_t *kcl = st->kc + (size_t)l * P.kv_elems_per_layer;
    uint16_t *vcl = st->vc + (size_t)l * P.kv_elems_per_layer;
    {
      GemvParams g = base_gemv(st, L.qkv, st->xn, P.ldh, batch);
      g.sumsq = st->sumsq;
      g.n_parts = P.n_parts;
      g.d_norm = P.d;
      g.eps = c.rms_eps;
      g.q = st->q;
      g.kcache = kcl;
      g.vcache = vcl;
      g.positions = st->pos;
      g.slots = st->slots;
      g.rope_cos = st->rope_cos;
      g.rope_sin = st->rope_sin;
      g.n_q_rows = P.qdim;
      g.n_kv_rows = P.kvdim;
      g.head_dim = P.hd;
      g.max_ctx = c.max_ctx;
      g.n_kv_heads = P.hkv;
      if (c.qk_norm) {
        g.qk_raw = st->qk_raw;
        g.ld_raw = P.ld_raw;
      }
      if (i4) g.xin = st->xn16;
      gemv(EPI_QKV, g);
    }
    {
      Phase x = {};
      x.kind = PH_ATTN;
      AttnParams &a = x.a;
      a.q = st->q;
      a.kcache = kcl;
      a.vcache = vcl;
      a.positions = st->pos;
      a.slots = st->slots;
      a.o = st->o;
      a.ldo = P.ldq;
      if (i4) a.o16 = st->o16;
      a.partial = st->attn_partial;
      a.tickets = st->attn_tickets;
      a.batch = batch;
      a.n_heads = P.hq;
      a.n_kv_heads = P.hkv;
      a.max_ctx = c.max_ctx;
      a.chunk = std::max(1, env_int("KFL_ATTN_MIN_CHUNK", 64) / 64) * 64;  // the kernels size the step's chunks from its positions (at least this)
      a.n_chunks = (c.max_ctx + 63) / 64;
      a.target_units = P.attn_units;
      if (!dataflow && P.attn_cluster_max >= 2) {
        // one cluster per (user, KV head): the largest power of two up to the maximum with at
        // most as many CTAs as fit the SMs at once (power-of-two clusters and two or three
        // CTAs per SM measured fastest; clusters sized to fill the SMs exactly and one CTA per SM
        // with a deeper ring were slower)
        int cl = 1;
        while (cl * 2 <= P.attn_cluster_max) cl *= 2;
        const long long slots = (long long)P.n_sm * (P.attn_stages <= 2 ? 3 : 2);
        while (cl > 2 && (long long)cl * batch * P.hkv > slots) cl >>= 1;
        a.stages = P.attn_stages;
        a.launch_at = P.o.bytes <= (size_t)P.attn_late_max_mb << 20 ? P.attn_launch_at : 0;
        // the clusters cannot balance ragged users or spread a long context over idle SMs, but
        // their CTAs stream without block barriers: they are taken unless a CTA would have more
        // than KFL_ATTN_CLUSTER_SUB 64-position sub-tiles at the longest context while the
        // clusters leave SMs idle (by default always: measured no slower than the unit kernel
        // on every workload, 72B int4 b=1 20.0 against 22.4 us per block)
        const int per_cta = (c.max_ctx + cl - 1) / cl;
        if (per_cta <= P.attn_cluster_sub * 64 || (long long)cl * batch * P.hkv >= P.n_sm) a.cluster = cl;
      }
      a.scale_log2 = (float)(1.4426950408889634 / std::sqrt((double)P.hd));
      a.err = st->err;
      if (c.qk_norm) {
        QkNormParams &n = x.qn;
        n.raw = st->qk_raw;
        n.ld_raw = P.ld_raw;
        n.g_q = L.g_q;
        n.g_k = L.g_k;
        n.q = st->q;
        n.kcache = kcl;
        n.vcache = vcl;
        n.positions = st->pos;
        n.slots = st->slots;
        n.rope_cos = st->rope_cos;
        n.rope_sin = st->rope_sin;
        n.batch = batch;
        n.n_heads = P.hq;
        n.n_kv_heads = P.hkv;
        n.head_dim = P.hd;
        n.max_ctx = c.max_ctx;
        n.eps = c.rms_eps;
      }
      ph.push_back(x);
    }
    {
      GemvParams g = base_gemv(st, L.o, st->o, P.ldq, batch);
      g.h = st->h;
      g.ldh = P.ldh;
      g.xn = st->xn;
      g.g_next = L.g_ffn;
      g.sumsq_out = st->sumsq;
      if (i4) {
        g.xin = st->o16;
        g.xout = st->xn16;
      }
      gemv(EPI_RESID, g);
    }
    {
      GemvParams g = base_gemv(st, L.gu, st->xn, P.ldh, batch);
      g.sumsq = st->sumsq;
      g.n_parts = P.n_parts;
      g.d_norm = P.d;
      g.eps = c.rms_eps;
      g.out = st->a;
      g.ldo = P.lda;
      if (i4) {
        g.xin = st->xn16;
        g.xout = st->a16;
      }
      gemv(EPI_SWIGLU, g);
    }
    {
      GemvParams g = base_gemv(st, L.down, st->a, P.lda, batch);
      g.h = st->h;
      g.ldh = P.ldh;
      g.xn = st->xn;
      g.g_next = (l + 1 < P.nl) ? st->layers[l + 1].g_attn : ((st->flags & KFL_LOGITS_OUT) ? st->g_final : nullptr);
      g.sumsq_out = st->sumsq;
      g.capture = st->capture ? st->capture + (size_t)l * c.max_batch * P.d : nullptr;
      if (i4) {
        g.xin = st->a16;
        g.xout = st->xn16;
      }
      gemv(EPI_RESID, g);
    }
  }
  if (st->flags & KFL_LOGITS_OUT) {
    GemvParams g = base_gemv(st, st->lm, st->xn, P.ldh, batch);
    g.sumsq = st->sumsq;
    g.n_parts = P.n_parts;
    g.d_norm = P.d;
    g.eps = c.rms_eps;
    g.cand_val = st->cand_val;
    g.cand_idx = st->cand_idx;
    g.argmax_ticket = st->am_ticket;
    g.next_ids = st->next_int;
    if (i4) g.xin = st->xn16;
    gemv(EPI_ARGMAX, g);
  }
  if (!dataflow && st->trace) {
    // one kernel per phase: each launch stamps its own slice of the trace
    const int tg = std::max(P.n_sm, P.gemv_grid_max);
    for (size_t k = 0; k < ph.size(); ++k) {
      unsigned long long *slice = st->trace + k * (size_t)tg * TRACE_SLOTS;
      if (ph[k].kind == PH_GEMV) {
        ph[k].g.trace = slice;
      } else {
        ph[k].a.trace = slice;
        ph[k].a.trace_grid = tg;
      }
    }
  }
  if (dataflow) {
    // readiness counters: phase k publishes in region k, the phase after it reads region k
    const int kk = tile_k(c.weight_fmt);
    const int G = P.hq / P.hkv;
    auto region = [&](int k) { return st->counters + (size_t)k * P.ctr_stride; };
    auto done = [&](int k) { return st->counters + (size_t)k * P.ctr_stride + P.ctr_stride - 1; };
    const int rb_d = (P.d + RB - 1) / RB;
    for (size_t k = 0; k < ph.size(); ++k) {
      Phase &x = ph[k];
      const bool lm = (int)k == 5 * P.nl;
      const int j = lm ? 5 : (int)(k % 5);  // 0 QKV, 1 attention, 2 O, 3 gate/up, 4 down, 5 lm_head
      if (x.kind == PH_ATTN) {
        x.a.in_ready = region((int)k - 1);
        x.a.in_need = (G + 2) * P.hd / RB;
        x.a.out_ready = region((int)k);
        continue;
      }
      GemvParams &g = x.g;
      if (j == 0 || j == 5) {  // input xn and the norm of h from the previous down (or none)
        if (k > 0) {
          g.in_kind = 1;
          g.in_ready = region((int)k - 1);
          g.in_len = P.d;
          g.in_unit = RB;
          g.norm_done = done((int)k - 1);
          g.norm_need = rb_d;
        }
      } else if (j == 2) {  // attention output o
        g.in_kind = 2;
        g.in_ready = region((int)k - 1);
        g.in_len = P.qdim;
        g.in_group = G;
        g.in_head_dim = P.hd;
        g.in_need = batch;
      } else if (j == 3) {  // xn and the norm of h from O
        g.in_kind = 1;
        g.in_ready = region((int)k - 1);
        g.in_len = P.d;
        g.in_unit = RB;
        g.norm_done = done((int)k - 1);
        g.norm_need = rb_d;
      } else if (j == 4) {  // a from gate/up
        g.in_kind = 1;
        g.in_ready = region((int)k - 1);
        g.in_len = P.F;
        g.in_unit = RB / 2;
      }
      if (j != 5) {
        g.out_ready = region((int)k);
        g.out_done = done((int)k);
        g.out_unit = (j == 3) ? RB / 2 : RB;
        g.out_kt = kk;
      }
    }
  }
  return ph;
}

// Kernel kind of phase i of a step (phases come in blocks of five, then lm_head).
int phase_kind_code(const Phase &ph, size_t i) {
  if (ph.kind == PH_ATTN) return KFL_KERNEL_ATTN;
  switch (ph.epi) {
    case EPI_QKV: return KFL_KERNEL_QKV;
    case EPI_SWIGLU: return KFL_KERNEL_GATEUP;
    case EPI_ARGMAX: return KFL_KERNEL_LMHEAD;
    default: return (i % 5 == 2) ? KFL_KERNEL_OPROJ : KFL_KERNEL_DOWN;
  }
}

// The launch shape of a GEMV phase in the one-kernel-per-phase mode: sets g's ring depth and
// cluster size and returns its grid.  Every shape is a stream-K split: CTA c streams tiles
// [c T / G, (c + 1) T / G) (a cluster of N CTAs per row block is the split with G = N n_rb).
int gemv_launch_shape(const kfl_stage *st, int batch, GemvParams &g, int big_cluster = 0) {
  const long long T = (long long)g.n_rb * g.n_kt;
  int grid = (int)(T < st->P.gemv_grid_max ? T : st->P.gemv_grid_max);
  if (big_cluster >= 2 && g.n_kt >= big_cluster && (long long)big_cluster * g.n_rb <= 2LL * st->P.n_sm &&
      st->P.ctas_per_sm > 1 && T > st->P.small_gemv_tiles) {
    const int N = big_cluster;
    const int per_sm = N * g.n_rb <= st->P.n_sm ? 1 : 2;
    g.cluster = N;
    g.stages = ring_depth(g.fmt, std::min(st->P.stages, gemv_stages_for(batch, g.fmt, N, per_sm)));
    return N * g.n_rb;
  }
  if (T <= st->P.small_gemv_tiles && T >= 2LL * st->P.n_sm && st->P.ctas_per_sm > 1) {
    // a small GEMV: one CTA per SM with a deeper ring, so that fewer CTAs share a row block;
    // with few enough row blocks, clusters of N CTAs split each one's K range and combine
    // through distributed shared memory (N row blocks' worth of CTAs at one or two per SM)
    grid = (int)(T < st->P.n_sm ? T : st->P.n_sm);
    g.stages = ring_depth(g.fmt, std::min(st->P.small_gemv_stages, gemv_max_stages(batch, g.fmt, st->smem_optin)));
    const int N = st->P.cluster;
    if (N >= 2 && g.n_kt >= N && (long long)N * g.n_rb <= 2LL * st->P.n_sm) {
      const int per_sm = N * g.n_rb <= st->P.n_sm ? 1 : 2;
      grid = N * g.n_rb;
      g.cluster = N;
      g.stages = ring_depth(g.fmt, std::min(st->P.small_gemv_stages, gemv_stages_for(batch, g.fmt, N, per_sm)));
    }
  }
  return grid;
}

// Per-kernel mode: one launch per phase on stream s (chained with PDL when pdl is set).  With
// `kinds` (profiling, no PDL) the k-th launch is bracketed by events ev[2(ev_base+k)] and
// ev[2(ev_base+k)+1] and its kind appended to *kinds.
int enqueue_body(kfl_stage *st, int batch, cudaStream_t s, bool pdl, std::vector<int> *kinds, int ev_base) {
  const std::vector<Phase> phases = build_phases(st, batch);
  int k = ev_base;
  for (size_t i = 0; i < phases.size(); ++i) {
    const Phase &ph = phases[i];
    if (kinds) {
      CK(cudaEventRecord(st->ev[2 * k], s));
      kinds->push_back(phase_kind_code(ph, i));
    }
    if (ph.kind == PH_GEMV) {
      GemvParams g = ph.g;
      const int grid = gemv_launch_shape(st, batch, g, i % 5 == 4 ? st->P.down_cluster : 0);
      CK(launch_gemv(g, ph.epi, grid, s, pdl));
    } else {
      if (ph.qn.raw) CK(launch_qknorm(ph.qn, s, pdl));  // QK-norm stages: norm, RoPE, KV append
      if (ph.a.cluster > 0)  // phases come five per block: Q/K/V, attention, O, gate/up, down
        CK(launch_attention_cluster(ph.a, st->kv_maps[2 * (i / 5)], st->kv_maps[2 * (i / 5) + 1], st->P.hd, s, pdl));
      else
        CK(launch_attention(ph.a, st->P.hd, s, pdl));
    }
    if (kinds) CK(cudaEventRecord(st->ev[2 * k + 1], s));
    ++k;
  }
  return KFL_OK;
}

// Persistent mode: the phase table of this batch size, uploaded once (outside any capture).
int upload_phases(kfl_stage *st, int batch) {
  if (st->phases_dev[batch]) return KFL_OK;
  const std::vector<Phase> phases = build_phases(st, batch, true);
  void *d = nullptr;
  if (cudaMalloc(&d, phases.size() * sizeof(Phase)) != cudaSuccess) {
    cudaGetLastError();
    return KFL_ERR_OOM;
  }
  st->phases_dev[batch] = static_cast<Phase *>(d);
  st->n_phases = (int)phases.size();
  CK(cudaMemcpy(d, phases.data(), phases.size() * sizeof(Phase), cudaMemcpyHostToDevice));
  return KFL_OK;
}

// Persistent mode: the whole step as one cooperative launch of the stage kernel.
int enqueue_persistent(kfl_stage *st, int batch, cudaStream_t s) {
  StageKernelParams kp = {};
  kp.phases = st->phases_dev[batch];
  kp.n_phases = st->n_phases;
  kp.stages = st->mk_stages[batch];
  kp.head_dim = st->P.hd;
  kp.attn_bytes = stage_kernel_attn_bytes(st->P.hd);
  kp.bar = st->bar;
  kp.abort_flag = reinterpret_cast<int *>(st->bar + 1);
  kp.err = st->err;
  kp.trace = st->trace;
  kp.positions = st->pos;
  kp.rope_cos = st->rope_cos;
  kp.rope_sin = st->rope_sin;
  kp.max_ctx = st->cfg.max_ctx;
  kp.l2_ahead = env_int("KFL_L2_AHEAD", 0);
  CK(cudaMemsetAsync(st->counters, 0, (size_t)std::max(1, st->n_phases) * st->P.ctr_stride * 4, s));
  CK(launch_stage_kernel(kp, batch, st->cfg.weight_fmt, st->P.n_sm, st->mk_smem[batch], s));
  return KFL_OK;
}

int ensure_graph(kfl_stage *st, int batch) {
  if (st->graph[batch]) return KFL_OK;
  if (!st->cap_stream) CK(cudaStreamCreateWithFlags(&st->cap_stream, cudaStreamNonBlocking));
  if (st->persistent) {
    int rc = upload_phases(st, batch);
    if (rc != KFL_OK) return rc;
  }
  cudaGraph_t g = nullptr;
  CK(cudaStreamBeginCapture(st->cap_stream, cudaStreamCaptureModeThreadLocal));
  int rc = st->persistent ? enqueue_persistent(st, batch, st->cap_stream)
                          : enqueue_body(st, batch, st->cap_stream, true, nullptr, 0);
  cudaError_t e = cudaStreamEndCapture(st->cap_stream, &g);
  if (rc != KFL_OK || e != cudaSuccess) {
    if (g) cudaGraphDestroy(g);
    cudaGetLastError();
    return rc != KFL_OK ? rc : KFL_ERR_CUDA;
  }
  e = cudaGraphInstantiate(&st->graph[batch], g, 0);
  cudaGraphDestroy(g);
  if (e != cudaSuccess) {
    st->graph[batch] = nullptr;
    cudaGetLastError();
    return KFL_ERR_CUDA;
  }
  return KFL_OK;
}

const float *input_g_next(const kfl_stage *st) {
  if (st->P.nl > 0) return st->layers[0].g_attn;
  if (st->flags & KFL_LOGITS_OUT) return st->g_final;
  return nullptr;
}

// One step over `batch` rows.  Row b's KV slot: users[b] (device) when users is non-NULL, else
// user_all for every row when user_all >= 0, else b.
int run_step(kfl_stage *st, const int32_t *ids, const float *hidden_in, const int32_t *positions,
             const int32_t *users, int user_all, int batch, float *hidden_out, int32_t *next_ids,
             cudaStream_t s) {
  const Plan &P = st->P;
  const bool embed = (st->flags & KFL_EMBED_IN) != 0;
  const bool body = P.nl > 0 || (st->flags & KFL_LOGITS_OUT);
  if (st->profile) {
    const int n_k = 2 + (int)build_phases(st, batch).size();
    while ((int)st->ev.size() < 2 * n_k) {
      cudaEvent_t e;
      CK(cudaEventCreate(&e));
      st->ev.push_back(e);
    }
    std::vector<int> kinds;
    CK(cudaEventRecord(st->ev[0], s));
    CK(launch_stage_input(ids, hidden_in, positions, batch, embed ? st->embed : nullptr, P.V, P.d, P.ldh,
                          input_g_next(st), st->h, st->xn, st->sumsq, st->pos, st->cfg.max_ctx, st->err, st->bar,
                          st->cfg.weight_fmt == KFL_INT4_G64 ? st->xn16 : Act16{}, users, user_all,
                          st->cfg.max_batch, st->slots, s));
    CK(cudaEventRecord(st->ev[1], s));
    kinds.push_back(KFL_KERNEL_INPUT);
    int rc = enqueue_body(st, batch, s, false, &kinds, 1);
    if (rc != KFL_OK) return rc;
    const int ko = (int)kinds.size();
    CK(cudaEventRecord(st->ev[2 * ko], s));
    CK(launch_stage_output(st->h, P.ldh, P.d, batch, hidden_out, st->next_int, next_ids, s, false));
    CK(cudaEventRecord(st->ev[2 * ko + 1], s));
    kinds.push_back(KFL_KERNEL_OUTPUT);
    CK(cudaEventSynchronize(st->ev[2 * ko + 1]));
    for (size_t k = 0; k < kinds.size(); ++k) {
      float ms = 0.f;
      CK(cudaEventElapsedTime(&ms, st->ev[2 * k], st->ev[2 * k + 1]));
      st->prof_ms[kinds[k]] += ms;
      st->prof_n[kinds[k]] += 1;
    }
    return KFL_OK;
  }
  CK(launch_stage_input(ids, hidden_in, positions, batch, embed ? st->embed : nullptr, P.V, P.d, P.ldh,
                        input_g_next(st), st->h, st->xn, st->sumsq, st->pos, st->cfg.max_ctx, st->err, st->bar,
                        st->cfg.weight_fmt == KFL_INT4_G64 ? st->xn16 : Act16{}, users, user_all,
                        st->cfg.max_batch, st->slots, s));
  if (body) {
    int rc = ensure_graph(st, batch);
    if (rc != KFL_OK) return rc;
    CK(cudaGraphLaunch(st->graph[batch], s));
  }
  CK(launch_stage_output(st->h, P.ldh, P.d, batch, hidden_out, st->next_int, next_ids, s, false));
  return KFL_OK;
}

// ---- dense prefill (bf16 weights) ---------------------------------------------------------
constexpr int PF_PASS = 2048;  // tokens per pass of the dense prefill

int pf_ld(int n) { return round_up(n, 64); }

// Workspace for passes of up to `tokens` tokens (grown, never shrunk) and the weight maps.
int ensure_prefill(kfl_stage *st, int tokens) {
  const Plan &P = st->P;
  const int cap = std::min(PF_PASS, round_up(tokens, PG_M));
  if (cap > st->pf_cap) {
    for (void *p : st->pf_allocs) cudaFree(p);
    st->pf_allocs.clear();
    st->pf_cap = 0;
    auto get = [&](void **p, size_t bytes) {
      if (cudaMalloc(p, bytes) != cudaSuccess) {
        cudaGetLastError();
        return false;
      }
      st->pf_allocs.push_back(*p);
      return true;
    };
    const int n_tiles = (P.V + PG_N - 1) / PG_N;
    bool ok = get((void **)&st->pf_h, (size_t)cap * P.ldh * 4) && get((void **)&st->pf_q, (size_t)cap * pf_ld(P.qdim) * 2);
    for (int j = 0; j < 2; ++j)
      ok = ok && get((void **)&st->pf_x[j], (size_t)cap * pf_ld(P.d) * 2) &&
           get((void **)&st->pf_o[j], (size_t)cap * pf_ld(P.qdim) * 2) &&
           get((void **)&st->pf_a[j], (size_t)cap * pf_ld(P.F) * 2);
    if (!ok || !get((void **)&st->pf_pos, (size_t)cap * 4) ||
        !get((void **)&st->pf_amax, (size_t)cap * n_tiles * 4) ||
        !get((void **)&st->pf_aidx, (size_t)cap * n_tiles * 4))
      return KFL_ERR_OOM;
    st->pf_cap = cap;
  }
  if (st->pf_maps.empty() && st->cfg.weight_fmt == KFL_INT4_G64) {
    // the fp16 scratch holds the largest matrix; its maps are per matrix kind
    const Mat *kinds[5] = {&P.qkv, &P.o, &P.gu, &P.down, &P.lm};
    const int n_kinds = (st->flags & KFL_LOGITS_OUT) ? 5 : 4;
    size_t most = 0;
    for (int j = 0; j < n_kinds; ++j) most = std::max(most, (size_t)kinds[j]->n_rb * 2 * kinds[j]->n_kt * TILE_BYTES);
    // each resource is made once (a call that failed part way keeps what it made, and the next
    // call completes the set; kfl_stage_destroy frees them)
    for (int b = 0; b < 2; ++b) {
      if (!st->pf_w16[b] && cudaMalloc((void **)&st->pf_w16[b], most) != cudaSuccess) {
        cudaGetLastError();
        st->pf_w16[b] = nullptr;
        return KFL_ERR_OOM;
      }
      if ((!st->pf_deq[b] && cudaEventCreateWithFlags(&st->pf_deq[b], cudaEventDisableTiming) != cudaSuccess) ||
          (!st->pf_used[b] && cudaEventCreateWithFlags(&st->pf_used[b], cudaEventDisableTiming) != cudaSuccess)) {
        cudaGetLastError();
        return KFL_ERR_CUDA;
      }
    }
    if (!st->pf_side && cudaStreamCreateWithFlags(&st->pf_side, cudaStreamNonBlocking) != cudaSuccess) {
      cudaGetLastError();
      st->pf_side = nullptr;
      return KFL_ERR_CUDA;
    }
    std::vector<CUtensorMap> maps(10);
    for (int b = 0; b < 2; ++b)
      for (int j = 0; j < n_kinds; ++j)
        if (encode_tiles_map(&maps[b * 5 + j], reinterpret_cast<const uint8_t *>(st->pf_w16[b]), 2 * kinds[j]->n_kt,
                             kinds[j]->n_rb))
          return KFL_ERR_CUDA;
    st->pf_maps = std::move(maps);
  }
  if (st->pf_maps.empty()) {
    std::vector<CUtensorMap> maps(4 * P.nl + 1);
    for (int l = 0; l < P.nl; ++l) {
      const LayerDev &L = st->layers[l];
      const Mat *m[4] = {&L.qkv, &L.o, &L.gu, &L.down};
      for (int j = 0; j < 4; ++j)
        if (encode_tiles_map(&maps[4 * l + j], m[j]->tiles, m[j]->n_kt, m[j]->n_rb)) return KFL_ERR_CUDA;
    }
    if ((st->flags & KFL_LOGITS_OUT) && encode_tiles_map(&maps[4 * P.nl], st->lm.tiles, st->lm.n_kt, st->lm.n_rb))
      return KFL_ERR_CUDA;
    st->pf_maps = std::move(maps);
  }
  return KFL_OK;
}

// Matrix j of block l (j = 4: lm_head).
const Mat &pf_mat(const kfl_stage *st, int l, int j) {
  if (j == 4) return st->lm;
  const LayerDev &L = st->layers[l];
  return j == 0 ? L.qkv : j == 1 ? L.o : j == 2 ? L.gu : L.down;
}

// The g-th GEMM of a pass multiplies matrix (g / 4, g % 4) of the blocks, then (head) the lm_head.
bool pf_seq_matrix(const kfl_stage *st, int g, int *l, int *j) {
  if (g < 4 * st->P.nl) {
    *l = g / 4;
    *j = g % 4;
    return true;
  }
  if (g == 4 * st->P.nl && (st->flags & KFL_LOGITS_OUT)) {
    *l = -1;
    *j = 4;
    return true;
  }
  return false;
}

// int4: dequantize the g-th matrix of the pass into buffer g % 2 on the side stream, once the GEMM
// that last read that buffer (g - 2) is done.
cudaError_t pf_dequant(kfl_stage *st, int g) {
  int l, j;
  if (!pf_seq_matrix(st, g, &l, &j)) return cudaSuccess;
  const Mat &m = pf_mat(st, l, j);
  cudaError_t err = cudaStreamWaitEvent(st->pf_side, st->pf_used[g % 2], 0);
  if (err == cudaSuccess) err = launch_dequant_int4_f16(m.tiles, m.n_rb, m.n_kt, st->pf_w16[g % 2], st->pf_side);
  if (err == cudaSuccess) err = cudaEventRecord(st->pf_deq[g % 2], st->pf_side);
  return err;
}

// int4: start of a pass on stream s: both buffers free once s's earlier work is done; the first
// matrix is dequantized.
cudaError_t pf_pass_begin(kfl_stage *st, cudaStream_t s) {
  st->pf_seq = 0;
  if (st->cfg.weight_fmt != KFL_INT4_G64) return cudaSuccess;
  cudaError_t err = cudaEventRecord(st->pf_used[0], s);
  if (err == cudaSuccess) err = cudaEventRecord(st->pf_used[1], s);
  if (err == cudaSuccess) err = pf_dequant(st, 0);
  return err;
}

// One prefill GEMM with matrix j of block l (j = 4: lm_head) and the split count chosen for its
// shape.  int4 stages read the matrix's fp16 copy, dequantized ahead on the side stream (the
// next one is started before this GEMM, so dequantization overlaps the products).
cudaError_t pf_gemm(kfl_stage *st, int mode, const CUtensorMap &a, const CUtensorMap &a2, int l, int j,
                    PrefillEpiParams e, cudaStream_t s) {
  const Mat &m = pf_mat(st, l, j);
  const bool i4 = st->cfg.weight_fmt == KFL_INT4_G64;
  int n_kt = m.n_kt;
  const CUtensorMap *b;
  const int g = st->pf_seq++;
  if (i4) {
    cudaError_t err = pf_dequant(st, g + 1);
    if (err == cudaSuccess) err = cudaStreamWaitEvent(s, st->pf_deq[g % 2], 0);
    if (err != cudaSuccess) return err;
    b = &st->pf_maps[(g % 2) * 5 + j];
    n_kt = 2 * m.n_kt;  // K tiles of 128 fp16
  } else {
    b = &st->pf_maps[j == 4 ? 4 * st->P.nl : 4 * l + j];
  }
  e.f16 = i4 ? 1 : 0;
  e.splits = mode == PE_ARGMAX ? 1 : prefill_splits(e.T, e.N, n_kt, st->P.n_sm);
  cudaError_t err = launch_prefill_gemm(mode, a, a2, *b, n_kt, e, s);
  if (err == cudaSuccess && i4) err = cudaEventRecord(st->pf_used[g % 2], s);
  return err;
}

// The prompt in passes of up to pf_cap tokens.  Per pass and block: RMSNorm -> Q/K/V GEMM (RoPE,
// K/V appended to the user's slot) -> causal attention over the slot -> O GEMM + residual ->
// RMSNorm -> gate/up GEMM (SwiGLU) -> down GEMM + residual; the head: final RMSNorm -> lm_head GEMM
// with the greedy argmax.
int run_prefill_dense(kfl_stage *st, const int32_t *ids, const float *hidden_in, const int32_t *positions, int user,
                      int T, float *hidden_out, int32_t *next_ids, cudaStream_t s) {
  const Plan &P = st->P;
  int rc = ensure_prefill(st, T);
  if (rc != KFL_OK) return rc;
  const bool embed = (st->flags & KFL_EMBED_IN) != 0;
  const int i4 = st->cfg.weight_fmt == KFL_INT4_G64 ? 1 : 0;
  const int ldx = pf_ld(P.d), ldq = pf_ld(P.qdim), lda = pf_ld(P.F);
  const float eps = st->cfg.rms_eps;
  for (int t0 = 0; t0 < T; t0 += st->pf_cap) {
    const int n = std::min(st->pf_cap, T - t0);
    CK(launch_prefill_input(ids ? ids + t0 : nullptr, hidden_in ? hidden_in + (size_t)t0 * P.d : nullptr,
                            positions + t0, n, embed ? st->embed : nullptr, P.V, P.d, P.ldh, st->pf_h, st->pf_pos,
                            st->cfg.max_ctx, st->err, s));
    CK(pf_pass_begin(st, s));
    CUtensorMap mx[2], mo[2], ma[2];
    for (int j = 0; j < 2; ++j)
      if (encode_act_map(&mx[j], st->pf_x[j], P.d, n, ldx) || encode_act_map(&mo[j], st->pf_o[j], P.qdim, n, ldq) ||
          encode_act_map(&ma[j], st->pf_a[j], P.F, n, lda))
        return KFL_ERR_CUDA;
    for (int l = 0; l < P.nl; ++l) {
      const LayerDev &L = st->layers[l];
      uint16_t *kcl = st->kc + (size_t)l * P.kv_elems_per_layer;
      uint16_t *vcl = st->vc + (size_t)l * P.kv_elems_per_layer;
      CK(launch_prefill_rmsnorm(st->pf_h, P.ldh, n, P.d, L.g_attn, eps, st->pf_x[0], st->pf_x[1], ldx, i4, st->err, s));
      PrefillEpiParams e = {};
      e.T = n;
      e.err = st->err;
      e.N = L.qkv.N;
      e.out16 = st->pf_q;
      e.ldo16 = ldq;
      e.kcache = kcl;
      e.vcache = vcl;
      e.positions = st->pf_pos;
      e.slot = user;
      e.hd = P.hd;
      e.hkv = P.hkv;
      e.qdim = P.qdim;
      e.kvdim = P.kvdim;
      e.max_ctx = st->cfg.max_ctx;
      e.rope_cos = st->rope_cos;
      e.rope_sin = st->rope_sin;
      CK(pf_gemm(st, PE_QKV, mx[0], mx[1], l, 0, e, s));
      PrefillAttnParams a = {};
      a.q = st->pf_q;
      a.ldq = ldq;
      a.o = st->pf_o[0];
      a.o_lo = st->pf_o[1];
      a.ldo = ldq;
      a.f16 = i4;
      a.kcache = kcl;
      a.vcache = vcl;
      a.positions = st->pf_pos;
      a.slot = user;
      a.T = n;
      a.n_heads = P.hq;
      a.n_kv_heads = P.hkv;
      a.max_ctx = st->cfg.max_ctx;
      a.scale_log2 = (float)(1.4426950408889634 / std::sqrt((double)P.hd));
      a.err = st->err;
      CK(launch_prefill_attention(a, P.hd, s));
      PrefillEpiParams r = {};
      r.T = n;
      r.err = st->err;
      r.N = P.d;
      r.out = st->pf_h;
      r.ldo = P.ldh;
      CK(pf_gemm(st, PE_RESID, mo[0], mo[1], l, 1, r, s));
      CK(launch_prefill_rmsnorm(st->pf_h, P.ldh, n, P.d, L.g_ffn, eps, st->pf_x[0], st->pf_x[1], ldx, i4, st->err, s));
      PrefillEpiParams g = {};
      g.T = n;
      g.err = st->err;
      g.N = 2 * P.F;
      g.out16 = st->pf_a[0];
      g.out16lo = st->pf_a[1];
      g.ldo16 = lda;
      CK(pf_gemm(st, PE_SWIGLU, mx[0], mx[1], l, 2, g, s));
      CK(pf_gemm(st, PE_RESID, ma[0], ma[1], l, 3, r, s));
    }
    if (st->flags & KFL_LOGITS_OUT) {
      CK(launch_prefill_rmsnorm(st->pf_h, P.ldh, n, P.d, st->g_final, eps, st->pf_x[0], st->pf_x[1], ldx, i4, st->err, s));
      PrefillEpiParams z = {};
      z.T = n;
      z.err = st->err;
      z.N = P.V;
      z.amax = st->pf_amax;
      z.aidx = st->pf_aidx;
      z.n_tiles = (P.V + PG_N - 1) / PG_N;
      CK(pf_gemm(st, PE_ARGMAX, mx[0], mx[1], -1, 4, z, s));
      CK(launch_prefill_argmax(st->pf_amax, st->pf_aidx, z.n_tiles, n, next_ids + t0, s));
    }
    if (hidden_out)
      CK(cudaMemcpy2DAsync(hidden_out + (size_t)t0 * P.d, (size_t)P.d * 4, st->pf_h, (size_t)P.ldh * 4,
                           (size_t)P.d * 4, n, cudaMemcpyDeviceToDevice, s));
  }
  return KFL_OK;
}

// host or device source -> device pointer (a temporary copy for host sources)
int to_device(kfl_stage *st, const void *src, size_t bytes, int on_device, void **out, std::vector<void *> &tmp) {
  if (on_device) {
    *out = const_cast<void *>(src);
    return KFL_OK;
  }
  void *d = nullptr;
  if (cudaMalloc(&d, bytes ? bytes : 16) != cudaSuccess) {
    cudaGetLastError();
    return KFL_ERR_OOM;
  }
  tmp.push_back(d);
  CK(cudaMemcpy(d, src, bytes, cudaMemcpyHostToDevice));
  *out = d;
  return KFL_OK;
}

void free_tmp(std::vector<void *> &tmp) {
  for (void *p : tmp) cudaFree(p);
  tmp.clear();
}

int load_gain(kfl_stage *st, const uint16_t *src, int n, int on_device, float *dst, std::vector<void *> &tmp) {
  void *d = nullptr;
  int rc = to_device(st, src, (size_t)n * 2, on_device, &d, tmp);
  if (rc) return rc;
  CK(launch_bf16_to_f32(static_cast<const uint16_t *>(d), dst, n, nullptr));
  return KFL_OK;
}

// Concatenate matrices (rows stacked) into one device buffer and repack with an optional row
// map.  parts: (matrix, rows).  For int4 the words and scales are concatenated separately.
int load_matrix(kfl_stage *st, Mat &m, const std::vector<std::pair<const kfl_matrix *, int>> &parts, int K,
                const std::vector<int> &row_map, int on_device, std::vector<void *> &tmp) {
  const bool bf = m.fmt == KFL_BF16;
  int n_src = 0;
  for (auto &pp : parts) {
    if (!pp.first || !pp.first->w || (!bf && !pp.first->scales)) return KFL_ERR_ARG;
    n_src += pp.second;
  }
  const size_t row_w = bf ? (size_t)K * 2 : (size_t)K / 2;  // bytes of codes per row
  const size_t row_s = bf ? 0 : (size_t)(K / 64) * 2;
  void *wcat = nullptr, *scat = nullptr;
  if (parts.size() == 1 && on_device) {
    wcat = const_cast<void *>(parts[0].first->w);
    scat = const_cast<void *>(parts[0].first->scales);
  } else {
    if (cudaMalloc(&wcat, n_src * row_w) != cudaSuccess) {
      cudaGetLastError();
      return KFL_ERR_OOM;
    }
    tmp.push_back(wcat);
    if (!bf) {
      if (cudaMalloc(&scat, n_src * row_s) != cudaSuccess) {
        cudaGetLastError();
        return KFL_ERR_OOM;
      }
      tmp.push_back(scat);
    }
    size_t off = 0;
    for (auto &pp : parts) {
      CK(cudaMemcpy(static_cast<uint8_t *>(wcat) + off * row_w, pp.first->w, pp.second * row_w, cudaMemcpyDefault));
      if (!bf)
        CK(cudaMemcpy(static_cast<uint8_t *>(scat) + off * row_s, pp.first->scales, pp.second * row_s,
                      cudaMemcpyDefault));
      off += pp.second;
    }
  }
  int *dmap = nullptr;
  if (!row_map.empty()) {
    if (cudaMalloc(&dmap, row_map.size() * sizeof(int)) != cudaSuccess) {
      cudaGetLastError();
      return KFL_ERR_OOM;
    }
    tmp.push_back(dmap);
    CK(cudaMemcpy(dmap, row_map.data(), row_map.size() * sizeof(int), cudaMemcpyHostToDevice));
  }
  if (bf)
    CK(launch_repack_bf16(static_cast<const uint16_t *>(wcat), n_src, K, dmap, m.N, m.n_rb, m.n_kt, m.tiles,
                          nullptr));
  else
    CK(launch_repack_int4(static_cast<const uint32_t *>(wcat), static_cast<const uint16_t *>(scat), n_src, K, dmap,
                          m.N, m.n_rb, m.n_kt, m.tiles, nullptr));
  CK(cudaDeviceSynchronize());
  return KFL_OK;
}

}  // namespace

// ============================================================================ C ABI

extern "C" int kfl_stage_memory_bytes(const kfl_model_cfg *cfg, int l0, int l1, int flags, size_t *out) {
  if (!out) return KFL_ERR_ARG;
  int rc = validate_cfg(cfg, l0, l1, flags);
  if (rc) return rc;
  Plan P;
  int n_sm = 152;
  int dev = 0;
  if (cudaGetDevice(&dev) == cudaSuccess) {
    int v = 0;
    if (cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev) == cudaSuccess && v > 0) n_sm = v;
  }
  cudaGetLastError();
  make_plan(cfg, l0, l1, flags, n_sm, &P);
  *out = P.bytes_weights + P.bytes_kv + P.bytes_ws;
  return KFL_OK;
}

extern "C" int kfl_stage_create(const kfl_model_cfg *cfg, int l0, int l1, int flags, kfl_stage **out) {
  if (!out) return KFL_ERR_ARG;
  *out = nullptr;
  int rc = validate_cfg(cfg, l0, l1, flags);
  if (rc) return rc;
  int dev = 0, n_sm = 0;
  CK(cudaGetDevice(&dev));
  CK(cudaDeviceGetAttribute(&n_sm, cudaDevAttrMultiProcessorCount, dev));
  CK(prepare_gemv());
  CK(prepare_attention());
  CK(prepare_attention_cluster());
  int smem_optin = 0;
  CK(cudaDeviceGetAttribute(&smem_optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev));
  kfl_stage *st = new kfl_stage();
  st->cfg = *cfg;
  st->l0 = l0;
  st->l1 = l1;
  st->flags = flags;
  st->dev = dev;
  st->smem_optin = smem_optin;
  st->fault_at = env_int("KFL_FAULT_ALLOC_AT", 0);
  make_plan(cfg, l0, l1, flags, n_sm, &st->P);
  Plan &P = st->P;
  {
    const int want = env_int("KFL_ATTN_CLUSTER", MAX_CLUSTER_ATT);
    P.attn_stages = std::max(2, std::min(ATT_RING_MAX, env_int("KFL_ATTN_STAGES", 3)));
    P.attn_cluster_max = want >= 2 ? attention_cluster_size(P.hd, std::min(want, MAX_CLUSTER_ATT), P.attn_stages) : 0;
  }
  auto fail = [&](int code) {
    kfl_stage_destroy(st);
    return code;
  };
#define AL(ptr, bytes)                                                  \
  do {                                                                  \
    int _r = st->alloc(reinterpret_cast<void **>(&(ptr)), (bytes));     \
    if (_r) return fail(_r);                                            \
  } while (0)
  st->layers.resize(P.nl);
  for (int l = 0; l < P.nl; ++l) {
    LayerDev &L = st->layers[l];
    L.qkv = P.qkv;
    L.o = P.o;
    L.gu = P.gu;
    L.down = P.down;
    AL(L.qkv.tiles, L.qkv.bytes);
    AL(L.o.tiles, L.o.bytes);
    AL(L.gu.tiles, L.gu.bytes);
    AL(L.down.tiles, L.down.bytes);
    AL(L.g_attn, (size_t)P.d * 4);
    AL(L.g_ffn, (size_t)P.d * 4);
    if (cfg->qk_norm) {
      AL(L.g_q, (size_t)P.hd * 4);
      AL(L.g_k, (size_t)P.hd * 4);
    }
  }
  if (flags & KFL_EMBED_IN) AL(st->embed, (size_t)P.V * P.d * 2);
  if (flags & KFL_LOGITS_OUT) {
    st->lm = P.lm;
    AL(st->lm.tiles, st->lm.bytes);
    AL(st->g_final, (size_t)P.d * 4);
  }
  if (P.nl > 0) {
    AL(st->kc, (size_t)P.nl * P.kv_elems_per_layer * 2);
    AL(st->vc, (size_t)P.nl * P.kv_elems_per_layer * 2);
  }
  AL(st->rope_cos, (size_t)cfg->max_ctx * (P.hd / 2) * 4);
  AL(st->rope_sin, (size_t)cfg->max_ctx * (P.hd / 2) * 4);
  AL(st->h, (size_t)MAXB * P.ldh * 4);
  AL(st->xn, (size_t)MAXB * P.ldh * 4);
  AL(st->q, (size_t)MAXB * P.ldq * 4);
  AL(st->o, (size_t)MAXB * P.ldq * 4);
  AL(st->a, (size_t)MAXB * P.lda * 4);
  if (cfg->qk_norm) AL(st->qk_raw, (size_t)MAXB * P.ld_raw * 4);
  AL(st->sumsq, (size_t)P.n_parts * MAXB * 4);
  {
    // int4 GEMV inputs (allocated for every stage; zero where nothing writes: the padding)
    Act16 *acts[3] = {&st->xn16, &st->o16, &st->a16};
    const int lds[3] = {P.ldh, P.ldq, P.lda};
    for (int i = 0; i < 3; ++i) {
      Act16 &x = *acts[i];
      x.ld = lds[i];
      x.rest = i == 0 ? 1 : 0;
      const size_t bytes = act16_bytes(x.ld, x.rest != 0);
      AL(x.base, bytes);
      if (cudaMemset(x.base, 0, bytes) != cudaSuccess) return fail(KFL_ERR_CUDA);
    }
  }
  AL(st->pos, MAXB * 4);
  AL(st->slots, MAXB * 4);
  AL(st->next_int, MAXB * 4);
  AL(st->gemv_partial, (size_t)4 * P.gemv_grid_max * 2 * RB * MAXB * 4);
  AL(st->tickets, (size_t)(4 * P.n_rb_max + 1) * 4);
  st->am_ticket = st->tickets + 4 * P.n_rb_max;
  AL(st->counters, (size_t)std::max(1, P.n_phases) * P.ctr_stride * 4);
  AL(st->cand_val, (size_t)P.n_rb_max * MAXB * 4);
  AL(st->cand_idx, (size_t)P.n_rb_max * MAXB * 4);
  AL(st->attn_partial, (size_t)MAXB * P.hkv * P.attn_nchunks_max * 8 * (P.hd + 4) * 4);
  AL(st->attn_tickets, (size_t)MAXB * P.hkv * 4);
  AL(st->err, 16);
  AL(st->io_pos, MAXB * 4);
  AL(st->io_ids, MAXB * 4);
  AL(st->io_hin, (size_t)MAXB * P.d * 4);
  AL(st->bar, 16);
#undef AL
  // zero everything that is read before it is written or whose padding must stay zero
  if (P.nl > 0) {
    if (cudaMemset(st->kc, 0, (size_t)P.nl * P.kv_elems_per_layer * 2) != cudaSuccess) return fail(KFL_ERR_CUDA);
    if (cudaMemset(st->vc, 0, (size_t)P.nl * P.kv_elems_per_layer * 2) != cudaSuccess) return fail(KFL_ERR_CUDA);
    // the attention clusters read each layer's cache through TMA tensor maps
    st->kv_maps.resize(2 * (size_t)P.nl);
    const long long rows = (long long)cfg->max_batch * P.hkv * cfg->max_ctx;
    for (int l = 0; l < P.nl; ++l)
      if (encode_kv_map(&st->kv_maps[2 * l], st->kc + (size_t)l * P.kv_elems_per_layer, P.hd, rows) ||
          encode_kv_map(&st->kv_maps[2 * l + 1], st->vc + (size_t)l * P.kv_elems_per_layer, P.hd, rows))
        return fail(KFL_ERR_CUDA);
  }
  if (cudaMemset(st->h, 0, (size_t)MAXB * P.ldh * 4) || cudaMemset(st->xn, 0, (size_t)MAXB * P.ldh * 4) ||
      cudaMemset(st->q, 0, (size_t)MAXB * P.ldq * 4) || cudaMemset(st->o, 0, (size_t)MAXB * P.ldq * 4) ||
      cudaMemset(st->a, 0, (size_t)MAXB * P.lda * 4) || cudaMemset(st->sumsq, 0, (size_t)P.n_parts * MAXB * 4) ||
      cudaMemset(st->pos, 0, MAXB * 4) || cudaMemset(st->slots, 0, MAXB * 4) ||
      cudaMemset(st->next_int, 0, MAXB * 4) ||
      cudaMemset(st->tickets, 0, (size_t)(4 * P.n_rb_max + 1) * 4) ||
      cudaMemset(st->counters, 0, (size_t)std::max(1, P.n_phases) * P.ctr_stride * 4) ||
      cudaMemset(st->attn_tickets, 0, (size_t)MAXB * P.hkv * 4) || cudaMemset(st->err, 0, 16) ||
      cudaMemset(st->bar, 0, 16))
    return fail(KFL_ERR_CUDA);
  // RoPE table: angle pos * theta^(-2i/hd) in fp64, stored as fp32 cos / sin
  {
    const int half = P.hd / 2;
    std::vector<float> cs((size_t)cfg->max_ctx * half), sn((size_t)cfg->max_ctx * half);
    for (int p = 0; p < cfg->max_ctx; ++p)
      for (int i = 0; i < half; ++i) {
        const double a = (double)p * std::pow((double)cfg->rope_theta, -2.0 * i / P.hd);
        cs[(size_t)p * half + i] = (float)std::cos(a);
        sn[(size_t)p * half + i] = (float)std::sin(a);
      }
    if (cudaMemcpy(st->rope_cos, cs.data(), cs.size() * 4, cudaMemcpyHostToDevice) != cudaSuccess ||
        cudaMemcpy(st->rope_sin, sn.data(), sn.size() * 4, cudaMemcpyHostToDevice) != cudaSuccess)
      return fail(KFL_ERR_CUDA);
  }
  // persistent stage kernel: the deepest ring that fits next to the attention buffers
  // the persistent stage kernel has no QK-norm phase: QK-norm stages run one kernel per phase
  st->persistent = env_int("KFL_PERSISTENT", 0) != 0 && !cfg->qk_norm;
  {
    const size_t static_smem = 8192;  // the kernel's own __shared__ variables
    size_t smem_max = 0;
    for (int b = 1; b <= cfg->max_batch; ++b) {
      // 96-128 KiB of weights in flight per SM streams fastest (deeper rings queue more)
      int stages = env_int("KFL_STAGE_KERNEL_STAGES", 8);
      if (stages > MAX_STAGES) stages = MAX_STAGES;
      while (stages > 2 && stage_kernel_smem(stages, P.hd, b, cfg->weight_fmt) + static_smem > (size_t)smem_optin)
        --stages;
      stages = ring_depth(cfg->weight_fmt, stages);
      st->mk_stages[b] = stages;
      st->mk_smem[b] = stage_kernel_smem(stages, P.hd, b, cfg->weight_fmt);
      if (st->mk_smem[b] > smem_max) smem_max = st->mk_smem[b];
    }
    if (prepare_stage_kernel(smem_max) != cudaSuccess) {
      cudaGetLastError();
      st->persistent = false;
    }
  }
  *out = st;
  return KFL_OK;
}

extern "C" int kfl_stage_load_layer(kfl_stage *st, int local, const kfl_layer_weights *w, int on_device) {
  if (!valid(st)) return KFL_ERR_STATE;
  if (!w) return KFL_ERR_ARG;
  if (local < 0 || local >= st->P.nl) return KFL_ERR_RANGE;
  if (!w->attn_norm || !w->ffn_norm) return KFL_ERR_ARG;
  if (st->cfg.qk_norm && (!w->q_norm || !w->k_norm)) return KFL_ERR_ARG;
  CK(cudaSetDevice(st->dev));
  const Plan &P = st->P;
  LayerDev &L = st->layers[local];
  std::vector<void *> tmp;
  int rc = KFL_OK;
  do {
    if ((rc = load_gain(st, w->attn_norm, P.d, on_device, L.g_attn, tmp))) break;
    if ((rc = load_gain(st, w->ffn_norm, P.d, on_device, L.g_ffn, tmp))) break;
    if (st->cfg.qk_norm) {
      if ((rc = load_gain(st, w->q_norm, P.hd, on_device, L.g_q, tmp))) break;
      if ((rc = load_gain(st, w->k_norm, P.hd, on_device, L.g_k, tmp))) break;
    }
    // Q/K/V: q and k rows of each head reordered so that the RoPE pair (i, i + hd/2) is adjacent
    std::vector<int> map(P.qdim + 2 * P.kvdim);
    for (int r = 0; r < (int)map.size(); ++r) {
      if (r < P.qdim + P.kvdim) {
        const int base = (r / P.hd) * P.hd, j = r % P.hd;
        map[r] = base + ((j & 1) ? (j >> 1) + P.hd / 2 : (j >> 1));
      } else {
        map[r] = r;
      }
    }
    if ((rc = load_matrix(st, L.qkv, {{&w->wq, P.qdim}, {&w->wk, P.kvdim}, {&w->wv, P.kvdim}}, P.d, map, on_device,
                          tmp)))
      break;
    if ((rc = load_matrix(st, L.o, {{&w->wo, P.d}}, P.qdim, {}, on_device, tmp))) break;
    // gate/up interleaved: row 2j = gate j, row 2j + 1 = up j
    std::vector<int> gmap(2 * P.F);
    for (int j = 0; j < P.F; ++j) {
      gmap[2 * j] = j;
      gmap[2 * j + 1] = P.F + j;
    }
    if ((rc = load_matrix(st, L.gu, {{&w->wg, P.F}, {&w->wu, P.F}}, P.d, gmap, on_device, tmp))) break;
    if ((rc = load_matrix(st, L.down, {{&w->wd, P.d}}, P.F, {}, on_device, tmp))) break;
    if (cudaDeviceSynchronize() != cudaSuccess) {
      rc = KFL_ERR_CUDA;
      break;
    }
    L.loaded = true;
    st->drop_graphs();
  } while (0);
  cudaGetLastError();
  free_tmp(tmp);
  return rc;
}

extern "C" int kfl_stage_load_head(kfl_stage *st, const uint16_t *embed, const uint16_t *final_norm,
                                   const kfl_matrix *lm_head, int on_device) {
  if (!valid(st)) return KFL_ERR_STATE;
  if (!(st->flags & (KFL_EMBED_IN | KFL_LOGITS_OUT))) return KFL_OK;
  if ((st->flags & KFL_EMBED_IN) && !embed) return KFL_ERR_ARG;
  if ((st->flags & KFL_LOGITS_OUT) && (!final_norm || !lm_head)) return KFL_ERR_ARG;
  CK(cudaSetDevice(st->dev));
  const Plan &P = st->P;
  std::vector<void *> tmp;
  int rc = KFL_OK;
  do {
    if (st->flags & KFL_EMBED_IN) {
      if (cudaMemcpy(st->embed, embed, (size_t)P.V * P.d * 2, cudaMemcpyDefault) != cudaSuccess) {
        rc = KFL_ERR_CUDA;
        break;
      }
    }
    if (st->flags & KFL_LOGITS_OUT) {
      if ((rc = load_gain(st, final_norm, P.d, on_device, st->g_final, tmp))) break;
      if ((rc = load_matrix(st, st->lm, {{lm_head, P.V}}, P.d, {}, on_device, tmp))) break;
    }
    if (cudaDeviceSynchronize() != cudaSuccess) {
      rc = KFL_ERR_CUDA;
      break;
    }
    st->head_loaded = true;
    st->drop_graphs();
  } while (0);
  cudaGetLastError();
  free_tmp(tmp);
  return rc;
}

extern "C" int kfl_stage_load_weights(kfl_stage *st, const kfl_weights *w) {
  if (!valid(st)) return KFL_ERR_STATE;
  if (!w || w->n_layers != st->P.nl || (st->P.nl > 0 && !w->layers)) return KFL_ERR_ARG;
  for (int l = 0; l < st->P.nl; ++l) {
    int rc = kfl_stage_load_layer(st, l, &w->layers[l], w->on_device);
    if (rc) return rc;
  }
  return kfl_stage_load_head(st, w->embed, w->final_norm, &w->lm_head, w->on_device);
}

static int check_decode_args(kfl_stage *st, const int32_t *ids, const float *hidden_in, const int32_t *positions,
                             int batch, float *hidden_out, int32_t *next_ids) {
  if (!valid(st)) return KFL_ERR_STATE;
  if (batch < 1) return KFL_ERR_ARG;
  if (batch > st->cfg.max_batch) return KFL_ERR_RANGE;
  if (!positions) return KFL_ERR_ARG;
  if ((st->flags & KFL_EMBED_IN) ? !ids : !hidden_in) return KFL_ERR_ARG;
  if ((st->flags & KFL_LOGITS_OUT) ? !next_ids : !hidden_out) return KFL_ERR_ARG;
  if (!st->loaded()) return KFL_ERR_STATE;
  return KFL_OK;
}

extern "C" int kfl_stage_decode(kfl_stage *st, const int32_t *token_ids, const float *hidden_in,
                                const int32_t *positions, int batch, float *hidden_out, int32_t *next_ids,
                                void *cuda_stream) {
  int rc = check_decode_args(st, token_ids, hidden_in, positions, batch, hidden_out, next_ids);
  if (rc) return rc;
  CK(cudaSetDevice(st->dev));
  return run_step(st, token_ids, hidden_in, positions, nullptr, -1, batch, hidden_out, next_ids,
                  static_cast<cudaStream_t>(cuda_stream));
}

extern "C" int kfl_stage_decode_users(kfl_stage *st, const int32_t *token_ids, const float *hidden_in,
                                      const int32_t *positions, const int32_t *users, int batch,
                                      float *hidden_out, int32_t *next_ids, void *cuda_stream) {
  int rc = check_decode_args(st, token_ids, hidden_in, positions, batch, hidden_out, next_ids);
  if (rc) return rc;
  if (!users) return KFL_ERR_ARG;
  CK(cudaSetDevice(st->dev));
  return run_step(st, token_ids, hidden_in, positions, users, -1, batch, hidden_out, next_ids,
                  static_cast<cudaStream_t>(cuda_stream));
}

extern "C" int kfl_stage_prefill(kfl_stage *st, const int32_t *token_ids, const float *hidden_in,
                                 const int32_t *positions, int user, int n_tokens, float *hidden_out,
                                 int32_t *next_ids, void *cuda_stream) {
  if (!valid(st)) return KFL_ERR_STATE;
  if (n_tokens < 1 || !positions) return KFL_ERR_ARG;
  if ((st->flags & KFL_EMBED_IN) ? !token_ids : !hidden_in) return KFL_ERR_ARG;
  if ((st->flags & KFL_LOGITS_OUT) ? !next_ids : !hidden_out) return KFL_ERR_ARG;
  if (user < 0 || user >= st->cfg.max_batch) return KFL_ERR_RANGE;
  if (!st->loaded()) return KFL_ERR_STATE;
  CK(cudaSetDevice(st->dev));
  cudaStream_t s = static_cast<cudaStream_t>(cuda_stream);
  // the dense path from KFL_PREFILL_DENSE_MIN tokens on (default 16); QK-norm stages take the
  // decode-step path (the dense path has no QK-norm epilogue)
  if (n_tokens >= env_int("KFL_PREFILL_DENSE_MIN", 16) && !st->cfg.qk_norm)
    return run_prefill_dense(st, token_ids, hidden_in, positions, user, n_tokens, hidden_out, next_ids, s);
  const int d = st->P.d;
  // else the prompt in chunks of max_batch consecutive tokens: each chunk is one decode step whose
  // rows all address the user's KV slot, so a token attends to the chunk's earlier tokens too
  for (int t0 = 0; t0 < n_tokens; t0 += st->cfg.max_batch) {
    const int n = std::min(st->cfg.max_batch, n_tokens - t0);
    const int rc = run_step(st, token_ids ? token_ids + t0 : nullptr, hidden_in ? hidden_in + (size_t)t0 * d : nullptr,
                            positions + t0, nullptr, user, n, hidden_out ? hidden_out + (size_t)t0 * d : nullptr,
                            next_ids ? next_ids + t0 : nullptr, s);
    if (rc != KFL_OK) return rc;
  }
  return KFL_OK;
}

extern "C" int kfl_stage_decode_host(kfl_stage *st, const int32_t *token_ids, const float *hidden_in,
                                     const int32_t *positions, int batch, float *hidden_out, int32_t *next_ids,
                                     void *cuda_stream) {
  int rc = check_decode_args(st, token_ids, hidden_in, positions, batch, hidden_out, next_ids);
  if (rc) return rc;
  CK(cudaSetDevice(st->dev));
  cudaStream_t s = static_cast<cudaStream_t>(cuda_stream);
  const Plan &P = st->P;
  const bool embed = (st->flags & KFL_EMBED_IN) != 0;
  CK(cudaMemcpyAsync(st->io_pos, positions, (size_t)batch * 4, cudaMemcpyHostToDevice, s));
  if (embed) CK(cudaMemcpyAsync(st->io_ids, token_ids, (size_t)batch * 4, cudaMemcpyHostToDevice, s));
  else CK(cudaMemcpyAsync(st->io_hin, hidden_in, (size_t)batch * P.d * 4, cudaMemcpyHostToDevice, s));
  rc = run_step(st, embed ? st->io_ids : nullptr, embed ? nullptr : st->io_hin, st->io_pos, nullptr, -1, batch,
                nullptr, nullptr, s);
  if (rc) return rc;
  if (hidden_out)
    CK(cudaMemcpy2DAsync(hidden_out, (size_t)P.d * 4, st->h, (size_t)P.ldh * 4, (size_t)P.d * 4, batch,
                         cudaMemcpyDeviceToHost, s));
  if (next_ids) CK(cudaMemcpyAsync(next_ids, st->next_int, (size_t)batch * 4, cudaMemcpyDeviceToHost, s));
  CK(cudaStreamSynchronize(s));
  return KFL_OK;
}

extern "C" int kfl_kv_reset(kfl_stage *st, int user) {
  if (!valid(st)) return KFL_ERR_STATE;
  if (user < -1 || user >= st->cfg.max_batch) return KFL_ERR_RANGE;
  CK(cudaSetDevice(st->dev));
  CK(cudaDeviceSynchronize());
  const Plan &P = st->P;
  const size_t per_user = (size_t)P.hkv * st->cfg.max_ctx * P.hd;
  for (int l = 0; l < P.nl; ++l) {
    for (int u = 0; u < st->cfg.max_batch; ++u) {
      if (user >= 0 && u != user) continue;
      const size_t off = (size_t)l * P.kv_elems_per_layer + (size_t)u * per_user;
      CK(cudaMemset(st->kc + off, 0, per_user * 2));
      CK(cudaMemset(st->vc + off, 0, per_user * 2));
    }
  }
  CK(cudaDeviceSynchronize());
  return KFL_OK;
}

extern "C" int kfl_kv_fill_seeded(kfl_stage *st, int user, int len, uint64_t seed) {
  if (!valid(st)) return KFL_ERR_STATE;
  if (user < -1 || user >= st->cfg.max_batch || len < 0 || len > st->cfg.max_ctx) return KFL_ERR_RANGE;
  CK(cudaSetDevice(st->dev));
  CK(cudaDeviceSynchronize());
  const Plan &P = st->P;
  const float c = (float)(1.0 * (1.0 / std::sqrt((65536.0 * 65536.0 - 1.0) / 3.0)));
  const size_t per_user = (size_t)P.hkv * st->cfg.max_ctx * P.hd;
  for (int l = 0; l < P.nl; ++l) {
    const int gl = st->l0 + l;
    for (int u = 0; u < st->cfg.max_batch; ++u) {
      if (user >= 0 && u != user) continue;
      for (int h = 0; h < P.hkv; ++h) {
        const size_t off = (size_t)l * P.kv_elems_per_layer + (size_t)u * per_user + (size_t)h * st->cfg.max_ctx * P.hd;
        const int64_t start = (((int64_t)u * P.hkv + h) << 20) * P.hd;
        for (int which = 0; which < 2; ++which) {
          uint16_t *dst = (which == 0 ? st->kc : st->vc) + off;
          int rc = kfl_synth_fill(dst, (int64_t)len * P.hd, seed, 0x4B560000ull + 2ull * gl + which,
                                  KFL_SYNTH_NORMAL_BF16, c, 0.0f, start, nullptr);
          if (rc) return rc;
        }
      }
    }
  }
  CK(cudaDeviceSynchronize());
  return KFL_OK;
}

extern "C" int kfl_kv_write(kfl_stage *st, int local, int user, const uint16_t *k, const uint16_t *v, int len,
                            int on_device) {
  if (!valid(st)) return KFL_ERR_STATE;
  if (!k || !v) return KFL_ERR_ARG;
  if (local < 0 || local >= st->P.nl || user < 0 || user >= st->cfg.max_batch || len < 0 || len > st->cfg.max_ctx)
    return KFL_ERR_RANGE;
  if (len == 0) return KFL_OK;
  CK(cudaSetDevice(st->dev));
  CK(cudaDeviceSynchronize());
  const Plan &P = st->P;
  const size_t per_user = (size_t)P.hkv * st->cfg.max_ctx * P.hd;
  const size_t off = (size_t)local * P.kv_elems_per_layer + (size_t)user * per_user;
  const size_t dpitch = (size_t)st->cfg.max_ctx * P.hd * 2, spitch = (size_t)len * P.hd * 2;
  const cudaMemcpyKind kind = on_device ? cudaMemcpyDeviceToDevice : cudaMemcpyHostToDevice;
  CK(cudaMemcpy2D(st->kc + off, dpitch, k, spitch, spitch, P.hkv, kind));
  CK(cudaMemcpy2D(st->vc + off, dpitch, v, spitch, spitch, P.hkv, kind));
  return KFL_OK;
}

extern "C" int kfl_kv_read(kfl_stage *st, int local, int user, uint16_t *k, uint16_t *v, int on_device) {
  if (!valid(st)) return KFL_ERR_STATE;
  if (!k || !v) return KFL_ERR_ARG;
  if (local < 0 || local >= st->P.nl || user < 0 || user >= st->cfg.max_batch) return KFL_ERR_RANGE;
  CK(cudaSetDevice(st->dev));
  CK(cudaDeviceSynchronize());
  const Plan &P = st->P;
  const size_t per_user = (size_t)P.hkv * st->cfg.max_ctx * P.hd;
  const size_t off = (size_t)local * P.kv_elems_per_layer + (size_t)user * per_user;
  const cudaMemcpyKind kind = on_device ? cudaMemcpyDeviceToDevice : cudaMemcpyDeviceToHost;
  CK(cudaMemcpy(k, st->kc + off, per_user * 2, kind));
  CK(cudaMemcpy(v, st->vc + off, per_user * 2, kind));
  return KFL_OK;
}

extern "C" int kfl_stage_debug_capture(kfl_stage *st, float *per_layer_hidden) {
  if (!valid(st)) return KFL_ERR_STATE;
  if (st->capture != per_layer_hidden) {
    st->capture = per_layer_hidden;
    st->drop_graphs();
  }
  return KFL_OK;
}

extern "C" int kfl_stage_trace(kfl_stage *st, uint64_t *buf) {
  if (!valid(st)) return KFL_ERR_STATE;
  if (st->trace != reinterpret_cast<unsigned long long *>(buf)) {
    st->trace = reinterpret_cast<unsigned long long *>(buf);
    st->drop_graphs();
  }
  return KFL_OK;
}

extern "C" int kfl_stage_trace_shape(kfl_stage *st, int batch, int *n_phases, int *grid, int *slots) {
  if (!valid(st)) return KFL_ERR_STATE;
  if (batch < 1 || batch > st->cfg.max_batch) return KFL_ERR_RANGE;
  if (n_phases) *n_phases = (int)build_phases(st, batch).size();
  if (grid) *grid = std::max(st->P.n_sm, st->P.gemv_grid_max);
  if (slots) *slots = TRACE_SLOTS;
  return KFL_OK;
}

extern "C" int kfl_stage_status(kfl_stage *st) {
  if (!valid(st)) return KFL_ERR_STATE;
  CK(cudaSetDevice(st->dev));
  CK(cudaDeviceSynchronize());
  unsigned e = 0;
  CK(cudaMemcpy(&e, st->err, 4, cudaMemcpyDeviceToHost));
  CK(cudaMemset(st->err, 0, 4));
  if (e & ERR_TIMEOUT) return KFL_ERR_TIMEOUT;
  if (e & (ERR_POSITION | ERR_TOKEN)) return KFL_ERR_RANGE;
  if (e & ERR_F16_RANGE) return KFL_ERR_OVERFLOW;
  return KFL_OK;
}

extern "C" int kfl_stage_profile(kfl_stage *st, int enable) {
  if (!valid(st)) return KFL_ERR_STATE;
  st->profile = enable != 0;
  return KFL_OK;
}

extern "C" int kfl_stage_profile_read(kfl_stage *st, double *ms, int64_t *launches, int n) {
  if (!valid(st)) return KFL_ERR_STATE;
  CK(cudaSetDevice(st->dev));
  CK(cudaDeviceSynchronize());
  for (int k = 0; k < KFL_KERNEL_KINDS && k < n; ++k) {
    if (ms) ms[k] = st->prof_ms[k];
    if (launches) launches[k] = st->prof_n[k];
    st->prof_ms[k] = 0.0;
    st->prof_n[k] = 0;
  }
  return KFL_KERNEL_KINDS;
}

extern "C" int kfl_stage_launches_per_step(kfl_stage *st, int batch) {
  if (!valid(st)) return KFL_ERR_STATE;
  (void)batch;
  const int body = 5 * st->P.nl + ((st->flags & KFL_LOGITS_OUT) ? 1 : 0);
  if (st->profile || !st->persistent) return 2 + body + (st->cfg.qk_norm ? st->P.nl : 0);
  return 2 + (body > 0 ? 1 : 0);
}

extern "C" void kfl_stage_destroy(kfl_stage *st) {
  if (!valid(st)) return;
  cudaSetDevice(st->dev);
  cudaDeviceSynchronize();
  st->drop_graphs();
  for (cudaEvent_t e : st->ev) cudaEventDestroy(e);
  if (st->cap_stream) cudaStreamDestroy(st->cap_stream);
  for (void *p : st->allocs) cudaFree(p);
  for (void *p : st->pf_allocs) cudaFree(p);
  for (int b = 0; b < 2; ++b) {
    if (st->pf_w16[b]) cudaFree(st->pf_w16[b]);
    if (st->pf_deq[b]) cudaEventDestroy(st->pf_deq[b]);
    if (st->pf_used[b]) cudaEventDestroy(st->pf_used[b]);
  }
  if (st->pf_side) cudaStreamDestroy(st->pf_side);
  cudaGetLastError();
  st->magic = 0;
  delete st;
}

extern "C" const char *kfl_last_error_detail(void) { return g_last_error; }

namespace kfl {
// Lets other translation units of the library (the allocation-free entry point) set the text
// that kfl_last_error_detail returns.
void set_error_detail(const char *msg) { snprintf(g_last_error, sizeof(g_last_error), "%s", msg); }
}  // namespace kfl

extern "C" const char *kfl_strerror(int code) {
  switch (code) {
    case KFL_OK: return "ok";
    case KFL_ERR_ARG: return "invalid argument";
    case KFL_ERR_RANGE: return "index, size, position or token id out of range";
    case KFL_ERR_OOM: return "device memory allocation failed";
    case KFL_ERR_CUDA: return "CUDA runtime error";
    case KFL_ERR_STATE: return "stage not ready (weights not loaded) or invalid";
    case KFL_ERR_TIMEOUT: return "a bounded device-side wait gave up";
    case KFL_ERR_OVERFLOW: return "an int4 prefill activation is beyond the fp16 range";
    case KFL_ERR_INFEASIBLE: return "no division of the blocks fits the devices";
    default: return "unknown error";
  }
}
