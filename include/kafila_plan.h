/* Kafila block placement over a ring of devices: host-side planner (no GPU needed).
 *
 * Follows the paper's planner: the stage cost of Eq. 2 (Section V-A), the exact chain-on-chain
 * block placement for a fixed device order (Section V-B "Block placement"), head
 * placement by rotation with a noise margin (Section V-B, the head paragraph), and the three
 * admission tiers with the final memory check (Section V-C "Admission").
 *
 * Conventions as in kafila_stage.h: KFL_OK (0) or a negative KFL_ERR_* code.  Every array is
 * owned by the caller and read (or, for outputs, written) only during the call.  Devices are
 * indexed in ring order 0..m-1; block counts are returned in that order, and the chain of blocks
 * starts at the head: the head holds blocks [0, n[head]), the next device around the ring the
 * following n[head+1], and so on.
 */
#ifndef KAFILA_PLAN_H
#define KAFILA_PLAN_H

#include <stddef.h>

#include "kafila_stage.h"

#ifdef __cplusplus
extern "C" {
#endif

#define KFL_ERR_INFEASIBLE (-7) /* no division of the blocks fits the devices (limits, or m > k) */

/* Exact chain-on-chain placement of k blocks on devices 0..m-1 in this order (Section V-B,
 * "Block placement": the problem the paper's Partition solves).  Device i holding n blocks costs
 * fixed[i] + n * per[i] (Eq. 2: fixed = o_i, plus beta_head / b_i for the head;
 * per = beta_block / b_i) and holds at most lim[i] blocks.  Writes n_out[i] >= 1 with sum k,
 * n_out[i] <= lim[i], minimizing the bottleneck max_i fixed[i] + n_out[i] * per[i], and that
 * bottleneck to *tau_out (the largest cost of the returned division, so exactly attained).
 * Method: each device starts with one block; the remaining k - m go one at a time to the device
 * whose cost after taking one more is lowest (the lower index on ties).  O(m + k log m).
 * Among the optimal divisions it returns the one this hand-out builds.
 * Errors: KFL_ERR_ARG (k < 1, m < 1, NULL arrays, a non-finite fixed or per, per <= 0, lim < 0),
 * KFL_ERR_INFEASIBLE (no division exists: a limit of 0, the limits sum below k, or m > k). */
int kfl_partition(int k, int m, const double *fixed, const double *per, const int *lim, int *n_out,
                  double *tau_out);

/* What the planner knows about one device (Section V-C).  A field <= 0 means "not measured". */
typedef struct {
  double o;           /* o_i: fixed stage time (time units of the plan) */
  double bw;          /* b_i: effective bandwidth (bytes per time unit); > 0: priced by Eq. 2 */
  double throughput;  /* raw arithmetic throughput (any common unit); > 0: reported */
  double working_set; /* reported working set (any common unit); > 0: reported */
  int lim_body;       /* block limit as a body member at the declared context and concurrency */
  int lim_head;       /* block limit as the head (the head also holds the embedding, lm_head) */
} kfl_plan_device;

typedef struct {
  int tier;          /* 1: Eq. 2 with head rotation; 2: throughput ratio, head at the anchor;
                        3: proportional to working set, head at the anchor */
  int head;          /* ring index of the head */
  double tau;        /* the division's bottleneck under the tier's cost (tier 3: 0) */
  double tau_anchor; /* tier 1: the bottleneck with the anchor as head (INFINITY if infeasible) */
  int undersized;    /* admission: the first device (from the head) whose share exceeds its
                        limit, else -1 */
} kfl_plan;

/* Plan k blocks over m devices in ring order (Sections V-B and V-C).
 *   Tier 1, every bw > 0: for every rotation (device r as head) Partition with
 *     fixed = o + (head ? beta_head / bw : 0), per = beta_block / bw, lim = lim_head or lim_body;
 *     the anchor stays head unless the best rotation's bottleneck is below
 *     tau_anchor * (1 - mu) (the paper's mu = 0.05).
 *   Tier 2, else if every throughput > 0: Partition from the anchor with per = 1 / throughput,
 *     no fixed or head term, the head at the anchor.
 *   Tier 3, else: blocks in proportion to working_set (kfl_divide), the head at the anchor.
 * Then admission: every device's share must be within its limit (head: lim_head).
 * Writes n_out[0..m-1] (ring order) and *plan.  Errors: KFL_ERR_ARG (bad sizes, NULL pointers,
 * anchor outside [0, m), mu outside [0, 1), tier 1 with beta_block <= 0 or beta_head < 0,
 * tier 3 with a working_set <= 0), KFL_ERR_INFEASIBLE (tiers 1 and 2: no division fits the
 * limits, plan->undersized = -1; tier 3: admission failed, plan->undersized names the device). */
int kfl_plan_ring(int k, int m, const kfl_plan_device *dev, int anchor, double beta_block, double beta_head,
                  double mu, int *n_out, kfl_plan *plan);

/* The baselines of the paper's evaluation (Section VII): weight == NULL, Uniform (GPipe): k / m
 * blocks each, the k mod m left over to the first devices; else Memory-proportional (exo): the
 * largest-remainder apportionment of k by weight (remainders tied: the lower index first), then
 * every device left with 0 blocks takes one from the device holding most (the lowest index on
 * ties).  Writes n_out[0..m-1].  Errors: KFL_ERR_ARG (k < m, m < 1, a weight <= 0 or non-finite). */
int kfl_divide(int k, int m, const double *weight, int *n_out);

/* lim(i) of Section V-B: the largest number of blocks n (0..cfg->n_layers_total) whose stage,
 * with the head's embedding and lm_head when is_head, needs at most room_bytes of device memory
 * at cfg's declared context (max_ctx) and concurrency (max_batch), as counted by
 * kfl_stage_memory_bytes.  Writes 0 if not even the smallest stage fits.  Errors: KFL_ERR_ARG. */
int kfl_block_limit(const kfl_model_cfg *cfg, size_t room_bytes, int is_head, int *lim_out);

#ifdef __cplusplus
}
#endif

#endif /* KAFILA_PLAN_H */
