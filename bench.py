"""Benchmark of the stage-decode step on GB300.

One step = one decode step of the 7B-shaped body stage (blocks [0, 14) of a 28-block Qwen
7B-shaped decoder, d_model 3584, 28/4 heads of 128, FFN 18944, bf16 weights, batch 1, KV
context 2048 pre-filled) unless --config picks another workload.  Each timed step decodes the
next position of the workload's 64-step run (positions wrap after 64 steps).

Prints one JSON line: metric "stage decode us/layer/token" (lower is better; the median of
--reps timed regions of --steps steps), the roofline of the dominant kernel (gate/up GEMV)
against the measured HBM copy bandwidth, the whole step's HBM fraction, an end-to-end figure
through the host-buffer C-ABI call, SM clocks sampled during the timed regions, and the CPU
oracle timed on a bounded sample (cpu_baseline).  With the default workload, ``also`` carries
the 32B-shaped head (b = 1), the 72B-shaped body with four ragged users (b = 4) and the 80-block
int4 72B-shaped model (b = 1 and b = 4), each timed the same way.

``--impl reference`` times the CPU oracle instead (this workload has no runnable reference
implementation: the paper ships none).
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "stage decode us/layer/token"
UNIT = "us/layer/token"


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--config", type=int, default=2)
    ap.add_argument("--profile-steps", type=int, default=20)
    ap.add_argument("--e2e-steps", type=int, default=500)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--reps", type=int, default=5, help="timed regions of --steps steps each (median reported)")
    ap.add_argument("--no-also", action="store_true",
                    help="skip the other workloads (32B head, 72B body b=4, 72B int4 b=1 and b=4)")
    ap.add_argument("--ring", action="store_true",
                    help="ring emulation: the 7B-shaped model as 4 stages of 7 blocks and the head's return "
                         "leg, 4 users served pipelined (one stream per stage) vs one at a time vs batched")
    ap.add_argument("--prefill", action="store_true",
                    help="time to first token of one user on the 7B-shaped model as one head stage: the "
                         "prompt's prefill (steps of 4 of its tokens) plus the first decode step")
    ap.add_argument("--prompt-lengths", default="128,512,2048",
                    help="--prefill: prompt lengths (comma-separated)")
    ap.add_argument("--prefill-gens", type=int, default=5,
                    help="--prefill: generations per case (the first is discarded)")
    ap.add_argument("--prefill-dense-only", action="store_true",
                    help="--prefill: skip the decode-step comparisons (for launch lists)")
    ap.add_argument("--prefill-config", type=int, default=2, choices=[2, 5],
                    help="--prefill: the model of this workload as one whole-model head stage "
                         "(2: 7B-shaped bf16, 5: 72B-shaped int4)")
    ap.add_argument("--prefill-layers", type=int, default=0,
                    help="--prefill: the head stage holds only the first N blocks (small case for profiling)")
    ap.add_argument("--layers", type=int, default=0,
                    help="small case for profiling: the first N blocks of the stage as a body stage "
                         "(no embedding, no head, no splits)")
    return ap.parse_args()


def dist_env():
    return int(os.environ.get("RANK", 0)), int(os.environ.get("LOCAL_RANK", 0)), int(os.environ.get("WORLD_SIZE", 1))


def max_over_ranks(x: float, dist, device) -> float:
    """The largest of every rank's x (the job is as slow as its slowest replica); x itself
    without a process group."""
    if dist is None:
        return x
    import torch
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


# ---------------------------------------------------------------------------- bytes

def kernel_bytes(work, kind: str) -> int:
    """Algorithmic HBM bytes of one launch of a kernel kind at the workload's first step:
    weights as stored once, activations in and out once, KV rows read over [0, P_b]."""
    from paper_2609_34045_gb300 import workload as wl
    m, b = work.model, work.batch
    d, q, kv, f, v = m.d_model, m.q_dim, m.kv_dim, m.ffn, m.vocab
    mb = lambda r, c: wl.matrix_bytes(r, c, m.weight_fmt)  # noqa: E731
    if kind == "qkv":
        return mb(q + 2 * kv, d) + b * (d + q) * 4 + b * 2 * kv * 2
    if kind == "attn":
        return sum(2 * kv * 2 * (p + 1) for p in work.contexts[:b]) + 2 * b * q * 4
    if kind == "oproj":
        return mb(d, q) + b * (q + 3 * d) * 4
    if kind == "gateup":
        return mb(2 * f, d) + b * (d + f) * 4
    if kind == "down":
        return mb(d, f) + b * (f + 3 * d) * 4
    if kind == "lmhead":
        return mb(v, d) + b * d * 4
    return 0


def measured_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            j = json.load(f)
        return float(j["hbm_gbs"]), "measured"
    return 6800.0, "fallback"


def kernel_source_hash() -> str:
    """Hash of the sources the GEMV kernels are built from: a committed DRAM-traffic figure
    counts only while they are unchanged."""
    h = hashlib.sha256()
    for name in ("gemv.cu", "gemv_core.cuh", "common.cuh"):
        with open(os.path.join(ROOT, "paper_2609_34045_gb300", "csrc", name), "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


def ncu_traffic(kind: str, config: int):
    """DRAM bytes per launch from the committed ncu summary, if it was taken on the current
    kernel source (else None)."""
    p = os.path.join(ROOT, "profiles", "traffic.json")
    if not os.path.exists(p):
        return None
    with open(p) as f:
        j = json.load(f)
    e = j.get(f"config{config}", {}).get(kind)
    if not e or e.get("source_hash") != kernel_source_hash():
        return None
    return e.get("dram_bytes_per_launch")


# ---------------------------------------------------------------------------- clocks

class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def start(self):
        try:
            fd, self.path = tempfile.mkstemp(prefix="kfl_clocks_", suffix=".csv")
            os.close(fd)
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "100"],
                                         stdout=self.f, stderr=subprocess.DEVNULL)
        except (OSError, FileNotFoundError):
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.f.close()
        rows = []
        with open(self.path) as f:
            for line in f:
                parts = [x.strip() for x in line.split(",")]
                if len(parts) >= 9:
                    rows.append(parts)
        os.unlink(self.path)
        if not rows:
            return None
        sm = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        mx = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        reasons = sorted({n for r in rows for n, v in zip(names, r[5:9]) if v.lower() == "active"})
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": reasons, "samples": len(rows)}


# ---------------------------------------------------------------------------- CPU oracle

def oracle_layer_seconds(work, n_layer_steps: int, warmup: int = 1, budget_s: float = 0.0):
    """Time the CPU oracle on single-block decode steps of the workload (weights and KV made
    before timing): n_layer_steps steps, or with budget_s > 0 as many as fit in about budget_s
    seconds (at least 2, at most n_layer_steps).  Returns (seconds per layer-token, layer-steps
    timed, threads)."""
    import numpy as np

    import oracle
    from paper_2609_34045_gb300 import workload as wl
    m = work.model
    st = oracle.OracleStage(m, work.l0, work.l0 + 1, False, False, work.batch, work.max_ctx)
    st.load_layer(0, wl.layer_weights(m, work.l0, work.seed))
    for u in range(work.batch):
        k, v = wl.kv_prefill(m, work.l0, u, work.contexts[u], work.seed)
        st.set_kv(0, u, k, v)
    h = wl.hidden_in(m, 0, work.batch, work.seed)
    pos = wl.positions(work, 0)
    for _ in range(warmup):
        st.decode(pos, hidden_in=h)
    t0 = time.perf_counter()
    n = 0
    while n < n_layer_steps:
        st.decode(pos, hidden_in=h)
        n += 1
        if budget_s > 0 and n >= 2 and time.perf_counter() - t0 >= budget_s:
            break
    dt = (time.perf_counter() - t0) / n
    return dt / work.batch, n, os.cpu_count()


def run_reference(args, work):
    rank, _, world = dist_env()
    if rank != 0:
        return 0
    sec, n, cores = oracle_layer_seconds(work, max(1, min(args.steps, 8)), warmup=min(args.warmup, 1))
    us = sec * 1e6
    line = {
        "impl": "reference", "metric": METRIC, "value": us, "unit": UNIT, "n_gpus": args.gpus, "steps": n,
        "warmup": min(args.warmup, 1), "ms_per_step": sec * 1e3 * work.batch, "higher_is_better": False,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic (seeded)",
        "config": {"workload": work.name, "layers_timed": 1, "batch": work.batch, "ctx": list(work.contexts),
                   "note": "the paper ships no implementation; the reference arm is the fp64 CPU oracle"},
        "cpu_baseline": {"value": us, "unit": UNIT, "cores": cores, "kind": "oracle",
                         "sample": f"{n} decode steps of one block (block {work.l0}) of {work.name}"},
        "e2e": {"value": us, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


# ---------------------------------------------------------------------------- ours

def run_splits(work, st_full, ids_all, hid_all, pos_all, args, stream):
    """The workload's stage splits ({13, 67} = blocks [0, 13) then [13, 80), ...) run as
    consecutive stages on this GPU, the hidden state handed over in a device buffer.  Each split
    is checked bit for bit against the single stage over its first steps (next ids and final
    hidden state), then timed.  Returns a list of per-split results."""
    import dataclasses

    import numpy as np
    import torch

    from paper_2609_34045_gb300 import device_inputs as di
    from paper_2609_34045_gb300 import stage as K

    m, b, d = work.model, work.batch, work.model.d_model
    n_check = 3
    n_time = max(10, min(200, args.steps // 10))
    cfg = K.model_cfg(m, work.max_ctx, b)
    res = []
    for split in work.splits:
        if len(split) < 2:
            continue
        bounds = [work.l0]
        for n in split:
            bounds.append(bounds[-1] + n)
        parts = []
        for i in range(len(split)):
            flags = (K.KFL_EMBED_IN if (i == 0 and work.embed_in) else 0) | \
                    (K.KFL_LOGITS_OUT if (i == len(split) - 1 and work.logits_out) else 0)
            s_ = K.kfl_stage_create(cfg, bounds[i], bounds[i + 1], flags)
            di.load_stage_seeded(s_, work, bounds[i], bounds[i + 1])
            parts.append(s_)
        hbuf = [torch.empty(b, d, dtype=torch.float32, device="cuda") for _ in range(len(split))]
        nxt = torch.empty(b, dtype=torch.int32, device="cuda") if work.logits_out else None

        def chain(i):
            j = i % work.steps
            for k, s_ in enumerate(parts):
                K.kfl_stage_decode(s_, ids_all[j] if (k == 0 and ids_all is not None) else None,
                                   (hid_all[j] if hid_all is not None else None) if k == 0 else hbuf[k - 1],
                                   pos_all[j], b, hbuf[k], nxt if k == len(parts) - 1 else None, stream.cuda_stream)

        exact = True
        ref_h = torch.empty(b, d, dtype=torch.float32, device="cuda")
        ref_n = torch.empty(b, dtype=torch.int32, device="cuda") if work.logits_out else None
        for i in range(n_check):
            chain(i)
            K.kfl_stage_decode(st_full, ids_all[i] if ids_all is not None else None,
                               hid_all[i] if hid_all is not None else None, pos_all[i], b, ref_h, ref_n,
                               stream.cuda_stream)
            torch.cuda.synchronize()
            exact = exact and torch.equal(ref_h, hbuf[-1]) and (ref_n is None or torch.equal(ref_n, nxt))
        for i in range(n_check, n_check + 3):
            chain(i)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize()
        e0.record(stream)
        for i in range(n_time):
            chain(n_check + 3 + i)
        e1.record(stream)
        torch.cuda.synchronize()
        ms = e0.elapsed_time(e1) / n_time
        # each stage of the chain on its own (events between the stages' launches)
        evs = [[torch.cuda.Event(enable_timing=True) for _ in range(len(parts) + 1)] for _ in range(n_time)]
        for i in range(n_time):
            j = (n_check + 3 + i) % work.steps
            for k, s_ in enumerate(parts):
                evs[i][k].record(stream)
                K.kfl_stage_decode(s_, ids_all[j] if (k == 0 and ids_all is not None) else None,
                                   (hid_all[j] if hid_all is not None else None) if k == 0 else hbuf[k - 1],
                                   pos_all[j], b, hbuf[k], nxt if k == len(parts) - 1 else None, stream.cuda_stream)
            evs[i][-1].record(stream)
        torch.cuda.synchronize()
        stage_ms = [float(np.median([evs[i][k].elapsed_time(evs[i][k + 1]) for i in range(n_time)]))
                    for k in range(len(parts))]
        stage_bytes = [dataclasses.replace(work, l0=bounds[k], l1=bounds[k + 1],
                                           embed_in=work.embed_in and k == 0,
                                           logits_out=work.logits_out and k == len(parts) - 1,
                                           splits=()).step_bytes(n_check + 3)
                       for k in range(len(parts))]
        for s_ in parts:
            if K.kfl_stage_status(s_) != 0:
                raise RuntimeError("device reported an error in a split stage")
            K.kfl_stage_destroy(s_)
        res.append({"split": list(split), "ms_per_step": ms, "us_per_layer_token": ms * 1e3 / (work.n_layers * b),
                    "steps_timed": n_time, "bit_exact_vs_single_stage": bool(exact),
                    "steps_compared": n_check, "stage_ms": stage_ms, "stage_bytes": stage_bytes})
    return res


def empty_stage_ms(work, stream, n=50):
    """The fixed per-stage time o of the cost model (Eq. 2): a stage with no blocks that only
    embeds the token (stage input and output kernels)."""
    import torch

    from paper_2609_34045_gb300 import device_inputs as di
    from paper_2609_34045_gb300 import stage as K
    from paper_2609_34045_gb300 import workload as wl

    m, b = work.model, work.batch
    st = K.kfl_stage_create(K.model_cfg(m, work.max_ctx, b), 0, 0, K.KFL_EMBED_IN)
    di.load_stage_seeded(st, work, 0, 0)
    ids = torch.tensor(wl.first_token_ids(m, b, work.seed), device="cuda")
    pos = torch.tensor(wl.positions(work, 0), device="cuda")
    out = torch.empty(b, m.d_model, dtype=torch.float32, device="cuda")
    for _ in range(5):
        K.kfl_stage_decode(st, ids, None, pos, b, out, None, stream.cuda_stream)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    e0.record(stream)
    for _ in range(n):
        K.kfl_stage_decode(st, ids, None, pos, b, out, None, stream.cuda_stream)
    e1.record(stream)
    torch.cuda.synchronize()
    K.kfl_stage_destroy(st)
    return e0.elapsed_time(e1) / n


def block_probe_stage(work, stream, o_ms, n=30):
    """The per-format bandwidth probe of Eq. 2: one block of the workload's model, in its weight
    format, at its batch and context, run as a body stage of its own (a device can time this
    before any division of the blocks).  b = the block's algorithmic bytes / (its step time - o),
    in GB/s, with o the empty stage's fixed time."""
    import dataclasses

    import torch

    from paper_2609_34045_gb300 import device_inputs as di
    from paper_2609_34045_gb300 import stage as K

    one = dataclasses.replace(work, l0=0, l1=1, embed_in=False, logits_out=False, splits=())
    st = K.kfl_stage_create(K.model_cfg(one.model, one.max_ctx, one.batch), 0, 1, 0)
    di.load_stage_seeded(st, one)
    inputs = step_inputs(one)
    times, _ = time_steps(st, one, inputs, n, 5, 3, stream, None)
    K.kfl_stage_destroy(st)
    ms = statistics.median(times)
    return one.step_bytes(0) / ((ms - o_ms) * 1e-3) / 1e9, ms


def plan_example(work, fit):
    """The planner (the exact fixed-order division with head rotation, section V) on a synthetic
    ring driven by this GPU's measured stage cost: four members stream at 1, 1/2, 1/4 and 1/8 of
    the probed rate b with the probed overhead o, and hold 35, 280, 140 and 70 GB; the bottleneck
    of the planned
    division against the evaluation's Uniform and Memory-proportional divisions under the same
    costs (Eq. 2, ms per step)."""
    import dataclasses

    from paper_2609_34045_gb300 import stage as K

    m = work.model
    k = m.n_layers_total
    cfg = K.model_cfg(m, work.max_ctx, work.batch)
    mid = dataclasses.replace(work, l0=0, l1=1, embed_in=False, logits_out=False, splits=())
    beta_block = float(mid.step_bytes(work.steps // 2))
    head = dataclasses.replace(work, l0=0, l1=0, embed_in=True, logits_out=True, splits=())
    beta_head = float(head.step_bytes(0))
    rates = [1.0, 0.5, 0.25, 0.125]
    rooms = [35e9, 280e9, 140e9, 70e9]
    bw = [fit["b_gbs"] * 1e6 * r for r in rates]  # bytes per ms
    devs = [dict(o=fit["o_us"] * 1e-3, bw=b, lim_body=K.kfl_block_limit(cfg, int(room), False),
                 lim_head=K.kfl_block_limit(cfg, int(room), True)) for b, room in zip(bw, rooms)]
    n, plan, rc = K.kfl_plan_ring(k, devs, 0, beta_block, beta_head, 0.05)

    def bottleneck(div, h):
        return max(devs[i]["o"] + (beta_head / bw[i] if i == h else 0.0) + div[i] * beta_block / bw[i]
                   for i in range(len(devs)))
    out = {"members_rate_of_measured": rates, "members_memory_gb": [r / 1e9 for r in rooms],
           "blocks": k, "beta_block_bytes": beta_block, "beta_head_bytes": beta_head,
           "lim_body": [d["lim_body"] for d in devs], "lim_head": [d["lim_head"] for d in devs]}
    if rc == 0:
        out.update(partition={"blocks": n, "head": plan["head"], "bottleneck_ms": plan["tau"]})
    for name, w in (("uniform", None), ("memory_proportional", rooms)):
        div = K.kfl_divide(k, len(devs), w)
        fits = all(div[i] <= (devs[i]["lim_head"] if i == 0 else devs[i]["lim_body"]) for i in range(len(devs)))
        out[name] = {"blocks": div, "head": 0, "bottleneck_ms": bottleneck(div, 0), "fits_memory": fits}
    return out


def cost_model(points, probe_gbs, o_ms, block_probe_gbs=None):
    """The paper's per-stage cost (Eq. 2), c = o + bytes / b: each stage's algorithmic HBM bytes
    (its blocks' weights and KV, and the head's embedding and unembedding) over a bandwidth b.
    points: [(bytes, measured ms)].  'probe' takes b from a copy benchmark and o from an empty
    stage; 'block_probe' (when given) takes b from one block of the model run in the stage's own
    weight format before any placement (block_probe_stage); both are what a planner can measure
    ahead of dividing the blocks.  'fitted' takes (o, b) from a least-squares line through the
    points (it needs the stages it predicts).  Returns each, with each stage's predicted time and
    relative error."""
    import numpy as np

    x = np.array([p[0] for p in points], dtype=np.float64)
    y = np.array([p[1] for p in points], dtype=np.float64)

    def evaluate(o, gbs):
        pred = o + x / (gbs * 1e6)
        err = (pred - y) / y
        return {"o_us": o * 1e3, "b_gbs": gbs, "pred_ms": pred.tolist(), "rel_err": err.tolist(),
                "median_abs_err": float(np.median(np.abs(err)))}

    out = {"stage_bytes": x.tolist(), "measured_ms": y.tolist(), "probe": evaluate(o_ms, probe_gbs)}
    if block_probe_gbs:
        out["block_probe"] = evaluate(o_ms, block_probe_gbs)
    if len(points) >= 2 and np.ptp(x) > 0:
        slope, icpt = np.polyfit(x, y, 1)
        out["fitted"] = evaluate(float(icpt), float(1.0 / (slope * 1e6)))
    return out


def step_inputs(work):
    """Device tensors of every step's positions and inputs (token ids, else hidden states)."""
    import numpy as np
    import torch

    from paper_2609_34045_gb300 import workload as wl
    m, b = work.model, work.batch
    pos_all = torch.tensor(np.stack([wl.positions(work, s) for s in range(work.steps)]), dtype=torch.int32,
                           device="cuda")
    if work.embed_in:
        ids_all = torch.tensor(np.stack([wl.token_ids(work.seed, wl.ids_tag(s), b, m.vocab)
                                         for s in range(work.steps)]), dtype=torch.int32, device="cuda")
        return pos_all, ids_all, None
    hid_all = torch.tensor(np.stack([wl.hidden_in(m, s, b, work.seed) for s in range(work.steps)]),
                           dtype=torch.float32, device="cuda")
    return pos_all, None, hid_all


def time_steps(st, work, inputs, steps, warmup, reps, stream, dist, clocks=None):
    """Decode steps of stage ``st``: ``warmup`` untimed, then ``reps`` timed regions of exactly
    ``steps`` steps, each bracketed by a barrier and a device synchronization, timed with CUDA
    events on the launching stream (the max over ranks).  Returns (ms per step of each region,
    clock record or None)."""
    import torch

    from paper_2609_34045_gb300 import stage as K
    pos_all, ids_all, hid_all = inputs
    b, d = work.batch, work.model.d_model
    out = torch.empty(b, d, dtype=torch.float32, device="cuda")
    nxt = torch.empty(b, dtype=torch.int32, device="cuda") if work.logits_out else None

    def step(s):
        i = s % work.steps
        K.kfl_stage_decode(st, ids_all[i] if ids_all is not None else None,
                           hid_all[i] if hid_all is not None else None, pos_all[i], b, out, nxt,
                           stream.cuda_stream)

    for s in range(warmup):
        step(s)
    torch.cuda.synchronize()
    if clocks is not None:
        clocks.start()
        time.sleep(0.3)  # let the sampler take its first reading
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    times = []
    for r in range(reps):
        if dist:
            dist.barrier()
        torch.cuda.synchronize()
        ev0.record(stream)
        for s in range(steps):
            step(warmup + r * steps + s)
        ev1.record(stream)
        torch.cuda.synchronize()
        times.append(max_over_ranks(ev0.elapsed_time(ev1) / steps, dist, "cuda"))
    clk = clocks.stop() if clocks is not None else None
    status = K.kfl_stage_status(st)
    if status != 0:
        raise RuntimeError(f"device reported {K.kfl_strerror(status)} during the benchmark")
    return times, clk


def per_kernel_profile(st, work, inputs, n_steps, stream):
    """Per-kernel time (the library's profile mode: CUDA events around each launch on the
    stage's stream) and achieved GB/s of each kernel kind."""
    from paper_2609_34045_gb300 import stage as K
    K.kfl_stage_profile(st, True)
    time_steps(st, work, inputs, n_steps, 0, 1, stream, None)
    prof = K.kfl_stage_profile_read(st)
    K.kfl_stage_profile(st, False)
    kinds = [k for k in ("qkv", "attn", "oproj", "gateup", "down", "lmhead") if prof[k][1] > 0]
    return {k: {"us": 1e3 * prof[k][0] / prof[k][1], "launches_per_step": prof[k][1] / n_steps,
                "gbs": (kernel_bytes(work, k) / (prof[k][0] / prof[k][1] * 1e-3) / 1e9) if prof[k][0] else None}
            for k in kinds}


def also_workloads(args, stream, local):
    """The batch-4 and int4 workloads measured in the same run, each as its own timed regions:
    the 32B-shaped head (b = 1), the 72B-shaped body with four ragged users (b = 4), and the
    80-block int4 72B-shaped model at b = 1 and b = 4 (one stage with four users' KV slots; b = 1
    decodes user 0).  Per workload: ms per step (median, min, max over the regions), the step's
    algorithmic bytes over its time, per-kernel times, and the clocks during its regions."""
    import dataclasses

    from paper_2609_34045_gb300 import device_inputs as di
    from paper_2609_34045_gb300 import stage as K
    from paper_2609_34045_gb300 import workload as wl

    peak, _ = measured_peaks()
    also_steps = max(1, min(args.steps, 40))
    res = {}

    def measure(work, st):
        inputs = step_inputs(work)
        times, clk = time_steps(st, work, inputs, also_steps, max(3, args.warmup), args.reps, stream, None,
                                ClockSampler(local))
        ms = statistics.median(times)
        sb = work.step_bytes(0)
        gbs = sb / (ms * 1e-3) / 1e9
        return {"workload": work.name, "batch": work.batch, "stage_layers": [work.l0, work.l1],
                "weights": work.model.weight_fmt, "ctx": list(work.contexts),
                "ms_per_step": ms, "ms_per_step_min": min(times), "ms_per_step_max": max(times),
                "regions": len(times), "steps_per_region": also_steps,
                "us_per_layer_token": ms * 1e3 / (max(1, work.n_layers) * work.batch),
                "tokens_per_s": work.batch / (ms * 1e-3),
                "step_roofline": {"bytes_per_step": sb, "achieved_gbs": gbs, "frac_of_measured": gbs / peak,
                                  "frac_of_8tbs": gbs / 8000.0},
                "per_kernel": per_kernel_profile(st, work, inputs, min(args.profile_steps, 10), stream),
                "clocks": clk}

    for n in (3, 4):
        work = wl.CONFIGS[n]
        st = K.kfl_stage_create(K.model_cfg(work.model, work.max_ctx, work.batch), work.l0, work.l1,
                                (K.KFL_EMBED_IN if work.embed_in else 0) | (K.KFL_LOGITS_OUT if work.logits_out else 0))
        di.load_stage_seeded(st, work)
        res[f"config{n}"] = measure(work, st)
        K.kfl_stage_destroy(st)
    w6 = wl.CONFIGS[6]
    st = K.kfl_stage_create(K.model_cfg(w6.model, w6.max_ctx, 4), w6.l0, w6.l1, K.KFL_IS_HEAD)
    di.load_stage_seeded(st, w6)
    w5 = dataclasses.replace(wl.CONFIGS[5], splits=())
    assert w5.max_ctx == w6.max_ctx and w5.contexts[0] == w6.contexts[0]
    res["config5"] = measure(w5, st)
    res["config6"] = measure(dataclasses.replace(w6, splits=()), st)
    K.kfl_stage_destroy(st)
    return res


def run_ours(args, work):
    import numpy as np
    import torch

    from paper_2609_34045_gb300 import device_inputs as di
    from paper_2609_34045_gb300 import stage as K
    from paper_2609_34045_gb300 import workload as wl

    rank, local, world = dist_env()
    torch.cuda.set_device(local)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    if not os.path.exists(K.LIB_PATH):
        from paper_2609_34045_gb300.build import build
        build()

    m = work.model
    flags = (K.KFL_EMBED_IN if work.embed_in else 0) | (K.KFL_LOGITS_OUT if work.logits_out else 0)
    cfg = K.model_cfg(m, work.max_ctx, work.batch)
    st = K.kfl_stage_create(cfg, work.l0, work.l1, flags)
    di.load_stage_seeded(st, work)
    b, d = work.batch, m.d_model
    stream = torch.cuda.current_stream()
    n_pos = work.steps
    inputs = step_inputs(work)
    pos_all, ids_all, hid_all = inputs

    times, clk = time_steps(st, work, inputs, args.steps, args.warmup, args.reps, stream, dist,
                            ClockSampler(local))
    ms = statistics.median(times)
    if dist:
        dist.barrier()

    n_layers = max(1, work.n_layers)
    value = ms * 1e3 / (n_layers * b) / world
    launches = K.kfl_stage_launches_per_step(st, b) * args.steps

    # per-kernel timing (kernels one by one with CUDA events on the launching stream)
    per_kernel = per_kernel_profile(st, work, inputs, args.profile_steps, stream)
    dom = max(per_kernel, key=lambda k: per_kernel[k]["us"] * per_kernel[k]["launches_per_step"])
    dom_ms = per_kernel[dom]["us"] * 1e-3
    dom_bytes = kernel_bytes(work, dom)
    peak, peak_kind = measured_peaks()
    achieved = dom_bytes / (dom_ms * 1e-3) / 1e9
    step_bytes = work.step_bytes(0)
    step_gbs = step_bytes / (ms * 1e-3) / 1e9

    # end to end through the host-buffer C-ABI call (pinned host memory, copies timed)
    e2e_steps = min(args.e2e_steps, args.steps)
    pos_h = torch.from_numpy(np.stack([wl.positions(work, s) for s in range(n_pos)])).pin_memory()
    if work.embed_in:
        in_h = torch.from_numpy(np.stack([wl.token_ids(work.seed, wl.ids_tag(s), b, m.vocab)
                                          for s in range(n_pos)])).pin_memory()
        h2d = b * 4 + b * 4
    else:
        in_h = torch.from_numpy(np.stack([wl.hidden_in(m, s, b, work.seed) for s in range(n_pos)])).pin_memory()
        h2d = b * d * 4 + b * 4
    out_h = torch.empty(b, d, dtype=torch.float32).pin_memory()
    nxt_h = torch.empty(b, dtype=torch.int32).pin_memory() if work.logits_out else None
    d2h = (b * 4) if work.logits_out else (b * d * 4)

    def e2e_step(s):
        i = s % n_pos
        K.kfl_stage_decode_host(st, in_h[i] if work.embed_in else None, None if work.embed_in else in_h[i],
                                pos_h[i], b, None if work.logits_out else out_h, nxt_h, stream.cuda_stream)

    for s in range(3):
        e2e_step(s)
    if dist:
        dist.barrier()
    t0 = time.perf_counter()
    for s in range(e2e_steps):
        e2e_step(s)
    e2e_s = (time.perf_counter() - t0) / e2e_steps
    e2e_s = max_over_ranks(e2e_s, dist, "cuda")
    e2e_value = e2e_s * 1e6 / (n_layers * b) / world

    splits = run_splits(work, st, ids_all, hid_all, pos_all, args, stream) if work.splits and world == 1 else None
    cost = None
    if splits:
        # Eq. 2 against every stage timed here: the whole model as one stage, and each split's stages
        points = [(work.step_bytes(work.steps // 2), ms)]
        for r in splits:
            points += list(zip(r["stage_bytes"], r["stage_ms"]))
        o_ms = empty_stage_ms(work, stream)
        probe_gbs, probe_ms = block_probe_stage(work, stream, o_ms)
        cost = cost_model(points, measured_peaks()[0], o_ms, probe_gbs)
        cost["block_probe_step_ms"] = probe_ms
        # the planner runs on what it can measure before placing blocks: the block probe
        cost["plan_example"] = plan_example(work, {"o_us": o_ms * 1e3, "b_gbs": probe_gbs})
    K.kfl_stage_destroy(st)

    also = None
    if world == 1 and args.config == 2 and args.layers == 0 and not args.no_also:
        also = also_workloads(args, stream, local)

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        sec, n, cores = oracle_layer_seconds(work, 64, budget_s=10.0)
        cpu = {"value": sec * 1e6, "unit": UNIT, "cores": cores, "kind": "oracle",
               "sample": f"{n} decode steps of one block (block {work.l0}) of {work.name}, fp64 numpy"}

    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": False, "scaling": "weak",
            # the arithmetic type of the weight products: fp32 FMAs on bf16 weights; fp16
            # tensor-core products (fp32 accumulation) on int4 weights
            "vs_baseline": None, "dtype": "f32" if m.weight_fmt == "bf16" else "f16", "data": "synthetic (seeded)",
            "config": {"workload": work.name, "stage_layers": [work.l0, work.l1], "batch": b,
                       "ctx": list(work.contexts), "weights": m.weight_fmt,
                       "arithmetic": ("fp32 FMA on bf16 weights" if m.weight_fmt == "bf16"
                                      else "fp16 x int4-as-fp16 tensor-core MMA, fp32 accumulation"),
                       "l2": "inputs larger than L2 (weights streamed once per step)",
                       "parallelism": f"replicas x{world}",
                       "timing": f"median of {len(times)} timed regions of {args.steps} steps each",
                       "execution": ("persistent stage kernel" if launches == 3 * args.steps
                                     else "one kernel per phase, CUDA graph + programmatic dependent launch")},
            "repeats": {"ms_per_step": times, "median": ms, "min": min(times), "max": max(times)},
            "tokens_per_s": b * world / (ms * 1e-3),
            "roofline": {"bound": "hbm", "kernel": dom, "achieved": achieved, "peak": peak, "unit": "GB/s",
                         "frac": achieved / peak, "peak_kind": f"{peak_kind} copy (MEASURED_PEAKS.json hbm_gbs)",
                         "bytes_per_launch": dom_bytes, "us_per_launch": dom_ms * 1e3,
                         "traffic": ncu_traffic(dom, args.config)},
            "step_roofline": {"bytes_per_step": step_bytes, "achieved_gbs": step_gbs, "frac_of_measured": step_gbs / peak,
                              "frac_of_8tbs": step_gbs / 8000.0},
            "per_kernel": per_kernel,
            "e2e": {"value": e2e_value, "unit": UNIT, "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
                    "steps": e2e_steps},
            "gpu_launches": launches * len(times),
            "clocks": clk,
            "cpu_baseline": cpu,
        }
        if splits is not None:
            line["splits"] = splits
            line["cost_model"] = cost
        if also is not None:
            line["also"] = also
        print(json.dumps(line), flush=True)
    if dist:
        dist.destroy_process_group()
    return 0


def run_ring(args):
    """Tokens per second of 4 users around a ring of stages on this GPU (section VII, "Serving
    several users at once"): pipelined (each stage on its own stream, working on one user's token
    while the stage after it works on another's), the same schedule on one stream, one user alone,
    and, for reference, all four users batched through one whole-model stage."""
    import dataclasses

    import torch

    from paper_2609_34045_gb300 import device_inputs as di
    from paper_2609_34045_gb300 import stage as K
    from paper_2609_34045_gb300 import workload as wl
    from paper_2609_34045_gb300.ring import Ring

    users, tokens = 4, 16
    base = wl.CONFIGS[2]
    m = base.model
    work = dataclasses.replace(base, name="7B-ring-4x7-u4-ctx2048", l0=0, l1=m.n_layers_total, embed_in=True,
                               logits_out=True, batch=users, contexts=(2048, 2048, 2048, 2048), steps=6 * tokens,
                               splits=())
    torch.cuda.set_device(0)
    ring = Ring(work, [7, 7, 7, 7], users)
    first = wl.first_token_ids(m, users, work.seed)

    def timed(fn):
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        out = fn()
        torch.cuda.synchronize()
        return time.perf_counter() - t0, out

    ring.run(first, 2)  # warm-up: every stage captures its graph
    res = {}
    t, ids_pipe = timed(lambda: ring.run(first, tokens, start=2))
    res["pipelined_4_users"] = users * tokens / t
    t, ids_seq = timed(lambda: ring.run(first, tokens, start=2 + tokens, sequential=True))
    res["sequential_4_users"] = users * tokens / t
    # one user alone: the same ring, users 1..3 idle
    ring1_first = [first[0]]
    ring.users, saved = 1, ring.users
    t, _ = timed(lambda: ring.run(ring1_first, tokens, start=2 + 2 * tokens))
    res["one_user"] = tokens / t
    ring.users = saved
    ring.close()
    # all four users batched through one whole-model (head) stage
    cfg = K.model_cfg(m, work.max_ctx, users)
    st = K.kfl_stage_create(cfg, 0, m.n_layers_total, K.KFL_IS_HEAD)
    di.load_stage_seeded(st, work)
    ids = torch.tensor(first, dtype=torch.int32, device="cuda")
    nxt = torch.zeros(users, dtype=torch.int32, device="cuda")
    stream = torch.cuda.current_stream().cuda_stream

    def batched(n, start):
        tok = ids.clone()
        for j in range(n):
            pos = torch.tensor([c + start + j for c in work.contexts], dtype=torch.int32, device="cuda")
            K.kfl_stage_decode(st, tok, None, pos, users, None, nxt, stream)
            tok.copy_(nxt)
    batched(2, 2 + 3 * tokens)
    t, _ = timed(lambda: batched(tokens, 4 + 3 * tokens))
    res["batched_4_users"] = users * tokens / t
    K.kfl_stage_destroy(st)
    line = {"metric": "ring tokens/s", "unit": "tokens/s", "higher_is_better": True, "n_gpus": 1,
            "config": {"workload": work.name, "stages": [7, 7, 7, 7, "return leg"], "users": users,
                       "tokens_per_user": tokens, "ctx": 2048, "weights": "bf16"},
            "tokens_per_s": res,
            "pipelined_over_sequential": res["pipelined_4_users"] / res["sequential_4_users"],
            "data": "synthetic (seeded)", "timing": "host wall clock around synchronized runs"}
    print(json.dumps(line), flush=True)
    return 0


def run_prefill(args):
    """Time to first token split into prefill and decode (section VI, instrumentation paragraph)
    on the 7B-shaped model as one head stage, one user from an empty cache: the prompt goes
    through kfl_stage_prefill, then one decode step.  The prefill is the dense path (tensor-core
    matrix products over the prompt's tokens); for comparison the 512-token prompt also in steps
    of max_batch = 4 tokens through the decode kernels, and one token per step
    (kfl_stage_decode_users at batch 1).  As in the paper's protocol, five generations per case,
    the first discarded as cold, the median of the rest; CUDA events on the launching stream."""
    import dataclasses
    import statistics

    import torch

    from paper_2609_34045_gb300 import device_inputs as di
    from paper_2609_34045_gb300 import stage as K
    from paper_2609_34045_gb300 import workload as wl

    lengths = tuple(int(x) for x in args.prompt_lengths.split(","))
    gens = max(2, args.prefill_gens)
    base = wl.CONFIGS[args.prefill_config]
    m = base.model
    nl = args.prefill_layers if 0 < args.prefill_layers < m.n_layers_total else m.n_layers_total
    shape = "7B" if args.prefill_config == 2 else "72B-int4"
    work = dataclasses.replace(base, name=f"{shape}-head-{nl}L-prefill", l0=0, l1=nl, embed_in=True,
                               logits_out=True, batch=4, contexts=(0, 0, 0, 0), steps=max(lengths) + 64,
                               splits=())
    torch.cuda.set_device(0)
    cfg = K.model_cfg(m, work.max_ctx, 4)
    st = K.kfl_stage_create(cfg, 0, nl, K.KFL_IS_HEAD)
    di.load_stage_seeded(st, work)
    stream = torch.cuda.current_stream()
    sp = stream.cuda_stream
    user = torch.zeros(1, dtype=torch.int32, device="cuda")
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(3)]

    def ttft(n, dense):
        os.environ["KFL_PREFILL_DENSE_MIN"] = "1" if dense else str(1 << 30)
        ids = torch.tensor(wl.token_ids(work.seed, 90, n, m.vocab), device="cuda")
        pos = torch.arange(n, dtype=torch.int32, device="cuda")
        nxt = torch.zeros(n, dtype=torch.int32, device="cuda")
        tok = torch.zeros(1, dtype=torch.int32, device="cuda")
        first = torch.zeros(1, dtype=torch.int32, device="cuda")
        pos_n = torch.tensor([n], dtype=torch.int32, device="cuda")
        times = []
        for g in range(gens):
            torch.cuda.synchronize()
            ev[0].record(stream)
            K.kfl_stage_prefill(st, ids, None, pos, 0, n, None, nxt, sp)
            ev[1].record(stream)
            tok.copy_(nxt[n - 1:])
            K.kfl_stage_decode_users(st, tok, None, pos_n, user, 1, None, first, sp)
            ev[2].record(stream)
            torch.cuda.synchronize()
            times.append((ev[0].elapsed_time(ev[1]), ev[1].elapsed_time(ev[2])))
        pre = statistics.median(x[0] for x in times[1:])
        dec = statistics.median(x[1] for x in times[1:])
        # the weight products only (attention's products excluded)
        flops = 2.0 * n * (nl * sum(r * c for r, c in m.matrix_shapes().values()) + m.vocab * m.d_model)
        return {"prefill_ms": pre, "decode_ms": dec, "ttft_ms": pre + dec, "prefill_tokens_per_s": n / pre * 1e3,
                "matmul_tflops": flops / pre / 1e9}

    rows = {n: ttft(n, True) for n in lengths}
    os.environ.pop("KFL_PREFILL_DENSE_MIN", None)
    if args.prefill_dense_only:
        K.kfl_stage_destroy(st)
        print(json.dumps({"metric": "time to first token", "unit": "ms", "higher_is_better": False, "n_gpus": 1,
                          "config": {"workload": work.name, "users": 1, "weights": m.weight_fmt,
                                     "prompt_lengths": list(lengths)},
                          "dense_by_prompt_length": {str(k): v for k, v in rows.items()}}), flush=True)
        return 0
    n = 512 if 512 in lengths else lengths[0]
    steps512 = ttft(n, False)
    os.environ.pop("KFL_PREFILL_DENSE_MIN", None)
    # one token per step
    ids = torch.tensor(wl.token_ids(work.seed, 90, n, m.vocab), dtype=torch.int32, device="cuda")
    pos = torch.arange(n, dtype=torch.int32, device="cuda")
    first = torch.zeros(1, dtype=torch.int32, device="cuda")
    times = []
    for g in range(min(gens, 3)):
        torch.cuda.synchronize()
        ev[0].record(stream)
        for t in range(n):
            K.kfl_stage_decode_users(st, ids[t:t + 1], None, pos[t:t + 1], user, 1, None, first, sp)
        ev[1].record(stream)
        torch.cuda.synchronize()
        times.append(ev[0].elapsed_time(ev[1]))
    one = statistics.median(times[1:])
    if K.kfl_stage_status(st) != 0:
        raise RuntimeError("device reported an error during the prefill runs")
    K.kfl_stage_destroy(st)
    line = {"metric": "time to first token", "unit": "ms", "higher_is_better": False, "n_gpus": 1,
            "config": {"workload": work.name, "users": 1, "weights": m.weight_fmt,
                       "prompt_lengths": list(lengths)},
            "dense_by_prompt_length": {str(k): v for k, v in rows.items()},
            f"steps_of_4_{n}": steps512,
            f"one_token_per_step_{n}": {"prefill_ms": one, "prefill_tokens_per_s": n / one * 1e3},
            "data": "synthetic (seeded)", "protocol": f"{gens} generations, first discarded, median",
            "timing": "CUDA events on the launching stream"}
    print(json.dumps(line), flush=True)
    return 0


def main():
    args = parse()
    if args.ring:
        return run_ring(args)
    if args.prefill:
        return run_prefill(args)
    import dataclasses

    from paper_2609_34045_gb300 import workload as wl
    work = wl.CONFIGS[args.config]
    if args.layers > 0 and args.layers < work.n_layers:
        work = dataclasses.replace(work, l1=work.l0 + args.layers, name=f"{work.name}-first{args.layers}",
                                   embed_in=False, logits_out=False, splits=())
    if args.impl == "reference":
        return run_reference(args, work)
    return run_ours(args, work)


if __name__ == "__main__":
    sys.exit(main())
