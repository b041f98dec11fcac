"""Write the oracle's expected values for one decode step of the 80-block int4 72B-shaped model.

The workload: the 72B-shaped decoder (d_model 8192, 64 query / 8 KV heads of 128, SwiGLU FFN
29568, vocab 152064) with every projection and the lm_head in int4 group-64 form, as one head
stage over all 80 blocks (embedding, blocks [0, 80), final RMSNorm, lm_head, greedy argmax),
four users each with 8192 pre-filled KV positions, seed 20260005, decoding step 0 (token ids
``first_token_ids``, every user at position 8192).  The batch-one workload is user 0 of this
batch: a row's result depends on that row's inputs only.

Only the oracle (``oracle``) and the seeded input generator (``paper_2609_34045_gb300.workload``)
are used.  The oracle runs the model one block at a time, as a chain of one-block stages
[l, l + 1): that a chain of stages equals one stage over the same blocks is the paper's own
invariant (section VI: every division gives the same output), pinned in the oracle's CPU tests.

Stored (``int4_72B_80L_step0.npz``):

* ``per_layer_rms[l][u]``: RMS of the hidden state after block l for user u (fp64);
* ``sample_cols``: 512 seeded column indices, and ``per_layer_sample[l][u]``: the hidden state
  after block l at those columns (fp32);
* ``full_layers`` = (13, 27, 80) and ``full_states``: the whole hidden state after those many
  blocks, the hand-over points of the stage splits {13, 67}, {27, 53} and {80} (fp32);
* ``next_ids``, ``margins`` (top-2 logit gap), ``top_ids`` / ``top_logits`` (the 16 largest
  logits per user);
* ``kv_layers`` and ``k_new`` / ``v_new``: the bf16 K and V rows written at position 8192 by
  those blocks;
* provenance: the seed, this script's SHA-256, the oracle's SHA-256.

Run from the repository root: ``python tests/golden/make_int4_72B_goldens.py [output.npz]``
(about 20 minutes on sixteen cores, 30 GB of host memory; the output defaults to the file beside
this script).
"""
from __future__ import annotations

import hashlib
import os
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
sys.path.insert(0, ROOT)

import oracle  # noqa: E402
from paper_2609_34045_gb300 import workload as wl  # noqa: E402

OUT = os.path.join(os.path.dirname(os.path.abspath(__file__)), "int4_72B_80L_step0.npz")
FULL_LAYERS = (13, 27, 80)
KV_LAYERS = (0, 12, 13, 26, 27, 79)
N_SAMPLE = 512
N_TOP = 16
SAMPLE_TAG = 0x474F4C44  # stream of the sampled column indices


def sha256(path: str) -> str:
    with open(path, "rb") as f:
        return hashlib.sha256(f.read()).hexdigest()


def sample_columns(d: int, seed: int) -> np.ndarray:
    """N_SAMPLE distinct columns of [0, d), sorted, from the seeded generator."""
    keys = wl.draws(wl.stream_key(seed, SAMPLE_TAG), 0, d)
    return np.sort(np.argsort(keys, kind="stable")[:N_SAMPLE]).astype(np.int64)


class Embedding:
    """Rows of the seeded embedding, generated on demand (only the batch's ids are read)."""

    def __init__(self, model, seed):
        self.model, self.seed = model, seed

    def __getitem__(self, ids):
        ids = np.atleast_1d(np.asarray(ids, dtype=np.int64))
        d = self.model.d_model
        idx = (ids[:, None] * d + np.arange(d)[None, :]).astype(np.uint64).ravel()
        return wl.normal_bf16_at(self.seed, wl.head_tag("embed"), idx, 0.02).reshape(len(ids), d)


def _no_huge_page_advice() -> None:
    """numpy asks the kernel for transparent huge pages on large arrays; where the kernel then
    compacts memory on every allocation, the oracle's multi-gigabyte temporaries crawl.  Only
    the allocation advice changes, not any value."""
    core = getattr(np, "_core", None) or getattr(np, "core", None)
    setter = getattr(getattr(core, "multiarray", None), "_set_madvise_hugepage", None)
    if setter is not None:
        setter(False)


def main(out: str = OUT) -> int:
    _no_huge_page_advice()
    work = wl.CONFIGS[6]
    m, seed, b = work.model, work.seed, work.batch
    assert work.contexts == (8192,) * 4 and wl.CONFIGS[5].seed == seed
    max_ctx = work.max_ctx
    pos = wl.positions(work, 0)
    ids = wl.first_token_ids(m, b, seed)
    cols = sample_columns(m.d_model, seed)
    n = m.n_layers_total
    rms = np.zeros((n, b))
    samp = np.zeros((n, b, N_SAMPLE), dtype=np.float32)
    full = {}
    k_new, v_new = [], []
    h = None
    t0 = time.time()
    for layer in range(n):
        first, last = layer == 0, layer == n - 1
        st = oracle.OracleStage(m, layer, layer + 1, first, last, b, max_ctx)
        st.load_layer(0, wl.layer_weights(m, layer, seed))
        head = {}
        if first:
            head["embed"] = Embedding(m, seed)
        if last:
            head.update(wl.head_weights(m, seed, embed=False, logits=True))
        st.load_head(head)
        for u in range(b):
            k, v = wl.kv_prefill(m, layer, u, work.contexts[u], seed)
            st.set_kv(0, u, k, v)
        o = st.decode(pos, token_ids=ids if first else None, hidden_in=None if first else h)
        h = o["hidden_out"]
        rms[layer] = np.sqrt(np.mean(h * h, axis=-1))
        samp[layer] = h[:, cols].astype(np.float32)
        if layer + 1 in FULL_LAYERS:
            full[layer + 1] = h.astype(np.float32)
        if layer in KV_LAYERS:
            k_new.append(np.stack([st.k_cache[0, u, :, pos[u]] for u in range(b)]))
            v_new.append(np.stack([st.v_cache[0, u, :, pos[u]] for u in range(b)]))
        if last:
            z = o["logits"]
            top = np.argsort(-z, axis=-1, kind="stable")[:, :N_TOP]
            next_ids, margins = o["next_ids"], o["margins"]
            top_logits = np.take_along_axis(z, top, axis=-1)
        print(f"block {layer}: rms {rms[layer].round(3).tolist()}  ({time.time() - t0:.0f} s)", flush=True)
        del st
    np.savez_compressed(
        out, seed=np.int64(seed), positions=pos.astype(np.int64), token_ids=ids.astype(np.int64),
        per_layer_rms=rms, sample_cols=cols, per_layer_sample=samp,
        full_layers=np.array(FULL_LAYERS, dtype=np.int64), full_states=np.stack([full[x] for x in FULL_LAYERS]),
        next_ids=next_ids.astype(np.int64), margins=margins, top_ids=top.astype(np.int64), top_logits=top_logits,
        kv_layers=np.array(KV_LAYERS, dtype=np.int64), k_new=np.stack(k_new), v_new=np.stack(v_new),
        script_sha256=np.array(sha256(os.path.abspath(__file__))),
        oracle_sha256=np.array(sha256(os.path.join(ROOT, "oracle", "stage.py"))))
    print("wrote", out, f"({time.time() - t0:.0f} s)")
    return 0


if __name__ == "__main__":
    sys.exit(main(*sys.argv[1:2]))
