"""Shared plumbing of the GPU parity tests: build both sides on the same seeded inputs, run
decode steps through the C ABI, and compare with the oracle."""
from __future__ import annotations

import os

import numpy as np
import torch

import oracle
from paper_2609_34045_gb300 import device_inputs as dev_in
from paper_2609_34045_gb300 import stage as K
from paper_2609_34045_gb300 import workload as wl

HIDDEN_TOL = 1e-2  # max-abs error per layer and user, relative to the oracle's RMS
ID_MARGIN = 1e-2   # argmax ids compared where the oracle's top-2 logit gap exceeds this


def ensure_built():
    if not os.path.exists(K.LIB_PATH):
        from paper_2609_34045_gb300.build import build
        build()


class LazyEmbedding:
    """Rows of the seeded embedding, generated on demand (the oracle reads only the rows of the
    ids it is given)."""

    def __init__(self, model, seed):
        self.model, self.seed = model, seed

    def __getitem__(self, ids):
        ids = np.atleast_1d(np.asarray(ids, dtype=np.int64))
        d = self.model.d_model
        idx = (ids[:, None] * d + np.arange(d)[None, :]).astype(np.uint64).ravel()
        return wl.normal_bf16_at(self.seed, wl.head_tag("embed"), idx, 0.02).reshape(len(ids), d)


class Pair:
    """A GPU stage and the oracle stage on identical weights and KV prefill."""

    def __init__(self, model, l0, l1, flags, batch, contexts, max_ctx, seed, device_weights=False,
                 max_batch=None):
        self.model, self.l0, self.l1, self.flags = model, l0, l1, flags
        self.batch, self.contexts, self.max_ctx, self.seed = batch, tuple(contexts), max_ctx, seed
        self.max_batch = max_batch or batch
        embed, logits = bool(flags & K.KFL_EMBED_IN), bool(flags & K.KFL_LOGITS_OUT)
        self.embed, self.logits = embed, logits
        cfg = K.model_cfg(model, max_ctx, self.max_batch)
        self.st = K.kfl_stage_create(cfg, l0, l1, flags)
        self.ora = oracle.OracleStage(model, l0, l1, embed, logits, self.max_batch, max_ctx)
        # weights: the oracle always from the host generator; the GPU from host arrays or from
        # the device twin of the generator (bit-identical, tested separately)
        for i, l in enumerate(range(l0, l1)):
            w = wl.layer_weights(model, l, seed)
            self.ora.load_layer(i, w)
            if device_weights:
                K.kfl_stage_load_layer(self.st, i, dev_in.layer_weights(model, l, seed), on_device=True)
            else:
                K.kfl_stage_load_layer(self.st, i, w, on_device=False)
        if embed or logits:
            if device_weights:
                head_o = {}
                if embed:
                    head_o["embed"] = LazyEmbedding(model, seed)
                if logits:
                    head_o.update(wl.head_weights(model, seed, embed=False, logits=True))
                self.ora.load_head(head_o)
                K.kfl_stage_load_head(self.st, dev_in.head_weights(model, seed, embed, logits), on_device=True)
            else:
                head = wl.head_weights(model, seed, embed, logits)
                self.ora.load_head(head)
                K.kfl_stage_load_head(self.st, head, on_device=False)
        for i, l in enumerate(range(l0, l1)):
            for u in range(batch):
                k, v = wl.kv_prefill(model, l, u, contexts[u], seed)
                self.ora.set_kv(i, u, k, v)
                if device_weights:
                    pass
                else:
                    K.kfl_kv_write(self.st, i, u, np.ascontiguousarray(k), np.ascontiguousarray(v), contexts[u],
                                   False)
        if device_weights:
            for u in range(batch):
                K.kfl_kv_fill_seeded(self.st, u, contexts[u], seed)
        self.k0 = self.ora.k_cache.copy()
        self.v0 = self.ora.v_cache.copy()
        self.written = set()
        n = max(1, l1 - l0)
        self.cap = torch.zeros(n, self.max_batch, model.d_model, dtype=torch.float32, device="cuda")
        K.kfl_stage_debug_capture(self.st, self.cap)

    def gpu_step(self, positions, ids=None, hidden=None, host=False):
        b = len(positions)
        d = self.model.d_model
        stream = torch.cuda.current_stream().cuda_stream
        if host:
            pos = np.ascontiguousarray(positions, dtype=np.int32)
            idt = np.ascontiguousarray(ids, dtype=np.int32) if ids is not None else None
            hid = np.ascontiguousarray(hidden, dtype=np.float32) if hidden is not None else None
            out = np.zeros((b, d), dtype=np.float32)
            nxt = np.zeros(b, dtype=np.int32) if self.logits else None
            K.kfl_stage_decode_host(self.st, idt, hid, pos, b, out, nxt, stream)
            return out, nxt
        pos = torch.tensor(np.asarray(positions), dtype=torch.int32, device="cuda")
        idt = torch.tensor(np.asarray(ids), dtype=torch.int32, device="cuda") if ids is not None else None
        hid = torch.tensor(np.asarray(hidden), dtype=torch.float32, device="cuda") if hidden is not None else None
        out = torch.zeros(b, d, dtype=torch.float32, device="cuda")
        nxt = torch.full((b,), -7, dtype=torch.int32, device="cuda") if self.logits else None
        K.kfl_stage_decode(self.st, idt, hid, pos, b, out, nxt, stream)
        torch.cuda.synchronize()
        return out.cpu().numpy(), (nxt.cpu().numpy() if nxt is not None else None)

    def step(self, s, ids=None, hidden=None, check=True):
        """Decode step ``s`` (positions contexts[b] + s) on both sides and compare; returns the
        oracle's output (its next ids drive the following step: teacher forcing)."""
        positions = np.array([self.contexts[u] + s for u in range(self.batch)], dtype=np.int32)
        for u in range(self.batch):
            self.written.add((u, int(positions[u])))
        o = self.ora.decode(positions, token_ids=ids, hidden_in=hidden, capture=True)
        g_out, g_next = self.gpu_step(positions, ids, hidden)
        if check:
            self.compare(o, g_out, g_next)
        return o, g_out, g_next

    def compare(self, o, g_out, g_next):
        b = self.batch
        cap = self.cap.cpu().numpy()
        for layer in range(self.l1 - self.l0):
            for u in range(b):
                ref = o["per_layer"][layer][u]
                err = np.max(np.abs(cap[layer, u] - ref))
                rms = np.sqrt(np.mean(ref * ref))
                assert err <= HIDDEN_TOL * rms, f"layer {layer} user {u}: max err {err:.3e} > {HIDDEN_TOL} x rms {rms:.3e}"
        ref = o["hidden_out"]
        for u in range(b):
            err = np.max(np.abs(g_out[u] - ref[u]))
            rms = np.sqrt(np.mean(ref[u] ** 2))
            assert err <= HIDDEN_TOL * rms, f"hidden_out user {u}: {err:.3e} vs rms {rms:.3e}"
        if self.logits:
            for u in range(b):
                if o["margins"][u] > ID_MARGIN:
                    assert int(g_next[u]) == int(o["next_ids"][u]), (u, g_next, o["next_ids"], o["margins"])
                else:
                    # a near tie: the GPU must still pick one of the (near-)maximal logits
                    z = o["logits"][u]
                    assert z[int(g_next[u])] >= np.max(z) - 2 * ID_MARGIN

    def compare_kv(self):
        """Slots never written are bit-identical to the prefill; written slots match the oracle."""
        hkv, hd = self.model.n_kv_heads, self.model.head_dim
        for layer in range(self.l1 - self.l0):
            for u in range(self.batch):
                kg = np.zeros((hkv, self.max_ctx, hd), dtype=np.uint16)
                vg = np.zeros_like(kg)
                K.kfl_kv_read(self.st, layer, u, kg, vg, False)
                written = sorted(p for (uu, p) in self.written if uu == u)
                mask = np.ones(self.max_ctx, dtype=bool)
                mask[written] = False
                assert np.array_equal(kg[:, mask], self.k0[layer, u][:, mask])
                assert np.array_equal(vg[:, mask], self.v0[layer, u][:, mask])
                if not written:
                    continue
                for cache_g, cache_o in ((kg, self.ora.k_cache), (vg, self.ora.v_cache)):
                    g = oracle.bf16_to_f64(cache_g[:, written])
                    r = oracle.bf16_to_f64(cache_o[layer, u][:, written])
                    rms = np.sqrt(np.mean(r * r))
                    assert np.all(np.abs(g - r) <= HIDDEN_TOL * rms + 2.0 ** -7 * np.abs(r))

    def close(self):
        K.kfl_stage_destroy(self.st)
