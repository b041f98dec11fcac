"""Seeded synthetic weights made directly in device memory (harness support).

The same values as ``workload.layer_weights`` / ``workload.head_weights`` (bit for bit: the
device generator ``kfl_synth_fill`` implements the generator defined in ``workload``), made
on the GPU so that multi-gigabyte stages load in seconds.  Tensors come from torch (device
memory only); the values come from the library's generator kernel.
"""
from __future__ import annotations

import numpy as np
import torch

from . import stage as K
from . import workload as wl


def _empty(n: int, dtype, device) -> torch.Tensor:
    return torch.empty(n, dtype=dtype, device=device)


def normal_bf16(seed: int, tag: int, n: int, std: float, mean: float = 0.0, device="cuda") -> torch.Tensor:
    t = _empty(n, torch.int16, device)
    K.kfl_synth_fill(t, n, seed, tag, K.SYNTH_NORMAL_BF16, float(wl.normal_scale(std)), float(np.float32(mean)))
    return t


def matrix(fmt: str, seed: int, tag: int, scale_tag: int, rows: int, cols: int, device="cuda"):
    if fmt == "bf16":
        return normal_bf16(seed, tag, rows * cols, 0.02, device=device).view(rows, cols)
    words = _empty(rows * cols // 8, torch.int32, device)
    K.kfl_synth_fill(words, words.numel(), seed, tag, K.SYNTH_INT4_WORDS, 0.0)
    scales = _empty(rows * cols // 64, torch.int16, device)
    K.kfl_synth_fill(scales, scales.numel(), seed, scale_tag, K.SYNTH_INT4_SCALES_BF16,
                     float(np.float32(wl.INT4_SCALE_C1)))
    return (words.view(rows, cols // 8), scales.view(rows, cols // 64))


def layer_weights(model: wl.ModelShape, layer: int, seed: int, device="cuda") -> dict:
    w = {}
    for name in ("attn_norm", "ffn_norm"):
        w[name] = normal_bf16(seed, wl.layer_tag(layer, name), model.d_model, 0.02, mean=1.0, device=device)
    if model.qk_norm:
        for name in ("q_norm", "k_norm"):
            w[name] = normal_bf16(seed, wl.layer_tag(layer, name), model.head_dim, 0.02, mean=1.0, device=device)
    for name, (rows, cols) in model.matrix_shapes().items():
        w[name] = matrix(model.weight_fmt, seed, wl.layer_tag(layer, name), wl.layer_tag(layer, name, True),
                         rows, cols, device)
    return w


def head_weights(model: wl.ModelShape, seed: int, embed: bool = True, logits: bool = True, device="cuda") -> dict:
    w = {}
    d, v = model.d_model, model.vocab
    if embed:
        w["embed"] = normal_bf16(seed, wl.head_tag("embed"), v * d, 0.02, device=device).view(v, d)
    if logits:
        w["final_norm"] = normal_bf16(seed, wl.head_tag("final_norm"), d, 0.02, mean=1.0, device=device)
        w["lm_head"] = matrix(model.weight_fmt, seed, wl.head_tag("lm_head"), wl.head_tag("lm_head", True), v, d,
                              device)
    return w


def load_stage_seeded(st: K.Stage, work: wl.Workload, l0: int | None = None, l1: int | None = None) -> None:
    """Generate and load every weight of stage ``st`` (blocks [l0, l1) of ``work.model``) on the
    device, one block at a time, then fill each user's KV cache over its pre-filled context."""
    l0 = st.l0 if l0 is None else l0
    l1 = st.l1 if l1 is None else l1
    m = work.model
    for local, layer in enumerate(range(l0, l1)):
        w = layer_weights(m, layer, work.seed)
        K.kfl_stage_load_layer(st, local, w, on_device=True)
        del w
    if st.flags & (K.KFL_EMBED_IN | K.KFL_LOGITS_OUT):
        head = head_weights(m, work.seed, embed=bool(st.flags & K.KFL_EMBED_IN),
                            logits=bool(st.flags & K.KFL_LOGITS_OUT))
        K.kfl_stage_load_head(st, head, on_device=True)
        del head
    for u in range(work.batch):
        if st.n_layers > 0:
            K.kfl_kv_fill_seeded(st, u, work.contexts[u], work.seed)
    torch.cuda.synchronize()
