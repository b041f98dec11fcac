"""fp64 oracle of one pipeline stage's decode step and prompt prefill (test infrastructure only).

What a stage computes comes from the paper:

* A session serves the model as a ring of members; a token leaves the head, passes through
  each member's contiguous range of decoder blocks and returns to the head (section III,
  "ring" paragraph).  A stage is therefore a block range [l0, l1) applied to a hidden state.
* The head holds the embedding, the unembedding and the sampler (section III, "head"
  paragraph); the sampler is greedy at a fixed seed so that every division produces the same
  output (section VI, testbed paragraph).  Hence a stage split [0,k)+[k,L) must equal [0,L).
* At batch one a stage reads each weight once and does two flops per weight (section V-A,
  Eq. 2); the work is the decoder forward pass of the served Qwen-family models.

The paper never spells out a block's internals.  The oracle takes the standard pre-norm
decoder of that family: RMSNorm, fused-free Q/K/V projections, rotate-half RoPE, causal
grouped-query attention over the cached positions, output projection with a residual add,
RMSNorm, SwiGLU feed-forward with a residual add.  Every reading of a point the paper leaves
open is listed in the design notes of the repository.

Arithmetic is fp64 throughout.  Stored values are the inputs' own formats: bf16 bit patterns
(uint16) for weights, gains, embedding and the KV cache; int4 group-64 codes with bf16
scales for quantised matrices.  The only rounding the method itself performs is the KV cache
store (bf16); the oracle takes that decision in the kernel's precision: fp64 -> fp32 -> bf16,
round to nearest even.
"""
from __future__ import annotations

import numpy as np

__all__ = [
    "bf16_to_f64", "round_to_bf16", "int4_codes", "dequant_int4_g64", "matrix_f64", "gemv",
    "rms_norm", "rope_angles", "rope_rotate", "softmax", "attention_gqa", "silu", "swiglu",
    "argmax_first", "top2_margin", "OracleStage",
]


# --------------------------------------------------------------------------- number formats

def bf16_to_f64(bits) -> np.ndarray:
    """bf16 bit patterns -> fp64.  A bf16 value is the top 16 bits of an fp32 value, so the
    conversion is exact."""
    u = np.asarray(bits, dtype=np.uint16).astype(np.uint32)
    u <<= np.uint32(16)
    with np.errstate(invalid="ignore"):
        return u.view(np.float32).astype(np.float64)


def round_to_bf16(x) -> np.ndarray:
    """fp64 -> bf16 bit patterns: first to fp32 (nearest even), then to bf16 by rounding the
    low 16 bits of the fp32 pattern to nearest, ties to even.  NaN maps to a quiet NaN."""
    f = np.ascontiguousarray(np.asarray(x, dtype=np.float64).astype(np.float32))
    u = f.view(np.uint32).astype(np.uint64)
    low = u & np.uint64(0xFFFF)
    high = u >> np.uint64(16)
    up = (low > np.uint64(0x8000)) | ((low == np.uint64(0x8000)) & ((high & np.uint64(1)) == np.uint64(1)))
    r = high + up.astype(np.uint64)
    isnan = np.isnan(f)
    r = np.where(isnan, np.uint64(0x7FC0), r)
    return r.astype(np.uint16)


# the signed value of each 4-bit pattern (two's complement: 0x8 -> -8, 0xF -> -1)
_NIBBLE_VALUE = np.array([n - 16 if n >= 8 else n for n in range(16)], dtype=np.int8)


def int4_codes(words) -> np.ndarray:
    """Signed 4-bit codes of packed words: code ``j`` of a uint32 word is bits [4j, 4j+4),
    low nibble first along K, two's complement (0x8 -> -8, 0xF -> -1).  Returns int8
    ``[..., 8 * words]``.  Byte ``i`` of a word (little-endian) holds codes 2i (its low nibble)
    and 2i + 1 (its high nibble)."""
    w = np.asarray(words, dtype=np.uint32)
    b = np.ascontiguousarray(w, dtype="<u4").view(np.uint8).reshape(*w.shape, 4)
    q = np.stack([_NIBBLE_VALUE[b & 0xF], _NIBBLE_VALUE[b >> 4]], axis=-1)
    return q.reshape(*w.shape[:-1], w.shape[-1] * 8)


def dequant_int4_g64(words, scales) -> np.ndarray:
    """Symmetric int4 group quantisation along K, group 64, bf16 scales, zero point 0:
    ``w[n][k] = code(n, k) * scale[n][k // 64]``."""
    q = int4_codes(words).astype(np.float64)
    s = bf16_to_f64(scales)
    groups = q.reshape(*q.shape[:-1], q.shape[-1] // 64, 64)  # [..., group][64 codes]
    return (groups * s[..., None]).reshape(q.shape)


def matrix_f64(m) -> np.ndarray:
    """A stored weight matrix ``[out][in]`` as fp64: bf16 bits, or (int4 words, bf16 scales)."""
    if isinstance(m, tuple):
        return dequant_int4_g64(*m)
    return bf16_to_f64(m)


# --------------------------------------------------------------------------- block parts

def gemv(w: np.ndarray, x: np.ndarray) -> np.ndarray:
    """Linear map of each row of ``x`` (``[b][in]``) by ``w`` (``[out][in]``): ``y = x W^T``.
    Batch-one decode applies every weight once with one multiply-add (section V-A, Eq. 2)."""
    return np.asarray(x, dtype=np.float64) @ np.asarray(w, dtype=np.float64).T


def rms_norm(h: np.ndarray, g: np.ndarray, eps: float) -> np.ndarray:
    """RMSNorm over the last axis: ``h / sqrt(mean(h^2) + eps) * g``."""
    h = np.asarray(h, dtype=np.float64)
    ms = np.mean(h * h, axis=-1, keepdims=True)
    return h / np.sqrt(ms + eps) * np.asarray(g, dtype=np.float64)


def rope_angles(pos: int, head_dim: int, theta: float) -> np.ndarray:
    """Rotation angles at ``pos``: ``pos * theta^(-2i/head_dim)`` for i in [0, head_dim/2)."""
    i = np.arange(head_dim // 2, dtype=np.float64)
    return float(pos) * np.power(float(theta), -2.0 * i / head_dim)


def rope_rotate(x: np.ndarray, pos: int, theta: float) -> np.ndarray:
    """Rotate-half rotary embedding of ``x`` (``[heads][head_dim]``) at position ``pos``: the pair
    (x_i, x_{i+hd/2}) is rotated by angle a_i."""
    x = np.asarray(x, dtype=np.float64)
    hd = x.shape[-1]
    a = rope_angles(pos, hd, theta)
    c, s = np.cos(a), np.sin(a)
    x1, x2 = x[..., : hd // 2], x[..., hd // 2:]
    return np.concatenate([x1 * c - x2 * s, x2 * c + x1 * s], axis=-1)


def softmax(s: np.ndarray) -> np.ndarray:
    """Softmax over the last axis, with the maximum subtracted first."""
    s = np.asarray(s, dtype=np.float64)
    e = np.exp(s - np.max(s, axis=-1, keepdims=True))
    return e / np.sum(e, axis=-1, keepdims=True)


def attention_gqa(q: np.ndarray, k: np.ndarray, v: np.ndarray) -> np.ndarray:
    """Causal decode attention of one user over its cached positions.

    ``q``: ``[Hq][hd]``; ``k``, ``v``: ``[Hkv][T][hd]`` holding positions [0, T) (the new token's
    own position included).  Query head h reads KV head ``h // (Hq / Hkv)``; scores are scaled
    by ``1/sqrt(hd)``.  Returns ``[Hq][hd]``."""
    hq, hd = q.shape
    hkv = k.shape[0]
    group = hq // hkv
    out = np.empty((hq, hd), dtype=np.float64)
    for h in range(hq):
        kh = h // group
        p = softmax(k[kh] @ q[h] / np.sqrt(hd))
        out[h] = p @ v[kh]
    return out


def silu(x: np.ndarray) -> np.ndarray:
    """``x * sigmoid(x) = x / (1 + e^{-x})``."""
    x = np.asarray(x, dtype=np.float64)
    return x / (1.0 + np.exp(-x))


def swiglu(gate: np.ndarray, up: np.ndarray) -> np.ndarray:
    return silu(gate) * np.asarray(up, dtype=np.float64)


def argmax_first(z: np.ndarray) -> int:
    """Greedy sampler: the index of the largest logit, the lowest index among equal maxima."""
    z = np.asarray(z, dtype=np.float64)
    return int(np.flatnonzero(z == np.max(z))[0])


def top2_margin(z: np.ndarray) -> float:
    """Largest minus second-largest logit (0 when the maximum is not unique)."""
    s = np.sort(np.asarray(z, dtype=np.float64))
    return float(s[-1] - s[-2]) if s.size > 1 else float("inf")


# --------------------------------------------------------------------------- the stage

class OracleStage:
    """A stage: decoder blocks [l0, l1) of a model, plus the head's parts when asked.

    ``embed_in``: the stage starts from token ids through the embedding (the head's first leg).
    ``logits_out``: the stage ends with final RMSNorm, unembedding and greedy argmax (the head's
    return leg).  The KV cache is held as bf16 bit patterns ``[layer][user][kv head][slot][hd]``;
    user ``b``'s token at position ``P_b`` attends to slots [0, P_b] and is stored at slot P_b.
    """

    def __init__(self, model, l0: int, l1: int, embed_in: bool, logits_out: bool, max_batch: int,
                 max_ctx: int):
        self.m = model
        self.l0, self.l1 = l0, l1
        self.embed_in, self.logits_out = embed_in, logits_out
        self.max_batch, self.max_ctx = max_batch, max_ctx
        self.layers = [None] * (l1 - l0)
        self.head = {}
        n = l1 - l0
        shape = (n, max_batch, model.n_kv_heads, max_ctx, model.head_dim)
        self.k_cache = np.zeros(shape, dtype=np.uint16)
        self.v_cache = np.zeros(shape, dtype=np.uint16)

    def load_layer(self, local: int, w: dict) -> None:
        self.layers[local] = w

    def load_head(self, w: dict) -> None:
        self.head = dict(w)

    def set_kv(self, local: int, user: int, k_bits: np.ndarray, v_bits: np.ndarray) -> None:
        """Cached K/V of ``user`` for slots [0, len) of stage layer ``local`` (``[Hkv][len][hd]``)."""
        n = k_bits.shape[1]
        self.k_cache[local, user, :, :n] = k_bits
        self.v_cache[local, user, :, :n] = v_bits

    def _block(self, local: int, h: np.ndarray, positions: np.ndarray, slots: np.ndarray) -> np.ndarray:
        m, w = self.m, self.layers[local]
        b = h.shape[0]
        hq, hkv, hd = m.n_heads, m.n_kv_heads, m.head_dim
        y = rms_norm(h, bf16_to_f64(w["attn_norm"]), m.rms_eps)
        q = gemv(matrix_f64(w["wq"]), y).reshape(b, hq, hd)
        k = gemv(matrix_f64(w["wk"]), y).reshape(b, hkv, hd)
        v = gemv(matrix_f64(w["wv"]), y).reshape(b, hkv, hd)
        # every row's K/V is stored before any row attends: rows of one user at several positions
        # (a prompt) see the earlier ones, as causal attention over the prompt does
        qs = []
        for u in range(b):
            p, sl = int(positions[u]), int(slots[u])
            qu, ku = q[u], k[u]
            if m.qk_norm:
                qu = rms_norm(qu, bf16_to_f64(w["q_norm"]), m.rms_eps)
                ku = rms_norm(ku, bf16_to_f64(w["k_norm"]), m.rms_eps)
            qs.append(rope_rotate(qu, p, m.rope_theta))
            self.k_cache[local, sl, :, p] = round_to_bf16(rope_rotate(ku, p, m.rope_theta))
            self.v_cache[local, sl, :, p] = round_to_bf16(v[u])
        o = np.empty((b, hq * hd), dtype=np.float64)
        for u in range(b):
            p, sl = int(positions[u]), int(slots[u])
            kc = bf16_to_f64(self.k_cache[local, sl, :, : p + 1])
            vc = bf16_to_f64(self.v_cache[local, sl, :, : p + 1])
            o[u] = attention_gqa(qs[u], kc, vc).reshape(hq * hd)
        h = h + gemv(matrix_f64(w["wo"]), o)
        y = rms_norm(h, bf16_to_f64(w["ffn_norm"]), m.rms_eps)
        a = swiglu(gemv(matrix_f64(w["wg"]), y), gemv(matrix_f64(w["wu"]), y))
        return h + gemv(matrix_f64(w["wd"]), a)

    def decode(self, positions, token_ids=None, hidden_in=None, capture: bool = False, users=None) -> dict:
        """One decode step for users ``0..b-1`` (``users``: row b serves user users[b]).  Returns
        ``hidden_out`` (fp64 ``[b][d]``), and with ``logits_out``: ``next_ids``, ``margins``
        (top-2 logit gap) and ``logits``; with ``capture``: ``per_layer`` (hidden after each
        block, ``[n][b][d]``)."""
        positions = np.asarray(positions, dtype=np.int64)
        b = positions.shape[0]
        if b > self.max_batch:
            raise ValueError("batch exceeds max_batch")
        slots = np.arange(b) if users is None else np.asarray(users, dtype=np.int64)
        return self._forward(positions, slots, token_ids, hidden_in, capture)

    def prefill(self, user: int, positions, token_ids=None, hidden_in=None) -> dict:
        """A prompt of one user in one pass: token t at positions[t] attends to the user's cached
        rows up to its position, the prompt's earlier tokens included (causal self-attention over
        the prompt).  Any number of tokens; the results as ``decode`` gives them, per token."""
        positions = np.asarray(positions, dtype=np.int64)
        if len(set(positions.tolist())) != positions.shape[0]:
            raise ValueError("a prompt's positions must be distinct")
        if not 0 <= user < self.max_batch:
            raise ValueError("user outside [0, max_batch)")
        return self._forward(positions, np.full(positions.shape[0], user), token_ids, hidden_in, False)

    def _forward(self, positions, slots, token_ids, hidden_in, capture) -> dict:
        b = positions.shape[0]
        if np.any(positions < 0) or np.any(positions >= self.max_ctx):
            raise ValueError("position outside [0, max_ctx)")
        if self.embed_in:
            ids = np.asarray(token_ids, dtype=np.int64)
            h = bf16_to_f64(self.head["embed"][ids])
        else:
            h = np.array(hidden_in, dtype=np.float64).reshape(b, self.m.d_model)
        per_layer = []
        for local in range(self.l1 - self.l0):
            h = self._block(local, h, positions, slots)
            if capture:
                per_layer.append(h.copy())
        out = {"hidden_out": h}
        if capture:
            out["per_layer"] = np.stack(per_layer) if per_layer else np.zeros((0, b, self.m.d_model))
        if self.logits_out:
            y = rms_norm(h, bf16_to_f64(self.head["final_norm"]), self.m.rms_eps)
            z = gemv(matrix_f64(self.head["lm_head"]), y)
            out["logits"] = z
            out["next_ids"] = np.array([argmax_first(z[u]) for u in range(b)], dtype=np.int32)
            out["margins"] = np.array([top2_margin(z[u]) for u in range(b)])
        return out
