"""Seeded synthetic inputs for the stage-decode path, and the shapes of its workloads.

Both sides of every parity check draw their inputs from here: the CUDA path (through the
device-side twin of this generator, ``csrc/synth.cu``, or through host arrays made here) and
the CPU oracle (host arrays made here).  The module holds none of the method's arithmetic:
only a counter-based random generator and the workload recipes.

Generator (one definition, implemented twice: here in numpy, and in ``csrc/synth.cu``):

* ``key(seed, tag) = mix64(seed XOR (tag * 0xD1B54A32D192ED03))``
* ``draw(key, i)   = mix64(key + (i + 1) * 0x9E3779B97F4A7C15)``   (all mod 2**64)

where ``mix64`` is the SplitMix64 output function of Steele, Lea and Flood, "Fast splittable
pseudorandom number generators" (OOPSLA 2014): ``z ^= z>>30; z *= 0xBF58476D1CE4E5B9;
z ^= z>>27; z *= 0x94D049BB133111EB; z ^= z>>31``.

Value kinds (every float step is a single IEEE fp32 operation, so host and device agree bit
for bit):

* ``normal``: Irwin-Hall sum of the four 16-bit fields of a draw, ``S`` in [0, 4*65535];
  ``z = fp32(S - 131070) * c`` with ``c = fp32(std / sqrt((65536**2 - 1) / 3))``, plus an
  optional fp32 ``mean``; stored as bf16 (round to nearest even).  Mean 0 and standard
  deviation ``std``, bounded at +-3.46 std: a stand-in for the workloads' N(0, std).
* ``int4 words``: the low 32 bits of a draw, i.e. eight independent nibbles uniform on the 16
  codes; read as signed 4-bit integers they are uniform on [-8, 7].
* ``int4 scales``: ``bf16(c1 * (0.5 + U))``, ``U = (draw >> 40) * 2**-24``, with
  ``c1 = fp32(0.02 / sqrt(21.25))`` (21.25 is the variance of a uniform integer on [-8, 7]),
  so a dequantised weight has a standard deviation near 0.02.
* ``token ids``: ``draw % vocab``.
"""
from __future__ import annotations

import concurrent.futures as _cf
import math
import os
from dataclasses import dataclass, replace

import numpy as np

M64 = (1 << 64) - 1
GAMMA = 0x9E3779B97F4A7C15
MIX1 = 0xBF58476D1CE4E5B9
MIX2 = 0x94D049BB133111EB
TAGMUL = 0xD1B54A32D192ED03
IH4_INV_STD = 1.0 / math.sqrt((65536.0 * 65536.0 - 1.0) / 3.0)
INT4_SCALE_C1 = 0.02 / math.sqrt(21.25)

# value kinds shared with the device generator (csrc/synth.cu, kfl_synth_fill)
KIND_NORMAL_BF16 = 0
KIND_INT4_WORDS = 1
KIND_INT4_SCALES_BF16 = 2

_CHUNK = 1 << 21
_THREADS = min(16, os.cpu_count() or 1)


def _chunked(n: int, out: np.ndarray, fill) -> np.ndarray:
    """Run ``fill(c0, c1)`` (which writes out[c0:c1]) over chunks, on threads for large n
    (numpy releases the GIL inside its array loops)."""
    starts = range(0, n, _CHUNK)
    if n > 4 * _CHUNK and _THREADS > 1:
        with _cf.ThreadPoolExecutor(_THREADS) as ex:
            list(ex.map(lambda c0: fill(c0, min(n, c0 + _CHUNK)), starts))
    else:
        for c0 in starts:
            fill(c0, min(n, c0 + _CHUNK))
    return out


def _mix64_int(z: int) -> int:
    z &= M64
    z = ((z ^ (z >> 30)) * MIX1) & M64
    z = ((z ^ (z >> 27)) * MIX2) & M64
    return z ^ (z >> 31)


def stream_key(seed: int, tag: int) -> int:
    """Key of the stream ``(seed, tag)``."""
    return _mix64_int((seed & M64) ^ ((tag * TAGMUL) & M64))


def _mix64(z: np.ndarray) -> np.ndarray:
    z = (z ^ (z >> np.uint64(30))) * np.uint64(MIX1)
    z = (z ^ (z >> np.uint64(27))) * np.uint64(MIX2)
    return z ^ (z >> np.uint64(31))


def draws(key: int, start: int, n: int) -> np.ndarray:
    """``draw(key, i)`` for ``i`` in ``[start, start + n)`` as uint64."""
    idx = np.arange(start + 1, start + n + 1, dtype=np.uint64)
    with np.errstate(over="ignore"):
        z = np.uint64(key) + idx * np.uint64(GAMMA)
        return _mix64(z)


def draws_at(key: int, idx: np.ndarray) -> np.ndarray:
    """``draw(key, i)`` for an arbitrary uint64 index array."""
    idx = np.asarray(idx, dtype=np.uint64)
    with np.errstate(over="ignore"):
        z = np.uint64(key) + (idx + np.uint64(1)) * np.uint64(GAMMA)
        return _mix64(z)


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round fp32 to bf16 (nearest, ties to even) and return the 16-bit patterns."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    nan = (u & np.uint32(0x7FFFFFFF)) > np.uint32(0x7F800000)
    r = (u + np.uint32(0x7FFF) + ((u >> np.uint32(16)) & np.uint32(1))) >> np.uint32(16)
    r = np.where(nan, np.uint32(0x7FC0), r)
    return r.astype(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    return (np.asarray(b, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


def normal_scale(std: float) -> np.float32:
    return np.float32(std * IH4_INV_STD)


def _normal_from_draws(d: np.ndarray, std: float, mean: float) -> np.ndarray:
    m16 = np.uint64(0xFFFF)
    s = (d & m16) + ((d >> np.uint64(16)) & m16) + ((d >> np.uint64(32)) & m16) + (d >> np.uint64(48))
    centred = (s.astype(np.int64) - 131070).astype(np.float32)
    z = centred * normal_scale(std)
    if mean != 0.0:
        z = np.float32(mean) + z
    return z


def normal_bf16(seed: int, tag: int, n: int, std: float, mean: float = 0.0, start: int = 0) -> np.ndarray:
    """``n`` bf16 bit patterns of the ``normal`` kind, stream ``(seed, tag)``, from index ``start``."""
    key = stream_key(seed, tag)
    out = np.empty(n, dtype=np.uint16)

    def fill(c0, c1):
        out[c0:c1] = f32_to_bf16_bits(_normal_from_draws(draws(key, start + c0, c1 - c0), std, mean))
    return _chunked(n, out, fill)


def normal_bf16_at(seed: int, tag: int, idx: np.ndarray, std: float, mean: float = 0.0) -> np.ndarray:
    key = stream_key(seed, tag)
    return f32_to_bf16_bits(_normal_from_draws(draws_at(key, idx), std, mean))


def int4_words(seed: int, tag: int, n: int) -> np.ndarray:
    key = stream_key(seed, tag)
    out = np.empty(n, dtype=np.uint32)

    def fill(c0, c1):
        out[c0:c1] = (draws(key, c0, c1 - c0) & np.uint64(0xFFFFFFFF)).astype(np.uint32)
    return _chunked(n, out, fill)


def int4_scales_bf16(seed: int, tag: int, n: int) -> np.ndarray:
    key = stream_key(seed, tag)
    out = np.empty(n, dtype=np.uint16)
    c1s = np.float32(INT4_SCALE_C1)

    def fill(c0, c1):
        u = (draws(key, c0, c1 - c0) >> np.uint64(40)).astype(np.float32) * np.float32(2.0 ** -24)
        out[c0:c1] = f32_to_bf16_bits(c1s * (np.float32(0.5) + u))
    return _chunked(n, out, fill)


def token_ids(seed: int, tag: int, n: int, vocab: int) -> np.ndarray:
    return (draws(stream_key(seed, tag), 0, n) % np.uint64(vocab)).astype(np.int32)


# --------------------------------------------------------------------------- tags

TENSOR_IDS = {
    "attn_norm": 1, "wq": 2, "wk": 3, "wv": 4, "wo": 5, "ffn_norm": 6,
    "wg": 7, "wu": 8, "wd": 9, "q_norm": 10, "k_norm": 11,
}
HEAD_IDS = {"embed": 1, "final_norm": 2, "lm_head": 3}
SCALES_OFFSET = 32
TAG_KV = 0x4B560000
TAG_HIDDEN = 0x53540000
TAG_IDS = 0x49440000
KV_USER_STRIDE = 1 << 20  # positions per (user, kv head) in the KV stream index; > any max_ctx


def layer_tag(layer: int, name: str, scales: bool = False) -> int:
    return ((layer + 1) << 8) | (TENSOR_IDS[name] + (SCALES_OFFSET if scales else 0))


def head_tag(name: str, scales: bool = False) -> int:
    return HEAD_IDS[name] + (SCALES_OFFSET if scales else 0)


def kv_tag(layer: int, which: int) -> int:
    return TAG_KV + 2 * layer + which


def hidden_tag(step: int) -> int:
    return TAG_HIDDEN + step


def ids_tag(step: int) -> int:
    return TAG_IDS + step


# --------------------------------------------------------------------------- shapes

@dataclass(frozen=True)
class ModelShape:
    n_layers_total: int
    d_model: int
    n_heads: int
    n_kv_heads: int
    head_dim: int
    ffn: int
    vocab: int
    rms_eps: float = 1e-6
    rope_theta: float = 1e6
    weight_fmt: str = "bf16"  # or "int4_g64"
    qk_norm: bool = False

    @property
    def q_dim(self) -> int:
        return self.n_heads * self.head_dim

    @property
    def kv_dim(self) -> int:
        return self.n_kv_heads * self.head_dim

    def matrix_shapes(self) -> dict:
        d, q, kv, f = self.d_model, self.q_dim, self.kv_dim, self.ffn
        return {"wq": (q, d), "wk": (kv, d), "wv": (kv, d), "wo": (d, q),
                "wg": (f, d), "wu": (f, d), "wd": (d, f)}

    def layer_weight_bytes(self) -> int:
        """Bytes of one decoder block's weights as stored (the paper's beta_block)."""
        n = 0
        for (rows, cols) in self.matrix_shapes().values():
            n += matrix_bytes(rows, cols, self.weight_fmt)
        n += 2 * self.d_model * 2
        if self.qk_norm:
            n += 2 * self.head_dim * 2
        return n


def matrix_bytes(rows: int, cols: int, fmt: str) -> int:
    if fmt == "bf16":
        return rows * cols * 2
    return rows * cols // 2 + rows * (cols // 64) * 2


@dataclass(frozen=True)
class Workload:
    """One synthetic decode workload: a stage [l0, l1) of a model, its users and steps."""
    name: str
    model: ModelShape
    l0: int
    l1: int
    embed_in: bool
    logits_out: bool
    batch: int
    contexts: tuple  # pre-filled KV length per user (the position of its first new token)
    steps: int
    seed: int
    splits: tuple = ()  # stage splits run back to back (config 5)

    @property
    def n_layers(self) -> int:
        return self.l1 - self.l0

    @property
    def max_ctx(self) -> int:
        """KV slots per user: the longest context plus every decode step, rounded up to 64."""
        need = max(self.contexts) + self.steps
        return (need + 63) // 64 * 64

    def step_bytes(self, step: int = 0) -> int:
        """Algorithmic HBM bytes of one decode step: every weight once, the KV rows read over
        positions [0, P_b] and the new K/V rows written, embedding rows, lm_head."""
        m = self.model
        n = self.n_layers * m.layer_weight_bytes()
        kv_row = m.kv_dim * 2
        for b in range(self.batch):
            p = self.contexts[b] + step
            n += self.n_layers * (2 * kv_row * (p + 1) + 2 * kv_row)
        if self.embed_in:
            n += self.batch * m.d_model * 2
        if self.logits_out:
            n += matrix_bytes(m.vocab, m.d_model, m.weight_fmt) + m.d_model * 2
        return n


QWEN_TINY = ModelShape(2, 512, 8, 2, 64, 1408, 4096)
QWEN_7B = ModelShape(28, 3584, 28, 4, 128, 18944, 152064)
QWEN_32B = ModelShape(64, 5120, 64, 8, 128, 27648, 152064)
QWEN_72B = ModelShape(80, 8192, 64, 8, 128, 29568, 152064)
QWEN_72B_INT4 = replace(QWEN_72B, weight_fmt="int4_g64")

CONFIGS = {
    1: Workload("tiny-head-body-2L-d512", QWEN_TINY, 0, 2, True, True, 1, (128,), 8, 20260001),
    2: Workload("7B-body-L0-14-b1-ctx2048", QWEN_7B, 0, 14, False, False, 1, (2048,), 64, 20260002),
    3: Workload("32B-head-L56-64-b1-ctx4096", QWEN_32B, 56, 64, True, True, 1, (4096,), 32, 20260003),
    4: Workload("72B-body-10L-b4-ragged", QWEN_72B, 0, 10, False, False, 4, (512, 1536, 3072, 4096), 64,
                20260004),
    5: Workload("72B-int4-80L-b1-ctx8192", QWEN_72B_INT4, 0, 80, True, True, 1, (8192,), 8, 20260005,
                splits=((80,), (13, 67), (27, 53))),
    6: Workload("72B-int4-80L-b4-ctx8192", QWEN_72B_INT4, 0, 80, True, True, 4, (8192,) * 4, 8, 20260005,
                splits=((80,), (13, 67), (27, 53))),
}


# --------------------------------------------------------------------------- host tensors

def layer_weights(model: ModelShape, layer: int, seed: int) -> dict:
    """Host weights of global layer ``layer``: norm gains (bf16 bits ``[n]``), matrices as bf16
    bits ``[out][in]`` or, for int4_g64, ``(words uint32 [out][in/8], scales bf16 [out][in/64])``."""
    w = {}
    for name in ("attn_norm", "ffn_norm"):
        w[name] = normal_bf16(seed, layer_tag(layer, name), model.d_model, 0.02, mean=1.0)
    if model.qk_norm:
        for name in ("q_norm", "k_norm"):
            w[name] = normal_bf16(seed, layer_tag(layer, name), model.head_dim, 0.02, mean=1.0)
    for name, (rows, cols) in model.matrix_shapes().items():
        w[name] = matrix(model.weight_fmt, seed, layer_tag(layer, name), layer_tag(layer, name, True),
                         rows, cols)
    return w


def matrix(fmt: str, seed: int, tag: int, scale_tag: int, rows: int, cols: int):
    if fmt == "bf16":
        return normal_bf16(seed, tag, rows * cols, 0.02).reshape(rows, cols)
    words = int4_words(seed, tag, rows * cols // 8).reshape(rows, cols // 8)
    scales = int4_scales_bf16(seed, scale_tag, rows * cols // 64).reshape(rows, cols // 64)
    return (words, scales)


def head_weights(model: ModelShape, seed: int, embed: bool = True, logits: bool = True) -> dict:
    w = {}
    d, v = model.d_model, model.vocab
    if embed:
        w["embed"] = normal_bf16(seed, head_tag("embed"), v * d, 0.02).reshape(v, d)
    if logits:
        w["final_norm"] = normal_bf16(seed, head_tag("final_norm"), d, 0.02, mean=1.0)
        w["lm_head"] = matrix(model.weight_fmt, seed, head_tag("lm_head"), head_tag("lm_head", True), v, d)
    return w


def kv_prefill(model: ModelShape, layer: int, user: int, length: int, seed: int):
    """K and V of global layer ``layer`` for ``user`` over positions [0, length), bf16 bits
    ``[n_kv_heads][length][head_dim]``, values ~N(0, 1)."""
    hkv, hd = model.n_kv_heads, model.head_dim
    out = []
    for which in (0, 1):
        arr = np.empty((hkv, length, hd), dtype=np.uint16)
        for h in range(hkv):
            start = ((user * hkv + h) * KV_USER_STRIDE) * hd
            arr[h] = normal_bf16(seed, kv_tag(layer, which), length * hd, 1.0, start=start).reshape(length, hd)
        out.append(arr)
    return out[0], out[1]


def hidden_in(model: ModelShape, step: int, batch: int, seed: int) -> np.ndarray:
    """Stage input for ``step``: bf16 N(0, 1) values held as fp32 ``[batch][d_model]``."""
    bits = normal_bf16(seed, hidden_tag(step), batch * model.d_model, 1.0)
    return bf16_bits_to_f32(bits).reshape(batch, model.d_model)


def first_token_ids(model: ModelShape, batch: int, seed: int) -> np.ndarray:
    return token_ids(seed, ids_tag(0), batch, model.vocab)


def positions(work: Workload, step: int) -> np.ndarray:
    return np.array([work.contexts[b] + step for b in range(work.batch)], dtype=np.int32)
