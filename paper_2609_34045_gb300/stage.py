"""Python binding of the C ABI in ``include/kafila_stage.h`` (argument marshalling only).

Every function here has the name of the C entry point it calls and does nothing but turn
Python objects (numpy arrays, torch tensors, ints) into pointers and structs.  All work of a
decode step runs in the CUDA library ``libkafila_stage.so``; if that library is missing this
module raises instead of falling back to anything else.
"""
from __future__ import annotations

import ctypes as C
import os

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libkafila_stage.so")

KFL_OK = 0
KFL_ERR_ARG, KFL_ERR_RANGE, KFL_ERR_OOM, KFL_ERR_CUDA, KFL_ERR_STATE, KFL_ERR_TIMEOUT = -1, -2, -3, -4, -5, -6
KFL_BF16 = 0
KFL_INT4_G64 = 1
KFL_EMBED_IN = 1
KFL_LOGITS_OUT = 2
KFL_IS_HEAD = 3
KERNEL_KINDS = ("input", "qkv", "attn", "oproj", "gateup", "down", "lmhead", "output")
SYNTH_NORMAL_BF16, SYNTH_INT4_WORDS, SYNTH_INT4_SCALES_BF16 = 0, 1, 2


class KflError(RuntimeError):
    def __init__(self, code: int, where: str):
        self.code = code
        detail = kfl_last_error_detail() if code == -4 else ""
        super().__init__(f"{where}: {kfl_strerror(code)} ({code}){': ' + detail if detail else ''}")


class kfl_model_cfg(C.Structure):
    _fields_ = [("n_layers_total", C.c_int), ("d_model", C.c_int), ("n_heads", C.c_int),
                ("n_kv_heads", C.c_int), ("head_dim", C.c_int), ("ffn", C.c_int), ("vocab", C.c_int),
                ("rms_eps", C.c_float), ("rope_theta", C.c_float), ("weight_fmt", C.c_int),
                ("max_ctx", C.c_int), ("max_batch", C.c_int), ("qk_norm", C.c_int)]


class kfl_matrix(C.Structure):
    _fields_ = [("w", C.c_void_p), ("scales", C.c_void_p)]


class kfl_layer_weights(C.Structure):
    _fields_ = [("attn_norm", C.c_void_p), ("ffn_norm", C.c_void_p)] + \
               [(n, kfl_matrix) for n in ("wq", "wk", "wv", "wo", "wg", "wu", "wd")] + \
               [("q_norm", C.c_void_p), ("k_norm", C.c_void_p)]


class kfl_weights(C.Structure):
    _fields_ = [("n_layers", C.c_int), ("on_device", C.c_int), ("layers", C.POINTER(kfl_layer_weights)),
                ("embed", C.c_void_p), ("final_norm", C.c_void_p), ("lm_head", kfl_matrix)]


class kfl_plan_device(C.Structure):
    _fields_ = [("o", C.c_double), ("bw", C.c_double), ("throughput", C.c_double), ("working_set", C.c_double),
                ("lim_body", C.c_int), ("lim_head", C.c_int)]


class kfl_plan(C.Structure):
    _fields_ = [("tier", C.c_int), ("head", C.c_int), ("tau", C.c_double), ("tau_anchor", C.c_double),
                ("undersized", C.c_int)]


KFL_ERR_INFEASIBLE = -7
KFL_ERR_OVERFLOW = -8

_lib = None


def lib() -> C.CDLL:
    """The loaded CUDA library (raises if it has not been built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is missing: build it first "
                               "(python -m paper_2609_34045_gb300.build); there is no fallback path")
        L = C.CDLL(LIB_PATH)
        vp, i, sz = C.c_void_p, C.c_int, C.c_size_t
        sigs = {
            "kfl_stage_memory_bytes": ([C.POINTER(kfl_model_cfg), i, i, i, C.POINTER(sz)], i),
            "kfl_stage_create": ([C.POINTER(kfl_model_cfg), i, i, i, C.POINTER(vp)], i),
            "kfl_stage_load_weights": ([vp, C.POINTER(kfl_weights)], i),
            "kfl_stage_load_layer": ([vp, i, C.POINTER(kfl_layer_weights), i], i),
            "kfl_stage_load_head": ([vp, vp, vp, C.POINTER(kfl_matrix), i], i),
            "kfl_stage_decode": ([vp, vp, vp, vp, i, vp, vp, vp], i),
            "kfl_stage_decode_host": ([vp, vp, vp, vp, i, vp, vp, vp], i),
            "kfl_stage_decode_users": ([vp, vp, vp, vp, vp, i, vp, vp, vp], i),
            "kfl_stage_prefill": ([vp, vp, vp, vp, i, i, vp, vp, vp], i),
            "kfl_matmul_bf16w": ([vp, i, i, i, vp, i, vp, i, vp], i),
            "kfl_kv_reset": ([vp, i], i),
            "kfl_kv_fill_seeded": ([vp, i, i, C.c_uint64], i),
            "kfl_kv_write": ([vp, i, i, vp, vp, i, i], i),
            "kfl_kv_read": ([vp, i, i, vp, vp, i], i),
            "kfl_stage_debug_capture": ([vp, vp], i),
            "kfl_stage_status": ([vp], i),
            "kfl_stage_trace": ([vp, vp], i),
            "kfl_stage_trace_shape": ([vp, i, C.POINTER(i), C.POINTER(i), C.POINTER(i)], i),
            "kfl_stage_profile": ([vp, i], i),
            "kfl_stage_profile_read": ([vp, C.POINTER(C.c_double), C.POINTER(C.c_int64), i], i),
            "kfl_stage_launches_per_step": ([vp, i], i),
            "kfl_stage_destroy": ([vp], None),
            "kfl_strerror": ([i], C.c_char_p),
            "kfl_last_error_detail": ([], C.c_char_p),
            "kfl_head_argmax_noalloc": ([vp, vp, vp, i, i, i, C.c_float, vp, vp], i),
            "kfl_synth_key": ([C.c_uint64, C.c_uint64], C.c_uint64),
            "kfl_synth_fill": ([vp, C.c_int64, C.c_uint64, C.c_uint64, i, C.c_float, C.c_float, C.c_int64, vp], i),
            "kfl_partition": ([i, i, vp, vp, vp, vp, C.POINTER(C.c_double)], i),
            "kfl_plan_ring": ([i, i, C.POINTER(kfl_plan_device), i, C.c_double, C.c_double, C.c_double, vp,
                               C.POINTER(kfl_plan)], i),
            "kfl_divide": ([i, i, vp, vp], i),
            "kfl_block_limit": ([C.POINTER(kfl_model_cfg), sz, i, C.POINTER(i)], i),
        }
        for name, (args, res) in sigs.items():
            f = getattr(L, name)
            f.argtypes = args
            f.restype = res
        _lib = L
    return _lib


def _ptr(x) -> int | None:
    """Address of a numpy array / torch tensor / int / None."""
    if x is None:
        return None
    if isinstance(x, int):
        return x
    if hasattr(x, "data_ptr"):
        return x.data_ptr()
    if hasattr(x, "ctypes"):
        if not x.flags["C_CONTIGUOUS"]:
            raise ValueError("arrays passed to the library must be C-contiguous")
        return x.ctypes.data
    raise TypeError(f"cannot pass {type(x)} as a pointer")


def _check(rc: int, where: str) -> int:
    if rc < 0:
        raise KflError(rc, where)
    return rc


def kfl_strerror(code: int) -> str:
    return lib().kfl_strerror(code).decode()


def kfl_last_error_detail() -> str:
    return lib().kfl_last_error_detail().decode()


def model_cfg(shape, max_ctx: int, max_batch: int) -> kfl_model_cfg:
    """kfl_model_cfg from a workload.ModelShape."""
    return kfl_model_cfg(shape.n_layers_total, shape.d_model, shape.n_heads, shape.n_kv_heads, shape.head_dim,
                         shape.ffn, shape.vocab, shape.rms_eps, shape.rope_theta,
                         KFL_BF16 if shape.weight_fmt == "bf16" else KFL_INT4_G64, max_ctx, max_batch,
                         1 if shape.qk_norm else 0)


def kfl_stage_memory_bytes(cfg: kfl_model_cfg, l0: int, l1: int, flags: int) -> int:
    out = C.c_size_t(0)
    _check(lib().kfl_stage_memory_bytes(C.byref(cfg), l0, l1, flags, C.byref(out)), "kfl_stage_memory_bytes")
    return out.value


class Stage:
    """A handle from kfl_stage_create; keeps the config it was made with."""

    def __init__(self, handle: int, cfg: kfl_model_cfg, l0: int, l1: int, flags: int):
        self.handle, self.cfg, self.l0, self.l1, self.flags = handle, cfg, l0, l1, flags

    @property
    def n_layers(self) -> int:
        return self.l1 - self.l0

    def __del__(self):
        if getattr(self, "handle", None) and _lib is not None:
            kfl_stage_destroy(self)


def kfl_stage_create(cfg: kfl_model_cfg, l0: int, l1: int, flags: int) -> Stage:
    h = C.c_void_p()
    _check(lib().kfl_stage_create(C.byref(cfg), l0, l1, flags, C.byref(h)), "kfl_stage_create")
    return Stage(h.value, cfg, l0, l1, flags)


def _matrix(m) -> kfl_matrix:
    if isinstance(m, tuple):
        return kfl_matrix(_ptr(m[0]), _ptr(m[1]))
    return kfl_matrix(_ptr(m), None)


def _layer(w: dict) -> kfl_layer_weights:
    lw = kfl_layer_weights()
    lw.attn_norm = _ptr(w["attn_norm"])
    lw.ffn_norm = _ptr(w["ffn_norm"])
    for n in ("wq", "wk", "wv", "wo", "wg", "wu", "wd"):
        setattr(lw, n, _matrix(w[n]))
    lw.q_norm = _ptr(w.get("q_norm"))
    lw.k_norm = _ptr(w.get("k_norm"))
    return lw


def kfl_stage_load_layer(st: Stage, local: int, w: dict, on_device: bool) -> None:
    """``w``: norm gains and matrices as in workload.layer_weights (numpy host arrays, or CUDA
    tensors with on_device=True)."""
    lw = _layer(w)
    _check(lib().kfl_stage_load_layer(st.handle, local, C.byref(lw), int(on_device)), "kfl_stage_load_layer")


def kfl_stage_load_head(st: Stage, head: dict, on_device: bool) -> None:
    lm = _matrix(head["lm_head"]) if "lm_head" in head else kfl_matrix(None, None)
    _check(lib().kfl_stage_load_head(st.handle, _ptr(head.get("embed")), _ptr(head.get("final_norm")),
                                     C.byref(lm), int(on_device)), "kfl_stage_load_head")


def kfl_stage_load_weights(st: Stage, layers: list, head: dict, on_device: bool) -> None:
    arr = (kfl_layer_weights * max(1, len(layers)))(*[_layer(w) for w in layers])
    w = kfl_weights()
    w.n_layers = len(layers)
    w.on_device = int(on_device)
    w.layers = arr
    w.embed = _ptr(head.get("embed"))
    w.final_norm = _ptr(head.get("final_norm"))
    w.lm_head = _matrix(head["lm_head"]) if "lm_head" in head else kfl_matrix(None, None)
    _check(lib().kfl_stage_load_weights(st.handle, C.byref(w)), "kfl_stage_load_weights")


def kfl_stage_decode(st: Stage, token_ids, hidden_in, positions, batch: int, hidden_out, next_ids,
                     cuda_stream: int | None = None) -> None:
    """Device buffers (CUDA tensors): int32 ids [batch], fp32 hidden_in [batch][d], int32
    positions [batch], fp32 hidden_out [batch][d], int32 next_ids [batch].  Asynchronous."""
    _check(lib().kfl_stage_decode(st.handle, _ptr(token_ids), _ptr(hidden_in), _ptr(positions), batch,
                                  _ptr(hidden_out), _ptr(next_ids), cuda_stream), "kfl_stage_decode")


def kfl_stage_decode_users(st: Stage, token_ids, hidden_in, positions, users, batch: int, hidden_out, next_ids,
                           cuda_stream: int | None = None) -> None:
    """kfl_stage_decode with batch row b serving user users[b] (int32 CUDA tensor [batch])."""
    _check(lib().kfl_stage_decode_users(st.handle, _ptr(token_ids), _ptr(hidden_in), _ptr(positions), _ptr(users),
                                        batch, _ptr(hidden_out), _ptr(next_ids), cuda_stream),
           "kfl_stage_decode_users")


def kfl_stage_prefill(st: Stage, token_ids, hidden_in, positions, user: int, n_tokens: int, hidden_out, next_ids,
                      cuda_stream: int | None = None) -> None:
    """n_tokens prompt tokens of one user (KV slot `user`) through the stage (the dense tensor-core
    path, or for short prompts steps of up to max_batch rows): int32 token_ids [n] or fp32
    hidden_in [n][d], int32 positions [n], fp32 hidden_out [n][d], int32 next_ids [n] (CUDA
    tensors).  Asynchronous."""
    _check(lib().kfl_stage_prefill(st.handle, _ptr(token_ids), _ptr(hidden_in), _ptr(positions), user, n_tokens,
                                   _ptr(hidden_out), _ptr(next_ids), cuda_stream), "kfl_stage_prefill")


def kfl_matmul_bf16w(x, T: int, K_: int, ldx: int, w, N: int, y, ldy: int, cuda_stream: int | None = None) -> None:
    """y[T][N] (fp32, row stride ldy) = x[T][K] (fp32, row stride ldx) times w[N][K]^T (bf16 bits)
    on the tensor cores: the prefill's matrix product on its own.  CUDA tensors; synchronous."""
    _check(lib().kfl_matmul_bf16w(_ptr(x), T, K_, ldx, _ptr(w), N, _ptr(y), ldy, cuda_stream), "kfl_matmul_bf16w")


def kfl_stage_decode_host(st: Stage, token_ids, hidden_in, positions, batch: int, hidden_out, next_ids,
                          cuda_stream: int | None = None) -> None:
    """As kfl_stage_decode with host buffers (numpy arrays or pinned CPU tensors); synchronous."""
    _check(lib().kfl_stage_decode_host(st.handle, _ptr(token_ids), _ptr(hidden_in), _ptr(positions), batch,
                                       _ptr(hidden_out), _ptr(next_ids), cuda_stream), "kfl_stage_decode_host")


def kfl_kv_reset(st: Stage, user: int = -1) -> None:
    _check(lib().kfl_kv_reset(st.handle, user), "kfl_kv_reset")


def kfl_kv_fill_seeded(st: Stage, user: int, length: int, seed: int) -> None:
    _check(lib().kfl_kv_fill_seeded(st.handle, user, length, seed), "kfl_kv_fill_seeded")


def kfl_kv_write(st: Stage, local: int, user: int, k, v, length: int, on_device: bool) -> None:
    _check(lib().kfl_kv_write(st.handle, local, user, _ptr(k), _ptr(v), length, int(on_device)), "kfl_kv_write")


def kfl_kv_read(st: Stage, local: int, user: int, k, v, on_device: bool) -> None:
    _check(lib().kfl_kv_read(st.handle, local, user, _ptr(k), _ptr(v), int(on_device)), "kfl_kv_read")


def kfl_stage_debug_capture(st: Stage, per_layer_hidden) -> None:
    _check(lib().kfl_stage_debug_capture(st.handle, _ptr(per_layer_hidden)), "kfl_stage_debug_capture")


def kfl_stage_trace(st: Stage, buf) -> None:
    _check(lib().kfl_stage_trace(st.handle, _ptr(buf)), "kfl_stage_trace")


def kfl_stage_trace_shape(st: Stage, batch: int) -> tuple:
    n, g, sl = C.c_int(), C.c_int(), C.c_int()
    _check(lib().kfl_stage_trace_shape(st.handle, batch, C.byref(n), C.byref(g), C.byref(sl)),
           "kfl_stage_trace_shape")
    return n.value, g.value, sl.value


def kfl_stage_status(st: Stage) -> int:
    """The device error word (0 or a negative code), cleared; does not raise."""
    return lib().kfl_stage_status(st.handle)


def kfl_stage_profile(st: Stage, enable: bool) -> None:
    _check(lib().kfl_stage_profile(st.handle, int(enable)), "kfl_stage_profile")


def kfl_stage_profile_read(st: Stage) -> dict:
    ms = (C.c_double * len(KERNEL_KINDS))()
    n = (C.c_int64 * len(KERNEL_KINDS))()
    _check(lib().kfl_stage_profile_read(st.handle, ms, n, len(KERNEL_KINDS)), "kfl_stage_profile_read")
    return {k: (ms[i], n[i]) for i, k in enumerate(KERNEL_KINDS)}


def kfl_stage_launches_per_step(st: Stage, batch: int) -> int:
    return _check(lib().kfl_stage_launches_per_step(st.handle, batch), "kfl_stage_launches_per_step")


def kfl_stage_destroy(st: Stage) -> None:
    if st.handle:
        lib().kfl_stage_destroy(st.handle)
        st.handle = None


def kfl_head_argmax_noalloc(hidden, final_norm, lm_head, batch: int, d_model: int, vocab: int, rms_eps: float,
                            next_ids, stream=None) -> None:
    """Greedy ids from device buffers without any device allocation (for callers that cannot
    allocate).  hidden fp32 [batch][d_model], final_norm bf16 [d_model], lm_head bf16
    [vocab][d_model] row-major, next_ids int32 [batch]; all device memory.  Enqueued on
    ``stream`` (an int handle or None); the library's static scratch is shared by every call."""
    rc = lib().kfl_head_argmax_noalloc(_ptr(hidden), _ptr(final_norm), _ptr(lm_head), batch, d_model, vocab,
                                       rms_eps, _ptr(next_ids), _ptr(stream))
    if rc < 0:
        raise RuntimeError(f"kfl_head_argmax_noalloc: {kfl_strerror(rc)} ({rc}): {kfl_last_error_detail()}")


def kfl_synth_key(seed: int, tag: int) -> int:
    return lib().kfl_synth_key(seed, tag)


def kfl_synth_fill(dst, n: int, seed: int, tag: int, kind: int, c: float, mean: float = 0.0, start: int = 0,
                   cuda_stream: int | None = None) -> None:
    _check(lib().kfl_synth_fill(_ptr(dst), n, seed, tag, kind, c, mean, start, cuda_stream), "kfl_synth_fill")


# ---- planner (include/kafila_plan.h): host code, no GPU needed ------------------------------

def kfl_partition(k: int, fixed, per, lim):
    """The exact fixed-order division of section V-B: (block counts, bottleneck), or raises
    KflError (KFL_ERR_INFEASIBLE)."""
    import numpy as np
    m = len(fixed)
    f = np.ascontiguousarray(fixed, dtype=np.float64)
    p = np.ascontiguousarray(per, dtype=np.float64)
    li = np.ascontiguousarray(lim, dtype=np.int32)
    n = np.zeros(m, dtype=np.int32)
    tau = C.c_double(0.0)
    _check(lib().kfl_partition(k, m, f.ctypes.data, p.ctypes.data, li.ctypes.data, n.ctypes.data, C.byref(tau)),
           "kfl_partition")
    return n.tolist(), tau.value


def kfl_plan_ring(k: int, devices, anchor: int, beta_block: float, beta_head: float, mu: float = 0.05):
    """(block counts in ring order, kfl_plan fields as a dict, return code); devices: dicts with the
    kfl_plan_device fields.  Does not raise on KFL_ERR_INFEASIBLE (the plan names the device)."""
    import numpy as np
    m = len(devices)
    arr = (kfl_plan_device * m)(*[kfl_plan_device(d.get("o", 0.0), d.get("bw", 0.0), d.get("throughput", 0.0),
                                                  d.get("working_set", 0.0), d["lim_body"], d["lim_head"])
                                  for d in devices])
    n = np.zeros(m, dtype=np.int32)
    plan = kfl_plan()
    rc = lib().kfl_plan_ring(k, m, arr, anchor, beta_block, beta_head, mu, n.ctypes.data, C.byref(plan))
    if rc < 0 and rc != KFL_ERR_INFEASIBLE:
        raise KflError(rc, "kfl_plan_ring")
    return n.tolist(), {f: getattr(plan, f) for f, _ in kfl_plan._fields_}, rc


def kfl_divide(k: int, m: int, weight=None):
    import numpy as np
    n = np.zeros(m, dtype=np.int32)
    w = None if weight is None else np.ascontiguousarray(weight, dtype=np.float64)
    _check(lib().kfl_divide(k, m, None if w is None else w.ctypes.data, n.ctypes.data), "kfl_divide")
    return n.tolist()


def kfl_block_limit(cfg: kfl_model_cfg, room_bytes: int, is_head: bool) -> int:
    out = C.c_int(0)
    _check(lib().kfl_block_limit(C.byref(cfg), room_bytes, 1 if is_head else 0, C.byref(out)), "kfl_block_limit")
    return out.value
