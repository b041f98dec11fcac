"""The C-ABI library builds, loads and exports every declared symbol; host-side argument checks
(no GPU needed: nothing here launches a kernel)."""
import glob
import os
import re

import pytest

from paper_2609_34045_gb300 import stage as K
from paper_2609_34045_gb300 import workload as wl

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    if not os.path.exists(K.LIB_PATH):
        from paper_2609_34045_gb300.build import build
        build()
    return K.lib()


def declared_symbols():
    names = set()
    for h in glob.glob(os.path.join(ROOT, "include", "*.h")):
        text = open(h).read()
        text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
        for m in re.finditer(r"\b(kfl_\w+)\s*\(", text):
            names.add(m.group(1))
    return sorted(names)


def test_header_declares_the_boundary():
    names = declared_symbols()
    for required in ("kfl_stage_create", "kfl_stage_load_weights", "kfl_stage_decode", "kfl_kv_reset",
                     "kfl_stage_memory_bytes", "kfl_stage_destroy", "kfl_strerror"):
        assert required in names


def test_every_declared_symbol_is_exported(lib):
    missing = [n for n in declared_symbols() if not hasattr(lib, n)]
    assert not missing, missing


def test_strerror(lib):
    assert K.kfl_strerror(0) == "ok"
    for code in range(-8, 0):
        assert K.kfl_strerror(code) != "unknown error"
    assert K.kfl_strerror(-99) == "unknown error"


def test_memory_bytes_counts_weights_and_cache(lib):
    w = wl.CONFIGS[2]
    cfg = K.model_cfg(w.model, w.max_ctx, w.batch)
    n = K.kfl_stage_memory_bytes(cfg, 0, 14, 0)
    weights = 14 * w.model.layer_weight_bytes()
    kv = 2 * 14 * w.batch * w.model.n_kv_heads * w.max_ctx * w.model.head_dim * 2
    assert weights + kv <= n <= weights + kv + 64 * 2**20
    # the head adds the embedding and the unembedding
    n_head = K.kfl_stage_memory_bytes(cfg, 0, 14, K.KFL_IS_HEAD)
    assert n_head - n >= 2 * w.model.vocab * w.model.d_model * 2


def test_qk_norm_stage_counts_its_gains_and_raw_projection(lib):
    # QK-norm adds two fp32 gains of head_dim per block and one raw Q/K/V row per user
    w = wl.CONFIGS[2]
    cfg = K.model_cfg(w.model, w.max_ctx, w.batch)
    n0 = K.kfl_stage_memory_bytes(cfg, 0, 14, 0)
    cfg.qk_norm = 1
    n1 = K.kfl_stage_memory_bytes(cfg, 0, 14, 0)
    m = w.model
    ld_raw = (m.q_dim + 2 * m.kv_dim + 255) // 256 * 256
    assert n1 - n0 == 14 * 2 * m.head_dim * 4 + 4 * ld_raw * 4


@pytest.mark.parametrize("field,value", [("max_batch", 5), ("max_batch", 0), ("head_dim", 96), ("qk_norm", 2),
                                         ("n_kv_heads", 3), ("max_ctx", 0), ("weight_fmt", 7)])
def test_bad_config_is_refused_before_any_allocation(lib, field, value):
    w = wl.CONFIGS[1]
    cfg = K.model_cfg(w.model, w.max_ctx, 1)
    setattr(cfg, field, value)
    with pytest.raises(K.KflError) as e:
        K.kfl_stage_memory_bytes(cfg, 0, 2, K.KFL_IS_HEAD)
    assert e.value.code == -1
    with pytest.raises(K.KflError) as e:
        K.kfl_stage_create(cfg, 0, 2, K.KFL_IS_HEAD)
    assert e.value.code == -1


@pytest.mark.parametrize("l0,l1,flags", [(-1, 2, 0), (1, 0, 0), (0, 3, 0), (0, 2, 4), (1, 1, 0)])
def test_bad_stage_range_is_refused(lib, l0, l1, flags):
    w = wl.CONFIGS[1]
    cfg = K.model_cfg(w.model, w.max_ctx, 1)
    with pytest.raises(K.KflError) as e:
        K.kfl_stage_create(cfg, l0, l1, flags)
    assert e.value.code == -1


def test_null_handles_are_rejected(lib):
    L = K.lib()
    assert L.kfl_stage_decode(None, None, None, None, 1, None, None, None) == -5
    assert L.kfl_kv_reset(None, -1) == -5
    assert L.kfl_stage_status(None) == -5
    L.kfl_stage_destroy(None)  # no-op


def test_prefill_and_matmul_argument_errors_without_a_gpu(lib):
    """The entry points refuse bad arguments before touching the device."""
    class NoStage:
        handle = None  # a NULL stage pointer

    with pytest.raises(K.KflError) as e:
        K.kfl_stage_prefill(NoStage(), None, None, None, 0, 4, None, None)
    assert e.value.code == K.KFL_ERR_STATE
    for args in ((None, 4, 64, 64, None, 8, None, 8),       # NULL pointers
                 (1 << 20, 0, 64, 64, 1 << 21, 8, 1 << 22, 8),  # T < 1
                 (1 << 20, 4, 64, 60, 1 << 21, 8, 1 << 22, 8),  # ldx < K
                 (1 << 20, 4, 64, 64, 1 << 21, 8, 1 << 22, 6),  # ldy < N
                 (1 << 20, 4, 64, 64, 1 << 21, 8, (1 << 22) + 4, 8)):  # y not 16-byte aligned
        with pytest.raises(K.KflError) as e:
            K.kfl_matmul_bf16w(*args)
        assert e.value.code == K.KFL_ERR_ARG
