"""The allocation-free greedy head, kfl_head_argmax_noalloc, against the stage decode path.

Some callers cannot allocate device memory (a host whose device memory is all held by its own
pool, or an embedding that forbids allocation from extension code), so this entry point keeps
its scratch in a fixed array inside the library instead of in a stage's workspace.  Its ids must
match those of kfl_stage_decode on a head-return-leg stage (l0 == l1 with KFL_LOGITS_OUT) over
the same hidden states and weights, wherever the top-2 logit margin exceeds the tolerance the
parity tests use; on a near tie both must pick a near-maximal logit.  Two calls in a row share
the scratch, so each test makes two with different inputs and batch sizes.  This file is named
to be collected last.
"""
import numpy as np
import pytest
import torch

import oracle
from gpu_helpers import ID_MARGIN, ensure_built
from paper_2609_34045_gb300 import device_inputs as dev_in
from paper_2609_34045_gb300 import stage as K
from paper_2609_34045_gb300 import workload as wl

pytestmark = pytest.mark.gpu

# d = 320 is 40 lanes' worth of 8-element loads (a ragged second pass), vocab 1000 leaves a
# 40-row last block
SMALL = wl.ModelShape(n_layers_total=3, d_model=320, n_heads=6, n_kv_heads=2, head_dim=64, ffn=712, vocab=1000)


@pytest.fixture(scope="module", autouse=True)
def _built():
    ensure_built()
    torch.cuda.init()


def _tail_stage(model, head_dev):
    cfg = K.model_cfg(model, 64, 4)
    st = K.kfl_stage_create(cfg, model.n_layers_total, model.n_layers_total, K.KFL_LOGITS_OUT)
    K.kfl_stage_load_head(st, head_dev, on_device=True)
    return st


def _stage_ids(st, h):
    b, d = h.shape
    stream = torch.cuda.current_stream().cuda_stream
    pos = torch.zeros(b, dtype=torch.int32, device="cuda")
    out = torch.empty(b, d, dtype=torch.float32, device="cuda")
    nxt = torch.full((b,), -7, dtype=torch.int32, device="cuda")
    K.kfl_stage_decode(st, None, h, pos, b, out, nxt, stream)
    torch.cuda.synchronize()
    return nxt.cpu().numpy()


def _noalloc_ids(model, h, final_norm, lm_head):
    b, d = h.shape
    nxt = torch.full((b,), -7, dtype=torch.int32, device="cuda")
    K.kfl_head_argmax_noalloc(h, final_norm, lm_head, b, d, model.vocab, model.rms_eps, nxt,
                              torch.cuda.current_stream().cuda_stream)
    torch.cuda.synchronize()
    return nxt.cpu().numpy()


def _check_ids(ids_a, ids_b, logits):
    """Equal where the top-2 margin exceeds ID_MARGIN; else both within 2 x ID_MARGIN of the max."""
    for u in range(len(ids_a)):
        z = logits[u]
        top2 = np.sort(z)[-2:]
        if top2[1] - top2[0] > ID_MARGIN:
            assert int(ids_a[u]) == int(ids_b[u]) == int(np.argmax(z)), (u, ids_a, ids_b)
        else:
            for ids in (ids_a, ids_b):
                assert 0 <= int(ids[u]) < len(z) and z[int(ids[u])] >= np.max(z) - 2 * ID_MARGIN


def test_noalloc_head_matches_stage_decode_two_calls():
    m, seed = SMALL, 31
    head = dev_in.head_weights(m, seed, embed=False, logits=True)
    st = _tail_stage(m, head)
    ora = oracle.OracleStage(m, m.n_layers_total, m.n_layers_total, False, True, 4, 64)
    ora.load_head(wl.head_weights(m, seed, embed=False, logits=True))
    free_after_first = None
    for call, batch in enumerate((4, 3)):
        h_np = wl.hidden_in(m, call, batch, seed)
        h = torch.tensor(h_np, device="cuda")
        ids_stage = _stage_ids(st, h)
        ids_noalloc = _noalloc_ids(m, h, head["final_norm"], head["lm_head"])
        o = ora.decode(np.zeros(batch, dtype=np.int32), hidden_in=h_np)
        _check_ids(ids_stage, ids_noalloc, o["logits"])
        torch.cuda.synchronize()
        free = torch.cuda.mem_get_info()[0]
        if free_after_first is None:
            free_after_first = free
        else:
            assert free == free_after_first, "device memory changed across an allocation-free call"
    K.kfl_stage_destroy(st)


def test_noalloc_head_full_vocab_width_two_calls():
    # the 32B model's head: d_model 5120, vocab 152064 (2376 row blocks); margins from an fp32
    # torch product of the same bf16 weights
    m, seed = wl.QWEN_32B, 20260003
    head = dev_in.head_weights(m, seed, embed=False, logits=True)
    st = _tail_stage(m, head)
    g = head["final_norm"].view(torch.bfloat16).float()
    w = head["lm_head"].view(torch.bfloat16)
    for call, batch in enumerate((2, 4)):
        h = torch.tensor(wl.hidden_in(m, call, batch, seed), device="cuda")
        ids_stage = _stage_ids(st, h)
        ids_noalloc = _noalloc_ids(m, h, head["final_norm"], head["lm_head"])
        inv = torch.rsqrt((h * h).mean(dim=1, keepdim=True) + m.rms_eps)
        logits = torch.cat([(h * inv * g) @ w[r:r + 16384].float().t() for r in range(0, m.vocab, 16384)], dim=1)
        _check_ids(ids_stage, ids_noalloc, logits.double().cpu().numpy())
    K.kfl_stage_destroy(st)


def test_noalloc_head_rejects_sizes_beyond_its_scratch():
    m = SMALL
    head = dev_in.head_weights(m, 32, embed=False, logits=True)
    h = torch.zeros(1, m.d_model, device="cuda")
    nxt = torch.zeros(5, dtype=torch.int32, device="cuda")
    for batch, d, vocab in ((5, m.d_model, m.vocab), (1, m.d_model, 262145), (1, 16392, m.vocab), (1, 324, m.vocab)):
        with pytest.raises(RuntimeError, match="outside the static scratch's limits"):
            K.kfl_head_argmax_noalloc(h, head["final_norm"], head["lm_head"], batch, d, vocab, m.rms_eps, nxt)
    with pytest.raises(RuntimeError, match="16-byte aligned"):
        K.kfl_head_argmax_noalloc(h.view(-1)[1:], head["final_norm"], head["lm_head"], 1, 8, 8, m.rms_eps, nxt)
