"""GPU parity of the prompt prefill (kfl_stage_prefill) against the oracle's prefill.

A prompt of one user goes through the stage either as steps of up to max_batch rows on the user's
KV slot (the decode kernels) or densely (tensor-core matrix products over all its tokens, causal
attention over the slot; int4 weights dequantized to fp16 first); the oracle runs the whole prompt
in one pass.  Bar as
for decode: every token's output within max-abs 1e-2 of the oracle's RMS, greedy ids equal where
the oracle's top-2 margin exceeds 1e-2, the user's written cache rows within tolerance and every
other row of every slot bit-identical.
"""
import dataclasses

import numpy as np
import pytest
import torch

from gpu_helpers import HIDDEN_TOL, ID_MARGIN, Pair, ensure_built
from paper_2609_34045_gb300 import stage as K
from paper_2609_34045_gb300 import workload as wl
from test_gpu_parity import RAGGED, RAGGED128, RAGGED_INT4

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    ensure_built()
    torch.cuda.init()


def _prefill(pair, user, start, n, seed, embed):
    """Prefill n tokens of `user` at positions start.. on both sides and compare."""
    d = pair.model.d_model
    positions = np.arange(start, start + n, dtype=np.int32)
    ids = wl.token_ids(seed, 77, n, pair.model.vocab) if embed else None
    hidden = None if embed else wl.hidden_in(pair.model, 3, n, seed)
    o = pair.ora.prefill(user, positions, token_ids=ids, hidden_in=hidden)
    for p in positions:
        pair.written.add((user, int(p)))
    pos = torch.tensor(positions, device="cuda")
    idt = torch.tensor(ids, device="cuda") if embed else None
    hid = None if embed else torch.tensor(hidden, dtype=torch.float32, device="cuda")
    out = torch.zeros(n, d, dtype=torch.float32, device="cuda")
    nxt = torch.full((n,), -7, dtype=torch.int32, device="cuda") if pair.logits else None
    K.kfl_stage_prefill(pair.st, idt, hid, pos, user, n, out, nxt, torch.cuda.current_stream().cuda_stream)
    assert K.kfl_stage_status(pair.st) == 0
    g_out = out.cpu().numpy()
    for t in range(n):
        ref = o["hidden_out"][t]
        err = np.max(np.abs(g_out[t] - ref))
        rms = np.sqrt(np.mean(ref * ref))
        assert err <= HIDDEN_TOL * rms, f"token {t}: max err {err:.3e} > {HIDDEN_TOL} x rms {rms:.3e}"
    if pair.logits:
        g_next = nxt.cpu().numpy()
        for t in range(n):
            if o["margins"][t] > ID_MARGIN:
                assert int(g_next[t]) == int(o["next_ids"][t]), (t, g_next, o["next_ids"])
            else:
                z = o["logits"][t]
                assert z[int(g_next[t])] >= np.max(z) - 2 * ID_MARGIN
    return o


@pytest.fixture(params=["steps", "dense"])
def path(request, monkeypatch):
    """Which prefill path a bf16 stage takes: the decode steps or the dense one."""
    monkeypatch.setenv("KFL_PREFILL_DENSE_MIN", "1" if request.param == "dense" else str(1 << 30))
    return request.param


# (model, stage layers, flags, contexts of users 0..2, prefilled user, tokens, max_ctx): prompts
# that end mid-step (11 = 4 + 4 + 3), fill whole steps, are one token, cross the 64-position
# sub-tiles and the dense path's 128-token tiles, start from an empty cache, and (2100 tokens)
# take two dense passes
CASES = [
    ("bf16-head-ragged", RAGGED, 0, 3, K.KFL_IS_HEAD, (5, 130, 58), 2, 11, 192),
    ("bf16-body-hidden", RAGGED, 1, 3, 0, (17, 40, 61), 1, 8, 192),
    ("bf16-one-token", RAGGED, 0, 2, K.KFL_IS_HEAD, (3, 9, 20), 0, 1, 192),
    ("hd128-empty-cache", RAGGED128, 0, 2, K.KFL_IS_HEAD, (0, 100, 7), 0, 9, 192),
    ("bf16-head-300", RAGGED, 0, 3, K.KFL_IS_HEAD, (5, 30, 70), 2, 300, 448),
    ("hd128-200", RAGGED128, 0, 2, K.KFL_IS_HEAD, (0, 100, 7), 1, 200, 320),
    ("int4-head", RAGGED_INT4, 0, 2, K.KFL_IS_HEAD, (9, 70, 131), 1, 7, 192),
    ("int4-head-260", RAGGED_INT4, 0, 2, K.KFL_IS_HEAD, (9, 70, 131), 2, 260, 448),
    # QK-norm stages prefill through decode steps whatever the prompt length
    ("qknorm-head-40", dataclasses.replace(RAGGED, qk_norm=True), 0, 3, K.KFL_IS_HEAD, (5, 30, 70), 1, 40, 192),
]


@pytest.mark.parametrize("name,model,l0,l1,flags,contexts,user,n,max_ctx", CASES, ids=[c[0] for c in CASES])
def test_prefill_matches_the_oracle(name, model, l0, l1, flags, contexts, user, n, max_ctx, path):
    if path == "steps" and n > 64:
        pytest.skip("long prompts: the dense path only (the steps path is covered by the short ones)")
    p = Pair(model, l0, l1, flags, 3, contexts, max_ctx, seed=23, max_batch=4)
    _prefill(p, user, contexts[user], n, 23, bool(flags & K.KFL_EMBED_IN))
    p.compare_kv()
    p.close()


def test_two_dense_passes(monkeypatch):
    """A prompt longer than one dense pass (2048 tokens): the second pass attends to the first's
    cache rows."""
    monkeypatch.setenv("KFL_PREFILL_DENSE_MIN", "1")
    small = wl.ModelShape(n_layers_total=1, d_model=128, n_heads=2, n_kv_heads=1, head_dim=64, ffn=256,
                          vocab=300)
    p = Pair(small, 0, 1, K.KFL_IS_HEAD, 1, (40,), 2176, seed=37, max_batch=1)
    _prefill(p, 0, 40, 2100, 37, True)
    p.compare_kv()
    p.close()


def test_decode_after_prefill_matches_the_oracle(path):
    """Prefill user 1's prompt, then decode all three users; user 1 continues after its prompt."""
    model, contexts, n = RAGGED, (20, 33, 64), 6
    p = Pair(model, 0, 3, K.KFL_IS_HEAD, 3, contexts, 192, seed=29, max_batch=4)
    _prefill(p, 1, contexts[1], n, 29, True)
    p.contexts = (contexts[0], contexts[1] + n, contexts[2])
    ids = wl.token_ids(29, 79, 3, model.vocab)
    for s in range(2):
        o, _, _ = p.step(s, ids=ids)
        ids = o["next_ids"]
    p.compare_kv()
    p.close()


def test_repeated_position_is_reported(path):
    """Two tokens of one user at the same position in one step: the later one is refused on the
    device (status KFL_ERR_RANGE) and the stage stays usable."""
    p = Pair(RAGGED, 0, 1, K.KFL_IS_HEAD, 2, (5, 6), 64, seed=31, max_batch=4)
    pos = torch.tensor([10, 10], dtype=torch.int32, device="cuda")
    ids = torch.tensor([1, 2], dtype=torch.int32, device="cuda")
    nxt = torch.zeros(2, dtype=torch.int32, device="cuda")
    K.kfl_stage_prefill(p.st, ids, None, pos, 0, 2, None, nxt, torch.cuda.current_stream().cuda_stream)
    assert K.kfl_stage_status(p.st) == -2
    with pytest.raises(K.KflError):
        K.kfl_stage_prefill(p.st, ids, None, pos, 4, 2, None, nxt, None)  # user outside [0, max_batch)
    pos = torch.tensor([10, 11], dtype=torch.int32, device="cuda")
    K.kfl_stage_prefill(p.st, ids, None, pos, 0, 2, None, nxt, torch.cuda.current_stream().cuda_stream)
    assert K.kfl_stage_status(p.st) == 0
    p.close()


def test_int4_dense_prefill_reports_fp16_overflow(monkeypatch):
    """The int4 dense prefill carries activations as fp16 terms.  Host-made RMSNorm gains of 2^17
    make every normalised input larger than fp16 can hold: kfl_stage_status reports
    KFL_ERR_OVERFLOW (a status read back on the host; nothing faults).  The same stage with its
    seeded gains reports nothing."""
    monkeypatch.setenv("KFL_PREFILL_DENSE_MIN", "1")
    m = RAGGED_INT4
    cfg = K.model_cfg(m, 128, 1)
    for big in (False, True):
        st = K.kfl_stage_create(cfg, 0, 1, K.KFL_IS_HEAD)
        w = wl.layer_weights(m, 0, 41)
        if big:
            w["attn_norm"] = np.full(m.d_model, 0x4800, dtype=np.uint16)  # bf16 2^17
        K.kfl_stage_load_layer(st, 0, w, on_device=False)
        K.kfl_stage_load_head(st, wl.head_weights(m, 41), on_device=False)
        n = 20
        ids = torch.tensor(wl.token_ids(41, 5, n, m.vocab), device="cuda")
        pos = torch.arange(n, dtype=torch.int32, device="cuda")
        nxt = torch.zeros(n, dtype=torch.int32, device="cuda")
        K.kfl_stage_prefill(st, ids, None, pos, 0, n, None, nxt, torch.cuda.current_stream().cuda_stream)
        assert K.kfl_stage_status(st) == (K.KFL_ERR_OVERFLOW if big else 0)
        K.kfl_stage_destroy(st)
