"""Pins of the CPU oracle to things other than itself (no GPU).

Each pin checks the oracle against a value fixed by the mathematics, a textbook or library
routine that the special case reduces to, an invariant, or brute force on tiny inputs.  The
``planted`` tests put a plausible mistake into the oracle (on the CPU) and check that at
least one pin fails, so the pins are known to be sharp.
"""
import math
import os

import numpy as np
import pytest
import torch
import torch.nn.functional as F

import oracle
import oracle.stage as ost
from paper_2609_34045_gb300 import workload as wl

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")
rng = np.random.default_rng(1234)


def _read_pairs(name):
    rows = []
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.split("#")[0].strip()
            if line:
                a, b = line.split()
                rows.append((a, b))
    return rows


# --------------------------------------------------------------------------- pins

def pin_bf16_golden():
    for fbits, bbits in _read_pairs("bf16_rne.txt"):
        f = np.array([int(fbits, 16)], dtype=np.uint32).view(np.float32).astype(np.float64)
        got = int(oracle.round_to_bf16(f)[0])
        assert got == int(bbits, 16), (fbits, hex(got), bbits)


def pin_bf16_vs_torch():
    x = np.concatenate([rng.standard_normal(20000) * 10.0 ** rng.integers(-30, 30, 20000),
                        rng.standard_normal(1000)])
    want = torch.from_numpy(x).to(torch.float32).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(oracle.round_to_bf16(x), want)
    # exact round trip of every finite bf16 pattern
    b = np.arange(0, 1 << 16, dtype=np.uint32).astype(np.uint16)
    f = oracle.bf16_to_f64(b)
    fin = np.isfinite(f)
    assert np.array_equal(oracle.round_to_bf16(f[fin]), b[fin])
    tf = torch.from_numpy(b.view(np.int16)).view(torch.bfloat16).to(torch.float64).numpy()
    assert np.array_equal(f[fin], tf[fin])


def pin_int4_exhaustive():
    table = {int(a, 16): int(b) for a, b in _read_pairs("int4_codes.txt")}
    for v in range(16):
        for j in range(8):
            word = np.array([[v << (4 * j)]], dtype=np.uint64).astype(np.uint32)
            codes = oracle.int4_codes(word)[0]
            want = np.zeros(8, dtype=np.int64)
            want[j] = table[v]
            assert np.array_equal(codes.astype(np.int64), want), (v, j, codes)


def pin_int4_groups():
    # one row, K = 128: two groups; scale 0 = 0.5, scale 1 = -2.0 (both exact in bf16)
    words = np.full((1, 16), 0x11111111, dtype=np.uint32)  # every code = 1
    scales = oracle.round_to_bf16(np.array([[0.5, -2.0]]))
    w = oracle.dequant_int4_g64(words, scales)[0]
    assert np.all(w[:64] == 0.5) and np.all(w[64:] == -2.0)


def pin_gemv_bruteforce():
    for (n, k, b) in [(3, 5, 1), (7, 4, 2), (1, 9, 3)]:
        w = rng.integers(-7, 8, size=(n, k)).astype(np.float64)
        x = rng.integers(-7, 8, size=(b, k)).astype(np.float64)
        y = oracle.gemv(w, x)
        assert y.shape == (b, n)
        for bb in range(b):
            for i in range(n):
                s = 0.0
                for j in range(k):
                    s += w[i, j] * x[bb, j]
                assert y[bb, i] == s


def pin_rms_norm():
    for eps in (1e-6, 0.5):
        h = rng.standard_normal((3, 40)) * 3
        y = oracle.rms_norm(h, np.ones(40), eps)
        ms = np.mean(h * h, axis=-1)
        got = np.sqrt(np.mean(y * y, axis=-1))
        assert np.allclose(got, np.sqrt(ms / (ms + eps)), rtol=1e-12)
        # constant vector c -> c / sqrt(c^2 + eps)
        c = 1.7
        yc = oracle.rms_norm(np.full((1, 16), c), np.ones(16), eps)
        assert np.allclose(yc, c / math.sqrt(c * c + eps), rtol=1e-14)
        g = rng.standard_normal(40)
        want = F.rms_norm(torch.from_numpy(h), (40,), weight=torch.from_numpy(g), eps=eps).numpy()
        assert np.allclose(oracle.rms_norm(h, g, eps), want, rtol=1e-12, atol=1e-14)


def pin_rope():
    hd, theta = 16, 1e6
    x = rng.standard_normal((3, hd))
    assert np.array_equal(oracle.rope_rotate(x, 0, theta), x)
    for p in (1, 7, 4095):
        r = oracle.rope_rotate(x, p, theta)
        assert np.allclose(np.linalg.norm(r, axis=-1), np.linalg.norm(x, axis=-1), rtol=1e-13)
    # complex form: z_i = x_i + i x_{i+hd/2}, multiplied by exp(i * p * theta^(-2i/hd))
    p = 5
    z = x[:, : hd // 2] + 1j * x[:, hd // 2:]
    freq = np.array([theta ** (-(2.0 * i) / hd) for i in range(hd // 2)])
    zr = z * np.exp(1j * p * freq)
    want = np.concatenate([zr.real, zr.imag], axis=-1)
    assert np.allclose(oracle.rope_rotate(x, p, theta), want, rtol=1e-12, atol=1e-14)
    # only the distance between positions matters for the score
    q, k = rng.standard_normal((1, hd)), rng.standard_normal((1, hd))
    for m, n in [(9, 4), (100, 37), (3000, 2999)]:
        lhs = float((oracle.rope_rotate(q, m, theta) @ oracle.rope_rotate(k, n, theta).T)[0, 0])
        rhs = float((oracle.rope_rotate(q, m - n, theta) @ k.T)[0, 0])
        assert abs(lhs - rhs) < 1e-10 * (1 + abs(rhs))


def pin_softmax():
    s = rng.standard_normal((5, 33)) * 20
    p = oracle.softmax(s)
    assert np.all(np.abs(p.sum(-1) - 1.0) <= 1e-12)
    import scipy.special
    assert np.allclose(p, scipy.special.softmax(s, axis=-1), rtol=1e-12)


def pin_attention():
    hq, hkv, hd = 6, 2, 8
    q = rng.standard_normal((hq, hd))
    # one cached position: the output is that position's V
    k1, v1 = rng.standard_normal((hkv, 1, hd)), rng.standard_normal((hkv, 1, hd))
    o = oracle.attention_gqa(q, k1, v1)
    for h in range(hq):
        assert np.array_equal(o[h], v1[h // 3, 0])
    # identical keys: uniform weights, output is the mean of V
    kk = np.repeat(rng.standard_normal((hkv, 1, hd)), 9, axis=1)
    vv = rng.standard_normal((hkv, 9, hd))
    o = oracle.attention_gqa(q, kk, vv)
    for h in range(hq):
        assert np.allclose(o[h], vv[h // 3].mean(0), rtol=1e-12, atol=1e-14)
    # library routine: scaled dot-product attention with KV heads repeated per group
    T = 13
    k, v = rng.standard_normal((hkv, T, hd)), rng.standard_normal((hkv, T, hd))
    tq = torch.from_numpy(q)[:, None, :]
    tk = torch.from_numpy(k).repeat_interleave(hq // hkv, 0)
    tv = torch.from_numpy(v).repeat_interleave(hq // hkv, 0)
    want = F.scaled_dot_product_attention(tq, tk, tv)[:, 0, :].numpy()
    assert np.allclose(oracle.attention_gqa(q, k, v), want, rtol=1e-12, atol=1e-14)


def pin_silu():
    assert oracle.silu(np.array([0.0]))[0] == 0.0
    assert abs(oracle.silu(np.array([1.0]))[0] - 0.7310585786300049) < 1e-15  # 1/(1+e^-1)
    assert abs(oracle.silu(np.array([-1.0]))[0] + 0.2689414213699951) < 1e-15  # -1/(1+e)
    x = rng.standard_normal(100) * 5
    assert np.allclose(oracle.silu(x), F.silu(torch.from_numpy(x)).numpy(), rtol=1e-14)
    u = rng.standard_normal(100)
    assert np.allclose(oracle.swiglu(x, u), F.silu(torch.from_numpy(x)).numpy() * u, rtol=1e-14)


def pin_argmax():
    z = np.array([1.0, 3.0, -2.0, 3.0, 0.5])
    assert oracle.argmax_first(z) == 1
    assert oracle.top2_margin(z) == 0.0
    z2 = rng.standard_normal(1000)
    assert oracle.argmax_first(z2) == int(np.argmax(z2))
    assert oracle.top2_margin(np.array([0.25, 1.5, 1.0])) == 0.5


# --------------------------------------------------------------------------- whole stage

SMALL = wl.ModelShape(n_layers_total=3, d_model=64, n_heads=4, n_kv_heads=2, head_dim=16, ffn=96,
                      vocab=50, rms_eps=1e-6, rope_theta=1e4)


def _small_stage(l0, l1, embed, logits, seed=77, max_ctx=32, batch=2, fill=(5, 9), model=SMALL):
    st = oracle.OracleStage(model, l0, l1, embed, logits, batch, max_ctx)
    for i, l in enumerate(range(l0, l1)):
        st.load_layer(i, wl.layer_weights(model, l, seed))
        for u in range(batch):
            k, v = wl.kv_prefill(model, l, u, fill[u], seed)
            st.set_kv(i, u, k, v)
    st.load_head(wl.head_weights(model, seed, embed, logits))
    return st


def _int4_by_lut(m):
    """int4 group-64 matrix -> fp64 through the golden code table (not the oracle's unpack)."""
    table = {int(a, 16): int(b) for a, b in _read_pairs("int4_codes.txt")}
    lut = np.array([table[v] for v in range(16)], dtype=np.float64)
    words, scales = m
    nib = np.stack([(words >> np.uint32(4 * j)) & np.uint32(15) for j in range(8)], -1)
    codes = lut[nib.reshape(words.shape[0], -1)]
    s = torch.from_numpy(scales.view(np.int16)).view(torch.bfloat16).to(torch.float64).numpy()
    return torch.from_numpy(codes * np.repeat(s, 64, axis=1))


def _torch_stage(model, layers, head, kcache, vcache, positions, ids):
    """An independent restatement with torch fp64 library ops (F.rms_norm, F.linear, complex
    rotation, F.scaled_dot_product_attention, F.silu, torch.argmax); bf16 decoded by torch."""
    def bf(bits):
        if isinstance(bits, tuple):
            return _int4_by_lut(bits)
        return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16).to(torch.float64)
    d, hq, hkv, hd = model.d_model, model.n_heads, model.n_kv_heads, model.head_dim
    h = bf(head["embed"][ids])
    kc = [bf(k.copy()) for k in kcache]
    vc = [bf(v.copy()) for v in vcache]
    freq = torch.tensor([model.rope_theta ** (-(2.0 * i) / hd) for i in range(hd // 2)], dtype=torch.float64)
    for li, w in enumerate(layers):
        y = F.rms_norm(h, (d,), weight=bf(w["attn_norm"]), eps=model.rms_eps)
        q = F.linear(y, bf(w["wq"])).view(-1, hq, hd)
        k = F.linear(y, bf(w["wk"])).view(-1, hkv, hd)
        v = F.linear(y, bf(w["wv"])).view(-1, hkv, hd)
        outs = []
        for u, p in enumerate(positions):
            rot = torch.polar(torch.ones_like(freq), p * freq)

            def rope(x):
                z = torch.complex(x[:, : hd // 2], x[:, hd // 2:]) * rot
                return torch.cat([z.real, z.imag], dim=-1)
            qu, ku = rope(q[u]), rope(k[u])
            kc[li][u, :, p] = ku.to(torch.float32).to(torch.bfloat16).to(torch.float64)
            vc[li][u, :, p] = v[u].to(torch.float32).to(torch.bfloat16).to(torch.float64)
            K = kc[li][u, :, : p + 1].repeat_interleave(hq // hkv, 0)
            V = vc[li][u, :, : p + 1].repeat_interleave(hq // hkv, 0)
            outs.append(F.scaled_dot_product_attention(qu[:, None, :], K, V)[:, 0, :].reshape(-1))
        h = h + F.linear(torch.stack(outs), bf(w["wo"]))
        y = F.rms_norm(h, (d,), weight=bf(w["ffn_norm"]), eps=model.rms_eps)
        h = h + F.linear(F.silu(F.linear(y, bf(w["wg"]))) * F.linear(y, bf(w["wu"])), bf(w["wd"]))
    y = F.rms_norm(h, (d,), weight=bf(head["final_norm"]), eps=model.rms_eps)
    z = F.linear(y, bf(head["lm_head"]))
    return h.numpy(), z.numpy(), torch.argmax(z, dim=-1).numpy(), kc, vc


def _check_stage_vs_torch(model, n_layers):
    st = _small_stage(0, n_layers, True, True, model=model)
    k0 = [st.k_cache[i].copy() for i in range(n_layers)]
    v0 = [st.v_cache[i].copy() for i in range(n_layers)]
    ids = np.array([7, 41]) % model.vocab
    pos = np.array([5, 9])
    out = st.decode(pos, token_ids=ids)
    layers = [st.layers[i] for i in range(n_layers)]
    h, z, am, kc, vc = _torch_stage(model, layers, st.head, k0, v0, pos, ids)
    assert np.allclose(out["hidden_out"], h, rtol=1e-11, atol=1e-12)
    assert np.allclose(out["logits"], z, rtol=1e-11, atol=1e-12)
    assert np.array_equal(out["next_ids"], am)
    for i in range(n_layers):
        assert np.array_equal(oracle.bf16_to_f64(st.k_cache[i]), kc[i].numpy())
        assert np.array_equal(oracle.bf16_to_f64(st.v_cache[i]), vc[i].numpy())


def pin_stage_vs_torch():
    _check_stage_vs_torch(SMALL, 3)


def pin_kv_slots():
    st = _small_stage(0, 2, True, False)
    k0, v0 = st.k_cache.copy(), st.v_cache.copy()
    pos = np.array([5, 9])
    st.decode(pos, token_ids=np.array([1, 2]))
    for u, p in enumerate(pos):
        other = np.ones(st.max_ctx, dtype=bool)
        other[p] = False
        assert np.array_equal(st.k_cache[:, u][:, :, other], k0[:, u][:, :, other])
        assert np.array_equal(st.v_cache[:, u][:, :, other], v0[:, u][:, :, other])
        assert not np.array_equal(st.k_cache[:, u, :, p], k0[:, u, :, p])


def pin_stage_split_associativity():
    full = _small_stage(0, 3, True, True)
    a = _small_stage(0, 1, True, False)
    b = _small_stage(1, 3, False, True)
    pos = np.array([5, 9])
    ids = np.array([3, 44])
    for step in range(3):
        p = pos + step
        o_full = full.decode(p, token_ids=ids, capture=True)
        o_a = a.decode(p, token_ids=ids, capture=True)
        o_b = b.decode(p, hidden_in=o_a["hidden_out"], capture=True)
        assert np.array_equal(o_full["hidden_out"], o_b["hidden_out"])
        assert np.array_equal(o_full["per_layer"], np.concatenate([o_a["per_layer"], o_b["per_layer"]]))
        assert np.array_equal(o_full["next_ids"], o_b["next_ids"])
        assert np.array_equal(full.k_cache[1:], b.k_cache) and np.array_equal(full.k_cache[:1], a.k_cache)
        ids = o_full["next_ids"]


def _torch_prefill(model, layers, head, kcache, vcache, start, ids, causal=True):
    """A prompt of one user (cache [layer][Hkv][ctx][hd] bf16 bits, filled below `start`) in
    matrix form: every token's K/V appended at start + t, then one masked attention with torch's
    F.scaled_dot_product_attention, token t seeing cache rows <= start + t (causal=False: the
    whole prompt, to show the check can fail)."""
    def bf(bits):
        if isinstance(bits, tuple):
            return _int4_by_lut(bits)
        return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16).to(torch.float64)
    d, hq, hkv, hd = model.d_model, model.n_heads, model.n_kv_heads, model.head_dim
    T = len(ids)
    h = bf(head["embed"][ids])
    kc = [bf(k.copy()) for k in kcache]
    vc = [bf(v.copy()) for v in vcache]
    pos = torch.arange(start, start + T, dtype=torch.float64)
    freq = torch.tensor([model.rope_theta ** (-(2.0 * i) / hd) for i in range(hd // 2)], dtype=torch.float64)
    rot = torch.polar(torch.ones(T, hd // 2, dtype=torch.float64), pos[:, None] * freq[None, :])

    def rope(x):  # [T][heads][hd]
        z = torch.complex(x[..., : hd // 2], x[..., hd // 2:]) * rot[:, None, :]
        return torch.cat([z.real, z.imag], dim=-1)
    ctx = start + T
    seen = torch.arange(ctx)[None, :] <= (start + torch.arange(T))[:, None]
    mask = seen if causal else torch.ones(T, ctx, dtype=torch.bool)
    for li, w in enumerate(layers):
        y = F.rms_norm(h, (d,), weight=bf(w["attn_norm"]), eps=model.rms_eps)
        q = rope(F.linear(y, bf(w["wq"])).view(T, hq, hd))
        k = rope(F.linear(y, bf(w["wk"])).view(T, hkv, hd))
        v = F.linear(y, bf(w["wv"])).view(T, hkv, hd)
        kc[li][:, start:ctx] = k.transpose(0, 1).to(torch.float32).to(torch.bfloat16).to(torch.float64)
        vc[li][:, start:ctx] = v.transpose(0, 1).to(torch.float32).to(torch.bfloat16).to(torch.float64)
        K = kc[li][:, :ctx].repeat_interleave(hq // hkv, 0)
        V = vc[li][:, :ctx].repeat_interleave(hq // hkv, 0)
        o = F.scaled_dot_product_attention(q.transpose(0, 1), K, V, attn_mask=mask)  # [hq][T][hd]
        h = h + F.linear(o.transpose(0, 1).reshape(T, hq * hd), bf(w["wo"]))
        y = F.rms_norm(h, (d,), weight=bf(w["ffn_norm"]), eps=model.rms_eps)
        h = h + F.linear(F.silu(F.linear(y, bf(w["wg"]))) * F.linear(y, bf(w["wu"])), bf(w["wd"]))
    y = F.rms_norm(h, (d,), weight=bf(head["final_norm"]), eps=model.rms_eps)
    z = F.linear(y, bf(head["lm_head"]))
    return h.numpy(), z.numpy(), kc, vc


def _check_prefill_vs_torch(model, n_layers):
    # user 1 (9 cached rows) takes a prompt of 6 tokens at positions 9..14; user 0 is untouched
    st = _small_stage(0, n_layers, True, True, model=model)
    k0 = [st.k_cache[i, 1].copy() for i in range(n_layers)]
    v0 = [st.v_cache[i, 1].copy() for i in range(n_layers)]
    other = (st.k_cache[:, 0].copy(), st.v_cache[:, 0].copy())
    ids = np.array([3, 44, 17, 17, 0, 39]) % model.vocab
    out = st.prefill(1, np.arange(9, 15), token_ids=ids)
    layers = [st.layers[i] for i in range(n_layers)]
    h, z, kc, vc = _torch_prefill(model, layers, st.head, k0, v0, 9, ids)
    assert np.allclose(out["hidden_out"], h, rtol=1e-11, atol=1e-12)
    assert np.allclose(out["logits"], z, rtol=1e-11, atol=1e-12)
    for i in range(n_layers):
        assert np.array_equal(oracle.bf16_to_f64(st.k_cache[i, 1]), kc[i].numpy())
        assert np.array_equal(oracle.bf16_to_f64(st.v_cache[i, 1]), vc[i].numpy())
    assert np.array_equal(st.k_cache[:, 0], other[0]) and np.array_equal(st.v_cache[:, 0], other[1])
    # the same check without the causal mask fails: it tests what each token sees
    h_all, _, _, _ = _torch_prefill(model, layers, st.head, k0, v0, 9, ids, causal=False)
    assert not np.allclose(out["hidden_out"], h_all, rtol=1e-6, atol=1e-6)


def pin_prefill_vs_torch():
    _check_prefill_vs_torch(SMALL, 3)


def pin_prefill_is_sequential_decode():
    # one pass over the prompt equals one decode step per token (and from an empty cache)
    for start in (0, 9):
        a = _small_stage(0, 3, True, True)
        b = _small_stage(0, 3, True, True)
        ids = np.array([8, 1, 30, 30, 12])
        pa = a.prefill(1, np.arange(start, start + 5), token_ids=ids)
        for t in range(5):
            ob = b.decode(np.array([start + t]), token_ids=ids[t:t + 1], users=[1])
            assert np.allclose(pa["hidden_out"][t], ob["hidden_out"][0], rtol=1e-12, atol=1e-13)
            assert pa["next_ids"][t] == ob["next_ids"][0]
        assert np.array_equal(a.k_cache, b.k_cache) and np.array_equal(a.v_cache, b.v_cache)


def pin_prefill_in_two_calls():
    # a prompt prefilled in two calls (the second attending to the first's cache rows) equals one call
    a = _small_stage(0, 3, True, True)
    b = _small_stage(0, 3, True, True)
    ids = np.array([8, 1, 30, 30, 12, 7, 49])
    one = a.prefill(0, np.arange(5, 12), token_ids=ids)
    first = b.prefill(0, np.arange(5, 8), token_ids=ids[:3])
    second = b.prefill(0, np.arange(8, 12), token_ids=ids[3:])
    both = np.concatenate([first["hidden_out"], second["hidden_out"]])
    assert np.allclose(one["hidden_out"], both, rtol=1e-12, atol=1e-13)
    assert np.array_equal(one["next_ids"], np.concatenate([first["next_ids"], second["next_ids"]]))
    assert np.array_equal(a.k_cache, b.k_cache) and np.array_equal(a.v_cache, b.v_cache)


def pin_steps_of_several_users_in_one_call():
    # two users' rows over three steps in one call (rows at positions P_u + s, each on its user's
    # slot) equal the three steps one at a time: a row sees its user's rows of earlier steps and
    # no later ones, and the other user's slot not at all
    def stage():
        st = oracle.OracleStage(SMALL, 0, 3, False, False, 6, 32)
        for i in range(3):
            st.load_layer(i, wl.layer_weights(SMALL, i, 78))
            for u, n in enumerate((5, 11)):
                st.set_kv(i, u, *wl.kv_prefill(SMALL, i, u, n, 78))
        return st
    a, b = stage(), stage()
    hid = [wl.hidden_in(SMALL, s, 2, 78) for s in range(3)]
    pos = [np.array([5 + s, 11 + s]) for s in range(3)]
    one = a.decode(np.concatenate(pos), hidden_in=np.concatenate(hid), users=[0, 1] * 3, capture=True)
    for s in range(3):
        o = b.decode(pos[s], hidden_in=hid[s], capture=True)
        assert np.allclose(one["hidden_out"][2 * s:2 * s + 2], o["hidden_out"], rtol=1e-12, atol=1e-13)
        assert np.allclose(one["per_layer"][:, 2 * s:2 * s + 2], o["per_layer"], rtol=1e-12, atol=1e-13)
    assert np.array_equal(a.k_cache, b.k_cache) and np.array_equal(a.v_cache, b.v_cache)


SMALL_INT4 = wl.ModelShape(n_layers_total=2, d_model=128, n_heads=4, n_kv_heads=2, head_dim=32, ffn=192,
                           vocab=40, weight_fmt="int4_g64")


def pin_int4_stage_vs_torch():
    _check_stage_vs_torch(SMALL_INT4, 2)


def pin_int4_prefill_vs_torch():
    # int4 weights decoded through the golden code table on the torch side
    _check_prefill_vs_torch(SMALL_INT4, 2)


PINS = [pin_bf16_golden, pin_bf16_vs_torch, pin_int4_exhaustive, pin_int4_groups, pin_gemv_bruteforce,
        pin_rms_norm, pin_rope, pin_softmax, pin_attention, pin_silu, pin_argmax, pin_stage_vs_torch,
        pin_kv_slots, pin_stage_split_associativity, pin_int4_stage_vs_torch, pin_prefill_vs_torch,
        pin_prefill_is_sequential_decode, pin_int4_prefill_vs_torch, pin_prefill_in_two_calls,
        pin_steps_of_several_users_in_one_call]


@pytest.mark.parametrize("pin", PINS, ids=[p.__name__ for p in PINS])
def test_pin(pin):
    pin()


# --------------------------------------------------------------------------- planted mistakes

def _rope_interleaved(x, pos, theta):
    x = np.asarray(x, dtype=np.float64)
    hd = x.shape[-1]
    a = oracle.rope_angles(pos, hd, theta)
    c, s = np.cos(a), np.sin(a)
    x1, x2 = x[..., 0::2], x[..., 1::2]
    out = np.empty_like(x)
    out[..., 0::2] = x1 * c - x2 * s
    out[..., 1::2] = x2 * c + x1 * s
    return out


def _rope_sign(x, pos, theta):
    x = np.asarray(x, dtype=np.float64)
    hd = x.shape[-1]
    a = oracle.rope_angles(pos, hd, theta)
    c, s = np.cos(a), np.sin(a)
    x1, x2 = x[..., : hd // 2], x[..., hd // 2:]
    return np.concatenate([x1 * c + x2 * s, x2 * c - x1 * s], axis=-1)


def _rms_no_eps(h, g, eps):
    h = np.asarray(h, dtype=np.float64)
    return h / np.sqrt(np.mean(h * h, axis=-1, keepdims=True)) * g


def _attn_mod_group(q, k, v):
    hq, hd = q.shape
    hkv = k.shape[0]
    out = np.empty((hq, hd))
    for h in range(hq):
        kh = h % hkv
        out[h] = ost.softmax(k[kh] @ q[h] / np.sqrt(hd)) @ v[kh]
    return out


def _attn_no_scale(q, k, v):
    hq, hd = q.shape
    g = hq // k.shape[0]
    return np.stack([ost.softmax(k[h // g] @ q[h]) @ v[h // g] for h in range(hq)])


def _codes_high_first(words):
    w = np.asarray(words, dtype=np.uint32)
    nib = np.stack([(w >> np.uint32(4 * (7 - j))) & np.uint32(0xF) for j in range(8)], -1).astype(np.int16)
    nib = np.where(nib >= 8, nib - 16, nib).astype(np.int8)
    return nib.reshape(*w.shape[:-1], w.shape[-1] * 8)


def _codes_unsigned(words):
    w = np.asarray(words, dtype=np.uint32)
    nib = np.stack([(w >> np.uint32(4 * j)) & np.uint32(0xF) for j in range(8)], -1).astype(np.int8)
    return nib.reshape(*w.shape[:-1], w.shape[-1] * 8)


def _silu_wrong(x):
    x = np.asarray(x, dtype=np.float64)
    return x / (1.0 + np.exp(x))


def _argmax_last(z):
    z = np.asarray(z)
    return int(np.flatnonzero(z == np.max(z))[-1])


def _gemv_transposed(w, x):
    w = np.asarray(w, dtype=np.float64)
    return np.asarray(x, dtype=np.float64) @ (w if w.shape[0] == w.shape[1] else w.T)


def _round_truncate(x):
    f = np.ascontiguousarray(np.asarray(x, dtype=np.float64).astype(np.float32))
    return (f.view(np.uint32) >> np.uint32(16)).astype(np.uint16)


MUTANTS = {
    "rope_interleaved": ("rope_rotate", _rope_interleaved),
    "rope_sign": ("rope_rotate", _rope_sign),
    "rms_no_eps": ("rms_norm", _rms_no_eps),
    "gqa_modulo": ("attention_gqa", _attn_mod_group),
    "attn_no_scale": ("attention_gqa", _attn_no_scale),
    "int4_high_first": ("int4_codes", _codes_high_first),
    "int4_unsigned": ("int4_codes", _codes_unsigned),
    "silu_sign": ("silu", _silu_wrong),
    "argmax_last": ("argmax_first", _argmax_last),
    "bf16_truncate": ("round_to_bf16", _round_truncate),
}


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_planted_mistake_is_caught(name, monkeypatch):
    attr, fn = MUTANTS[name]
    monkeypatch.setattr(ost, attr, fn)
    monkeypatch.setattr(oracle, attr, fn)
    failed = []
    for pin in PINS:
        try:
            pin()
        except AssertionError:
            failed.append(pin.__name__)
        except Exception:  # a shape error from a transposed operand also counts as caught
            failed.append(pin.__name__)
    assert failed, f"no pin caught the planted mistake {name}"


def test_planted_transposed_gemv_is_caught(monkeypatch):
    monkeypatch.setattr(ost, "gemv", _gemv_transposed)
    monkeypatch.setattr(oracle, "gemv", _gemv_transposed)
    # the block's square O projection (d x Hq*hd = 64 x 64) is where a transposed operand
    # would silently survive; the torch cross-check must catch it
    with pytest.raises(AssertionError):
        pin_stage_vs_torch()


def test_planted_residual_drop_is_caught(monkeypatch):
    orig = ost.OracleStage._block

    def no_residual(self, local, h, positions, slots):
        return orig(self, local, h, positions, slots) - h

    monkeypatch.setattr(ost.OracleStage, "_block", no_residual)
    with pytest.raises(AssertionError):
        pin_stage_vs_torch()
