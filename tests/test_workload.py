"""The seeded input generator (no GPU): its published core, determinism and value kinds."""
import numpy as np

from paper_2609_34045_gb300 import workload as wl


def test_splitmix64_published_sequence():
    # SplitMix64 (Steele, Lea, Flood 2014) from state 0: the reference implementation's first
    # three outputs
    d = wl.draws(0, 0, 3)
    assert [int(x) for x in d] == [0xE220A8397B1DCDAF, 0x6E789E6AA1B965F4, 0x06C45D188009454F]


def test_draws_at_matches_range():
    key = wl.stream_key(5, 77)
    idx = np.array([0, 3, 1000, 123456], dtype=np.uint64)
    assert np.array_equal(wl.draws_at(key, idx), wl.draws(key, 0, 123457)[idx.astype(np.int64)])


def test_normal_kind_statistics_and_bounds():
    x = wl.bf16_bits_to_f32(wl.normal_bf16(3, 11, 1_000_000, 0.02)).astype(np.float64)
    assert abs(x.mean()) < 1e-4
    assert abs(x.std() - 0.02) < 2e-4
    assert np.abs(x).max() <= 0.02 * 3.47
    g = wl.bf16_bits_to_f32(wl.normal_bf16(3, 12, 100_000, 0.02, mean=1.0)).astype(np.float64)
    assert abs(g.mean() - 1.0) < 1e-3


def test_chunked_and_threaded_generation_is_position_pure():
    n = 11 * (1 << 21) + 5
    full = wl.normal_bf16(9, 1, n, 1.0)
    part = wl.normal_bf16(9, 1, 1000, 1.0, start=n - 1000)
    assert np.array_equal(full[-1000:], part)
    idx = np.array([0, 7, n - 1], dtype=np.uint64)
    assert np.array_equal(wl.normal_bf16_at(9, 1, idx, 1.0), full[idx.astype(np.int64)])


def test_int4_words_and_scales():
    w = wl.int4_words(1, 2, 200_000)
    nib = np.stack([(w >> np.uint32(4 * j)) & np.uint32(15) for j in range(8)]).ravel()
    counts = np.bincount(nib, minlength=16)
    assert counts.min() > 0.9 * counts.mean() and counts.max() < 1.1 * counts.mean()
    s = wl.bf16_bits_to_f32(wl.int4_scales_bf16(1, 3, 100_000)).astype(np.float64)
    c1 = wl.INT4_SCALE_C1
    assert s.min() >= 0.49 * c1 and s.max() <= 1.51 * c1


def test_kv_prefill_is_independent_of_cache_size():
    m = wl.QWEN_TINY
    k1, v1 = wl.kv_prefill(m, 1, 0, 10, 42)
    k2, v2 = wl.kv_prefill(m, 1, 0, 20, 42)
    assert np.array_equal(k1, k2[:, :10]) and np.array_equal(v1, v2[:, :10])
    k3, _ = wl.kv_prefill(m, 1, 1, 10, 42)
    assert not np.array_equal(k1, k3)


def test_workload_bytes():
    w = wl.CONFIGS[2]
    per_layer = w.model.layer_weight_bytes()
    assert abs(per_layer - 466.1e6) < 0.2e6  # d 3584, F 18944, 28/4 heads of 128
    assert abs(w.step_bytes() - 6.58e9) < 0.02e9
