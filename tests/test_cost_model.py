"""The stage cost model (Eq. 2) that bench.py evaluates against measured stage times: with the
probe's overhead and bandwidth it is the straight line o + bytes / b, and a least-squares fit
recovers (o, b) from points on such a line."""
import bench


def test_probe_prediction_is_overhead_plus_bytes_over_bandwidth():
    r = bench.cost_model([(6e9, 2.0), (12e9, 3.0)], 6000.0, 0.5)["probe"]
    # 0.5 ms + 6e9 B / 6e12 B/s = 1.5 ms, + 12e9 / 6e12 = 2.5 ms
    assert abs(r["pred_ms"][0] - 1.5) < 1e-12 and abs(r["pred_ms"][1] - 2.5) < 1e-12
    assert abs(r["rel_err"][0] - (-0.25)) < 1e-12 and abs(r["rel_err"][1] - (-1 / 6)) < 1e-12
    assert abs(r["median_abs_err"] - (0.25 + 1 / 6) / 2) < 1e-12


def test_fit_recovers_overhead_and_bandwidth():
    o_ms, gbs = 0.02, 4500.0
    pts = [(n, o_ms + n / (gbs * 1e6)) for n in (1e9, 3e9, 7e9, 2e10)]
    f = bench.cost_model(pts, 6000.0, 0.0)["fitted"]
    assert abs(f["o_us"] - 20.0) < 1e-6 and abs(f["b_gbs"] - gbs) < 1e-6
    assert f["median_abs_err"] < 1e-12


def test_block_probe_is_evaluated_like_the_copy_probe():
    pts = [(6e9, 2.0), (12e9, 3.0)]
    r = bench.cost_model(pts, 6000.0, 0.5, block_probe_gbs=4000.0)
    # 0.5 ms + 6e9 B / 4e12 B/s = 2.0 ms (exact), 0.5 + 3.0 = 3.5 ms (+1/6)
    b = r["block_probe"]
    assert abs(b["pred_ms"][0] - 2.0) < 1e-12 and abs(b["pred_ms"][1] - 3.5) < 1e-12
    assert abs(b["median_abs_err"] - (0 + 1 / 6) / 2) < 1e-12
    assert "block_probe" not in bench.cost_model(pts, 6000.0, 0.5)


def test_single_point_has_no_fit():
    assert "fitted" not in bench.cost_model([(1e9, 1.0)], 6000.0, 0.1)
