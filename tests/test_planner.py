"""Ring planner (the exact fixed-order division, head rotation, admission tiers): the brute-force oracle pinned by
hand-derived cases, then the C library's planner against the oracle on random instances.  Host
code only: no GPU."""
import math
import os
import random

import pytest

from oracle import planner as P
from paper_2609_34045_gb300 import stage as K
from paper_2609_34045_gb300 import workload as wl


@pytest.fixture(scope="module")
def lib():
    if not os.path.exists(K.LIB_PATH):
        from paper_2609_34045_gb300.build import build
        build()
    return K.lib()


# ---- pins of the oracle (values derived by hand) ------------------------------------------

def test_pin_two_equal_devices_split_evenly():
    tau, divs = P.partition(4, [0.0, 0.0], [1.0, 1.0], [10, 10])
    assert tau == 2.0 and divs == [(2, 2)]


def test_pin_speed_ratio_three():
    # max(n1, n2 / 3) with n1 + n2 = 8: (2, 6) gives 2; (1, 7) gives 7/3; (3, 5) gives 3
    tau, divs = P.partition(8, [0.0, 0.0], [1.0, 1.0 / 3.0], [10, 10])
    assert tau == 2.0 and divs == [(2, 6)]


def test_pin_limit_binds():
    tau, divs = P.partition(5, [0.0, 0.0], [1.0, 1.0], [1, 10])
    assert tau == 4.0 and divs == [(1, 4)]


def test_pin_infeasible():
    assert P.partition(5, [0.0, 0.0], [1.0, 1.0], [2, 2]) is None  # limits hold 4 < 5
    assert P.partition(2, [0.0] * 3, [1.0] * 3, [5] * 3) is None    # more devices than blocks


def test_pin_fixed_cost_shifts_blocks():
    # the head term 0.5 on device 0: (1, 3) gives max(1.5, 3) = 3, (2, 2) gives 2.5
    tau, divs = P.partition(4, [0.5, 0.0], [1.0, 1.0], [10, 10])
    assert tau == 2.5 and divs == [(2, 2)]
    tau, divs = P.partition(5, [0.5, 0.0], [1.0, 1.0], [10, 10])
    assert tau == 3.0 and divs == [(2, 3)]


def test_pin_head_rotation_moves_to_the_faster_device():
    # A (bw 1) and B (bw 3), beta_block 1, beta_head 0.5, 8 blocks.  A as head: fixed 0.5, per 1
    # vs per 1/3: best (1, 7) = max(1.5, 7/3) = 7/3.  B as head: fixed 1/6, per 1/3 vs per 1:
    # (6, 2) = max(1/6 + 2, 2) = 13/6 < 7/3 * 0.95
    devs = [dict(o=0.0, bw=1.0, lim_body=10, lim_head=10), dict(o=0.0, bw=3.0, lim_body=10, lim_head=10)]
    r = P.plan_ring(8, devs, 0, 1.0, 0.5)
    assert r["tier"] == 1 and r["head"] == 1
    assert abs(r["tau"] - 13.0 / 6.0) < 1e-12 and abs(r["tau_anchor"] - 7.0 / 3.0) < 1e-12
    assert r["divisions"] == [[2, 6]]


def test_pin_anchor_kept_within_margin():
    # B is 1% faster per block: its rotation wins by less than 5%, the anchor stays head
    devs = [dict(o=0.0, bw=1.0, lim_body=10, lim_head=10), dict(o=0.0, bw=1.01, lim_body=10, lim_head=10)]
    r = P.plan_ring(8, devs, 0, 1.0, 0.1)
    assert r["head"] == 0


def test_pin_tiers():
    devs = [dict(throughput=1.0, lim_body=10, lim_head=10), dict(throughput=3.0, lim_body=10, lim_head=10)]
    r = P.plan_ring(8, devs, 0, 1.0, 0.5)
    assert r["tier"] == 2 and r["head"] == 0 and r["divisions"] == [[2, 6]]
    devs = [dict(working_set=w, lim_body=10, lim_head=10) for w in (1.0, 1.0, 8.0)]
    r = P.plan_ring(10, devs, 0, 1.0, 0.5)
    assert r["tier"] == 3 and r["divisions"] == [[1, 1, 8]] and r["feasible"]
    devs[2]["lim_body"] = 7
    r = P.plan_ring(10, devs, 0, 1.0, 0.5)
    assert not r["feasible"] and r["undersized"] == 2


def test_pin_baselines():
    assert P.divide(10, 3) == [4, 3, 3]
    # shares 5/102, 500/102, 5/102: floors (0, 4, 0), the remainder to device 1, then devices 0
    # and 2 each take one block from the largest holder
    assert P.divide(5, 3, [1.0, 100.0, 1.0]) == [1, 3, 1]
    assert P.divide(10, 3, [1.0, 1.0, 8.0]) == [1, 1, 8]


# ---- the library against the oracle -------------------------------------------------------

def _random_instance(rng, k, m):
    fixed = [rng.choice([0.0, rng.uniform(0, 3)]) for _ in range(m)]
    per = [rng.choice([1.0, 0.5, 0.25, rng.uniform(0.1, 2.0)]) for _ in range(m)]
    lim = [rng.randint(0, k) for _ in range(m)]
    return fixed, per, lim


def test_partition_matches_brute_force(lib):
    rng = random.Random(20260917)
    seen_infeasible = seen_feasible = 0
    for _ in range(600):
        k, m = rng.randint(1, 11), rng.randint(1, 4)
        fixed, per, lim = _random_instance(rng, k, m)
        want = P.partition(k, fixed, per, lim)
        if want is None:
            with pytest.raises(K.KflError) as e:
                K.kfl_partition(k, fixed, per, lim)
            assert e.value.code == K.KFL_ERR_INFEASIBLE
            seen_infeasible += 1
            continue
        n, tau = K.kfl_partition(k, fixed, per, lim)
        assert tau == want[0]
        assert tuple(n) in want[1]
        seen_feasible += 1
    assert seen_feasible > 100 and seen_infeasible > 50


def test_plan_ring_matches_brute_force(lib):
    rng = random.Random(7)
    tiers = {1: 0, 2: 0, 3: 0}
    for _ in range(400):
        k, m = rng.randint(1, 10), rng.randint(1, 4)
        tier = rng.choice([1, 2, 3])
        devs = []
        for _ in range(m):
            lb = rng.randint(1, k)
            d = {"lim_body": lb, "lim_head": rng.randint(0, lb)}
            if tier == 1:
                d.update(o=rng.choice([0.0, rng.uniform(0, 0.2)]), bw=rng.choice([1.0, 2.0, 3.0, rng.uniform(0.5, 4)]))
            elif tier == 2:
                d.update(throughput=rng.choice([1.0, 2.0, rng.uniform(0.5, 4)]), bw=rng.choice([0.0, 1.0]))
            else:
                d.update(working_set=rng.choice([1.0, 2.0, rng.uniform(0.5, 8)]))
            devs.append(d)
        if tier == 2 and all(d["bw"] > 0 for d in devs):
            devs[0]["bw"] = 0.0
        anchor = rng.randrange(m)
        bb, bh = rng.choice([1.0, 0.5]), rng.choice([0.0, 0.3, 1.0])
        want = P.plan_ring(k, devs, anchor, bb, bh, 0.05)
        n, plan, rc = K.kfl_plan_ring(k, devs, anchor, bb, bh, 0.05)
        assert plan["tier"] == want["tier"]
        tiers[want["tier"]] += 1
        if not want["feasible"]:
            assert rc == K.KFL_ERR_INFEASIBLE and plan["undersized"] == want["undersized"]
            continue
        assert rc == 0
        assert plan["head"] == want["head"]
        assert n in want["divisions"]
        if want["tier"] in (1, 2):
            assert plan["tau"] == want["tau"]
        if want["tier"] == 1:
            assert plan["tau_anchor"] == want["tau_anchor"]
    assert min(tiers.values()) > 50


def test_divide_matches_oracle(lib):
    rng = random.Random(11)
    for _ in range(300):
        m = rng.randint(1, 6)
        k = rng.randint(m, 40)
        w = None if rng.random() < 0.2 else [rng.choice([1.0, 2.0, rng.uniform(0.01, 10)]) for _ in range(m)]
        assert K.kfl_divide(k, m, w) == P.divide(k, m, w)


def test_partition_never_worse_than_the_baselines(lib):
    # on any feasible instance without limits, the exact bottleneck is at most that of Uniform and
    # of Memory-proportional divisions
    rng = random.Random(3)
    for _ in range(200):
        m = rng.randint(1, 5)
        k = rng.randint(m, 30)
        fixed = [rng.uniform(0, 1) for _ in range(m)]
        per = [rng.uniform(0.1, 2) for _ in range(m)]
        n, tau = K.kfl_partition(k, fixed, per, [k] * m)
        for base in (K.kfl_divide(k, m), K.kfl_divide(k, m, [rng.uniform(1, 4) for _ in range(m)])):
            assert tau <= max(fixed[i] + base[i] * per[i] for i in range(m))


def test_argument_errors(lib):
    with pytest.raises(K.KflError):
        K.kfl_partition(0, [0.0], [1.0], [1])
    with pytest.raises(K.KflError):
        K.kfl_partition(3, [0.0], [0.0], [3])      # per must be positive
    with pytest.raises(K.KflError):
        K.kfl_partition(3, [math.inf], [1.0], [3])
    with pytest.raises(K.KflError):
        K.kfl_divide(2, 3)
    assert K.kfl_strerror(K.KFL_ERR_INFEASIBLE) != "unknown error"


def test_block_limit_is_the_largest_stage_that_fits(lib):
    m = wl.QWEN_72B_INT4
    cfg = K.model_cfg(m, 8256, 4)
    per_block = K.kfl_stage_memory_bytes(cfg, 0, 2, 0) - K.kfl_stage_memory_bytes(cfg, 0, 1, 0)
    for room in (0, 10 * per_block, 37 * per_block + 12345, 10 ** 13):
        for head in (False, True):
            lim = K.kfl_block_limit(cfg, room, head)
            flags = K.KFL_IS_HEAD if head else 0

            def need(n):
                return 0 if (n == 0 and not head) else K.kfl_stage_memory_bytes(cfg, 0, n, flags)
            if lim > 0 or head is False:
                assert need(lim) <= room or lim == 0
            if lim < m.n_layers_total:
                assert need(lim + 1) > room
    # the head holds the embedding and lm_head: it fits fewer blocks in the same room
    room = 40 * per_block
    assert K.kfl_block_limit(cfg, room, True) < K.kfl_block_limit(cfg, room, False)
