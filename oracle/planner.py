"""Brute-force oracle of the ring planner (test infrastructure only).

What the planner computes comes from the paper:

* A device i holding n blocks costs fixed(i) + n per(i): Eq. 2 (section V-A) with
  fixed(i) = o_i, plus beta_head / b_i for the head, and per(i) = beta_block / b_i.  Device i
  holds at most lim(i) blocks at the session's declared context and concurrency (section V-B,
  "Block placement").
* Block placement for a fixed ring order: a contiguous chain of k blocks over the devices in
  that order, every device holding at least one block, minimizing the largest stage cost
  (section V-B; Algorithm 1 solves it exactly).  The oracle is that definition written out: it
  tries every division and keeps the smallest bottleneck, with no candidate set, binary search
  or greedy pass.
* Head placement: one exact solve per rotation (device r as head, the ring taken from r); the
  anchor stays head unless the best rotation's bottleneck is below tau_anchor (1 - mu), with
  mu = 0.05 (section V-B, the head paragraph).
* Admission (section V-C): the full cost model when every device is priced; else per(i) from
  raw throughput with no head term and the head at the anchor; else blocks in proportion to the
  reported working set; then the division is checked against every device's limit and the
  undersized device is named.

Readings of what the paper leaves open (listed in the repository's design notes): among rotations
of equal bottleneck the first from the anchor around the ring wins; the tier-2 cost has no fixed
term; the proportional division is the largest-remainder apportionment (lower index first on
equal remainders) after which a device with no block takes one from the device holding most
(lower index first); the uniform division gives the k mod m left over to the first devices.

Only tests/ may import this module.
"""
from __future__ import annotations

import itertools
import math

__all__ = ["stage_cost", "partition", "plan_ring", "divide"]


def stage_cost(fixed: float, per: float, n: int) -> float:
    """Eq. 2 for n blocks: fixed + n per."""
    return fixed + n * per


def _divisions(k: int, caps: list):
    """Every (n_1 .. n_m) with 1 <= n_i <= caps[i] and sum k."""
    m = len(caps)
    for cut in itertools.combinations(range(1, k), m - 1):
        bounds = (0,) + cut + (k,)
        n = tuple(bounds[i + 1] - bounds[i] for i in range(m))
        if all(n[i] <= caps[i] for i in range(m)):
            yield n


def partition(k: int, fixed: list, per: list, lim: list):
    """(smallest bottleneck, every division reaching it), or None when no division exists."""
    best, arg = math.inf, []
    for n in _divisions(k, list(lim)):
        b = max(stage_cost(fixed[i], per[i], n[i]) for i in range(len(n)))
        if b < best:
            best, arg = b, [n]
        elif b == best:
            arg.append(n)
    return None if not arg else (best, arg)


def divide(k: int, m: int, weight=None) -> list:
    """The evaluation's baselines: Uniform (weight None) or Memory-proportional (k >= m: every
    member of a ring holds a block)."""
    assert k >= m >= 1
    if weight is None:
        return [k // m + (1 if i < k % m else 0) for i in range(m)]
    total = sum(weight)
    share = [k * w / total for w in weight]
    n = [math.floor(s) for s in share]
    order = sorted(range(m), key=lambda i: (-(share[i] - n[i]), i))
    for j in range(k - sum(n)):
        n[order[j]] += 1
    for i in range(m):
        if n[i] == 0:
            big = max(range(m), key=lambda j: (n[j], -j))
            n[big] -= 1
            n[i] += 1
    return n


def plan_ring(k: int, devices: list, anchor: int, beta_block: float, beta_head: float, mu: float = 0.05) -> dict:
    """The planner's outcome: tier, head, bottleneck, block counts in ring order (every optimal
    division for tiers 1 and 2), feasibility and the undersized device."""
    m = len(devices)

    def rotated(r, priced):
        order = [(r + j) % m for j in range(m)]
        fixed, per, lim = [], [], []
        for j, d in enumerate(order):
            dev = devices[d]
            head = j == 0
            if priced:
                fixed.append(dev["o"] + (beta_head / dev["bw"] if head else 0.0))
                per.append(beta_block / dev["bw"])
            else:
                fixed.append(0.0)
                per.append(1.0 / dev["throughput"])
            lim.append(dev["lim_head"] if head else dev["lim_body"])
        return order, partition(k, fixed, per, lim)

    def unrotated(order, n):
        out = [0] * m
        for j, d in enumerate(order):
            out[d] = n[j]
        return out

    if all(d.get("bw", 0) > 0 for d in devices):
        sols = {r: rotated(r, True) for r in range(m)}
        taus = {r: (sols[r][1][0] if sols[r][1] else math.inf) for r in range(m)}
        ring = [(anchor + j) % m for j in range(m)]
        best = min(ring, key=lambda r: (taus[r], ring.index(r)))
        if taus[best] == math.inf:
            return {"tier": 1, "feasible": False, "undersized": -1, "tau_anchor": taus[anchor]}
        head = best if taus[best] < taus[anchor] * (1 - mu) else anchor
        order, (tau, divs) = sols[head]
        return {"tier": 1, "feasible": True, "head": head, "tau": tau, "tau_anchor": taus[anchor],
                "divisions": [unrotated(order, n) for n in divs], "undersized": -1}
    if all(d.get("throughput", 0) > 0 for d in devices):
        order, sol = rotated(anchor, False)
        if sol is None:
            return {"tier": 2, "feasible": False, "undersized": -1}
        return {"tier": 2, "feasible": True, "head": anchor, "tau": sol[0],
                "divisions": [unrotated(order, n) for n in sol[1]], "undersized": -1}
    order = [(anchor + j) % m for j in range(m)]
    if m > k:
        return {"tier": 3, "feasible": False, "undersized": -1}
    n = unrotated(order, divide(k, m, [devices[d]["working_set"] for d in order]))
    for d in order:
        if n[d] > (devices[d]["lim_head"] if d == anchor else devices[d]["lim_body"]):
            return {"tier": 3, "feasible": False, "head": anchor, "divisions": [n], "undersized": d}
    return {"tier": 3, "feasible": True, "head": anchor, "divisions": [n], "undersized": -1}
