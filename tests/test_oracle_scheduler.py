"""Pins for the oracle's urgency scheduler (Section 4, Algorithm 1, Eqs. 1-3)."""
import json
import os
from fractions import Fraction

import numpy as np

from oracle.scheduler import classify, schedule, utility

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "schedule_round.json")


def test_schedule_golden_round():
    g = json.load(open(GOLDEN))
    for r in g["requests"]:
        assert classify(r["started"], r["play_buffer_us"], g["p_safe_us"]) == g["expect_classes"][str(r["id"])]
    for rid, want in g["expect_utility"].items():
        r = g["requests"][int(rid)]
        u = utility(r["kv_pages"], r["play_buffer_us"], g["p_safe_us"], g["alpha"], g["beta"],
                    g["occupied"], g["allocatable"])
        assert u == Fraction(want)
    order, batch = schedule(g["requests"], g["p_safe_us"], g["alpha"], g["beta"], g["occupied"],
                            g["allocatable"], g["token_budget"], g["kv_budget"])
    assert order == g["expect_order"] and batch == g["expect_batch"]


def _random_round(rng, n):
    reqs = []
    for i in range(n):
        started = int(rng.random() < 0.7)
        reqs.append(dict(id=i, started=started,
                         play_buffer_us=int(rng.integers(0, 6)) * 1_000_000 if started else 0,
                         ready_age_us=int(rng.integers(0, 5)) * 500_000,
                         kv_pages=int(rng.integers(0, 4)) * 100, tokens=int(rng.integers(1, 300)),
                         kv_needed=int(rng.integers(0, 40))))
    return reqs


def test_schedule_properties_on_random_rounds():
    rng = np.random.default_rng(4)
    for trial in range(200):
        reqs = _random_round(rng, int(rng.integers(1, 40)))
        ps, a, b = 2_000_000, int(rng.integers(1, 8)), int(rng.integers(1, 4))
        occ, alloc = int(rng.integers(0, 1000)), 1000
        tb, kb = int(rng.integers(0, 3000)), int(rng.integers(0, 300))
        order, batch = schedule(reqs, ps, a, b, occ, alloc, tb, kb)
        by_id = {r["id"]: r for r in reqs}
        assert sorted(order) == list(range(len(reqs)))
        cls = [classify(by_id[i]["started"], by_id[i]["play_buffer_us"], ps) for i in order]
        assert cls == sorted(cls)                                   # U0, then U1, then U2
        for x, y in zip(order, order[1:]):
            rx, ry = by_id[x], by_id[y]
            cx = classify(rx["started"], rx["play_buffer_us"], ps)
            if cx != classify(ry["started"], ry["play_buffer_us"], ps):
                continue
            if cx == 0:
                kx, ky = rx["play_buffer_us"], ry["play_buffer_us"]
            elif cx == 1:
                kx, ky = -rx["ready_age_us"], -ry["ready_age_us"]
            else:
                kx = -utility(rx["kv_pages"], rx["play_buffer_us"], ps, a, b, occ, alloc)
                ky = -utility(ry["kv_pages"], ry["play_buffer_us"], ps, a, b, occ, alloc)
            assert (kx, x) < (ky, y)
        # the batch is the longest prefix that fits both budgets
        assert batch == order[:len(batch)]
        tok = sum(by_id[i]["tokens"] for i in batch)
        kv = sum(by_id[i]["kv_needed"] for i in batch)
        assert tok <= tb and kv <= kb
        if len(batch) < len(order):
            nxt = by_id[order[len(batch)]]
            assert tok + nxt["tokens"] > tb or kv + nxt["kv_needed"] > kb


def test_utility_directions():
    """More resident KV under pressure raises U2 priority; a deeper buffer lowers it."""
    u = lambda k, p: utility(k, p, 2_000_000, 2, 1, 800, 1000)
    assert u(200, 3_000_000) > u(100, 3_000_000)
    assert u(100, 5_000_000) < u(100, 3_000_000)
    assert u(100, 2_000_000) == u(100, 1_000_000)        # no penalty within the safe buffer
