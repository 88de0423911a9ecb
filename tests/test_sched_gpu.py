"""lv_schedule (Section 4, Algorithm 1) against the oracle's scheduler: the golden
round, random ready sets up to the 4096-request limit, and degenerate sizes."""
import json
import os

import numpy as np
import pytest

pytestmark = pytest.mark.gpu

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "schedule_round.json")


def _run(pool, reqs, ps, a, b, occ, alloc, tb, kb):
    from paper_2606_22983_gb300 import lv
    arr = np.zeros(len(reqs), dtype=lv.REQUEST_DTYPE)
    for i, r in enumerate(reqs):
        for k in lv.REQUEST_DTYPE.names:
            arr[i][k] = r[k]
    q = lv.lv_sched_params(p_safe_us=ps, alpha=a, beta=b, occupied=occ, allocatable=alloc,
                           token_budget=tb, kv_budget=kb)
    order = np.full(max(1, len(reqs)), -1, np.int32)
    batch = np.full(1, -1, np.int32)
    lv.lv_schedule(pool.handle, q, arr, len(reqs), order, batch, pool.stream)
    pool.sync()
    return order[:len(reqs)].tolist(), order[:int(batch[0])].tolist()


@pytest.fixture(scope="module")
def pool():
    from paper_2606_22983_gb300.pool import KVPool
    p = KVPool(layers=1, kv_heads=1, head_dim=8, max_sessions=4, max_blocks=4, hbm_pages=16,
               hbm_budget_pages=16, host_pages=16)
    yield p
    p.close()


def test_schedule_golden_round(pool):
    g = json.load(open(GOLDEN))
    order, batch = _run(pool, g["requests"], g["p_safe_us"], g["alpha"], g["beta"], g["occupied"],
                        g["allocatable"], g["token_budget"], g["kv_budget"])
    assert order == g["expect_order"] and batch == g["expect_batch"]


@pytest.mark.parametrize("n", [0, 1, 7, 64, 1000, 4096])
def test_schedule_matches_oracle(pool, n):
    from oracle.scheduler import schedule
    rng = np.random.default_rng(n)
    for trial in range(6 if n < 4096 else 2):
        reqs = []
        for i in range(n):
            started = int(rng.random() < 0.7)
            reqs.append(dict(id=int(rng.integers(0, 1 << 30)), started=started,
                             play_buffer_us=int(rng.integers(0, 8)) * 700_000 if started else 0,
                             ready_age_us=int(rng.integers(0, 6)) * 400_000,
                             kv_pages=int(rng.integers(0, 5)) * 250, tokens=int(rng.integers(0, 400)),
                             kv_needed=int(rng.integers(0, 50))))
        args = (2_000_000, int(rng.integers(0, 9)), int(rng.integers(0, 4)), int(rng.integers(0, 40_000)),
                40_000, int(rng.integers(0, 30 * max(n, 1))), int(rng.integers(0, 5 * max(n, 1))))
        want = schedule(reqs, *args)
        got = _run(pool, reqs, *args)
        assert got == want, (n, trial)
    assert pool.sync(raise_on_error=False) == 0
