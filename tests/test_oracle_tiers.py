"""Pins for the oracle's inclusive tiers (clean host copies kept after a reload).

The paper does not say whether the host copy survives a reload, so the
inclusive mode is a reading; these tests tie it to facts that do not depend on
that reading: the tier mode never changes a decision (victims, pages, order),
every block's bytes -- wherever they sit -- equal what the seeded generator
wrote for its tokens, and with no appends the copied pages are exactly the
blocks that were first evicted from their initial HBM placement."""
import numpy as np
import pytest

from oracle import OracleManager
from oracle.pool import OraclePool, OracleError, _enc_host
from workloads import make_workload, pool_spec, value_table

DECISIONS = ("victims", "in_blocks", "in_pages", "append_pages", "order", "preload", "k")


def _manager(name, tiers, seed=0, with_bytes=True, rank_on="all", **over):
    wl = make_workload(name, seed, spec=pool_spec(name).with_(tiers=tiers), **over)
    content = (seed, value_table(seed)) if with_bytes else None
    return OracleManager(wl, with_bytes=with_bytes, content=content, rank_on=rank_on)


def _check_bytes(om):
    """Every block's bytes at its location, and at its clean copy, are the generator's."""
    pool = om.pool
    for s in range(pool.S):
        ctx = int(pool.ctx[s])
        for b in range(int(pool.nblocks[s])):
            want = om._subpage_content(s, b, ctx)
            e = int(pool.tables[s, b])
            got = pool.hbm[:, e, :] if e >= 0 else pool.host[-(e + 2)]
            assert np.array_equal(got, want), ("location", s, b, e)
            g = int(pool.shadow[s, b])
            if g >= 0:
                assert np.array_equal(pool.host[g], want), ("clean copy", s, b, g)


@pytest.mark.parametrize("seed", [0, 1])
def test_tier_mode_changes_no_decision(seed):
    ex = _manager("tiny", 0, seed, with_bytes=False)
    inc = _manager("tiny", 1, seed, with_bytes=False)
    moved_out = 0
    for i in range(ex.wl.n_events):
        a, b = ex.step(i), inc.step(i)
        for key in DECISIONS:
            assert (key in a) == (key in b), (i, key)
            if key in a:
                assert np.array_equal(np.asarray(a[key]), np.asarray(b[key])), (i, key)
        # HBM placement is identical; host slots may differ
        assert np.array_equal(ex.pool.tables >= 0, inc.pool.tables >= 0), i
        assert np.array_equal(np.where(ex.pool.tables >= 0, ex.pool.tables, -1),
                              np.where(inc.pool.tables >= 0, inc.pool.tables, -1)), i
        moved_out += len(a.get("slots", ()))        # victims actually swapped out
    inc.pool.check_invariants()
    ex.pool.check_invariants()
    page = ex.pool.J * ex.pool.P
    assert ex.pool.bytes_in == inc.pool.bytes_in
    assert ex.pool.bytes_out == moved_out * page
    assert inc.pool.bytes_out + inc.pool.clean_out * page == ex.pool.bytes_out
    assert inc.pool.clean_out > 0 and inc.pool.bytes_out < ex.pool.bytes_out


def test_inclusive_bytes_are_the_generators():
    om = _manager("tiny", 1, 0, rank_on="none")
    for i in range(om.wl.n_events):
        om.step(i)
        if i % 100 == 99:
            _check_bytes(om)
            om.pool.check_invariants()
    assert om.pool.clean_dropped > 0          # appends into clean tails happened


def test_a_stale_tail_copy_is_caught():
    """Planted mistake: keep the clean copy of a tail block that gains rows."""
    om = _manager("tiny", 1, 0, rank_on="none")
    pool = om.pool
    real_append = OraclePool.append

    def append_keeping_copy(sid, n_tokens):
        b = int(pool.nblocks[sid]) - 1
        g = int(pool.shadow[sid, b]) if b >= 0 else -1
        out = real_append(pool, sid, n_tokens)
        if g >= 0 and pool.shadow[sid, b] < 0:    # undo the drop
            pool.shadow[sid, b] = g
            pool.host_used[g] = True
            pool.owner_host[g] = (sid, b)
        return out

    pool.append = append_keeping_copy
    with pytest.raises(AssertionError):
        for i in range(om.wl.n_events):
            om.step(i)
            if i % 25 == 24:
                _check_bytes(om)


def test_without_appends_only_first_evictions_copy():
    """Turn-driven sessions never append: a block is copied out only the first time
    it leaves its initial HBM page; every later eviction finds a clean copy."""
    om = _manager("thinker", 1, 0, with_bytes=False, rank_on="none", n_turns=40)
    init = om.pool.tables.copy()
    first = set()
    total = 0
    for i in range(om.wl.n_events):
        r = om.step(i)
        if "slots" not in r:                        # nothing was swapped out
            continue
        for s, b, _ in r["victims"]:
            total += 1
            if init[s, b] >= 0:
                first.add((int(s), int(b)))
    page = om.pool.J * om.pool.P
    assert total > 0
    assert om.pool.bytes_out == len(first) * page
    assert om.pool.clean_out == total - len(first)
    om.pool.check_invariants()


def _small_pool(inclusive=True):
    p = OraclePool(1, 1, 8, 16, 2, n_sessions=2, max_blocks=8, hbm_pages=8, hbm_budget_pages=8,
                   host_pages=8, with_bytes=True, inclusive=inclusive)
    placement = np.full((2, 8), -1, np.int64)
    placement[0, :3] = [_enc_host(0), _enc_host(1), _enc_host(2)]      # 40 tokens on the host
    p.import_placement(placement, np.array([40, 0]))
    for h in range(3):
        p.host[h] = h + 1
    return p


def test_hand_scenario_clean_copies_and_the_tail():
    p = _small_pool()
    pages = p.swap_in(0, [0, 1, 2])
    p.remap([0, 0, 0], [0, 1, 2], pages)
    assert list(p.shadow[0, :3]) == [0, 1, 2] and p.host_used[:3].all()
    p.append(0, 4)                                # 44 tokens: block 2 (8 rows) gains 4
    assert list(p.shadow[0, :3]) == [0, 1, -1] and not p.host_used[2] and p.clean_dropped == 1
    p.hbm[:, pages[2], :] = 9                      # the new rows
    before = p.bytes_out
    slots = p.swap_out([0, 0, 0], [2, 1, 0], [pages[2], pages[1], pages[0]])
    assert list(slots) == [2, 1, 0]               # dirty tail: lowest free slot; others: copies
    assert p.bytes_out - before == p.J * p.P and p.clean_out == 2
    assert (p.host[2] == 9).all() and (p.host[0] == 1).all() and (p.host[1] == 2).all()
    p.remap([0, 0, 0], [2, 1, 0], _enc_host(slots))
    assert list(p.tables[0, :3]) == [_enc_host(0), _enc_host(1), _enc_host(2)]
    assert (p.shadow < 0).all() and not p.hbm_used.any()
    p.check_invariants()


def test_exclusive_hand_scenario_frees_slots():
    p = _small_pool(inclusive=False)
    pages = p.swap_in(0, [0, 1, 2])
    p.remap([0, 0, 0], [0, 1, 2], pages)
    assert (p.shadow < 0).all() and not p.host_used.any()
    slots = p.swap_out([0], [2], [pages[2]])
    assert list(slots) == [0] and p.clean_out == 0


def test_cancel_leaves_clean_copies_and_frees_reservations():
    p = _small_pool()
    pages = p.swap_in(0, [0, 1, 2])
    p.remap([0, 0, 0], [0, 1, 2], pages)
    p.append(0, 4)                                 # block 2 loses its copy
    slots = p.swap_out([0, 0], [1, 2], [pages[1], pages[2]])
    assert list(slots) == [1, 2]
    p.cancel(_enc_host(slots))                     # slot 1 is block 1's copy, slot 2 a reservation
    assert p.shadow[0, 1] == 1 and p.host_used[1] and not p.host_used[2]
    assert list(p.tables[0, :3]) == list(pages)
    p.check_invariants()
    with pytest.raises(OracleError):
        p.cancel([_enc_host(5)])                   # neither


def test_commit_elsewhere_drops_the_copy():
    p = _small_pool()
    pages = p.swap_in(0, [0])
    p.remap([0], [0], pages)
    assert p.shadow[0, 0] == 0
    h = p.alloc_host(1)                            # a different slot than the copy
    p.remap([0], [0], _enc_host(h))
    assert p.shadow[0, 0] == -1 and not p.host_used[0] and p.tables[0, 0] == _enc_host(int(h[0]))
    p.check_invariants()


def test_tier_mode_changes_no_controller_decision():
    """Under the Section 5.2 preload controller (admissions, deferred commits,
    cancellations) the inclusive tiers still change where bytes sit only."""
    from oracle.preload import ControlledOracleManager, PreloadController
    runs = []
    for tiers in (0, 1):
        wl = make_workload("tiny", 0, spec=pool_spec("tiny").with_(tiers=tiers))
        om = ControlledOracleManager(wl, PreloadController(link_bytes_per_us=1, lead_prior_us=1_000_000,
                                                           cap_pages=40),
                                     with_bytes=False, rank_on="none")
        runs.append((om, om.run()))
    (ex, ra), (inc, rb) = runs
    for a, b in zip(ra, rb):
        for key in DECISIONS + ("admitted", "completed", "cancelled", "unprotected"):
            assert (key in a) == (key in b), key
            if key in a and key != "admitted":
                assert np.array_equal(np.asarray(a[key]), np.asarray(b[key])), key
    assert ex.counters == inc.counters
    assert inc.pool.clean_out > 0 and inc.pool.bytes_out < ex.pool.bytes_out
    inc.pool.check_invariants()
