"""Pins for the oracle's allocation, copy and remap (Sections 5.1, 5.2, 6).

Allocation is checked against brute force, copies against plain slicing of a
pool with one layer and against the round-trip identity, remap against the
owner/table bijection, the budget, and its error cases.
"""
import numpy as np
import pytest

from oracle.pool import OraclePool, OracleError


def _pool(L=2, H=1, D=8, T=4, S=4, maxb=6, pages=16, budget=16, slots=32, with_bytes=True):
    return OraclePool(L, H, D, T, 2, S, maxb, pages, budget, slots, with_bytes=with_bytes)


def _fill_random(pool, rng, ctx):
    """Place sessions' blocks on consecutive pages and give every page random bytes."""
    place = np.full((pool.S, pool.max_blocks), -1, dtype=np.int64)
    p = 0
    for s, c in enumerate(ctx):
        for b in range(-(-c // pool.T)):
            place[s, b] = p
            p += 1
    pool.import_placement(place, np.asarray(ctx))
    if pool.with_bytes:
        pool.hbm[:] = rng.integers(0, 256, pool.hbm.shape, dtype=np.uint8)
        pool.host[:] = rng.integers(0, 256, pool.host.shape, dtype=np.uint8)


def _logical_bytes(pool):
    """bytes of every (sid, blk), read through the block tables."""
    out = {}
    for s in range(pool.S):
        for b in range(int(pool.nblocks[s])):
            e = int(pool.tables[s, b])
            out[(s, b)] = (pool.hbm[:, e, :].copy() if e >= 0 else pool.host[-(e + 2)].copy())
    return out


def test_alloc_lowest_free_brute_force():
    rng = np.random.default_rng(0)
    for _ in range(50):
        n = int(rng.integers(1, 200))
        pool = _pool(pages=n, budget=n, slots=n, with_bytes=False)
        used = rng.random(n) < 0.5
        pool.hbm_used[:] = used
        free = [i for i in range(n) if not used[i]]       # brute force
        k = int(rng.integers(0, len(free) + 1))
        got = pool.alloc_hbm(k)
        assert got.tolist() == free[:k]
        assert pool.hbm_used[got].all() and int(pool.hbm_used.sum()) == int(used.sum()) + k
        with pytest.raises(OracleError) as ei:
            pool.alloc_hbm(len(free) - k + 1)
        assert ei.value.code == "NO_HBM"


def test_alloc_respects_budget_not_just_capacity():
    pool = _pool(pages=16, budget=5, with_bytes=False)
    assert pool.alloc_hbm(5).tolist() == [0, 1, 2, 3, 4]
    with pytest.raises(OracleError):
        pool.alloc_hbm(1)


def test_swap_out_single_layer_is_plain_memcpy():
    rng = np.random.default_rng(1)
    pool = _pool(L=1, S=1, maxb=2, pages=4, budget=4, slots=3)
    _fill_random(pool, rng, [8])                   # two blocks on pages 0, 1
    pool.host_used[0] = True                       # slot 0 taken: lowest free is 1
    src_k, src_v = pool.hbm[0, 1].copy(), pool.hbm[1, 1].copy()
    slots = pool.swap_out([0], [1], [1])
    assert slots.tolist() == [1]
    assert np.array_equal(pool.host[1, 0], src_k) and np.array_equal(pool.host[1, 1], src_v)
    assert pool.bytes_out == 2 * pool.P
    # the tables are untouched until the commit
    assert pool.tables[0, 1] == 1


def test_round_trip_identity_and_invariants():
    rng = np.random.default_rng(2)
    for trial in range(20):
        pool = _pool(S=4, maxb=6, pages=24, budget=20, slots=40)
        ctx = rng.integers(1, 6 * pool.T + 1, 4)
        while sum(-(-int(c) // pool.T) for c in ctx) > 20:
            ctx = rng.integers(1, 6 * pool.T + 1, 4)
        _fill_random(pool, rng, ctx)
        before = _logical_bytes(pool)
        for rnd in range(6):
            res = [(s, b) for s in range(4) for b in range(int(pool.nblocks[s])) if pool.tables[s, b] >= 0]
            if res:
                pick = rng.permutation(len(res))[:int(rng.integers(1, len(res) + 1))]
                vs = [res[i][0] for i in pick]
                vb = [res[i][1] for i in pick]
                vp = [int(pool.tables[s, b]) for s, b in zip(vs, vb)]
                n0 = pool.bytes_out
                slots = pool.swap_out(vs, vb, vp)
                assert pool.bytes_out - n0 == len(vs) * 2 * pool.L * pool.P
                pool.remap(vs, vb, -(slots + 2))
                pool.check_invariants()
            s = int(rng.integers(0, 4))
            hb = pool.host_blocks(s)
            if hb.size and pool.free_budget() >= hb.size:
                order = rng.permutation(hb)             # any list order
                pages = pool.swap_in(s, order)
                pool.remap(np.full(hb.size, s), order, pages)
                pool.check_invariants()
            assert pool.resident_count() <= pool.budget
        after = _logical_bytes(pool)
        assert before.keys() == after.keys()
        for key in before:
            assert np.array_equal(before[key], after[key]), key


def test_exclusive_tiers_free_host_slot_on_commit():
    rng = np.random.default_rng(4)
    pool = _pool(S=1, maxb=2, pages=4, budget=4, slots=4)
    _fill_random(pool, rng, [8])
    slots = pool.swap_out([0], [1], [1])
    pool.remap([0], [1], -(slots + 2))
    assert not pool.hbm_used[1] and pool.host_used[slots[0]]
    pages = pool.swap_in(0, [1])
    pool.remap([0], [1], pages)
    assert pages.tolist() == [1]                  # the lowest free page again
    assert not pool.host_used[slots[0]] and pool.owner_host[slots[0], 0] == -1
    pool.check_invariants()


def test_remap_errors():
    rng = np.random.default_rng(5)
    pool = _pool(S=2, maxb=4, pages=8, budget=8, slots=8)
    _fill_random(pool, rng, [8, 8])               # pages 0,1 and 2,3
    with pytest.raises(OracleError) as e:
        pool.remap([0], [0], [2])                 # page 2 is owned by (1, 0)
    assert e.value.code == "DOUBLE_MAP"
    with pytest.raises(OracleError) as e:
        pool.remap([0], [0], [5])                 # page 5 was never reserved
    assert e.value.code == "DOUBLE_MAP"
    pages = pool.alloc_hbm(2)
    with pytest.raises(OracleError) as e:
        pool.remap([0, 0], [0, 0], pages)         # the same block twice in one batch
    assert e.value.code == "DOUBLE_MAP"
    with pytest.raises(OracleError) as e:
        pool.remap([0], [3], [int(pages[1])])     # block 3 is beyond the context
    assert e.value.code == "BOUNDS"


def test_cancel_releases_reservation_and_keeps_old_mapping():
    rng = np.random.default_rng(6)
    pool = _pool(S=1, maxb=2, pages=4, budget=4, slots=4)
    _fill_random(pool, rng, [8])
    before = _logical_bytes(pool)
    slots = pool.swap_out([0], [1], [1])
    pool.cancel(-(slots + 2))                     # the transfer is abandoned
    assert not pool.host_used.any()
    assert pool.tables[0, 1] == 1
    after = _logical_bytes(pool)
    assert all(np.array_equal(before[k], after[k]) for k in before)
    with pytest.raises(OracleError):
        pool.cancel([0])                          # an owned page is not a reservation


def test_append_takes_lowest_free_pages():
    pool = _pool(S=2, maxb=6, pages=10, budget=10, slots=4, with_bytes=False)
    place = np.full((2, 6), -1)
    place[0, 0], place[1, 0], place[1, 1] = 1, 0, 3
    pool.import_placement(place, np.array([3, 8]))
    got = pool.append(0, 6)                       # 3 -> 9 tokens: blocks 1, 2 needed
    assert got.tolist() == [2, 4]
    assert pool.tables[0, :3].tolist() == [1, 2, 4] and pool.ctx[0] == 9
    assert pool.append(0, 3).tolist() == []       # 12 tokens still fit in 3 blocks
    pool.check_invariants()


def test_swap_rejects_stale_victim():
    rng = np.random.default_rng(8)
    pool = _pool(S=1, maxb=2, pages=4, budget=4, slots=4)
    _fill_random(pool, rng, [8])
    with pytest.raises(OracleError) as e:
        pool.swap_out([0], [1], [0])              # block 1 lives on page 1, not 0
    assert e.value.code == "STATE"
    with pytest.raises(OracleError) as e:
        pool.swap_in(0, [0])                      # block 0 is not in the host tier
    assert e.value.code == "STATE"
