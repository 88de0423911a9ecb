"""Workload-level pins of the oracle's KV manager, and planted-mistake checks that
show each pin catches the kind of error it is meant to catch."""
import numpy as np
import pytest

import oracle
from oracle import OracleManager
from oracle import policy as opol
from oracle import pool as opool
from oracle import sessions as se
from workloads import make_workload, value_table
from workloads.content import subpage_offsets, subpage_values_np, valid_rows

from . import test_oracle_policy as tpol
from . import test_oracle_pool as tpool


def _expected_block_bytes(seed, table, shape, sid, blk, ctx):
    J = 2 * shape.layers
    off = subpage_offsets(seed, np.full(J, sid), np.full(J, blk), np.arange(J) // 2,
                          np.arange(J) % 2, shape)
    rows = np.full(J, int(valid_rows(ctx, blk, shape)))
    return subpage_values_np(table, off, rows, shape).view(np.uint8).reshape(J, -1)


def _check_content_follows_ownership(m, seed, table):
    pool = m.pool
    for s in range(pool.S):
        for b in range(int(pool.nblocks[s])):
            want = _expected_block_bytes(seed, table, m.shape, s, b, int(pool.ctx[s]))
            e = int(pool.tables[s, b])
            got = pool.hbm[:, e, :] if e >= 0 else pool.host[-(e + 2)]
            assert np.array_equal(got, want), (s, b, e)


def test_tiny_workload_invariants_and_bytes():
    seed = 0
    wl = make_workload("tiny", seed)
    table = value_table(seed)
    m = OracleManager(wl, with_bytes=True, content=(seed, table), rank_on="none")
    for i in range(wl.n_events):
        rec = m.step(i)
        pool = m.pool
        assert pool.resident_count() <= pool.budget
        if rec["kind"] in (1, 2):
            # the turn's session is fully resident afterwards and k = deficit exactly
            assert pool.host_blocks(rec["sid"]).size == 0
            if "victims" in rec:
                assert rec["victims"].shape[0] == rec["k"]
                assert rec["sid"] not in rec["victims"][:, 0]
        if i % 100 == 99:
            pool.check_invariants()
            _check_content_follows_ownership(m, seed, table)
    c = m.counters
    # the workload exercises every path: evictions, reloads, preloads, growth
    assert c["pages_out"] > 500 and c["pages_in"] > 500 and c["preloads"] > 10
    assert c["appended"] > 100 and c["turns"] > 50


def test_thinker_turns_reload_one_session_each():
    wl = make_workload("thinker", 0, n_turns=30)
    m = OracleManager(wl, with_bytes=False, rank_on="none")
    for i in range(wl.n_events):
        rec = m.step(i)
        if rec["kind"] == 2:
            sid = rec["sid"]
            assert m.pool.host_blocks(sid).size == 0
            assert rec["in_pages"].size > 0                 # every turn reloads
            assert rec["k"] == rec["victims"].shape[0]
            # exactly the deficit: the pool is full again after the turn
            assert m.pool.free_budget() == 0
    m.pool.check_invariants()


def test_workload_scripts_are_deterministic_and_ordered():
    a = make_workload("tiny", 3)
    b = make_workload("tiny", 3)
    c = make_workload("tiny", 4)
    assert np.array_equal(a.t_us, b.t_us) and np.array_equal(a.kind, b.kind)
    assert not (np.array_equal(a.t_us, c.t_us) and np.array_equal(a.sid, c.sid))
    assert np.all(np.diff(a.t_us) >= 0)
    t = make_workload("thinker", 1, n_turns=5)
    assert t.perms.shape == (5, 64)
    assert int(t.meta["total_pages"]) >= t.spec.hbm_budget_pages + t.spec.max_blocks


def test_load_keys_reproduce_the_scatter_order_of_any_subset():
    """The device driver passes a scattered reload order as per-block keys: for every
    subset of blocks, ascending (key, block id) must be the scatter order the oracle
    uses for that subset."""
    from paper_2606_22983_gb300 import build
    build()                      # the manager module loads liblv (no GPU call)
    from paper_2606_22983_gb300.manager import load_keys
    from workloads import scatter_order
    rng = np.random.default_rng(4)
    for trial in range(40):
        nb = int(rng.integers(1, 300))
        key = int(rng.integers(0, 1 << 40))
        keys = load_keys(scatter_order, key, nb)
        assert sorted(keys.tolist()) == list(range(nb))
        sub = np.sort(rng.choice(nb, size=int(rng.integers(0, nb + 1)), replace=False))
        want = scatter_order(key, sub)
        got = sub[np.lexsort((sub, keys[sub]))]
        assert np.array_equal(got, want), (trial, nb)


def test_content_numpy_and_torch_agree():
    import torch
    from workloads import TINY_SHAPE, THINKER_SHAPE, subpage_values_torch
    table = value_table(5)
    for shape in (TINY_SHAPE, THINKER_SHAPE):
        n = 7
        off = subpage_offsets(5, np.arange(n), np.arange(n) * 3, np.arange(n) % 4, np.arange(n) % 2, shape)
        rows = np.array([0, 1, 5, 16, 16, 3, 15])
        a = subpage_values_np(table, off, rows, shape)
        b = subpage_values_torch(torch.from_numpy(table.view(np.int16)), torch.from_numpy(off),
                                 torch.from_numpy(rows), shape).numpy().view(np.uint16)
        assert np.array_equal(a, b)
        assert (a[0] == 0).all() and (a[3] != 0).any()
    v = torch.from_numpy(table.view(np.int16)).view(torch.bfloat16).float()
    assert abs(float(v.mean())) < 0.01 and abs(float(v.std()) - 1.0) < 0.01


# ----------------------------------------------------------------- planted mistakes
def _fails(fn, *a, **kw):
    try:
        fn(*a, **kw)
    except (AssertionError, opool.OracleError):
        return True
    return False


def test_pins_catch_dropped_reply_term(monkeypatch):
    real = opol.t_next

    def bad(st, mode, prior, unit):
        return max(0, st.gen_us - st.play_us) if mode == 0 else real(st, mode, prior, unit)
    monkeypatch.setattr(opol, "t_next", bad)
    monkeypatch.setattr(tpol, "t_next", bad)
    assert _fails(tpol.test_next_use_golden)


def test_pins_catch_wrong_ema_weight(monkeypatch):
    real = se.apply_event

    def bad(st, kind, t, a=0, b=0, protect_us=0):
        if kind == se.SE_SPEECH_STOP and st.flags & se.DONE_VALID and st.reply_n > 0:
            st.reply_ema_us = (st.reply_ema_us + (t - st.t_done_us)) // 2
            st.reply_n += 1
            st.flags &= ~(se.IMMEDIATE | se.DONE_VALID)
            return
        real(st, kind, t, a, b, protect_us)
    monkeypatch.setattr(se, "apply_event", bad)
    assert _fails(tpol.test_reply_interval_golden)


def test_pins_catch_wrong_sort_direction(monkeypatch):
    real = opol.order_global

    def bad(*a, **kw):
        s, b, p = real(*a, **kw)
        return s[::-1].copy(), b[::-1].copy(), p[::-1].copy()
    monkeypatch.setattr(opol, "order_global", bad)
    monkeypatch.setattr(tpol, "order_global", bad)
    assert _fails(tpol.test_order_pairwise_and_formulations_agree, opol.SUFFIX_FIRST, False)
    assert _fails(tpol.test_paper_scenario_next_use_beats_lru)


def test_pins_catch_prefix_first(monkeypatch):
    """Evicting prefix blocks first (the opposite of Section 5.1's suffix-first rule)."""
    real = opol.order_global

    def bad(tables, nblocks, sessions, now, mode, prior, unit, within=0, fallback=False):
        return real(tables, nblocks, sessions, now, mode, prior, unit, 1 - within, fallback)
    monkeypatch.setattr(opol, "order_global", bad)
    monkeypatch.setattr(tpol, "order_global", bad)
    assert _fails(tpol.test_paper_scenario_next_use_beats_lru)
    assert _fails(tpol.test_special_cases)


def test_pins_catch_protection_ignored(monkeypatch):
    monkeypatch.setattr(opol, "is_eligible", lambda st, now: not (st.flags & se.RUNNING))
    assert _fails(tpol.test_order_pairwise_and_formulations_agree, opol.SUFFIX_FIRST, False)
    assert _fails(tpol.test_protection_window_expires)


def test_pins_catch_wrong_subpage_copied(monkeypatch):
    real = opool.OraclePool.swap_out

    def bad(self, sid, blk, page):
        slots = real(self, sid, blk, page)
        if self.with_bytes and self.J > 1:
            for p, h in zip(np.asarray(page), slots):
                self.host[h, 0, :] = self.hbm[1, p, :]          # layer 0 K <- layer 0 V
        return slots
    monkeypatch.setattr(opool.OraclePool, "swap_out", bad)
    assert _fails(tpool.test_round_trip_identity_and_invariants)


def test_pins_catch_highest_free_allocation(monkeypatch):
    def bad(self, used, n, cap, code):
        free = np.nonzero(~used)[0][::-1]
        if int(used.sum()) + n > cap or free.size < n:
            raise opool.OracleError(code)
        got = free[:n].astype(np.int64)
        used[got] = True
        return got
    monkeypatch.setattr(opool.OraclePool, "_alloc_lowest", bad)
    assert _fails(tpool.test_alloc_lowest_free_brute_force)


def test_pins_catch_remap_without_free(monkeypatch):
    real = opool.OraclePool.remap

    def bad(self, sid, blk, new_loc):
        keep = self.hbm_used.copy()
        real(self, sid, blk, new_loc)
        self.hbm_used |= keep & (self.owner_hbm[:, 0] == -1) & ~self.hbm_used
    monkeypatch.setattr(opool.OraclePool, "remap", bad)
    assert _fails(tpool.test_exclusive_tiers_free_host_slot_on_commit)


def test_next_use_versus_lru_on_the_voice_workloads():
    """NEXT f3 (Sections 2.3 and 5): the same scripts under the paper's next-use
    order with speech-triggered preload, and under the LRU baseline that loads at
    turn start.  Next-use must move fewer reloads onto the turns' critical path."""
    rows = {}
    for name in ("tiny", "mixed"):
        for policy in (0, 1):
            from workloads import pool_spec
            wl = make_workload(name, 0)
            wl.spec = wl.spec.with_(policy=policy)
            m = OracleManager(wl, with_bytes=False, rank_on="none")
            m.run()
            m.pool.check_invariants()
            rows[(name, policy)] = dict(m.counters)
    for name in ("tiny", "mixed"):
        nu, lru = rows[(name, 0)], rows[(name, 1)]
        assert nu["sync_loads"] < lru["sync_loads"], (name, nu, lru)


def test_turns_preload_fallback_and_eviction_hand_worked():
    """Every decision of a small script worked by hand (tests/golden/manager_turns_hand.json):
    a preload, turns with growth, the foreground fallback tier and an eviction request
    with fewer candidates than asked for."""
    from oracle.manager import OracleManager
    from ._hand import hand_workload, load
    g = load("manager_turns_hand.json")
    m = OracleManager(hand_workload(g), with_bytes=True, content="tagged", rank_on="none")
    for i, want in enumerate(g["expect"]):
        rec = m.step(i)
        got = {k: np.asarray(rec[k]).tolist() for k in want if k in rec}
        assert got == want, (i, got)
        assert not any(k in rec for k in ("k", "victims", "in_blocks", "append_pages") if k not in want), i
        m.pool.check_invariants()
    assert m.pool.tables.tolist() == g["expect_tables"]
    assert [s.ctx_tokens for s in m.sessions] == g["expect_ctx_tokens"]
    assert [s.protect_until_us for s in m.sessions] == g["expect_protect_until_us"]
    assert {k: m.counters[k] for k in g["expect_counters"]} == g["expect_counters"]
