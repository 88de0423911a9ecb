"""Pins for the oracle's next-use estimate, eligibility and victim order (Section 5.1).

Nothing here re-types the oracle's formulas: expected values are worked by hand
(tests/golden), victim sets are found by brute-force enumeration, and the order
is checked pairwise against a comparator written from the paper's wording.
"""
import itertools
import json
import os

import numpy as np
import pytest

from oracle import sessions as se
from oracle.policy import (t_next, order_global, order_scan, select_victims, SUFFIX_FIRST,
                           ASCENDING)

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _load(name):
    with open(os.path.join(GOLDEN, name)) as f:
        return json.load(f)


def test_next_use_golden():
    g = _load("next_use.json")
    for c in g["cases"]:
        st = se.SessionState(gen_us=c["gen_us"], play_us=c["play_us"], reply_n=c["reply_n"],
                             reply_ema_us=c["reply_ema_us"], reply_tokens=c["reply_tokens"],
                             flags=se.RESP_OPEN if c["resp_open"] else 0)
        got = t_next(st, c["mode"], g["reply_prior_us"], g["unit_us"])
        assert got == c["expect"], c["what"]


_EV = {"PLAYBACK": se.SE_PLAYBACK, "SPEECH_START": se.SE_SPEECH_START,
       "SPEECH_STOP": se.SE_SPEECH_STOP, "BARGE_IN": se.SE_BARGE_IN,
       "TURN_BEGIN": se.SE_TURN_BEGIN, "TURN_END": se.SE_TURN_END}


def test_reply_interval_golden():
    g = _load("reply_interval.json")
    ini = g["initial"]
    st = se.SessionState(gen_us=ini["gen_us"], play_us=ini["play_us"],
                         flags=se.RESP_OPEN if ini["resp_open"] else 0)
    checked = 0
    for e in g["events"]:
        se.apply_event(st, _EV[e["ev"]], e["t"], e.get("a", 0), e.get("b", 0))
        for key, want in e.get("expect", {}).items():
            if key == "t_next":
                got = t_next(st, se.MODE_PLAYBACK, g["reply_prior_us"], 80000)
            else:
                got = getattr(st, key)
            assert got == want, (e, key)
            checked += 1
    assert checked >= 12


def _mk_sessions(spec):
    out = []
    for d in spec:
        fl = 0
        for name in d.get("flags", "").split():
            fl |= getattr(se, name)
        out.append(se.SessionState(gen_us=d["gen_us"], play_us=d["play_us"], flags=fl))
    return out


def test_paper_scenario_next_use_beats_lru():
    g = _load("scenario_lru_vs_next_use.json")
    sess = _mk_sessions(g["sessions"])
    S = len(sess)
    maxb = 8
    tables = np.full((S, maxb), -1, dtype=np.int64)
    nblocks = np.zeros(S, dtype=np.int64)
    page = 0
    for s, d in enumerate(g["sessions"]):
        nblocks[s] = d["resident_blocks"]
        for b in range(d["resident_blocks"]):
            tables[s, b] = page
            page += 1
    prior = g["reply_prior_us"]
    for sid, want in g["expect_t_next"].items():
        assert t_next(sess[int(sid)], 0, prior, 80000) == want
    vs, vb, _ = select_victims(tables, nblocks, sess, g["now_us"], g["k"], 0, prior, 80000)
    assert [[int(a), int(b)] for a, b in zip(vs, vb)] == g["expect_next_use_victims"]
    # LRU contrast: least recently used session first (written here, not in the oracle)
    lru_order = sorted(range(S), key=lambda s: g["sessions"][s]["last_use_us"])
    lru = []
    for s in lru_order:
        if "RUNNING" in g["sessions"][s]["flags"]:
            continue
        for b in range(int(nblocks[s]) - 1, -1, -1):
            if len(lru) < g["k"]:
                lru.append(s)
    assert lru == g["expect_lru_victims_sessions"]
    # barge-in on session 1 makes it immediate reuse: protected
    se.apply_event(sess[1], se.SE_BARGE_IN, g["now_us"])
    vs, vb, _ = select_victims(tables, nblocks, sess, g["now_us"], g["k"], 0, prior, 80000)
    assert [[int(a), int(b)] for a, b in zip(vs, vb)] == g["barge_in_variant"]["expect_victims"]


# ----------------------------------------------------------------------------- random pools
def _random_pool(rng, S, maxb, fallback_states=True):
    sess = []
    for s in range(S):
        st = se.SessionState()
        st.gen_us = int(rng.integers(0, 5)) * 1_000_000     # few distinct values: many ties
        st.play_us = int(rng.integers(0, st.gen_us + 1)) if st.gen_us else 0
        if rng.random() < 0.5:
            st.reply_n = 1
            st.reply_ema_us = int(rng.integers(0, 3)) * 1_000_000
        r = rng.random()
        if r < 0.15:
            st.flags |= se.RUNNING
        elif r < 0.3:
            st.flags |= se.IMMEDIATE
        elif r < 0.45 and fallback_states:
            st.protect_until_us = 10_000_000
        sess.append(st)
    tables = np.full((S, maxb), -1, dtype=np.int64)
    nblocks = rng.integers(0, maxb + 1, S)
    page = 0
    for s in range(S):
        for b in range(int(nblocks[s])):
            if rng.random() < 0.7:
                tables[s, b] = page
                page += 1
            else:
                tables[s, b] = -2 - b          # host-resident: never a victim
    return sess, tables, nblocks


def _prefers(x, y, keyof, within):
    """True when candidate x must be evicted before candidate y (Section 5.1 wording).

    keyof(sid) -> (tier, T_next).  The normally eligible tier comes first; then the
    session with the later predicted next use; equal estimates by smaller session id;
    within a session the suffix (larger block id) first, or the smaller block id
    under ASCENDING."""
    (sx, bx), (sy, by) = x, y
    tx, nx = keyof(sx)
    ty, ny = keyof(sy)
    if tx != ty:
        return tx < ty
    if nx != ny:
        return nx > ny
    if sx != sy:
        return sx < sy
    return bx > by if within == SUFFIX_FIRST else bx < by


@pytest.mark.parametrize("within", [SUFFIX_FIRST, ASCENDING])
@pytest.mark.parametrize("fallback", [False, True])
def test_order_pairwise_and_formulations_agree(within, fallback):
    rng = np.random.default_rng(1234 + within + 2 * fallback)
    now = 5_000_000
    prior = 3_000_000
    for trial in range(60):
        sess, tables, nblocks = _random_pool(rng, int(rng.integers(1, 9)), int(rng.integers(1, 7)))
        a = order_global(tables, nblocks, sess, now, 0, prior, 80000, within, fallback)
        b = order_scan(tables, nblocks, sess, now, 0, prior, 80000, within, fallback=fallback)
        assert [list(map(int, x)) for x in a] == [list(map(int, x)) for x in b]

        # the candidate set, written from the eligibility rules directly
        def tier_of(s):
            st = sess[s]
            if st.flags & se.RUNNING:
                return None
            protected = bool(st.flags & se.IMMEDIATE) or now < st.protect_until_us
            if not protected:
                return 0
            return 1 if fallback else None
        cand = {(s, bb) for s in range(len(sess)) for bb in range(int(nblocks[s]))
                if tables[s, bb] >= 0 and tier_of(s) is not None}
        got = list(zip(a[0].tolist(), a[1].tolist()))
        assert set(got) == cand and len(got) == len(cand)

        def keyof(s):
            return tier_of(s), t_next(sess[s], 0, prior, 80000)
        for i in range(len(got)):
            for j in range(i + 1, len(got)):
                assert _prefers(got[i], got[j], keyof, within), (got[i], got[j])
        assert all(a[2][i] == tables[got[i]] for i in range(len(got)))


def test_topk_is_the_unique_dominating_subset_brute_force():
    """For tiny pools, enumerate every k-subset of candidates: exactly one subset has
    every member ranked before every non-member, and it is the oracle's top-k."""
    rng = np.random.default_rng(7)
    now, prior = 5_000_000, 3_000_000
    n_checked = 0
    for trial in range(40):
        sess, tables, nblocks = _random_pool(rng, int(rng.integers(2, 5)), 4)
        full = order_global(tables, nblocks, sess, now, 0, prior, 80000)
        cand = list(zip(full[0].tolist(), full[1].tolist()))
        if not 1 <= len(cand) <= 12:
            continue

        def keyof(s):
            return 0, t_next(sess[s], 0, prior, 80000)
        for k in range(0, len(cand) + 2):
            winners = []
            for sub in itertools.combinations(cand, min(k, len(cand))):
                rest = [c for c in cand if c not in sub]
                if all(_prefers(x, y, keyof, SUFFIX_FIRST) for x in sub for y in rest):
                    winners.append(set(sub))
            assert len(winners) == 1
            vs, vb, _ = select_victims(tables, nblocks, sess, now, k, 0, prior, 80000)
            assert set(zip(vs.tolist(), vb.tolist())) == winners[0]
            n_checked += 1
    assert n_checked > 50


def test_special_cases():
    rng = np.random.default_rng(3)
    sess, tables, nblocks = _random_pool(rng, 6, 5)
    now, prior = 5_000_000, 3_000_000
    full = order_global(tables, nblocks, sess, now, 0, prior, 80000)
    n = full[0].size
    assert select_victims(tables, nblocks, sess, now, 0, 0, prior, 80000)[0].size == 0
    assert select_victims(tables, nblocks, sess, now, n + 5, 0, prior, 80000)[0].size == n
    for s in full[0]:
        st = sess[int(s)]
        assert not st.flags & (se.RUNNING | se.IMMEDIATE) and now >= st.protect_until_us
    # within a session the victims taken first are its highest resident blocks
    for s in set(full[0].tolist()):
        bl = full[1][full[0] == s].tolist()
        assert bl == sorted(bl, reverse=True)
        res = [b for b in range(int(nblocks[s])) if tables[s, b] >= 0]
        assert sorted(bl) == res
    # no session resident at all
    empty = np.full_like(tables, -1)
    assert order_global(empty, nblocks, sess, now, 0, prior, 80000)[0].size == 0


def test_protection_window_expires():
    st = se.SessionState()
    se.apply_event(st, se.SE_PRELOADED, 1_000_000, protect_us=2_000_000)
    tables = np.array([[0, 1]], dtype=np.int64)
    nb = np.array([2])
    assert order_global(tables, nb, [st], 2_999_999, 0, 3_000_000, 80000)[0].size == 0
    assert order_global(tables, nb, [st], 3_000_000, 0, 3_000_000, 80000)[0].size == 2
    se.apply_event(st, se.SE_TURN_BEGIN, 1_500_000)
    assert st.protect_until_us == 0


def test_lru_baseline_order_pairwise():
    """The LRU baseline (Sections 2.3 and 5: rank by last use, not next use):
    only running KV is pinned; least recently used session first, equal times by
    smaller session id, suffix blocks first."""
    from oracle.policy import order_lru
    rng = np.random.default_rng(99)
    for trial in range(40):
        sess, tables, nblocks = _random_pool(rng, int(rng.integers(1, 9)), int(rng.integers(1, 6)))
        for st in sess:
            st.last_use_us = int(rng.integers(0, 4)) * 1_000_000
        s_, b_, p_ = order_lru(tables, nblocks, sess)
        got = list(zip(s_.tolist(), b_.tolist()))
        cand = {(s, b) for s in range(len(sess)) for b in range(int(nblocks[s]))
                if tables[s, b] >= 0 and not (sess[s].flags & se.RUNNING)}
        assert set(got) == cand and len(got) == len(cand)
        for i in range(len(got)):
            for j in range(i + 1, len(got)):
                (sx, bx), (sy, by) = got[i], got[j]
                tx, ty = sess[sx].last_use_us, sess[sy].last_use_us
                assert (tx < ty) or (tx == ty and (sx < sy or (sx == sy and bx > by))), (got[i], got[j])


def test_lru_picks_the_older_session_in_the_paper_scenario():
    from oracle.policy import order_lru
    g = _load("scenario_lru_vs_next_use.json")
    sess = _mk_sessions(g["sessions"])
    for st, d in zip(sess, g["sessions"]):
        st.last_use_us = d["last_use_us"]
    tables = np.full((3, 8), -1, dtype=np.int64)
    nblocks = np.zeros(3, dtype=np.int64)
    page = 0
    for s, d in enumerate(g["sessions"]):
        nblocks[s] = d["resident_blocks"]
        for b in range(d["resident_blocks"]):
            tables[s, b] = page
            page += 1
    s_, _, _ = order_lru(tables, nblocks, sess)
    assert s_[:g["k"]].tolist() == g["expect_lru_victims_sessions"]
