"""The hand-worked values of the policy goldens checked on the library directly, with no
oracle in between: the Section 5.1 scenario where next-use and LRU disagree (and its
barge-in variant), and the reply-interval average driven by monitor events."""
import json
import os

import numpy as np
import pytest

pytestmark = pytest.mark.gpu

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _load(name):
    with open(os.path.join(GOLDEN, name)) as f:
        return json.load(f)


def _pool(S, maxb, reply_prior_us, policy):
    from paper_2606_22983_gb300.pool import KVPool
    return KVPool(layers=2, kv_heads=2, head_dim=64, max_sessions=S, max_blocks=maxb, hbm_pages=16,
                  hbm_budget_pages=16, host_pages=16, reply_prior_us=reply_prior_us, policy=policy)


@pytest.mark.parametrize("policy", ["next_use", "lru"])
def test_scenario_next_use_versus_lru(policy):
    from paper_2606_22983_gb300 import lv
    g = _load("scenario_lru_vs_next_use.json")
    S, maxb, T = len(g["sessions"]), 8, 16
    pol = lv.LV_POLICY_NEXT_USE if policy == "next_use" else lv.LV_POLICY_LRU
    pool = _pool(S, maxb, g["reply_prior_us"], pol)
    try:
        placement = np.full((S, maxb), -1, np.int32)
        ctx = np.zeros(S, np.int32)
        page = 0
        for s, d in enumerate(g["sessions"]):
            ctx[s] = d["resident_blocks"] * T
            for b in range(d["resident_blocks"]):
                placement[s, b] = page
                page += 1
        pool.import_placement(placement, ctx)
        st = np.zeros(S, dtype=lv.SESSION_DTYPE)
        for s, d in enumerate(g["sessions"]):
            st[s]["gen_us"], st[s]["play_us"] = d["gen_us"], d["play_us"]
            st[s]["last_use_us"] = d["last_use_us"]
            st[s]["flags"] = lv.LV_RUNNING if "RUNNING" in d["flags"] else 0
        pool.set_sessions(st)
        vic, n = pool.select(g["now_us"], g["k"])
        got = vic[:n].cpu().numpy()
        if policy == "next_use":
            assert got[:, :2].tolist() == g["expect_next_use_victims"]
            ev = np.zeros(1, dtype=lv.EVENT_DTYPE)
            ev[0]["kind"], ev[0]["sid"], ev[0]["t_us"] = lv.LV_EV_BARGE_IN, 1, g["now_us"]
            pool.events(ev)
            vic, n = pool.select(g["now_us"], g["k"])
            assert vic[:n].cpu().numpy()[:, :2].tolist() == g["barge_in_variant"]["expect_victims"]
        else:
            assert got[:, 0].tolist() == g["expect_lru_victims_sessions"]
            assert got[:, 1].tolist() == [3, 2, 1]          # suffix first within the session
    finally:
        pool.close()


def test_reply_interval_events():
    from paper_2606_22983_gb300 import lv
    g = _load("reply_interval.json")
    kinds = {"PLAYBACK": lv.LV_EV_PLAYBACK, "SPEECH_START": lv.LV_EV_SPEECH_START,
             "SPEECH_STOP": lv.LV_EV_SPEECH_STOP, "BARGE_IN": lv.LV_EV_BARGE_IN,
             "TURN_BEGIN": lv.LV_EV_TURN_BEGIN, "TURN_END": lv.LV_EV_TURN_END}
    pool = _pool(1, 4, g["reply_prior_us"], lv.LV_POLICY_NEXT_USE)
    try:
        pool.import_placement(np.full((1, 4), -1, np.int32), np.zeros(1, np.int32))
        st = np.zeros(1, dtype=lv.SESSION_DTYPE)
        ini = g["initial"]
        st[0]["gen_us"], st[0]["play_us"] = ini["gen_us"], ini["play_us"]
        st[0]["flags"] = lv.LV_RESP_OPEN if ini["resp_open"] else 0
        pool.set_sessions(st)
        checked = 0
        for e in g["events"]:
            ev = np.zeros(1, dtype=lv.EVENT_DTYPE)
            ev[0]["kind"], ev[0]["sid"], ev[0]["t_us"] = kinds[e["ev"]], 0, e["t"]
            ev[0]["a"], ev[0]["b"] = e.get("a", 0), e.get("b", 0)
            pool.events(ev)
            now = pool.get_sessions()[0]
            for key, want in e.get("expect", {}).items():
                if key == "t_next":
                    continue            # not a stored field; the ranker's order is compared elsewhere
                assert int(now[key]) == want, (e, key)
                checked += 1
        assert checked >= 8
        assert pool.sync() == 0
    finally:
        pool.close()


def test_scenario_on_the_allocation_free_ranker():
    """The same scenario through lv_select_victims_noalloc, from caller-held session and
    block tables: the next-use victims, then the state a barge-in of session 1 leaves
    (its unplayed audio dropped, immediate reuse)."""
    import torch
    from paper_2606_22983_gb300 import lv
    g = _load("scenario_lru_vs_next_use.json")
    S, maxb, T = len(g["sessions"]), 8, 16
    st = np.zeros(S, dtype=lv.SESSION_DTYPE)
    tables = np.full((S, maxb), -1, np.int32)
    page = 0
    for s, d in enumerate(g["sessions"]):
        st[s]["ctx_tokens"] = d["resident_blocks"] * T
        st[s]["gen_us"], st[s]["play_us"] = d["gen_us"], d["play_us"]
        st[s]["flags"] = lv.LV_RUNNING if "RUNNING" in d["flags"] else 0
        for b in range(d["resident_blocks"]):
            tables[s, b] = page
            page += 1
    prm = lv.lv_rank_params(num_sessions=S, max_blocks=maxb, page_tokens=T, within_order=0,
                            t_play_mode=0, flags=0, reply_prior_us=g["reply_prior_us"], unit_us=80_000)
    tab = torch.from_numpy(tables).cuda()
    cap = 16

    def rank(states):
        sess = torch.from_numpy(states.view(np.uint8).copy()).cuda()
        out = torch.full((cap, 3), -7, dtype=torch.int32, device="cuda")
        cnt = torch.full((1,), -1, dtype=torch.int64, device="cuda")
        lv.lv_select_victims_noalloc(prm, sess, tab, g["now_us"], g["k"], out, cap, cnt, None)
        torch.cuda.synchronize()
        return out[:int(cnt.item())].cpu().numpy()

    assert rank(st)[:, :2].tolist() == g["expect_next_use_victims"]
    st[1]["gen_us"] = st[1]["play_us"]
    st[1]["flags"] |= lv.LV_IMMEDIATE
    assert rank(st)[:, :2].tolist() == g["barge_in_variant"]["expect_victims"]
