"""Pins for the oracle's preload controller (Section 5.2): properties that the
paper's description fixes, checked on its decisions rather than re-typed."""
import numpy as np
import pytest

from oracle.preload import ControlledOracleManager, PreloadController
from workloads import make_workload

CASES = [("tiny", 1, 1_000_000, 40), ("mixed", 2_000, 2_000_000, 2000), ("mixed", 5_000, 3_000_000, 3000)]


@pytest.mark.parametrize("name,bw,lead,cap", CASES)
def test_controller_properties(name, bw, lead, cap):
    wl = make_workload(name, 0)
    m = ControlledOracleManager(wl, PreloadController(link_bytes_per_us=bw, lead_prior_us=lead,
                                                      cap_pages=cap), with_bytes=False, rank_on="none")
    intervals = []
    page_bytes = wl.spec.shape.page_bytes
    for i in range(wl.n_events):
        rec = m.step(i)
        for sid, start, finish, t_pred, pages in rec.get("admitted", []):
            # admitted only when the copy can finish unseen: the transfer ends by the predicted turn
            assert finish <= t_pred
            assert start >= rec["t"] and finish - start == -(-len(pages) * page_bytes // bw)
            intervals.append((start, finish))
        if rec.get("completed"):
            # the cap on warmed (protected) KV holds after every completion
            now = rec["t"]
            prot = [s for s, st in enumerate(m.sessions) if st.protect_until_us > now]
            res = sum(int((m.pool.tables[s, :int(m.pool.nblocks[s])] >= 0).sum()) for s in prot)
            assert res <= cap
        if i % 200 == 0:
            m.pool.check_invariants()
    m.pool.check_invariants()
    # transfers are serialised on the modelled link
    intervals.sort()
    for (a0, b0), (a1, b1) in zip(intervals, intervals[1:]):
        assert a1 >= b0
    c = m.counters
    assert c["admitted"] == c["completed"] + c["cancelled"] + len(m.pending)
    assert c["hits"] <= c["completed"]


def test_controller_exercises_every_path():
    wl = make_workload("tiny", 0)
    m = ControlledOracleManager(wl, PreloadController(link_bytes_per_us=1, lead_prior_us=1_000_000,
                                                      cap_pages=40), with_bytes=False, rank_on="none")
    recs = m.run()
    c = m.counters
    assert c["waited"] > 0 and c["given_up"] > 0 and c["cancelled"] > 0 and c["hits"] > 0
    assert sum(len(r.get("unprotected", [])) for r in recs) > 0


def test_fast_link_admits_every_preload_and_hides_reloads():
    """With a link fast enough and HBM for about half of all KV (the mixed workload with
    128 sessions), every preload is admitted and completes, and most turns find their
    KV already resident (the paper's prefetch hit).  At the stated 256 sessions the 60 GB
    budget holds a third of the KV, so preloads evict one another before their turns."""
    from workloads import pool_spec
    wl = make_workload("mixed", 0, spec=pool_spec("mixed").with_(n_sessions=128))
    m = ControlledOracleManager(wl, PreloadController(link_bytes_per_us=200_000), with_bytes=False,
                                rank_on="none")
    m.run()
    c = m.counters
    assert c["admitted"] == c["completed"] and c["given_up"] == 0 and c["cancelled"] == 0
    assert c["hits"] > 0.6 * c["turns"] and c["sync_loads"] < 0.1 * c["turns"]


# ------------------------------------------------------ hand-worked scenarios
from ._hand import hand_workload, load as _load_hand


@pytest.mark.parametrize("index", [0, 1])
def test_controller_hand_worked_scenarios(index):
    """Every decision of two small scenarios, worked by hand from the controller's
    reading of Section 5.2 (tests/golden/preload_controller_hand.json)."""
    sc = _load_hand("preload_controller_hand.json")["scenarios"][index]
    c = sc["controller"]
    m = ControlledOracleManager(hand_workload(sc), PreloadController(link_bytes_per_us=c["link_bytes_per_us"],
                                                                     lead_prior_us=c["lead_prior_us"],
                                                                     cap_pages=c["cap_pages"]),
                                with_bytes=True, content="tagged", rank_on="none")
    admitted, victims, completed, cancelled, unprotected = [], {}, {}, {}, {}
    for i in range(m.wl.n_events):
        rec = m.step(i)
        for sid, start, finish, deadline, pages in rec.get("admitted", []):
            admitted.append({"event": i, "sid": sid, "start": start, "finish": finish,
                             "deadline": deadline, "pages": [int(x) for x in pages]})
        if rec.get("preload_victims"):
            victims[str(i)] = np.concatenate(rec["preload_victims"]).tolist()
        if rec.get("completed"):
            completed[str(i)] = list(rec["completed"])
        if "cancelled" in rec:
            cancelled[str(i)] = rec["cancelled"]
        if rec.get("unprotected"):
            unprotected[str(i)] = list(rec["unprotected"])
        m.pool.check_invariants()
    assert admitted == sc["expect_admitted"]
    assert victims == sc["expect_preload_victims"]
    assert completed == sc["expect_completed"]
    assert cancelled == sc["expect_cancelled"]
    assert unprotected == sc["expect_unprotected"]
    assert {k: m.counters[k] for k in sc["expect_counters"]} == sc["expect_counters"]
    assert {str(k): list(v) for k, v in m.lead.items()} == sc["expect_lead"]
    assert m.link_free_at == sc["expect_link_free_at"]
    assert m.pool.tables.tolist() == sc["expect_tables"]
