"""The Section 5.2 preload controller through liblv against the oracle's controller:
admissions (with their modelled start, finish and deadline), reserved pages,
completions, cancellations, dropped protections and every eviction and load,
event by event; byte images on the tiny pool, tables and sampled bytes on the
mixed pool at full size."""
import numpy as np
import pytest

from workloads import make_workload, scatter_order, value_table

pytestmark = pytest.mark.gpu


def _compare_controller(ro, rg, where):
    from ._lockstep import compare_records
    compare_records(ro, rg, where)
    ao, ag = ro.get("admitted", []), rg.get("admitted", [])
    assert len(ao) == len(ag), (where, ao, ag)
    for x, y in zip(ao, ag):
        assert tuple(int(v) for v in x[:4]) == tuple(int(v) for v in y[:4]), (where, x, y)
        assert np.array_equal(np.asarray(x[4], np.int64), np.asarray(y[4], np.int64)), where
    for key in ("completed", "unprotected"):
        assert list(map(int, ro.get(key, []))) == list(map(int, rg.get(key, []))), (where, key)
    assert ro.get("cancelled") == rg.get("cancelled"), where
    vo, vg = ro.get("preload_victims", []), rg.get("preload_victims", [])
    assert len(vo) == len(vg) and all(np.array_equal(np.asarray(a, np.int64), np.asarray(b, np.int64))
                                      for a, b in zip(vo, vg)), where


@pytest.mark.parametrize("name,bw,lead,cap,with_bytes,tiers", [
    ("tiny", 1, 1_000_000, 40, True, 0),
    ("tiny", 1, 1_000_000, 40, True, 1),
    ("mixed", 2_000, 2_000_000, 2000, False, 0),
])
def test_controller_matches_oracle(name, bw, lead, cap, with_bytes, tiers):
    import torch
    from oracle.preload import ControlledOracleManager, PreloadController
    from paper_2606_22983_gb300.controller import ControlledKVManager
    from paper_2606_22983_gb300.harness import ContentWriter, pool_for, zero_host
    from ._lockstep import compare_state

    from workloads import host_tier_limit, pool_spec
    wl = make_workload(name, 0, spec=pool_spec(name).with_(tiers=tiers),
                       host_limit=host_tier_limit() if name == "mixed" else None)
    table = value_table(wl.seed)
    om = ControlledOracleManager(wl, PreloadController(link_bytes_per_us=bw, lead_prior_us=lead,
                                                       cap_pages=cap),
                                 with_bytes=with_bytes, content=(wl.seed, table) if with_bytes else None,
                                 rank_on="none")
    pool = pool_for(wl)
    try:
        writer = ContentWriter(pool, wl)
        zero_host(pool)
        writer.write_initial(wl)
        gm = ControlledKVManager(pool, link_bytes_per_us=bw, lead_prior_us=lead, cap_pages=cap,
                                 perms=wl.perms, on_append=writer.write_appended,
                                 order_fn=scatter_order)
        for i in range(wl.n_events):
            ro, rg = om.step(i), gm.step(wl.event(i), i)
            _compare_controller(ro, rg, (i, wl.event(i)))
            if with_bytes and i % 100 == 99:
                compare_state(om, pool, i, True)
        compare_state(om, pool, "end", with_bytes)
        for k in ("admitted", "completed", "waited", "given_up", "cancelled", "hits", "sync_loads",
                  "pages_in", "pages_out"):
            assert om.counters[k] == gm.counters[k], k
        assert gm.counters["given_up"] > 0 and gm.counters["admitted"] > 0
        if name == "tiny":
            assert gm.counters["cancelled"] > 0
        else:
            # 256 sessions on a 60 GB budget: the host tier is tight, so most preloads wait
            # for room and are given up; the admitted ones complete before their turns
            assert gm.counters["waited"] > 0 and gm.counters["hits"] > 0
    finally:
        torch.cuda.synchronize()
        pool.close()
        torch.cuda.empty_cache()


@pytest.mark.parametrize("index", [0, 1])
def test_controller_hand_worked_scenarios(index):
    """The two scenarios of tests/golden/preload_controller_hand.json through the native
    controller: every decision against the oracle's, which the CPU tests pin to the
    hand-worked values; byte images compared after every event."""
    import torch
    from oracle.preload import ControlledOracleManager, PreloadController
    from paper_2606_22983_gb300.controller import ControlledKVManager
    from paper_2606_22983_gb300.harness import ContentWriter, pool_for, zero_host
    from ._hand import hand_workload, load
    from ._lockstep import compare_state

    sc = load("preload_controller_hand.json")["scenarios"][index]
    c = sc["controller"]
    wl = hand_workload(sc)
    om = ControlledOracleManager(wl, PreloadController(link_bytes_per_us=c["link_bytes_per_us"],
                                                       lead_prior_us=c["lead_prior_us"],
                                                       cap_pages=c["cap_pages"]),
                                 with_bytes=True, content=(wl.seed, value_table(wl.seed)),
                                 rank_on="none")
    pool = pool_for(wl)
    try:
        writer = ContentWriter(pool, wl)
        zero_host(pool)
        writer.write_initial(wl)
        gm = ControlledKVManager(pool, link_bytes_per_us=c["link_bytes_per_us"],
                                 lead_prior_us=c["lead_prior_us"],
                                 cap_pages=c["cap_pages"],
                                 perms=wl.perms, on_append=writer.write_appended,
                                 order_fn=scatter_order)
        for i in range(wl.n_events):
            ro, rg = om.step(i), gm.step(wl.event(i), i)
            _compare_controller(ro, rg, (i, wl.event(i)))
            compare_state(om, pool, i, True)
        for k, v in sc["expect_counters"].items():
            if k in gm.counters:
                assert gm.counters[k] == v, k
        assert om.pool.tables.tolist() == sc["expect_tables"]
    finally:
        torch.cuda.synchronize()
        pool.close()
