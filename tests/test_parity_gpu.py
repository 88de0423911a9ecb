"""GPU vs oracle parity through the C ABI, bit for bit (victim lists, host slots,
HBM pages, block and owner tables, session states, and KV bytes)."""
import numpy as np
import pytest

from workloads import make_workload

from ._lockstep import run_lockstep

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("seed,driver,mode", [(0, "device", 0), (1, "device", 0), (0, "exchange", 0),
                                              (1, "sequential", 0), (0, "exchange", 2),
                                              (1, "sequential", 2)])
def test_tiny_workload_full_images(seed, driver, mode):
    """1000 scripted events of the tiny pool: every ranking (full order after
    each event), eviction, preload, reload and growth, with full HBM and host
    byte images compared every 50 events -- through lv_make_resident, through
    select + lv_swap_exchange, and through the four sequential calls, with
    zero-copy kernels (mode 0) and with the staged copy-engine path (mode 2)."""
    wl = make_workload("tiny", seed)
    om, gm = run_lockstep(wl, with_bytes=True, check_every=50, driver=driver, mode=mode)
    assert om.counters == gm.counters
    assert gm.counters["pages_out"] > 500 and gm.counters["preloads"] > 10


def test_tiny_workload_ascending_and_counters_mode():
    """The literal block-ascending tie-break and the progress-counter T_play."""
    wl = make_workload("tiny", 2)
    wl.spec = wl.spec.with_(within_order=1, t_play_mode=1)
    om, gm = run_lockstep(wl, with_bytes=True, check_every=100, n_events=400)
    assert om.counters == gm.counters


def _expected_block(seed, table, shape, sid, blk, ctx):
    from workloads.content import subpage_offsets, subpage_values_np, valid_rows
    J = 2 * shape.layers
    off = subpage_offsets(seed, np.full(J, sid), np.full(J, blk), np.arange(J) // 2,
                          np.arange(J) % 2, shape)
    rows = np.full(J, int(valid_rows(ctx, blk, shape)))
    return subpage_values_np(table, off, rows, shape).view(np.uint8).reshape(J, -1)


@pytest.mark.parametrize("driver,mode", [("device", 0), ("exchange", 0), ("exchange", 2)])
def test_thinker_full_size_sampled_bytes(driver, mode):
    """The thinker pool at full size (40 GB HBM budget, 1.5 MiB pages), in the
    launch configuration the benchmark times: every turn's victims, host slots
    and pages match the oracle; afterwards the tables and owners match, and
    the bytes of sampled blocks (plus every block of the last turn) are the
    content of their logical position."""
    import torch
    from oracle import OracleManager
    from paper_2606_22983_gb300.harness import ContentWriter, pool_for
    from paper_2606_22983_gb300.manager import KVManager
    from workloads import value_table
    from ._lockstep import compare_records, compare_state

    wl = make_workload("thinker", 0, n_turns=6)
    om = OracleManager(wl, with_bytes=False, rank_on="turns")
    pool = pool_for(wl)
    try:
        writer = ContentWriter(pool, wl)
        writer.write_initial(wl)
        gm = KVManager(pool, perms=wl.perms, rank_on="turns", driver=driver, mode=mode)
        last = None
        for i in range(wl.n_events):
            ro, rg = om.step(i), gm.step(wl.event(i), i)
            compare_records(ro, rg, i)
            if ro["kind"] == 2:
                last = ro
        compare_state(om, pool, "end", with_bytes=False)
        table = value_table(wl.seed)
        rng = np.random.default_rng(0)
        t = om.pool.tables
        sample = set()
        placed = np.argwhere(t != -1)
        for r in rng.choice(len(placed), 48, replace=False):
            sample.add(tuple(int(x) for x in placed[r]))
        for s, b, _ in last["victims"][:32]:
            sample.add((int(s), int(b)))
        for b in last["in_blocks"][:32]:
            sample.add((int(last["sid"]), int(b)))
        for s, b in sorted(sample):
            e = int(t[s, b])
            want = _expected_block(wl.seed, table, wl.spec.shape, s, b, int(om.pool.ctx[s]))
            got = pool.kv[:, e, :].cpu().numpy() if e >= 0 else pool.host[-(e + 2)]
            assert np.array_equal(got, want), (s, b, e)
    finally:
        torch.cuda.synchronize()
        pool.close()
