"""GPU vs oracle parity through the C ABI, bit for bit (victim lists, host slots,
HBM pages, block and owner tables, session states, and KV bytes)."""
import numpy as np
import pytest

from workloads import make_workload

from ._lockstep import run_lockstep

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("seed,driver,mode", [(0, "device", 0), (1, "device", 0), (0, "exchange", 0),
                                              (1, "sequential", 0), (0, "exchange", 2),
                                              (1, "sequential", 2), (2, "exchange", 18),
                                              (3, "device", 0), (4, "device", 0)])
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


@pytest.mark.parametrize("driver,mode", [("device", 0), ("exchange", 2)])
def test_tiny_workload_address_tagged_bytes(driver, mode):
    """The tiny script with address-tagged KV contents (every 16-byte chunk holds its
    session, token, layer, K/V and chunk): full byte images after every 25 events, so a
    misplaced byte would be reported with where it came from."""
    wl = make_workload("tiny", 5)
    om, gm = run_lockstep(wl, with_bytes=True, check_every=25, driver=driver, mode=mode, tagged=True)
    assert om.counters == gm.counters and gm.counters["pages_out"] > 300


@pytest.mark.parametrize("driver", ["device", "exchange"])
def test_tiny_workload_tma_exchange_copy(driver, monkeypatch):
    """The exchange's copies moved by TMA bulk copies (LV_EXCHANGE_KERNEL=tma) instead of
    16-byte loads and stores: the tiny script with address-tagged contents, every
    decision and full byte images after every 25 events."""
    monkeypatch.setenv("LV_EXCHANGE_KERNEL", "tma")
    wl = make_workload("tiny", 6)
    om, gm = run_lockstep(wl, with_bytes=True, check_every=25, driver=driver, mode=0, tagged=True)
    assert om.counters == gm.counters and gm.counters["pages_out"] > 300


@pytest.mark.parametrize("driver,mode", [("device", 0), ("exchange", 0), ("exchange", 2),
                                         ("sequential", 0)])
def test_hand_worked_turns(driver, mode):
    """The hand-worked script of tests/golden/manager_turns_hand.json (a preload, growth,
    the foreground fallback tier, an eviction with a shortfall): every decision and the
    state with address-tagged bytes after every event."""
    from ._hand import hand_workload, load
    g = load("manager_turns_hand.json")
    om, gm = run_lockstep(hand_workload(g), with_bytes=True, check_every=1, driver=driver,
                          mode=mode, tagged=True)
    assert om.pool.tables.tolist() == g["expect_tables"]


@pytest.mark.parametrize("driver", ["device", "sequential"])
def test_tiny_workload_lru_baseline(driver):
    """The LRU baseline policy on the same kernels (NEXT f3): every ranking and
    every move of the tiny script, with full byte images."""
    wl = make_workload("tiny", 3)
    wl.spec = wl.spec.with_(policy=1)
    om, gm = run_lockstep(wl, with_bytes=True, check_every=100, driver=driver)
    assert om.counters == gm.counters and gm.counters["preloads"] == 0


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


def _sampled_full_size(wl, driver, mode, n_sample=48, rank_on="turns", record=True,
                       async_copy=False):
    """Every event's decisions (when recorded), the final tables/owners/sessions, and
    the bytes of sampled blocks (plus blocks the last movements touched) against the
    oracle."""
    import torch
    from oracle import OracleManager
    from paper_2606_22983_gb300.harness import ContentWriter, pool_for
    from paper_2606_22983_gb300.manager import KVManager
    from workloads import scatter_order, value_table
    from ._lockstep import compare_records, compare_state

    om = OracleManager(wl, with_bytes=False, rank_on=rank_on)
    pool = pool_for(wl)
    try:
        writer = ContentWriter(pool, wl)
        writer.write_initial(wl)
        gm = KVManager(pool, perms=wl.perms, rank_on=rank_on if record else "none", driver=driver,
                       mode=mode, order_fn=scatter_order, on_append=writer.write_appended,
                       record=record, async_copy=async_copy,
                       # unrecorded runs take the script's load keys from the device
                       script=None if record else wl)
        touched = []
        for i in range(wl.n_events):
            ro, rg = om.step(i), gm.step(wl.event(i), i)
            if record:
                compare_records(ro, rg, i)
            if "victims" in ro and len(ro["victims"]):
                touched += [(int(a), int(b)) for a, b, _ in ro["victims"][:8]]
            if "in_blocks" in ro:
                touched += [(int(ro["sid"]), int(b)) for b in ro["in_blocks"][:8]]
        compare_state(om, pool, "end", with_bytes=False)
        table = value_table(wl.seed)
        rng = np.random.default_rng(0)
        t = om.pool.tables
        placed = np.argwhere(t != -1)
        sample = {tuple(int(x) for x in placed[r])
                  for r in rng.choice(len(placed), min(n_sample, len(placed)), replace=False)}
        sample |= set(touched[-64:])
        for s_, b in sorted(sample):
            e = int(t[s_, b])
            want = _expected_block(wl.seed, table, wl.spec.shape, s_, b, int(om.pool.ctx[s_]))
            got = pool.kv[:, e, :].cpu().numpy() if e >= 0 else pool.host[-(e + 2)]
            assert np.array_equal(got, want), (s_, b, e)
        assert om.counters["pages_out"] > 0 and om.counters["pages_in"] > 0
        return om, gm
    finally:
        torch.cuda.synchronize()
        pool.close()
        torch.cuda.empty_cache()


def test_thinker_full_size_pipelined_staged_exchanges():
    """Staged (copy-engine) exchanges with LV_MODE_ASYNC: each call's transfers and
    unpacks overlap the next calls, ordered transfer by transfer; no byte readback
    between turns.  The end state and sampled bytes equal the oracle's."""
    _sampled_full_size(make_workload("thinker", 3, n_turns=30), "exchange", 2, record=False,
                       async_copy=True)


def test_thinker_full_size_async_copies():
    """Thinker turns with each turn's copy on the pool's copy stream and no host
    round trip between turns (the next turn ranks and plans while the previous
    turn's pages still move): the end state and sampled bytes equal the oracle's."""
    _sampled_full_size(make_workload("thinker", 1, n_turns=30), "device", 0, record=False,
                       async_copy=True)


def test_thinker_full_size_tma_exchange_copy(monkeypatch):
    """Thinker turns at full size with the TMA exchange copy and asynchronous copies
    (nothing read back between turns): end state and sampled bytes equal the oracle's."""
    monkeypatch.setenv("LV_EXCHANGE_KERNEL", "tma")
    _sampled_full_size(make_workload("thinker", 2, n_turns=30), "device", 0, record=False,
                       async_copy=True)


@pytest.mark.parametrize("driver,mode", [("device", 0), ("exchange", 0), ("exchange", 2)])
def test_thinker_full_size_sampled_bytes(driver, mode):
    """The thinker pool at full size (40 GB HBM budget, 1.5 MiB pages), in the
    launch configuration the benchmark times."""
    _sampled_full_size(make_workload("thinker", 0, n_turns=6), driver, mode)


def _at_stated_size(name, seed):
    """The workload at its stated session count (256 mixed, 1024 frag) when this host
    can page-lock its host tier within min(400 GB, 0.8 * MemAvailable), else scaled
    down to that limit; the sizing is printed (pytest -rP shows it) and checked."""
    from workloads import STATED_SESSIONS, host_tier_limit, mem_available_bytes
    mem = mem_available_bytes()
    wl = make_workload(name, seed, host_limit=host_tier_limit(mem))
    sz = wl.meta["sizing"]
    print(f"sizing {name} seed {seed}: MemAvailable {mem} B, limit {sz['host_limit_bytes']} B, "
          f"sessions {sz['sessions']} of {sz['stated_sessions']}, host tier {sz['host_tier_bytes']} B")
    assert sz["host_tier_bytes"] <= sz["host_limit_bytes"]
    assert sz["stated_sessions"] == STATED_SESSIONS[name]
    if not sz["scaled"]:
        assert wl.spec.n_sessions == STATED_SESSIONS[name]
    return wl


def test_mixed_realtime_full_size():
    """Mixed realtime load: 256 sessions (log-uniform 2k-16k tokens) with Poisson
    next-speech arrivals, barge-ins, speech-triggered preloads and turns with
    growth; 60 GB HBM budget, a ~115-135 GB host tier; 3000 events."""
    om, gm = _sampled_full_size(_at_stated_size("mixed", 0), "device", 0)
    assert om.counters["preloads"] > 50 and om.counters == gm.counters


def test_mixed_realtime_full_size_async_copies():
    """The mixed workload with every turn's and preload's copy left running on the pool's
    copy stream (turns, preloads and growth overlap earlier copies): the end state and
    sampled bytes equal the oracle's."""
    om, gm = _sampled_full_size(_at_stated_size("mixed", 1), "device", 0, record=False,
                                async_copy=True)


def test_long_multimodal_full_size_pipelined_staged():
    """The long workload's multi-GB turns through the copy-engine path with pipelined
    (asynchronous) staged exchanges: the staging runs grow to several GB and are reused
    by alternate calls.  The end state and sampled bytes equal the oracle's."""
    _sampled_full_size(make_workload("long", 1), "exchange", 2, record=False, async_copy=True)


def test_long_multimodal_full_size():
    """16 sessions of 32k-64k tokens (3-6 GB each, 30 % frame tokens); every turn
    evicts and reloads several GB at once through the exchange."""
    om, gm = _sampled_full_size(make_workload("long", 0), "device", 0)
    assert om.counters["pages_in"] > 16 * 1000


@pytest.mark.parametrize("driver,async_copy", [("exchange", False), ("device", False),
                                               ("device", True)])
def test_fragmentation_full_size(driver, async_copy):
    """Pages randomly permuted over a 100 GB HBM budget, 1024 sessions of
    256-4096 tokens (~219 GB of KV, a ~148 GB host tier); 10 000 events alternating
    "free k pages" with turns whose reload list comes in a scattered order (with the
    device driver, the evictions run through lv_evict and the turns through lv_turn
    with load keys; with asynchronous copies, nothing is read back between events)."""
    om, gm = _sampled_full_size(_at_stated_size("frag", 0), driver, 0, rank_on="none",
                                record=not async_copy, async_copy=async_copy)
    assert om.counters["turns"] == 5000
