"""Inclusive tiers on the GPU against the oracle, bit for bit: every decision,
every host slot (a clean copy where the block has one), the block and owner
tables, the clean-copy counters and the KV bytes of both tiers."""
import pytest

from workloads import make_workload, pool_spec

from ._lockstep import run_lockstep
from .test_parity_gpu import _sampled_full_size

pytestmark = pytest.mark.gpu


def _inclusive(name, seed, **over):
    return make_workload(name, seed, spec=pool_spec(name).with_(tiers=1), **over)


@pytest.mark.parametrize("seed,driver,mode", [(0, "device", 0), (1, "exchange", 0),
                                              (0, "sequential", 0), (1, "device", 2),
                                              (0, "exchange", 2), (1, "sequential", 2)])
def test_tiny_inclusive_full_images(seed, driver, mode):
    """1000 tiny events with clean copies kept: evictions that find one move no
    bytes, appends into a clean tail drop it; full byte images every 50 events."""
    om, gm = run_lockstep(_inclusive("tiny", seed), with_bytes=True, check_every=50,
                          driver=driver, mode=mode)
    assert om.counters == gm.counters
    assert om.pool.clean_out > 200 and om.pool.clean_dropped > 10
    page = om.pool.J * om.pool.P
    assert om.pool.bytes_out == (om.counters["pages_out"] - om.pool.clean_out) * page


def test_thinker_inclusive_full_size():
    """Thinker turns with clean copies: after a session has been reloaded once,
    evicting it again moves no bytes (turns never append)."""
    om, gm = _sampled_full_size(_inclusive("thinker", 0, n_turns=20), "device", 0)
    assert om.pool.clean_out > 0
    assert om.pool.clean_dropped == 0


def test_tiny_inclusive_lru_baseline():
    """Inclusive tiers under the LRU baseline policy (no preloads)."""
    wl = make_workload("tiny", 3, spec=pool_spec("tiny").with_(tiers=1, policy=1))
    om, gm = run_lockstep(wl, with_bytes=True, check_every=100, driver="device")
    assert om.counters == gm.counters and om.pool.clean_out > 0


def test_thinker_inclusive_async_copies():
    """Inclusive tiers with asynchronous turn copies and no host round trip."""
    om, gm = _sampled_full_size(_inclusive("thinker", 2, n_turns=30), "device", 0, record=False,
                                async_copy=True)
    assert om.pool.clean_out > 0


def test_inclusive_swap_out_over_several_chunks():
    """One swap-out of 1500 victims (more than a CTA's 1024 threads), 800 without a
    clean copy and 700 with one, in suffix-first order: the in-place spread of the
    compact slot allocation over two chunks gives the oracle's slots, tables and bytes."""
    import numpy as np
    import torch
    from oracle.pool import OraclePool, _enc_host
    from paper_2606_22983_gb300.pool import KVPool
    S, B, N = 2, 2048, 2000
    pool = KVPool(layers=1, kv_heads=1, head_dim=8, max_sessions=S, max_blocks=B, hbm_pages=4096,
                  hbm_budget_pages=4096, host_pages=4096, tiers=1)
    om = OraclePool(1, 1, 8, 16, 2, S, B, 4096, 4096, 4096, with_bytes=True, inclusive=True)
    try:
        rng = np.random.default_rng(7)
        placement = np.full((S, B), -1, np.int64)
        order = rng.permutation(N)
        hbm_blocks, host_blocks = np.sort(order[:800]), np.sort(order[800:])
        placement[0, hbm_blocks] = rng.permutation(4096)[:800]
        placement[0, host_blocks] = -(rng.permutation(4096)[:1200] + 2)
        ctx = np.array([N * 16, 0])
        om.import_placement(placement, ctx)
        pool.import_placement(placement.astype(np.int32), ctx.astype(np.int32))
        om.hbm[:] = rng.integers(0, 256, om.hbm.shape, dtype=np.uint8)
        om.host[:] = rng.integers(0, 256, om.host.shape, dtype=np.uint8)
        pool.kv.copy_(torch.from_numpy(om.hbm).to(pool.device))
        pool.host[:] = om.host
        torch.cuda.synchronize()
        # reload 700 of the host blocks: they keep their slots as clean copies
        back = np.sort(rng.permutation(host_blocks)[:700])
        pages = om.swap_in(0, back)
        om.remap(np.zeros(700, np.int64), back, pages)
        gp, commit = pool.swap_in(0, torch.from_numpy(back.astype(np.int32)).to(pool.device), 700)
        pool.remap(commit, 700)
        assert np.array_equal(gp.cpu().numpy(), pages.astype(np.int32))
        assert om.clean_copies() == 700
        # evict every resident block at once
        from oracle import sessions as se
        from oracle.policy import select_victims
        vs, vb, vp = select_victims(om.tables, om.nblocks, [se.SessionState(ctx_tokens=N * 16),
                                                            se.SessionState()], 0, 1500, 0,
                                    3_000_000, 80_000)
        victims, n = pool.select(0, 1500)
        assert n == 1500 and np.array_equal(victims.cpu().numpy(), np.stack([vs, vb, vp], 1).astype(np.int32))
        slots = om.swap_out(vs, vb, vp)
        gs, commit = pool.swap_out(victims, n)
        assert np.array_equal(gs.cpu().numpy(), slots.astype(np.int32))
        om.remap(vs, vb, _enc_host(slots))
        pool.remap(commit, n)
        assert pool.sync(raise_on_error=False) == 0
        assert om.clean_out == 700
        t, oh, oo = pool.tables()
        assert np.array_equal(t, om.tables.astype(np.int32))
        assert np.array_equal(pool.host, om.host)
        st = pool.stats()
        assert st["clean_out"] == 700 and st["clean_copies"] == 0
        assert st["host_allocated"] == int(om.host_used.sum())
    finally:
        torch.cuda.synchronize()
        pool.close()
