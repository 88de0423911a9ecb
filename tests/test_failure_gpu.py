"""Failure paths without a GPU fault: an allocation that fails, a copy-engine
transfer that is never issued, a device wait that runs out.  After each, the old
mapping and every byte are intact (Section 5.2: a failed or cancelled transfer
affects latency, not correctness), and the pool keeps working."""
import numpy as np
import pytest

pytestmark = pytest.mark.gpu


def _setup():
    from paper_2606_22983_gb300.harness import ContentWriter, pool_for, zero_host
    from workloads import make_workload, pool_spec
    wl = make_workload("tiny", 0, spec=pool_spec("tiny").with_(hbm_budget_pages=128), all_resident=False)
    pool = pool_for(wl)
    w = ContentWriter(pool, wl)
    zero_host(pool)
    w.write_initial(wl)
    return wl, pool


def _snapshot(pool):
    t, oh, oo = pool.tables()
    st = pool.stats()
    return (t.copy(), oh.copy(), oo.copy(), st["hbm_allocated"], st["host_allocated"],
            pool.kv.cpu().numpy().copy(), pool.host.copy())


def _same(a, b):
    return all(np.array_equal(x, y) if isinstance(x, np.ndarray) else x == y for x, y in zip(a, b))


def test_injected_allocation_failures_change_nothing():
    from paper_2606_22983_gb300 import lv
    wl, pool = _setup()
    try:
        victims, n = pool.select(0, 6)
        before = _snapshot(pool)
        lv.lv_inject_fault(pool.handle, lv.LV_FAULT_HOST_ALLOC, 0)
        pool.swap_out(victims, n)
        assert pool.sync(raise_on_error=False) == lv.LV_ERR_NO_HOST
        pool.clear_error()
        assert _same(before, _snapshot(pool))
        # a swap-out that completes but is abandoned: its host reservations are
        # released and nothing else changes (the slots' bytes are scratch)
        slots, commit = pool.swap_out(victims, n)
        assert pool.sync(raise_on_error=False) == 0
        pool.cancel((-(slots.long() + 2)).to(torch_int32()), n)
        assert pool.sync(raise_on_error=False) == 0
        assert _same(before[:6], _snapshot(pool)[:6])
        # the same swap-out, committed: its blocks are now in the host tier
        slots, commit = pool.swap_out(victims, n)
        pool.remap(commit, n)
        assert pool.sync(raise_on_error=False) == 0
        mid = _snapshot(pool)
        # an HBM-side failure on their reload (host reservations do not count:
        # the swap-in's is the first HBM allocation after arming)
        _, host = pool.counts()
        sid = int(np.nonzero(host)[0][0])
        blks, nb = pool.blocks(sid, 1)
        lv.lv_inject_fault(pool.handle, lv.LV_FAULT_HBM_ALLOC, 0)
        pool.swap_in(sid, blks, nb)
        assert pool.sync(raise_on_error=False) == lv.LV_ERR_NO_HBM
        pool.clear_error()
        assert _same(mid, _snapshot(pool))
        # and the pool still works: the reload now succeeds and commits
        pages, commit = pool.swap_in(sid, blks, nb)
        pool.remap(commit, nb)
        assert pool.sync(raise_on_error=False) == 0
    finally:
        pool.close()


def torch_int32():
    import torch
    return torch.int32


def test_unissued_copy_engine_transfer_leaves_the_old_mapping():
    from paper_2606_22983_gb300 import lv
    wl, pool = _setup()
    try:
        victims, n = pool.select(0, 6)                                # give some blocks a host slot
        slots, commit = pool.swap_out(victims, n)
        pool.remap(commit, n)
        assert pool.sync(raise_on_error=False) == 0
        _, host = pool.counts()
        sid = int(np.nonzero(host)[0][0])
        blks, nb = pool.blocks(sid, 1)
        before = _snapshot(pool)
        lv.lv_inject_fault(pool.handle, lv.LV_FAULT_COPY, 0)
        with pytest.raises(lv.LvError) as e:
            pool.swap_in(sid, blks, nb, lv.LV_MODE_STAGED)
        assert e.value.status == lv.LV_ERR_CUDA
        pages = pool.pages[:nb].clone()
        pool.cancel(pages, nb)                                        # release the reservations
        assert pool.sync(raise_on_error=False) == 0
        assert _same(before, _snapshot(pool))
        # a clean retry through the same path loads exactly the host bytes
        pages, commit = pool.swap_in(sid, blks, nb, lv.LV_MODE_STAGED)
        pool.remap(commit, nb)
        assert pool.sync(raise_on_error=False) == 0
        t, _, _ = pool.tables()
        for b, p in zip(blks.cpu().tolist(), pages.cpu().tolist()):
            slot = -(int(before[0][sid, b]) + 2)
            assert t[sid, b] == p
            assert np.array_equal(pool.kv[:, p, :].cpu().numpy(), before[6][slot])
    finally:
        pool.close()


def test_bounded_device_wait_reports_a_timeout_and_the_context_survives():
    from paper_2606_22983_gb300 import lv
    wl, pool = _setup()
    try:
        lv.lv_selftest_wait(pool.handle, 200_000, pool.stream)        # 0.2 s, nothing completes it
        assert pool.sync(raise_on_error=False) == lv.LV_ERR_TIMEOUT
        pool.clear_error()
        victims, n = pool.select(0, 3)
        slots, commit = pool.swap_out(victims, n)
        pool.remap(commit, n)
        assert pool.sync(raise_on_error=False) == 0
    finally:
        pool.close()
