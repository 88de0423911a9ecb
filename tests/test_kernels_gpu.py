"""Kernel-level GPU tests through the C ABI: the ranker against the oracle on random
session states (and at 2^20 resident pages), pack/unpack against the content
definition, remap / cancel / allocation error paths, degenerate sizes, and host
versus device pointer arguments."""
import os
import time

import numpy as np
import pytest

pytestmark = pytest.mark.gpu


def _tiny_pool(**kw):
    from paper_2606_22983_gb300.pool import KVPool
    args = dict(layers=2, kv_heads=2, head_dim=64, max_sessions=8, max_blocks=16, hbm_pages=64,
                hbm_budget_pages=64, host_pages=64)
    args.update(kw)
    return KVPool(**args)


def _oracle_states(st):
    from oracle import sessions as se
    out = []
    for r in st:
        out.append(se.SessionState(ctx_tokens=int(r["ctx_tokens"]), flags=int(r["flags"]),
                                   gen_us=int(r["gen_us"]), play_us=int(r["play_us"]),
                                   t_done_us=int(r["t_done_us"]), reply_ema_us=int(r["reply_ema_us"]),
                                   reply_n=int(r["reply_n"]), reply_tokens=int(r["reply_tokens"]),
                                   protect_until_us=int(r["protect_until_us"]),
                                   last_use_us=int(r["last_use_us"])))
    return out


def _random_states(rng, S):
    from paper_2606_22983_gb300 import lv
    st = np.zeros(S, dtype=lv.SESSION_DTYPE)
    st["gen_us"] = rng.integers(0, 6, S) * 1_000_000
    st["play_us"] = (rng.random(S) * st["gen_us"]).astype(np.int64) // 500_000 * 500_000
    st["reply_n"] = rng.integers(0, 2, S)
    st["reply_ema_us"] = rng.integers(0, 4, S) * 700_000
    st["reply_tokens"] = rng.integers(0, 80, S)
    fl = np.zeros(S, np.int32)
    fl |= np.where(rng.random(S) < 0.5, lv.LV_RESP_OPEN, 0).astype(np.int32)
    r = rng.random(S)
    fl |= np.where(r < 0.15, lv.LV_RUNNING, 0).astype(np.int32)
    fl |= np.where((r >= 0.15) & (r < 0.3), lv.LV_IMMEDIATE, 0).astype(np.int32)
    st["flags"] = fl
    st["protect_until_us"] = np.where((r >= 0.3) & (r < 0.45), 10_000_000, 0)
    return st


def _random_placement(rng, S, maxb, T, hbm_pages, host_pages, p_host=0.3):
    ctx = rng.integers(0, maxb * T + 1, S).astype(np.int32)
    nb = -(-ctx // T)
    placement = np.full((S, maxb), -1, np.int32)
    pages = rng.permutation(hbm_pages)
    slots = rng.permutation(host_pages)
    pi = hi = 0
    for s in range(S):
        for b in range(nb[s]):
            if rng.random() < p_host and hi < host_pages:
                placement[s, b] = -(int(slots[hi]) + 2)
                hi += 1
            elif pi < hbm_pages:
                placement[s, b] = int(pages[pi])
                pi += 1
            else:
                placement[s, b] = -(int(slots[hi]) + 2)
                hi += 1
    return placement, ctx


@pytest.mark.parametrize("within,tplay", [(0, 0), (1, 0), (0, 1)])
def test_ranker_matches_oracle_on_random_states(within, tplay):
    from paper_2606_22983_gb300 import lv
    from oracle.policy import order_global
    rng = np.random.default_rng(11 + within + 2 * tplay)
    S, maxb, T = 64, 24, 16
    pool = _tiny_pool(max_sessions=S, max_blocks=maxb, hbm_pages=1024, hbm_budget_pages=1024,
                      host_pages=1024, within_order=within, t_play_mode=tplay,
                      reply_prior_us=1_500_000, unit_us=40_000)
    try:
        for trial in range(12):
            placement, ctx = _random_placement(rng, S, maxb, T, 1024, 1024)
            pool.import_placement(placement, ctx)
            st = _random_states(rng, S)
            pool.set_sessions(st)
            pool.sync()
            gs = pool.get_sessions()
            osess = _oracle_states(gs)
            tables = placement.astype(np.int64)
            nb = -(-ctx.astype(np.int64) // T)
            now = int(rng.integers(0, 12_000_000))
            for fallback in (False, True):
                want = np.stack(order_global(tables, nb, osess, now, tplay, 1_500_000, 40_000,
                                             within, fallback), axis=1)
                flags = lv.LV_SELECT_FALLBACK if fallback else 0
                got, n = pool.select(now, lv.LV_ALL, flags)
                assert np.array_equal(got.cpu().numpy().astype(np.int64), want), (trial, fallback)
                for k in (0, 1, 7, len(want), len(want) + 3):
                    got, n = pool.select(now, k, flags)
                    assert n == min(k, len(want))
                    assert np.array_equal(got.cpu().numpy().astype(np.int64), want[:n])
        assert pool.sync(raise_on_error=False) == 0
    finally:
        pool.close()


def test_ranker_at_two_to_the_twenty_resident_pages():
    """1024 sessions x 1024 blocks all resident (a metadata-sized page shape):
    the full order and a top-256 match the oracle; reports microseconds per decision."""
    import torch
    from paper_2606_22983_gb300 import lv
    from oracle.policy import order_global
    rng = np.random.default_rng(5)
    S, maxb, T = 1024, 1024, 16
    n = S * maxb
    pool = _tiny_pool(layers=1, kv_heads=1, head_dim=8, max_sessions=S, max_blocks=maxb,
                      hbm_pages=n, hbm_budget_pages=n, host_pages=16)
    try:
        placement = rng.permutation(n).astype(np.int32).reshape(S, maxb)
        ctx = np.full(S, maxb * T, np.int32)
        pool.import_placement(placement, ctx)
        st = _random_states(rng, S)
        st["flags"] &= ~(lv.LV_RUNNING | lv.LV_IMMEDIATE)
        st["protect_until_us"] = 0
        st["gen_us"] = rng.integers(0, 10_000_000, S)          # distinct-ish keys
        st["play_us"] = 0
        pool.set_sessions(st)
        pool.sync()
        osess = _oracle_states(pool.get_sessions())
        want = np.stack(order_global(placement.astype(np.int64), np.full(S, maxb), osess, 0, 0,
                                     3_000_000, 80_000), axis=1)
        assert want.shape[0] == n
        got, cnt = pool.select(0, lv.LV_ALL, 0, capacity=n)
        assert cnt == n and np.array_equal(got.cpu().numpy().astype(np.int64), want)
        out = torch.empty((256, 3), dtype=torch.int32, device="cuda")
        cnt_d = torch.zeros(1, dtype=torch.int64, device="cuda")
        for _ in range(5):
            lv.lv_select_victims(pool.handle, 0, 256, 0, out, 256, cnt_d, pool.stream)
        torch.cuda.synchronize()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record()
        reps = 50
        for _ in range(reps):
            lv.lv_select_victims(pool.handle, 0, 256, 0, out, 256, cnt_d, pool.stream)
        b.record()
        torch.cuda.synchronize()
        us = a.elapsed_time(b) * 1e3 / reps
        assert np.array_equal(out.cpu().numpy().astype(np.int64), want[:256])
        print(f"\nranker, 2^20 resident pages, k=256: {us:.1f} us per decision")
    finally:
        pool.close()


@pytest.mark.parametrize("kernel", ["tma", "lsu"])
def test_pack_unpack_pages(kernel, monkeypatch):
    import torch
    from paper_2606_22983_gb300 import lv
    monkeypatch.setenv("LV_STAGE_KERNEL", kernel)
    pool = _tiny_pool(hbm_pages=300, hbm_budget_pages=300)
    try:
        rng = np.random.default_rng(1)
        kv = rng.integers(0, 256, tuple(pool.kv.shape), dtype=np.uint8)
        pool.kv.copy_(torch.from_numpy(kv))
        pages = rng.permutation(300)[:173].astype(np.int32)
        run = torch.zeros((173, pool.J, pool.P), dtype=torch.uint8, device="cuda")
        lv.lv_pack_pages(pool.handle, pages, 173, run, pool.stream)
        pool.sync()
        want = np.stack([kv[:, p, :] for p in pages])
        assert np.array_equal(run.cpu().numpy(), want)
        # unpack a fresh run into other pages; the rest of the pool is untouched
        src = rng.integers(0, 256, (90, pool.J, pool.P), dtype=np.uint8)
        dst_pages = rng.permutation(300)[:90].astype(np.int32)
        lv.lv_unpack_pages(pool.handle, torch.from_numpy(src).cuda(), torch.from_numpy(dst_pages).cuda(),
                           90, pool.stream)
        pool.sync()
        after = pool.kv.cpu().numpy()
        expect = kv.copy()
        for i, p in enumerate(dst_pages):
            expect[:, p, :] = src[i]
        assert np.array_equal(after, expect)
        # an out-of-range page is reported and skipped, not faulted
        bad = np.array([3, 300, 5], dtype=np.int32)
        lv.lv_pack_pages(pool.handle, bad, 3, run, pool.stream)
        assert pool.sync(raise_on_error=False) == lv.LV_ERR_BOUNDS
        pool.clear_error()
        assert pool.sync(raise_on_error=False) == 0
    finally:
        pool.close()


def test_remap_cancel_and_allocation_errors():
    from paper_2606_22983_gb300 import lv
    pool = _tiny_pool(hbm_pages=64, hbm_budget_pages=10, host_pages=8)
    try:
        placement = np.full((8, 16), -1, np.int32)
        placement[0, :4] = [0, 1, 2, 3]
        placement[1, :2] = [4, -2]                     # block (1, 1) on host slot 0
        ctx = np.zeros(8, np.int32)
        ctx[0], ctx[1] = 64, 32
        pool.import_placement(placement, ctx)
        assert pool.sync(raise_on_error=False) == 0
        st = pool.stats()
        assert st["hbm_allocated"] == 5 and st["host_allocated"] == 1

        def remap(entries):
            e = np.array(entries, dtype=np.int32).reshape(-1, 3)
            pool.remap(e, len(e))
            return pool.sync(raise_on_error=False)

        assert remap([[0, 0, 4]]) == lv.LV_ERR_DOUBLE_MAP     # page 4 is owned by (1, 0)
        pool.clear_error()
        assert remap([[0, 0, 20]]) == lv.LV_ERR_DOUBLE_MAP    # page 20 was never reserved
        pool.clear_error()
        assert remap([[0, 9, 20]]) == lv.LV_ERR_BOUNDS        # block 9 is past the context
        pool.clear_error()
        assert remap([[0, 0, -1]]) == lv.LV_ERR_BOUNDS        # no location
        pool.clear_error()
        # a reservation, committed twice in one call: one is a double map
        pages, _ = pool.swap_in(1, np.array([1], np.int32), 1)
        p = int(pages.cpu()[0])
        assert remap([[1, 1, p], [1, 1, p]]) == lv.LV_ERR_DOUBLE_MAP
        pool.clear_error()
        t, own, _ = pool.tables()
        assert t[1, 1] == p and own[p] == (1 << 16) | 1
        # cancel: an owned page is refused, a pending reservation is released
        pool.cancel(np.array([p], np.int32), 1)
        assert pool.sync(raise_on_error=False) == lv.LV_ERR_STATE
        pool.clear_error()
        v = np.array([[0, 3, 3]], np.int32)
        slots, commit = pool.swap_out(v, 1)
        s0 = int(slots.cpu()[0])
        pool.cancel(np.array([-(s0 + 2)], np.int32), 1)
        assert pool.sync(raise_on_error=False) == 0
        assert pool.stats()["host_allocated"] == 0
        # the budget: 6 pages used of 10, 6 more cannot be reserved and nothing changes
        before = pool.stats()["hbm_allocated"]
        lv.lv_session_append(pool.handle, 2, 6 * 16, pool.pages, None, pool.stream)
        assert pool.sync(raise_on_error=False) == lv.LV_ERR_NO_HBM
        pool.clear_error()
        assert pool.stats()["hbm_allocated"] == before
        assert int(pool.get_sessions()["ctx_tokens"][2]) == 0
        # a stale victim (block 0 does not live on page 3) is refused by swap-out
        pool.swap_out(np.array([[0, 0, 3]], np.int32), 1)
        assert pool.sync(raise_on_error=False) == lv.LV_ERR_STATE
        pool.clear_error()
    finally:
        pool.close()


def _owner_words(owner, used):
    """The oracle's owners as the library's owner words (sid << 16 | blk, reserved, free)."""
    w = np.where(used, -2, -1).astype(np.int64)
    own = owner[:, 0] >= 0
    w[own] = (owner[own, 0] << 16) | owner[own, 1]
    return w.astype(np.int32)


@pytest.mark.parametrize("per_thread", [1, 2, 4])
def test_remap_batch_with_refused_entries(per_thread, monkeypatch):
    """A 32 768-entry commit (every page of a pool to the host tier) in which 600
    entries are refused -- 400 name another block's HBM page as their new location (a
    double map), 200 name a block past its session's context -- at 1, 2 and 4 entries
    per thread.  A refused entry changes nothing (its block stays on its page, its
    reserved slot stays reserved) and every other entry is committed: tables, owner
    words and allocation counts equal the oracle's after it commits the accepted
    entries alone, and the allocation bitmaps agree with it on the next reservations."""
    import torch
    from oracle.pool import OraclePool
    from paper_2606_22983_gb300 import lv
    from paper_2606_22983_gb300.pool import KVPool
    monkeypatch.setenv("LV_REMAP_ENTRIES_PER_THREAD", str(per_thread))
    rng = np.random.default_rng(per_thread)
    S, B = 64, 512
    N = S * B
    pool = KVPool(layers=1, kv_heads=1, head_dim=8, max_sessions=S, max_blocks=B, hbm_pages=N,
                  hbm_budget_pages=N, host_pages=N)
    om = OraclePool(1, 1, 8, 16, 2, S, B, N, N, N, with_bytes=False)
    try:
        placement = rng.permutation(N).astype(np.int32).reshape(S, B)
        ctx = np.full(S, B * 16, np.int32)
        ctx[-1] = (B - 8) * 16          # the last session's last 8 blocks lie past its context
        placement[-1, B - 8:] = -1
        pool.import_placement(placement, ctx)
        om.import_placement(placement, ctx)
        victims, nv = pool.select(0, lv.LV_ALL, 0)
        v = victims.cpu().numpy().astype(np.int64)
        slots, commit = pool.swap_out(victims, nv)
        assert np.array_equal(slots.cpu().numpy(), om.swap_out(v[:, 0], v[:, 1], v[:, 2]))
        reserved = commit.cpu().numpy().copy()
        e = reserved.copy()
        bad = rng.choice(nv, 600, replace=False)
        owned, past = bad[:400], bad[400:]
        good = np.setdiff1d(np.arange(nv), bad)
        e[owned, 2] = v[rng.choice(good, owned.size), 2]
        e[past, 0] = S - 1
        e[past, 1] = B - 1 - rng.integers(0, 8, past.size)
        pool.remap(torch.from_numpy(e).to(pool.device), nv)
        assert pool.sync(raise_on_error=False) in (lv.LV_ERR_DOUBLE_MAP, lv.LV_ERR_BOUNDS)
        pool.clear_error()
        om.remap(e[good, 0], e[good, 1], e[good, 2])
        t, oh, oo = pool.tables()
        assert np.array_equal(t, om.tables.astype(np.int32))
        assert np.array_equal(oh, _owner_words(om.owner_hbm, om.hbm_used))
        assert np.array_equal(oo, _owner_words(om.owner_host, om.host_used))
        st = pool.stats()
        assert st["hbm_allocated"] == int(om.hbm_used.sum()) == 600
        assert st["host_allocated"] == int(om.host_used.sum()) == nv
        # the refused entries' slots are still reservations: releasing them works
        refused_slots = reserved[bad, 2]
        pool.cancel(torch.from_numpy(refused_slots.astype(np.int32)).to(pool.device), bad.size)
        assert pool.sync(raise_on_error=False) == 0
        om.cancel(refused_slots)
        # and the next reservations take the same lowest free slots as the oracle's
        victims2, n2 = pool.select(0, 50, 0)
        v2 = victims2.cpu().numpy().astype(np.int64)
        slots2, _ = pool.swap_out(victims2, n2)
        assert np.array_equal(slots2.cpu().numpy(), om.swap_out(v2[:, 0], v2[:, 1], v2[:, 2]))
        assert pool.sync(raise_on_error=False) == 0
        assert pool.stats()["host_allocated"] == int(om.host_used.sum())
    finally:
        pool.close()


def test_degenerate_sizes_and_host_pointer_arguments():
    import torch
    from paper_2606_22983_gb300 import lv
    pool = _tiny_pool(max_sessions=1, max_blocks=4, hbm_pages=8, hbm_budget_pages=8, host_pages=8)
    try:
        placement = np.full((1, 4), -1, np.int32)
        placement[0, :3] = [5, 6, 7]
        pool.import_placement(placement, np.array([40], np.int32))
        # k = 0, n = 0, empty exchange: no work, no error
        got, n = pool.select(0, 0)
        assert n == 0
        pool.swap_out(np.zeros((0, 3), np.int32), 0)
        lv.lv_swap_exchange(pool.handle, None, 0, 0, None, 0, None, None, 0, pool.stream)
        lv.lv_session_append(pool.handle, 0, 0, None, None, pool.stream)
        assert pool.sync(raise_on_error=False) == 0
        # the same swap-out with host (numpy) and device (torch) arguments
        v_host = np.array([[0, 2, 7], [0, 1, 6]], np.int32)
        slots_h = np.full(2, -9, np.int32)
        commit_h = np.zeros((2, 3), np.int32)
        lv.lv_swap_out(pool.handle, v_host, 2, slots_h, commit_h, 0, pool.stream)
        pool.sync()
        assert slots_h.tolist() == [0, 1]
        assert commit_h.tolist() == [[0, 2, -2], [0, 1, -3]]
        pool.cancel(np.array([-2, -3], np.int32), 2)
        v_dev = torch.from_numpy(v_host).cuda()
        slots_d = torch.full((2,), -9, dtype=torch.int32, device="cuda")
        commit_d = torch.zeros((2, 3), dtype=torch.int32, device="cuda")
        lv.lv_swap_out(pool.handle, v_dev, 2, slots_d, commit_d, 0, pool.stream)
        pool.sync()
        assert slots_d.cpu().tolist() == [0, 1]
        assert np.array_equal(commit_d.cpu().numpy(), commit_h)
        assert np.array_equal(pool.host[0], pool.kv[:, 7].cpu().numpy())
        # page-locked host arguments are used in place: the commit's entries are read and
        # a victim list is written over the host link, in stream order
        commit_p = torch.from_numpy(commit_h).pin_memory()
        pool.remap(commit_p, 2)
        cnt_p = torch.full((1,), -7, dtype=torch.int64).pin_memory()
        out_p = torch.full((4, 3), -7, dtype=torch.int32).pin_memory()
        lv.lv_select_victims(pool.handle, 0, lv.LV_ALL, 0, out_p, 4, cnt_p, pool.stream)
        assert pool.sync(raise_on_error=False) == 0
        t, _, _ = pool.tables()
        assert t[0, :3].tolist() == [5, -3, -2]
        assert int(cnt_p[0]) == 1
        assert out_p[0].tolist() == [0, 0, 5] and out_p[1].tolist() == [-7, -7, -7]
    finally:
        pool.close()


def test_largest_pool_shape_and_ids():
    """The largest shape the descriptor allows: 4096 sessions x 65536 blocks per
    session.  Session 4095 holds a full 65536-block table (its top 1536 blocks in HBM,
    the rest on the host), so its owner words carry the largest session and block ids.
    The full victim order matches the oracle; evicting the top 1536 blocks fills the
    host tier to its last slot; the tables, owners and bytes follow, and the highest
    block comes back."""
    import torch
    from paper_2606_22983_gb300 import lv
    from oracle.policy import order_global
    S, maxb, T, hbm, host = 4096, 65536, 16, 2048, 65536
    rng = np.random.default_rng(23)
    pool = _tiny_pool(layers=1, kv_heads=1, head_dim=8, max_sessions=S, max_blocks=maxb,
                      hbm_pages=hbm, hbm_budget_pages=hbm, host_pages=host)
    try:
        g = torch.Generator().manual_seed(23)
        pool.kv.copy_(torch.randint(0, 256, tuple(pool.kv.shape), generator=g, dtype=torch.uint8))
        kv0 = pool.kv.cpu().numpy()
        pages = rng.permutation(hbm).astype(np.int32)
        placement = np.full((S, maxb), -1, np.int32)
        ctx = np.zeros(S, np.int32)
        top, n_top = S - 1, 1536
        ctx[top] = maxb * T
        placement[top, :maxb - n_top] = -(np.arange(maxb - n_top, dtype=np.int32) + 2)
        placement[top, maxb - n_top:] = pages[:n_top]
        ctx[0], ctx[2047] = 70, 100 * T
        placement[0, :5] = pages[n_top:n_top + 5]
        placement[2047, :100] = pages[n_top + 5:n_top + 105]
        pool.import_placement(placement, ctx)
        st = np.zeros(S, dtype=lv.SESSION_DTYPE)
        st["reply_n"] = 1
        st["reply_ema_us"] = 1_000_000
        st["reply_ema_us"][top], st["reply_ema_us"][0], st["reply_ema_us"][2047] = 9e6, 5e6, 2e6
        pool.set_sessions(st)
        pool.sync()
        osess = _oracle_states(pool.get_sessions())
        nb = -(-ctx.astype(np.int64) // T)
        want = np.stack(order_global(placement, nb, osess, 0, 0, 3_000_000, 80_000), axis=1)
        assert want.shape[0] == n_top + 105
        got, n = pool.select(0, lv.LV_ALL, 0, capacity=len(want))
        assert n == len(want) and np.array_equal(got.cpu().numpy().astype(np.int64), want)
        # evict the top 1536: blocks 65535 .. 64000 of session 4095 into slots 64000 ..
        v, n = pool.select(0, n_top)
        assert n == n_top and np.array_equal(v.cpu().numpy().astype(np.int64), want[:n_top])
        slots, commit = pool.swap_out(v, n)
        pool.remap(commit, n)
        pool.sync()
        blk = np.arange(maxb - 1, maxb - 1 - n_top, -1)
        want_slots = np.arange(maxb - n_top, maxb)
        assert np.array_equal(slots.cpu().numpy(), want_slots)
        tables, own_hbm, own_host = pool.tables()
        assert np.array_equal(tables[top, blk], -(want_slots + 2))
        assert np.array_equal(own_host[want_slots].astype(np.int64), (top << 16) | blk)
        assert own_host[want_slots[0]] == (4095 << 16) | 65535
        assert np.all(own_host[:maxb - n_top] == ((top << 16) | np.arange(maxb - n_top)))
        assert np.all(own_hbm[pages[:n_top]] == -1)
        host_img = pool.host.reshape(host, pool.J, pool.P)
        for i in (0, 1, 700, n_top - 1):
            assert np.array_equal(host_img[want_slots[i]], kv0[:, pages[n_top - 1 - i]])
        assert pool.stats()["host_allocated"] == host
        # the highest block comes back into the lowest free HBM page
        free = np.sort(pages[:n_top])
        pg, commit = pool.swap_in(top, torch.tensor([maxb - 1], dtype=torch.int32,
                                                    device="cuda"), 1)
        pool.remap(commit, 1)
        pool.sync()
        assert int(pg[0]) == free[0]
        assert np.array_equal(pool.kv[:, free[0]].cpu().numpy(), kv0[:, pages[n_top - 1]])
        tables, own_hbm, own_host = pool.tables()
        assert tables[top, maxb - 1] == free[0] and own_hbm[free[0]] == (4095 << 16) | 65535
        assert own_host[maxb - n_top] == -1
        assert pool.sync(raise_on_error=False) == 0
    finally:
        pool.close()


def test_turn_picks_the_first_candidate_with_host_blocks():
    """lv_turn with sid = -1: the first listed session that has a block in the host
    tier (else the first listed), then turn begin, make resident, turn end -- the
    same state as the separate calls."""
    import torch
    from paper_2606_22983_gb300 import lv
    S, B, T = 8, 16, 16
    placement = np.full((S, B), -1, np.int32)
    ctx = np.zeros(S, np.int32)
    # sessions 1 and 3: 4 blocks in HBM; session 5: 3 blocks on the host; session 6: 2 + 2
    nxt = 0
    for s, (n_hbm, n_host) in {1: (4, 0), 3: (4, 0), 5: (0, 3), 6: (2, 2)}.items():
        for b in range(n_hbm + n_host):
            placement[s, b] = nxt if b < n_hbm else -(s * 4 + b + 2)
            nxt += b < n_hbm
        ctx[s] = (n_hbm + n_host) * T
    results = []
    for how in ("turn", "calls"):
        pool = _tiny_pool(max_sessions=S, max_blocks=B, hbm_pages=64, hbm_budget_pages=64, host_pages=64)
        try:
            pool.import_placement(placement, ctx)
            res = np.zeros(1, dtype=lv.RESIDENT_DTYPE)
            if how == "turn":
                cand = torch.tensor([3, 1, 6, 5], dtype=torch.int32, device=pool.device)
                lv.lv_turn(pool.handle, -1, 7_000_000, 20, 4_000_000, 50, result_out=res,
                           candidates=cand, num_candidates=4, stream=pool.stream)
            else:
                ev = np.zeros(1, dtype=lv.EVENT_DTYPE)
                ev["kind"], ev["sid"], ev["t_us"] = lv.LV_EV_TURN_BEGIN, 6, 7_000_000
                pool.events(ev)
                lv.lv_make_resident(pool.handle, 6, 7_000_000, 20, 0, -1, None, None, None, None,
                                    None, res, pool.stream)
                ev["kind"], ev["a"], ev["b"] = lv.LV_EV_TURN_END, 4_000_000, 50
                pool.events(ev)
            assert pool.sync(raise_on_error=False) == 0
            r = res[0]
            assert int(r["sid"]) == 6 and int(r["status"]) == lv.LV_RESIDENT_DONE
            assert int(r["n_loaded"]) == 2 and int(r["n_appended"]) == 2
            results.append((pool.tables(), pool.get_sessions().copy(), pool.stats()))
        finally:
            pool.close()
    (ta, sa, xa), (tb, sb, xb) = results
    for a, b in zip(ta, tb):
        assert np.array_equal(a, b)
    assert np.array_equal(sa, sb)
    assert sa[6]["gen_us"] == 4_000_000 and not (sa[6]["flags"] & lv.LV_RUNNING)
    for k in ("hbm_allocated", "host_allocated", "pages_in", "appended_pages", "events"):
        assert xa[k] == xb[k], k


def test_turn_pick_fallback_and_bad_candidate():
    import torch
    from paper_2606_22983_gb300 import lv
    pool = _tiny_pool()
    try:
        placement = np.full((8, 16), -1, np.int32)
        placement[2, :2] = [0, 1]
        pool.import_placement(placement, np.array([0, 0, 32, 0, 0, 0, 0, 0], np.int32))
        res = np.zeros(1, dtype=lv.RESIDENT_DTYPE)
        cand = torch.tensor([4, 2], dtype=torch.int32, device=pool.device)
        lv.lv_turn(pool.handle, -1, 1_000, 0, 0, 0, result_out=res, candidates=cand,
                   num_candidates=2, stream=pool.stream)
        assert pool.sync(raise_on_error=False) == 0
        assert int(res[0]["sid"]) == 4 and int(res[0]["n_loaded"]) == 0   # nobody offloaded
        bad = torch.tensor([8 + 3], dtype=torch.int32, device=pool.device)
        lv.lv_turn(pool.handle, -1, 2_000, 16, 0, 0, result_out=res, candidates=bad,
                   num_candidates=1, stream=pool.stream)
        assert pool.sync(raise_on_error=False) == lv.LV_ERR_BOUNDS
        assert int(res[0]["status"]) == lv.LV_RESIDENT_FAILED and int(res[0]["sid"]) == -1
        assert pool.stats()["appended_pages"] == 0
        pool.clear_error()
        with pytest.raises(lv.LvError):
            lv.lv_turn(pool.handle, -1, 3_000, 0, 0, 0, candidates=None, num_candidates=0,
                       stream=pool.stream)
    finally:
        pool.close()


@pytest.mark.parametrize("shape", [(2, 2, 64), (48, 4, 128)])
def test_page_checksums_match_the_oracle(shape):
    """lv_page_checksums against the oracle's definition on the same bytes: every
    page of a randomly filled pool (tiny and thinker-shaped sub-pages), host and
    device argument buffers, and a page id outside the pool."""
    import torch
    from oracle.pool import OraclePool
    from paper_2606_22983_gb300 import lv
    L, H, D = shape
    pages = 64 if L == 2 else 24
    pool = _tiny_pool(layers=L, kv_heads=H, head_dim=D, hbm_pages=pages, hbm_budget_pages=pages,
                      host_pages=4)
    try:
        g = torch.Generator(device=pool.device).manual_seed(5)
        pool.kv.copy_(torch.randint(0, 256, pool.kv.shape, generator=g, device=pool.device,
                                    dtype=torch.int32).to(torch.uint8))
        om = OraclePool(L, H, D, 16, 2, n_sessions=1, max_blocks=1, hbm_pages=pages,
                        hbm_budget_pages=pages, host_pages=0)
        om.hbm[:] = pool.kv.cpu().numpy()
        want = np.array([om.page_checksum(q) for q in range(pages)], dtype=np.uint64)
        order = np.random.default_rng(0).permutation(pages).astype(np.int32)
        got_h = np.zeros(pages, np.uint64)
        lv.lv_page_checksums(pool.handle, order, pages, got_h, pool.stream)
        assert pool.sync(raise_on_error=False) == 0
        assert np.array_equal(got_h, want[order])
        got_d = torch.zeros(pages, dtype=torch.int64, device=pool.device)
        lv.lv_page_checksums(pool.handle, torch.from_numpy(order).to(pool.device), pages, got_d,
                             pool.stream)
        assert np.array_equal(got_d.cpu().numpy().view(np.uint64), want[order])
        bad = np.array([1, pages + 7], np.int32)
        sums = np.ones(2, np.uint64)
        lv.lv_page_checksums(pool.handle, bad, 2, sums, pool.stream)
        assert pool.sync(raise_on_error=False) == lv.LV_ERR_BOUNDS
        assert sums[0] == want[1] and sums[1] == 0
    finally:
        pool.close()


def test_async_copy_is_joined_by_the_next_reader():
    """lv_make_resident with LV_RESIDENT_ASYNC_COPY moves 96 thinker pages on the
    pool's copy stream; lv_page_checksums queued right after it on the same stream,
    with no host wait, must see every moved byte (it joins the copies first)."""
    import torch
    from oracle.pool import OraclePool
    from paper_2606_22983_gb300 import lv
    n = 96
    pool = _tiny_pool(layers=48, kv_heads=4, head_dim=128, max_sessions=2, max_blocks=128,
                      hbm_pages=256, hbm_budget_pages=256, host_pages=128)
    try:
        placement = np.full((2, 128), -1, np.int32)
        placement[0, :n] = -(np.arange(n, dtype=np.int32) + 2)         # session 0 on the host
        pool.import_placement(placement, np.array([n * 16, 0], np.int32))
        g = torch.Generator(device=pool.device).manual_seed(9)
        pool.host_dev[:n].copy_(torch.randint(0, 256, pool.host_dev[:n].shape, generator=g,
                                              device=pool.device, dtype=torch.int32).to(torch.uint8))
        torch.cuda.synchronize()
        om = OraclePool(48, 4, 128, 16, 2, n_sessions=1, max_blocks=1, hbm_pages=1,
                        hbm_budget_pages=1, host_pages=0)
        want = []
        for h in range(n):
            om.hbm[:, 0, :] = pool.host[h]
            want.append(om.page_checksum(0))
        blocks = torch.empty(128, dtype=torch.int32, device=pool.device)
        pages = torch.empty(128, dtype=torch.int32, device=pool.device)
        sums = torch.zeros(n, dtype=torch.int64, device=pool.device)
        res = torch.zeros(lv.RESIDENT_DTYPE.itemsize, dtype=torch.uint8).pin_memory()
        lv.lv_make_resident(pool.handle, 0, 1_000, 0, lv.LV_RESIDENT_ASYNC_COPY, -1, None, None,
                            blocks, pages, None, res, pool.stream)
        lv.lv_page_checksums(pool.handle, pages, n, sums, pool.stream)
        assert pool.sync(raise_on_error=False) == 0
        r = res.numpy().view(lv.RESIDENT_DTYPE)[0]
        assert int(r["n_loaded"]) == n and int(r["status"]) == lv.LV_RESIDENT_DONE
        assert np.array_equal(blocks[:n].cpu().numpy(), np.arange(n))
        assert np.array_equal(sums.cpu().numpy().view(np.uint64), np.array(want, np.uint64))
    finally:
        pool.close()


def test_large_subpages_fall_back_to_plain_copies():
    """Sub-pages too large for two TMA stages (32 KV heads x 128, 16 tokens, bf16 =
    128 KiB) are packed and staged with 16-byte copies: a round trip through the
    staged swap path returns every byte."""
    import torch
    from paper_2606_22983_gb300 import lv
    pool = _tiny_pool(layers=1, kv_heads=32, head_dim=128, max_sessions=2, max_blocks=8,
                      hbm_pages=8, hbm_budget_pages=8, host_pages=8)
    try:
        placement = np.full((2, 8), -1, np.int32)
        placement[0, :4] = [0, 1, 2, 3]
        pool.import_placement(placement, np.array([64, 0], np.int32))
        g = torch.Generator(device=pool.device).manual_seed(3)
        pool.kv.copy_(torch.randint(0, 256, pool.kv.shape, generator=g, device=pool.device,
                                    dtype=torch.int32).to(torch.uint8))
        before = pool.kv[:, :4, :].clone()
        victims, n = pool.select(0, 4)
        slots, commit = pool.swap_out(victims, n, lv.LV_MODE_STAGED)
        pool.remap(commit, n)
        assert pool.sync(raise_on_error=False) == 0
        blks, nb = pool.blocks(0, 1)
        pool.kv[:, :4, :].zero_()
        pages, commit = pool.swap_in(0, blks, nb, lv.LV_MODE_STAGED)
        pool.remap(commit, nb)
        assert pool.sync(raise_on_error=False) == 0
        t, _, _ = pool.tables()
        for b in range(4):
            assert torch.equal(pool.kv[:, int(t[0, b]), :], before[:, b, :])
    finally:
        pool.close()


@pytest.mark.parametrize("S", [1025, 1500, 4096])
def test_ranker_beyond_a_thousand_sessions(S):
    """More sessions than the sort kernel's threads (up to the 4096 maximum): the
    shared-memory sorting network, against the oracle's full order."""
    from paper_2606_22983_gb300 import lv
    from oracle.policy import order_global
    rng = np.random.default_rng(S)
    maxb, T = 4, 16
    pages = S * maxb
    pool = _tiny_pool(max_sessions=S, max_blocks=maxb, hbm_pages=pages, hbm_budget_pages=pages,
                      host_pages=pages)
    try:
        placement, ctx = _random_placement(rng, S, maxb, T, pages, pages)
        pool.import_placement(placement, ctx)
        st = _random_states(rng, S)
        pool.set_sessions(st)
        pool.sync()
        osess = _oracle_states(pool.get_sessions())
        nb = -(-ctx.astype(np.int64) // T)
        now = int(rng.integers(0, 12_000_000))
        for fallback in (False, True):
            want = np.stack(order_global(placement.astype(np.int64), nb, osess, now, 0, 3_000_000,
                                         80_000, 0, fallback), axis=1)
            got, n = pool.select(now, lv.LV_ALL, lv.LV_SELECT_FALLBACK if fallback else 0)
            assert np.array_equal(got.cpu().numpy().astype(np.int64), want), fallback
            got, n = pool.select(now, 100, lv.LV_SELECT_FALLBACK if fallback else 0)
            assert np.array_equal(got.cpu().numpy().astype(np.int64), want[:100]), fallback
        assert pool.sync(raise_on_error=False) == 0
    finally:
        pool.close()
