"""lv_select_victims_noalloc: the ranker for callers that cannot allocate.

Some callers of this library must not allocate GPU memory while they rank victims:
an engine that gave almost all free HBM to its KV pages (one more cudaMalloc may
fail or fragment that reservation), or a scheduler thread that cannot take the
device synchronisation an allocation may cause.  This entry point keeps its working
memory in a fixed array compiled into liblv.  The tests check that it returns what
the pool's own ranker returns, on two calls in a row; that it matches the oracle's
victim order element by element at the compiled-in maximum of 4096 sessions, under
both policies; that warmed-up calls leave the device's free memory unchanged; and
that it takes mapped page-locked host outputs and refuses pageable host memory.

The file sorts last so that a run stopping at the first failure has run every
other test first.
"""
import numpy as np
import pytest

pytestmark = pytest.mark.gpu


def _prm(lv, S, B, T, **kw):
    d = dict(num_sessions=S, max_blocks=B, page_tokens=T, within_order=0, t_play_mode=0,
             flags=0, reply_prior_us=3_000_000, unit_us=80_000, policy=0, reserved=0)
    d.update(kw)
    return lv.lv_rank_params(**d)


@pytest.mark.parametrize("policy", [0, 1])
def test_noalloc_ranker_matches_pool_ranker_on_two_calls(policy):
    import torch
    from paper_2606_22983_gb300 import build
    build()
    from paper_2606_22983_gb300 import lv
    from paper_2606_22983_gb300.harness import pool_for
    from paper_2606_22983_gb300.manager import KVManager
    from workloads import make_workload, pool_spec

    wl = make_workload("tiny", 5, spec=pool_spec("tiny").with_(policy=policy))
    pool = pool_for(wl)
    try:
        gm = KVManager(pool, perms=wl.perms, record=False)
        for i in range(300):                      # sessions in varied states, some on the host
            gm.step(wl.event(i), i)
        S, B = pool.S, pool.max_blocks
        sess = torch.empty(S * lv.SESSION_DTYPE.itemsize, dtype=torch.uint8, device="cuda")
        lv.lv_session_get(pool.handle, sess, 0, S, pool.stream)
        tables = torch.from_numpy(pool.tables()[0]).cuda()
        prm = _prm(lv, S, B, pool.T, within_order=wl.spec.within_order,
                   t_play_mode=wl.spec.t_play_mode, reply_prior_us=wl.spec.reply_prior_us,
                   unit_us=wl.spec.unit_us, policy=policy)
        cap = pool.budget
        now = int(wl.t_us[299])
        calls = [(now, lv.LV_ALL, 0), (now + 1_500_000, 37, lv.LV_SELECT_FALLBACK)]
        for now_us, k, flags in calls:
            want, n_want = pool.select(now_us, k, flags)
            want = want.cpu().numpy()
            prm.flags = flags
            out = torch.full((cap, 3), -7, dtype=torch.int32, device="cuda")
            cnt = torch.full((1,), -1, dtype=torch.int64, device="cuda")
            lv.lv_select_victims_noalloc(prm, sess, tables, now_us, k, out, cap, cnt, pool.stream)
            torch.cuda.synchronize()
            n = int(cnt.item())
            assert n == n_want and n > 0
            assert np.array_equal(out[:n].cpu().numpy(), want)
        # sizes beyond the compiled-in maximum are refused, not run
        prm.num_sessions = lv.LV_NOALLOC_MAX_SESSIONS + 1
        with pytest.raises(lv.LvError) as e:
            lv.lv_select_victims_noalloc(prm, sess, tables, now, 1, out, cap, cnt, pool.stream)
        assert e.value.status == lv.LV_ERR_INVALID
        assert pool.sync(raise_on_error=False) == 0
    finally:
        torch.cuda.synchronize()
        pool.close()


def _random_state(seed, S, B, T):
    """S sessions with random interaction states and block tables: resident pages
    (distinct), host-tier entries and unplaced blocks past each context."""
    from oracle import sessions as se
    rng = np.random.default_rng(seed)
    ctx = rng.integers(0, B * T + 1, S).astype(np.int32)
    nb = -(-ctx // T)
    tables = np.full((S, B), -1, np.int32)
    pages = rng.permutation(S * B).astype(np.int32)
    for s in range(S):
        n = int(nb[s])
        host = rng.random(n) < 0.3
        row = pages[s * B:s * B + n].copy()
        row[host] = -(rng.integers(0, 1 << 20, int(host.sum())) + 2)
        tables[s, :n] = row
    st = np.zeros(S, dtype=[("ctx_tokens", "<i4"), ("flags", "<i4"), ("gen_us", "<i8"),
                            ("play_us", "<i8"), ("t_done_us", "<i8"), ("reply_ema_us", "<i8"),
                            ("reply_n", "<i4"), ("pad", "<i4"), ("reply_tokens", "<i8"),
                            ("protect_until_us", "<i8"), ("last_use_us", "<i8")])
    st["ctx_tokens"] = ctx
    r = rng.random(S)
    st["flags"] = np.where(r < 0.1, se.RUNNING, np.where(r < 0.2, se.IMMEDIATE, 0)) | \
        np.where(rng.random(S) < 0.5, se.RESP_OPEN, 0)
    st["gen_us"] = rng.integers(0, 30_000_000, S)
    st["play_us"] = rng.integers(0, 30_000_000, S)
    st["reply_n"] = rng.integers(0, 3, S)
    st["reply_ema_us"] = rng.integers(0, 9_000_000, S)
    st["reply_tokens"] = rng.integers(0, 400, S)
    st["protect_until_us"] = np.where(rng.random(S) < 0.15, 5_000_000, 0)
    st["last_use_us"] = rng.integers(0, 1 << 31, S)
    states = [se.SessionState(ctx_tokens=int(x["ctx_tokens"]), flags=int(x["flags"]),
                              gen_us=int(x["gen_us"]), play_us=int(x["play_us"]),
                              reply_ema_us=int(x["reply_ema_us"]), reply_n=int(x["reply_n"]),
                              reply_tokens=int(x["reply_tokens"]),
                              protect_until_us=int(x["protect_until_us"]),
                              last_use_us=int(x["last_use_us"])) for x in st]
    return tables, nb.astype(np.int64), st, states


@pytest.mark.parametrize("policy,within,mode,fallback", [(0, 0, 0, False), (0, 1, 1, True),
                                                         (1, 0, 0, False)])
def test_noalloc_at_the_maximum_session_count_matches_the_oracle(policy, within, mode, fallback):
    """4096 sessions (the compiled-in maximum) x 64 blocks: the whole victim order,
    element by element, against the oracle's global sort."""
    import torch
    from paper_2606_22983_gb300 import build
    build()
    from paper_2606_22983_gb300 import lv
    from oracle.policy import order_global, order_lru

    S, B, T = lv.LV_NOALLOC_MAX_SESSIONS, 64, 16
    tables, nb, st, states = _random_state(7 + policy + within, S, B, T)
    assert st.dtype == lv.SESSION_DTYPE
    now = 2_000_000
    if policy == 1:
        want = order_lru(tables, nb, states, within)
    else:
        want = order_global(tables, nb, states, now, mode, 3_000_000, 80_000, within, fallback)
    want = np.stack([np.asarray(w, np.int64) for w in want], axis=1).astype(np.int32)
    assert len(want) > 10_000
    dev = torch.device("cuda")
    sess = torch.from_numpy(st.view(np.uint8).copy()).to(dev)
    tab = torch.from_numpy(tables).to(dev)
    prm = _prm(lv, S, B, T, within_order=within, t_play_mode=mode, policy=policy,
               flags=lv.LV_SELECT_FALLBACK if fallback else 0)
    cap = S * B
    for k in (lv.LV_ALL, 1000):
        out = torch.full((cap, 3), -7, dtype=torch.int32, device=dev)
        cnt = torch.full((1,), -1, dtype=torch.int64, device=dev)
        lv.lv_select_victims_noalloc(prm, sess, tab, now, k, out, cap, cnt, None)
        torch.cuda.synchronize()
        n = int(cnt.item())
        m = min(len(want), cap if k == lv.LV_ALL else k)
        assert n == m
        assert np.array_equal(out[:n].cpu().numpy(), want[:m])
        assert (out[n:n + 16].cpu().numpy() == -7).all()


def test_noalloc_calls_allocate_nothing_and_take_mapped_host_outputs():
    """After one warm-up call (which may load liblv's kernels), further calls leave the
    device's free memory and torch's reservations unchanged; outputs in page-locked
    (mapped) host memory give the same victims; pageable host memory is refused."""
    import torch
    from paper_2606_22983_gb300 import build
    build()
    from paper_2606_22983_gb300 import lv

    S, B, T = 512, 64, 16
    tables, nb, st, _ = _random_state(3, S, B, T)
    dev = torch.device("cuda")
    sess = torch.from_numpy(st.view(np.uint8).copy()).to(dev)
    tab = torch.from_numpy(tables).to(dev)
    prm = _prm(lv, S, B, T)
    cap = S * B
    out = torch.full((cap, 3), -7, dtype=torch.int32, device=dev)
    cnt = torch.zeros(1, dtype=torch.int64, device=dev)
    lv.lv_select_victims_noalloc(prm, sess, tab, 0, lv.LV_ALL, out, cap, cnt, None)   # warm-up
    torch.cuda.synchronize()
    want = out[:int(cnt.item())].cpu().numpy().copy()
    out_h = torch.full((cap, 3), -7, dtype=torch.int32, pin_memory=True)
    cnt_h = torch.zeros(1, dtype=torch.int64, pin_memory=True)
    torch.cuda.synchronize()
    free0, _ = torch.cuda.mem_get_info()
    res0 = torch.cuda.memory_reserved()
    for i in range(20):
        lv.lv_select_victims_noalloc(prm, sess, tab, 0, lv.LV_ALL, out, cap, cnt, None)
        lv.lv_select_victims_noalloc(prm, sess, tab, 0, lv.LV_ALL, out_h, cap, cnt_h, None)
    torch.cuda.synchronize()
    free1, _ = torch.cuda.mem_get_info()
    assert free1 == free0 and torch.cuda.memory_reserved() == res0
    n = int(cnt_h.item())
    assert n == len(want) and np.array_equal(out_h[:n].numpy(), want)
    assert np.array_equal(out[:n].cpu().numpy(), want)
    # pageable host memory cannot be staged without an allocation: refused, nothing runs
    pageable = np.full((cap, 3), -7, np.int32)
    with pytest.raises(lv.LvError) as e:
        lv.lv_select_victims_noalloc(prm, sess, tab, 0, lv.LV_ALL, pageable, cap, cnt, None)
    assert e.value.status == lv.LV_ERR_INVALID
    torch.cuda.synchronize()
    assert (pageable == -7).all()
    # an unknown policy or a non-zero reserved field is refused too
    for bad in (dict(policy=2), dict(reserved=1)):
        with pytest.raises(lv.LvError) as e:
            lv.lv_select_victims_noalloc(_prm(lv, S, B, T, **bad), sess, tab, 0, 1, out, cap, cnt, None)
        assert e.value.status == lv.LV_ERR_INVALID
