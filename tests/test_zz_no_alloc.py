"""lv_select_victims_noalloc against lv_select_victims.

The no-allocation ranker serves callers that must not allocate GPU memory while
they rank (an engine that gave almost all free HBM to its KV pages, or a
scheduler thread that cannot afford the device synchronisation an allocation
may cause).  It must return exactly what the pool's ranker returns: here both
rank the same sessions and block tables, on two calls in a row, and the
victim lists and counts must be equal bit for bit.
"""
import numpy as np
import pytest

pytestmark = pytest.mark.gpu


def test_noalloc_ranker_matches_pool_ranker_on_two_calls():
    import torch
    from paper_2606_22983_gb300 import build
    build()
    from paper_2606_22983_gb300 import lv
    from paper_2606_22983_gb300.harness import pool_for
    from paper_2606_22983_gb300.manager import KVManager
    from workloads import make_workload

    wl = make_workload("tiny", 5)
    pool = pool_for(wl)
    try:
        gm = KVManager(pool, perms=wl.perms, record=False)
        for i in range(300):                      # sessions in varied states, some on the host
            gm.step(wl.event(i), i)
        S, B = pool.S, pool.max_blocks
        sess = torch.empty(S * lv.SESSION_DTYPE.itemsize, dtype=torch.uint8, device="cuda")
        lv.lv_session_get(pool.handle, sess, 0, S, pool.stream)
        tables = torch.from_numpy(pool.tables()[0]).cuda()
        prm = lv.lv_rank_params(num_sessions=S, max_blocks=B, page_tokens=pool.T,
                                within_order=wl.spec.within_order, t_play_mode=wl.spec.t_play_mode,
                                flags=0, reply_prior_us=wl.spec.reply_prior_us,
                                unit_us=wl.spec.unit_us)
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
