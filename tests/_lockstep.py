"""Runs a workload through the oracle and through liblv side by side and
compares everything each event decides, bit for bit."""
from __future__ import annotations

import numpy as np
import torch

from oracle import OracleManager
from paper_2606_22983_gb300 import lv
from paper_2606_22983_gb300.harness import ContentWriter, pool_for, zero_host
from paper_2606_22983_gb300.manager import KVManager
from workloads import scatter_order, value_table

REC_KEYS = ("sid", "k", "victims", "slots", "in_blocks", "in_pages", "append_pages", "order", "preload")
SESSION_FIELDS = ("ctx_tokens", "flags", "gen_us", "play_us", "t_done_us", "reply_ema_us",
                  "reply_n", "reply_tokens", "protect_until_us", "last_use_us")


def compare_records(ro, rg, where):
    for key in REC_KEYS:
        a, b = ro.get(key), rg.get(key)
        if a is None and b is None:
            continue
        assert a is not None and b is not None, (where, key, a, b)
        if isinstance(a, (int, str)) or isinstance(b, (int, str)):
            assert a == b, (where, key, a, b)
            continue
        a = np.asarray(a, np.int64)
        b = np.asarray(b, np.int64)
        assert a.shape == b.shape and np.array_equal(a, b), (where, key, a, b)


def owners_encoded(owner_pairs, used):
    """The C ABI's owner words: sid << 16 | blk when owned, -2 when reserved by a
    swap and not yet committed, -1 when free."""
    sid, blk = owner_pairs[:, 0], owner_pairs[:, 1]
    return np.where(sid >= 0, (sid << 16) | blk, np.where(used, -2, -1)).astype(np.int32)


def compare_state(om: OracleManager, pool, where, with_bytes):
    tables, own_hbm, own_host = pool.tables()
    assert np.array_equal(om.pool.tables.astype(np.int32), tables), where
    assert np.array_equal(owners_encoded(om.pool.owner_hbm, om.pool.hbm_used), own_hbm), where
    assert np.array_equal(owners_encoded(om.pool.owner_host, om.pool.host_used), own_host), where
    st = pool.stats()
    assert st["error"] == 0, (where, st)
    assert st["hbm_allocated"] == int(om.pool.hbm_used.sum()), where
    assert st["host_allocated"] == int(om.pool.host_used.sum()), where
    assert st["clean_copies"] == om.pool.clean_copies(), where
    assert st["clean_out"] == om.pool.clean_out, where
    assert st["clean_dropped"] == om.pool.clean_dropped, where
    gs = pool.get_sessions()
    oa = om.session_arrays()
    for f in SESSION_FIELDS:
        assert np.array_equal(gs[f].astype(np.int64), oa[f]), (where, f)
    if with_bytes:
        hbm = pool.kv.cpu().numpy()
        assert np.array_equal(hbm, om.pool.hbm), (where, "hbm bytes", _first_difference(hbm, om.pool.hbm))
        assert np.array_equal(pool.host, om.pool.host), (where, "host bytes",
                                                         _first_difference(pool.host, om.pool.host))


def _first_difference(got, want):
    """Where two byte images first differ, with both 16-byte chunks decoded as
    address tags (meaningful when the contents are address-tagged)."""
    from workloads.content import decode_tag
    g, w = np.ascontiguousarray(got).reshape(-1), np.ascontiguousarray(want).reshape(-1)
    bad = np.nonzero(g != w)[0]
    if not bad.size:
        return None
    at = int(bad[0]) // 16 * 16
    return {"byte": int(bad[0]), "got (sid, token, layer, kv, chunk)": decode_tag(g[at:at + 16]),
            "want": decode_tag(w[at:at + 16])}


def make_pair(workload, with_bytes, rank_on="all", mode=lv.LV_MODE_AUTO, driver="device",
              tagged=False):
    seed = workload.seed
    content = None
    if with_bytes:
        content = "tagged" if tagged else (seed, value_table(seed))
    om = OracleManager(workload, with_bytes=with_bytes, content=content, rank_on=rank_on)
    pool = pool_for(workload)
    writer = None
    if with_bytes:
        writer = ContentWriter(pool, workload, tagged=tagged)
        zero_host(pool)
        writer.write_initial(workload)
    gm = KVManager(pool, perms=workload.perms,
                   on_append=writer.write_appended if writer else None,
                   rank_on=rank_on, mode=mode, driver=driver, order_fn=scatter_order)
    return om, pool, gm


def run_lockstep(workload, with_bytes=True, check_every=50, n_events=None, rank_on="all",
                 mode=lv.LV_MODE_AUTO, driver="device", tagged=False):
    om, pool, gm = make_pair(workload, with_bytes, rank_on, mode, driver, tagged)
    n = workload.n_events if n_events is None else n_events
    try:
        compare_state(om, pool, "initial", with_bytes)
        for i in range(n):
            ev = workload.event(i)
            ro = om.step(i)
            rg = gm.step(ev, i)
            compare_records(ro, rg, (i, ev))
            if check_every and (i % check_every == check_every - 1 or i == n - 1):
                compare_state(om, pool, (i, ev), with_bytes)
        return om, gm
    finally:
        torch.cuda.synchronize()
        pool.close()
