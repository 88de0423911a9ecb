"""Randomized differential test of the C ABI against the oracle: random sequences of
ranking, swap-out, swap-in, commit, cancel, exchange, growth, monitor events, whole
device-driven turns (lv_turn, most with their copies left running on the pool's copy
stream) and device-driven evictions (lv_evict) on a tiny pool with random bytes, plus single-item calls that must be refused
with the right status and change nothing.  After a random half of the calls (so that a
turn's copies are often still in flight when the next call starts, and that call must
join them), and after the last one, the block and owner tables, allocation counts,
clean copies, session states and both byte images are compared."""
import numpy as np
import pytest

pytestmark = pytest.mark.gpu

S, B, T = 6, 24, 16          # sessions, blocks per session, tokens per page
HBM, BUDGET, HOST = 96, 80, 160


def _setup(seed, tiers):
    import torch
    from oracle import sessions as se
    from oracle.pool import OraclePool
    from paper_2606_22983_gb300 import lv
    from paper_2606_22983_gb300.pool import KVPool
    rng = np.random.default_rng(seed)
    pool = KVPool(layers=1, kv_heads=1, head_dim=64, max_sessions=S, max_blocks=B, hbm_pages=HBM,
                  hbm_budget_pages=BUDGET, host_pages=HOST, tiers=tiers)
    om = OraclePool(1, 1, 64, T, 2, S, B, HBM, BUDGET, HOST, with_bytes=True, inclusive=tiers == 1)
    # a random placement: each session's blocks split between HBM and the host tier
    ctx = rng.integers(0, B * T - 40, S)
    nb = -(-ctx // T)
    placement = np.full((S, B), -1, np.int64)
    pages, slots = list(rng.permutation(HBM)), list(rng.permutation(HOST))
    used = 0
    for s in range(S):
        for b in range(nb[s]):
            if used < BUDGET - 10 and rng.random() < 0.6:
                placement[s, b] = pages.pop()
                used += 1
            else:
                placement[s, b] = -(slots.pop() + 2)
    om.import_placement(placement, ctx)
    pool.import_placement(placement.astype(np.int32), ctx.astype(np.int32))
    om.hbm[:] = rng.integers(0, 256, om.hbm.shape, dtype=np.uint8)
    om.host[:] = rng.integers(0, 256, om.host.shape, dtype=np.uint8)
    pool.kv.copy_(torch.from_numpy(om.hbm).to(pool.device))
    pool.host[:] = om.host
    sts = [se.SessionState(ctx_tokens=int(ctx[s])) for s in range(S)]
    torch.cuda.synchronize()
    assert pool.sync(raise_on_error=False) == 0
    return rng, pool, om, sts, lv, se


def _compare(pool, om, sts, where):
    from ._lockstep import owners_encoded
    t, oh, oo = pool.tables()
    assert np.array_equal(t, om.tables.astype(np.int32)), where
    assert np.array_equal(oh, owners_encoded(om.owner_hbm, om.hbm_used)), where
    assert np.array_equal(oo, owners_encoded(om.owner_host, om.host_used)), where
    st = pool.stats()
    assert st["error"] == 0, (where, st["error"])
    assert st["hbm_allocated"] == int(om.hbm_used.sum()), where
    assert st["host_allocated"] == int(om.host_used.sum()), where
    assert st["clean_copies"] == om.clean_copies(), where
    g = pool.get_sessions()
    for f in ("ctx_tokens", "flags", "gen_us", "play_us", "t_done_us", "reply_ema_us", "reply_n",
              "reply_tokens", "protect_until_us", "last_use_us"):
        assert np.array_equal(g[f].astype(np.int64), np.array([getattr(x, f) for x in sts])), (where, f)
    assert np.array_equal(pool.kv.cpu().numpy(), om.hbm), (where, "hbm bytes")
    assert np.array_equal(pool.host, om.host), (where, "host bytes")


def _refused(pool, lv, code, where):
    got = pool.sync(raise_on_error=False)
    assert got == code, (where, got, code)
    pool.clear_error()


@pytest.mark.parametrize("seed,tiers", [(0, 0), (1, 0), (2, 1), (3, 1)])
def test_random_call_sequences_match_the_oracle(seed, tiers):
    import torch
    from oracle.policy import select_victims
    from oracle.pool import OracleError, _enc_host
    rng, pool, om, sts, lv, se = _setup(seed, tiers)
    now = 1_000_000
    done = dict.fromkeys(("select", "out", "in", "exchange", "append", "events", "turn", "evict",
                          "bad"), 0)
    try:
        for step in range(300):
            now += int(rng.integers(0, 400_000))
            op = rng.choice(["select", "out", "in", "exchange", "append", "events", "turn", "evict",
                             "bad"], p=[0.07, 0.15, 0.15, 0.12, 0.09, 0.14, 0.14, 0.09, 0.05])
            where = (seed, tiers, step, op)
            if op in ("select", "out", "exchange"):
                k = int(rng.integers(0, 12))
                fb = bool(rng.random() < 0.3)
                vs, vb, vp = select_victims(om.tables, om.nblocks, sts, now, k, 0, 3_000_000,
                                            80_000, 0, fb)
                victims, n = pool.select(now, k, lv.LV_SELECT_FALLBACK if fb else 0)
                assert np.array_equal(victims.cpu().numpy(), np.stack([vs, vb, vp], 1).astype(np.int32)), where
                if op == "select":
                    done["select"] += 1
                if op == "select" or n == 0:
                    continue
                # host slots the victims need (a clean copy needs none)
                need = int(sum(om.shadow[s_, b_] < 0 for s_, b_ in zip(vs, vb)))
                if need > HOST - int(om.host_used.sum()):
                    continue
                if op == "out":
                    slots = om.swap_out(vs, vb, vp)
                    gs, commit = pool.swap_out(victims, n)
                    assert np.array_equal(gs.cpu().numpy(), slots.astype(np.int32)), where
                    if rng.random() < 0.75:
                        om.remap(vs, vb, _enc_host(slots))
                        pool.remap(commit, n)
                    else:
                        om.cancel(_enc_host(slots))
                        pool.cancel((-(gs.long() + 2)).to(torch.int32), n)
                else:   # exchange: evict these victims and reload a session's host blocks
                    sid = int(rng.integers(0, S))
                    hb = om.host_blocks(sid)
                    free_after = BUDGET - int(om.hbm_used.sum()) + n
                    hb = hb[:max(0, min(len(hb), free_after))]
                    slots = om.swap_out(vs, vb, vp)
                    om.remap(vs, vb, _enc_host(slots))
                    pages = om.swap_in(sid, hb)
                    om.remap(np.full(hb.size, sid), hb, pages)
                    blks = torch.from_numpy(hb.astype(np.int32)).to(pool.device)
                    gs, gp = pool.exchange(victims, n, sid, blks, int(hb.size))
                    assert np.array_equal(gs.cpu().numpy(), slots.astype(np.int32)), where
                    assert np.array_equal(gp.cpu().numpy(), pages.astype(np.int32)), where
            elif op == "in":
                cand = [s for s in range(S) if om.host_blocks(s).size]
                if not cand:
                    continue
                sid = int(rng.choice(cand))
                hb = om.host_blocks(sid)
                hb = rng.permutation(hb)[:int(rng.integers(1, hb.size + 1))]
                hb = hb[:max(0, BUDGET - int(om.hbm_used.sum()))]
                if hb.size == 0:
                    continue
                mode = lv.LV_MODE_STAGED if rng.random() < 0.3 else lv.LV_MODE_AUTO
                pages = om.swap_in(sid, hb)
                blks = torch.from_numpy(hb.astype(np.int32)).to(pool.device)
                gp, commit = pool.swap_in(sid, blks, int(hb.size), mode)
                assert np.array_equal(gp.cpu().numpy(), pages.astype(np.int32)), where
                if rng.random() < 0.75:
                    om.remap(np.full(hb.size, sid), hb, pages)
                    pool.remap(commit, int(hb.size))
                else:
                    om.cancel(pages)
                    pool.cancel(gp.clone(), int(hb.size))
            elif op == "append":
                cand = [s for s in range(S) if om.host_blocks(s).size == 0]
                if not cand:
                    continue
                sid = int(rng.choice(cand))
                room = min(B * T - int(om.ctx[sid]), (BUDGET - int(om.hbm_used.sum())) * T)
                if room <= 0:
                    continue
                n_tok = int(rng.integers(1, min(room, 50) + 1))
                pages = om.append(sid, n_tok)
                sts[sid].ctx_tokens = int(om.ctx[sid])
                got = pool.append(sid, n_tok)
                assert np.array_equal(got.cpu().numpy(), pages.astype(np.int32)), where
                # the model writes the new rows: same random bytes on both sides
                rb = 64 * 2
                old_ctx = int(om.ctx[sid]) - n_tok
                for b in range(old_ctx // T, -(-int(om.ctx[sid]) // T)):
                    lo = max(old_ctx, b * T) - b * T
                    hi = min(int(om.ctx[sid]), (b + 1) * T) - b * T
                    data = rng.integers(0, 256, (2, (hi - lo) * rb), dtype=np.uint8)
                    p = int(om.tables[sid, b])
                    om.hbm[:, p, lo * rb:hi * rb] = data
                    pool.kv[:, p, lo * rb:hi * rb] = torch.from_numpy(data).to(pool.device)
            elif op == "events":
                n_ev = int(rng.integers(1, 6))
                ev = np.zeros(n_ev, dtype=lv.EVENT_DTYPE)
                for e in range(n_ev):
                    kind = int(rng.integers(1, 8))
                    sid = int(rng.integers(0, S))
                    a = int(rng.integers(0, 3_000_000)) if kind in (2, 3) else 0
                    bb = int(rng.integers(0, 60)) if kind == 2 else 0
                    ev[e] = (kind, sid, now, a, bb)
                    se.apply_event(sts[sid], kind, now, a, bb, protect_us=2_000_000)
                pool.events(ev)
            elif op == "turn":
                # the oracle's turn (Section 5.1): turn begin, evict the first k of the
                # order (protected KV as a last resort), reload every host block in block
                # order, grow, turn end -- tried on copies first, since a turn that
                # cannot fit is an error on the GPU
                sid = int(rng.integers(0, S))
                n_app = min(int(rng.integers(0, 40)) if rng.random() < 0.5 else 0,
                            B * T - int(om.ctx[sid]))
                trial = [x.copy() for x in sts]
                se.apply_event(trial[sid], se.SE_TURN_BEGIN, now)
                hb = om.host_blocks(sid)
                new_blocks = -(-(int(om.ctx[sid]) + n_app) // T) - int(om.nblocks[sid])
                k = max(0, int(hb.size) + new_blocks - (BUDGET - int(om.hbm_used.sum())))
                vs, vb, vp = select_victims(om.tables, om.nblocks, trial, now, k, 0, 3_000_000,
                                            80_000, 0, True)
                need = int(sum(om.shadow[s_, b_] < 0 for s_, b_ in zip(vs, vb)))
                if vs.size < k or need > HOST - int(om.host_used.sum()):
                    continue
                sts[sid] = trial[sid]
                if k:
                    slots = om.swap_out(vs, vb, vp)
                    om.remap(vs, vb, _enc_host(slots))
                if hb.size:
                    pages = om.swap_in(sid, hb)
                    om.remap(np.full(hb.size, sid), hb, pages)
                if n_app:
                    om.append(sid, n_app)
                    sts[sid].ctx_tokens = int(om.ctx[sid])
                audio, units = int(rng.integers(0, 3_000_000)), int(rng.integers(0, 60))
                se.apply_event(sts[sid], se.SE_TURN_END, now, audio, units)
                flags = lv.LV_RESIDENT_ASYNC_COPY if rng.random() < 0.7 else 0
                lv.lv_turn(pool.handle, sid, now, n_app, audio, units, stream=pool.stream,
                           flags=flags)
            elif op == "evict":
                # lv_evict (Section 5.1 under outside pressure): the first k of the normal
                # order, fewer when there are fewer, evicted with no load
                k = int(rng.integers(0, 16))
                vs, vb, vp = select_victims(om.tables, om.nblocks, sts, now, k, 0, 3_000_000,
                                            80_000, 0, False)
                need = int(sum(om.shadow[s_, b_] < 0 for s_, b_ in zip(vs, vb)))
                if need > HOST - int(om.host_used.sum()):
                    continue
                if vs.size:
                    slots = om.swap_out(vs, vb, vp)
                    om.remap(vs, vb, _enc_host(slots))
                res = np.zeros(1, dtype=lv.RESIDENT_DTYPE)
                flags = lv.LV_RESIDENT_ASYNC_COPY if rng.random() < 0.5 else 0
                lv.lv_evict(pool.handle, now, k, flags, pool.victims, pool.slots, res, pool.stream)
                pool.sync()
                assert int(res["n_victims"][0]) == vs.size and int(res["k"][0]) == k, where
                assert int(res["status"][0]) == (lv.LV_RESIDENT_DONE if vs.size else
                                                 lv.LV_RESIDENT_NOTHING), where
                got = pool.victims[:vs.size].cpu().numpy()
                assert np.array_equal(got, np.stack([vs, vb, vp], 1).astype(np.int32)), where
                if vs.size:
                    assert np.array_equal(pool.slots[:vs.size].cpu().numpy(), slots.astype(np.int32)), where
            else:   # a single-item call that must be refused and change nothing
                which = int(rng.integers(0, 3))
                if which == 0:      # commit to a page nobody reserved
                    free = np.nonzero(~om.hbm_used)[0]
                    res = [s for s in range(S) if om.nblocks[s] > 0]
                    if not free.size or not res:
                        continue
                    e = np.array([[res[0], 0, int(free[0])]], np.int32)
                    pool.remap(torch.from_numpy(e).to(pool.device), 1)
                    _refused(pool, lv, lv.LV_ERR_DOUBLE_MAP, where)
                    with pytest.raises(OracleError):
                        om.remap([res[0]], [0], [int(free[0])])
                elif which == 1:    # a victim that is not where it says
                    res = np.argwhere(om.tables >= 0)
                    if not len(res):
                        continue
                    s_, b_ = (int(x) for x in res[0])
                    wrong = (int(om.tables[s_, b_]) + 1) % HBM
                    v = np.array([[s_, b_, wrong]], np.int32)
                    if int(om.host_used.sum()) >= HOST:
                        continue
                    pool.swap_out(torch.from_numpy(v).to(pool.device), 1)
                    _refused(pool, lv, lv.LV_ERR_STATE, where)
                    # the refused victim's reserved slot is released again
                    pool.cancel(torch.tensor([-(int(pool.slots[0]) + 2)], dtype=torch.int32,
                                             device=pool.device), 1)
                    assert pool.sync(raise_on_error=False) == 0, where
                    with pytest.raises(OracleError):
                        om.swap_out([s_], [b_], [wrong])
                else:               # cancel an owned page
                    owned = np.nonzero(om.owner_hbm[:, 0] >= 0)[0]
                    if not owned.size:
                        continue
                    pool.cancel(torch.tensor([int(owned[0])], dtype=torch.int32, device=pool.device), 1)
                    _refused(pool, lv, lv.LV_ERR_STATE, where)
                    with pytest.raises(OracleError):
                        om.cancel([int(owned[0])])
            if op == "bad" or rng.random() < 0.5:
                _compare(pool, om, sts, where)
            done[op] += 1
        _compare(pool, om, sts, (seed, tiers, "end"))
        om.check_invariants()
        # every kind of call ran, not only the ones that are always possible
        assert min(done.values()) >= 5, done
        if tiers == 1:
            assert om.clean_out > 0, "no eviction found a clean copy"
    finally:
        torch.cuda.synchronize()
        pool.close()
