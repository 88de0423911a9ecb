"""The KV manager's procedure over an event script (Sections 5.1 and 5.2).

For each script event (see ``workloads.scripts`` for the kinds):

  PLAYBACK      session state update only.
  SPEECH_START  immediate reuse; preload trigger (Section 5.2).
  BARGE_IN      unplayed reply discarded; immediate reuse; preload trigger.
  SPEECH_STOP   session state update (reply-interval sample).
  TURN          the request runs: the session's KV is made fully resident
                (a synchronous, foreground load of any host blocks), its
                context grows, then the reply is recorded.
  TURN_SCATTER  a turn whose host blocks are reloaded in a given scattered order.
  EVICT         k pages are freed now, in the victim order of Section 5.1.

Making a session resident with ``need`` missing pages (host blocks plus new
blocks) first evicts ``k = need - free`` pages when the HBM budget is short,
in the victim order of Section 5.1 (exactly k pages, never rounded up to a
whole session), then swaps the host blocks in, in ascending block order.
A foreground turn ranks with the fallback tier (protected, non-running KV
after all normally eligible KV); a preload does not.

Preload (Section 5.2): only when the session has host blocks.  Admission is
"always" unless ``admit`` is given.  A preload that cannot find k eligible
victims is skipped (nothing moves) and the next turn loads synchronously.
After a completed preload the warmed KV is protected for ``protect_us``.

Every event (or every turn, with ``rank_on="turns"``) ends with a full-order
ranking (k = all) that the parity tests compare.
"""
from __future__ import annotations

import numpy as np

from . import sessions as se
from .policy import LRU, order_global, order_lru, select_victims
from .pool import OraclePool, OracleError, _enc_host

# script event kinds (the published script format)
EV_TURN, EV_TURN_ANY, EV_PLAYBACK, EV_SPEECH_START, EV_BARGE_IN, EV_SPEECH_STOP = 1, 2, 3, 4, 5, 6
EV_TURN_SCATTER, EV_EVICT = 7, 8


class OracleManager:
    """The KV manager of Section 5 over an event script: turns make their session
    resident (Section 5.1 eviction, Section 6 loading), speech start and barge-in
    trigger preloads (Section 5.2), monitor events update the sessions (Section 3)."""
    def __init__(self, workload, with_bytes=True, content=None, admit=None, rank_on="all"):
        spec = workload.spec
        sh = spec.shape
        self.wl = workload
        self.spec = spec
        self.shape = sh
        self.pool = OraclePool(sh.layers, sh.kv_heads, sh.head_dim, sh.page_tokens, sh.elem_bytes,
                               spec.n_sessions, spec.max_blocks, spec.hbm_pages,
                               spec.hbm_budget_pages, spec.host_pages, with_bytes=with_bytes,
                               inclusive=spec.tiers == 1)
        init = workload.init
        self.pool.import_placement(init.placement, init.ctx_tokens)
        self.sessions = []
        for s in range(spec.n_sessions):
            st = se.SessionState(ctx_tokens=int(init.ctx_tokens[s]), gen_us=int(init.gen_us[s]),
                                 play_us=int(init.play_us[s]), reply_tokens=int(init.reply_tokens[s]))
            if int(init.resp_open[s]):
                st.flags |= se.RESP_OPEN
            self.sessions.append(st)
        self.content = content        # (seed, value table) or "tagged": how KV bytes are made
        self.admit = admit
        self.rank_on = rank_on          # 'all' events, 'turns' only, or 'none'
        self.counters = dict(victims=0, pages_out=0, pages_in=0, preloads=0,
                             preload_skipped=0, turns=0, sync_loads=0, appended=0)
        if with_bytes and content is not None:
            self._write_initial_bytes()

    # ------------------------------------------------------------ content
    def _subpage_content(self, sid, blk, ctx):
        from workloads.content import (subpage_offsets, subpage_values_np, tagged_values_np,
                                       valid_rows)
        sh = self.shape
        J = 2 * sh.layers
        layer = np.arange(J) // 2
        kv = np.arange(J) % 2
        if self.content == "tagged":      # address-tagged chunks (a debugging mode)
            rows = np.full(J, int(valid_rows(ctx, blk, sh)))
            return tagged_values_np(np.full(J, sid), np.full(J, blk), layer, kv, rows,
                                    sh).view(np.uint8).reshape(J, sh.subpage_bytes)
        seed, table = self.content
        off = subpage_offsets(seed, np.full(J, sid), np.full(J, blk), layer, kv, sh)
        rows = np.full(J, int(valid_rows(ctx, blk, sh)))
        return subpage_values_np(table, off, rows, sh).view(np.uint8).reshape(J, sh.subpage_bytes)

    def _write_initial_bytes(self):
        pool = self.pool
        for s in range(pool.S):
            for b in range(int(pool.nblocks[s])):
                data = self._subpage_content(s, b, int(pool.ctx[s]))
                e = int(pool.tables[s, b])
                if e >= 0:
                    pool.hbm[:, e, :] = data
                else:
                    pool.host[-(e + 2)] = data

    def _write_appended_rows(self, sid, old_ctx, new_ctx):
        """The model writes K/V of the appended tokens into their (resident) pages.

        A block that already existed gets only its new rows; a newly allocated
        block is written whole, rows past the context end as zeros."""
        pool, sh = self.pool, self.shape
        T, rb = sh.page_tokens, sh.row_elems * sh.elem_bytes
        old_blocks = -(-old_ctx // T)
        for b in range(old_ctx // T, -(-new_ctx // T)):
            lo = max(old_ctx, b * T) - b * T if b < old_blocks else 0
            hi = min(new_ctx, (b + 1) * T) - b * T if b < old_blocks else T
            data = self._subpage_content(sid, b, new_ctx)
            p = int(pool.tables[sid, b])
            pool.hbm[:, p, lo * rb:hi * rb] = data[:, lo * rb:hi * rb]

    # ------------------------------------------------------------- ranking
    def full_order(self, now_us):
        """The whole victim order at now_us: Section 5.1 (Eq. 4 keys), or the LRU
        baseline of Sections 2.3 and 5."""
        sp = self.spec
        if sp.policy == LRU:
            return order_lru(self.pool.tables, self.pool.nblocks, self.sessions, sp.within_order)
        return order_global(self.pool.tables, self.pool.nblocks, self.sessions, now_us,
                            sp.t_play_mode, sp.reply_prior_us, sp.unit_us, sp.within_order)

    def select(self, now_us, k, fallback=False):
        """The first k victims of the order (Section 5.1); with ``fallback`` the
        protected, non-running tier follows the normal one (Section 5.2)."""
        sp = self.spec
        if sp.policy == LRU:
            s_, b_, p_ = order_lru(self.pool.tables, self.pool.nblocks, self.sessions, sp.within_order)
            k = min(int(k), s_.size)
            return s_[:k], b_[:k], p_[:k]
        return select_victims(self.pool.tables, self.pool.nblocks, self.sessions, now_us, k,
                              sp.t_play_mode, sp.reply_prior_us, sp.unit_us, sp.within_order,
                              fallback)

    # ------------------------------------------------------------ movement
    def make_resident(self, sid, now_us, append_tokens, foreground, rec, order_key=None):
        """Make session sid fully resident, then grow it: evict exactly the deficit in
        the Section 5.1 order, load the host blocks (Sections 5.2 and 6; block order, or
        the script's scattered order), allocate pages for new tokens (Section 5.1 keeps
        block-level allocation).  False when a preload finds too few victims."""
        pool = self.pool
        host_blks = pool.host_blocks(sid)
        if order_key is not None:
            from workloads.scripts import scatter_order
            host_blks = scatter_order(order_key, host_blks)
        new_ctx = int(pool.ctx[sid]) + int(append_tokens)
        new_blocks = -(-new_ctx // pool.T) - int(pool.nblocks[sid])
        need = int(host_blks.size) + new_blocks
        k = max(0, need - pool.free_budget())
        rec["k"] = k
        if k > 0:
            # a preload may evict only later-use idle KV (Section 5.2); a foreground
            # turn may also take protected, non-running KV as a last resort
            vs, vb, vp = self.select(now_us, k, fallback=foreground)
            rec["victims"] = np.stack([vs, vb, vp], axis=1) if vs.size else np.zeros((0, 3), np.int64)
            if vs.size < k:
                if foreground:
                    raise OracleError("NO_HBM", f"turn of session {sid} needs {k} victims, "
                                      f"{vs.size} eligible")
                return False
            slots = pool.swap_out(vs, vb, vp)
            rec["slots"] = slots
            pool.remap(vs, vb, _enc_host(slots))
            self.counters["victims"] += k
            self.counters["pages_out"] += k
        if host_blks.size:
            pages = pool.swap_in(sid, host_blks)
            rec["in_blocks"] = host_blks
            rec["in_pages"] = pages
            pool.remap(np.full(host_blks.size, sid), host_blks, pages)
            self.counters["pages_in"] += int(host_blks.size)
        if append_tokens:
            old_ctx = int(pool.ctx[sid])
            pages = pool.append(sid, append_tokens)
            rec["append_pages"] = pages
            self.sessions[sid].ctx_tokens = int(pool.ctx[sid])
            self.counters["appended"] += int(pages.size)
            if pool.with_bytes and self.content is not None:
                self._write_appended_rows(sid, old_ctx, int(pool.ctx[sid]))
        return True

    def preload(self, sid, now_us, rec):
        """Speech-triggered preload of sid's host blocks (Section 5.2): admitted by
        ``admit`` when given, skipped when too few victims, protected once complete."""
        if self.spec.policy == LRU:
            return              # the baseline loads at turn start only
        host_blks = self.pool.host_blocks(sid)
        if host_blks.size == 0:
            return
        if self.admit is not None and not self.admit(self, sid, now_us, int(host_blks.size)):
            self.counters["preload_skipped"] += 1
            rec["preload"] = "skipped"
            return
        if self.make_resident(sid, now_us, 0, foreground=False, rec=rec):
            se.apply_event(self.sessions[sid], se.SE_PRELOADED, now_us,
                           protect_us=self.spec.protect_us)
            self.counters["preloads"] += 1
            rec["preload"] = "done"
        else:
            self.counters["preload_skipped"] += 1
            rec["preload"] = "skipped"

    def evict(self, now_us, k, rec):
        """Free k pages now (memory pressure from elsewhere): the first k of the
        Section 5.1 victim order with normal eligibility, or all candidates when there
        are fewer."""
        pool = self.pool
        vs, vb, vp = self.select(now_us, k)
        rec["k"] = int(k)
        rec["victims"] = np.stack([vs, vb, vp], axis=1) if vs.size else np.zeros((0, 3), np.int64)
        if vs.size:
            slots = pool.swap_out(vs, vb, vp)
            rec["slots"] = slots
            pool.remap(vs, vb, _enc_host(slots))
            self.counters["victims"] += int(vs.size)
            self.counters["pages_out"] += int(vs.size)

    def turn_target(self, perm_row):
        """The session a TURN_ANY / TURN_SCATTER event picks: the first of the script's
        seeded order that has offloaded KV (a workload construct, not from the paper)."""
        perm = self.wl.perms[perm_row]
        for s in perm:
            if self.pool.host_blocks(int(s)).size:
                return int(s)
        return int(perm[0])

    # --------------------------------------------------------------- events
    def step(self, i):
        """Process script event i (Section 3 monitor events; the decisions of Sections
        5.1 and 5.2); returns a record of everything it decided."""
        t, kind, sid, a, b, c, d = self.wl.event(i)
        rec = {"i": i, "t": t, "kind": kind}
        sts = self.sessions
        if kind == EV_PLAYBACK:
            se.apply_event(sts[sid], se.SE_PLAYBACK, t, a)
        elif kind == EV_SPEECH_START:
            se.apply_event(sts[sid], se.SE_SPEECH_START, t)
            self.preload(sid, t, rec)
        elif kind == EV_BARGE_IN:
            se.apply_event(sts[sid], se.SE_BARGE_IN, t)
            self.preload(sid, t, rec)
        elif kind == EV_SPEECH_STOP:
            se.apply_event(sts[sid], se.SE_SPEECH_STOP, t)
        elif kind in (EV_TURN, EV_TURN_ANY, EV_TURN_SCATTER):
            order_key = None
            if kind == EV_TURN_SCATTER:
                sid = self.turn_target(d)
                order_key, a = a, 0
            elif kind == EV_TURN_ANY:
                sid = self.turn_target(d)
            se.apply_event(sts[sid], se.SE_TURN_BEGIN, t)
            if self.pool.host_blocks(sid).size:
                self.counters["sync_loads"] += 1
            self.make_resident(sid, t, a, foreground=True, rec=rec, order_key=order_key)
            se.apply_event(sts[sid], se.SE_TURN_END, t, b, c)
            self.counters["turns"] += 1
        elif kind == EV_EVICT:
            self.evict(t, a, rec)
        else:
            raise ValueError(f"unknown script event kind {kind}")
        rec["sid"] = sid
        if self.rank_on == "all" or (self.rank_on == "turns" and kind in (EV_TURN, EV_TURN_ANY,
                                                                           EV_TURN_SCATTER)):
            rec["order"] = np.stack(self.full_order(t), axis=1)
        return rec

    def run(self, lo=0, hi=None):
        """Process script events lo..hi (harness helper)."""
        hi = self.wl.n_events if hi is None else hi
        return [self.step(i) for i in range(lo, hi)]

    # ------------------------------------------------------------- snapshot
    def session_arrays(self):
        """The session table as arrays (harness helper for comparisons)."""
        keys = ("ctx_tokens", "flags", "gen_us", "play_us", "t_done_us", "reply_ema_us",
                "reply_n", "reply_tokens", "protect_until_us", "last_use_us")
        return {k: np.array([getattr(s, k) for s in self.sessions], dtype=np.int64) for k in keys}
