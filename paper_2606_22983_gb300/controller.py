"""The preload controller of Section 5.2 over liblv: admission, brief wait and
re-check, deferred commit with cancellation, and the cap on protected KV.

  * A preload of B bytes requested at speech start (or barge-in) is admitted at
    time t if, queued behind the transfers already on the modelled host->device
    link (``link_bytes_per_us``), it finishes by the predicted start of the
    session's LLM stage, t_speech + lead, and if the pages it must evict fit in
    the host tier with one session's worth of slots (max_blocks) still free.
    lead is the session's moving average of (turn start - speech start),
    integer EMA of weight 1/4 (the first sample sets it), or ``lead_prior_us``.
  * A refused preload waits and is re-checked at every later event (its slack
    shrinks) until it is admitted, its deadline passes, or the turn arrives.
  * An admitted preload evicts what it needs (next-use order, no fallback tier),
    commits those evictions, then reserves and fills HBM pages (lv_swap_in) but
    commits them (lv_remap) only at the first event at or after its modelled
    finish; a turn that arrives first cancels the reservation (lv_cancel) and
    loads synchronously.  A synchronous load also occupies the modelled link.
  * A completed preload protects the session until finish + protect_us; when
    the protected sessions' resident pages exceed ``cap_pages`` the oldest
    protections (smallest protect_until, then lower session id) are dropped.

All data movement and table updates are liblv calls; this class keeps only the
controller's host-side schedule.
"""
from __future__ import annotations

import numpy as np
import torch

from . import lv
from .manager import EV_TURN, EV_TURN_ANY, EV_TURN_SCATTER, KVManager, _event


class ControlledKVManager(KVManager):
    def __init__(self, pool, link_bytes_per_us=200_000, lead_prior_us=2_000_000, cap_pages=None,
                 **kw):
        kw.setdefault("driver", "exchange")
        super().__init__(pool, **kw)
        self.bw = int(link_bytes_per_us)
        self.lead_prior_us = int(lead_prior_us)
        self.cap_pages = cap_pages
        self.link_free_at = 0
        self.lead = {}
        self.speech_t = {}
        self.waiting = {}
        self.pending = {}
        self.completed = set()
        for k in ("admitted", "completed", "waited", "given_up", "cancelled", "hits"):
            self.counters[k] = 0

    def _lead(self, sid):
        ema, n = self.lead.get(sid, (0, 0))
        return ema if n > 0 else self.lead_prior_us

    def _duration(self, n_pages):
        b = n_pages * self.pool.J * self.pool.P
        return -(-b // self.bw)

    def _host_free(self):
        st = self.pool.stats()
        return st["host_pages"] - st["host_allocated"]

    def _try_admit(self, sid, t, rec):
        pool = self.pool
        w = self.waiting[sid]
        blks, n = self.host_blocks(sid)
        if n == 0:
            del self.waiting[sid]
            return
        start = max(t, self.link_free_at)
        finish = start + self._duration(n)
        if finish > w["t_pred"]:
            w["refused"] += 1
            return
        k = max(0, n - self.free_budget())
        if k > self._host_free() - pool.max_blocks:
            w["refused"] += 1
            return
        if k > 0:
            victims, nv = pool.select(t, k, 0)
            if nv < k:
                w["refused"] += 1
                return
            rec.setdefault("preload_victims", []).append(victims.cpu().numpy().astype(np.int64))
            pool.exchange(victims, nv, 0, None, 0, self.mode)
            self.counters["victims"] += k
            self.counters["pages_out"] += k
            self.bytes_moved += k * pool.J * pool.P
        blks = blks.clone()
        pages, commit = pool.swap_in(sid, blks, n, self.mode)
        pages, commit = pages.clone(), commit.clone()
        self.pending[sid] = {"finish": finish, "n": n, "pages": pages, "commit": commit}
        self.counters["pages_in"] += n
        self.bytes_moved += n * pool.J * pool.P
        self.link_free_at = finish
        self.counters["admitted"] += 1
        if w["refused"]:
            self.counters["waited"] += 1
        t_pred = w["t_pred"]
        del self.waiting[sid]
        rec.setdefault("admitted", []).append((sid, start, finish, t_pred,
                                               pages.cpu().numpy().astype(np.int64)))

    def _complete(self, sid, rec):
        pool = self.pool
        p = self.pending.pop(sid)
        pool.remap(p["commit"], p["n"])
        pool.events(_event(lv.LV_EV_PRELOADED, sid, p["finish"]))
        self.counters["completed"] += 1
        self.counters["preloads"] += 1
        self.completed.add(sid)
        self._enforce_cap(p["finish"], rec)
        rec.setdefault("completed", []).append(sid)

    def _enforce_cap(self, now, rec):
        if self.cap_pages is None:
            return
        st = self.pool.get_sessions()
        prot = sorted((int(st["protect_until_us"][s]), s) for s in range(self.pool.S)
                      if int(st["protect_until_us"][s]) > now)
        if not prot:
            return
        hbm, _ = self.pool.counts()
        total = sum(int(hbm[s]) for _, s in prot)
        drop = []
        for _, s in prot:
            if total <= self.cap_pages:
                break
            drop.append(s)
            total -= int(hbm[s])
        if drop:
            ev = np.zeros(len(drop), dtype=lv.EVENT_DTYPE)
            ev["kind"], ev["sid"], ev["t_us"] = lv.LV_EV_UNPROTECT, drop, now
            self.pool.events(ev)
            rec.setdefault("unprotected", []).extend(drop)

    def _housekeeping(self, t, rec):
        for sid in sorted(self.pending, key=lambda s: (self.pending[s]["finish"], s)):
            if self.pending[sid]["finish"] <= t:
                self._complete(sid, rec)
        for sid in sorted(self.waiting):
            if t >= self.waiting[sid]["t_pred"]:
                del self.waiting[sid]
                self.counters["given_up"] += 1
            else:
                self._try_admit(sid, t, rec)

    def _before_turn(self, sid, t, rec):
        if sid in self.speech_t:
            x = max(0, t - self.speech_t.pop(sid))
            ema, n = self.lead.get(sid, (0, 0))
            self.lead[sid] = (x if n == 0 else (3 * ema + x) // 4, n + 1)
        if sid in self.waiting:
            del self.waiting[sid]
            self.counters["given_up"] += 1
        if sid in self.pending:
            p = self.pending.pop(sid)
            self.pool.cancel(p["pages"], p["n"])
            self.counters["cancelled"] += 1
            rec["cancelled"] = sid
        if sid in self.completed:
            self.completed.discard(sid)
            if self.host_blocks(sid)[1] == 0:
                self.counters["hits"] += 1

    def preload(self, sid, now_us, rec):
        self.speech_t.setdefault(sid, now_us)
        if sid in self.pending or sid in self.waiting:
            return
        if self.host_blocks(sid)[1] == 0:
            return
        self.waiting[sid] = {"t_pred": self.speech_t[sid] + self._lead(sid), "refused": 0}
        self._try_admit(sid, now_us, rec)

    def step(self, ev, index=None):
        t, kind, sid, a, b, c, d = (int(x) for x in ev)
        pre = {}
        self._housekeeping(t, pre)
        if kind in (EV_TURN, EV_TURN_ANY, EV_TURN_SCATTER):
            target = sid if kind == EV_TURN else self.turn_target(d)
            self._before_turn(target, t, pre)
        loaded0 = self.counters["pages_in"]
        rec = super().step(ev, index)
        rec.update(pre)
        loaded = self.counters["pages_in"] - loaded0
        if kind in (EV_TURN, EV_TURN_ANY, EV_TURN_SCATTER) and loaded:
            self.link_free_at = max(t, self.link_free_at) + self._duration(loaded)
        return rec
