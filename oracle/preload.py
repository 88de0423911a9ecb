"""The preload controller of Section 5.2, on top of the oracle's KV manager.

Readings (the paper describes the controller in prose; every constant below is a
reading -- parity unpinned against the paper):

  * Admission: a preload of B bytes is admitted at time t only if its transfer,
    queued behind the transfers already on the host->device link, finishes by
    the predicted start of the session's LLM stage:
        start  = max(t, link_free_at);  finish = start + ceil(B / link_bytes_per_us)
        admit  iff finish <= t_speech + lead
    (the transfer must be hidden before the turn under the current load), and only
    if the victims it must evict fit in the host tier with ``max_blocks`` slots
    still free (room for a foreground turn's synchronous eviction).  lead is
    the session's moving average of (turn start - speech start) -- integer EMA
    with weight 1/4, first sample sets it -- or ``lead_prior_us`` before any
    sample.  t_speech is the first speech start (or barge-in) since the session's
    last turn: later ones before the same turn move neither the deadline nor the
    sample.  A sync load at a turn also occupies the link.
  * Brief wait and re-check: a preload that is not admitted waits; at every later
    event before the turn it is re-evaluated at that event's time (the slack
    shrinks as time passes) and given up once t >= t_speech + lead.
  * An admitted preload evicts what it needs (next-use order, normal tier only)
    and reserves and copies at once, but commits only when its transfer
    completes (at the first event with time >= finish).  If the turn arrives
    first, the reservation is cancelled and the turn loads synchronously (the
    paper's fallback).
  * Protection and its cap: a completed preload protects the session until
    finish + protect_us; if the protected sessions' resident pages then exceed
    ``cap_pages``, the oldest protections (smallest protect_until, then lower
    session id) are dropped until they fit -- the new one too if it alone
    exceeds the cap.

The code is pinned to these readings by two scenarios whose every decision was
worked by hand (tests/golden/preload_controller_hand.json: admission, queueing on
the link, victims, waiting, completion, cancellation, the cap, hits, give-ups,
the lead average) and by properties on the generated workloads.

Counters: admitted, completed, waited (admitted after at least one refusal),
given_up, cancelled, hits (turns whose session needed no synchronous load after
a completed preload), sync_loads.
"""
from __future__ import annotations

import numpy as np

from . import sessions as se
from .manager import (OracleManager, EV_TURN, EV_TURN_ANY, EV_TURN_SCATTER, EV_SPEECH_START,
                      EV_BARGE_IN)
from .pool import _enc_host


class PreloadController:
    """The preload controller's constants (Section 5.2): the host link's speed, the
    prior speech-to-turn lead and an optional cap on warmed pages."""

    def __init__(self, link_bytes_per_us=200_000, lead_prior_us=2_000_000, cap_pages=None):
        self.bw = int(link_bytes_per_us)
        self.lead_prior_us = int(lead_prior_us)
        self.cap_pages = cap_pages


class ControlledOracleManager(OracleManager):
    """OracleManager whose preloads go through the Section 5.2 controller."""

    def __init__(self, workload, controller: PreloadController, **kw):
        super().__init__(workload, **kw)
        self.ctl = controller
        self.link_free_at = 0
        self.lead = {}        # sid -> (ema_us, n)
        self.speech_t = {}    # sid -> time of the speech start (or barge-in) before its turn
        self.waiting = {}     # sid -> {"t_pred", "refused"}
        self.pending = {}     # sid -> {"finish", "blks", "pages"}
        self.completed = set()
        for k in ("admitted", "completed", "waited", "given_up", "cancelled", "hits"):
            self.counters[k] = 0

    # ------------------------------------------------------------ helpers
    def _lead(self, sid):
        ema, n = self.lead.get(sid, (0, 0))
        return ema if n > 0 else self.ctl.lead_prior_us

    def _duration(self, n_pages):
        b = n_pages * self.pool.J * self.pool.P
        return -(-b // self.ctl.bw)

    def _try_admit(self, sid, t, rec):
        w = self.waiting[sid]
        blks = self.pool.host_blocks(sid)
        if blks.size == 0:
            del self.waiting[sid]
            return
        start = max(t, self.link_free_at)
        finish = start + self._duration(int(blks.size))
        if finish > w["t_pred"]:
            w["refused"] += 1
            return
        k = max(0, int(blks.size) - self.pool.free_budget())
        host_free = self.pool.host_pages - int(self.pool.host_used.sum())
        if k > host_free - self.spec.max_blocks:
            w["refused"] += 1
            return
        if k > 0:
            vs, vb, vp = self.select(t, k, fallback=False)
            if vs.size < k:
                w["refused"] += 1
                return
            slots = self.pool.swap_out(vs, vb, vp)
            self.pool.remap(vs, vb, _enc_host(slots))
            self.counters["victims"] += k
            self.counters["pages_out"] += k
            rec.setdefault("preload_victims", []).append(np.stack([vs, vb, vp], axis=1))
        pages = self.pool.swap_in(sid, blks)
        self.counters["pages_in"] += int(blks.size)
        self.pending[sid] = {"finish": finish, "blks": blks, "pages": pages}
        self.link_free_at = finish
        self.counters["admitted"] += 1
        if w["refused"]:
            self.counters["waited"] += 1
        del self.waiting[sid]
        rec.setdefault("admitted", []).append((sid, start, finish, w["t_pred"], pages))

    def _complete(self, sid, rec):
        p = self.pending.pop(sid)
        self.pool.remap(np.full(p["blks"].size, sid), p["blks"], p["pages"])
        se.apply_event(self.sessions[sid], se.SE_PRELOADED, p["finish"], protect_us=self.spec.protect_us)
        self.counters["completed"] += 1
        self.counters["preloads"] += 1
        self.completed.add(sid)
        self._enforce_cap(p["finish"], rec)
        rec.setdefault("completed", []).append(sid)

    def _enforce_cap(self, now, rec):
        cap = self.ctl.cap_pages
        if cap is None:
            return
        prot = [(st.protect_until_us, s) for s, st in enumerate(self.sessions)
                if st.protect_until_us > now]
        res = {s: int((self.pool.tables[s, :int(self.pool.nblocks[s])] >= 0).sum()) for _, s in prot}
        total = sum(res.values())
        for _, s in sorted(prot):                 # oldest protection first
            if total <= cap:
                break
            self.sessions[s].protect_until_us = 0
            total -= res[s]
            rec.setdefault("unprotected", []).append(s)

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

    # ------------------------------------------------------------- events
    def preload(self, sid, now_us, rec):
        """A speech start (or barge-in) asks for ``sid``'s host blocks; the request waits
        until the link can finish it before the predicted turn (Section 5.2)."""
        self.speech_t.setdefault(sid, now_us)
        if sid in self.pending or sid in self.waiting:
            return
        if self.pool.host_blocks(sid).size == 0:
            return
        self.waiting[sid] = {"t_pred": self.speech_t[sid] + self._lead(sid), "refused": 0}
        self._try_admit(sid, now_us, rec)

    def step(self, i):
        """One event, with the controller's admissions, completions and lead updates
        around it (Section 5.2)."""
        t, kind, sid, a, b, c, d = self.wl.event(i)
        pre = {}
        self._housekeeping(t, pre)
        if kind in (EV_TURN, EV_TURN_ANY, EV_TURN_SCATTER):
            target = sid
            if kind != EV_TURN:
                target = self.turn_target(d)
            self._before_turn(target, t, pre)
        rec = super().step(i)
        rec.update({k: v for k, v in pre.items()})
        if kind in (EV_TURN, EV_TURN_ANY, EV_TURN_SCATTER) and "in_blocks" in rec:
            self.link_free_at = max(t, self.link_free_at) + self._duration(len(rec["in_blocks"]))
        return rec

    def _before_turn(self, sid, t, rec):
        if sid in self.speech_t:
            x = max(0, t - self.speech_t.pop(sid))
            ema, n = self.lead.get(sid, (0, 0))
            self.lead[sid] = (x if n == 0 else (3 * ema + x) // 4, n + 1)
        if sid in self.waiting:
            del self.waiting[sid]
            self.counters["given_up"] += 1
        if sid in self.pending:
            p = self.pending.pop(sid)           # still in flight: cancel, load synchronously
            self.pool.cancel(p["pages"])
            self.counters["cancelled"] += 1
            rec["cancelled"] = sid
        if sid in self.completed:
            self.completed.discard(sid)
            if self.pool.host_blocks(sid).size == 0:
                self.counters["hits"] += 1
