"""The preload controller of Section 5.2 (lv_controller_* in liblv) driven from the
KV manager's event loop.

The controller itself -- admission against a modelled host->device link and the
predicted turn start, the brief wait and re-check, the deferred commit with
cancellation, the cap on protected KV -- is native code in liblv (see the
lv_controller_* declarations in include/lv.h for its readings).  This class calls
its hooks in event order (tick at every event, turn begin before a turn, speech at
a speech start or barge-in, turn loaded after a turn's own load) and turns its
decision log into the per-event records the manager reports.
"""
from __future__ import annotations

import numpy as np

from . import lv
from .manager import EV_TURN, EV_TURN_ANY, EV_TURN_SCATTER, KVManager


class ControlledKVManager(KVManager):
    def __init__(self, pool, link_bytes_per_us=200_000, lead_prior_us=2_000_000, cap_pages=None,
                 **kw):
        kw.setdefault("driver", "exchange")
        super().__init__(pool, **kw)
        self.ctl = lv.lv_controller_create(pool.handle, int(link_bytes_per_us), int(lead_prior_us),
                                           cap_pages, self.mode)
        pool.attach(self)       # the controller goes before the pool
        self._native = lv.lv_controller_counters_get(self.ctl)
        for k in ("admitted", "completed", "waited", "given_up", "cancelled", "hits"):
            self.counters[k] = 0

    def close(self):
        if getattr(self, "ctl", None) and getattr(self.pool, "handle", None):
            lv.lv_controller_destroy(self.ctl, self.pool.stream)
        self.ctl = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    # ---------------------------------------------------------- native log
    def _drain(self, rec):
        """Moves the controller's new decisions into ``rec`` and its counters into
        the manager's."""
        recs, data = lv.lv_controller_records(self.ctl)
        for r in recs:
            kind, sid, n, off = int(r["kind"]), int(r["sid"]), int(r["n"]), int(r["data_offset"])
            if kind == lv.LV_CTL_ADMITTED:
                rec.setdefault("admitted", []).append(
                    (sid, int(r["start_us"]), int(r["finish_us"]), int(r["deadline_us"]),
                     data[off:off + n].astype(np.int64)))
            elif kind == lv.LV_CTL_EVICTED:
                rec.setdefault("preload_victims", []).append(
                    data[off:off + 3 * n].reshape(n, 3).astype(np.int64))
            elif kind == lv.LV_CTL_COMPLETED:
                rec.setdefault("completed", []).append(sid)
            elif kind == lv.LV_CTL_UNPROTECTED:
                rec.setdefault("unprotected", []).append(sid)
            elif kind == lv.LV_CTL_CANCELLED:
                rec["cancelled"] = sid
        now = lv.lv_controller_counters_get(self.ctl)
        d = {k: now[k] - self._native[k] for k in now}
        self._native = now
        for k in ("admitted", "completed", "waited", "given_up", "cancelled", "hits"):
            self.counters[k] += d[k]
        self.counters["victims"] += d["victims"]
        self.counters["pages_out"] += d["victims"]
        self.counters["pages_in"] += d["pages_in"]
        self.counters["preloads"] += d["completed"]
        self.bytes_moved += (d["victims"] + d["pages_in"]) * self.pool.J * self.pool.P

    # ------------------------------------------------------------- events
    def preload(self, sid, now_us, rec):
        lv.lv_controller_speech(self.ctl, sid, now_us, self.pool.stream)
        self._drain(rec)

    def step(self, ev, index=None):
        t, kind, sid, a, b, c, d = (int(x) for x in ev)
        pre = {}
        lv.lv_controller_tick(self.ctl, t, self.pool.stream)
        self._drain(pre)
        turn = kind in (EV_TURN, EV_TURN_ANY, EV_TURN_SCATTER)
        if turn:
            target = sid if kind == EV_TURN else self.turn_target(d)
            lv.lv_controller_turn_begin(self.ctl, target, t, self.pool.stream)
            self._drain(pre)
        loaded0 = self.counters["pages_in"]
        rec = super().step(ev, index)
        rec.update(pre)
        loaded = self.counters["pages_in"] - loaded0
        if turn and loaded:
            lv.lv_controller_turn_loaded(self.ctl, t, loaded)
        return rec
