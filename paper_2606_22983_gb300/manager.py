"""The KV manager's turn and preload procedure over liblv (Sections 5.1 and 5.2).

Consumes monitor event scripts (records ``(t_us, kind, sid, a, b, c, d)``):

  kind 1 TURN(sid, a=append_tokens, b=reply_audio_us, c=reply_tokens)
  kind 2 TURN_ANY(d=row of perms): the first session in perms[d] with blocks in
         the host tier takes the turn (perms[d][0] when none has)
  kind 3 PLAYBACK(sid, a=delta_us)    kind 4 SPEECH_START(sid)
  kind 5 BARGE_IN(sid)                kind 6 SPEECH_STOP(sid)
  kind 7 TURN_SCATTER(d=row, a=key): as TURN_ANY, host blocks reloaded in the
         order ``order_fn(key, blocks)`` (given by the caller; it must order blocks
         by a key of each block alone, so that the device driver can pass it as
         per-block load keys)
  kind 8 EVICT(a=k): free k pages now, in the next-use order

A turn makes the session fully resident (a synchronous foreground load),
grows its context, then records the reply.  By default (``driver="device"``)
each step is one lv_make_resident call that decides and moves everything on the
GPU without a host round trip; ``driver="exchange"`` ranks, reads the count back
and calls lv_swap_exchange; ``driver="sequential"`` issues swap-out, commit,
swap-in, commit one after the other.  All three give the same result.  Speech start and barge-in trigger a
best-effort preload of the session's host blocks.  Making a session resident
with ``need`` missing pages first evicts exactly ``k = need - free`` pages in
the next-use order (foreground turns may also take protected, non-running KV
after every normally eligible block; a preload may not), swaps them out, commits,
then swaps the host blocks in (ascending block order) and commits.  A preload
that finds fewer than k victims is skipped; a completed one protects the
warmed KV for the pool's protection window.

Every step runs in liblv's kernels; this class only decides which calls to
make (and, on the host-driven paths, reads back the few counts it needs).
"""
from __future__ import annotations

import numpy as np
import torch

from . import lv
from .pool import KVPool

EV_TURN, EV_TURN_ANY, EV_PLAYBACK, EV_SPEECH_START, EV_BARGE_IN, EV_SPEECH_STOP = 1, 2, 3, 4, 5, 6
EV_TURN_SCATTER, EV_EVICT = 7, 8

_STATE_EVENT = {EV_PLAYBACK: lv.LV_EV_PLAYBACK, EV_SPEECH_START: lv.LV_EV_SPEECH_START,
                EV_BARGE_IN: lv.LV_EV_BARGE_IN, EV_SPEECH_STOP: lv.LV_EV_SPEECH_STOP}


def _event(kind, sid, t, a=0, b=0):
    e = np.zeros(1, dtype=lv.EVENT_DTYPE)
    e["kind"], e["sid"], e["t_us"], e["a"], e["b"] = kind, sid, t, a, b
    return e


def load_keys(order_fn, order_key, n_blocks):
    """Per-block keys (uint64 [n_blocks]) whose ascending order is ``order_fn(order_key,
    blocks)`` for any set of blocks: the rank of each block in the order of all of them.
    ``order_fn`` must order blocks by a key of each block alone (ties by block id), as the
    workloads' scatter order does; then its order of any subset is the subset's order in
    the whole."""
    perm = np.asarray(order_fn(order_key, np.arange(n_blocks)), dtype=np.int64)
    keys = np.empty(n_blocks, dtype=np.uint64)
    keys[perm] = np.arange(n_blocks, dtype=np.uint64)
    return keys


class KVManager:
    def __init__(self, pool: KVPool, perms=None, on_append=None, rank_on="none", admit=None,
                 mode=lv.LV_MODE_AUTO, record=True, driver="device", order_fn=None,
                 async_copy=False, script=None):
        self.pool = pool
        # device driver: turns' page copies on the pool's copy stream, overlapping the
        # next turn's decisions (LV_RESIDENT_ASYNC_COPY); exchange driver, staged mode:
        # consecutive exchanges pipelined (LV_MODE_ASYNC); pool.sync() joins them
        self.async_copy = async_copy
        self.perms = perms
        self.on_append = on_append      # callback(sid, old_ctx, new_ctx, pages) after growth
        self.rank_on = rank_on          # 'all' events, 'turns' only, or 'none'
        self.admit = admit              # callback(manager, sid, now, n_host_blocks) -> bool
        self.mode = mode
        self.record = record
        if driver not in ("device", "exchange", "sequential"):
            raise ValueError(f"unknown driver {driver!r}")
        # device: one lv_make_resident per step, no host round trip;
        # exchange: select, then one lv_swap_exchange; sequential: the four calls
        self.driver = driver
        self.order_fn = order_fn        # (key, blocks) -> blocks, for TURN_SCATTER
        self.res_h = torch.zeros(lv.RESIDENT_DTYPE.itemsize, dtype=torch.uint8).pin_memory()
        # the turn-target candidate rows, resident for lv_turn's on-device pick
        self.perms_dev = None
        if perms is not None and len(perms):
            self.perms_dev = torch.from_numpy(np.ascontiguousarray(perms, dtype=np.int32)).to(pool.device)
            # a row's device address, without building a tensor view per turn
            self._perm_row = (self.perms_dev.data_ptr(), self.perms_dev.shape[1] * 4,
                              int(self.perms_dev.shape[1]))
        self.counters = dict(victims=0, pages_out=0, pages_in=0, preloads=0,
                             preload_skipped=0, turns=0, sync_loads=0, appended=0)
        self.bytes_moved = 0
        self.timer = None               # optional start(name) / stop(name, bytes) hooks
        self.last_readback_bytes = 0    # bytes of lists read back to the host by the last step
        # the load keys of a script's scattered-reload turns, resident on the device
        self._keys_dev, self._keys_row = None, {}
        if script is not None and order_fn is not None:
            self.stage_load_keys(script)

    def stage_load_keys(self, wl):
        """Uploads once the per-block load keys of every scattered-reload turn of the
        script ``wl``.  They are script input, like the events: a turn then passes a
        device pointer to its row instead of computing its keys and staging them."""
        sel = np.nonzero(np.asarray(wl.kind) == EV_TURN_SCATTER)[0]
        order_keys = sorted({int(k) for k in np.asarray(wl.a)[sel]})
        if not order_keys:
            return
        rows = np.stack([self._load_keys(k) for k in order_keys])
        self._keys_dev = torch.from_numpy(rows.view(np.int64)).to(self.pool.device)
        base, stride = self._keys_dev.data_ptr(), rows.shape[1] * 8
        self._keys_row = {k: base + i * stride for i, k in enumerate(order_keys)}

    # ------------------------------------------------------------- queries
    def free_budget(self) -> int:
        st = self.pool.stats()
        if st["error"]:
            raise lv.LvError(st["error"], "device error")
        return st["hbm_budget_pages"] - st["hbm_allocated"]

    def host_blocks(self, sid):
        return self.pool.blocks(sid, 1)

    def ctx_tokens(self, sid) -> int:
        return int(self.pool.get_sessions()["ctx_tokens"][sid])

    # ------------------------------------------------------------ movement
    def _device(self, sid, now_us, append_tokens, foreground, rec):
        pool = self.pool
        flags = 0 if foreground else lv.LV_RESIDENT_PRELOAD
        rec_bufs = self.record or self.on_append is not None
        old_ctx = self.ctx_tokens(sid) if (append_tokens and self.on_append is not None) else 0
        outs = (pool.victims, pool.slots, pool.blks, pool.pages, pool.app) if rec_bufs else (None,) * 5
        if self.timer:
            self.timer.start("resident")
        lv.lv_make_resident(pool.handle, sid, now_us, append_tokens, flags, -1, *outs,
                            self.res_h, pool.stream)
        # prepare, census, emit, plan (with the step's end), copy; or the append with the end
        pool.launches += 5 + pool.rank_extra + (1 if append_tokens else 0)
        if self.timer:
            self.timer.stop("resident", None)
        if not rec_bufs:
            return None
        pool.sync()
        r = self.res_h.numpy().view(lv.RESIDENT_DTYPE)[0]
        k, found, nv, nl, na, status = (int(r["k"]), int(r["n_found"]), int(r["n_victims"]),
                                        int(r["n_loaded"]), int(r["n_appended"]), int(r["status"]))
        if status == lv.LV_RESIDENT_NOTHING:
            return status
        rec["k"] = k
        if self.record:
            if k > 0:
                rec["victims"] = pool.victims[:found].cpu().numpy().astype(np.int64)
                self.last_readback_bytes += found * 12
            if nv:
                rec["slots"] = pool.slots[:nv].cpu().numpy().astype(np.int64)
                self.last_readback_bytes += nv * 4
            if nl:
                rec["in_blocks"] = pool.blks[:nl].cpu().numpy().astype(np.int64)
                rec["in_pages"] = pool.pages[:nl].cpu().numpy().astype(np.int64)
                self.last_readback_bytes += nl * 8
            if append_tokens:
                rec["append_pages"] = pool.app[:na].cpu().numpy().astype(np.int64)
        self.counters["victims"] += nv
        self.counters["pages_out"] += nv
        self.counters["pages_in"] += nl
        self.counters["appended"] += na
        self.bytes_moved += (nv + nl) * pool.J * pool.P
        if foreground and nl:
            self.counters["sync_loads"] += 1
        if status == lv.LV_RESIDENT_DONE and append_tokens and self.on_append is not None:
            self.on_append(sid, old_ctx, old_ctx + append_tokens)
        return status

    def _load_keys(self, order_key):
        return load_keys(self.order_fn, order_key, self.pool.max_blocks)

    def _device_turn(self, sid, row, now_us, append_tokens, reply_us, reply_units, rec,
                     load_keys=None):
        """One lv_turn: (pick,) turn begin, make resident, turn end -- no host round trip
        unless the decisions are recorded.  Returns the session id (-1 when not read back)."""
        pool = self.pool
        cand, n_cand = None, 0
        if sid < 0:
            base, stride, n_cand = self._perm_row
            cand = base + row * stride
        rec_bufs = self.record or (self.on_append is not None and append_tokens > 0)
        outs = (pool.victims, pool.slots, pool.blks, pool.pages, pool.app) if self.record else (None,) * 5
        lv.lv_turn(pool.handle, sid, now_us, append_tokens, reply_us, reply_units, outs, self.res_h,
                   cand, n_cand, pool.stream, lv.LV_RESIDENT_ASYNC_COPY if self.async_copy else 0,
                   load_keys)
        pool.launches += 1 if load_keys is not None else 0
        pool.launches += 5 + pool.rank_extra + (1 if sid < 0 else 0) + (1 if append_tokens else 0)
        if not rec_bufs:
            return sid
        pool.sync(raise_on_error=False)
        r = self.res_h.numpy().view(lv.RESIDENT_DTYPE)[0]
        sid = int(r["sid"])
        status = int(r["status"])
        if status == lv.LV_RESIDENT_FAILED:
            raise lv.LvError(pool.sync(raise_on_error=False) or lv.LV_ERR_NO_HBM, f"turn of session {sid}")
        k, found, nv, nl, na = (int(r["k"]), int(r["n_found"]), int(r["n_victims"]),
                                int(r["n_loaded"]), int(r["n_appended"]))
        rec["k"] = k
        if self.record:
            if k > 0:
                rec["victims"] = pool.victims[:found].cpu().numpy().astype(np.int64)
                self.last_readback_bytes += found * 12
            if nv:
                rec["slots"] = pool.slots[:nv].cpu().numpy().astype(np.int64)
                self.last_readback_bytes += nv * 4
            if nl:
                rec["in_blocks"] = pool.blks[:nl].cpu().numpy().astype(np.int64)
                rec["in_pages"] = pool.pages[:nl].cpu().numpy().astype(np.int64)
                self.last_readback_bytes += nl * 8
            if append_tokens:
                rec["append_pages"] = pool.app[:na].cpu().numpy().astype(np.int64)
        self.counters["victims"] += nv
        self.counters["pages_out"] += nv
        self.counters["pages_in"] += nl
        self.counters["appended"] += na
        self.bytes_moved += (nv + nl) * pool.J * pool.P
        if nl:
            self.counters["sync_loads"] += 1
        if append_tokens and self.on_append is not None:
            new_ctx = self.ctx_tokens(sid)
            self.on_append(sid, new_ctx - append_tokens, new_ctx)
        return sid

    def make_resident(self, sid, now_us, append_tokens, foreground, rec, order_key=None):
        if self.driver == "device" and order_key is None:
            status = self._device(sid, now_us, append_tokens, foreground, rec)
            if status == lv.LV_RESIDENT_FAILED:
                raise lv.LvError(self.pool.sync(raise_on_error=False) or lv.LV_ERR_NO_HBM,
                                 f"turn of session {sid}")
            return status
        pool = self.pool
        hblk, nh = self.host_blocks(sid)
        if order_key is not None and nh:
            order = np.asarray(self.order_fn(order_key, hblk.cpu().numpy()), dtype=np.int32)
            hblk = torch.from_numpy(order).to(pool.device)
        new_blocks = 0
        if append_tokens:
            ctx = self.ctx_tokens(sid)
            T = pool.T
            new_blocks = -(-(ctx + append_tokens) // T) - (-(-ctx // T))
        need = nh + new_blocks
        k = max(0, need - self.free_budget())
        rec["k"] = k
        if self.driver != "sequential":
            if not self._exchange(sid, now_us, k, hblk, nh, foreground, rec):
                return False
        else:
            if not self._sequential(sid, now_us, k, hblk, nh, foreground, rec):
                return False
        if append_tokens:
            old_ctx = self.ctx_tokens(sid)
            pages = pool.append(sid, append_tokens)
            if self.record:
                rec["append_pages"] = pages.cpu().numpy().astype(np.int64)
            self.counters["appended"] += int(pages.numel())
            if self.on_append is not None:
                self.on_append(sid, old_ctx, old_ctx + append_tokens)
        return True

    def _xmode(self):
        """The exchange's mode: staged exchanges are pipelined across calls when the
        manager runs with asynchronous copies (LV_MODE_ASYNC; pool.sync() joins)."""
        if self.async_copy and self.mode == lv.LV_MODE_STAGED:
            return self.mode | lv.LV_MODE_ASYNC
        return self.mode

    def _victims(self, sid, now_us, k, foreground, rec):
        flags = lv.LV_SELECT_FALLBACK if foreground else 0
        victims, n = self.pool.select(now_us, k, flags)
        if self.record:
            rec["victims"] = victims.cpu().numpy().astype(np.int64)
            self.last_readback_bytes += n * 12
        if n < k:
            if foreground:
                raise lv.LvError(lv.LV_ERR_NO_HBM, f"turn of session {sid} needs {k} victims, {n} found")
            return None, n
        return victims, n

    def _exchange(self, sid, now_us, k, hblk, nh, foreground, rec):
        pool = self.pool
        victims, n = None, 0
        if k > 0:
            victims, n = self._victims(sid, now_us, k, foreground, rec)
            if victims is None:
                return False
        if n == 0 and nh == 0:
            return True
        nbytes = (n + nh) * pool.J * pool.P
        if self.timer:
            self.timer.start("exchange")
        slots, pages = pool.exchange(victims, n, sid, hblk, nh, self._xmode())
        if self.timer:
            self.timer.stop("exchange", nbytes)
        if self.record:
            if n:
                rec["slots"] = slots.cpu().numpy().astype(np.int64)
                self.last_readback_bytes += n * 4
            if nh:
                rec["in_blocks"] = hblk.cpu().numpy().astype(np.int64)
                rec["in_pages"] = pages.cpu().numpy().astype(np.int64)
                self.last_readback_bytes += nh * 8
        self.counters["victims"] += n
        self.counters["pages_out"] += n
        self.counters["pages_in"] += nh
        self.bytes_moved += nbytes
        return True

    def _sequential(self, sid, now_us, k, hblk, nh, foreground, rec):
        pool = self.pool
        if k > 0:
            victims, n = self._victims(sid, now_us, k, foreground, rec)
            if victims is None:
                return False
            if self.timer:
                self.timer.start("swap_out")
            slots, commit = pool.swap_out(victims, n, self.mode)
            if self.timer:
                self.timer.stop("swap_out", n * pool.J * pool.P)
            pool.remap(commit, n)
            if self.record:
                rec["slots"] = slots.cpu().numpy().astype(np.int64)
                self.last_readback_bytes += n * 4
            self.counters["victims"] += n
            self.counters["pages_out"] += n
            self.bytes_moved += n * pool.J * pool.P
        if nh:
            if self.timer:
                self.timer.start("swap_in")
            pages, commit = pool.swap_in(sid, hblk, nh, self.mode)
            if self.timer:
                self.timer.stop("swap_in", nh * pool.J * pool.P)
            pool.remap(commit, nh)
            if self.record:
                rec["in_blocks"] = hblk.cpu().numpy().astype(np.int64)
                rec["in_pages"] = pages.cpu().numpy().astype(np.int64)
                self.last_readback_bytes += nh * 8
            self.counters["pages_in"] += nh
            self.bytes_moved += nh * pool.J * pool.P
        return True

    def preload(self, sid, now_us, rec):
        if self.pool.policy == lv.LV_POLICY_LRU:
            return              # the LRU baseline loads at turn start only
        if self.driver == "device" and self.admit is None:
            status = self._device(sid, now_us, 0, False, rec)
            if status == lv.LV_RESIDENT_DONE:
                self.counters["preloads"] += 1
                rec["preload"] = "done"
            elif status == lv.LV_RESIDENT_SKIPPED:
                self.counters["preload_skipped"] += 1
                rec["preload"] = "skipped"
            return
        _, nh = self.host_blocks(sid)
        if nh == 0:
            return
        if self.admit is not None and not self.admit(self, sid, now_us, nh):
            self.counters["preload_skipped"] += 1
            rec["preload"] = "skipped"
            return
        if self.make_resident(sid, now_us, 0, foreground=False, rec=rec):
            self.pool.events(_event(lv.LV_EV_PRELOADED, sid, now_us))
            self.counters["preloads"] += 1
            rec["preload"] = "done"
        else:
            self.counters["preload_skipped"] += 1
            rec["preload"] = "skipped"

    def evict(self, now_us, k, rec):
        """Free k pages now: the first k of the victim order (fewer if there are fewer)."""
        pool = self.pool
        if self.driver == "device":
            self._device_evict(now_us, k, rec)
            return
        victims, n = pool.select(now_us, k, 0)
        rec["k"] = int(k)
        if self.record:
            rec["victims"] = victims.cpu().numpy().astype(np.int64)
        if n == 0:
            return
        if self.driver == "sequential":
            slots, commit = pool.swap_out(victims, n, self.mode)
            pool.remap(commit, n)
        else:
            slots, _ = pool.exchange(victims, n, 0, None, 0, self._xmode())
        if self.record:
            rec["slots"] = slots.cpu().numpy().astype(np.int64)
        self.counters["victims"] += n
        self.counters["pages_out"] += n
        self.bytes_moved += n * pool.J * pool.P

    def _device_evict(self, now_us, k, rec):
        """lv_evict: ranking and eviction on the device, no host round trip unless the
        decisions are recorded."""
        pool = self.pool
        outs = (pool.victims, pool.slots) if self.record else (None, None)
        lv.lv_evict(pool.handle, now_us, int(k), lv.LV_RESIDENT_ASYNC_COPY if self.async_copy else 0,
                    *outs, self.res_h, pool.stream)
        pool.launches += 5 + pool.rank_extra
        rec["k"] = int(k)
        if not self.record:
            return
        pool.sync()
        r = self.res_h.numpy().view(lv.RESIDENT_DTYPE)[0]
        n = int(r["n_victims"])
        rec["victims"] = pool.victims[:int(r["n_found"])].cpu().numpy().astype(np.int64)
        if n:
            rec["slots"] = pool.slots[:n].cpu().numpy().astype(np.int64)
        self.counters["victims"] += n
        self.counters["pages_out"] += n
        self.bytes_moved += n * pool.J * pool.P

    def turn_target(self, row):
        _, host = self.pool.counts()
        for s in self.perms[row]:
            if host[int(s)] > 0:
                return int(s)
        return int(self.perms[row][0])

    # --------------------------------------------------------------- events
    def step(self, ev, index=None):
        t, kind, sid, a, b, c, d = (int(x) for x in ev)
        self.last_readback_bytes = 0
        rec = {"i": index, "t": t, "kind": kind}
        pool = self.pool
        if kind in _STATE_EVENT:
            pool.events(_event(_STATE_EVENT[kind], sid, t, a))
            if kind in (EV_SPEECH_START, EV_BARGE_IN):
                self.preload(sid, t, rec)
        elif kind in (EV_TURN, EV_TURN_ANY) and self.driver == "device":
            sid = self._device_turn(sid if kind == EV_TURN else -1, d, t, a, b, c, rec)
            self.counters["turns"] += 1
        elif kind == EV_TURN_SCATTER and self.driver == "device" and self.order_fn is not None:
            # the reload order is the script's scatter order, given as per-block keys
            keys = self._keys_row.get(a)        # the row's device address, if staged
            if keys is None:
                keys = self._load_keys(a)
            sid = self._device_turn(-1, d, t, 0, b, c, rec, load_keys=keys)
            self.counters["turns"] += 1
        elif kind in (EV_TURN, EV_TURN_ANY, EV_TURN_SCATTER):
            order_key = None
            if kind == EV_TURN_SCATTER:
                sid = self.turn_target(d)
                order_key, a = a, 0
            elif kind == EV_TURN_ANY:
                sid = self.turn_target(d)
            pool.events(_event(lv.LV_EV_TURN_BEGIN, sid, t))
            host_path = self.driver != "device" or order_key is not None
            if host_path and self.host_blocks(sid)[1]:
                self.counters["sync_loads"] += 1
            self.make_resident(sid, t, a, foreground=True, rec=rec, order_key=order_key)
            pool.events(_event(lv.LV_EV_TURN_END, sid, t, b, c))
            self.counters["turns"] += 1
        elif kind == EV_EVICT:
            self.evict(t, a, rec)
        else:
            raise ValueError(f"unknown script event kind {kind}")
        rec["sid"] = sid
        if self.rank_on == "all" or (self.rank_on == "turns" and kind in (EV_TURN, EV_TURN_ANY,
                                                                           EV_TURN_SCATTER)):
            order, n = pool.select(t, lv.LV_ALL, 0)
            rec["order"] = order.cpu().numpy().astype(np.int64)
        return rec
