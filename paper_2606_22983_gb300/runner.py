"""Runs a seeded workload script through liblv one event at a time and reports how
fast each kind of event moved KV over the host link.

Each event's calls are bracketed by CUDA events on the pool's stream and followed by a
host wait, so an event's device time is its own (no overlap between events).  Bytes
come from the pool's counters.  The link fraction of a set of events is the link's
best time for each event's own mix of bytes out and in, summed, over their measured
time: max(out / d2h, in / h2d, (out + in) / bidir) per event, with the peaks of
contiguous page-locked copies measured in the same process (``harness.link_peaks``).
"""
from __future__ import annotations

import time

import numpy as np


def run_events(torch, pool, gm, wl, n, before_event=None, copy_times=None):
    """Events 0..n of ``wl`` through ``gm``; returns per-event moves
    [(ms, bytes out, bytes in, kind)], the turns' times and the wall time.
    ``before_event(i)`` runs before each event is issued (a co-running consumer
    tops up its queue there).  ``copy_times`` (a dict) receives the copy kernels'
    launches and summed device time (liblv's timing instrument, CUDA events around
    each copy launch)."""
    from . import lv
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    turn_ms, load_ms, moves = [], [], []
    if copy_times is not None:
        lv.lv_timing_read(pool.handle, reset=True)
        lv.lv_timing_enable(pool.handle, True)
    st0 = pool.stats()
    w0 = time.perf_counter()
    for i in range(n):
        e = wl.event(i)
        if before_event is not None:
            before_event(i)
        a.record()
        gm.step(e, i)
        b.record()
        b.synchronize()
        ms = a.elapsed_time(b)
        st1 = pool.stats()
        out, inn = st1["bytes_out"] - st0["bytes_out"], st1["bytes_in"] - st0["bytes_in"]
        st0 = st1
        if out or inn:
            moves.append((ms, out, inn, int(e[1])))
        if int(e[1]) in (1, 2, 7):
            turn_ms.append(ms)
            if inn:
                load_ms.append(ms)
    assert pool.sync(raise_on_error=False) == 0
    wall = time.perf_counter() - w0
    if copy_times is not None:
        lv.lv_timing_enable(pool.handle, False)
        for name, t in lv.lv_timing_read(pool.handle, reset=True).items():
            if t["launches"]:
                copy_times[name] = {"launches": t["launches"], "total_s": round(t["total_ms"] / 1e3, 4)}
    return moves, turn_ms, load_ms, wall


def peak_bytes(pool, moves):
    """Byte count for the link-peak copies: half the mean move, within 64 MiB..1 GiB
    and what the pool's HBM and host arrays hold."""
    mv = np.array(moves, dtype=np.float64).reshape(-1, 4)
    mean_move = float(mv[:, 1:3].sum(axis=1).mean()) if len(mv) else 0.0
    nbytes = int(min(max(mean_move / 2, 1 << 26), 1 << 30, pool.kv.numel(),
                     pool.host.size // 2 if pool.host is not None else 0))
    return nbytes // 4096 * 4096


def link_summary(moves, peaks, event_names):
    """GB/s and link fraction of all moving events, by event kind, and by direction:
    events that only offloaded (against the D2H peak), only reloaded (against the
    H2D peak), or did both (against the mix's best time)."""
    mv = np.array(moves, dtype=np.float64).reshape(-1, 4)
    if not len(mv) or "bidir" not in peaks:
        return None
    d2h, h2d, bi = peaks["d2h"] * 1e9, peaks["h2d"] * 1e9, peaks["bidir"] * 1e9
    best_s = np.maximum(np.maximum(mv[:, 1] / d2h, mv[:, 2] / h2d), (mv[:, 1] + mv[:, 2]) / bi)
    t_s = mv[:, 0] / 1e3

    def part(sel):
        ts = float(t_s[sel].sum())
        if ts <= 0:
            return None
        return {"events": int(sel.sum()), "device_s": round(ts, 4),
                "gb_out": round(float(mv[sel, 1].sum()) / 1e9, 3),
                "gb_in": round(float(mv[sel, 2].sum()) / 1e9, 3),
                "gbs": round(float(mv[sel, 1:3].sum()) / ts / 1e9, 1),
                "link_best_s": round(float(best_s[sel].sum()), 6),
                "link_frac": round(float(best_s[sel].sum()) / ts, 3)}

    out = part(np.ones(len(mv), bool))
    out["peaks_gbs"] = {k: round(v, 1) for k, v in peaks.items()}
    out["by_event_kind"] = {}
    for kind in sorted(set(mv[:, 3].astype(int).tolist())):
        out["by_event_kind"][event_names.get(kind, str(kind))] = part(mv[:, 3] == kind)
    out["by_direction"] = {"offload_only": part((mv[:, 2] == 0) & (mv[:, 1] > 0)),
                           "reload_only": part((mv[:, 1] == 0) & (mv[:, 2] > 0)),
                           "both": part((mv[:, 1] > 0) & (mv[:, 2] > 0))}
    return out


def quantiles(xs):
    q = lambda f: round(float(np.percentile(xs, f)), 3) if xs else None
    return {"mean": round(float(np.mean(xs)), 3) if xs else None, "p50": q(50), "p90": q(90),
            "max": q(100)}
