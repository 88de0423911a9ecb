"""Run one of the synthetic workloads through liblv on the current GPU.

    python -m paper_2606_22983_gb300 --workload mixed --seed 0 --driver device

Prints one JSON line: the workload's size, the bytes moved each way, the device time of
every event that moved bytes (CUDA events around each event's calls, with a host wait per
event so that each event's time is its own), the turns' latencies, the wall time, the
pool's counters (and, with --record, the manager's, whose decision read-back then falls
inside the timed events), and the host link's peaks measured afterwards in the same
process.  ``link_frac`` compares the moving events' time with the link's best time for
each event's own mix of bytes out and in: max(out / d2h, in / h2d, (out + in) / bidir).
Workloads: tiny, thinker, mixed, long, frag (see workloads.configs)."""
from __future__ import annotations

import argparse
import json
import time

import numpy as np


def main(argv=None) -> int:
    from workloads import CONFIG_NAMES, make_workload, pool_spec, scatter_order
    from workloads.scripts import EVENT_NAMES
    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("--workload", choices=CONFIG_NAMES, default="tiny")
    ap.add_argument("--seed", type=int, default=0)
    ap.add_argument("--driver", choices=("device", "exchange", "sequential"), default="device")
    ap.add_argument("--mode", type=int, default=0, help="0 auto, 1 zero-copy, 2 staged")
    ap.add_argument("--tiers", type=int, choices=(0, 1), default=0, help="1: inclusive tiers")
    ap.add_argument("--policy", type=int, choices=(0, 1), default=0, help="1: LRU baseline")
    ap.add_argument("--events", type=int, default=0, help="run only the first N events")
    ap.add_argument("--controller", type=int, default=0, metavar="BYTES_PER_US",
                    help="preloads through the Section 5.2 controller with this modelled link "
                         "(host-driven exchange driver; 0: every preload admitted)")
    ap.add_argument("--cap-pages", type=int, default=-1, help="the controller's protected-KV cap")
    ap.add_argument("--record", action="store_true",
                    help="read every decision back to the host (inside the timed events) and "
                         "report the manager's counters")
    args = ap.parse_args(argv)

    import torch
    from . import build
    build()
    from .harness import fill_random, link_peaks, pool_for
    from .manager import KVManager

    spec = pool_spec(args.workload).with_(tiers=args.tiers, policy=args.policy)
    wl = make_workload(args.workload, args.seed, spec=spec)
    pool = pool_for(wl)
    try:
        fill_random(pool, args.seed)
        if args.controller > 0:
            from .controller import ControlledKVManager
            gm = ControlledKVManager(pool, link_bytes_per_us=args.controller,
                                     cap_pages=None if args.cap_pages < 0 else args.cap_pages,
                                     perms=wl.perms, mode=args.mode, order_fn=scatter_order)
        else:
            gm = KVManager(pool, perms=wl.perms, rank_on="none", record=args.record, driver=args.driver,
                           mode=args.mode, order_fn=scatter_order)
        n = wl.n_events if args.events <= 0 else min(args.events, wl.n_events)
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        page = pool.J * pool.P
        turn_ms, load_ms, moves = [], [], []      # moves: (ms, bytes out, bytes in)
        st0 = pool.stats()
        w0 = time.perf_counter()
        for i in range(n):
            e = wl.event(i)
            torch.cuda.synchronize()
            a.record()
            gm.step(e, i)
            b.record()
            torch.cuda.synchronize()
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
        st = pool.stats()
        mv = np.array(moves, dtype=np.float64).reshape(-1, 4)
        mean_move = float(mv[:, 1:].sum(axis=1).mean()) if len(mv) else 0.0
        nbytes = int(min(max(mean_move / 2, 1 << 26), 1 << 30, pool.kv.numel(),
                         pool.host.size // 2 if pool.host is not None else 0))
        nbytes = nbytes // 4096 * 4096
        peaks = link_peaks(pool, nbytes) if nbytes > 0 else {}
        link = None
        if len(mv) and "bidir" in peaks:
            best_s = np.maximum(np.maximum(mv[:, 1] / (peaks["d2h"] * 1e9), mv[:, 2] / (peaks["h2d"] * 1e9)),
                                (mv[:, 1] + mv[:, 2]) / (peaks["bidir"] * 1e9))
            t_s = mv[:, 0].sum() / 1e3
            link = {"moving_events": int(len(mv)), "device_s": round(float(t_s), 4),
                    "gbs": round(float(mv[:, 1:3].sum() / t_s / 1e9), 1),
                    "link_best_s": round(float(best_s.sum()), 4),
                    "link_frac": round(float(best_s.sum() / t_s), 3),
                    "peaks_gbs": {k: round(v, 1) for k, v in peaks.items()},
                    "peak_copy_bytes": nbytes, "by_event_kind": {}}
            for kind in sorted(set(mv[:, 3].astype(int).tolist())):
                sel = mv[:, 3] == kind
                ts = float(mv[sel, 0].sum()) / 1e3
                link["by_event_kind"][EVENT_NAMES.get(kind, str(kind))] = {
                    "events": int(sel.sum()), "device_s": round(ts, 4),
                    "gb_out": round(float(mv[sel, 1].sum()) / 1e9, 3),
                    "gb_in": round(float(mv[sel, 2].sum()) / 1e9, 3),
                    "link_frac": round(float(best_s[sel].sum()) / ts, 3) if ts > 0 else None}
        q = lambda xs, f: round(float(np.percentile(xs, f)), 3) if xs else None
        print(json.dumps({
            "workload": args.workload, "seed": args.seed, "events": n, "driver": args.driver,
            "mode": args.mode, "tiers": args.tiers, "policy": args.policy,
            "controller_link_bytes_per_us": args.controller or None,
            "sessions": spec.n_sessions, "hbm_budget_pages": spec.hbm_budget_pages,
            "host_pages": wl.spec.host_pages, "page_bytes": page,
            "moves": link,
            "turns": len(turn_ms), "turns_loading_on_path": len(load_ms),
            "turn_ms": {"mean": round(float(np.mean(turn_ms)), 3) if turn_ms else None,
                        "p50": q(turn_ms, 50), "p90": q(turn_ms, 90), "max": q(turn_ms, 100)},
            "gb_out": round(st["bytes_out"] / 1e9, 3), "gb_in": round(st["bytes_in"] / 1e9, 3),
            "wall_s": round(wall, 2), "manager": gm.counters if args.record or args.controller > 0 else None,
            "pool": {k: st[k] for k in ("selects", "victims", "shortfalls", "pages_out", "pages_in",
                                        "remap_entries", "appended_pages", "preloads",
                                        "preloads_skipped", "clean_out", "clean_dropped")}}))
    finally:
        torch.cuda.synchronize()
        pool.close()
    return 0


if __name__ == "__main__":
    raise SystemExit(main())
