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


def main(argv=None) -> int:
    from workloads import CONFIG_NAMES, host_tier_limit, make_workload, pool_spec, scatter_order
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
    from .runner import link_summary, peak_bytes, quantiles, run_events

    spec = pool_spec(args.workload).with_(tiers=args.tiers, policy=args.policy)
    wl = make_workload(args.workload, args.seed, spec=spec, host_limit=host_tier_limit())
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
                           mode=args.mode, order_fn=scatter_order, script=wl)
        n = wl.n_events if args.events <= 0 else min(args.events, wl.n_events)
        copies = {}
        moves, turn_ms, load_ms, wall = run_events(torch, pool, gm, wl, n, copy_times=copies)
        nbytes = peak_bytes(pool, moves)
        peaks = link_peaks(pool, nbytes) if nbytes > 0 else {}
        link = link_summary(moves, peaks, EVENT_NAMES)
        if link is not None:
            link["peak_copy_bytes"] = nbytes
        st = pool.stats()
        print(json.dumps({
            "workload": args.workload, "seed": args.seed, "events": n, "driver": args.driver,
            "mode": args.mode, "tiers": args.tiers, "policy": args.policy,
            "controller_link_bytes_per_us": args.controller or None,
            "sessions": wl.spec.n_sessions, "sizing": wl.meta.get("sizing"),
            "hbm_budget_pages": spec.hbm_budget_pages,
            "host_pages": wl.spec.host_pages, "page_bytes": pool.J * pool.P,
            "moves": link, "copy_kernels": copies,
            "turns": len(turn_ms), "turns_loading_on_path": len(load_ms),
            "turn_ms": quantiles(turn_ms),
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
