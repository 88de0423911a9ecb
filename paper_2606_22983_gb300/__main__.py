"""Run one of the synthetic workloads through liblv on the current GPU.

    python -m paper_2606_22983_gb300 --workload mixed --seed 0 --driver device

Prints one JSON line: the workload's size, the bytes moved each way, the device time
of the turns (CUDA events around each turn's calls, with a host wait per turn so that
each turn's time is its own), the wall time, and the manager's and pool's counters.
Workloads: tiny, thinker, mixed, long, frag (see workloads.configs)."""
from __future__ import annotations

import argparse
import json
import time

import numpy as np


def main(argv=None) -> int:
    from workloads import CONFIG_NAMES, make_workload, pool_spec, scatter_order
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
    args = ap.parse_args(argv)

    import torch
    from . import build
    build()
    from .harness import fill_random, pool_for
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
            gm = KVManager(pool, perms=wl.perms, rank_on="none", record=True, driver=args.driver,
                           mode=args.mode, order_fn=scatter_order)
        n = wl.n_events if args.events <= 0 else min(args.events, wl.n_events)
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        turn_ms, load_ms = [], []
        w0 = time.perf_counter()
        for i in range(n):
            e = wl.event(i)
            if int(e[1]) not in (1, 2, 7):
                gm.step(e, i)
                continue
            torch.cuda.synchronize()
            a.record()
            rec = gm.step(e, i)
            b.record()
            torch.cuda.synchronize()
            ms = a.elapsed_time(b)
            turn_ms.append(ms)
            if len(rec.get("in_blocks", ())):
                load_ms.append(ms)
        assert pool.sync(raise_on_error=False) == 0
        wall = time.perf_counter() - w0
        st = pool.stats()
        q = lambda xs, f: round(float(np.percentile(xs, f)), 3) if xs else None
        print(json.dumps({
            "workload": args.workload, "seed": args.seed, "events": n, "driver": args.driver,
            "mode": args.mode, "tiers": args.tiers, "policy": args.policy,
            "controller_link_bytes_per_us": args.controller or None,
            "sessions": spec.n_sessions, "hbm_budget_pages": spec.hbm_budget_pages,
            "host_pages": wl.spec.host_pages, "page_bytes": pool.J * pool.P,
            "turns": len(turn_ms), "turns_loading_on_path": len(load_ms),
            "turn_ms": {"mean": round(float(np.mean(turn_ms)), 3) if turn_ms else None,
                        "p50": q(turn_ms, 50), "p90": q(turn_ms, 90), "max": q(turn_ms, 100)},
            "gb_out": round(st["bytes_out"] / 1e9, 3), "gb_in": round(st["bytes_in"] / 1e9, 3),
            "wall_s": round(wall, 2), "manager": gm.counters,
            "pool": {k: st[k] for k in ("selects", "victims", "shortfalls", "pages_out", "pages_in",
                                        "remap_entries", "appended_pages", "preloads",
                                        "preloads_skipped", "clean_out", "clean_dropped")}}))
    finally:
        torch.cuda.synchronize()
        pool.close()
    return 0


if __name__ == "__main__":
    raise SystemExit(main())
