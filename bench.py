#!/usr/bin/env python
"""KV reload/offload throughput of the interaction-aware swap path on GB300.

One step = one turn of the thinker-shaped workload (48 layers, 4 KV heads x
128, 16-token pages of 1.5 MiB, 64 sessions with log-uniform 2k-16k token
contexts, 40 GB HBM budget): playback reports for every session, then the
turn's session is made fully resident -- next-use ranking (census, then
rank and top-k emission), host-slot allocation, swap-out, commit, HBM-page
allocation, swap-in, commit -- in one lv_turn with no host round trip.  ``value`` is the payload moved over the host link in both
directions per second (GB/s, 1e9 B) with every input resident before timing;
``e2e`` is the same through the C ABI with host buffers (every step copies its
event batch in from page-locked host memory and reads the turn's result back
into it), timed on the host clock.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

N > 1 runs N independent replicas (one pool per GPU, one process per GPU, no
collective on the data path); ``value`` is then the sum over replicas divided
by the slowest rank's time.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import select
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "KV reload+offload payload GB/s on 1 GB300 (thinker-shaped pages, 40 GB HBM budget)"
UNIT = "GB/s"
WORKLOAD = "thinker"


def _hbm_peak():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return float(json.load(f)["hbm_gbs"])
    except (OSError, KeyError, ValueError):
        return 6800.0          # the profiling recipe's fallback HBM figure


HBM_PEAK = _hbm_peak()


def _dist():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def aggregate(per_rank_bytes, per_rank_seconds):
    """Whole-job throughput: all ranks' bytes over the slowest rank's time."""
    t = max(per_rank_seconds)
    return (sum(per_rank_bytes) / t) if t > 0 else 0.0


# ------------------------------------------------------------------ clocks
class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.gpu = gpu_index
        self.proc = None
        self.first = ""

    def start(self, wait_s=10.0):
        """Starts sampling and returns once the first sample is in (or after wait_s), so
        that nvidia-smi's start-up (NVML initialisation) is over before the caller's
        timed region begins."""
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "50"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except (OSError, ValueError):
            self.proc = None
            return
        ready, _, _ = select.select([self.proc.stdout], [], [], wait_s)
        if ready:
            self.first = self.proc.stdout.readline()

    def stop(self):
        if not self.proc:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
            out, _ = self.proc.communicate()
        if not out.strip():       # nothing after the start-up sample: report that one
            out = self.first
        sm, mx, reasons = [], [], set()
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        for line in out.strip().splitlines():
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                mx.append(float(parts[2]))
            except ValueError:
                continue
            for n, v in zip(names, parts[5:9]):
                if v.lower() == "active":
                    reasons.add(n)
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None, "reasons": sorted(reasons),
                "samples": len(sm)}


# --------------------------------------------------------------- our arm
def run_turns(gm, wl, lo, hi, dev_events=None):
    """Turns lo..hi of a turn-driven script (playback batch, then the turn)."""
    from paper_2606_22983_gb300 import lv
    S = wl.spec.n_sessions
    per_turn = S + 1
    for i in range(lo, hi):
        base = i * per_turn
        if dev_events is not None:
            lv.lv_session_events(gm.pool.handle, dev_events[i], S, gm.pool.stream)
            gm.pool.launches += 1
        else:
            ev = np.zeros(S, dtype=lv.EVENT_DTYPE)
            ev["kind"], ev["sid"], ev["t_us"], ev["a"] = (lv.LV_EV_PLAYBACK, wl.sid[base:base + S],
                                                          int(wl.t_us[base]), wl.a[base:base + S])
            gm.pool.events(ev)
        gm.step(wl.event(base + S), base + S)


def _moved_pages(pool):
    """Pages whose bytes crossed the host link (an eviction that found a clean
    copy under inclusive tiers moves none): (both ways, out, in)."""
    st = pool.stats()
    page = pool.J * pool.P
    out, inn = st["bytes_out"] // page, st["bytes_in"] // page
    return out + inn, out, inn


def ours(args, torch):
    from paper_2606_22983_gb300 import build, lv
    build()
    from paper_2606_22983_gb300.harness import fill_random, link_peaks, pool_for
    from paper_2606_22983_gb300.manager import KVManager
    from workloads import make_workload

    ws, rank, local = _dist()
    torch.cuda.set_device(local)
    dist = None
    if ws > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    K, W = args.steps, args.warmup
    KO = OVERLAP_TURNS if (args.overlap and args.driver == "device") else 0
    wl = _arm_spec(args, args.seed + rank)
    pool = pool_for(wl)
    fill_random(pool, args.seed + rank)
    page_bytes = pool.J * pool.P
    gm = KVManager(pool, perms=wl.perms, rank_on="none", mode=args.mode, record=False,
                   driver=args.driver, async_copy=args.async_copy)
    S = wl.spec.n_sessions
    # the PLAYBACK batches of the device-timed pass, resident before timing
    dev_events = []
    for i in range(W + K):
        base = i * (S + 1)
        ev = np.zeros(S, dtype=lv.EVENT_DTYPE)
        ev["kind"], ev["sid"], ev["t_us"], ev["a"] = (lv.LV_EV_PLAYBACK, wl.sid[base:base + S],
                                                      int(wl.t_us[base]), wl.a[base:base + S])
        dev_events.append(torch.from_numpy(ev.view(np.uint8).copy()).to(pool.device))
    torch.cuda.synchronize()

    # the clock sampler's start-up (NVML initialisation) is over before the warm-up, and
    # it samples throughout the timed region
    clocks = ClockSampler(local)
    clocks.start()
    run_turns(gm, wl, 0, W, dev_events)                         # warm-up
    pool.sync()
    p0, o0, i0 = _moved_pages(pool)
    lv.lv_timing_read(pool.handle, reset=True)
    lv.lv_timing_enable(pool.handle, True)
    if dist:
        dist.barrier()
    torch.cuda.synchronize()
    l0 = pool.launches
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    t0.record()
    run_turns(gm, wl, W, W + K, dev_events)
    lv.lv_join(pool.handle, pool.stream)       # every turn's copy is inside the timed region
    t1.record()
    torch.cuda.synchronize()
    if dist:
        dist.barrier()
    launches = pool.launches - l0
    clk = clocks.stop()
    lv.lv_timing_enable(pool.handle, False)
    timing = lv.lv_timing_read(pool.handle, reset=True)
    dev_s = t0.elapsed_time(t1) / 1e3
    assert pool.sync(raise_on_error=False) == 0, "device error during the timed turns"
    p1, o1, i1 = _moved_pages(pool)
    moved = (p1 - p0) * page_bytes
    kern = {}
    for name, t in timing.items():
        if t["launches"]:
            pages = {"swap_out": o1 - o0, "swap_in": i1 - i0, "pack": o1 - o0,
                     "unpack": i1 - i0}.get(name, p1 - p0)
            nb = pages * page_bytes
            kern[name] = {"launches": t["launches"], "total_ms": t["total_ms"],
                          "avg_ms": t["total_ms"] / t["launches"],
                          "bytes_per_launch": nb / t["launches"],
                          "gbs": nb / 1e9 / (t["total_ms"] / 1e3)}

    # e2e: K further turns through the public API from host buffers, timed on the host
    # clock: every step moves its event batch from page-locked host memory to the device
    # and the turn's result (lv_resident_result) back into page-locked host memory, in
    # stream order (the library's kernels read and write page-locked arguments in place,
    # over the host link); the results are checked after the final join
    gm.record = False
    ev_h = torch.empty((K, S * lv.EVENT_DTYPE.itemsize), dtype=torch.uint8).pin_memory()
    for j, i in enumerate(range(W + K, W + 2 * K)):
        base = i * (S + 1)
        ev = ev_h[j].numpy().view(lv.EVENT_DTYPE)
        ev["kind"], ev["sid"], ev["t_us"], ev["a"], ev["b"] = (
            lv.LV_EV_PLAYBACK, wl.sid[base:base + S], int(wl.t_us[base]), wl.a[base:base + S], 0)
    res_h = torch.zeros((K, lv.RESIDENT_DTYPE.itemsize), dtype=torch.uint8).pin_memory()
    own_res = gm.res_h
    h2d = K * S * lv.EVENT_DTYPE.itemsize
    d2h = K * lv.RESIDENT_DTYPE.itemsize
    torch.cuda.synchronize()
    q0, qo0, qi0 = _moved_pages(pool)
    w0 = time.perf_counter()
    for j, i in enumerate(range(W + K, W + 2 * K)):
        lv.lv_session_events(pool.handle, ev_h[j], S, pool.stream)
        gm.res_h = res_h[j]
        gm.step(wl.event(i * (S + 1) + S), i * (S + 1) + S)
    lv.lv_join(pool.handle, pool.stream)
    torch.cuda.synchronize()
    e2e_s = time.perf_counter() - w0
    gm.res_h = own_res
    status = res_h.numpy().view(lv.RESIDENT_DTYPE)["status"]
    assert (status == lv.LV_RESIDENT_DONE).all(), "a turn of the end-to-end pass failed"
    q1, qo1, qi1 = _moved_pages(pool)
    moved_e2e = (q1 - q0) * page_bytes
    e2e_out, e2e_in = (qo1 - qo0) * page_bytes, (qi1 - qi0) * page_bytes
    if dist:
        tt = torch.tensor([dev_s, e2e_s, moved, moved_e2e], dtype=torch.float64, device="cuda")
        gathered = [torch.zeros_like(tt) for _ in range(ws)]
        dist.all_gather(gathered, tt)
        g = torch.stack(gathered).cpu().numpy()
        value = aggregate(g[:, 2], g[:, 0]) / 1e9
        e2e_value = aggregate(g[:, 3], g[:, 1]) / 1e9
        t_max = float(g[:, 0].max())
    else:
        value = moved / dev_s / 1e9
        e2e_value = moved_e2e / e2e_s / 1e9
        t_max = dev_s

    line = None
    if rank == 0:
        mean_turn = moved / K / 2
        peaks = link_peaks(pool, int(min(mean_turn, 1 << 30)) // 4096 * 4096)
        # roofline of the dominant kernel (longest total time) among the link-bound copies;
        # the staged path's pack/unpack are HBM-bound and reported against the HBM peak
        link_kern = {n: d for n, d in kern.items() if n in ("swap_out", "swap_in", "exchange")}
        hbm_kern = {}
        for n in ("pack", "unpack"):
            if n in kern:
                rw = 2 * kern[n]["gbs"]          # each payload byte is read and written in HBM
                hbm_kern[n] = {"achieved_gbs": round(rw, 1), "peak_gbs": HBM_PEAK,
                               "frac": round(rw / HBM_PEAK, 3), "launches": kern[n]["launches"],
                               "avg_ms": round(kern[n]["avg_ms"], 4)}
        if link_kern:
            dom = max(link_kern, key=lambda n: kern[n]["total_ms"])
            dk = kern[dom]
            peak = {"swap_out": peaks["d2h"], "swap_in": peaks["h2d"]}.get(dom)
            peak_dir = {"swap_out": "D2H", "swap_in": "H2D"}.get(dom)
            if peak is None:
                # the exchange moves O bytes out and I in at once: the link's best time for
                # that mix is max(O / d2h, I / h2d, (O + I) / bidir)
                O, I = (o1 - o0) * page_bytes, (i1 - i0) * page_bytes
                best_s = max(O / peaks["d2h"], I / peaks["h2d"], (O + I) / peaks["bidir"])
                peak = (O + I) / best_s if best_s > 0 else peaks["bidir"]
                peak_dir = (f"D2H and H2D concurrently, weighted by this run's mix: "
                            f"{O / 1e9:.1f} GB out, {I / 1e9:.1f} GB in")
            # the profiled DRAM ratio holds for the exclusive tiers' two-way mix only
            traffic = _profiled_traffic(dom, dk["bytes_per_launch"]) if args.tiers == 0 else None
            roof = {"kernel": dom, "bound": "host_link", "achieved": round(dk["gbs"], 1),
                    "peak": round(peak, 1), "unit": "GB/s", "frac": round(dk["gbs"] / peak, 3),
                    "traffic": traffic,
                    "peak_source": "same-run contiguous page-locked cudaMemcpyAsync "
                                   f"({peak_dir}, mean-turn byte count)"}
        else:   # staged: the copy engines carry the link traffic, the kernels are HBM-bound
            dom = max(hbm_kern, key=lambda n: kern[n]["total_ms"])
            h = hbm_kern[dom]
            roof = {"kernel": dom, "bound": "hbm", "achieved": h["achieved_gbs"], "peak": HBM_PEAK,
                    "unit": "GB/s", "frac": h["frac"],
                    "traffic": _profiled_traffic(dom, 2 * kern[dom]["bytes_per_launch"]),
                    "peak_source": "MEASURED_PEAKS.json hbm_gbs (of measured)"}
        line = {
            "metric": METRIC, "value": round(value, 3), "unit": UNIT, "n_gpus": ws,
            "steps": K, "warmup": W, "ms_per_step": round(t_max * 1e3 / K, 4),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "u8", "data": "synthetic",
            "config": arm_config(args, wl.spec, ws),
            "mean_turn_mb_each_way": round(mean_turn / 1e6, 1),
            "blocks_per_s": round(moved / page_bytes / t_max, 1),
            "turns_per_s": round(K * ws / t_max, 2),
            "link_peak_gbs": {k: round(v, 1) for k, v in peaks.items()},
            "link_frac": round(value / peaks["bidir"], 3) if "bidir" in peaks else None,
            "roofline": roof,
            "kernels": {n: {k: round(v, 3) for k, v in d.items()} for n, d in kern.items()},
            "in_turn_hbm_kernels": hbm_kern or None,
            "e2e": {"value": round(e2e_value, 3), "unit": UNIT,
                    "h2d_bytes_per_step": int(h2d / K), "d2h_bytes_per_step": int(d2h / K),
                    # its own turns (the K after the device-timed ones) and their link roofline
                    "mean_turn_mb_each_way": round(moved_e2e / K / 2 / 1e6, 1),
                    "link_frac": (round(max(e2e_out / peaks["d2h"], e2e_in / peaks["h2d"],
                                            moved_e2e / peaks["bidir"]) / 1e9 / e2e_s, 3)
                                  if "bidir" in peaks and ws == 1 else None)},
            "gpu_launches": int(launches),
            "clocks": clk,
        }
    if line is not None and KO:
        line["overlap"] = overlap_measure(torch, pool, wl, W + 2 * K, KO)
    if line is not None and args.directions:
        line["directions"] = direction_legs(torch, pool, int(wl.t_us[-1]) + 1_000_000)
    if line is not None and args.micro:
        micro = kernel_micro(torch, pool, args.seed)
        line["ranker"] = micro.pop("ranker")
        line["scheduler"] = micro.pop("scheduler")
        line["hbm_kernels"] = micro
    pool.close()
    if line is not None and args.five:
        line["workloads"] = five_workloads(torch, args.seed)
    if line is not None and args.cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(args, args.cpu_seconds, args.seed)
    if dist:
        dist.destroy_process_group()
    return line


OVERLAP_TURNS = 40
# The commit's algorithmic bytes per entry: the entry 12; read and write of the table
# word 4+4 and of the new location's owner word 4+4; write of the old location's owner
# word 4; read and write of the old location's bitmap word 4+4.  The per-block epoch
# mark (duplicate detection) and the read of the old location's owner word (a
# consistency check) are the implementation's own and are not counted.
REMAP_BYTES_PER_ENTRY = 40


class ChecksumConsumer:
    """Stands in for the engine's attention reads of resident KV: lv_page_checksums
    over n resident pages (HBM-bound, every byte read once) issued on its own stream
    through a second liblv pool over the same KV arrays, so that its reads never wait
    for the first pool's copies.  A call reads 512 pages (0.8 GB, about 0.11 ms alone),
    the length of a serving step's larger kernels, so that its SMs are handed back as
    often as a serving engine's would be; ``top_up`` keeps ``depth`` calls queued, so it
    runs without gaps while the other work is issued."""

    def __init__(self, torch, pool, n_pages=512, seed=0, depth=24):
        from paper_2606_22983_gb300.pool import KVPool
        self.torch = torch
        self.stream = torch.cuda.Stream(device=pool.device)
        elems = pool.P // 2                       # bf16 elements of one sub-page
        self.cp = KVPool(layers=pool.L, kv_heads=1, head_dim=elems // pool.T, page_tokens=pool.T,
                         max_sessions=1, max_blocks=1, hbm_pages=pool.hbm_pages, hbm_budget_pages=1,
                         host_pages=0, device=pool.device, stream=self.stream, kv=pool.kv)
        g = torch.Generator(device=pool.device).manual_seed(seed)
        n = min(n_pages, pool.hbm_pages)
        self.pages = torch.randperm(pool.hbm_pages, generator=g, device=pool.device)[:n].to(torch.int32)
        self.n = n
        self.sums = torch.empty(n, dtype=torch.int64, device=pool.device)
        self.bytes_per_call = n * pool.J * pool.P
        self.depth = depth
        self.pending = []
        self.ends = []
        self.calls = 0
        self.call_ms = 1.0

    def describe(self):
        return (f"lv_page_checksums over {self.n} resident pages ({self.bytes_per_call / 1e9:.1f} GB "
                f"read per call, {self.depth} calls kept queued), its own stream and pool over the "
                "same KV arrays")

    def issue(self):
        from paper_2606_22983_gb300 import lv
        lv.lv_page_checksums(self.cp.handle, self.pages, self.n, self.sums, self.stream)
        ev = self.torch.cuda.Event(enable_timing=True)
        ev.record(self.stream)
        self.pending.append(ev)
        self.ends.append(ev)
        self.calls += 1

    def start(self):
        """Starts a window: the consumer's calls from now on are counted."""
        self.ends = []
        self.top_up()

    def keep_busy_until(self, ev):
        """Keeps calls queued until event ``ev`` (recorded on another stream) has
        completed, then returns the end events of the window's calls."""
        while not ev.query():
            self.top_up()
            time.sleep(0.0002)
        self.top_up()
        return list(self.ends)

    def rate_within(self, ends, t0, t1):
        """The consumer's GB/s within the window [t0, t1] of another stream (after a
        synchronize): calls completed in it, the call running at t1 counted by the
        part of it inside the window; and whether the consumer ran past t1."""
        T = t0.elapsed_time(t1)
        x = [t0.elapsed_time(e) for e in ends]
        done = sum(1 for v in x if 0 < v <= T)
        later = [v for v in x if v > T]
        if later:
            prev = max([v for v in x if v <= T], default=0.0)
            span = later[0] - prev
            if span > 0:
                done += (T - prev) / span
        return done * self.bytes_per_call / (T / 1e3) / 1e9, bool(later)

    def top_up(self, *_):
        self.pending = [e for e in self.pending if not e.query()]
        while len(self.pending) < self.depth:
            self.issue()

    def alone_gbs(self, reps=10):
        torch = self.torch
        for _ in range(2):
            self.issue()
        torch.cuda.synchronize()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(self.stream)
        for _ in range(reps):
            self.issue()
        b.record(self.stream)
        torch.cuda.synchronize()
        self.call_ms = a.elapsed_time(b) / reps
        return self.bytes_per_call * reps / (a.elapsed_time(b) / 1e3) / 1e9

    def window(self):
        """Starts counting: returns a closure that, after a synchronize, gives the
        consumer's GB/s over the window."""
        torch = self.torch
        a = torch.cuda.Event(enable_timing=True)
        a.record(self.stream)
        c0 = self.calls

        def done():
            b = torch.cuda.Event(enable_timing=True)
            b.record(self.stream)
            torch.cuda.synchronize()
            return (self.calls - c0) * self.bytes_per_call / (a.elapsed_time(b) / 1e3) / 1e9
        return done

    def close(self):
        self.torch.cuda.synchronize()
        self.cp.close()


def overlap_measure(torch, pool, wl, first_turn, n_turns):
    """Config 3's overlap of KV movement with serving work: a consumer reading resident
    KV at HBM speed (lv_page_checksums over 4096 resident pages, 6.4 GB per call, on
    its own stream) runs alone, then throughout n_turns thinker turns moved by the
    zero-copy device-driven path (SM copies, async) and then by the staged path (copy
    engines).  The turns' calls are issued on a high-priority stream (the KV manager's
    work gates the turns; the exchange copy's own stream has the highest priority), the
    consumer's on a stream of normal priority.  The consumer's pages may change under
    it; its sums are not used."""
    torch.cuda.synchronize()
    with torch.cuda.stream(torch.cuda.Stream(device=pool.device, priority=-1)):
        return _overlap_measure(torch, pool, wl, first_turn, n_turns)


def _overlap_measure(torch, pool, wl, first_turn, n_turns):
    from paper_2606_22983_gb300 import lv
    from paper_2606_22983_gb300.manager import KVManager
    cons = ChecksumConsumer(torch, pool)
    alone = cons.alone_gbs()
    out = {"consumer": cons.describe(),
           "consumer_alone_gbs": round(alone, 1), "consumer_alone_hbm_frac": round(alone / HBM_PEAK, 3)}
    page_bytes = pool.J * pool.P
    ev = lambda: torch.cuda.Event(enable_timing=True)
    turn = first_turn
    for label, driver, mode, async_copy in (("zero_copy_sm", "device", 0, True),
                                            ("staged_copy_engine", "exchange", 2, True)):
        gm = KVManager(pool, perms=wl.perms, rank_on="none", mode=mode, record=False,
                       driver=driver, async_copy=async_copy)
        # warm-up of this driver (the staged path's staging runs grow during its first calls)
        run_turns(gm, wl, turn, turn + 10, None)
        turn += 10
        lv.lv_join(pool.handle, pool.stream)
        torch.cuda.synchronize()
        # the turns alone
        p0 = _moved_pages(pool)[0]
        t0, t1 = ev(), ev()
        t0.record()
        run_turns(gm, wl, turn, turn + n_turns, None)
        lv.lv_join(pool.handle, pool.stream)
        t1.record()
        torch.cuda.synchronize()
        alone_ms = t0.elapsed_time(t1)
        alone_gbs = (_moved_pages(pool)[0] - p0) * page_bytes / (alone_ms / 1e3) / 1e9
        turn += n_turns
        # the turns with the consumer running throughout (kept topped up from the host
        # until the turns are done)
        p0 = _moved_pages(pool)[0]
        cons.start()
        t0.record()
        for i in range(turn, turn + n_turns):
            cons.top_up()
            run_turns(gm, wl, i, i + 1, None)
        lv.lv_join(pool.handle, pool.stream)
        t1.record()
        ends = cons.keep_busy_until(t1)
        torch.cuda.synchronize()
        cons_gbs, covered = cons.rate_within(ends, t0, t1)
        turn += n_turns
        both_gbs = (_moved_pages(pool)[0] - p0) * page_bytes / (t0.elapsed_time(t1) / 1e3) / 1e9
        out[label] = {"turns": n_turns, "turns_alone_gbs": round(alone_gbs, 1),
                      "turns_with_consumer_gbs": round(both_gbs, 1),
                      "consumer_with_turns_gbs": round(cons_gbs, 1),
                      "consumer_frac_kept": round(cons_gbs / alone, 3),
                      "consumer_ran_throughout": covered}
    cons.close()
    assert pool.sync(raise_on_error=False) == 0, "device error during the overlap turns"
    return out


def direction_legs(torch, pool, now_us, rounds=8, k_pages=1100):
    """Each link direction on its own, device-driven: lv_evict of up to k_pages pages
    (the ranking's first k, as many as the host tier has room for; offload only), then
    preloads (lv_make_resident with LV_RESIDENT_PRELOAD) of the sessions with the most
    host-tier blocks that fit in the free HBM pages, one after the other while one fits
    (reload only, no eviction).  Copies run on the caller's stream; each call is timed
    with CUDA events on it.  The peaks are same-run contiguous page-locked copies of the
    mean call's byte count, D2H and H2D."""
    from paper_2606_22983_gb300 import lv
    from paper_2606_22983_gb300.harness import link_peaks
    res = torch.zeros(lv.RESIDENT_DTYPE.itemsize, dtype=torch.uint8, device=pool.device)
    page = pool.J * pool.P
    ev = lambda: torch.cuda.Event(enable_timing=True)
    off_ms, off_pages, in_ms, in_pages = [], [], [], []
    t = now_us
    for r in range(rounds):
        t += 100_000
        st0 = pool.stats()
        k = min(k_pages, pool.host_pages - st0["host_allocated"] - 64)
        if k < 64:
            break
        a, b = ev(), ev()
        a.record()
        lv.lv_evict(pool.handle, t, k, 0, None, None, res, pool.stream)
        b.record()
        b.synchronize()
        st1 = pool.stats()
        assert st1["bytes_in"] == st0["bytes_in"]
        off_ms.append(a.elapsed_time(b))
        off_pages.append((st1["bytes_out"] - st0["bytes_out"]) // page)
        for _ in range(8):
            free = pool.budget - st1["hbm_allocated"]
            _, host = pool.counts()
            fits = np.where(host <= free, host, -1)
            sid = int(np.argmax(fits))
            if fits[sid] <= 0:
                break
            a.record()
            lv.lv_make_resident(pool.handle, sid, t, 0, lv.LV_RESIDENT_PRELOAD, -1, None, None, None,
                                None, None, res, pool.stream)
            b.record()
            b.synchronize()
            st2 = pool.stats()
            assert st2["bytes_out"] == st1["bytes_out"]
            in_ms.append(a.elapsed_time(b))
            in_pages.append((st2["bytes_in"] - st1["bytes_in"]) // page)
            st1 = st2
    assert pool.sync(raise_on_error=False) == 0, "device error during the direction legs"
    out_b, in_b = sum(off_pages) * page, sum(in_pages) * page
    mean = int(min(max((out_b + in_b) / max(len(off_ms) + len(in_ms), 1), 1 << 26), 1 << 30))
    peaks = link_peaks(pool, mean // 4096 * 4096)
    res = {}
    for name, nb, ms, peak in (("offload_only", out_b, off_ms, peaks["d2h"]),
                               ("reload_only", in_b, in_ms, peaks["h2d"])):
        if not ms:
            continue
        gbs = nb / (sum(ms) / 1e3) / 1e9
        res[name] = {"calls": len(ms), "gb": round(nb / 1e9, 2), "gbs": round(gbs, 1),
                     "blocks_per_s": round(nb / page / (sum(ms) / 1e3), 1),
                     "peak_gbs": round(peak, 1), "frac": round(gbs / peak, 3),
                     "ms_p50": round(float(np.median(ms)), 3)}
    if "offload_only" in res:
        res["offload_only"]["call"] = "lv_evict (rank, plan, out-only exchange copy)"
    if "reload_only" in res:
        res["reload_only"]["call"] = "lv_make_resident with LV_RESIDENT_PRELOAD (no eviction)"
    res["peak_source"] = (f"same-run contiguous page-locked cudaMemcpyAsync of {mean // 4096 * 4096} B "
                          "per direction")
    return res


def _restart(pool, wl):
    """Puts a pool back in the workload's initial state (placement and sessions)."""
    from paper_2606_22983_gb300.harness import initial_sessions
    init = wl.init
    pool.import_placement(init.placement, init.ctx_tokens)
    pool.set_sessions(initial_sessions(wl))
    pool.sync()


def _streamed(torch, pool, wl, moves, seed, with_consumer=True):
    """The whole script issued without a host wait between events (turns and preloads
    with their copies on the pool's copy stream, each event's decisions overlapping the
    copies before it), from the initial state, alone and then (``with_consumer``) with the
    checksum consumer kept running throughout on a stream of normal priority (the
    manager's calls on a high-priority one).  Link fraction: the link's best time for
    every moving event's own mix (from the event-by-event pass of the same script) over
    the elapsed device time."""
    from paper_2606_22983_gb300 import lv
    from paper_2606_22983_gb300.manager import KVManager
    from workloads import scatter_order
    best_s = moves["link_best_s"]
    out = {}
    cons = None
    for label in ("alone", "with_consumer") if with_consumer else ("alone",):
        _restart(pool, wl)
        st0 = pool.stats()
        with torch.cuda.stream(torch.cuda.Stream(device=pool.device, priority=-1)):
            gm = KVManager(pool, perms=wl.perms, rank_on="none", record=False, driver="device",
                           order_fn=scatter_order, async_copy=True, script=wl)
            ends = None
            if label == "with_consumer":
                cons = ChecksumConsumer(torch, pool, seed=seed)
                cons_alone = cons.alone_gbs()
                cons.start()
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record()
            for i in range(wl.n_events):
                if cons is not None:
                    cons.top_up()
                gm.step(wl.event(i), i)
            lv.lv_join(pool.handle, pool.stream)
            b.record()
            if cons is not None:
                ends = cons.keep_busy_until(b)
            torch.cuda.synchronize()
        assert pool.sync(raise_on_error=False) == 0
        st1 = pool.stats()
        moved = st1["bytes_out"] + st1["bytes_in"] - st0["bytes_out"] - st0["bytes_in"]
        ms = a.elapsed_time(b)
        out[label] = {"ms": round(ms, 2), "gb": round(moved / 1e9, 2),
                      "gbs": round(moved / (ms / 1e3) / 1e9, 1),
                      "link_frac": round(best_s / (ms / 1e3), 3)}
        if ends is not None:
            got, covered = cons.rate_within(ends, a, b)
            out[label].update({"consumer_alone_gbs": round(cons_alone, 1),
                               "consumer_with_events_gbs": round(got, 1),
                               "consumer_frac_kept": round(got / cons_alone, 3),
                               "consumer_ran_throughout": covered})
            cons.close()
    return out


def five_workloads(torch, seed, consumer_on="mixed", streamed=("mixed", "long", "frag")):
    """All five seeded workloads through the device driver, one event at a time
    (paper_2606_22983_gb300.runner): GB/s and link fraction overall, by event kind and
    by direction.  Mixed and frag run at their stated session counts (256, 1024) where
    the host can page-lock their host tier within min(400 GB, 0.8 * MemAvailable), else
    scaled to it (``sizing``).  The ``streamed`` workloads run a second time from the same
    initial state without a host wait between events (``_streamed``).  The mixed script
    also runs with the checksum consumer reading resident KV throughout (its calls on a
    stream of normal priority, the manager's on a high-priority one), so that its speech
    start and barge-in preloads are measured next to serving work."""
    from paper_2606_22983_gb300.harness import fill_random, link_peaks, pool_for
    from paper_2606_22983_gb300.manager import KVManager
    from paper_2606_22983_gb300.runner import link_summary, peak_bytes, quantiles, run_events
    from workloads import CONFIG_NAMES, EVENT_NAMES, host_tier_limit, make_workload, mem_available_bytes, scatter_order
    out = {"mem_available_bytes": mem_available_bytes()}
    for name in CONFIG_NAMES:
        wl = make_workload(name, seed, host_limit=host_tier_limit())
        pool = pool_for(wl)
        try:
            fill_random(pool, seed)
            gm = KVManager(pool, perms=wl.perms, rank_on="none", record=False, driver="device",
                           order_fn=scatter_order, script=wl)
            copies = {}
            moves, turn_ms, _, wall = run_events(torch, pool, gm, wl, wl.n_events, copy_times=copies)
            nbytes = peak_bytes(pool, moves)
            peaks = link_peaks(pool, nbytes)
            r = {"sessions": wl.spec.n_sessions, "events": wl.n_events,
                 "host_pages": wl.spec.host_pages, "sizing": wl.meta.get("sizing"),
                 "turn_ms": quantiles(turn_ms), "wall_s": round(wall, 1),
                 "moves": link_summary(moves, peaks, EVENT_NAMES),
                 "copy_kernels": copies}
            if name in streamed:
                r["streamed"] = _streamed(torch, pool, wl, r["moves"], seed,
                                          with_consumer=name == consumer_on)
            if name == consumer_on:
                _restart(pool, wl)
                cons = ChecksumConsumer(torch, pool, seed=seed)
                alone = cons.alone_gbs()
                gm2 = KVManager(pool, perms=wl.perms, rank_on="none", record=False, driver="device",
                                order_fn=scatter_order, script=wl)
                with torch.cuda.stream(torch.cuda.Stream(device=pool.device, priority=-1)):
                    cons.top_up()
                    done = cons.window()
                    moves2, turn2, _, _ = run_events(torch, pool, gm2, wl, wl.n_events,
                                                     before_event=cons.top_up)
                    got = done()
                cons.close()
                r["with_consumer"] = {"consumer": cons.describe(),
                                      "consumer_alone_gbs": round(alone, 1),
                                      "consumer_with_events_gbs": round(got, 1),
                                      "consumer_frac_kept": round(got / alone, 3),
                                      "turn_ms": quantiles(turn2),
                                      "moves": link_summary(moves2, peaks, EVENT_NAMES)}
            out[name] = r
        finally:
            torch.cuda.synchronize()
            pool.close()
            torch.cuda.empty_cache()
    return out


def ab_measure(torch, seed, n_events):
    """NEXT rows f1 and f3 on the GPU: the mixed real-time workload at full size
    (128 sessions, 60 GB HBM budget) under three policies -- next-use ranking with
    the Section 5.2 preload controller (a 200 GB/s modelled link), next-use with
    every preload admitted, and the LRU baseline (no preloads).  For each turn it
    records whether the session's KV had to be loaded at turn start, on the turn's
    critical path, and the device time of the turn's calls (CUDA events, a host wait
    per turn to read its decisions)."""
    from paper_2606_22983_gb300.controller import ControlledKVManager
    from paper_2606_22983_gb300.harness import pool_for
    from paper_2606_22983_gb300.manager import KVManager
    from workloads import host_tier_limit, make_workload, pool_spec, scatter_order
    out = {"workload": f"mixed (256 sessions or as the host allows, 60 GB HBM budget), "
                       f"{n_events} events, seed {seed}"}
    turn_kinds = (1, 2, 7)
    for label in ("next_use_controller", "next_use_preload", "lru"):
        spec = pool_spec("mixed").with_(policy=1 if label == "lru" else 0)
        wl = make_workload("mixed", seed, spec=spec, n_events=n_events, host_limit=host_tier_limit())
        pool = pool_for(wl)
        try:
            if label == "next_use_controller":
                gm = ControlledKVManager(pool, link_bytes_per_us=200_000, lead_prior_us=2_000_000,
                                         cap_pages=spec.hbm_budget_pages // 10, perms=wl.perms,
                                         order_fn=scatter_order)
            else:
                gm = KVManager(pool, perms=wl.perms, rank_on="none", record=True, driver="device",
                               order_fn=scatter_order)
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            on_path_ms, on_path_pages, turn_ms = [], [], []
            w0 = time.perf_counter()
            for i in range(wl.n_events):
                e = wl.event(i)
                if int(e[1]) not in turn_kinds:
                    gm.step(e, i)
                    continue
                torch.cuda.synchronize()
                a.record()
                rec = gm.step(e, i)
                b.record()
                torch.cuda.synchronize()
                ms = a.elapsed_time(b)
                turn_ms.append(ms)
                loaded = len(rec.get("in_blocks", ()))
                if loaded:
                    on_path_ms.append(ms)
                    on_path_pages.append(loaded)
            wall = time.perf_counter() - w0
            assert pool.sync(raise_on_error=False) == 0, f"device error in the {label} run"
            st = pool.stats()
            q = lambda xs, f: round(float(np.percentile(xs, f)), 3) if xs else None
            out[label] = {
                "turns": len(turn_ms), "turns_loading_on_path": len(on_path_ms),
                "on_path_load_ms": {"mean": round(float(np.mean(on_path_ms)), 3) if on_path_ms else None,
                                    "p50": q(on_path_ms, 50), "p90": q(on_path_ms, 90),
                                    "max": q(on_path_ms, 100)},
                "on_path_pages_mean": round(float(np.mean(on_path_pages)), 1) if on_path_pages else 0,
                "turn_ms_mean": round(float(np.mean(turn_ms)), 3),
                "preloads": int(gm.counters.get("preloads", 0)),
                "gb_out": round(st["bytes_out"] / 1e9, 2), "gb_in": round(st["bytes_in"] / 1e9, 2),
                "wall_s": round(wall, 1)}
            for k in ("admitted", "completed", "cancelled", "given_up", "hits"):
                if k in gm.counters:
                    out[label][k] = int(gm.counters[k])
        finally:
            torch.cuda.synchronize()
            pool.close()
            torch.cuda.empty_cache()
    return out


def kernel_micro(torch, pool, seed=0):
    """Standalone timings of the HBM-bound kernels and the ranker (rank 0, after the turns).

    pack/unpack: 4096 scattered pages of the bench pool to / from one contiguous 6.4 GB
    run (each payload byte is read once and written once in HBM); ranker and remap:
    a metadata-sized pool (16-token pages of 256 B) with 2^20 resident pages in 1024
    sessions -- one top-256 decision, and one commit of all 2^20 pages to the host tier."""
    from paper_2606_22983_gb300 import lv
    from paper_2606_22983_gb300.pool import KVPool
    out = {}
    g = torch.Generator(device=pool.device).manual_seed(seed)
    n = min(4096, pool.hbm_pages)
    pages = torch.randperm(pool.hbm_pages, generator=g, device=pool.device)[:n].to(torch.int32)
    payload = n * pool.J * pool.P
    run = torch.empty(payload, dtype=torch.uint8, device=pool.device)
    for _ in range(2):
        lv.lv_pack_pages(pool.handle, pages, n, run, pool.stream)
        lv.lv_unpack_pages(pool.handle, run, pages, n, pool.stream)   # writes back the same bytes
    pool.sync()
    lv.lv_timing_read(pool.handle, reset=True)
    lv.lv_timing_enable(pool.handle, True)
    for _ in range(5):
        lv.lv_pack_pages(pool.handle, pages, n, run, pool.stream)
        lv.lv_unpack_pages(pool.handle, run, pages, n, pool.stream)
    t = lv.lv_timing_read(pool.handle, reset=True)
    lv.lv_timing_enable(pool.handle, False)
    assert pool.sync(raise_on_error=False) == 0
    for name in ("pack", "unpack"):
        ms = t[name]["total_ms"] / t[name]["launches"]
        gbs = 2 * payload / (ms / 1e3) / 1e9
        out[name] = {"pages": n, "bytes_per_launch": 2 * payload, "avg_ms": round(ms, 4),
                     "achieved_gbs": round(gbs, 1), "peak_gbs": HBM_PEAK, "frac": round(gbs / HBM_PEAK, 3)}
    del run
    # page checksums (an HBM-bound reader): the same scattered pages, each read once
    sums = torch.empty(n, dtype=torch.int64, device=pool.device)
    for _ in range(2):
        lv.lv_page_checksums(pool.handle, pages, n, sums, pool.stream)
    torch.cuda.synchronize()
    c0, c1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    c0.record()
    for _ in range(5):
        lv.lv_page_checksums(pool.handle, pages, n, sums, pool.stream)
    c1.record()
    torch.cuda.synchronize()
    assert pool.sync(raise_on_error=False) == 0
    ms = c0.elapsed_time(c1) / 5
    gbs = payload / (ms / 1e3) / 1e9
    out["checksum"] = {"pages": n, "bytes_per_launch": payload, "avg_ms": round(ms, 4),
                       "achieved_gbs": round(gbs, 1), "peak_gbs": HBM_PEAK, "frac": round(gbs / HBM_PEAK, 3)}
    del sums
    # one urgency-scheduling round over 4096 ready requests (Algorithm 1)
    rng = np.random.default_rng(seed)
    R = lv.LV_SCHED_MAX_REQUESTS
    reqs = np.zeros(R, dtype=lv.REQUEST_DTYPE)
    reqs["id"] = np.arange(R)
    reqs["started"] = rng.random(R) < 0.7
    reqs["play_buffer_us"] = rng.integers(0, 8, R) * 700_000
    reqs["ready_age_us"] = rng.integers(0, 10_000_000, R)
    reqs["kv_pages"] = rng.integers(0, 2048, R)
    reqs["tokens"] = rng.integers(1, 512, R)
    reqs["kv_needed"] = rng.integers(0, 64, R)
    q = lv.lv_sched_params(p_safe_us=2_000_000, alpha=4, beta=1, occupied=30_000, allocatable=40_000,
                           token_budget=8192, kv_budget=4096)
    reqs_d = torch.from_numpy(reqs.view(np.uint8).copy()).to(pool.device)
    order = torch.empty(R, dtype=torch.int32, device=pool.device)
    nb = torch.empty(1, dtype=torch.int32, device=pool.device)
    for _ in range(5):
        lv.lv_schedule(pool.handle, q, reqs_d, R, order, nb, pool.stream)
    torch.cuda.synchronize()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record()
    for _ in range(50):
        lv.lv_schedule(pool.handle, q, reqs_d, R, order, nb, pool.stream)
    b.record()
    torch.cuda.synchronize()
    out["scheduler"] = {"ready_requests": R, "us_per_round": round(a.elapsed_time(b) * 1e3 / 50, 2),
                        "admitted": int(nb.item())}
    # a metadata-sized pool: 1024 sessions x 1024 resident blocks = 2^20 pages
    S = B = 1024
    N = S * B
    mp = KVPool(layers=1, kv_heads=1, head_dim=8, max_sessions=S, max_blocks=B, hbm_pages=N,
                hbm_budget_pages=N, host_pages=N, device=pool.device, stream=pool.stream)
    try:
        rng = np.random.default_rng(seed)
        mp.import_placement(rng.permutation(N).astype(np.int32).reshape(S, B),
                            np.full(S, B * 16, np.int32))
        st = np.zeros(S, dtype=lv.SESSION_DTYPE)
        st["gen_us"] = rng.integers(0, 10_000_000, S)
        mp.set_sessions(st)
        mp.sync()
        o = torch.empty((256, 3), dtype=torch.int32, device=pool.device)
        c = torch.zeros(1, dtype=torch.int64, device=pool.device)
        for _ in range(5):
            lv.lv_select_victims(mp.handle, 0, 256, 0, o, 256, c, mp.stream)
        torch.cuda.synchronize()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record()
        for _ in range(50):
            lv.lv_select_victims(mp.handle, 0, 256, 0, o, 256, c, mp.stream)
        b.record()
        torch.cuda.synchronize()
        out["ranker"] = {"resident_pages": N, "sessions": S, "k": 256,
                         "us_per_decision": round(a.elapsed_time(b) * 1e3 / 50, 2)}
        out["ranker"]["sessions_4096"] = _ranker_4096(torch, pool, seed)
        # remap: the commit of all 2^20 pages to the host tier.  Each repetition
        # re-imports the placement, swaps everything out, flushes L2 (a 256 MB
        # write) and times one lv_remap call (its commit and release passes); the first
        # repetition is untimed.
        placement = rng.permutation(N).astype(np.int32).reshape(S, B)
        ctx = np.full(S, B * 16, np.int32)
        flush = torch.empty(256 << 20, dtype=torch.uint8, device=pool.device)
        ms_1m = []
        for rep in range(4):
            mp.import_placement(placement, ctx)
            victims, nv = mp.select(0, lv.LV_ALL, 0)
            assert nv == N
            slots, commit = mp.swap_out(victims, nv)
            flush.fill_(rep)
            a.record()
            mp.remap(commit, nv)
            b.record()
            torch.cuda.synchronize()
            assert mp.sync(raise_on_error=False) == 0 and mp.stats()["host_allocated"] == N
            if rep:
                ms_1m.append(a.elapsed_time(b))
        ms = float(np.mean(ms_1m))
        gbs = REMAP_BYTES_PER_ENTRY * N / (ms / 1e3) / 1e9
        out["remap_1m"] = {"entries": N, "bytes_per_entry": REMAP_BYTES_PER_ENTRY, "ms": round(ms, 4),
                           "entries_per_s": round(N / (ms / 1e3)), "achieved_gbs": round(gbs, 1),
                           "peak_gbs": HBM_PEAK, "frac": round(gbs / HBM_PEAK, 3),
                           "l2": "flushed before each launch"}
        # and at a turn's size: 1024 entries (one whole thinker session), latency
        mp.import_placement(placement, ctx)
        lat = []
        for rep in range(6):
            victims, nv = mp.select(0, 1024, 0)
            slots, commit = mp.swap_out(victims, nv)
            mp.sync()
            a.record()
            mp.remap(commit, nv)
            b.record()
            torch.cuda.synchronize()
            if rep:
                lat.append(a.elapsed_time(b) * 1e3)
        assert mp.sync(raise_on_error=False) == 0
        # the stream is idle when the first event is recorded, so this is the whole
        # call as a caller sees it: binding, argument checks, launch and kernel
        out["remap_turn"] = {"entries": 1024, "us_per_call": round(float(np.median(lat)), 2),
                             "what": "lv_remap call latency on an idle stream"}
        del flush
    finally:
        mp.close()
    return out


def _ranker_4096(torch, pool, seed):
    """One top-256 decision over 4096 sessions x 256 resident blocks (2^20 pages, the
    most sessions a pool takes), 50 back to back, CUDA events."""
    from paper_2606_22983_gb300 import lv
    from paper_2606_22983_gb300.pool import KVPool
    S, B = 4096, 256
    N = S * B
    mp = KVPool(layers=1, kv_heads=1, head_dim=8, max_sessions=S, max_blocks=B, hbm_pages=N,
                hbm_budget_pages=N, host_pages=0, device=pool.device, stream=pool.stream)
    try:
        rng = np.random.default_rng(seed)
        mp.import_placement(rng.permutation(N).astype(np.int32).reshape(S, B), np.full(S, B * 16, np.int32))
        st = np.zeros(S, dtype=lv.SESSION_DTYPE)
        st["gen_us"] = rng.integers(0, 10_000_000, S)
        mp.set_sessions(st)
        mp.sync()
        o = torch.empty((256, 3), dtype=torch.int32, device=pool.device)
        c = torch.zeros(1, dtype=torch.int64, device=pool.device)
        for _ in range(5):
            lv.lv_select_victims(mp.handle, 0, 256, 0, o, 256, c, mp.stream)
        torch.cuda.synchronize()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record()
        for _ in range(50):
            lv.lv_select_victims(mp.handle, 0, 256, 0, o, 256, c, mp.stream)
        b.record()
        torch.cuda.synchronize()
        assert mp.sync(raise_on_error=False) == 0 and int(c.item()) == 256
        return {"resident_pages": N, "sessions": S, "k": 256,
                "us_per_decision": round(a.elapsed_time(b) * 1e3 / 50, 2)}
    finally:
        mp.close()


def micro_only(args, torch):
    """kernel_micro on a 2048-page thinker-shaped pool (3.2 GB) instead of the bench pool."""
    from paper_2606_22983_gb300 import build
    build()
    from paper_2606_22983_gb300.harness import fill_random
    from paper_2606_22983_gb300.pool import KVPool
    pool = KVPool(layers=48, kv_heads=4, head_dim=128, max_sessions=8, max_blocks=16,
                  hbm_pages=2048, hbm_budget_pages=2048, host_pages=16)
    try:
        fill_random(pool, args.seed)
        return {"micro": kernel_micro(torch, pool, args.seed)}
    finally:
        pool.close()


def kernel_source_sha(kernel):
    """sha256 of one kernel's definition in lv_kernels.cu (from its name to the
    closing brace), with the launch-shape constants it uses."""
    import hashlib
    import re
    src = os.path.join(ROOT, "paper_2606_22983_gb300", "csrc", "lv_kernels.cu")
    with open(src) as f:
        text = f.read()
    start = text.index("\nk_" + kernel + "(")
    end = text.index("\n}\n", start)
    consts = "".join(m.group(0) for m in re.finditer(r"constexpr int kCopy\w+ = \d+;", text))
    return hashlib.sha256((consts + text[start:end]).encode()).hexdigest()


def _profiled_traffic(kernel, bytes_per_launch):
    """DRAM bytes per launch from the committed ncu summary, or None when that
    summary does not cover this kernel or the kernel changed since."""
    try:
        with open(os.path.join(ROOT, "profiles", "traffic.json")) as f:
            d = json.load(f)[kernel]
        if kernel_source_sha(d["kernel"]) != d["kernel_source_sha256"]:
            return None
        return round(d["dram_bytes_per_payload_byte"] * bytes_per_launch)
    except (OSError, KeyError, ValueError):
        return None


# ----------------------------------------------------------- the oracle arm
def _oracle_for(wl):
    """The oracle over the whole workload, with full byte images (a 40 GB HBM image and
    the host tier for the thinker pool), touched once so that no timed turn pays for
    first-touch page faults."""
    from oracle import OracleManager
    om = OracleManager(wl, with_bytes=True, content=None, rank_on="none")
    om.pool.hbm.fill(1)
    om.pool.host.fill(1)
    return om


def _oracle_turn(om, S, i):
    """Turn i of a turn-driven script on the oracle (its playback batch, then the
    turn); returns the bytes it moved."""
    b0 = om.pool.bytes_out + om.pool.bytes_in
    for j in range(i * (S + 1), (i + 1) * (S + 1)):
        om.step(j)
    return om.pool.bytes_out + om.pool.bytes_in - b0


def cpu_baseline(args, seconds, seed):
    """The oracle (single thread, numpy memcpy per sub-page) on a bounded sample of the
    benchmark's own workload: the same pool and script, its first turns until about
    ``seconds`` of CPU time."""
    wl = _arm_spec(args, seed)
    om = _oracle_for(wl)
    S = wl.spec.n_sessions
    moved, turns = 0, 0
    t0 = time.perf_counter()
    el = 0.0
    while (turns + 1) * (S + 1) <= wl.n_events and el < seconds:
        moved += _oracle_turn(om, S, turns)
        turns += 1
        el = time.perf_counter() - t0
    return {"value": round(moved / el / 1e9, 4), "unit": UNIT, "cores": 1, "kind": "oracle",
            "sample": f"the first {turns} turns of the benchmark's workload (the same "
                      f"{S}-session pool with a {wl.spec.hbm_budget_pages}-page HBM image and "
                      f"{wl.spec.host_pages} host slots), {moved / 1e9:.2f} GB moved in {el:.1f} s",
            "seconds": round(el, 2), "ranker": _oracle_ranker(seed)}


def oracle_configs(seed, seconds=8.0):
    """The oracle as it stands (one host core, byte images) on a bounded sample of each
    of the five workloads at the sizes the GPU runs them: events in script order until
    about ``seconds`` of CPU time.  The tiny and thinker images are touched before
    timing; the larger ones (mixed 60 + ~134 GB, long 40 + ~50 GB, frag 100 + ~148 GB)
    are left untouched, so their timed events include first-touch page faults, and
    only the pages the sample writes take host memory."""
    from oracle import OracleManager
    from workloads import CONFIG_NAMES, host_tier_limit, make_workload
    out = {}
    for name in CONFIG_NAMES:
        wl = make_workload(name, seed, host_limit=host_tier_limit())
        om = OracleManager(wl, with_bytes=True, content=None, rank_on="none")
        touched = name in ("tiny", "thinker")
        if touched:
            om.pool.hbm.fill(1)
            om.pool.host.fill(1)
        b0 = om.pool.bytes_out + om.pool.bytes_in
        t0 = time.perf_counter()
        i = 0
        el = 0.0
        while i < wl.n_events and el < seconds:
            om.step(i)
            i += 1
            el = time.perf_counter() - t0
        moved = om.pool.bytes_out + om.pool.bytes_in - b0
        page = wl.spec.shape.page_bytes
        out[name] = {"sessions": wl.spec.n_sessions, "events": i, "of_events": wl.n_events,
                     "gb_moved": round(moved / 1e9, 3), "seconds": round(el, 2),
                     "gbs": round(moved / el / 1e9, 4), "blocks_per_s": round(moved / page / el, 1),
                     "images_touched_first": touched, "cores": 1}
        del om
    return out


def _oracle_ranker(seed):
    """The oracle's top-256 decision over the 2^20-page metadata state the GPU ranker is
    timed on (1024 sessions x 1024 resident blocks, random placement and states)."""
    from oracle import sessions as se
    from oracle.policy import select_victims
    rng = np.random.default_rng(seed)
    S = B = 1024
    tables = rng.permutation(S * B).reshape(S, B).astype(np.int64)
    nblocks = np.full(S, B, np.int64)
    sts = [se.SessionState(gen_us=int(g)) for g in rng.integers(0, 10_000_000, S)]
    t0 = time.perf_counter()
    n = 0
    while True:
        select_victims(tables, nblocks, sts, 0, 256, se.MODE_PLAYBACK, 3_000_000, 80_000)
        n += 1
        el = time.perf_counter() - t0
        if el > 2.0 or n >= 5:
            break
    return {"ms_per_decision": round(el * 1e3 / n, 1), "resident_pages": S * B, "k": 256,
            "decisions": n}


def arm_config(args, spec, ws):
    """The workload description both arms report (identical for the same arguments)."""
    return {"workload": "thinker: 48 layers, 4 KV heads x 128, bf16, 16-token pages (1.5 MiB), "
                        f"{spec.n_sessions} sessions log-uniform 2k-16k tokens, "
                        f"{spec.hbm_budget_pages}-page HBM budget, one turn = evict + reload",
            "hbm_budget_pages": spec.hbm_budget_pages, "host_pages": spec.host_pages,
            "mode": {0: "auto", 1: "zero_copy", 2: "staged"}[args.mode],
            "driver": args.driver,
            "tiers": ("exclusive", "inclusive")[args.tiers],
            "async_copy": bool(args.async_copy and (args.driver == "device" or args.mode == 2)),
            "l2": "inputs larger than L2 (a turn moves about 0.6 GB each way out of a "
                  "40 GB pool)",
            "parallelism": f"replicas x{ws}"}


def _arm_spec(args, seed):
    """The pool spec of the timed workload, as ours() builds it."""
    from workloads import make_workload, pool_spec
    over = {}
    if args.sessions or args.budget_pages or args.tiers:
        sp = pool_spec(WORKLOAD)
        b = args.budget_pages or sp.hbm_budget_pages
        over["spec"] = sp.with_(n_sessions=args.sessions or sp.n_sessions, hbm_pages=b,
                                hbm_budget_pages=b, tiers=args.tiers)
    KO = OVERLAP_TURNS if (args.overlap and args.driver == "device") else 0
    return make_workload(WORKLOAD, seed, n_turns=args.warmup + 2 * args.steps + 4 * KO + 26,
                         **over)


def reference(args):
    """The oracle as it stands, on the host cores, over the benchmark's own workload: W
    warm-up turns, then K timed turns of the same script, pool and sizes as our arm."""
    ws, rank, _ = _dist()
    if rank != 0:
        return None
    K, W = args.steps, args.warmup
    wl = _arm_spec(args, args.seed)
    om = _oracle_for(wl)
    S = wl.spec.n_sessions
    assert (W + K) * (S + 1) <= wl.n_events
    for i in range(W):
        _oracle_turn(om, S, i)
    t0 = time.perf_counter()
    moved = sum(_oracle_turn(om, S, i) for i in range(W, W + K))
    el = time.perf_counter() - t0
    v = moved / el / 1e9
    return {"impl": "reference", "metric": METRIC, "value": round(v, 4), "unit": UNIT,
            "n_gpus": ws, "steps": K, "warmup": W, "ms_per_step": round(el * 1e3 / K, 3),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "u8",
            "data": "synthetic",
            "config": arm_config(args, wl.spec, ws),
            "cpu_baseline": {"value": round(v, 4), "unit": UNIT, "cores": 1, "kind": "oracle",
                             "sample": f"{K} turns of this workload after {W} warm-up turns, "
                                       f"{moved / 1e9:.2f} GB moved (the whole workload: "
                                       f"{S} sessions, {wl.spec.hbm_budget_pages}-page HBM image)"},
            "e2e": {"value": round(v, 4), "unit": UNIT, "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}


def main():
    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=("ours", "reference"), default="ours")
    ap.add_argument("--mode", type=int, default=0, help="0 auto, 1 zero-copy, 2 staged")
    ap.add_argument("--driver", choices=("device", "exchange", "sequential"), default="device",
                    help="device: one lv_make_resident per turn; exchange: select + "
                         "lv_swap_exchange; sequential: swap-out, commit, swap-in, commit")
    ap.add_argument("--seed", type=int, default=0)
    ap.add_argument("--cpu-seconds", type=float, default=15.0)
    ap.add_argument("--no-cpu-baseline", dest="cpu_baseline", action="store_false")
    ap.add_argument("--micro-only", action="store_true",
                    help="only the standalone kernel timings, on a small pool (profiling case)")
    ap.add_argument("--no-micro", dest="micro", action="store_false",
                    help="skip the standalone pack/unpack/remap/ranker timings")
    ap.add_argument("--sessions", type=int, default=0,
                    help="smaller case for profiling: number of sessions")
    ap.add_argument("--budget-pages", type=int, default=0,
                    help="smaller case for profiling: HBM budget in pages")
    ap.add_argument("--oracle-configs", action="store_true",
                    help="only the oracle's bounded samples of all five workloads (host cores)")
    ap.add_argument("--ab", action="store_true",
                    help="only the policy A/B on the mixed workload (NEXT rows f1 and f3)")
    ap.add_argument("--ab-events", type=int, default=3000)
    ap.add_argument("--no-overlap", dest="overlap", action="store_false",
                    help="skip the consumer-overlap measurement")
    ap.add_argument("--no-directions", dest="directions", action="store_false",
                    help="skip the offload-only and reload-only legs")
    ap.add_argument("--no-five", dest="five", action="store_false",
                    help="skip the five workloads run event by event")
    ap.add_argument("--no-async-copy", dest="async_copy", action="store_false",
                    help="device driver: copy on the caller's stream (no overlap of the next "
                         "turn's decisions with this turn's copy)")
    ap.add_argument("--tiers", type=int, default=0, choices=(0, 1),
                    help="0 exclusive tiers, 1 inclusive (clean host copies kept)")
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be at least 3")
    if args.impl == "reference":
        line = reference(args)
    elif args.oracle_configs:
        line = {"oracle_configs": oracle_configs(args.seed, args.cpu_seconds)}
    elif args.micro_only:
        import torch
        line = micro_only(args, torch)
    elif args.ab:
        import torch
        from paper_2606_22983_gb300 import build
        build()
        line = {"ab": ab_measure(torch, args.seed, args.ab_events)}
    else:
        import torch
        line = ours(args, torch)
    if line is not None:
        print(json.dumps(line), flush=True)


if __name__ == "__main__":
    main()
