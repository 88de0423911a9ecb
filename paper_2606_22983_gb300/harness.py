"""Sets up a KVPool for a seeded synthetic workload (``workloads``).

Everything here prepares inputs: the initial placement and session states,
and the KV bytes (tagged by logical position, ``workloads.content``) written
with plain torch indexing, standing in for the model that produced the KV.
"""
from __future__ import annotations

import numpy as np
import torch

from workloads.content import (subpage_offsets, subpage_values_torch, tagged_values_torch,
                               valid_rows, value_table)

from . import lv
from .pool import KVPool


def zero_host(pool: KVPool):
    if pool.host_dev is not None:
        pool.host_dev.zero_()
        torch.cuda.synchronize(pool.device)


def pool_for(workload, device=None, stream=None, kv=None) -> KVPool:
    spec = workload.spec
    sh = spec.shape
    pool = KVPool(layers=sh.layers, kv_heads=sh.kv_heads, head_dim=sh.head_dim,
                  page_tokens=sh.page_tokens, elem_bytes=sh.elem_bytes,
                  max_sessions=spec.n_sessions, max_blocks=spec.max_blocks,
                  hbm_pages=spec.hbm_pages, hbm_budget_pages=spec.hbm_budget_pages,
                  host_pages=spec.host_pages, reply_prior_us=spec.reply_prior_us,
                  protect_us=spec.protect_us, unit_us=spec.unit_us,
                  within_order=spec.within_order, t_play_mode=spec.t_play_mode,
                  device=device, stream=stream, kv=kv, policy=spec.policy, tiers=spec.tiers)
    init = workload.init
    pool.import_placement(init.placement, init.ctx_tokens)
    pool.set_sessions(initial_sessions(workload))
    pool.sync()
    return pool


def initial_sessions(workload) -> np.ndarray:
    """The session table a workload starts from (lv_session_state [S])."""
    init = workload.init
    st = np.zeros(workload.spec.n_sessions, dtype=lv.SESSION_DTYPE)
    st["flags"] = np.where(init.resp_open != 0, lv.LV_RESP_OPEN, 0)
    st["gen_us"] = init.gen_us
    st["play_us"] = init.play_us
    st["reply_tokens"] = init.reply_tokens
    return st


class ContentWriter:
    """Writes tagged KV contents into a pool's HBM arrays and host pool."""

    def __init__(self, pool: KVPool, workload, seed=None, chunk=2048, tagged=False):
        self.pool = pool
        self.shape = workload.spec.shape
        self.seed = workload.seed if seed is None else seed
        self.tagged = tagged            # address-tagged chunks instead of seeded values
        if not tagged:
            self.table_np = value_table(self.seed)
            self.table = torch.from_numpy(self.table_np.view(np.int16)).to(pool.device)
        self.chunk = chunk

    def _values(self, sids, blks, layer, kv, rows):
        if self.tagged:
            return tagged_values_torch(sids, blks, layer, kv, rows, self.shape, self.pool.device)
        off = subpage_offsets(self.seed, sids, blks, np.full(len(sids), layer),
                              np.full(len(sids), kv), self.shape)
        return subpage_values_torch(self.table, torch.from_numpy(off).to(self.pool.device),
                                    torch.from_numpy(np.asarray(rows, np.int64)).to(self.pool.device),
                                    self.shape)

    def write_blocks(self, sids, blks, locs, ctx_of):
        """Whole sub-pages of blocks (sid, blk) at encoded locations ``locs``."""
        pool = self.pool
        sids = np.asarray(sids, np.int64)
        blks = np.asarray(blks, np.int64)
        locs = np.asarray(locs, np.int64)
        rows = valid_rows(np.asarray([ctx_of[s] for s in sids], np.int64), blks, self.shape)
        hbm = locs >= 0
        for j in range(pool.J):
            layer, kv = j // 2, j % 2
            for lo in range(0, len(sids), self.chunk):
                sl = slice(lo, lo + self.chunk)
                m = hbm[sl]
                vals = self._values(sids[sl], blks[sl], layer, kv, rows[sl])
                if m.any():
                    idx = torch.from_numpy(locs[sl][m]).to(pool.device)
                    pool.kv[j].index_copy_(0, idx, vals[torch.from_numpy(m).to(pool.device)].view(torch.uint8))
                if (~m).any():
                    slots = torch.from_numpy(-(locs[sl][~m] + 2)).to(pool.device)
                    host_vals = vals[torch.from_numpy(~m).to(pool.device)].view(torch.uint8)
                    pool.host_dev[:, j, :].index_copy_(0, slots, host_vals)   # GPU writes over the link
        torch.cuda.synchronize(pool.device)

    def write_initial(self, workload):
        init = workload.init
        S, B = init.placement.shape
        s_idx, b_idx = np.nonzero(init.placement != -1)
        self.write_blocks(s_idx, b_idx, init.placement[s_idx, b_idx], init.ctx_tokens)

    def write_appended(self, sid, old_ctx, new_ctx):
        """The model writes K/V of appended tokens: new rows of the old tail block,
        whole sub-pages (zero past the context end) of new blocks."""
        pool, T = self.pool, self.shape.page_tokens
        tables, _, _ = pool.tables()
        rb = self.shape.row_elems * self.shape.elem_bytes
        old_blocks = -(-old_ctx // T)
        for b in range(old_ctx // T, -(-new_ctx // T)):
            page = int(tables[sid, b])
            lo = (max(old_ctx, b * T) - b * T) if b < old_blocks else 0
            hi = (min(new_ctx, (b + 1) * T) - b * T) if b < old_blocks else T
            for j in range(pool.J):
                vals = self._values(np.array([sid]), np.array([b]), j // 2, j % 2, [valid_rows(new_ctx, b, self.shape)])
                pool.kv[j][page, lo * rb:hi * rb] = vals.view(torch.uint8)[0, lo * rb:hi * rb]
        torch.cuda.synchronize(pool.device)


def fill_random(pool: KVPool, seed: int = 0):
    """bf16 ~N(0,1) bytes in every HBM page and host slot (throughput runs)."""
    g = torch.Generator(device=pool.device).manual_seed(seed)
    for j in range(pool.J):
        v = torch.randn((pool.hbm_pages, pool.P // 2), generator=g, device=pool.device,
                        dtype=torch.float32).to(torch.bfloat16)
        pool.kv[j].copy_(v.view(torch.uint8).view(pool.hbm_pages, pool.P))
        del v
    if pool.host is not None:
        step = max(1, (256 << 20) // (pool.J * pool.P))
        for lo in range(0, pool.host_pages, step):
            n = min(step, pool.host_pages - lo)
            v = torch.randn((n, pool.J * pool.P // 2), generator=g, device=pool.device,
                            dtype=torch.float32).to(torch.bfloat16)
            pool.host_dev[lo:lo + n].copy_(v.view(torch.uint8).view(n, pool.J, pool.P))
    torch.cuda.synchronize(pool.device)


def link_peaks(pool: KVPool, nbytes: int, reps: int = 5) -> dict:
    """The host link's measured peaks in GB/s: a contiguous page-locked cudaMemcpyAsync of
    nbytes device-to-host, host-to-device, and both at once ('bidir', counting both).
    It overwrites the first 2 * nbytes of the host pool: measure after the workload."""
    src = pool.kv.view(-1)[:nbytes]
    host = torch.from_numpy(pool.host.reshape(-1)[:nbytes])
    dev2 = torch.empty(nbytes, dtype=torch.uint8, device=pool.device)
    host2 = torch.from_numpy(pool.host.reshape(-1)[nbytes:2 * nbytes]) \
        if pool.host.size >= 2 * nbytes else None
    res = {}
    for name, fn in (("d2h", lambda: host.copy_(src, non_blocking=True)),
                     ("h2d", lambda: dev2.copy_(host, non_blocking=True))):
        best = 1e30
        for _ in range(reps):
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record()
            fn()
            b.record()
            b.synchronize()
            best = min(best, a.elapsed_time(b))
        res[name] = nbytes / (best / 1e3) / 1e9
    if host2 is not None:
        s2 = torch.cuda.Stream()
        best = 1e30
        for _ in range(reps):
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record()
            s2.wait_event(a)
            host.copy_(src, non_blocking=True)
            with torch.cuda.stream(s2):
                dev2.copy_(host2, non_blocking=True)
            torch.cuda.current_stream().wait_stream(s2)
            b.record()
            b.synchronize()
            best = min(best, a.elapsed_time(b))
        res["bidir"] = 2 * nbytes / (best / 1e3) / 1e9
    del dev2
    return res
