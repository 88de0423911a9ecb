"""Paged KV block pool with an HBM tier and a host tier (Section 5, Fig. 6; Section 6).

State
  tables[s, b]   location of block b of session s: >= 0 HBM page, -1 none,
                 <= -2 host slot ``-(e + 2)``
  nblocks[s]     blocks in use by session s (ceil(context / T))
  owner_*        (sid, blk) that owns a page / slot, (-1, -1) when none
  *_used         page / slot is allocated (reserved by a swap, or owned)
  hbm[j, p]      bytes of sub-page j (= 2*layer + kv) of HBM page p   [2L][pages][P]
  host[h, j]     bytes of sub-page j of host slot h                   [slots][2L][P]

Operations follow their plain definitions:
  * allocation takes the lowest-numbered free pages / slots, in ascending
    order, and hands them out in request order; the HBM tier may hold at most
    ``budget`` allocated pages (the block allocator is kept, Section 5.1);
  * swap-out copies every sub-page of each victim page to its host slot and
    swap-in copies every sub-page of a host slot back, one ``memcpy`` per
    sub-page; neither changes the block tables;
  * remap commits (sid, blk, new location) entries: the table points to the
    new location, which becomes owned, and the old location is freed.  A
    failed or cancelled transfer is never committed, so the old mapping stays
    valid (Section 5.2: a preload that fails only costs time; the result stays right).

Tiers (the paper does not say whether the host copy is kept after a reload):
  * exclusive (default): a block lives in exactly one tier; its host slot is
    freed when the block is committed back to HBM.
  * inclusive: the host slot of a block committed back to HBM stays allocated
    and owned by the block as its *clean copy* (``shadow[s, b]``), as long as
    the block's bytes are unchanged.  KV rows are written once, when their
    token is appended, so only a session's last, partially filled block can
    change: appending tokens into it drops its clean copy (the slot is freed).
    Evicting a block that has a clean copy moves no bytes: its "slot" is the
    clean copy, no slot is reserved, and the commit points the table back to
    it.  Committing a block to any other host slot drops its clean copy.
    Clean copies are never reclaimed for other blocks, so the host tier must
    be able to hold every block (otherwise an eviction fails with NO_HOST,
    exactly as in the exclusive mode).

Parity status: allocation, copy and remap are pinned by closed forms and
invariants (owners and tables stay inverse, every byte lands where its block
is mapped, a failed transfer leaves the mapping unchanged).  The inclusive
tier is a reading: it is pinned by invariance (the same workload leaves the
same bytes and tables under both tiers) and is otherwise parity unpinned.
"""
from __future__ import annotations

import numpy as np


class OracleError(Exception):
    def __init__(self, code: str, msg: str = ""):
        super().__init__(f"{code}: {msg}" if msg else code)
        self.code = code


def _is_host(e: int) -> bool:
    return e <= -2


def _slot_of(e: int) -> int:
    return -(e + 2)


def _enc_host(slot: int) -> int:
    return -(slot + 2)


class OraclePool:
    def __init__(self, layers, kv_heads, head_dim, page_tokens, elem_bytes, n_sessions,
                 max_blocks, hbm_pages, hbm_budget_pages, host_pages, with_bytes=True,
                 inclusive=False):
        self.L, self.T = layers, page_tokens
        self.P = page_tokens * kv_heads * head_dim * elem_bytes
        self.J = 2 * layers
        self.S, self.max_blocks = n_sessions, max_blocks
        self.hbm_pages, self.budget, self.host_pages = hbm_pages, hbm_budget_pages, host_pages
        self.tables = np.full((n_sessions, max_blocks), -1, dtype=np.int64)
        self.nblocks = np.zeros(n_sessions, dtype=np.int64)
        self.ctx = np.zeros(n_sessions, dtype=np.int64)
        self.owner_hbm = np.full((hbm_pages, 2), -1, dtype=np.int64)
        self.owner_host = np.full((host_pages, 2), -1, dtype=np.int64)
        self.hbm_used = np.zeros(hbm_pages, dtype=bool)
        self.host_used = np.zeros(host_pages, dtype=bool)
        self.with_bytes = with_bytes
        if with_bytes:
            self.hbm = np.zeros((self.J, hbm_pages, self.P), dtype=np.uint8)
            self.host = np.zeros((host_pages, self.J, self.P), dtype=np.uint8)
        self.bytes_out = 0
        self.bytes_in = 0
        self.inclusive = bool(inclusive)
        self.shadow = np.full((n_sessions, max_blocks), -1, dtype=np.int64)   # clean copies
        self.clean_out = 0        # evictions that moved no bytes
        self.clean_dropped = 0    # clean copies dropped because their block changed

    # ---------------------------------------------------------------- set-up
    def import_placement(self, placement: np.ndarray, ctx_tokens: np.ndarray) -> None:
        """Load an initial placement (encoded block tables) and context lengths (Section 6,
        paged KV tables)."""
        S = self.S
        for s in range(S):
            self.ctx[s] = int(ctx_tokens[s])
            nb = -(-int(ctx_tokens[s]) // self.T)
            if nb > self.max_blocks:
                raise OracleError("INVALID", f"session {s} needs {nb} blocks")
            self.nblocks[s] = nb
            for b in range(self.max_blocks):
                e = int(placement[s, b])
                if b >= nb:
                    if e != -1:
                        raise OracleError("INVALID", f"entry beyond the context at ({s},{b})")
                    continue
                if e >= 0:
                    if e >= self.hbm_pages or self.hbm_used[e]:
                        raise OracleError("DOUBLE_MAP", f"page {e}")
                    self.hbm_used[e] = True
                    self.owner_hbm[e] = (s, b)
                elif _is_host(e):
                    h = _slot_of(e)
                    if h >= self.host_pages or self.host_used[h]:
                        raise OracleError("DOUBLE_MAP", f"slot {h}")
                    self.host_used[h] = True
                    self.owner_host[h] = (s, b)
                else:
                    raise OracleError("INVALID", f"block ({s},{b}) has no location")
                self.tables[s, b] = e
        if int(self.hbm_used.sum()) > self.budget:
            raise OracleError("BUDGET", "initial placement exceeds the HBM budget")

    # ------------------------------------------------------------ allocation
    def _alloc_lowest(self, used: np.ndarray, n: int, cap: int, code: str) -> np.ndarray:
        """The n lowest-numbered free entries of ``used`` in ascending order."""
        n = int(n)
        if n < 0:
            raise OracleError("INVALID", "negative count")
        if int(used.sum()) + n > cap:
            raise OracleError(code, f"{n} requested, {cap - int(used.sum())} available")
        free = np.nonzero(~used)[0]
        if free.size < n:
            raise OracleError(code, f"{n} requested, {free.size} free")
        got = free[:n].astype(np.int64)
        used[got] = True
        return got

    def alloc_hbm(self, n: int) -> np.ndarray:
        """Reserve the n lowest free HBM pages within the budget (Section 5.1)."""
        return self._alloc_lowest(self.hbm_used, n, self.budget, "NO_HBM")

    def alloc_host(self, n: int) -> np.ndarray:
        """Reserve the n lowest free host slots of the swap pool (Section 5.1)."""
        return self._alloc_lowest(self.host_used, n, self.host_pages, "NO_HOST")

    # ------------------------------------------------------------------ copy
    def swap_out(self, sid, blk, page) -> np.ndarray:
        """Copy victim pages to freshly reserved host slots; returns the slots (Section 5,
        the swap-out of Fig. 6).

        Inclusive tiers: a victim with a clean copy gets that slot and moves no
        bytes; the others reserve the lowest free slots, in victim order."""
        sid, blk, page = (np.asarray(x, dtype=np.int64) for x in (sid, blk, page))
        for s, b, p in zip(sid, blk, page):
            s, b, p = int(s), int(b), int(p)
            if not (0 <= s < self.S and 0 <= b < self.nblocks[s] and 0 <= p < self.hbm_pages):
                raise OracleError("BOUNDS", f"victim ({s},{b},{p})")
            if self.tables[s, b] != p or tuple(self.owner_hbm[p]) != (s, b):
                raise OracleError("STATE", f"victim ({s},{b},{p}) is not resident there")
        clean = np.array([self.inclusive and self.shadow[int(s), int(b)] >= 0
                          for s, b in zip(sid, blk)], dtype=bool)
        slots = np.empty(sid.size, dtype=np.int64)
        slots[~clean] = self.alloc_host(int((~clean).sum()))
        slots[clean] = self.shadow[sid[clean], blk[clean]]
        if self.with_bytes:
            for p, h, c in zip(page, slots, clean):
                if c:
                    continue
                for j in range(self.J):
                    self.host[h, j, :] = self.hbm[j, p, :]
        self.bytes_out += int((~clean).sum()) * self.J * self.P
        self.clean_out += int(clean.sum())
        return slots

    def swap_in(self, sid: int, blks) -> np.ndarray:
        """Copy host-resident blocks of ``sid`` into freshly reserved HBM pages
        (Sections 5.2 and 6)."""
        blks = np.asarray(blks, dtype=np.int64)
        slots = []
        for b in blks:
            b = int(b)
            if not (0 <= sid < self.S and 0 <= b < self.nblocks[sid]):
                raise OracleError("BOUNDS", f"block ({sid},{b})")
            e = int(self.tables[sid, b])
            if not _is_host(e) or tuple(self.owner_host[_slot_of(e)]) != (sid, b):
                raise OracleError("STATE", f"block ({sid},{b}) is not in the host tier")
            slots.append(_slot_of(e))
        pages = self.alloc_hbm(blks.size)
        if self.with_bytes:
            for h, p in zip(slots, pages):
                for j in range(self.J):
                    self.hbm[j, p, :] = self.host[h, j, :]
        self.bytes_in += int(blks.size) * self.J * self.P
        return pages

    # ----------------------------------------------------------------- remap
    def remap(self, sid, blk, new_loc) -> None:
        """Commit (sid, blk, new location) entries in order (Section 6, block-table update)."""
        seen = set()
        for s, b, e in zip(np.asarray(sid), np.asarray(blk), np.asarray(new_loc)):
            s, b, e = int(s), int(b), int(e)
            if not (0 <= s < self.S and 0 <= b < self.nblocks[s]):
                raise OracleError("BOUNDS", f"entry ({s},{b})")
            if (s, b) in seen:
                raise OracleError("DOUBLE_MAP", f"block ({s},{b}) twice in one batch")
            seen.add((s, b))
            if e >= 0:
                if e >= self.hbm_pages:
                    raise OracleError("BOUNDS", f"page {e}")
                if not self.hbm_used[e] or self.owner_hbm[e, 0] != -1:
                    raise OracleError("DOUBLE_MAP", f"page {e} is not a free reservation")
                self.owner_hbm[e] = (s, b)
            elif _is_host(e):
                h = _slot_of(e)
                if h >= self.host_pages:
                    raise OracleError("BOUNDS", f"slot {h}")
                own_copy = self.inclusive and self.shadow[s, b] == h
                if not own_copy and (not self.host_used[h] or self.owner_host[h, 0] != -1):
                    raise OracleError("DOUBLE_MAP", f"slot {h} is not a free reservation")
                self.owner_host[h] = (s, b)
            else:
                raise OracleError("BOUNDS", "new location -1")
            old = int(self.tables[s, b])
            self.tables[s, b] = e
            if _is_host(e):
                g = int(self.shadow[s, b])
                if g >= 0 and g != _slot_of(e):          # committed elsewhere: the copy goes
                    self._free_host(g)
                self.shadow[s, b] = -1
            if old >= 0:
                self.owner_hbm[old] = (-1, -1)
                self.hbm_used[old] = False
            elif _is_host(old):
                if self.inclusive and e >= 0:            # the host copy stays, clean
                    self.shadow[s, b] = _slot_of(old)
                else:
                    self._free_host(_slot_of(old))
        if int(self.hbm_used.sum()) > self.budget:
            raise OracleError("BUDGET", "HBM budget exceeded after commit")

    def _free_host(self, h: int) -> None:
        self.owner_host[h] = (-1, -1)
        self.host_used[h] = False

    def cancel(self, locs) -> None:
        """Release reservations that were never committed (Section 5.2, a cancelled preload)."""
        for e in np.asarray(locs):
            e = int(e)
            if e >= 0:
                if not self.hbm_used[e] or self.owner_hbm[e, 0] != -1:
                    raise OracleError("STATE", f"page {e} is not a pending reservation")
                self.hbm_used[e] = False
            elif _is_host(e):
                h = _slot_of(e)
                o_s, o_b = (int(x) for x in self.owner_host[h])
                if self.inclusive and o_s >= 0 and self.shadow[o_s, o_b] == h:
                    continue                             # a clean copy: nothing was reserved
                if not self.host_used[h] or o_s != -1:
                    raise OracleError("STATE", f"slot {h} is not a pending reservation")
                self.host_used[h] = False

    # ---------------------------------------------------------------- growth
    def append(self, sid: int, n_tokens: int) -> np.ndarray:
        """Grow a session's context; new blocks take the lowest free HBM pages (Section 5.1)."""
        new_ctx = int(self.ctx[sid]) + int(n_tokens)
        nb = -(-new_ctx // self.T)
        if nb > self.max_blocks:
            raise OracleError("BOUNDS", f"session {sid} would need {nb} blocks")
        first = int(self.nblocks[sid])
        pages = self.alloc_hbm(nb - first)
        tail = int(self.ctx[sid]) % self.T
        if n_tokens > 0 and tail and self.shadow[sid, first - 1] >= 0:
            # the partially filled last block gains rows: its clean copy is stale
            self._free_host(int(self.shadow[sid, first - 1]))
            self.shadow[sid, first - 1] = -1
            self.clean_dropped += 1
        for i, p in enumerate(pages):
            b = first + i
            self.tables[sid, b] = int(p)
            self.owner_hbm[p] = (sid, b)
        self.nblocks[sid] = nb
        self.ctx[sid] = new_ctx
        return pages

    # ----------------------------------------------------------------- views
    def page_checksum(self, page: int) -> int:
        """Position-weighted sum of an HBM page (an instrument, not from the paper):
        the 2L sub-pages concatenated in order, read as little-endian 64-bit words
        w_q, and sum_q w_q * (2q + 1) mod 2^64."""
        data = np.ascontiguousarray(self.hbm[:, int(page), :]).reshape(-1)
        w = data.view("<u8")
        weights = 2 * np.arange(w.size, dtype=np.uint64) + np.uint64(1)
        return int(np.sum(w * weights, dtype=np.uint64))

    def host_blocks(self, sid: int) -> np.ndarray:
        """Block indices of ``sid`` that live in host slots (Section 6)."""
        row = self.tables[sid, :int(self.nblocks[sid])]
        return np.nonzero(row <= -2)[0].astype(np.int64)

    def resident_count(self) -> int:
        """HBM pages in use (Section 5.1, the capacity check)."""
        return int(self.hbm_used.sum())

    def free_budget(self) -> int:
        """HBM pages still free under the budget (Section 5.1)."""
        return self.budget - self.resident_count()

    def clean_copies(self) -> int:
        """Host slots that still hold a clean copy of a resident block (inclusive tiers,
        a reading of Section 5)."""
        return int((self.shadow >= 0).sum())

    def check_invariants(self) -> None:
        """Owner tables and block tables (plus clean copies) are mutually inverse;
        budget holds (Section 6)."""
        n_hbm = n_host = n_clean = 0
        for s in range(self.S):
            for b in range(self.max_blocks):
                e = int(self.tables[s, b])
                g = int(self.shadow[s, b])
                if b >= self.nblocks[s]:
                    assert e == -1 and g == -1, (s, b, e, g)
                    continue
                if e >= 0:
                    assert tuple(self.owner_hbm[e]) == (s, b), (s, b, e)
                    n_hbm += 1
                else:
                    assert _is_host(e), (s, b, e)
                    assert tuple(self.owner_host[_slot_of(e)]) == (s, b), (s, b, e)
                    n_host += 1
                if g >= 0:
                    assert self.inclusive and e >= 0, (s, b, e, g)
                    assert tuple(self.owner_host[g]) == (s, b) and self.host_used[g], (s, b, g)
                    n_clean += 1
        assert int((self.owner_hbm[:, 0] >= 0).sum()) == n_hbm
        assert int((self.owner_host[:, 0] >= 0).sum()) == n_host + n_clean
        assert np.all(self.hbm_used[self.owner_hbm[:, 0] >= 0])
        assert np.all(self.host_used[self.owner_host[:, 0] >= 0])
        assert int(self.hbm_used.sum()) <= self.budget
