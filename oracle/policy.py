"""Next-use estimate, eviction eligibility and victim order (Section 5.1).

Victim order, two formulations that must agree exactly:
  A (``order_global``): every eligible HBM-resident block, sorted by
    (T_next descending, session id ascending, block id descending).
  B (``order_scan``): the paper's procedure -- order eligible sessions by
    decreasing T_next, take blocks from the farthest session, suffix blocks
    first, then continue with the next session.

Readings:
  * Ties in T_next are broken by session id ascending; within a session the
    suffix-first rule (Section 5.1, last paragraph) orders blocks by
    decreasing block id.  ``ASCENDING`` orders them by increasing block id
    instead (the literal "(session id, block id) ascending" tie-break).
  * T_next is clamped to [0, 2^32 - 1] microseconds; the paper asks only for
    an ordering signal, not a precise forecast of the time (Section 5.1).
  * T_play in the progress-counter mode is the current reply's length in
    units times ``unit_us`` while the reply is unfinished, else 0 (the paper
    reads a reply that is still long and open as reuse further away, Section
    5.1); like the playback
    horizon it is never negative.
  * Protection holds against *normal* eviction only (Section 5.1), and warmed
    KV may still be evicted before it is reused (Section 5.2).  With ``fallback`` set (a
    foreground turn that cannot otherwise run), protected sessions that are
    not running form a second tier, ordered by the same rule after every
    normally eligible block.  Pinned running KV is never a candidate.

Parity status: formulation A is pinned against formulation B, against brute
force over all block orders on tiny pools, and against hand-worked orders of
Section 5.1's rules.  The tie-breaks and the T_play reading of the counter
mode are readings: parity unpinned against the paper for those choices.
"""
from __future__ import annotations

import numpy as np

from .sessions import (SessionState, RUNNING, IMMEDIATE, RESP_OPEN, MODE_PLAYBACK,
                       MODE_COUNTERS)

KEY_MAX = 2**32 - 1
SUFFIX_FIRST = 0
ASCENDING = 1
NEXT_USE = 0        # the paper's order (Section 5.1)
LRU = 1             # the substrate's least-recently-used baseline (Sections 2.3, 5)


def t_next(st: SessionState, mode: int, reply_prior_us: int, unit_us: int) -> int:
    """Eq. 4: T_next = T_play + T_reply for one session (clamped to 32 bits)."""
    if mode == MODE_PLAYBACK:
        t_play = max(0, st.gen_us - st.play_us)            # audio still to play
    elif mode == MODE_COUNTERS:
        t_play = max(0, st.reply_tokens * unit_us) if (st.flags & RESP_OPEN) else 0
    else:
        raise ValueError(f"unknown T_play mode {mode}")
    # the session's own average once it has a sample, else the workload prior
    t_reply = st.reply_ema_us if st.reply_n > 0 else reply_prior_us
    return min(KEY_MAX, max(0, t_play + t_reply))


next_use_key = t_next


def is_eligible(st: SessionState, now_us: int) -> bool:
    """Eviction takes only multi-turn KV that sits in HBM unused (Section 5.1, Eviction policy):
    pinned running KV, immediate-reuse sessions (speech start / barge-in) and
    preload-protected sessions (Section 5.2) are excluded."""
    if st.flags & (RUNNING | IMMEDIATE):
        return False
    if now_us < st.protect_until_us:
        return False
    return True


def tier(st: SessionState, now_us: int, fallback: bool):
    """0: normally eligible; 1: protected, a candidate only with ``fallback``; None: never (Section 5.1 eligibility; Section 5.2 protection)."""
    if is_eligible(st, now_us):
        return 0
    if fallback and not (st.flags & RUNNING):
        return 1
    return None


def order_lru(tables, nblocks, sessions, within=SUFFIX_FIRST):
    """The LRU baseline: every HBM-resident block of a session that is not running,
    least recently used session first (last turn time ascending, then session id
    ascending), suffix blocks first within a session.  Immediate reuse and preload
    protection do not exist for it (Sections 2.3 and 5)."""
    cands = [(s, st.last_use_us) for s, st in enumerate(sessions) if not (st.flags & RUNNING)]
    cands.sort(key=lambda c: (min(max(c[1], 0), KEY_MAX), c[0]))
    out_s, out_b, out_p = [], [], []
    for s, _ in cands:
        n = int(nblocks[s])
        rng = range(n - 1, -1, -1) if within == SUFFIX_FIRST else range(n)
        for b in rng:
            e = int(tables[s][b])
            if e >= 0:
                out_s.append(s)
                out_b.append(b)
                out_p.append(e)
    return (np.array(out_s, dtype=np.int64), np.array(out_b, dtype=np.int64),
            np.array(out_p, dtype=np.int64))


def _resident_blocks(table_row: np.ndarray, nblocks: int) -> np.ndarray:
    row = table_row[:nblocks]
    return np.nonzero(row >= 0)[0]


def order_global(tables, nblocks, sessions, now_us, mode, reply_prior_us, unit_us,
                 within=SUFFIX_FIRST, fallback=False):
    """Formulation A. Returns int64 arrays (sid, blk, page) of the full victim order (Section 5.1)."""
    sids, blks, keys, tiers = [], [], [], []
    for s, st in enumerate(sessions):
        tr = tier(st, now_us, fallback)
        if tr is None:
            continue
        b = _resident_blocks(tables[s], int(nblocks[s]))
        if b.size == 0:
            continue
        sids.append(np.full(b.size, s, dtype=np.int64))
        blks.append(b.astype(np.int64))
        keys.append(np.full(b.size, t_next(st, mode, reply_prior_us, unit_us), dtype=np.int64))
        tiers.append(np.full(b.size, tr, dtype=np.int64))
    if not sids:
        z = np.zeros(0, dtype=np.int64)
        return z, z.copy(), z.copy()
    sid = np.concatenate(sids)
    blk = np.concatenate(blks)
    key = np.concatenate(keys)
    tr = np.concatenate(tiers)
    blk_key = -blk if within == SUFFIX_FIRST else blk
    # np.lexsort sorts by the LAST key first: tier, then -T_next, then sid, then block
    order = np.lexsort((blk_key, sid, -key, tr))
    sid, blk = sid[order], blk[order]
    page = np.asarray(tables)[sid, blk].astype(np.int64)
    return sid, blk, page


def order_scan(tables, nblocks, sessions, now_us, mode, reply_prior_us, unit_us,
               within=SUFFIX_FIRST, k=None, fallback=False):
    """Formulation B (the paper's session scan). Returns (sid, blk, page) lists (Section 5.1)."""
    elig = []
    for s, st in enumerate(sessions):
        tr = tier(st, now_us, fallback)
        if tr is not None:
            elig.append((tr, t_next(st, mode, reply_prior_us, unit_us), s))
    # normal tier first; decreasing T_next; equal T_next by increasing session id
    elig.sort(key=lambda e: (e[0], -e[1], e[2]))
    out_s, out_b, out_p = [], [], []
    for _, _, s in elig:
        n = int(nblocks[s])
        rng = range(n - 1, -1, -1) if within == SUFFIX_FIRST else range(n)
        for b in rng:
            if k is not None and len(out_s) >= k:
                return out_s, out_b, out_p
            e = int(tables[s][b])
            if e >= 0:
                out_s.append(s)
                out_b.append(b)
                out_p.append(e)
    return out_s, out_b, out_p


def select_victims(tables, nblocks, sessions, now_us, k, mode, reply_prior_us, unit_us,
                   within=SUFFIX_FIRST, fallback=False):
    """The first min(k, #candidates) blocks of the victim order (Section 5.1)."""
    sid, blk, page = order_global(tables, nblocks, sessions, now_us, mode,
                                  reply_prior_us, unit_us, within, fallback)
    k = min(int(k), sid.size)
    return sid[:k], blk[:k], page[:k]
