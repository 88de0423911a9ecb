"""Seeded event scripts and initial placements for the five workloads.

An event script is what the runtime monitor would deliver to the KV manager
(Section 3: playback progress, speech activity, barge-in; Section 5.2: speech
start and barge-in are preload triggers).  Events are plain records; what each
event *does* is defined by the consumer (the oracle or the library driver).

Script event kinds and arguments:

  EV_TURN(sid, a=append_tokens, b=reply_audio_us, c=reply_tokens)
      The session's next turn reaches the LLM stage: its context grows by
      ``append_tokens`` and it produces a reply of ``reply_audio_us`` of audio
      (``reply_tokens`` units for the progress-counter estimate).
  EV_TURN_ANY(sid=-1, d=row, a, b, c)
      As EV_TURN, but the session is the first id in ``perms[row]`` that has at
      least one block in the host tier at that moment (``perms[row][0]`` when
      none has).  Used by the turn-driven workloads so every turn reloads.
  EV_PLAYBACK(sid, a=delta_us)
      The client reports ``delta_us`` more of the current reply as played.
  EV_SPEECH_START(sid), EV_BARGE_IN(sid), EV_SPEECH_STOP(sid)
      Voice-activity signals; a barge-in is speech that starts while the
      session's reply is still playing.
  EV_TURN_SCATTER(sid=-1, d=row, a=scatter_key, b=reply_audio_us, c=reply_tokens)
      As EV_TURN_ANY (no context growth), but the session's host blocks are
      reloaded in the order ``scatter_order(scatter_key, blocks)`` instead of
      ascending block order.
  EV_EVICT(a=k)
      Memory pressure from elsewhere: k pages must be freed now.

Block-table placement encoding (the C-ABI's published encoding): entry >= 0 is
an HBM page id, -1 is "no block", entry <= -2 is host slot ``-(entry + 2)``.
"""
from __future__ import annotations

import heapq
from dataclasses import dataclass, field

import numpy as np

from .configs import PoolSpec, pool_spec

EV_TURN = 1
EV_TURN_ANY = 2
EV_PLAYBACK = 3
EV_SPEECH_START = 4
EV_BARGE_IN = 5
EV_SPEECH_STOP = 6
EV_TURN_SCATTER = 7
EV_EVICT = 8
EVENT_NAMES = {EV_TURN: "TURN", EV_TURN_ANY: "TURN_ANY", EV_PLAYBACK: "PLAYBACK",
               EV_SPEECH_START: "SPEECH_START", EV_BARGE_IN: "BARGE_IN",
               EV_SPEECH_STOP: "SPEECH_STOP", EV_TURN_SCATTER: "TURN_SCATTER",
               EV_EVICT: "EVICT"}

LOC_NONE = -1
SEC = 1_000_000


def encode_host(slot):
    """Host slot -> block-table entry (placement encoding of this module's docstring)."""
    return -(np.asarray(slot, dtype=np.int64) + 2)


def is_host(entry):
    return np.asarray(entry) <= -2


def host_slot(entry):
    return -(np.asarray(entry, dtype=np.int64) + 2)


@dataclass
class InitialState:
    ctx_tokens: np.ndarray       # int32 [S]
    placement: np.ndarray        # int32 [S, max_blocks], encoded locations
    gen_us: np.ndarray           # int64 [S] audio generated for the current reply
    play_us: np.ndarray          # int64 [S] audio of it already played
    resp_open: np.ndarray        # int32 [S] 1 while the current reply is unfinished
    reply_tokens: np.ndarray     # int32 [S] length of the current reply in units


@dataclass
class Workload:
    spec: PoolSpec
    seed: int
    init: InitialState
    t_us: np.ndarray             # int64 [E], non-decreasing
    kind: np.ndarray             # int32 [E]
    sid: np.ndarray              # int32 [E]
    a: np.ndarray                # int64 [E]
    b: np.ndarray                # int64 [E]
    c: np.ndarray                # int64 [E]
    d: np.ndarray                # int32 [E] row of ``perms`` for EV_TURN_ANY, else -1
    perms: np.ndarray            # int32 [R, S]
    meta: dict = field(default_factory=dict)

    @property
    def n_events(self) -> int:
        return int(self.t_us.shape[0])

    def event(self, i: int):
        return (int(self.t_us[i]), int(self.kind[i]), int(self.sid[i]), int(self.a[i]),
                int(self.b[i]), int(self.c[i]), int(self.d[i]))


def scatter_order(key, blocks) -> np.ndarray:
    """A seeded permutation of ``blocks`` (the random scatter order of a reload)."""
    from .content import _splitmix64
    blocks = np.asarray(blocks, dtype=np.int64)
    h = _splitmix64(np.uint64(key & 0xFFFFFFFFFFFF) * np.uint64(1 << 16)
                    + blocks.astype(np.uint64) * np.uint64(2654435761))
    return blocks[np.argsort(h, kind="stable")]


def _pack_events(rows, S):
    if rows:
        arr = np.array([r[:7] for r in rows], dtype=np.int64)
    else:
        arr = np.zeros((0, 7), dtype=np.int64)
    return (arr[:, 0].copy(), arr[:, 1].astype(np.int32), arr[:, 2].astype(np.int32),
            arr[:, 3].copy(), arr[:, 4].copy(), arr[:, 5].copy(), arr[:, 6].astype(np.int32))


def _pages(ctx, T):
    return (np.asarray(ctx, dtype=np.int64) + T - 1) // T


def _place_fill(n_pages, max_blocks, budget, host_pages, page_perm=None):
    """Blocks in (sid, blk) order take HBM pages until ``budget`` is used, then host slots.

    ``page_perm`` (optional) maps the k-th HBM page handed out to a physical page id,
    which scatters sessions across the pool.
    """
    S = len(n_pages)
    placement = np.full((S, max_blocks), LOC_NONE, dtype=np.int32)
    next_page, next_slot = 0, 0
    for s in range(S):
        for blk in range(int(n_pages[s])):
            if next_page < budget:
                p = next_page if page_perm is None else int(page_perm[next_page])
                placement[s, blk] = p
                next_page += 1
            else:
                if next_slot >= host_pages:
                    raise ValueError("initial placement does not fit in the host pool")
                placement[s, blk] = int(encode_host(next_slot))
                next_slot += 1
    return placement


def _log_uniform_tokens(rng, lo, hi, n):
    return np.round(np.exp(rng.uniform(np.log(lo), np.log(hi), n))).astype(np.int64)


# --------------------------------------------------------------------------------------
# Interactive sessions (tiny, mixed): per-session voice loop
#   TURN -> playback reports -> (speech start | barge-in) -> speech stop -> TURN ...
# The next user speech arrives a random gap after the turn; if that gap ends before
# the reply has finished playing the speech is a barge-in.
# --------------------------------------------------------------------------------------
def _interactive(spec: PoolSpec, seed: int, n_events: int, ctx_lo: int, ctx_hi: int,
                 log_uniform_ctx: bool, gap_mean_us: int, gap_exponential: bool,
                 reply_lo_us: int, reply_hi_us: int, speech_lo_us: int, speech_hi_us: int,
                 append_lo: int, append_hi: int, report_us: int = SEC,
                 delay_lo_us: int = 50_000, delay_hi_us: int = 300_000,
                 all_resident: bool = True) -> Workload:
    rng = np.random.default_rng(seed)
    S, T = spec.n_sessions, spec.shape.page_tokens
    cap_tokens = spec.max_blocks * T
    size_host_after = spec.host_pages == 0 and not all_resident
    if log_uniform_ctx:
        ctx = _log_uniform_tokens(rng, ctx_lo, ctx_hi, S)
    else:
        ctx = rng.integers(ctx_lo, ctx_hi + 1, S).astype(np.int64)
    ctx = np.minimum(ctx, cap_tokens)
    n_pages = _pages(ctx, T)
    if all_resident and int(n_pages.sum()) > spec.hbm_budget_pages:
        raise ValueError("initial contexts exceed the HBM budget")
    host_pages = spec.host_pages
    if host_pages == 0:
        # room for every session, plus growth; shrunk below once the script is known
        host_pages = int(n_pages.sum()) + S * spec.max_blocks
        spec = spec.with_(host_pages=host_pages)
    placement = _place_fill(n_pages, spec.max_blocks, spec.hbm_budget_pages, host_pages)

    def gap():
        if gap_exponential:
            return int(rng.exponential(gap_mean_us))
        return int(rng.uniform(0.25 * gap_mean_us, 1.75 * gap_mean_us))

    gen0 = rng.integers(reply_lo_us, reply_hi_us + 1, S).astype(np.int64)
    play0 = (rng.uniform(0.0, 1.0, S) * gen0).astype(np.int64)
    play0 = (play0 // report_us) * report_us                 # positions the client reported
    rtok0 = (gen0 // spec.unit_us).astype(np.int32)
    resp_open = (play0 < gen0).astype(np.int32)
    init = InitialState(ctx.astype(np.int32), placement, gen0, play0.copy(), resp_open, rtok0)

    rows = []
    heap = []          # (t, seq, sid, action, payload)
    seq = 0

    def push(t, s, action, payload=None):
        nonlocal seq
        heapq.heappush(heap, (int(t), seq, s, action, payload))
        seq += 1

    # per-session generator state
    gen = gen0.copy()
    play = play0.copy()
    cur_ctx = ctx.copy()
    for s in range(S):
        # the reply started play0 ago; the next user speech comes `gap` after it started
        t_start = -int(play0[s])
        t_speech = t_start + gap()
        if t_speech <= 0:
            t_speech = int(rng.integers(0, report_us))
        if play[s] < gen[s]:
            push(report_us, s, "report", t_speech)
        else:
            push(max(t_speech, 1), s, "speech", None)

    while len(rows) < n_events and heap:
        t, _, s, action, payload = heapq.heappop(heap)
        if action == "report":
            t_speech = payload
            if t_speech <= t and play[s] < gen[s]:
                # the user speaks while the reply is still playing: barge-in
                tb = max(t_speech, t - report_us + 1)
                rows.append((tb, EV_BARGE_IN, s, 0, 0, 0, -1))
                gen[s] = play[s]
                push(tb + int(rng.integers(speech_lo_us, speech_hi_us + 1)), s, "stop", None)
                continue
            delta = int(min(report_us, gen[s] - play[s]))
            rows.append((t, EV_PLAYBACK, s, delta, 0, 0, -1))
            play[s] += delta
            if play[s] < gen[s]:
                push(t + report_us, s, "report", t_speech)
            else:
                push(max(t_speech, t + 1), s, "speech", None)
        elif action == "speech":
            rows.append((t, EV_SPEECH_START, s, 0, 0, 0, -1))
            push(t + int(rng.integers(speech_lo_us, speech_hi_us + 1)), s, "stop", None)
        elif action == "stop":
            rows.append((t, EV_SPEECH_STOP, s, 0, 0, 0, -1))
            push(t + int(rng.integers(delay_lo_us, delay_hi_us + 1)), s, "turn", None)
        elif action == "turn":
            app = int(rng.integers(append_lo, append_hi + 1))
            app = int(min(app, cap_tokens - cur_ctx[s]))
            cur_ctx[s] += app
            reply = int(rng.integers(reply_lo_us, reply_hi_us + 1))
            rtok = reply // spec.unit_us
            rows.append((t, EV_TURN, s, app, reply, rtok, -1))
            gen[s], play[s] = reply, 0
            push(t + report_us, s, "report", t + gap())
    rows.sort(key=lambda r: r[0])   # stable: equal times keep generation order
    rows = rows[:n_events]
    t_us, kind, sid, a, b, c, d = _pack_events(rows, S)
    meta = {}
    if size_host_after:
        # every block that can exist, minus what the budget holds, plus two sessions of slack
        grown = ctx.copy()
        for r in rows:
            if r[1] == EV_TURN:
                grown[r[2]] += r[3]
        total = int(_pages(grown, T).sum())
        host = max(int(n_pages.sum()) - spec.hbm_budget_pages, total - spec.hbm_budget_pages, 0) \
            + 2 * spec.max_blocks
        if spec.tiers == 1:          # inclusive tiers: room for a host copy of every block
            host = total + 2 * spec.max_blocks
        spec = spec.with_(host_pages=host)
        meta["total_pages_final"] = total
    meta["total_pages"] = int(n_pages.sum())
    return Workload(spec, seed, init, t_us, kind, sid, a, b, c, d,
                    np.zeros((0, S), dtype=np.int32), meta=meta)


# --------------------------------------------------------------------------------------
# Turn-driven sessions (thinker): every turn reloads an offloaded session.
# --------------------------------------------------------------------------------------
def _turns(spec: PoolSpec, seed: int, n_turns: int, ctx_lo: int, ctx_hi: int,
           reply_lo_us: int, reply_hi_us: int, step_us: int, ctx_dist: str = "log",
           frame_fraction: float = 0.0) -> Workload:
    rng = np.random.default_rng(seed)
    S, T = spec.n_sessions, spec.shape.page_tokens
    need = spec.hbm_budget_pages + spec.max_blocks
    # Contexts are log-uniform (or uniform); draws whose total KV exceeds the budget by
    # less than one largest possible session are redrawn, so every turn must evict.
    for _ in range(1000):
        if ctx_dist == "log":
            raw = _log_uniform_tokens(rng, ctx_lo, ctx_hi, S)
        else:
            raw = rng.integers(ctx_lo, ctx_hi + 1, S).astype(np.int64)
        ctx = np.minimum(raw, spec.max_blocks * T)
        n_pages = _pages(ctx, T)
        if int(n_pages.sum()) >= need:
            break
    else:
        raise RuntimeError("could not draw contexts that exceed the budget")
    total = int(n_pages.sum())
    host_pages = spec.host_pages or (total - spec.hbm_budget_pages + 2 * spec.max_blocks
                                     if spec.tiers == 0 else total + 2 * spec.max_blocks)
    spec = spec.with_(host_pages=host_pages)
    placement = _place_fill(n_pages, spec.max_blocks, spec.hbm_budget_pages, host_pages)
    gen0 = rng.integers(reply_lo_us, reply_hi_us + 1, S).astype(np.int64)
    play0 = (rng.uniform(0.0, 1.0, S) * gen0).astype(np.int64)
    rtok0 = (gen0 // spec.unit_us).astype(np.int32)
    init = InitialState(ctx.astype(np.int32), placement, gen0, play0, np.ones(S, np.int32), rtok0)
    rows = []
    perms = np.zeros((n_turns, S), dtype=np.int32)
    for i in range(n_turns):
        t = (i + 1) * step_us
        for s in range(S):
            rows.append((t, EV_PLAYBACK, s, step_us, 0, 0, -1))
        perms[i] = rng.permutation(S)
        reply = int(rng.integers(reply_lo_us, reply_hi_us + 1))
        rows.append((t, EV_TURN_ANY, -1, 0, reply, reply // spec.unit_us, i))
    t_us, kind, sid, a, b, c, d = _pack_events(rows, S)
    meta = {"total_pages": total}
    if frame_fraction > 0:
        meta["frame_spans"] = _frame_spans(rng, ctx, frame_fraction)
    return Workload(spec, seed, init, t_us, kind, sid, a, b, c, d, perms, meta=meta)


def _frame_spans(rng, ctx, fraction, frame_tokens=256):
    """Token spans that came from dense image / video frames (a modality tag only:
    the KV of a frame token moves like any other)."""
    spans = []
    for c in ctx:
        want = int(fraction * int(c)) // frame_tokens
        starts = np.sort(rng.choice(max(1, int(c) // frame_tokens), size=min(want, max(1, int(c) // frame_tokens)),
                                    replace=False)) * frame_tokens
        spans.append([(int(x), frame_tokens) for x in starts])
    return spans


# --------------------------------------------------------------------------------------
# Fragmentation stress (frag): a pool whose pages start randomly permuted; events
# alternate "free k pages" and a turn whose reload list comes in a scattered order.
# --------------------------------------------------------------------------------------
def _frag(spec: PoolSpec, seed: int, n_events: int, ctx_lo: int, ctx_hi: int,
          evict_lo: int, evict_hi: int, reply_lo_us: int, reply_hi_us: int, step_us: int) -> Workload:
    rng = np.random.default_rng(seed)
    S, T = spec.n_sessions, spec.shape.page_tokens
    for _ in range(1000):
        ctx = np.minimum(rng.integers(ctx_lo, ctx_hi + 1, S).astype(np.int64), spec.max_blocks * T)
        n_pages = _pages(ctx, T)
        if int(n_pages.sum()) >= spec.hbm_budget_pages + 2 * spec.max_blocks:
            break
    else:
        raise RuntimeError("could not draw contexts that exceed the budget")
    total = int(n_pages.sum())
    keep = total if spec.tiers == 1 else total - spec.hbm_budget_pages   # inclusive: every block
    host_pages = spec.host_pages or (keep + max(total // 10, 2 * spec.max_blocks) + evict_hi)
    spec = spec.with_(host_pages=host_pages)
    perm = rng.permutation(spec.hbm_pages)
    placement = _place_fill(n_pages, spec.max_blocks, spec.hbm_budget_pages, host_pages, page_perm=perm)
    gen0 = rng.integers(reply_lo_us, reply_hi_us + 1, S).astype(np.int64)
    play0 = (rng.uniform(0.0, 1.0, S) * gen0).astype(np.int64)
    rtok0 = (gen0 // spec.unit_us).astype(np.int32)
    init = InitialState(ctx.astype(np.int32), placement, gen0, play0, np.ones(S, np.int32), rtok0)
    rows = []
    n_turns = (n_events + 1) // 2
    perms = np.zeros((n_turns, S), dtype=np.int32)
    for i in range(n_events):
        t = (i + 1) * step_us
        if i % 2 == 0:
            rows.append((t, EV_EVICT, -1, int(rng.integers(evict_lo, evict_hi + 1)), 0, 0, -1))
        else:
            r = i // 2
            perms[r] = rng.permutation(S)
            reply = int(rng.integers(reply_lo_us, reply_hi_us + 1))
            rows.append((t, EV_TURN_SCATTER, -1, int(rng.integers(0, 2**40)), reply,
                         reply // spec.unit_us, r))
    t_us, kind, sid, a, b, c, d = _pack_events(rows, S)
    return Workload(spec, seed, init, t_us, kind, sid, a, b, c, d, perms[: (n_events // 2)],
                    meta={"total_pages": total})


def make_workload(name: str, seed: int = 0, host_limit=None, **over) -> Workload:
    """Build the seeded workload ``name`` (see ``workloads.configs.CONFIG_NAMES``).

    Keyword overrides change the scale (e.g. ``n_events``, ``n_turns``, ``spec``).
    ``host_limit`` (bytes, for a caller that page-locks the host tier): when the
    workload's host tier would exceed it, the session count is scaled down by the
    ratio of the two and the script drawn again (then by 1 % steps until it fits);
    ``meta["sizing"]`` records the limit, the stated and the used session counts.
    """
    if host_limit is None:
        return _make(name, seed, **over)
    wl = _make(name, seed, **dict(over))
    n0 = wl.spec.n_sessions
    need = wl.spec.host_pages * wl.spec.shape.page_bytes
    n = n0
    # the host tier is about (all pages - budget + slack): linear in the session count
    per_session = (need + wl.spec.hbm_budget_pages * wl.spec.shape.page_bytes) / max(n0, 1)
    while need > host_limit and n > 1:
        guess = int((host_limit + wl.spec.hbm_budget_pages * wl.spec.shape.page_bytes) / per_session)
        n = max(1, min(n - 1, guess))
        sp = (over.get("spec") or pool_spec(name)).with_(n_sessions=n)
        wl = _make(name, seed, **dict(over, spec=sp))
        need = wl.spec.host_pages * wl.spec.shape.page_bytes
    # the estimate may undershoot: take the largest count that still fits
    while wl.spec.n_sessions < n0 and need <= host_limit:
        sp = (over.get("spec") or pool_spec(name)).with_(n_sessions=wl.spec.n_sessions + 1)
        nxt = _make(name, seed, **dict(over, spec=sp))
        nneed = nxt.spec.host_pages * nxt.spec.shape.page_bytes
        if nneed > host_limit:
            break
        wl, need = nxt, nneed
    wl.meta["sizing"] = {"host_limit_bytes": int(host_limit), "stated_sessions": n0,
                         "sessions": wl.spec.n_sessions, "host_tier_bytes": int(need),
                         "scaled": wl.spec.n_sessions != n0}
    return wl


def _make(name: str, seed: int = 0, **over) -> Workload:
    spec = over.pop("spec", None) or pool_spec(name)
    if name == "tiny":
        kw = dict(n_events=1000, ctx_lo=64, ctx_hi=512, log_uniform_ctx=False,
                  gap_mean_us=6 * SEC, gap_exponential=False,
                  reply_lo_us=2 * SEC, reply_hi_us=12 * SEC,
                  speech_lo_us=1 * SEC, speech_hi_us=4 * SEC,
                  append_lo=16, append_hi=96)
        kw.update(over)
        return _interactive(spec, seed, **kw)
    if name == "thinker":
        kw = dict(n_turns=210, ctx_lo=2048, ctx_hi=16384,
                  reply_lo_us=5 * SEC, reply_hi_us=30 * SEC, step_us=500_000)
        kw.update(over)
        return _turns(spec, seed, **kw)
    if name == "mixed":
        kw = dict(n_events=3000, ctx_lo=2048, ctx_hi=16384, log_uniform_ctx=True,
                  gap_mean_us=8 * SEC, gap_exponential=True,
                  reply_lo_us=5 * SEC, reply_hi_us=30 * SEC,
                  speech_lo_us=2 * SEC, speech_hi_us=10 * SEC,
                  append_lo=16, append_hi=96, all_resident=False)
        kw.update(over)
        return _interactive(spec, seed, **kw)
    if name == "long":
        kw = dict(n_turns=16, ctx_lo=32768, ctx_hi=65536, ctx_dist="uniform",
                  reply_lo_us=5 * SEC, reply_hi_us=30 * SEC, step_us=500_000, frame_fraction=0.3)
        kw.update(over)
        return _turns(spec, seed, **kw)
    if name == "frag":
        kw = dict(n_events=10_000, ctx_lo=256, ctx_hi=4096, evict_lo=8, evict_hi=128,
                  reply_lo_us=5 * SEC, reply_hi_us=30 * SEC, step_us=100_000)
        kw.update(over)
        return _frag(spec, seed, **kw)
    raise ValueError(f"unknown workload {name!r}")
