"""Per-session interaction state and how monitor events change it.

The runtime monitor (Section 3) reports how far playback has got, whether the user speaks, and
barge-ins; the KV manager keeps per-session side tables with the next-use
estimate's inputs and the preload-protection state (Section 6, "Hierarchical
KV cache manager").  This module is that state, updated one event at a time in
event order.  Times are integer microseconds.

Readings (the paper does not fix these):
  * T_reply is a moving average, kept per session, of how long the user takes
    to finish speaking again once the reply has played out (Section 5.1,
    after Eq. 4).
    Reading: an integer exponential moving average with weight 1/4,
    ``ema <- floor((3*ema + x) / 4)``; the first sample sets ``ema = x``.
  * A sample is taken at SPEECH_STOP (the user input is complete) when the
    current reply finished playing; a reply cut by a barge-in gives no sample.
  * Immediate-reuse protection (Section 5.1) lasts from speech start or
    barge-in until speech stop or the turn start.  Preload protection
    (Section 5.2) lasts ``protect_us`` from the preload's completion and ends
    at the next turn start (the warmed KV has then been reused).
  * A barge-in discards the unplayed part of the reply (Section 3), so the
    remaining playback becomes zero and the reply is finished without a
    completion time.

Parity status: the event updates are pinned by hand-worked timelines and by
invariants (a barge-in leaves no playback, protection ends at the turn start).
The EMA weight 1/4, the first-sample rule and the protection window are
readings: parity unpinned against the paper for those constants.
"""
from __future__ import annotations

from dataclasses import dataclass

# flag bits
RUNNING = 1        # the session's request is executing (pinned running KV)
IMMEDIATE = 2      # speech start or barge-in seen: immediate reuse
RESP_OPEN = 4      # the current reply is still unfinished
DONE_VALID = 8     # t_done_us holds the completion time of the current reply

# next-use estimate modes (Section 5.1)
MODE_PLAYBACK = 0  # T_play from playback accounting
MODE_COUNTERS = 1  # T_play from progress counters (fallback)

# state-level event kinds
SE_TURN_BEGIN = 1
SE_TURN_END = 2
SE_PLAYBACK = 3
SE_SPEECH_START = 4
SE_BARGE_IN = 5
SE_SPEECH_STOP = 6
SE_PRELOADED = 7

INT32_MAX = 2**31 - 1


@dataclass
class SessionState:
    """What the interaction monitor knows about one session (Section 5.1)."""

    ctx_tokens: int = 0
    flags: int = 0
    gen_us: int = 0            # audio generated for the current reply
    play_us: int = 0           # audio of it reported as played
    t_done_us: int = 0         # when playback of the current reply completed
    reply_ema_us: int = 0      # moving average of the reply interval
    reply_n: int = 0           # samples in the moving average
    reply_tokens: int = 0      # length of the current reply in progress units
    protect_until_us: int = 0  # preload protection ends at this time
    last_use_us: int = 0       # last turn begin or end (the LRU baseline's recency)

    def copy(self) -> "SessionState":
        return SessionState(**self.__dict__)


def apply_event(st: SessionState, kind: int, t_us: int, a: int = 0, b: int = 0,
                protect_us: int = 0) -> None:
    """Apply one monitor event to ``st`` in place (Sections 5.1 and 5.2)."""
    if kind == SE_TURN_BEGIN:
        # The turn's request runs: its KV is pinned running KV (Section 5, Fig. 6),
        # immediate-reuse ends, warmed KV has been reused (Section 5.2).
        st.flags = (st.flags | RUNNING) & ~IMMEDIATE
        st.protect_until_us = 0
        st.last_use_us = t_us
    elif kind == SE_TURN_END:
        # The LLM stage produced a reply of a = audio us, b = units; playback restarts.
        st.last_use_us = t_us
        st.flags &= ~(RUNNING | DONE_VALID)
        st.gen_us, st.play_us, st.reply_tokens = int(a), 0, int(b)
        if st.gen_us > 0:
            st.flags |= RESP_OPEN
        else:
            st.flags = (st.flags & ~RESP_OPEN) | DONE_VALID
            st.t_done_us = t_us
    elif kind == SE_PLAYBACK:
        # The client reports a more microseconds of audio as played (Section 3).
        if st.flags & RESP_OPEN:
            st.play_us = min(st.gen_us, st.play_us + int(a))
            if st.play_us >= st.gen_us:
                st.flags = (st.flags & ~RESP_OPEN) | DONE_VALID
                st.t_done_us = t_us
    elif kind == SE_SPEECH_START:
        st.flags |= IMMEDIATE
    elif kind == SE_BARGE_IN:
        # Audio not yet played is dropped on a barge-in (Section 3, barge-in handling).
        st.gen_us = st.play_us
        st.flags = (st.flags | IMMEDIATE) & ~(RESP_OPEN | DONE_VALID)
    elif kind == SE_SPEECH_STOP:
        # The next user input is complete: one sample of the reply interval.
        if st.flags & DONE_VALID:
            x = max(0, t_us - st.t_done_us)
            if st.reply_n == 0:
                st.reply_ema_us = x
            else:
                st.reply_ema_us = (3 * st.reply_ema_us + x) // 4
            st.reply_n = min(INT32_MAX, st.reply_n + 1)
        st.flags &= ~(IMMEDIATE | DONE_VALID)
    elif kind == SE_PRELOADED:
        # Warmed KV stays protected for a short time after the preload (Section 5.2).
        st.protect_until_us = t_us + protect_us
    else:
        raise ValueError(f"unknown session event kind {kind}")
