"""The interaction-aware request scheduler of Section 4 (Algorithm 1, Eqs. 1-3).

For one scheduling round of one stage:
  * each ready request i has a playback buffer P_i (microseconds of audio the
    client holds), whether it has produced its first playable audio, a ready
    age A_i, the KV pages it occupies K_i, and the token and KV-block cost of
    admitting it;
  * class 0 (playback urgency): started and P_i <= P_safe, ordered by P_i
    ascending; class 1 (first-audio urgency): not started, ordered by A_i
    descending (FCFS aging); class 2 (efficiency): started and P_i > P_safe,
    ordered by the utility U_i descending, with (Eqs. 1-3)
        U_i = beta * U_kv - alpha * C_barge,
        C_barge = max(0, P_i - P_safe) / P_safe,   U_kv = K_i * R_occ,
        R_occ = occupied / allocatable GPU KV;
  * the classes are concatenated 0-1-2 and scanned: admission stops at the
    first request that does not fit the remaining token or KV budget.

Readings: ties inside a class keep the ready set's order (the earlier request
first); the utility is evaluated in exact rational arithmetic (no rounding).  Parity unpinned for the
stage constants (P_safe, alpha, beta), which the paper tunes offline.
"""
from __future__ import annotations

from fractions import Fraction


def classify(started: bool, play_buffer_us: int, p_safe_us: int) -> int:
    """Urgency class (Section 4.1): 0 playback at risk, 1 not yet started, 2 safe."""
    if not started:
        return 1
    return 0 if play_buffer_us <= p_safe_us else 2


def utility(kv_pages, play_buffer_us, p_safe_us, alpha, beta, occupied, allocatable) -> Fraction:
    """Eq. 1 with Eq. 2 (barge-in exposure) and Eq. 3 (KV-pressure benefit)."""
    c_barge = Fraction(max(0, play_buffer_us - p_safe_us), p_safe_us)
    u_kv = kv_pages * Fraction(occupied, allocatable)
    return beta * u_kv - alpha * c_barge


def schedule(requests, p_safe_us, alpha, beta, occupied, allocatable, token_budget, kv_budget):
    """Algorithm 1.  ``requests``: dicts with id, started, play_buffer_us, ready_age_us,
    kv_pages, tokens, kv_needed.  Returns (priority order of ids, admitted batch of ids)."""
    c = {0: [], 1: [], 2: []}
    for pos, r in enumerate(requests):
        g = classify(bool(r["started"]), r["play_buffer_us"], p_safe_us)
        if g == 0:
            c[0].append((r["play_buffer_us"], pos, r))
        elif g == 1:
            c[1].append((-r["ready_age_us"], pos, r))
        else:
            u = utility(r["kv_pages"], r["play_buffer_us"], p_safe_us, alpha, beta, occupied, allocatable)
            c[2].append((-u, pos, r))
    order = []
    for g in (0, 1, 2):
        order += [x[2] for x in sorted(c[g], key=lambda x: (x[0], x[1]))]
    batch = []
    tok, kv = token_budget, kv_budget
    for r in order:
        if r["tokens"] > tok or r["kv_needed"] > kv:
            break
        batch.append(r["id"])
        tok -= r["tokens"]
        kv -= r["kv_needed"]
    return [r["id"] for r in order], batch
