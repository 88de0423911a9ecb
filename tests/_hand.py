"""Builds a Workload from a hand-written scenario (tests/golden/*_hand.json): a tiny-shape
pool, an initial placement and an event list.  Inputs only; no decision is made here."""
import json
import os

import numpy as np

from workloads.configs import PoolSpec, TINY_SHAPE
from workloads.scripts import (InitialState, Workload, EV_TURN, EV_PLAYBACK, EV_SPEECH_START,
                               EV_SPEECH_STOP, EV_BARGE_IN, EV_EVICT)

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")
KINDS = {"TURN": EV_TURN, "PLAYBACK": EV_PLAYBACK, "SPEECH_START": EV_SPEECH_START,
         "SPEECH_STOP": EV_SPEECH_STOP, "BARGE_IN": EV_BARGE_IN, "EVICT": EV_EVICT}


def load(name):
    with open(os.path.join(GOLDEN, name)) as f:
        return json.load(f)


def hand_workload(sc, seed=0):
    """sc: {"pool": {...}, "initial": {"ctx_tokens", "placement"}, "events": [...]}; every
    session starts with no reply in progress."""
    p = sc["pool"]
    spec = PoolSpec("hand", TINY_SHAPE, n_sessions=p["n_sessions"], max_blocks=p["max_blocks"],
                    hbm_pages=p["hbm_pages"], hbm_budget_pages=p["hbm_budget_pages"],
                    host_pages=p["host_pages"], reply_prior_us=p["reply_prior_us"],
                    protect_us=p["protect_us"])
    S, ev = spec.n_sessions, sc["events"]
    z = np.zeros(S, np.int64)
    init = InitialState(ctx_tokens=np.array(sc["initial"]["ctx_tokens"], np.int32),
                        placement=np.array(sc["initial"]["placement"], np.int32),
                        gen_us=z.copy(), play_us=z.copy(), resp_open=np.zeros(S, np.int32),
                        reply_tokens=np.zeros(S, np.int32))
    col = lambda key, dt: np.array([e.get(key, 0) for e in ev], dt)
    return Workload(spec=spec, seed=seed, init=init, t_us=col("t", np.int64),
                    kind=np.array([KINDS[e["ev"]] for e in ev], np.int32),
                    sid=np.array([e.get("sid", -1) for e in ev], np.int32),
                    a=col("a", np.int64), b=col("b", np.int64), c=np.zeros(len(ev), np.int64),
                    d=np.full(len(ev), -1, np.int32), perms=np.zeros((0, S), np.int32))
