"""Seeded synthetic inputs for the KV swap path: pool shapes, initial placements,
event scripts and KV page contents.

This package generates INPUTS only.  It holds none of the method's arithmetic
(no next-use score, no eligibility rule, no victim order, no allocation rule,
no copy or remap semantics); both the CPU oracle and the CUDA path consume the
same generated inputs, and neither is imported here.
"""
from .configs import (  # noqa: F401
    KVShape, PoolSpec, TINY_SHAPE, THINKER_SHAPE, CONFIG_NAMES, pool_spec, GB,
    STATED_SESSIONS, host_tier_limit, mem_available_bytes,
)
from .scripts import (  # noqa: F401
    Workload, InitialState, make_workload,
    EV_TURN, EV_TURN_ANY, EV_PLAYBACK, EV_SPEECH_START, EV_BARGE_IN, EV_SPEECH_STOP,
    EV_TURN_SCATTER, EV_EVICT, EVENT_NAMES, LOC_NONE, encode_host, is_host, host_slot,
    scatter_order,
)
from .content import (  # noqa: F401
    TABLE_LEN, value_table, subpage_offsets, subpage_values_np, subpage_values_torch,
    valid_rows,
)
