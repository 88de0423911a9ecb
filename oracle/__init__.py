"""CPU oracle for the interaction-aware KV swap path (test infrastructure only).

This package is the plain, slow, obviously-correct reference that the CUDA
library is checked against.  It is NOT part of the product: only the test
suite, ``__graft_entry__.smoke()`` and the CPU-baseline leg of ``bench.py`` may
import it.  It shares no code with the CUDA path and does not import it.

Modules
  sessions  per-session interaction state and its event updates (Sections 3, 5.1, 5.2)
  policy    next-use estimate (Eq. 4), eligibility, victim order (Section 5.1)
  pool      paged block pool: block tables, owners, allocation, copy, remap;
            exclusive and inclusive tiers; page checksums (an instrument)
  manager   the KV manager's turn / preload procedure driven by an event script
  preload   the preload controller (Section 5.2): admission, wait, deferred
            commit, cancellation, the cap on protected KV
  scheduler the interaction-aware request scheduler (Section 4, Algorithm 1)

Readings of the paper where it is silent or ambiguous are listed in each
function's docstring (and collected in the repository's design notes).

Parity status: the victim order, allocation, copy and remap are pinned by
brute force, closed forms and invariants in ``tests/test_oracle_*.py``.  The
policy constants (EMA weight 1/4, the 3 s reply prior, the 2 s protection
window) are readings, not values printed by the paper: parity unpinned
against the paper for those constants.  The same holds for the inclusive-tier
rules, the controller's admission model and the scheduler's constants; each
module's header lists its readings and which of them stay unpinned.
"""
from .sessions import (  # noqa: F401
    SessionState, RUNNING, IMMEDIATE, RESP_OPEN, DONE_VALID, apply_event,
    MODE_PLAYBACK, MODE_COUNTERS,
)
from .policy import (  # noqa: F401
    t_next, next_use_key, is_eligible, order_global, order_scan, select_victims,
    SUFFIX_FIRST, ASCENDING, KEY_MAX,
)
from .pool import OraclePool, OracleError  # noqa: F401
from .manager import OracleManager  # noqa: F401
