"""Inclusive tiers on the GPU against the oracle, bit for bit: every decision,
every host slot (a clean copy where the block has one), the block and owner
tables, the clean-copy counters and the KV bytes of both tiers."""
import pytest

from workloads import make_workload, pool_spec

from ._lockstep import run_lockstep
from .test_parity_gpu import _sampled_full_size

pytestmark = pytest.mark.gpu


def _inclusive(name, seed, **over):
    return make_workload(name, seed, spec=pool_spec(name).with_(tiers=1), **over)


@pytest.mark.parametrize("seed,driver,mode", [(0, "device", 0), (1, "exchange", 0),
                                              (0, "sequential", 0), (1, "device", 2),
                                              (0, "exchange", 2), (1, "sequential", 2)])
def test_tiny_inclusive_full_images(seed, driver, mode):
    """1000 tiny events with clean copies kept: evictions that find one move no
    bytes, appends into a clean tail drop it; full byte images every 50 events."""
    om, gm = run_lockstep(_inclusive("tiny", seed), with_bytes=True, check_every=50,
                          driver=driver, mode=mode)
    assert om.counters == gm.counters
    assert om.pool.clean_out > 200 and om.pool.clean_dropped > 10
    page = om.pool.J * om.pool.P
    assert om.pool.bytes_out == (om.counters["pages_out"] - om.pool.clean_out) * page


def test_thinker_inclusive_full_size():
    """Thinker turns with clean copies: after a session has been reloaded once,
    evicting it again moves no bytes (turns never append)."""
    om, gm = _sampled_full_size(_inclusive("thinker", 0, n_turns=20), "device", 0)
    assert om.pool.clean_out > 0
    assert om.pool.clean_dropped == 0


def test_tiny_inclusive_lru_baseline():
    """Inclusive tiers under the LRU baseline policy (no preloads)."""
    wl = make_workload("tiny", 3, spec=pool_spec("tiny").with_(tiers=1, policy=1))
    om, gm = run_lockstep(wl, with_bytes=True, check_every=100, driver="device")
    assert om.counters == gm.counters and om.pool.clean_out > 0


def test_thinker_inclusive_async_copies():
    """Inclusive tiers with asynchronous turn copies and no host round trip."""
    om, gm = _sampled_full_size(_inclusive("thinker", 2, n_turns=30), "device", 0, record=False,
                                async_copy=True)
    assert om.pool.clean_out > 0
