"""The five synthetic workloads against the sizes and distributions they are stated with:
shapes, session counts, context ranges, HBM budgets (decimal GB floored to whole pages),
event counts and kinds, the long workload's frame-token share and the frag workload's
scattered initial placement.  CPU only: the generators hold no arithmetic of the method."""
import numpy as np
import pytest

from workloads import make_workload
from workloads.configs import GB, THINKER_SHAPE, TINY_SHAPE

EV_TURN_SCATTER, EV_EVICT = 7, 8


def _ctx(wl):
    return np.asarray(wl.init.ctx_tokens, dtype=np.int64)


def _hbm_pages_used(wl):
    pl = np.asarray(wl.init.placement)
    return pl[pl >= 0]


def test_tiny():
    wl = make_workload("tiny", 0)
    sp = wl.spec
    assert sp.shape == TINY_SHAPE and sp.shape.subpage_bytes == 4096 and sp.shape.page_bytes == 16384
    assert (sp.n_sessions, sp.hbm_pages, sp.host_pages) == (8, 256, 1024)
    ctx = _ctx(wl)
    assert ctx.min() >= 64 and ctx.max() <= 512
    assert wl.n_events == 1000


def test_thinker_every_turn_must_evict():
    wl = make_workload("thinker", 0)
    sp = wl.spec
    assert sp.shape == THINKER_SHAPE and sp.shape.page_bytes == 1572864
    assert sp.n_sessions == 64
    assert sp.hbm_budget_pages == 40 * GB // 1572864 == 25431
    ctx = _ctx(wl)
    assert ctx.min() >= 2048 and ctx.max() <= 16384
    # log-uniform: about as many contexts below the geometric middle (~5.8k) as above
    mid = np.sqrt(2048 * 16384)
    assert 0.25 < float(np.mean(ctx < mid)) < 0.75
    pages = -(-ctx // 16)
    # the KV exceeds the budget by at least one largest possible session, so every turn
    # (which reloads a whole session) must evict
    assert pages.sum() >= sp.hbm_budget_pages + sp.max_blocks


def test_mixed_at_its_stated_size():
    wl = make_workload("mixed", 0)
    sp = wl.spec
    assert sp.shape == THINKER_SHAPE and sp.n_sessions == 256
    assert sp.hbm_budget_pages == 60 * GB // 1572864 == 38146
    ctx = _ctx(wl)
    assert ctx.min() >= 2048 and ctx.max() <= 16384
    assert wl.n_events == 3000


def test_long_contexts_and_frame_share():
    wl = make_workload("long", 0)
    sp = wl.spec
    assert sp.shape == THINKER_SHAPE and sp.n_sessions == 16
    assert sp.hbm_budget_pages == 25431
    ctx = _ctx(wl)
    assert ctx.min() >= 32768 and ctx.max() <= 65536
    spans = wl.meta["frame_spans"]
    frame_tokens = sum(n for sess in spans for _, n in sess)
    assert frame_tokens / ctx.sum() == pytest.approx(0.30, abs=0.02)
    for s, sess in enumerate(spans):                       # frames lie inside their context
        assert all(0 <= a and a + n <= ctx[s] for a, n in sess)


def test_frag_scattered_and_alternating():
    wl = make_workload("frag", 0)
    sp = wl.spec
    assert sp.shape == THINKER_SHAPE and sp.n_sessions == 1024
    assert sp.hbm_budget_pages == 100 * GB // 1572864 == 63578
    ctx = _ctx(wl)
    assert ctx.min() >= 256 and ctx.max() <= 4096
    assert wl.n_events == 10000
    kinds = np.asarray(wl.kind)
    assert int((kinds == EV_EVICT).sum()) == 5000 and int((kinds == EV_TURN_SCATTER).sum()) == 5000
    k = np.asarray(wl.a)[kinds == EV_EVICT]
    assert k.min() >= 8 and k.max() <= 128
    pages = _hbm_pages_used(wl)
    assert len(np.unique(pages)) == len(pages)           # no page twice
    # a random permutation of the pool, not the blocks' order: consecutive blocks of a
    # session rarely sit on consecutive pages
    pl = np.asarray(wl.init.placement)
    row = pl[0][pl[0] >= 0]
    assert len(row) > 8 and float(np.mean(np.diff(row) == 1)) < 0.1
