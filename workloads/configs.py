"""Pool shapes and sizes of the five synthetic workloads.

Notation: L layers, H KV heads, D head dim, T tokens per page.  A *sub-page*
is one layer's K (or V) for one page: T*H*D*elem bytes, laid out [T][H][D].
A *page* (the paper's KV "block", Section 5.1) is the allocation and eviction
unit: T tokens across all L layers and both K and V, i.e. 2L sub-pages.

Budgets quoted in GB are decimal (1e9 bytes), floored to whole pages.
"""
from __future__ import annotations

from dataclasses import dataclass, replace

GB = 1_000_000_000


@dataclass(frozen=True)
class KVShape:
    layers: int
    kv_heads: int
    head_dim: int
    page_tokens: int = 16
    elem_bytes: int = 2

    @property
    def row_elems(self) -> int:          # one token row of one sub-page
        return self.kv_heads * self.head_dim

    @property
    def subpage_elems(self) -> int:
        return self.page_tokens * self.row_elems

    @property
    def subpage_bytes(self) -> int:      # P
        return self.subpage_elems * self.elem_bytes

    @property
    def subpages(self) -> int:           # 2L sub-pages per page
        return 2 * self.layers

    @property
    def page_bytes(self) -> int:
        return self.subpages * self.subpage_bytes


# 2-layer GQA, 2 KV heads x 64: P = 4 KiB, page = 16 KiB.
TINY_SHAPE = KVShape(layers=2, kv_heads=2, head_dim=64)
# Thinker-shaped KV: 48 layers, 4 KV heads x 128: P = 16 KiB, page = 1.5 MiB.
THINKER_SHAPE = KVShape(layers=48, kv_heads=4, head_dim=128)


@dataclass(frozen=True)
class PoolSpec:
    """Static parameters of one pool (shared by every workload of a config)."""
    name: str
    shape: KVShape
    n_sessions: int
    max_blocks: int              # block-table capacity per session
    hbm_pages: int               # pages in each of the 2L device arrays
    hbm_budget_pages: int        # pages that may be allocated at once
    host_pages: int              # host pool slots (filled in by the generator when 0)
    reply_prior_us: int = 3_000_000
    protect_us: int = 2_000_000
    within_order: int = 0        # 0: suffix blocks first, 1: ascending block id
    t_play_mode: int = 0         # 0: playback accounting, 1: progress counters
    unit_us: int = 80_000        # progress-counter unit (one audio token)
    policy: int = 0              # 0: next-use order, 1: LRU baseline
    tiers: int = 0               # 0: exclusive, 1: inclusive (clean host copies kept)

    def with_(self, **kw) -> "PoolSpec":
        return replace(self, **kw)


CONFIG_NAMES = ("tiny", "thinker", "mixed", "long", "frag")

# Session counts of the two workloads whose host tier is the largest.  Where the host
# cannot page-lock that much, the count is scaled down (``host_tier_limit``).
STATED_SESSIONS = {"mixed": 256, "frag": 1024}
HOST_TIER_CAP = 400 * GB       # the mixed workload's stated host tier


def mem_available_bytes(path: str = "/proc/meminfo"):
    """MemAvailable of this host in bytes, or None where /proc/meminfo has none."""
    try:
        with open(path) as f:
            for line in f:
                if line.startswith("MemAvailable:"):
                    return int(line.split()[1]) * 1024
    except OSError:
        pass
    return None


def host_tier_limit(mem_available=None) -> int:
    """Page-locked host tier a workload may take: min(400 GB, 0.8 * MemAvailable)."""
    m = mem_available_bytes() if mem_available is None else int(mem_available)
    if m is None:
        return HOST_TIER_CAP
    return min(HOST_TIER_CAP, int(0.8 * m))


def pages_for_bytes(nbytes: int, shape: KVShape) -> int:
    return nbytes // shape.page_bytes


def pool_spec(name: str) -> PoolSpec:
    """Base pool parameters of a named workload (host_pages may be 0 = sized later)."""
    if name == "tiny":
        # 8 sessions, contexts grow by turns up to 2048 tokens (128 pages).
        return PoolSpec("tiny", TINY_SHAPE, n_sessions=8, max_blocks=128,
                        hbm_pages=256, hbm_budget_pages=256, host_pages=1024)
    if name == "thinker":
        b = pages_for_bytes(40 * GB, THINKER_SHAPE)          # 25 431 pages
        return PoolSpec("thinker", THINKER_SHAPE, n_sessions=64, max_blocks=1024,
                        hbm_pages=b, hbm_budget_pages=b, host_pages=0)
    if name == "mixed":
        # 256 sessions: the host tier comes to ~115-135 GB of page-locked memory
        b = pages_for_bytes(60 * GB, THINKER_SHAPE)          # 38 146 pages
        return PoolSpec("mixed", THINKER_SHAPE, n_sessions=STATED_SESSIONS["mixed"],
                        max_blocks=1024, hbm_pages=b, hbm_budget_pages=b, host_pages=0)
    if name == "long":
        b = pages_for_bytes(40 * GB, THINKER_SHAPE)
        return PoolSpec("long", THINKER_SHAPE, n_sessions=16, max_blocks=4096,
                        hbm_pages=b, hbm_budget_pages=b, host_pages=0)
    if name == "frag":
        # 1024 sessions of 256-4096 tokens hold ~219 GB: a host tier of ~140-150 GB
        b = pages_for_bytes(100 * GB, THINKER_SHAPE)         # 63 578 pages
        return PoolSpec("frag", THINKER_SHAPE, n_sessions=STATED_SESSIONS["frag"],
                        max_blocks=256, hbm_pages=b, hbm_budget_pages=b, host_pages=0)
    raise ValueError(f"unknown workload {name!r}; expected one of {CONFIG_NAMES}")
