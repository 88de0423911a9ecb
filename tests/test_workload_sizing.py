"""Sizing of the two workloads with the largest host tiers (mixed, frag): the stated
session counts, and the rule that scales them down where the host cannot page-lock
the tier, min(400 GB, 0.8 * MemAvailable)."""
from workloads import GB, STATED_SESSIONS, host_tier_limit, make_workload, mem_available_bytes


def test_limit_is_min_of_cap_and_four_fifths_of_available():
    assert host_tier_limit(100 * GB) == 80 * GB
    assert host_tier_limit(1000 * GB) == 400 * GB
    assert host_tier_limit(0) == 0


def test_meminfo_parse(tmp_path):
    f = tmp_path / "meminfo"
    f.write_text("MemTotal:       209230784 kB\nMemFree: 1 kB\nMemAvailable:   206747328 kB\n")
    assert mem_available_bytes(str(f)) == 206747328 * 1024
    assert mem_available_bytes(str(tmp_path / "absent")) is None


def test_stated_sizes_fit_a_grace_host():
    """With the GPU machine's MemAvailable (206.7 GB), both workloads run at their stated
    session counts."""
    lim = host_tier_limit(206747328 * 1024)
    for name in ("mixed", "frag"):
        wl = make_workload(name, 0, host_limit=lim)
        sz = wl.meta["sizing"]
        assert not sz["scaled"] and wl.spec.n_sessions == STATED_SESSIONS[name]
        assert sz["host_tier_bytes"] == wl.spec.host_pages * wl.spec.shape.page_bytes <= lim


def test_scaled_down_to_the_limit():
    for name in ("mixed", "frag"):
        full = make_workload(name, 0)
        need = full.spec.host_pages * full.spec.shape.page_bytes
        lim = need // 2
        wl = make_workload(name, 0, host_limit=lim)
        sz = wl.meta["sizing"]
        assert sz["scaled"] and sz["host_tier_bytes"] <= lim
        assert 1 <= wl.spec.n_sessions < STATED_SESSIONS[name]
        # the largest count that fits: one more session would not
        more = make_workload(name, 0, spec=full.spec.with_(n_sessions=wl.spec.n_sessions + 1,
                                                              host_pages=0))
        assert more.spec.host_pages * more.spec.shape.page_bytes > lim or \
            wl.spec.n_sessions + 1 == STATED_SESSIONS[name]
