"""ctypes binding of liblv.so (include/lv.h), with the same function names.

This module only marshals arguments: every step of the KV swap path runs in the
library's CUDA kernels.  Array arguments may be torch tensors, numpy arrays or
raw integer addresses (device or host memory, as the C ABI allows).  A
non-``LV_OK`` status raises :class:`LvError`.  If liblv.so is missing the import
fails loudly; there is no fallback.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "liblv.so")

LV_OK = 0
STATUS_NAMES = {0: "LV_OK", 1: "LV_ERR_INVALID", 2: "LV_ERR_OOM", 3: "LV_ERR_CUDA",
                4: "LV_ERR_NO_HBM", 5: "LV_ERR_NO_HOST", 6: "LV_ERR_BOUNDS",
                7: "LV_ERR_DOUBLE_MAP", 8: "LV_ERR_BUDGET", 9: "LV_ERR_TIMEOUT",
                10: "LV_ERR_STATE"}
LV_ERR_INVALID, LV_ERR_OOM, LV_ERR_CUDA, LV_ERR_NO_HBM, LV_ERR_NO_HOST = 1, 2, 3, 4, 5
LV_ERR_BOUNDS, LV_ERR_DOUBLE_MAP, LV_ERR_BUDGET, LV_ERR_TIMEOUT, LV_ERR_STATE = 6, 7, 8, 9, 10
LV_ALL = 2**63 - 1
LV_SUFFIX_FIRST, LV_ASCENDING = 0, 1
LV_PLAY_PLAYBACK, LV_PLAY_COUNTERS = 0, 1
LV_MODE_AUTO, LV_MODE_ZERO_COPY, LV_MODE_STAGED = 0, 1, 2
LV_SELECT_FALLBACK = 1
LV_POLICY_NEXT_USE, LV_POLICY_LRU = 0, 1
LV_TIERS_EXCLUSIVE, LV_TIERS_INCLUSIVE = 0, 1
LV_RESIDENT_ASYNC_COPY = 2
LV_VERSION = 3                     # include/lv.h
EMIT_SCAN_MAX = 1024               # above this many sessions a ranking runs one more kernel
LV_MODE_ASYNC = 16
LV_RUNNING, LV_IMMEDIATE, LV_RESP_OPEN, LV_DONE_VALID = 1, 2, 4, 8
(LV_EV_TURN_BEGIN, LV_EV_TURN_END, LV_EV_PLAYBACK, LV_EV_SPEECH_START, LV_EV_BARGE_IN,
 LV_EV_SPEECH_STOP, LV_EV_PRELOADED, LV_EV_UNPROTECT) = 1, 2, 3, 4, 5, 6, 7, 8


class LvError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = int(status)
        super().__init__(f"{where}: {STATUS_NAMES.get(self.status, self.status)}")


class lv_pool_desc(ctypes.Structure):
    _fields_ = [("num_layers", ctypes.c_int32), ("num_kv_heads", ctypes.c_int32),
                ("head_dim", ctypes.c_int32), ("page_tokens", ctypes.c_int32),
                ("elem_bytes", ctypes.c_int32), ("max_sessions", ctypes.c_int32),
                ("max_blocks", ctypes.c_int32), ("within_order", ctypes.c_int32),
                ("hbm_pages", ctypes.c_int64), ("hbm_budget_pages", ctypes.c_int64),
                ("host_pages", ctypes.c_int64), ("hbm_kv", ctypes.POINTER(ctypes.c_void_p)),
                ("host_kv", ctypes.c_void_p), ("reply_prior_us", ctypes.c_int64),
                ("protect_us", ctypes.c_int64), ("unit_us", ctypes.c_int64),
                ("t_play_mode", ctypes.c_int32), ("policy", ctypes.c_int32),
                ("tiers", ctypes.c_int32), ("reserved", ctypes.c_int32)]


class lv_turn_desc(ctypes.Structure):
    _fields_ = [("sid", ctypes.c_int32), ("num_candidates", ctypes.c_int32),
                ("candidates", ctypes.c_void_p), ("now_us", ctypes.c_int64),
                ("reply_audio_us", ctypes.c_int64), ("reply_units", ctypes.c_int64),
                ("append_tokens", ctypes.c_int32), ("flags", ctypes.c_uint32),
                ("load_keys", ctypes.c_void_p)]


class lv_controller_desc(ctypes.Structure):
    _fields_ = [("link_bytes_per_us", ctypes.c_int64), ("lead_prior_us", ctypes.c_int64),
                ("cap_pages", ctypes.c_int64), ("mode", ctypes.c_int32), ("reserved", ctypes.c_int32)]


class lv_controller_counters(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int64) for n in ("admitted", "completed", "waited", "given_up",
                                               "cancelled", "hits", "victims", "pages_in")]

    def as_dict(self):
        return {n: int(getattr(self, n)) for n, _ in self._fields_}


class lv_stats(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int64) for n in (
        "hbm_allocated", "host_allocated", "hbm_budget_pages", "host_pages", "error",
        "error_detail", "last_select_count", "last_select_total", "selects", "victims",
        "shortfalls", "pages_out", "pages_in", "bytes_out", "bytes_in", "remap_entries",
        "appended_pages", "cancels", "events", "fallback_selects", "preloads",
        "preloads_skipped", "clean_copies", "clean_out", "clean_dropped")]

    def as_dict(self):
        return {n: int(getattr(self, n)) for n, _ in self._fields_}


class lv_kernel_timing(ctypes.Structure):
    _fields_ = [("launches", ctypes.c_int64), ("total_ms", ctypes.c_double),
                ("min_ms", ctypes.c_double), ("max_ms", ctypes.c_double)]


LV_TIMING_SWAP_OUT, LV_TIMING_SWAP_IN, LV_TIMING_EXCHANGE, LV_TIMING_PACK, LV_TIMING_UNPACK = 0, 1, 2, 3, 4
LV_TIMING_KINDS = 5
TIMING_NAMES = ("swap_out", "swap_in", "exchange", "pack", "unpack")


class lv_rank_params(ctypes.Structure):
    _fields_ = [("num_sessions", ctypes.c_int32), ("max_blocks", ctypes.c_int32),
                ("page_tokens", ctypes.c_int32), ("within_order", ctypes.c_int32),
                ("t_play_mode", ctypes.c_int32), ("flags", ctypes.c_uint32),
                ("reply_prior_us", ctypes.c_int64), ("unit_us", ctypes.c_int64),
                ("policy", ctypes.c_int32), ("reserved", ctypes.c_int32)]


class lv_sched_params(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int64) for n in ("p_safe_us", "alpha", "beta", "occupied",
                                               "allocatable", "token_budget", "kv_budget")]


REQUEST_DTYPE = np.dtype([("id", "<i4"), ("started", "<i4"), ("play_buffer_us", "<i8"),
                          ("ready_age_us", "<i8"), ("kv_pages", "<i8"), ("tokens", "<i8"),
                          ("kv_needed", "<i8")])
LV_SCHED_MAX_REQUESTS = 4096
LV_NOALLOC_MAX_SESSIONS = 4096
LV_RESIDENT_PRELOAD = 1
LV_RESIDENT_DONE, LV_RESIDENT_SKIPPED, LV_RESIDENT_NOTHING, LV_RESIDENT_FAILED = 0, 1, 2, 3

# numpy views of the ABI's array element types
SESSION_DTYPE = np.dtype([("ctx_tokens", "<i4"), ("flags", "<i4"), ("gen_us", "<i8"),
                          ("play_us", "<i8"), ("t_done_us", "<i8"), ("reply_ema_us", "<i8"),
                          ("reply_n", "<i4"), ("pad", "<i4"), ("reply_tokens", "<i8"),
                          ("protect_until_us", "<i8"), ("last_use_us", "<i8")])
EVENT_DTYPE = np.dtype([("kind", "<i4"), ("sid", "<i4"), ("t_us", "<i8"), ("a", "<i8"), ("b", "<i8")])
VICTIM_DTYPE = np.dtype([("sid", "<i4"), ("blk", "<i4"), ("page", "<i4")])
RESIDENT_DTYPE = np.dtype([("k", "<i8"), ("n_found", "<i8"), ("n_victims", "<i8"), ("n_loaded", "<i8"),
                           ("n_appended", "<i8"), ("status", "<i4"), ("sid", "<i4")])
REMAP_DTYPE = np.dtype([("sid", "<i4"), ("blk", "<i4"), ("loc", "<i4")])
CTL_RECORD_DTYPE = np.dtype([("kind", "<i4"), ("sid", "<i4"), ("start_us", "<i8"), ("finish_us", "<i8"),
                             ("deadline_us", "<i8"), ("n", "<i8"), ("data_offset", "<i8")])
LV_CTL_ADMITTED, LV_CTL_COMPLETED, LV_CTL_CANCELLED, LV_CTL_GIVEN_UP, LV_CTL_UNPROTECTED, \
    LV_CTL_EVICTED = 1, 2, 3, 4, 5, 6
assert SESSION_DTYPE.itemsize == 72 and EVENT_DTYPE.itemsize == 32
assert VICTIM_DTYPE.itemsize == 12 and REMAP_DTYPE.itemsize == 12


def _load():
    if not os.path.exists(LIB_PATH):
        raise ImportError(f"{LIB_PATH} is missing: build it with "
                          "paper_2606_22983_gb300._build.build() (nvcc, sm_103a)")
    lib = ctypes.CDLL(LIB_PATH)
    vp, i32, i64, u32 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_uint32
    sigs = {
        "lv_pool_create": [ctypes.POINTER(lv_pool_desc), vp, ctypes.POINTER(vp)],
        "lv_pool_destroy": [vp, vp],
        "lv_pool_import": [vp, vp, vp, vp],
        "lv_session_set": [vp, vp, i32, i32, vp],
        "lv_session_get": [vp, vp, i32, i32, vp],
        "lv_session_events": [vp, vp, i64, vp],
        "lv_select_victims": [vp, i64, i64, u32, vp, i64, vp, vp],
        "lv_swap_out": [vp, vp, i64, vp, vp, i32, vp],
        "lv_swap_in": [vp, i32, vp, i64, vp, vp, i32, vp],
        "lv_swap_exchange": [vp, vp, i64, i32, vp, i64, vp, vp, i32, vp],
        "lv_make_resident": [vp, i32, i64, i32, u32, i64, vp, vp, vp, vp, vp, vp, vp],
        "lv_turn": [vp, ctypes.POINTER(lv_turn_desc), vp, vp, vp, vp, vp, vp, vp],
        "lv_join": [vp, vp],
        "lv_evict": [vp, i64, i64, u32, vp, vp, vp, vp],
        "lv_page_checksums": [vp, vp, i64, vp, vp],
        "lv_controller_create": [vp, ctypes.POINTER(lv_controller_desc), ctypes.POINTER(vp)],
        "lv_controller_destroy": [vp, vp],
        "lv_controller_tick": [vp, i64, vp],
        "lv_controller_speech": [vp, i32, i64, vp],
        "lv_controller_turn_begin": [vp, i32, i64, vp],
        "lv_controller_turn_loaded": [vp, i64, i64],
        "lv_controller_records": [vp, vp, i64, vp, vp, i64, vp],
        "lv_controller_counters_get": [vp, ctypes.POINTER(lv_controller_counters)],
        "lv_timing_enable": [vp, i32],
        "lv_pack_pages": [vp, vp, i64, vp, vp],
        "lv_schedule": [vp, ctypes.POINTER(lv_sched_params), vp, i32, vp, vp, vp],
        "lv_inject_fault": [vp, i32, i32],
        "lv_selftest_wait": [vp, i64, vp],
        "lv_unpack_pages": [vp, vp, vp, i64, vp],
        "lv_timing_read": [vp, ctypes.POINTER(lv_kernel_timing), i32],
        "lv_remap": [vp, vp, i64, vp],
        "lv_cancel": [vp, vp, i64, vp],
        "lv_session_append": [vp, i32, i32, vp, vp, vp],
        "lv_session_counts": [vp, vp, vp, vp],
        "lv_session_blocks": [vp, i32, i32, vp, vp, vp],
        "lv_read_tables": [vp, vp, vp, vp, vp],
        "lv_sync": [vp, vp],
        "lv_get_stats": [vp, ctypes.POINTER(lv_stats), vp],
        "lv_clear_error": [vp, vp],
        "lv_select_victims_noalloc": [ctypes.POINTER(lv_rank_params), vp, vp, i64, i64, vp, i64,
                                      vp, vp],
    }
    for name, args in sigs.items():
        f = getattr(lib, name)
        f.argtypes = args
        f.restype = ctypes.c_int
    lib.lv_pool_host_ptr.argtypes = [vp]
    lib.lv_pool_host_ptr.restype = vp
    lib.lv_pool_host_device_ptr.argtypes = [vp]
    lib.lv_pool_host_device_ptr.restype = vp
    lib.lv_status_str.argtypes = [ctypes.c_int]
    lib.lv_status_str.restype = ctypes.c_char_p
    lib.lv_version.argtypes = []
    lib.lv_version.restype = i32
    if lib.lv_version() != LV_VERSION:
        raise ImportError(f"{LIB_PATH} implements interface version {lib.lv_version()}, this "
                          f"binding version {LV_VERSION}: rebuild it")
    return lib


_lib = _load()

EXPORTED = ("lv_pool_create", "lv_pool_destroy", "lv_pool_host_ptr", "lv_pool_import",
            "lv_session_set", "lv_session_get", "lv_session_events", "lv_select_victims",
            "lv_swap_out", "lv_swap_in", "lv_swap_exchange", "lv_make_resident", "lv_remap", "lv_cancel", "lv_session_append",
            "lv_session_counts", "lv_session_blocks", "lv_read_tables", "lv_sync",
            "lv_get_stats", "lv_clear_error", "lv_status_str", "lv_version",
            "lv_select_victims_noalloc", "lv_timing_enable", "lv_timing_read", "lv_pack_pages",
            "lv_unpack_pages", "lv_pool_host_device_ptr", "lv_schedule", "lv_inject_fault",
            "lv_selftest_wait", "lv_turn", "lv_evict", "lv_join", "lv_page_checksums",
            "lv_controller_create", "lv_controller_destroy", "lv_controller_tick",
            "lv_controller_speech", "lv_controller_turn_begin", "lv_controller_turn_loaded",
            "lv_controller_records", "lv_controller_counters_get")


def lib():
    return _lib


def ptr(x):
    """Address of a tensor / array / integer, or None."""
    if x is None:
        return None
    if isinstance(x, int):
        return x
    if hasattr(x, "data_ptr"):
        return x.data_ptr()
    if isinstance(x, np.ndarray):
        if not x.flags["C_CONTIGUOUS"]:
            raise ValueError("array arguments must be C-contiguous")
        return x.ctypes.data
    if isinstance(x, ctypes.Array):
        return ctypes.addressof(x)
    raise TypeError(f"cannot pass {type(x).__name__} as an array argument")


def stream_handle(stream):
    """cudaStream_t of a torch stream (None: the current stream of the current device)."""
    if stream is None:
        import torch
        stream = torch.cuda.current_stream()
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def _check(status, where):
    if status != LV_OK:
        raise LvError(status, where)


# ----------------------------------------------------------------- entry points
def lv_pool_create(desc: lv_pool_desc, stream=None):
    h = ctypes.c_void_p()
    _check(_lib.lv_pool_create(ctypes.byref(desc), stream_handle(stream), ctypes.byref(h)),
           "lv_pool_create")
    return h.value


def lv_pool_destroy(pool, stream=None):
    _check(_lib.lv_pool_destroy(pool, stream_handle(stream)), "lv_pool_destroy")


def lv_pool_host_ptr(pool) -> int:
    return _lib.lv_pool_host_ptr(pool)


def lv_pool_host_device_ptr(pool) -> int:
    return _lib.lv_pool_host_device_ptr(pool)


def lv_pack_pages(pool, pages, n, dst, stream=None):
    _check(_lib.lv_pack_pages(pool, ptr(pages), n, ptr(dst), stream_handle(stream)), "lv_pack_pages")


def lv_unpack_pages(pool, src, pages, n, stream=None):
    _check(_lib.lv_unpack_pages(pool, ptr(src), ptr(pages), n, stream_handle(stream)), "lv_unpack_pages")


def lv_pool_import(pool, placement, ctx_tokens, stream=None):
    _check(_lib.lv_pool_import(pool, ptr(placement), ptr(ctx_tokens), stream_handle(stream)),
           "lv_pool_import")


def lv_session_set(pool, states, first, n, stream=None):
    _check(_lib.lv_session_set(pool, ptr(states), first, n, stream_handle(stream)), "lv_session_set")


def lv_session_get(pool, out, first, n, stream=None):
    _check(_lib.lv_session_get(pool, ptr(out), first, n, stream_handle(stream)), "lv_session_get")


def lv_session_events(pool, events, n, stream=None):
    _check(_lib.lv_session_events(pool, ptr(events), n, stream_handle(stream)), "lv_session_events")


def lv_select_victims(pool, now_us, k, flags, out, capacity, count_out, stream=None):
    _check(_lib.lv_select_victims(pool, now_us, k, flags, ptr(out), capacity, ptr(count_out),
                                  stream_handle(stream)), "lv_select_victims")


def lv_swap_out(pool, victims, n, slots_out, commit_out, mode=LV_MODE_AUTO, stream=None):
    _check(_lib.lv_swap_out(pool, ptr(victims), n, ptr(slots_out), ptr(commit_out), mode,
                            stream_handle(stream)), "lv_swap_out")


def lv_swap_in(pool, sid, blks, n, pages_out, commit_out, mode=LV_MODE_AUTO, stream=None):
    _check(_lib.lv_swap_in(pool, sid, ptr(blks), n, ptr(pages_out), ptr(commit_out), mode,
                           stream_handle(stream)), "lv_swap_in")


def lv_swap_exchange(pool, victims, n_out, sid, blks, n_in, slots_out, pages_out,
                     mode=LV_MODE_AUTO, stream=None):
    _check(_lib.lv_swap_exchange(pool, ptr(victims), n_out, sid, ptr(blks), n_in, ptr(slots_out),
                                 ptr(pages_out), mode, stream_handle(stream)), "lv_swap_exchange")


def lv_make_resident(pool, sid, now_us, append_tokens, flags, max_load_pages, victims_out,
                     slots_out, blocks_out, pages_out, append_out, result_out, stream=None):
    _check(_lib.lv_make_resident(pool, sid, now_us, append_tokens, flags, max_load_pages,
                                 ptr(victims_out), ptr(slots_out), ptr(blocks_out), ptr(pages_out),
                                 ptr(append_out), ptr(result_out), stream_handle(stream)),
           "lv_make_resident")


def lv_turn(pool, sid, now_us, append_tokens, reply_audio_us, reply_units, outs=(None,) * 5,
            result_out=None, candidates=None, num_candidates=0, stream=None, flags=0,
            load_keys=None):
    """One turn (pick when sid == -1, turn begin, make resident, turn end); outs =
    (victims, slots, blocks, pages, append) as for lv_make_resident; load_keys (uint64
    [max_blocks]) orders the loads."""
    d = lv_turn_desc(sid=sid, num_candidates=num_candidates, candidates=ptr(candidates),
                     now_us=now_us, reply_audio_us=reply_audio_us, reply_units=reply_units,
                     append_tokens=append_tokens, flags=flags, load_keys=ptr(load_keys))
    _check(_lib.lv_turn(pool, ctypes.byref(d), *(ptr(o) for o in outs), ptr(result_out),
                        stream_handle(stream)), "lv_turn")


def lv_evict(pool, now_us, k, flags=0, victims_out=None, slots_out=None, result_out=None,
             stream=None):
    _check(_lib.lv_evict(pool, now_us, k, flags, ptr(victims_out), ptr(slots_out), ptr(result_out),
                         stream_handle(stream)), "lv_evict")


def lv_page_checksums(pool, pages, n, sums_out, stream=None):
    _check(_lib.lv_page_checksums(pool, ptr(pages), n, ptr(sums_out), stream_handle(stream)),
           "lv_page_checksums")


def lv_controller_create(pool, link_bytes_per_us, lead_prior_us, cap_pages=None, mode=LV_MODE_AUTO):
    d = lv_controller_desc(link_bytes_per_us=link_bytes_per_us, lead_prior_us=lead_prior_us,
                           cap_pages=-1 if cap_pages is None else cap_pages, mode=mode, reserved=0)
    out = ctypes.c_void_p()
    _check(_lib.lv_controller_create(pool, ctypes.byref(d), ctypes.byref(out)), "lv_controller_create")
    return out.value


def lv_controller_destroy(ctl, stream=None):
    _check(_lib.lv_controller_destroy(ctl, stream_handle(stream)), "lv_controller_destroy")


def lv_controller_tick(ctl, now_us, stream=None):
    _check(_lib.lv_controller_tick(ctl, now_us, stream_handle(stream)), "lv_controller_tick")


def lv_controller_speech(ctl, sid, now_us, stream=None):
    _check(_lib.lv_controller_speech(ctl, sid, now_us, stream_handle(stream)), "lv_controller_speech")


def lv_controller_turn_begin(ctl, sid, now_us, stream=None):
    _check(_lib.lv_controller_turn_begin(ctl, sid, now_us, stream_handle(stream)),
           "lv_controller_turn_begin")


def lv_controller_turn_loaded(ctl, now_us, pages):
    _check(_lib.lv_controller_turn_loaded(ctl, now_us, pages), "lv_controller_turn_loaded")


def lv_controller_records(ctl):
    """The decision records since the last call and their int32 data."""
    n, nd = ctypes.c_int64(), ctypes.c_int64()
    st = _lib.lv_controller_records(ctl, None, 0, ctypes.byref(n), None, 0, ctypes.byref(nd))
    if st == LV_OK:
        return np.zeros(0, CTL_RECORD_DTYPE), np.zeros(0, np.int32)
    recs = np.zeros(n.value, CTL_RECORD_DTYPE)
    data = np.zeros(max(nd.value, 1), np.int32)
    _check(_lib.lv_controller_records(ctl, recs.ctypes.data, n.value, ctypes.byref(n), data.ctypes.data,
                                      data.size, ctypes.byref(nd)), "lv_controller_records")
    return recs, data[:nd.value]


def lv_controller_counters_get(ctl) -> dict:
    c = lv_controller_counters()
    _check(_lib.lv_controller_counters_get(ctl, ctypes.byref(c)), "lv_controller_counters_get")
    return c.as_dict()


def lv_join(pool, stream=None):
    _check(_lib.lv_join(pool, stream_handle(stream)), "lv_join")


def lv_remap(pool, entries, n, stream=None):
    _check(_lib.lv_remap(pool, ptr(entries), n, stream_handle(stream)), "lv_remap")


def lv_cancel(pool, locs, n, stream=None):
    _check(_lib.lv_cancel(pool, ptr(locs), n, stream_handle(stream)), "lv_cancel")


def lv_session_append(pool, sid, n_tokens, pages_out, count_out, stream=None):
    _check(_lib.lv_session_append(pool, sid, n_tokens, ptr(pages_out), ptr(count_out),
                                  stream_handle(stream)), "lv_session_append")


def lv_session_counts(pool, hbm_blocks, host_blocks, stream=None):
    _check(_lib.lv_session_counts(pool, ptr(hbm_blocks), ptr(host_blocks), stream_handle(stream)),
           "lv_session_counts")


def lv_session_blocks(pool, sid, where, blks_out, count_out, stream=None):
    _check(_lib.lv_session_blocks(pool, sid, where, ptr(blks_out), ptr(count_out),
                                  stream_handle(stream)), "lv_session_blocks")


def lv_read_tables(pool, tables, hbm_owner, host_owner, stream=None):
    _check(_lib.lv_read_tables(pool, ptr(tables), ptr(hbm_owner), ptr(host_owner),
                               stream_handle(stream)), "lv_read_tables")


def lv_sync(pool, stream=None, raise_on_error=True) -> int:
    st = _lib.lv_sync(pool, stream_handle(stream))
    if raise_on_error:
        _check(st, "lv_sync")
    return st


def lv_get_stats(pool, stream=None) -> dict:
    s = lv_stats()
    _check(_lib.lv_get_stats(pool, ctypes.byref(s), stream_handle(stream)), "lv_get_stats")
    return s.as_dict()


def lv_clear_error(pool, stream=None):
    _check(_lib.lv_clear_error(pool, stream_handle(stream)), "lv_clear_error")


def lv_select_victims_noalloc(params: lv_rank_params, sessions, tables, now_us, k, out, capacity,
                              count_out, stream=None):
    _check(_lib.lv_select_victims_noalloc(ctypes.byref(params), ptr(sessions), ptr(tables), now_us,
                                          k, ptr(out), capacity, ptr(count_out),
                                          stream_handle(stream)), "lv_select_victims_noalloc")


def lv_timing_enable(pool, enable=True):
    _check(_lib.lv_timing_enable(pool, 1 if enable else 0), "lv_timing_enable")


def lv_timing_read(pool, reset=False) -> dict:
    arr = (lv_kernel_timing * LV_TIMING_KINDS)()
    _check(_lib.lv_timing_read(pool, arr, 1 if reset else 0), "lv_timing_read")
    return {TIMING_NAMES[i]: {"launches": int(arr[i].launches), "total_ms": arr[i].total_ms,
                              "min_ms": arr[i].min_ms, "max_ms": arr[i].max_ms}
            for i in range(LV_TIMING_KINDS)}


def lv_schedule(pool, params: lv_sched_params, reqs, n, order_out, batch_out, stream=None):
    _check(_lib.lv_schedule(pool, ctypes.byref(params), ptr(reqs), n, ptr(order_out), ptr(batch_out),
                            stream_handle(stream)), "lv_schedule")


LV_FAULT_NONE, LV_FAULT_HOST_ALLOC, LV_FAULT_HBM_ALLOC, LV_FAULT_COPY = 0, 1, 2, 3


def lv_inject_fault(pool, kind, after=0):
    _check(_lib.lv_inject_fault(pool, kind, after), "lv_inject_fault")


def lv_selftest_wait(pool, limit_us, stream=None):
    _check(_lib.lv_selftest_wait(pool, limit_us, stream_handle(stream)), "lv_selftest_wait")


def lv_status_str(status: int) -> str:
    return _lib.lv_status_str(status).decode()


def lv_version() -> int:
    return _lib.lv_version()
