"""KVPool: one liblv pool with its HBM KV arrays held as torch device memory.

PyTorch provides only the device memory (the 2L sub-page arrays and small
scratch buffers) and the stream; every operation is a liblv call.
"""
from __future__ import annotations

import ctypes

import numpy as np
import torch

from . import lv


class _CudaArray:
    """__cuda_array_interface__ of a raw device address (no ownership)."""

    def __init__(self, ptr, nbytes):
        self.__cuda_array_interface__ = {"shape": (nbytes,), "typestr": "|u1",
                                         "data": (int(ptr), False), "version": 3, "strides": None}


class KVPool:
    def __init__(self, *, layers, kv_heads, head_dim, max_sessions, max_blocks, hbm_pages,
                 hbm_budget_pages, host_pages, page_tokens=16, elem_bytes=2,
                 reply_prior_us=3_000_000, protect_us=2_000_000, unit_us=80_000,
                 within_order=lv.LV_SUFFIX_FIRST, t_play_mode=lv.LV_PLAY_PLAYBACK,
                 device=None, stream=None, kv=None, policy=lv.LV_POLICY_NEXT_USE,
                 tiers=lv.LV_TIERS_EXCLUSIVE):
        if not torch.cuda.is_available():
            raise RuntimeError("KVPool needs a CUDA device (liblv has no CPU path)")
        self.device = torch.device(device or "cuda", torch.cuda.current_device()) \
            if device is None else torch.device(device)
        self.stream = stream
        self.L, self.T = layers, page_tokens
        self.J = 2 * layers
        self.P = page_tokens * kv_heads * head_dim * elem_bytes
        self.S, self.max_blocks = max_sessions, max_blocks
        self.hbm_pages, self.budget, self.host_pages = hbm_pages, hbm_budget_pages, host_pages
        self.launches = 0      # liblv kernels launched through this object
        # a ranking is two kernels, three above 1024 sessions (liblv's k_rank_prefix)
        self.rank_extra = 1 if max_sessions > lv.EMIT_SCAN_MAX else 0
        self.policy = policy
        self.tiers = tiers
        with torch.cuda.device(self.device):
            if kv is None:
                # one allocation, viewed as 2L sub-page arrays [hbm_pages][P]
                kv = torch.zeros((self.J, hbm_pages, self.P), dtype=torch.uint8, device=self.device)
            self.kv = kv
            ptrs = (ctypes.c_void_p * self.J)(*[self.kv[j].data_ptr() for j in range(self.J)])
            self._ptrs = ptrs
            d = lv.lv_pool_desc()
            d.num_layers, d.num_kv_heads, d.head_dim = layers, kv_heads, head_dim
            d.page_tokens, d.elem_bytes = page_tokens, elem_bytes
            d.max_sessions, d.max_blocks, d.within_order = max_sessions, max_blocks, within_order
            d.hbm_pages, d.hbm_budget_pages, d.host_pages = hbm_pages, hbm_budget_pages, host_pages
            d.hbm_kv = ctypes.cast(ptrs, ctypes.POINTER(ctypes.c_void_p))
            d.host_kv = None
            d.reply_prior_us, d.protect_us, d.unit_us = reply_prior_us, protect_us, unit_us
            d.t_play_mode, d.policy, d.tiers = t_play_mode, policy, tiers
            self.handle = lv.lv_pool_create(d, stream)
            cap = max(hbm_budget_pages, max_blocks, 1)
            self.cap = cap
            dev = self.device
            self.victims = torch.empty((cap, 3), dtype=torch.int32, device=dev)
            self.commit = torch.empty((cap, 3), dtype=torch.int32, device=dev)
            self.slots = torch.empty(cap, dtype=torch.int32, device=dev)
            self.pages = torch.empty(cap, dtype=torch.int32, device=dev)
            self.blks = torch.empty(max_blocks, dtype=torch.int32, device=dev)
            self.app = torch.empty(max_blocks + 2, dtype=torch.int32, device=dev)
            self.count_h = torch.zeros(4, dtype=torch.int64).pin_memory()
        hp = lv.lv_pool_host_ptr(self.handle)
        self.host = None
        self.host_dev = None
        if host_pages:
            nbytes = host_pages * self.J * self.P
            buf = (ctypes.c_uint8 * nbytes).from_address(hp)
            self.host = np.frombuffer(buf, dtype=np.uint8).reshape(host_pages, self.J, self.P)
            # the same host pool as a CUDA tensor (device-side alias of the mapped memory)
            cai = _CudaArray(lv.lv_pool_host_device_ptr(self.handle), nbytes)
            with torch.cuda.device(self.device):
                self.host_dev = torch.as_tensor(cai, device=self.device).view(host_pages, self.J, self.P)

    # ------------------------------------------------------------------ life
    def attach(self, obj):
        """Objects holding native state over this pool (a preload controller); they are
        closed before the pool is destroyed."""
        if not hasattr(self, "_attached"):
            self._attached = []
        self._attached.append(obj)

    def close(self):
        if getattr(self, "handle", None):
            for obj in getattr(self, "_attached", []):
                obj.close()
            self._attached = []
            self.host_dev = None
            lv.lv_pool_destroy(self.handle, self.stream)
            self.handle = None
            self.host = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    # ----------------------------------------------------------------- calls
    def import_placement(self, placement: np.ndarray, ctx_tokens: np.ndarray):
        pl = np.ascontiguousarray(placement, dtype=np.int32)
        cx = np.ascontiguousarray(ctx_tokens, dtype=np.int32)
        lv.lv_pool_import(self.handle, pl, cx, self.stream)
        self.launches += 2

    def set_sessions(self, states: np.ndarray, first: int = 0):
        states = np.ascontiguousarray(states, dtype=lv.SESSION_DTYPE)
        lv.lv_session_set(self.handle, states, first, len(states), self.stream)
        self.launches += 1

    def get_sessions(self) -> np.ndarray:
        out = np.zeros(self.S, dtype=lv.SESSION_DTYPE)
        lv.lv_session_get(self.handle, out, 0, self.S, self.stream)
        self.sync()
        return out

    def events(self, ev: np.ndarray):
        ev = np.ascontiguousarray(ev, dtype=lv.EVENT_DTYPE)
        if len(ev):
            lv.lv_session_events(self.handle, ev, len(ev), self.stream)
            self.launches += 1

    def select(self, now_us: int, k: int, flags: int = 0, capacity=None):
        """Victims (device int32 [n, 3] view) and n; synchronises to read n."""
        cap = self.cap if capacity is None else capacity
        out = self.victims if cap <= self.cap else torch.empty((cap, 3), dtype=torch.int32,
                                                                device=self.device)
        lv.lv_select_victims(self.handle, now_us, min(k, lv.LV_ALL), flags, out, cap,
                             self.count_h[0:1], self.stream)
        self.launches += 2 + self.rank_extra
        self.sync()
        n = int(self.count_h[0])
        return out[:n], n

    def swap_out(self, victims, n: int, mode=lv.LV_MODE_AUTO):
        lv.lv_swap_out(self.handle, victims, n, self.slots, self.commit, mode, self.stream)
        self.launches += 2
        return self.slots[:n], self.commit[:n]

    def swap_in(self, sid: int, blks, n: int, mode=lv.LV_MODE_AUTO):
        lv.lv_swap_in(self.handle, sid, blks, n, self.pages, self.commit, mode, self.stream)
        self.launches += 2
        return self.pages[:n], self.commit[:n]

    def exchange(self, victims, n_out: int, sid: int, blks, n_in: int, mode=lv.LV_MODE_AUTO):
        """Evict n_out victims and load n_in host blocks of sid, committed, in one step."""
        lv.lv_swap_exchange(self.handle, victims, n_out, sid, blks, n_in, self.slots, self.pages,
                            mode, self.stream)
        self.launches += 2
        return self.slots[:n_out], self.pages[:n_in]

    def remap(self, entries, n: int):
        lv.lv_remap(self.handle, entries, n, self.stream)
        self.launches += 2 if n > 0 else 0

    def cancel(self, locs, n: int):
        lv.lv_cancel(self.handle, locs, n, self.stream)
        self.launches += 1

    def append(self, sid: int, n_tokens: int):
        cap = n_tokens // self.T + 2
        pages = torch.empty(cap, dtype=torch.int32, device=self.device)
        cnt = torch.zeros(1, dtype=torch.int32).pin_memory()
        lv.lv_session_append(self.handle, sid, n_tokens, pages, cnt, self.stream)
        self.launches += 1
        self.sync()
        return pages[:int(cnt[0])]

    def counts(self):
        a = np.zeros(self.S, dtype=np.int32)
        b = np.zeros(self.S, dtype=np.int32)
        lv.lv_session_counts(self.handle, a, b, self.stream)
        self.launches += 1
        self.sync()
        return a, b

    def blocks(self, sid: int, where: int):
        """Blocks of ``sid`` in HBM (0) or the host tier (1): device view and count."""
        lv.lv_session_blocks(self.handle, sid, where, self.blks, self.count_h[1:2], self.stream)
        self.launches += 1
        self.sync()
        n = int(self.count_h[1])
        return self.blks[:n], n

    def tables(self):
        t = np.zeros((self.S, self.max_blocks), dtype=np.int32)
        oh = np.zeros(self.hbm_pages, dtype=np.int32)
        oo = np.zeros(max(self.host_pages, 1), dtype=np.int32)
        lv.lv_read_tables(self.handle, t, oh, oo if self.host_pages else None, self.stream)
        self.sync()
        return t, oh, oo[:self.host_pages]

    def stats(self) -> dict:
        return lv.lv_get_stats(self.handle, self.stream)

    def sync(self, raise_on_error=True) -> int:
        return lv.lv_sync(self.handle, self.stream, raise_on_error)

    def clear_error(self):
        lv.lv_clear_error(self.handle, self.stream)
