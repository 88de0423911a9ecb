"""Seeded KV page contents, tagged by logical position.

Every sub-page (session ``sid``, block ``blk``, layer ``l``, ``kv`` in {0: K, 1: V})
holds bf16 values drawn ~N(0,1): a window of ``T*H*D`` consecutive entries of
one seeded value table, starting at an offset hashed from (seed, sid, blk, l, kv).
Token rows at or beyond the session's context length are zero.

Because the content is a function of the logical position only, the expected
bytes at any physical location follow from which block owns it, which is what
the parity tests use at sizes where full byte images do not fit in host RAM.

Two implementations of the same definition are given: numpy (host) and torch
(any device, used to fill device pools quickly).  Both use exact integer
operations only (a table gather and a row mask), so they agree bit for bit.
"""
from __future__ import annotations

import numpy as np

from .configs import KVShape

TABLE_LEN = 1 << 22   # 4 Mi bf16 values = 8 MiB

_SM_GAMMA = np.uint64(0x9E3779B97F4A7C15)
_SM_M1 = np.uint64(0xBF58476D1CE4E5B9)
_SM_M2 = np.uint64(0x94D049BB133111EB)


def _splitmix64(x: np.ndarray) -> np.ndarray:
    """SplitMix64 output function (Steele, Lea, Flood 2014) on uint64 arrays."""
    with np.errstate(over="ignore"):
        z = (x + _SM_GAMMA).astype(np.uint64)
        z = (z ^ (z >> np.uint64(30))) * _SM_M1
        z = (z ^ (z >> np.uint64(27))) * _SM_M2
        return z ^ (z >> np.uint64(31))


def value_table(seed: int) -> np.ndarray:
    """``TABLE_LEN`` bf16 values ~N(0,1) as uint16 bit patterns, from ``seed``."""
    import torch
    g = torch.Generator().manual_seed(int(seed) * 1_000_003 + 17)
    v = torch.randn(TABLE_LEN, generator=g, dtype=torch.float32).to(torch.bfloat16)
    return v.view(torch.int16).numpy().view(np.uint16).copy()


def subpage_offsets(seed: int, sid, blk, layer, kv, shape: KVShape) -> np.ndarray:
    """Start offset in the value table of each sub-page's window (int64 array)."""
    sid = np.asarray(sid, dtype=np.uint64)
    blk = np.asarray(blk, dtype=np.uint64)
    layer = np.asarray(layer, dtype=np.uint64)
    kv = np.asarray(kv, dtype=np.uint64)
    key = ((np.uint64(seed & 0xFFFF) << np.uint64(48)) | ((sid & np.uint64(0xFFFF)) << np.uint64(32))
           | ((blk & np.uint64(0x3FFFFF)) << np.uint64(10)) | ((layer & np.uint64(0x1FF)) << np.uint64(1))
           | (kv & np.uint64(1)))
    span = np.uint64(TABLE_LEN - shape.subpage_elems + 1)
    return (_splitmix64(key) % span).astype(np.int64)


def valid_rows(ctx_tokens, blk, shape: KVShape) -> np.ndarray:
    """Token rows of block ``blk`` that lie inside a context of ``ctx_tokens`` (0..T)."""
    T = shape.page_tokens
    r = np.asarray(ctx_tokens, dtype=np.int64) - np.asarray(blk, dtype=np.int64) * T
    return np.clip(r, 0, T)


def subpage_values_np(table: np.ndarray, offsets, rows, shape: KVShape) -> np.ndarray:
    """uint16 [n, T*H*D] contents of n sub-pages (host)."""
    offsets = np.atleast_1d(np.asarray(offsets, dtype=np.int64))
    rows = np.atleast_1d(np.asarray(rows, dtype=np.int64))
    idx = offsets[:, None] + np.arange(shape.subpage_elems, dtype=np.int64)[None, :]
    out = table[idx]
    tok = np.arange(shape.subpage_elems, dtype=np.int64) // shape.row_elems
    out[tok[None, :] >= rows[:, None]] = 0
    return out


def subpage_values_torch(table_t, offsets_t, rows_t, shape: KVShape):
    """int16 [n, T*H*D] contents of n sub-pages on ``table_t``'s device.

    ``table_t`` is the value table as an int16 tensor; ``offsets_t`` and ``rows_t``
    are int64 tensors on the same device.
    """
    import torch
    dev = table_t.device
    ar = torch.arange(shape.subpage_elems, dtype=torch.int64, device=dev)
    idx = offsets_t[:, None] + ar[None, :]
    out = table_t[idx]
    tok = ar // shape.row_elems
    out.masked_fill_(tok[None, :] >= rows_t[:, None], 0)
    return out


# ------------------------------------------------------------- address-tagged content
# A debugging mode: every 16-byte chunk of a sub-page holds where it belongs, as four
# little-endian uint32 words (sid, token = blk * T + row, 2 * layer + kv, chunk within
# the row), so a byte found in the wrong place says which token, layer and chunk it
# is.  Rows past the context end are zero, as in the seeded mode.  Needs token rows
# of a multiple of 16 bytes.

def tagged_values_np(sid, blk, layer, kv, rows, shape: KVShape) -> np.ndarray:
    """uint16 [n, T*H*D] address-tagged contents of n sub-pages (host)."""
    sid = np.atleast_1d(np.asarray(sid, dtype=np.uint32))
    n = sid.size
    blk = np.broadcast_to(np.asarray(blk, dtype=np.uint32), (n,))
    jj = np.broadcast_to(np.asarray(layer, dtype=np.uint32) * 2 + np.asarray(kv, dtype=np.uint32), (n,))
    rows = np.broadcast_to(np.asarray(rows, dtype=np.int64), (n,))
    T = shape.page_tokens
    cpr = shape.row_elems * shape.elem_bytes // 16           # chunks per token row
    assert cpr * 16 == shape.row_elems * shape.elem_bytes
    w = np.zeros((n, T, cpr, 4), dtype=np.uint32)
    w[..., 0] = sid[:, None, None]
    w[..., 1] = blk[:, None, None] * np.uint32(T) + np.arange(T, dtype=np.uint32)[None, :, None]
    w[..., 2] = jj[:, None, None]
    w[..., 3] = np.arange(cpr, dtype=np.uint32)[None, None, :]
    w[np.arange(T)[None, :] >= rows[:, None]] = 0
    return w.reshape(n, -1).view(np.uint16).reshape(n, shape.subpage_elems)


def tagged_values_torch(sid, blk, layer, kv, rows, shape: KVShape, device):
    """int16 [n, T*H*D]: the same contents built on ``device``."""
    import torch
    as_t = lambda a: torch.as_tensor(np.asarray(a, dtype=np.int64), device=device)
    sid, blk, rows = as_t(sid), as_t(blk), as_t(rows)
    jj = as_t(np.asarray(layer) * 2 + np.asarray(kv)).expand(sid.shape[0])
    n = sid.shape[0]
    T = shape.page_tokens
    cpr = shape.row_elems * shape.elem_bytes // 16
    tok = torch.arange(T, device=device, dtype=torch.int64)
    w = torch.zeros((n, T, cpr, 4), dtype=torch.int64, device=device)
    w[..., 0] = sid[:, None, None]
    w[..., 1] = blk[:, None, None] * T + tok[None, :, None]
    w[..., 2] = jj[:, None, None]
    w[..., 3] = torch.arange(cpr, device=device, dtype=torch.int64)[None, None, :]
    w.masked_fill_((tok[None, :] >= rows[:, None])[:, :, None, None], 0)
    return w.to(torch.int32).reshape(n, -1).view(torch.int16).reshape(n, shape.subpage_elems)


def decode_tag(chunk16: bytes):
    """(sid, token, layer, kv, chunk) of a 16-byte address-tagged chunk."""
    w = np.frombuffer(bytes(chunk16), dtype="<u4")
    return int(w[0]), int(w[1]), int(w[2]) // 2, int(w[2]) % 2, int(w[3])
