"""Address-tagged KV contents: the generators agree, and the oracle's byte images
decode to their owners.

With tagged contents every 16-byte chunk names the (session, token, layer, K/V,
chunk) it belongs to, so the oracle's copy semantics can be checked in closed form:
after any sequence of evictions, reloads, preloads and growth, every chunk of every
block, wherever the block lives, must name exactly that block's token and place."""
import numpy as np

from oracle import OracleManager
from workloads import make_workload
from workloads.configs import TINY_SHAPE
from workloads.content import decode_tag, tagged_values_np, tagged_values_torch


def test_numpy_and_torch_generators_agree_and_decode():
    rng = np.random.default_rng(0)
    n = 40
    sid = rng.integers(0, 4096, n)
    blk = rng.integers(0, 4096, n)
    layer = rng.integers(0, 2, n)
    kv = rng.integers(0, 2, n)
    rows = rng.integers(0, 17, n)
    a = tagged_values_np(sid, blk, layer, kv, rows, TINY_SHAPE)
    b = tagged_values_torch(sid, blk, layer, kv, rows, TINY_SHAPE, "cpu").numpy().view(np.uint16)
    assert np.array_equal(a, b)
    T, cpr = TINY_SHAPE.page_tokens, TINY_SHAPE.row_elems * 2 // 16
    for i in range(n):
        by = a[i].view(np.uint8)
        for r in (0, int(rows[i]) - 1, T - 1):
            if r < 0:
                continue
            for c in (0, cpr - 1):
                at = (r * cpr + c) * 16
                got = decode_tag(by[at:at + 16])
                if r < rows[i]:
                    assert got == (int(sid[i]), int(blk[i]) * T + r, int(layer[i]), int(kv[i]), c)
                else:
                    assert got == (0, 0, 0, 0, 0)


def test_oracle_bytes_decode_to_their_owner():
    wl = make_workload("tiny", 5)
    om = OracleManager(wl, with_bytes=True, content="tagged", rank_on="none")
    for i in range(600):
        om.step(i)
    pool, sh = om.pool, TINY_SHAPE
    T, cpr = sh.page_tokens, sh.row_elems * 2 // 16
    assert om.counters["pages_out"] > 100 and om.counters["pages_in"] > 50
    checked = 0
    for s in range(pool.S):
        for b in range(int(pool.nblocks[s])):
            e = int(pool.tables[s, b])
            img = pool.hbm[:, e, :] if e >= 0 else pool.host[-(e + 2)]
            rows = max(0, min(T, int(pool.ctx[s]) - b * T))
            w = img.reshape(2 * sh.layers, T, cpr, 4, 4).view(np.uint32).reshape(2 * sh.layers, T, cpr, 4)
            for j in range(2 * sh.layers):
                want = np.zeros((T, cpr, 4), np.uint32)
                want[:rows, :, 0] = s
                want[:rows, :, 1] = b * T + np.arange(rows)[:, None]
                want[:rows, :, 2] = j
                want[:rows, :, 3] = np.arange(cpr)[None, :]
                assert np.array_equal(w[j], want), (s, b, j)
                checked += 1
    assert checked > 100
