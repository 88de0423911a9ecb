"""Pins for the oracle's page checksum: Python integers mod 2^64 (no numpy
wrap-around), unit vectors, zero pages, and sensitivity to word order."""
import numpy as np

from oracle.pool import OraclePool

M = 1 << 64


def _pool(seed):
    p = OraclePool(2, 1, 8, 16, 2, n_sessions=1, max_blocks=4, hbm_pages=4, hbm_budget_pages=4,
                   host_pages=0)
    rng = np.random.default_rng(seed)
    p.hbm[:] = rng.integers(0, 256, p.hbm.shape, dtype=np.uint8)
    return p


def _by_python_ints(p, page):
    raw = bytes(np.ascontiguousarray(p.hbm[:, page, :]).reshape(-1))
    total = 0
    for q in range(len(raw) // 8):
        w = int.from_bytes(raw[8 * q:8 * q + 8], "little")
        total = (total + w * (2 * q + 1)) % M
    return total


def test_checksum_equals_the_definition_in_python_integers():
    for seed in range(3):
        p = _pool(seed)
        for page in range(4):
            assert p.page_checksum(page) == _by_python_ints(p, page)


def test_checksum_special_cases():
    p = _pool(0)
    p.hbm[:, 1, :] = 0
    assert p.page_checksum(1) == 0
    J, P = p.hbm.shape[0], p.hbm.shape[2]
    q = (J * P // 8) - 3                       # a word in the last sub-page
    j, off = divmod(q * 8, P)
    p.hbm[j, 1, off] = 1                       # w_q = 1
    assert p.page_checksum(1) == 2 * q + 1
    p.hbm[:, 2, :] = 0xFF                      # every word 2^64 - 1: sum = -(sum of weights)
    m = J * P // 8
    assert p.page_checksum(2) == (-(m * m)) % M


def test_checksum_depends_on_word_order():
    p = _pool(1)
    before = p.page_checksum(0)
    a = p.hbm[0, 0, :8].copy()
    p.hbm[0, 0, :8] = p.hbm[1, 0, :8]
    p.hbm[1, 0, :8] = a                        # swap two words in different sub-pages
    assert p.page_checksum(0) != before
