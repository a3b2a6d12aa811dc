"""Pins for the paged KV cache oracle (CPU only): append and commit.

Checked against what the layout and the step fix, written independently
here with numpy indexing:

* read-back: after the append, the rows at key positions L_b-n .. L_b-1 of
  every request, gathered through the page table, are the new rows, and
  every other slot of both pools is unchanged;
* rows whose position is negative (a context shorter than the new rows) or
  whose page id is out of range are not written;
* appending a context's rows one position at a time equals appending them
  all at once, and equals scattering the dense context into its pages;
* commit keeps L - k + a rows and never goes below zero.
"""
import numpy as np
import pytest

import oracle


def pools(rng, P, H, ps, D=128):
    k = rng.integers(0, 1 << 16, size=(P, H, ps, D), dtype=np.uint16)
    v = rng.integers(0, 1 << 16, size=(P, H, ps, D), dtype=np.uint16)
    return k, v


def gather(pool, page_table, b, pos, ps):
    return pool[page_table[b, pos // ps], :, pos % ps, :]


@pytest.mark.parametrize("B,n,H,ps,seed", [(3, 5, 2, 16, 0), (2, 1, 4, 8, 1), (4, 17, 1, 32, 2), (1, 9, 8, 256, 3)])
def test_read_back_and_untouched_slots(B, n, H, ps, seed):
    rng = np.random.default_rng(seed)
    max_pages = 6
    P = B * max_pages
    kp, vp = pools(rng, P, H, ps)
    k0, v0 = kp.copy(), vp.copy()
    pt = rng.permutation(P).astype(np.int32).reshape(B, max_pages)
    L = rng.integers(n, max_pages * ps + 1, size=B).astype(np.int32)
    nk = rng.integers(0, 1 << 16, size=(B, n, H, 128), dtype=np.uint16)
    nv = rng.integers(0, 1 << 16, size=(B, n, H, 128), dtype=np.uint16)
    oracle.kv_append(nk, nv, kp, vp, pt, L)
    written = np.zeros(kp.shape[:3], dtype=bool)
    for b in range(B):
        for i in range(n):
            pos = L[b] - n + i
            np.testing.assert_array_equal(gather(kp, pt, b, pos, ps), nk[b, i])
            np.testing.assert_array_equal(gather(vp, pt, b, pos, ps), nv[b, i])
            written[pt[b, pos // ps], :, pos % ps] = True
    np.testing.assert_array_equal(kp[~written], k0[~written])
    np.testing.assert_array_equal(vp[~written], v0[~written])


def test_short_contexts_and_bad_pages_write_nothing():
    rng = np.random.default_rng(4)
    B, n, H, ps, max_pages, P = 4, 6, 2, 16, 4, 8
    kp, vp = pools(rng, P, H, ps)
    k0 = kp.copy()
    pt = np.array([[0, 1, 2, 3], [4, 5, 6, 7], [-1, 99, 8, 1 << 30], [3, 2, 1, 0]], dtype=np.int32)
    L = np.array([3, 0, 40, -5], dtype=np.int32)     # 3 < n: only rows 3..5; 0 and -5: nothing
    nk = rng.integers(0, 1 << 16, size=(B, n, H, 128), dtype=np.uint16)
    oracle.kv_append(nk, nk, kp, vp, pt, L)
    for i in range(n):
        pos = 3 - n + i
        if pos >= 0:
            np.testing.assert_array_equal(kp[pt[0, pos // ps], :, pos % ps], nk[0, i])
    # request 2 lands in page ids -1, 99, 8, 2^30: all outside [0, 8), so the
    # pool changes only where request 0 wrote
    changed = np.any(kp != k0, axis=-1)
    assert changed.sum() == 3 * H


def test_one_at_a_time_equals_all_at_once_equals_dense_scatter():
    rng = np.random.default_rng(5)
    B, H, ps, max_pages = 3, 2, 16, 5
    P = B * max_pages
    pt = rng.permutation(P).astype(np.int32).reshape(B, max_pages)
    L = np.array([37, 80, 5], dtype=np.int32)
    dense_k = rng.integers(0, 1 << 16, size=(B, 80, H, 128), dtype=np.uint16)
    dense_v = rng.integers(0, 1 << 16, size=(B, 80, H, 128), dtype=np.uint16)
    a_k, a_v = np.zeros((P, H, ps, 128), np.uint16), np.zeros((P, H, ps, 128), np.uint16)
    b_k, b_v = a_k.copy(), a_v.copy()
    c_k, c_v = a_k.copy(), a_v.copy()
    # all at once: the last L_b rows of a context of L_b (per request)
    for b in range(B):
        one = lambda arr: np.ascontiguousarray(arr[b:b + 1, :L[b]])
        oracle.kv_append(one(dense_k), one(dense_v), a_k, a_v, pt[b:b + 1], L[b:b + 1])
    # one position at a time, the context growing by one each call
    for b in range(B):
        for t in range(1, L[b] + 1):
            oracle.kv_append(np.ascontiguousarray(dense_k[b:b + 1, t - 1:t]),
                             np.ascontiguousarray(dense_v[b:b + 1, t - 1:t]), b_k, b_v, pt[b:b + 1],
                             np.array([t], np.int32))
    # the layout written directly
    for b in range(B):
        for pos in range(L[b]):
            c_k[pt[b, pos // ps], :, pos % ps] = dense_k[b, pos]
            c_v[pt[b, pos // ps], :, pos % ps] = dense_v[b, pos]
    for x, y in ((a_k, b_k), (a_k, c_k), (a_v, b_v), (a_v, c_v)):
        np.testing.assert_array_equal(x, y)


def test_commit():
    L = np.array([10, 6, 0, 3, 100], dtype=np.int32)
    a = np.array([0, 5, 0, 0, 2], dtype=np.int32)
    np.testing.assert_array_equal(oracle.kv_commit(L, a, 5), [5, 6, 0, 0, 97])
    rng = np.random.default_rng(6)
    for k in (1, 4, 16):
        L = rng.integers(k + 1, 10000, size=64).astype(np.int32)
        a = rng.integers(0, k + 1, size=64).astype(np.int32)
        got = oracle.kv_commit(L, a, k)
        assert ((got <= L) & (got >= L - k)).all()
        np.testing.assert_array_equal(got, L - k + a)
