"""Pins for the fp64 verify-attention oracle (CPU only).

The oracle is checked against things other than itself:
* torch's float64 scaled_dot_product_attention (a library routine) on tiny
  shapes, fed from DENSE K/V that the test scatters into pages itself;
* the prefix form of the causal verify mask: draft row i is ordinary,
  unmasked attention over the first L-k+i keys;
* closed forms (a single key, all-equal keys, one dominant key, distinct
  constant V per KV head that exposes the query-head -> KV-head map);
* exact invariances (page permutation, contiguous vs paged layout) and the
  defined degenerate cases (rows with no key, clamped context, bad page ids).
"""
import math

import numpy as np
import pytest
import torch
import torch.nn.functional as F

import oracle


def bf16_round(x: np.ndarray) -> tuple[np.ndarray, np.ndarray]:
    """(bf16 bit patterns, exact float64 values) of x rounded to bf16 by torch."""
    t = torch.from_numpy(np.asarray(x, dtype=np.float32)).to(torch.bfloat16)
    return t.view(torch.int16).numpy().view(np.uint16), t.to(torch.float64).numpy()


def make_case(rng, B, k, Hq, Hkv, D, ps, lens, extra_pages=3, contiguous=False):
    """Dense fp64 tensors plus the same data scattered into a paged pool by slicing."""
    lens = [int(L) for L in lens]
    max_pages = max(1, max(-(-L // ps) for L in lens))
    Lpad = max_pages * ps
    q_bits, q = bf16_round(rng.standard_normal((B, k + 1, Hq, D)))
    k_bits_d, k_dense = bf16_round(rng.standard_normal((B, Hkv, Lpad, D)))
    v_bits_d, v_dense = bf16_round(rng.standard_normal((B, Hkv, Lpad, D)))
    n_pages = [-(-L // ps) for L in lens]
    P = sum(n_pages) + extra_pages
    order = np.arange(P) if contiguous else rng.permutation(P)
    # unused pool slots hold unrelated data
    kpool, _ = bf16_round(rng.standard_normal((P, Hkv, ps, D)))
    vpool, _ = bf16_round(rng.standard_normal((P, Hkv, ps, D)))
    table = np.full((B, max_pages), -1, dtype=np.int32)
    nxt = 0
    for b in range(B):
        for j in range(n_pages[b]):
            pid = int(order[nxt])
            nxt += 1
            table[b, j] = pid
            kpool[pid] = k_bits_d[b, :, j * ps:(j + 1) * ps, :]
            vpool[pid] = v_bits_d[b, :, j * ps:(j + 1) * ps, :]
    return dict(q_bits=q_bits, q=q, k_dense=k_dense, v_dense=v_dense, kpool=kpool,
                vpool=vpool, table=table, lens=np.asarray(lens, dtype=np.int32), k=k)


def run_oracle(c, scale=0.0):
    return oracle.verify_attention(c["q_bits"], c["kpool"], c["vpool"], c["table"],
                                   c["lens"], c["k"], scale)


def sdpa_masked(c, Hq, Hkv, scale=None):
    """torch float64 SDPA with an explicit boolean causal-verify mask."""
    B, rows = c["q"].shape[:2]
    G = Hq // Hkv
    out = np.zeros_like(c["q"])
    for b in range(B):
        L = int(c["lens"][b])
        q = torch.from_numpy(c["q"][b]).transpose(0, 1)                 # [Hq, rows, D]
        kk = torch.from_numpy(c["k_dense"][b, :, :L]).repeat_interleave(G, dim=0)
        vv = torch.from_numpy(c["v_dense"][b, :, :L]).repeat_interleave(G, dim=0)
        i = torch.arange(rows)[:, None]
        j = torch.arange(L)[None, :]
        mask = j <= (L - rows + i)                                      # [rows, L]
        o = F.scaled_dot_product_attention(q, kk, vv, attn_mask=mask, scale=scale)
        out[b] = o.transpose(0, 1).numpy()
    return out


def sdpa_prefix(c, Hq, Hkv, scale=None):
    """Row i as plain unmasked attention over the first L-k+i keys."""
    B, rows = c["q"].shape[:2]
    G = Hq // Hkv
    out = np.zeros_like(c["q"])
    for b in range(B):
        L = int(c["lens"][b])
        for i in range(rows):
            n = L - rows + 1 + i
            q = torch.from_numpy(c["q"][b, i])[:, None, :]               # [Hq, 1, D]
            kk = torch.from_numpy(c["k_dense"][b, :, :n]).repeat_interleave(G, dim=0)
            vv = torch.from_numpy(c["v_dense"][b, :, :n]).repeat_interleave(G, dim=0)
            out[b, i] = F.scaled_dot_product_attention(q, kk, vv, scale=scale)[:, 0].numpy()
    return out


@pytest.mark.parametrize("seed", range(6))
def test_matches_torch_sdpa_masked(seed):
    rng = np.random.default_rng(100 + seed)
    B = int(rng.integers(1, 3))
    k = int(rng.integers(1, 4))
    Hkv = 2
    Hq = 4
    D = 8
    ps = int(rng.choice([2, 4, 8]))
    lens = rng.integers(k + 1, 41, size=B)
    c = make_case(rng, B, k, Hq, Hkv, D, ps, lens)
    got = run_oracle(c)
    ref = sdpa_masked(c, Hq, Hkv)
    np.testing.assert_allclose(got, ref, rtol=1e-12, atol=1e-13)


@pytest.mark.parametrize("seed", range(4))
def test_matches_prefix_form(seed):
    rng = np.random.default_rng(200 + seed)
    k = int(rng.integers(1, 5))
    c = make_case(rng, 2, k, 8, 2, 16, 4, rng.integers(k + 1, 60, size=2))
    np.testing.assert_allclose(run_oracle(c), sdpa_prefix(c, 8, 2), rtol=1e-12, atol=1e-13)


def test_last_row_is_full_decode_attention():
    rng = np.random.default_rng(7)
    c = make_case(rng, 1, 3, 4, 4, 8, 4, [23])
    got = run_oracle(c)[0, 3]
    q = torch.from_numpy(c["q"][0, 3])[:, None, :]
    ref = F.scaled_dot_product_attention(q, torch.from_numpy(c["k_dense"][0, :, :23]),
                                         torch.from_numpy(c["v_dense"][0, :, :23]))[:, 0]
    np.testing.assert_allclose(got, ref.numpy(), rtol=1e-12, atol=1e-13)


def test_custom_scale():
    rng = np.random.default_rng(8)
    c = make_case(rng, 2, 2, 4, 2, 8, 4, [9, 17])
    np.testing.assert_allclose(run_oracle(c, scale=0.77), sdpa_masked(c, 4, 2, scale=0.77),
                               rtol=1e-12, atol=1e-13)


def test_single_key_returns_its_value():
    # L = k+1: row 0 sees exactly key 0, so o = V_0 whatever q is
    rng = np.random.default_rng(9)
    k = 3
    c = make_case(rng, 1, k, 4, 2, 8, 4, [k + 1])
    got = run_oracle(c)
    for h in range(4):
        np.testing.assert_array_equal(got[0, 0, h], c["v_dense"][0, h // 2, 0])


def test_equal_keys_give_mean_of_values():
    rng = np.random.default_rng(10)
    k, L = 2, 13
    c = make_case(rng, 1, k, 2, 1, 8, 4, [L])
    # make every K row identical, in both the dense copy and the pool
    c["k_dense"][:] = c["k_dense"][0, 0, 0]
    c["kpool"][:] = c["kpool"][c["table"][0, 0], 0, 0]
    got = run_oracle(c)
    for i in range(k + 1):
        n = L - k + i
        np.testing.assert_allclose(got[0, i, 0], c["v_dense"][0, 0, :n].mean(axis=0),
                                   rtol=1e-12, atol=1e-14)


def test_dominant_key():
    # q = 0 except one coordinate; K_5 has a huge value there: softmax ~ one-hot on key 5
    rng = np.random.default_rng(11)
    k, L, D = 1, 12, 8
    c = make_case(rng, 1, k, 1, 1, D, 4, [L])
    qb, qv = bf16_round(np.eye(1, D, 0) * 8.0)
    c["q_bits"][0, :, 0] = qb[0]
    c["q"][0, :, 0] = qv[0]
    pid, slot = c["table"][0, 5 // 4], 5 % 4
    kb, _ = bf16_round(np.full((D,), 64.0))
    c["kpool"][pid, 0, slot] = kb
    got = run_oracle(c)
    np.testing.assert_allclose(got[0, 1, 0], c["v_dense"][0, 0, 5], rtol=0, atol=1e-60)


def test_gqa_head_map_consecutive_query_heads_share_a_kv_head():
    # V of KV head g is the constant g+1, so every output coordinate names its KV head
    rng = np.random.default_rng(12)
    Hq, Hkv = 12, 3
    c = make_case(rng, 2, 2, Hq, Hkv, 8, 4, [10, 7])
    for g in range(Hkv):
        bits, _ = bf16_round(np.full((8,), float(g + 1)))
        c["vpool"][:, g] = bits
    got = run_oracle(c)
    for h in range(Hq):
        np.testing.assert_allclose(got[:, :, h], h // (Hq // Hkv) + 1.0, rtol=1e-14)


def test_page_permutation_invariance_is_exact():
    rng = np.random.default_rng(13)
    c = make_case(rng, 3, 3, 4, 2, 8, 4, [17, 30, 9])
    base = run_oracle(c)
    P = c["kpool"].shape[0]
    perm = rng.permutation(P)            # new slot of old page p is perm[p]
    kp = np.empty_like(c["kpool"])
    vp = np.empty_like(c["vpool"])
    kp[perm] = c["kpool"]
    vp[perm] = c["vpool"]
    table = np.where(c["table"] >= 0, perm[np.maximum(c["table"], 0)], -1).astype(np.int32)
    got = oracle.verify_attention(c["q_bits"], kp, vp, table, c["lens"], c["k"])
    np.testing.assert_array_equal(got, base)


def test_contiguous_equals_paged():
    rng1 = np.random.default_rng(14)
    rng2 = np.random.default_rng(14)
    c1 = make_case(rng1, 2, 2, 4, 2, 8, 8, [20, 33], contiguous=True)
    c2 = make_case(rng2, 2, 2, 4, 2, 8, 8, [20, 33], contiguous=False)
    np.testing.assert_array_equal(run_oracle(c1), run_oracle(c2))


def test_rows_without_keys_are_zero():
    # L < k+1: row i has keys iff L-(k+1)+i >= 0
    rng = np.random.default_rng(15)
    k = 4
    c = make_case(rng, 1, k, 2, 1, 8, 4, [k + 1])
    c["lens"][0] = 2
    got = run_oracle(c)
    for i in range(k + 1):
        if 2 - (k + 1) + i < 0:
            assert np.all(got[0, i] == 0.0)
        else:
            n = 2 - k + i
            assert n >= 1 and np.all(np.isfinite(got[0, i]))
    c["lens"][0] = 0
    assert np.all(run_oracle(c) == 0.0)


def test_context_longer_than_table_is_clamped():
    rng = np.random.default_rng(16)
    c = make_case(rng, 1, 2, 2, 1, 8, 4, [12], extra_pages=0)
    assert c["table"].shape[1] * 4 == 12
    base = run_oracle(c)
    c["lens"][0] = 12 + 50
    np.testing.assert_array_equal(run_oracle(c), base)


def test_out_of_range_page_reads_zeros():
    rng = np.random.default_rng(17)
    k, ps = 1, 4
    c = make_case(rng, 1, k, 2, 1, 8, ps, [12])
    P = c["kpool"].shape[0]
    c["table"][0, 1] = P + 5          # keys 4..7 now read as zero rows
    c["k_dense"][0, :, 4:8] = 0.0
    c["v_dense"][0, :, 4:8] = 0.0
    np.testing.assert_allclose(run_oracle(c), sdpa_masked(c, 2, 1), rtol=1e-12, atol=1e-13)
    c["table"][0, 1] = -7
    np.testing.assert_allclose(run_oracle(c), sdpa_masked(c, 2, 1), rtol=1e-12, atol=1e-13)


def test_empty_batch():
    out = oracle.verify_attention(np.zeros((0, 2, 2, 8), np.uint16), np.zeros((1, 1, 4, 8), np.uint16),
                                  np.zeros((1, 1, 4, 8), np.uint16), np.zeros((0, 1), np.int32),
                                  np.zeros((0,), np.int32), 1)
    assert out.shape == (0, 2, 2, 8)


def test_bf16_widening_is_exact():
    # bf16 bit patterns with known values: 0x3F80 = 1, 0xC000 = -2, 0x3E00 = 0.125
    q = np.zeros((1, 1, 1, 8), np.uint16)
    kp = np.zeros((1, 1, 4, 8), np.uint16)
    vp = np.zeros((1, 1, 4, 8), np.uint16)
    vp[0, 0, 0, :3] = [0x3F80, 0xC000, 0x3E00]
    out = oracle.verify_attention(q, kp, vp, np.zeros((1, 1), np.int32), np.array([1], np.int32), 0)
    assert out[0, 0, 0, :3].tolist() == [1.0, -2.0, 0.125]
    assert math.isclose(out[0, 0, 0, 3], 0.0)


def test_large_values_match_torch_sdpa():
    """V entries across bf16's whole range (up to ~3.39e38, far beyond fp16's
    65504) are exact in fp64: the oracle still equals torch's float64 SDPA."""
    rng = np.random.default_rng(77)
    B, k, Hq, Hkv, D, ps = 2, 3, 4, 2, 8, 4
    c = make_case(rng, B, k, Hq, Hkv, D, ps, [29, 38])
    big = [3.3e38, -3.0e38, 1.0e5, -65536.0, 65280.0, 2.0e20]
    for b in range(B):
        L = int(c["lens"][b])
        for h in range(Hkv):
            for val, d in zip(big, rng.choice(D, len(big), replace=False)):
                key = int(rng.integers(0, L))
                bits, exact = bf16_round(np.array([val]))
                page, slot = int(c["table"][b, key // ps]), key % ps
                c["vpool"][page, h, slot, d] = bits[0]
                c["v_dense"][b, h, key, d] = exact[0]
    got = run_oracle(c)
    ref = sdpa_masked(c, Hq, Hkv)
    assert np.isfinite(got).all() and np.abs(ref).max() > 1e37
    np.testing.assert_allclose(got, ref, rtol=1e-12, atol=1e-13 * np.abs(ref).max())
