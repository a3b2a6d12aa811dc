"""Pins for the fp64 token-tree oracle (CPU only): tree attention, the
multi-candidate acceptance walk and the commit of the accepted path.

The oracle is checked against facts other than itself:

* attention: torch's float64 scaled_dot_product_attention with an explicit
  boolean mask whose tree part comes from networkx's ancestor sets, fed from
  dense K/V that the test scatters into pages; a chain tree equals the chain
  verify attention; closed forms (equal keys give the mean of the visible
  values); page-permutation invariance; detached nodes;
* acceptance: exact enumeration on an 8-token vocabulary, where every accept
  threshold and draw cell is located by bisection on fp64 uniforms: with
  sibling tokens drawn independently from the parent's draft distribution,
  the first emitted token follows p_root and, after an accepted child with
  token v, the next one follows that child's target distribution (the
  defining property of lossless multi-candidate speculative sampling);
  disjoint supports reject every sibling and draw from p; p == q accepts the
  first child; a chain tree reproduces the chain acceptance; greedy walks
  follow numpy's argmax; Monte Carlo histogram of the first emitted token;
* commit: numpy read-back of every slot of the pool.
"""
import math

import networkx as nx
import numpy as np
import pytest
import torch
import torch.nn.functional as F
from scipy.special import softmax

import oracle

TOP = float(np.nextafter(1.0, 0.0))


def bf16_round(x):
    t = torch.from_numpy(np.asarray(x, dtype=np.float32)).to(torch.bfloat16)
    return t.view(torch.int16).numpy().view(np.uint16), t.to(torch.float64).numpy()


def ancestors_or_self(parents):
    """Per node, the set of its ancestors and itself, from a networkx DiGraph."""
    g = nx.DiGraph()
    n = len(parents)
    g.add_nodes_from(range(n))
    for c in range(1, n):
        if 0 <= parents[c] < c:
            g.add_edge(int(parents[c]), c)
    return [nx.ancestors(g, i) | {i} for i in range(n)]


def paged_case(rng, B, n, Hq, Hkv, D, ps, lens, extra_pages=2):
    lens = [int(L) for L in lens]
    max_pages = max(1, max(-(-L // ps) for L in lens))
    Lpad = max_pages * ps
    q_bits, q = bf16_round(rng.standard_normal((B, n, Hq, D)))
    kb, kd = bf16_round(rng.standard_normal((B, Hkv, Lpad, D)))
    vb, vd = bf16_round(rng.standard_normal((B, Hkv, Lpad, D)))
    n_pages = [-(-L // ps) for L in lens]
    P = sum(n_pages) + extra_pages
    order = rng.permutation(P)
    kpool, _ = bf16_round(rng.standard_normal((P, Hkv, ps, D)))
    vpool, _ = bf16_round(rng.standard_normal((P, Hkv, ps, D)))
    table = np.full((B, max_pages), -1, np.int32)
    nxt = 0
    for b in range(B):
        for j in range(n_pages[b]):
            pid = int(order[nxt])
            nxt += 1
            table[b, j] = pid
            kpool[pid] = kb[b, :, j * ps:(j + 1) * ps]
            vpool[pid] = vb[b, :, j * ps:(j + 1) * ps]
    return dict(q_bits=q_bits, q=q, kd=kd, vd=vd, kpool=kpool, vpool=vpool, table=table,
                lens=np.asarray(lens, np.int32))


def random_parents(rng, n):
    par = np.full(n, -1, np.int32)
    for c in range(1, n):
        par[c] = rng.integers(0, c)
    return par


# --------------------------------------------------------------- attention
@pytest.mark.parametrize("seed,B,n,Hq,Hkv,ps,lens", [
    (0, 2, 5, 4, 2, 4, [13, 9]),
    (1, 1, 7, 6, 3, 8, [30]),
    (2, 3, 4, 2, 1, 5, [4, 11, 7]),
])
def test_tree_attention_matches_sdpa_with_ancestor_mask(seed, B, n, Hq, Hkv, ps, lens):
    rng = np.random.default_rng(seed)
    D = 8
    c = paged_case(rng, B, n, Hq, Hkv, D, ps, lens)
    parents = np.stack([random_parents(rng, n) for _ in range(B)])
    got = oracle.tree_attention(c["q_bits"], c["kpool"], c["vpool"], c["table"], c["lens"], parents)
    G = Hq // Hkv
    for b in range(B):
        L = int(lens[b])
        anc = ancestors_or_self(parents[b])
        mask = np.zeros((n, L), bool)
        for i in range(n):
            for j in range(L):
                m = j - (L - n)
                mask[i, j] = m < 0 or m in anc[i]
        q = torch.from_numpy(c["q"][b]).permute(1, 0, 2)                       # [Hq, n, D]
        kk = torch.from_numpy(c["kd"][b, :, :L]).repeat_interleave(G, dim=0)   # [Hq, L, D]
        vv = torch.from_numpy(c["vd"][b, :, :L]).repeat_interleave(G, dim=0)
        ref = F.scaled_dot_product_attention(q, kk, vv, attn_mask=torch.from_numpy(mask))
        np.testing.assert_allclose(got[b], ref.permute(1, 0, 2).numpy(), rtol=1e-12, atol=1e-12)


def test_chain_tree_equals_chain_attention():
    rng = np.random.default_rng(3)
    B, k = 2, 4
    c = paged_case(rng, B, k + 1, 8, 2, 16, 4, [17, 23])
    chain = np.tile(np.arange(-1, k, dtype=np.int32), (B, 1))
    a = oracle.tree_attention(c["q_bits"], c["kpool"], c["vpool"], c["table"], c["lens"], chain)
    b = oracle.verify_attention(c["q_bits"], c["kpool"], c["vpool"], c["table"], c["lens"], k)
    assert np.array_equal(a, b)


def test_star_tree_with_equal_keys_averages_root_and_self():
    rng = np.random.default_rng(4)
    n, D = 5, 8
    c = paged_case(rng, 1, n, 2, 1, D, 4, [n])          # no prefix: the tree is the whole context
    row = c["kpool"][c["table"][0, 0], 0, 0].copy()
    for j in range(n):                                   # every key the same vector
        c["kpool"][c["table"][0, j // 4], 0, j % 4] = row
    parents = np.array([[-1, 0, 0, 0, 0]], np.int32)
    got = oracle.tree_attention(c["q_bits"], c["kpool"], c["vpool"], c["table"], c["lens"], parents)
    vals = np.stack([bf16_round(0)[1] * 0 + c["vd"][0, 0, j] for j in range(n)])
    np.testing.assert_allclose(got[0, 0, :, :], np.broadcast_to(vals[0], (2, D)), rtol=1e-12, atol=1e-12)
    for i in range(1, n):
        np.testing.assert_allclose(got[0, i, 0], 0.5 * (vals[0] + vals[i]), rtol=1e-12, atol=1e-12)


def test_page_permutation_invariance_and_detached_nodes():
    rng = np.random.default_rng(5)
    n = 6
    c = paged_case(rng, 1, n, 4, 2, 8, 4, [21])
    parents = np.array([[-1, 0, 1, 7, 0, -3]], np.int32)   # nodes 3 and 5 are detached
    a = oracle.tree_attention(c["q_bits"], c["kpool"], c["vpool"], c["table"], c["lens"], parents)
    perm = rng.permutation(c["kpool"].shape[0])
    inv = np.argsort(perm)
    t2 = np.where(c["table"] >= 0, inv[np.maximum(c["table"], 0)], -1).astype(np.int32)
    b = oracle.tree_attention(c["q_bits"], c["kpool"][perm], c["vpool"][perm], t2, c["lens"], parents)
    assert np.array_equal(a, b)
    # a detached node sees the prefix and itself: same as a child of nobody in a star
    star = np.array([[-1, 0, 1, -1, 0, -1]], np.int32)
    s = oracle.tree_attention(c["q_bits"], c["kpool"], c["vpool"], c["table"], c["lens"], star)
    assert np.array_equal(a, s)


def test_short_context_drops_missing_keys():
    rng = np.random.default_rng(6)
    n = 6
    c = paged_case(rng, 1, n, 2, 1, 8, 4, [3])           # L < n: nodes 0..2 have no row
    parents = np.array([[-1, 0, 1, 2, 3, 4]], np.int32)
    got = oracle.tree_attention(c["q_bits"], c["kpool"], c["vpool"], c["table"], c["lens"], parents)
    assert np.all(got[0, :3] == 0.0)
    chain = oracle.verify_attention(c["q_bits"], c["kpool"], c["vpool"], c["table"], c["lens"], n - 1)
    assert np.array_equal(got, chain)


# --------------------------------------------------------------- acceptance
def boundary(pred, B):
    """Per row, the b in [0, 1] with pred False on [0, b) and True on [b, 1)."""
    lo, hi = np.zeros(B), np.ones(B)
    top = pred(np.full(B, TOP))
    zero = pred(np.zeros(B))
    for _ in range(64):
        mid = 0.5 * (lo + hi)
        r = pred(mid)
        hi = np.where(r, mid, hi)
        lo = np.where(r, lo, mid)
    return np.where(~top, 1.0, np.where(zero, 0.0, hi))


class Batch:
    """Many single-tree requests run through the oracle together."""

    def __init__(self, zt, zd, parents, tokens, T):
        self.zt, self.zd, self.par, self.x, self.T = zt, zd, parents, tokens, T
        self.B, self.n = tokens.shape

    def run(self, u):
        return oracle.tree_accept(self.zt, self.zd, self.par, self.x, u, self.T)

    def threshold(self, base_u, col, pred_from):
        def pred(v):
            u = base_u.copy()
            u[:, col] = v
            return pred_from(self.run(u))
        return boundary(pred, self.B)

    def draw_law(self, base_u, pos, V):
        law = np.zeros((self.B, V))
        prev = np.zeros(self.B)
        for v in range(V):
            b = self.threshold(base_u, self.n - 1, lambda r, v=v: r["tokens"][:, pos] > v)
            law[:, v] = b - prev
            prev = b
        return law


def combos(V, m):
    grids = np.meshgrid(*[np.arange(V)] * m, indexing="ij")
    return np.stack([g.reshape(-1) for g in grids], axis=1)


@pytest.mark.parametrize("T,seed,dtype", [(1.0, 0, "f32"), (0.7, 1, "bf16"), (1.6, 2, "f32")])
def test_two_level_tree_is_lossless_by_enumeration(T, seed, dtype):
    """Root with two children, each with one child; tokens drawn i.i.d. from the
    parent's draft distribution.  First emitted token ~ p_root; after accepting a
    child with token v the second ~ P1[v] (that child's target row)."""
    V = 8
    rng = np.random.default_rng(seed)
    raw = lambda *s: rng.standard_normal(s) * 1.5
    zt_root, zd_root = raw(V), None
    zd_root = zt_root + raw(V)
    P1, Q1 = raw(V, V), None                     # target / draft rows of a depth-1 node, by its token
    Q1 = P1 + raw(V, V)
    leaf = raw(V)
    if dtype == "bf16":
        to = lambda a: bf16_round(a)
    else:
        to = lambda a: (np.asarray(a, np.float32), np.asarray(a, np.float32).astype(np.float64))
    # node order: 0 root, 1 = c1, 2 = c2, 3 = child of c1, 4 = child of c2
    parents = np.array([-1, 0, 0, 1, 2], np.int32)
    X = combos(V, 4)                             # (x_c1, x_c2, x_d1, x_d2)
    B = X.shape[0]
    zt = np.zeros((B, 5, V))
    zd = np.zeros((B, 5, V))
    zt[:, 0], zd[:, 0] = zt_root, zd_root
    zt[:, 1], zd[:, 1] = P1[X[:, 0]], Q1[X[:, 0]]
    zt[:, 2], zd[:, 2] = P1[X[:, 1]], Q1[X[:, 1]]
    zt[:, 3] = zt[:, 4] = leaf
    zd[:, 3] = zd[:, 4] = leaf
    zt_in, zt64 = to(zt)
    zd_in, zd64 = to(zd)
    tokens = np.zeros((B, 5), np.int32)
    tokens[:, 1:] = X
    req = Batch(zt_in, zd_in, np.tile(parents, (B, 1)), tokens, T)
    p_root, q_root = softmax(zt64[0, 0] / T), softmax(zd64[0, 0] / T)
    P1p = softmax(np.stack([zt64[np.argmax(X[:, 0] == v), 1] for v in range(V)]) / T, axis=-1)
    Q1p = softmax(np.stack([zd64[np.argmax(X[:, 0] == v), 1] for v in range(V)]) / T, axis=-1)
    w = q_root[X[:, 0]] * q_root[X[:, 1]] * Q1p[X[:, 0], X[:, 2]] * Q1p[X[:, 1], X[:, 3]]
    assert w.sum() == pytest.approx(1.0, abs=1e-12)

    zero = np.zeros((B, 5))
    th1 = req.threshold(zero, 0, lambda r: r["path"][:, 0] != 1)
    u_rej1 = zero.copy()
    u_rej1[:, 0] = TOP
    th2 = req.threshold(u_rej1, 1, lambda r: r["path"][:, 0] != 2)
    u_rej12 = u_rej1.copy()
    u_rej12[:, 1] = TOP
    root_draw = req.draw_law(u_rej12, 0, V)
    first = np.zeros((B, V))
    first[np.arange(B), X[:, 0]] += th1
    first[np.arange(B), X[:, 1]] += (1 - th1) * th2
    first += ((1 - th1) * (1 - th2))[:, None] * root_draw
    np.testing.assert_allclose((w[:, None] * first).sum(0), p_root, rtol=0, atol=1e-12)

    # second token after an accepted child, through c1 and through c2
    joint = np.zeros((V, V))
    for via, (u_path, col, d_node) in enumerate([(zero, 2, 3), (u_rej1, 3, 4)]):
        weight = th1 if via == 0 else (1 - th1) * th2
        th_d = req.threshold(u_path, col, lambda r, d=d_node: r["path"][:, 1] != d)
        u_rej = u_path.copy()
        u_rej[:, col] = TOP
        law_d = req.draw_law(u_rej, 1, V)
        second = np.zeros((B, V))
        second[np.arange(B), X[:, 2 + via]] += th_d
        second += (1 - th_d)[:, None] * law_d
        np.add.at(joint, X[:, via], (w * weight)[:, None] * second)
    accepted_first = joint.sum(1)
    assert np.all(accepted_first > 0)
    np.testing.assert_allclose(joint / accepted_first[:, None], P1p, rtol=0, atol=1e-11)


def test_disjoint_supports_reject_all_siblings_and_draw_from_p():
    V, T = 8, 1.0
    zt = np.full((1, 4, V), -1.0e4, np.float32)
    zt[0, 0, :4] = np.log([0.1, 0.2, 0.3, 0.4])
    zd = np.full((1, 4, V), -1.0e4, np.float32)
    zd[0, 0, 4:] = 0.0
    parents = np.array([[-1, 0, 0, 0]], np.int32)
    tokens = np.array([[0, 4, 6, 7]], np.int32)
    req = Batch(zt, zd, parents, tokens, T)
    for col in range(3):
        u = np.zeros((1, 4))
        u[0, :col] = TOP
        th = req.threshold(u, col, lambda r, c=col: r["path"][:, 0] != c + 1)
        assert th[0] == 0.0
    law = req.draw_law(np.full((1, 4), TOP), 0, V)
    np.testing.assert_allclose(law[0], [0.1, 0.2, 0.3, 0.4, 0, 0, 0, 0], atol=1e-7)


def test_equal_distributions_accept_the_first_child():
    rng = np.random.default_rng(7)
    V, n = 8, 4
    z = rng.standard_normal((1, n, V)).astype(np.float32)
    parents = np.array([[-1, 0, 0, 1]], np.int32)
    for _ in range(50):
        x = np.concatenate([[0], rng.integers(0, V, n - 1)]).astype(np.int32)[None]
        r = oracle.tree_accept(z, z.copy(), parents, x, rng.random((1, n)), 0.9)
        assert r["path"][0, 0] == 1 and r["path"][0, 1] == 3 and r["n_accepted"][0] == 2


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_chain_tree_reproduces_chain_acceptance(dtype):
    rng = np.random.default_rng(8)
    B, k, V, T = 300, 4, 40, 0.8
    z = rng.standard_normal((B, k + 1, V)) * 2
    zd = z[:, :k] + rng.standard_normal((B, k, V))
    if dtype == "bf16":
        zt_in, zd_in = bf16_round(z)[0], bf16_round(zd)[0]
        zd_full = np.concatenate([zd_in, zd_in[:, :1]], 1)
    else:
        zt_in, zd_in = z.astype(np.float32), zd.astype(np.float32)
        zd_full = np.concatenate([zd_in, np.full((B, 1, V), np.nan, np.float32)], 1)   # leaf row unread
    x = rng.integers(0, V, (B, k)).astype(np.int32)
    u = rng.random((B, k + 1))
    out, acc, _ = oracle.spec_accept(zt_in, zd_in, x, u, T)
    tok = np.concatenate([np.zeros((B, 1), np.int32), x], 1)
    par = np.tile(np.arange(-1, k, dtype=np.int32), (B, 1))
    r = oracle.tree_accept(zt_in, zd_full, par, tok, u, T)
    assert np.array_equal(r["tokens"], out)
    assert np.array_equal(r["n_accepted"], acc)
    for b in range(B):
        a = acc[b]
        assert list(r["path"][b, :a]) == list(range(1, a + 1)) and np.all(r["path"][b, a:] == -1)


def test_greedy_walk_follows_argmax():
    rng = np.random.default_rng(9)
    B, n, V = 200, 9, 6
    z = rng.standard_normal((B, n, V)).astype(np.float32)
    z[::4, :, 2] = z[::4, :, 4] = 5.0                     # planted ties: lowest id wins
    par = np.stack([random_parents(rng, n) for _ in range(B)])
    g = np.argmax(z, axis=-1)
    tok = rng.integers(0, V, (B, n)).astype(np.int32)
    for b in range(B):                                    # make some children agree with the argmax
        for c in range(1, n):
            if rng.random() < 0.6:
                tok[b, c] = g[b, par[b, c]]
    r = oracle.tree_accept(z, None, par, tok, np.zeros((B, n), np.float32), 0.0)
    for b in range(B):
        a, node = int(r["n_accepted"][b]), 0
        for j in range(a):
            c = int(r["path"][b, j])
            kids = [m for m in range(1, n) if par[b, m] == node and tok[b, m] == g[b, node]]
            assert c == min(kids) and r["tokens"][b, j] == g[b, node]
            node = c
        assert r["tokens"][b, a] == g[b, node]
        assert not any(par[b, m] == node and tok[b, m] == g[b, node] for m in range(1, n))
        assert np.all(r["tokens"][b, a + 1:] == -1) and np.all(r["path"][b, a:] == -1)


def test_monte_carlo_first_token_histogram():
    rng = np.random.default_rng(10)
    V, n, T, N = 8, 4, 1.0, 30000
    zt = rng.standard_normal((n, V)).astype(np.float32)
    zd = (zt + rng.standard_normal((n, V)) * 1.5).astype(np.float32)
    q0 = softmax(zd[0].astype(np.float64) / T)
    tok = np.zeros((N, n), np.int32)
    tok[:, 1:] = rng.choice(V, size=(N, n - 1), p=q0)
    par = np.tile(np.array([-1, 0, 0, 0], np.int32), (N, 1))
    r = oracle.tree_accept(np.repeat(zt[None], N, 0), np.repeat(zd[None], N, 0), par, tok,
                           rng.random((N, n)).astype(np.float32), T)
    p0 = softmax(zt[0].astype(np.float64) / T)
    counts = np.bincount(r["tokens"][:, 0], minlength=V)
    chi2 = float(((counts - N * p0) ** 2 / (N * p0)).sum())
    assert chi2 < 30.0
    # three candidates accept more often than one: 1 - prod of rejection masses
    assert r["n_accepted"].mean() > np.minimum(p0, q0).sum()


# --------------------------------------------------------------- commit
def test_tree_commit_moves_the_accepted_rows_next_to_the_root():
    rng = np.random.default_rng(11)
    B, n, Hkv, D, ps = 3, 7, 2, 8, 4
    lens = [19, 25, 7]
    c = paged_case(rng, B, n, 2, Hkv, D, ps, lens)
    path = np.full((B, n), -1, np.int32)
    path[0, :3] = [2, 4, 6]
    path[1, :2] = [1, 5]
    na = np.array([3, 2, 0], np.int32)
    kp, vp = c["kpool"].copy(), c["vpool"].copy()
    new_len = oracle.kv_commit_tree(kp, vp, c["table"], c["lens"], path, na, n)

    def row(pool, b, pos, h):
        return pool[c["table"][b, pos // ps], h, pos % ps]

    for b in range(B):
        L, a = lens[b], int(na[b])
        assert new_len[b] == L - n + 1 + a
        moved = {L - n + 1 + i: L - n + path[b, i] for i in range(a)}
        for pos in range(L):
            for h in range(Hkv):
                src = moved.get(pos, pos)
                assert np.array_equal(row(kp, b, pos, h), row(c["kpool"], b, src, h))
                assert np.array_equal(row(vp, b, pos, h), row(c["vpool"], b, src, h))
