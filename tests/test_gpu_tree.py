"""GPU parity of token-tree verification against the fp64 oracle (through the
C ABI): tree attention, the multi-candidate acceptance walk and the commit of
the accepted path, plus one tree step chained through all of them.

Attention outputs must lie within |d| <= 2e-3 + 1e-2 |ref|.  Tokens, paths and
accepted counts must equal the oracle's, except near-ties, which are counted:
an accept test with |u - r(x)/q(x)| < 1e-5, or a draw with u within 1e-6 of
either CDF value bracketing the drawn token.  The commit is bit-exact.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_20507_gb300 import binding
from paper_2607_20507_gb300 import workloads as W

pytestmark = pytest.mark.gpu

DEV = "cuda:0"
from parity_bands import DRAW_TIE, NEAR_TIE, check_band_mismatches


def random_parents(rng, B, n, detach=0.0):
    par = np.full((B, n), -1, np.int32)
    for b in range(B):
        for c in range(1, n):
            par[b, c] = rng.integers(0, c)
            if rng.random() < detach:
                par[b, c] = c + rng.integers(0, 3)       # not in [0, c): detached
    return par


def tree_attn_case(B, n, Hq, Hkv, ps, ctx, seed, parents=None):
    w = W.Workload(90 + seed, f"tree-attn-{seed}", batch=B, n_draft=n - 1, vocab=100, logit_dtype="bf16",
                   draft_sigma=1.0, temperatures=(1.0,), n_q_heads=Hq, n_kv_heads=Hkv, head_dim=128,
                   ctx=ctx, page_size=ps)
    inp = W.attention_inputs(w, DEV)
    rng = np.random.default_rng(seed)
    par = random_parents(rng, B, n, detach=0.1) if parents is None else parents
    inp["parents"] = torch.from_numpy(par).to(DEV)
    return inp


def attn_gpu(inp):
    out = binding.cs_tree_verify_attention(inp["q"], inp["k_pages"], inp["v_pages"], inp["page_table"],
                                           inp["ctx_lens"], inp["parents"])
    torch.cuda.synchronize()
    return out


def attn_ref(inp):
    return oracle.tree_attention(W.host_bits(inp["q"]), W.host_bits(inp["k_pages"]), W.host_bits(inp["v_pages"]),
                                 inp["page_table"].cpu().numpy(), inp["ctx_lens"].cpu().numpy(),
                                 inp["parents"].cpu().numpy())


def assert_close(got, ref):
    got = got.float().cpu().numpy()
    bad = np.abs(got - ref) > 2e-3 + 1e-2 * np.abs(ref)
    assert not bad.any(), f"{int(bad.sum())} of {bad.size} outside tolerance, max {np.abs(got - ref).max()}"


@pytest.mark.parametrize("B,n,Hq,Hkv,ps,ctx,seed", [
    (3, 9, 32, 8, 16, ("uniform", 40, 700), 0),        # several tiles, ragged tails
    (2, 34, 32, 8, 16, ("uniform", 300, 1200), 1),     # 136 rows: one row block
    (2, 32, 64, 8, 32, ("uniform", 100, 900), 2),      # 256 rows: two row blocks
    (1, 64, 28, 4, 16, ("const", 2000), 3),            # 448 rows: four row blocks, 64 nodes
    (4, 12, 16, 4, 8, ("uniform", 5, 60), 4),          # contexts shorter than a tile, some L < n
    (3, 16, 32, 8, 16, ("uniform", 20, 700), 5),       # 64 rows: the tcgen05 form
    (2, 30, 16, 4, 32, ("uniform", 40, 900), 6),       # 120 rows: the tcgen05 form, 32-token pages
])
def test_tree_attention_matches_oracle(B, n, Hq, Hkv, ps, ctx, seed):
    inp = tree_attn_case(B, n, Hq, Hkv, ps, ctx, seed)
    assert_close(attn_gpu(inp), attn_ref(inp))


def test_chain_tree_attention_equals_chain_attention_bitwise():
    w = W.WORKLOADS[2]
    inp = W.attention_inputs(w, DEV)
    k = w.n_draft
    chain = binding.cs_verify_attention(inp["q"], inp["k_pages"], inp["v_pages"], inp["page_table"],
                                        inp["ctx_lens"], k)
    par = torch.arange(-1, k, dtype=torch.int32, device=DEV).repeat(w.batch, 1)
    tree = binding.cs_tree_verify_attention(inp["q"], inp["k_pages"], inp["v_pages"], inp["page_table"],
                                            inp["ctx_lens"], par)
    torch.cuda.synchronize()
    assert torch.equal(chain, tree)


def test_tree_attention_bench_workload_sampled():
    w = W.TREE_WORKLOADS[2]
    inp = W.tree_attention_inputs(w, DEV)
    got = attn_gpu(inp)
    for b in (0, w.batch - 1):
        sub = W.attention_subset(dict(inp, n_draft=w.n_nodes - 1), [b])
        ref = oracle.tree_attention(W.host_bits(sub["q"]), W.host_bits(sub["k_pages"]), W.host_bits(sub["v_pages"]),
                                    sub["page_table"].cpu().numpy(), sub["ctx_lens"].cpu().numpy(),
                                    inp["parents"][b:b + 1].cpu().numpy())
        assert_close(got[b:b + 1], ref)


# ---------------------------------------------------------------- acceptance
def accept_gpu(inp, T):
    tok, path, n = binding.cs_tree_accept(inp["target"], inp["draft"] if T > 0 else None, inp["parents"],
                                          inp["node_tokens"], inp["uniforms"], T)
    torch.cuda.synchronize()
    return tok.cpu().numpy(), path.cpu().numpy(), n.cpu().numpy()


def accept_ref(inp, T):
    r = oracle.tree_accept(W.host_bits(inp["target"]), W.host_bits(inp["draft"]) if T > 0 else None,
                           inp["parents"].cpu().numpy(), inp["node_tokens"].cpu().numpy(),
                           inp["uniforms"].cpu().numpy(), T)
    return r, (r["margin"] < NEAR_TIE) | (r["draw_margin"] < DRAW_TIE)


def assert_accept_parity(inp, T, what):
    tok, path, n = accept_gpu(inp, T)
    r, tie = accept_ref(inp, T)
    mism = np.any(tok != r["tokens"], axis=1) | np.any(path != r["path"], axis=1) | (n != r["n_accepted"])
    bad = mism & ~tie
    assert not bad.any(), f"{what}: {int(bad.sum())} requests differ outside the near-tie band"
    check_band_mismatches(int((mism & tie).sum()), len(n), what)
    print(f"{what}: {len(n)} requests, mean accepted {n.mean():.2f}, near-ties {int(tie.sum())}, "
          f"of which differ {int((mism & tie).sum())}")
    nn = tok.shape[1]
    V = inp["target"].shape[2]
    par = inp["parents"].cpu().numpy()
    for b in range(len(n)):
        a = int(n[b])
        assert 0 <= a < nn and 0 <= tok[b, a] < V and (tok[b, a + 1:] == -1).all() and (path[b, a:] == -1).all()
        node = 0
        for j in range(a):                                  # the path descends the tree
            assert par[b, path[b, j]] == node
            node = path[b, j]
    return n


def random_tree_accept(B, n, V, dtype, sigma, T, seed, detach=0.0):
    rng = np.random.default_rng(seed)
    g = torch.Generator(device=DEV).manual_seed(seed)
    dt = torch.float32 if dtype == "f32" else torch.bfloat16
    target = (torch.randn((B, n, V), generator=g, device=DEV) * 3.0).to(dt)
    draft = (target.float() + sigma * torch.randn((B, n, V), generator=g, device=DEV)).to(dt)
    par = random_parents(rng, B, n, detach)
    tokens = np.zeros((B, n), np.int32)
    dz = draft.float().cpu().numpy()
    for b in range(B):
        for c in range(1, n):
            u = par[b, c]
            if 0 <= u < c:
                if T > 0:
                    z = dz[b, u] / T
                    tokens[b, c] = np.argmax(z - np.log(-np.log(rng.random(V).clip(1e-12, 1 - 1e-7))))
                else:
                    tokens[b, c] = np.argmax(dz[b, u]) if rng.random() < 0.7 else rng.integers(0, V)
            else:
                tokens[b, c] = rng.integers(0, V)
    tokens[rng.random((B, n)) < 0.03] = V + 5           # a few invalid ids: never accepted
    return dict(target=target, draft=draft, parents=torch.from_numpy(par).to(DEV),
                node_tokens=torch.from_numpy(tokens).to(DEV),
                uniforms=torch.rand((B, n), generator=g, device=DEV))


@pytest.mark.parametrize("B,n,V,dtype,sigma,T,seed", [
    (64, 9, 32000, "f32", 1.0, 1.0, 0),
    (32, 20, 128256, "bf16", 0.5, 0.7, 1),
    (16, 64, 5000, "bf16", 2.0, 1.3, 2),
    (128, 6, 151936, "bf16", 0.1, 1.0, 3),
    (64, 9, 32000, "f32", 1.0, 0.0, 4),
    (32, 40, 128256, "bf16", 0.5, 0.0, 5),
    (8, 1, 1000, "bf16", 1.0, 0.8, 6),                  # a root alone: the draw of p_root
])
def test_tree_accept_matches_oracle(B, n, V, dtype, sigma, T, seed):
    inp = random_tree_accept(B, n, V, dtype, sigma, T, seed, detach=0.05)
    assert_accept_parity(inp, T, f"random trees B={B} n={n} V={V} T={T}")


@pytest.mark.parametrize("T", [0.0, 0.7])
def test_tree_accept_bench_workload(T):
    inp = W.tree_accept_inputs(W.TREE_WORKLOADS[2], T, DEV)
    n = assert_accept_parity(inp, T, f"{W.TREE_WORKLOADS[2].name} T={T}")
    if T > 0:
        assert n.mean() > 1.0      # three candidates per level accept more than one in most requests


@pytest.mark.parametrize("T", [0.0, 0.9])
def test_chain_tree_accept_equals_chain_accept(T):
    w = W.WORKLOADS[3]
    inp = W.accept_inputs(w, T, DEV)
    B, k, V = w.batch, w.n_draft, w.vocab
    out, na = binding.cs_spec_accept(inp["target"], inp["draft"] if T > 0 else None, inp["draft_tokens"],
                                     inp["uniforms"], T)
    draft = torch.cat([inp["draft"], inp["draft"][:, :1]], 1).contiguous()       # leaf row: not read
    tokens = torch.cat([torch.zeros((B, 1), dtype=torch.int32, device=DEV), inp["draft_tokens"]], 1).contiguous()
    par = torch.arange(-1, k, dtype=torch.int32, device=DEV).repeat(B, 1)
    tok, path, n = binding.cs_tree_accept(inp["target"], draft if T > 0 else None, par, tokens, inp["uniforms"], T)
    torch.cuda.synchronize()
    _, _, margin, dmargin = oracle.spec_accept(W.host_bits(inp["target"]),
                                               W.host_bits(inp["draft"]) if T > 0 else None,
                                               inp["draft_tokens"].cpu().numpy(), inp["uniforms"].cpu().numpy(), T,
                                               with_draw_margin=True)
    tie = (margin < NEAR_TIE) | (dmargin < DRAW_TIE)
    diff = (tok != out).any(1).cpu().numpy() | (n != na).cpu().numpy()
    assert not (diff & ~tie).any()
    a = n.cpu().numpy()
    p = path.cpu().numpy()
    for b in range(B):
        assert list(p[b, :a[b]]) == list(range(1, a[b] + 1))


# -------------------------------------------------------------------- commit
def test_kv_commit_tree_matches_oracle_bitwise():
    B, n = 6, 20
    inp = tree_attn_case(B, n, 32, 8, 16, ("uniform", 10, 400), 7)
    rng = np.random.default_rng(7)
    par = inp["parents"].cpu().numpy()
    path = np.full((B, n), -1, np.int32)
    na = np.zeros(B, np.int32)
    for b in range(B):                     # a random root-to-node path of each tree
        node, j = 0, 0
        while True:
            kids = [c for c in range(1, n) if par[b, c] == node]
            if not kids or rng.random() < 0.2:
                break
            node = int(rng.choice(kids))
            path[b, j] = node
            j += 1
        na[b] = j
    kp, vp = W.host_bits(inp["k_pages"]).copy(), W.host_bits(inp["v_pages"]).copy()
    exp_len = oracle.kv_commit_tree(kp, vp, inp["page_table"].cpu().numpy(), inp["ctx_lens"].cpu().numpy(), path,
                                    na, n)
    lens = inp["ctx_lens"].clone()
    binding.cs_kv_commit_tree(inp["k_pages"], inp["v_pages"], inp["page_table"], lens,
                              torch.from_numpy(path).to(DEV), torch.from_numpy(na).to(DEV))
    torch.cuda.synchronize()
    assert np.array_equal(lens.cpu().numpy(), exp_len)
    assert np.array_equal(W.host_bits(inp["k_pages"]), kp)
    assert np.array_equal(W.host_bits(inp["v_pages"]), vp)


def test_one_tree_step_through_the_c_abi():
    """append the n tree rows -> tree attention -> tree acceptance -> commit, each
    checked against the oracle run on the same data."""
    B, n, Hq, Hkv, V, T = 4, 14, 32, 8, 20000, 0.8
    inp = tree_attn_case(B, n, Hq, Hkv, 16, ("uniform", 200, 900), 8,
                         parents=np.tile(np.array(W.tree_parents((3, 2, 1))[:n], np.int32), (4, 1)))
    g = torch.Generator(device=DEV).manual_seed(8)
    new_k = torch.randn((B, n, Hkv, 128), generator=g, device=DEV).to(torch.bfloat16)
    new_v = torch.randn((B, n, Hkv, 128), generator=g, device=DEV).to(torch.bfloat16)
    kp, vp = W.host_bits(inp["k_pages"]).copy(), W.host_bits(inp["v_pages"]).copy()
    binding.cs_kv_append(new_k, new_v, inp["k_pages"], inp["v_pages"], inp["page_table"], inp["ctx_lens"])
    oracle.kv_append(W.host_bits(new_k), W.host_bits(new_v), kp, vp, inp["page_table"].cpu().numpy(),
                     inp["ctx_lens"].cpu().numpy())
    torch.cuda.synchronize()
    assert np.array_equal(W.host_bits(inp["k_pages"]), kp)
    assert_close(attn_gpu(inp), attn_ref(inp))
    acc = random_tree_accept(B, n, V, "bf16", 0.5, T, 8)
    acc["parents"] = inp["parents"]
    tok, path, na = accept_gpu(acc, T)
    r, tie = accept_ref(acc, T)
    assert not ((np.any(tok != r["tokens"], 1) | (na != r["n_accepted"])) & ~tie).any()
    lens = inp["ctx_lens"].clone()
    binding.cs_kv_commit_tree(inp["k_pages"], inp["v_pages"], inp["page_table"], lens,
                              torch.from_numpy(path).to(DEV), torch.from_numpy(na).to(DEV))
    exp_len = oracle.kv_commit_tree(kp, vp, inp["page_table"].cpu().numpy(), inp["ctx_lens"].cpu().numpy(), path,
                                    na, n)
    torch.cuda.synchronize()
    assert np.array_equal(lens.cpu().numpy(), exp_len)
    assert np.array_equal(W.host_bits(inp["k_pages"]), kp) and np.array_equal(W.host_bits(inp["v_pages"]), vp)
