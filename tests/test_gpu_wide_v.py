"""Verify attention with V entries of any finite bf16 magnitude, against the
fp64 oracle.

Every kernel form takes P.V on bf16 tensor cores with V as stored and P as
two bf16 terms (hi + lo), formed as P * 2^-64 (the row sum carries the same
factor): no partial sum can overflow fp32 for any finite bf16 V, and split
partials are stored normalised, so the merge cannot overflow either.  These
tests plant entries far beyond fp16's range (up to ~3.3e38, near bf16's
largest) in the middle of contexts, in draft rows (seen by later rows only)
and in spans that are cut across CTAs (split partials and the merge), for
each kernel form and for tree attention.  Outputs are compared element by
element with |gpu - oracle| <= 2e-3 + 1e-2 |oracle|.
"""
import dataclasses

import numpy as np
import pytest
import torch

import oracle
from paper_2607_20507_gb300 import binding
from paper_2607_20507_gb300 import workloads as W

pytestmark = pytest.mark.gpu

DEV = "cuda:0"
ATOL, RTOL = 2e-3, 1e-2


def plant(inp, rng, values):
    """Writes `values` into V at random visible keys of every (request, KV head):
    at most one planted entry per (request, head, dim), so that no output
    element sums two huge terms of opposite sign."""
    vp = inp["v_pages"]
    ps, Hkv, D = vp.shape[2], vp.shape[1], vp.shape[3]
    table = inp["page_table"].cpu().numpy()
    lens = inp["ctx_lens"].cpu().numpy()
    rows = inp["q"].shape[1]
    planted = 0
    for b, L in enumerate(lens.tolist()):
        if L < rows + 2:
            continue
        for h in range(Hkv):
            dims = rng.choice(D, len(values), replace=False)
            for val, d in zip(values, dims):
                # a key in the prefix's middle, or one of the draft rows
                key = int(rng.integers(L // 3, L)) if rng.random() < 0.8 else L - int(rng.integers(1, rows))
                page = int(table[b, key // ps])
                vp[page, h, key % ps, int(d)] = torch.tensor(val, dtype=torch.bfloat16)
                planted += 1
    return planted


def check(got, expect, what):
    got = got.float().cpu().numpy().astype(np.float64)
    assert np.isfinite(got).all(), f"{what}: non-finite output"
    err = np.abs(got - expect)
    tol = ATOL + RTOL * np.abs(expect)
    bad = err > tol
    assert not bad.any(), (f"{what}: {int(bad.sum())} of {bad.size} elements outside tolerance; "
                           f"worst excess {float((err - tol).max()):.3e}")


VALUES = [1.0e5, -2.5e5, 65536.0, -3.0e38, 3.3e38, 65280.0, -7.0e4]


def small(B, k, Hq, Hkv, ps, lo, hi, cell):
    return W.Workload(96, "wide-v", batch=B, n_draft=k, vocab=64, logit_dtype="bf16", draft_sigma=1.0,
                      temperatures=(1.0,), n_q_heads=Hq, n_kv_heads=Hkv, head_dim=128, ctx=("uniform", lo, hi),
                      page_size=ps, cell=cell)


@pytest.mark.parametrize("k,Hq,Hkv,ps,form", [
    (5, 32, 8, 16, "key-split mma.sync (24 rows)"),
    (1, 32, 8, 16, "key-split mma.sync (8 rows)"),
    (4, 28, 4, 16, "tcgen05 (35 rows)"),
    (4, 28, 4, 8, "mma.sync without key split (35 rows, 8-token pages)"),
    (8, 64, 8, 32, "tcgen05 (72 rows)"),
    (15, 64, 8, 16, "tcgen05 (128 rows)"),
    (16, 64, 8, 16, "mma.sync row blocks (136 rows)"),
])
def test_wide_v_matches_oracle(k, Hq, Hkv, ps, form):
    rng = np.random.default_rng(k * 100 + Hq)
    # few requests with long contexts: every span is cut over several CTAs
    inp = W.attention_inputs(small(3, k, Hq, Hkv, ps, 600, 3000, cell=k * 10 + ps), DEV)
    assert plant(inp, rng, VALUES) > 0
    out = binding.cs_verify_attention(inp["q"], inp["k_pages"], inp["v_pages"], inp["page_table"],
                                      inp["ctx_lens"], k)
    torch.cuda.synchronize()
    expect = oracle.verify_attention(W.host_bits(inp["q"]), W.host_bits(inp["k_pages"]), W.host_bits(inp["v_pages"]),
                                     inp["page_table"].cpu().numpy(), inp["ctx_lens"].cpu().numpy(), k)
    assert np.abs(expect).max() > 1e30          # the planted entries reach the output
    check(out, expect, form)


def test_wide_v_many_short_spans_and_status():
    """Many requests (uncut spans written whole, cut ones merged), the
    workspace's status word clean afterwards, and the same call twice."""
    rng = np.random.default_rng(7)
    inp = W.attention_inputs(small(48, 4, 32, 8, 16, 40, 700, cell=5), DEV)
    plant(inp, rng, VALUES[:4])
    d = binding.attn_dims(inp["q"], inp["k_pages"], inp["page_table"])
    ws = torch.zeros(binding.load_library().cs_verify_attention_workspace_bytes(d, 4), dtype=torch.uint8,
                     device=DEV)
    expect = oracle.verify_attention(W.host_bits(inp["q"]), W.host_bits(inp["k_pages"]), W.host_bits(inp["v_pages"]),
                                     inp["page_table"].cpu().numpy(), inp["ctx_lens"].cpu().numpy(), 4)
    for call in range(2):
        out = binding.cs_verify_attention(inp["q"], inp["k_pages"], inp["v_pages"], inp["page_table"],
                                          inp["ctx_lens"], 4, workspace=ws)
        torch.cuda.synchronize()
        check(out, expect, f"call {call}")
    assert binding.cs_read_device_status(ws) == 0


def test_wide_v_tree_attention():
    tw = dataclasses.replace(W.TREE_WORKLOADS[2], batch=3)
    inp = W.tree_attention_inputs(tw, DEV)
    rng = np.random.default_rng(11)
    plant(inp, rng, VALUES)
    out = binding.cs_tree_verify_attention(inp["q"], inp["k_pages"], inp["v_pages"], inp["page_table"],
                                           inp["ctx_lens"], inp["parents"])
    torch.cuda.synchronize()
    expect = oracle.tree_attention(W.host_bits(inp["q"]), W.host_bits(inp["k_pages"]), W.host_bits(inp["v_pages"]),
                                   inp["page_table"].cpu().numpy(), inp["ctx_lens"].cpu().numpy(),
                                   inp["parents"].cpu().numpy())
    check(out, expect, "tree")


def test_values_at_the_edge_of_fp16():
    """65280 (the largest bf16 value fp16 holds) and its negative: the edge
    where an fp16 P.V product would begin to overflow."""
    inp = W.attention_inputs(small(2, 5, 32, 8, 16, 300, 900, cell=9), DEV)
    rng = np.random.default_rng(3)
    plant(inp, rng, [65280.0, -65280.0])
    out = binding.cs_verify_attention(inp["q"], inp["k_pages"], inp["v_pages"], inp["page_table"],
                                      inp["ctx_lens"], 5)
    torch.cuda.synchronize()
    expect = oracle.verify_attention(W.host_bits(inp["q"]), W.host_bits(inp["k_pages"]), W.host_bits(inp["v_pages"]),
                                     inp["page_table"].cpu().numpy(), inp["ctx_lens"].cpu().numpy(), 5)
    check(out, expect, "65280")
