"""GPU parity of cs_kv_append / cs_kv_commit against the oracle (byte-exact),
and one whole draft-and-verify step chained through the C ABI:
append -> verify attention (which must see the appended rows) -> acceptance
-> commit, against the same chain in the oracle."""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_20507_gb300 import binding
from paper_2607_20507_gb300 import workloads as W

pytestmark = pytest.mark.gpu

DEV = "cuda:0"


def bits(t):
    return W.host_bits(t)


def setup(B, n, H, ps, max_pages, seed, P=None, short=False):
    g = torch.Generator().manual_seed(seed)
    P = P or B * max_pages
    kp = torch.randn(P, H, ps, 128, generator=g).bfloat16()
    vp = torch.randn(P, H, ps, 128, generator=g).bfloat16()
    pt = torch.randperm(P, generator=g)[:B * max_pages].reshape(B, max_pages).to(torch.int32)
    lo = 0 if short else n
    L = torch.randint(lo, max_pages * ps + 1, (B,), generator=g).to(torch.int32)
    nk = torch.randn(B, n, H, 128, generator=g).bfloat16()
    nv = torch.randn(B, n, H, 128, generator=g).bfloat16()
    return kp, vp, pt, L, nk, nv


def run_both(kp, vp, pt, L, nk, nv):
    gk, gv = kp.to(DEV), vp.to(DEV)
    binding.cs_kv_append(nk.to(DEV), nv.to(DEV), gk, gv, pt.to(DEV), L.to(DEV))
    torch.cuda.synchronize()
    ok, ov = bits(kp).copy(), bits(vp).copy()
    oracle.kv_append(bits(nk), bits(nv), ok, ov, pt.numpy(), L.numpy())
    np.testing.assert_array_equal(bits(gk.cpu()), ok)
    np.testing.assert_array_equal(bits(gv.cpu()), ov)


@pytest.mark.parametrize("B,n,H,ps,max_pages", [(3, 5, 2, 16, 6), (8, 6, 8, 16, 256), (64, 5, 4, 16, 24),
                                               (16, 9, 8, 32, 20), (2, 17, 8, 8, 40), (5, 1, 1, 64, 4),
                                               (4, 6, 8, 128, 3), (3, 4, 2, 256, 2), (256, 9, 8, 32, 4)])
def test_append_parity(B, n, H, ps, max_pages):
    run_both(*setup(B, n, H, ps, max_pages, seed=B * 31 + n * 7 + ps))


def test_append_short_contexts_and_bad_pages():
    kp, vp, pt, L, nk, nv = setup(12, 6, 2, 16, 5, seed=3, short=True)
    L[:4] = torch.tensor([0, 2, 5, -3], dtype=torch.int32)
    L[4] = 10 ** 6                       # clamped to max_pages * ps
    pt[5] = torch.tensor([-1, 1 << 30, 70, -7, 60], dtype=torch.int32)   # pool has 60 pages
    run_both(kp, vp, pt, L, nk, nv)


def test_commit_parity():
    g = torch.Generator().manual_seed(4)
    for k in (1, 5, 16):
        L = torch.randint(0, 5000, (1000,), generator=g).to(torch.int32)
        a = torch.randint(0, k + 1, (1000,), generator=g).to(torch.int32)
        gl = L.to(DEV)
        binding.cs_kv_commit(gl, a.to(DEV), k)
        np.testing.assert_array_equal(gl.cpu().numpy(), oracle.kv_commit(L.numpy(), a.numpy(), k))


def test_one_step_chained_through_the_c_abi():
    # workload-2 geometry, 8 requests: the verify rows are appended, then
    # attention reads them, the acceptance decides, and commit keeps the prefix
    w = W.WORKLOADS[2]
    inp = W.attention_inputs(w, DEV)
    B, R, Hq, D = inp["q"].shape
    Hkv, k = w.n_kv_heads, w.n_draft
    g = torch.Generator().manual_seed(5)
    nk = torch.randn(B, R, Hkv, D, generator=g).bfloat16().to(DEV)
    nv = torch.randn(B, R, Hkv, D, generator=g).bfloat16().to(DEV)
    kp0, vp0 = bits(inp["k_pages"].cpu()).copy(), bits(inp["v_pages"].cpu()).copy()
    binding.cs_kv_append(nk, nv, inp["k_pages"], inp["v_pages"], inp["page_table"], inp["ctx_lens"])
    out = binding.cs_verify_attention(inp["q"], inp["k_pages"], inp["v_pages"], inp["page_table"],
                                      inp["ctx_lens"], k)
    acc = W.accept_inputs(w, 0.7, DEV)
    tokens, n_acc = binding.cs_spec_accept(acc["target"], acc["draft"], acc["draft_tokens"], acc["uniforms"], 0.7)
    lens = inp["ctx_lens"].clone()
    binding.cs_kv_commit(lens, n_acc, k)
    torch.cuda.synchronize()
    # the oracle chain on the same inputs
    oracle.kv_append(bits(nk.cpu()), bits(nv.cpu()), kp0, vp0, inp["page_table"].cpu().numpy(),
                     inp["ctx_lens"].cpu().numpy())
    np.testing.assert_array_equal(bits(inp["k_pages"].cpu()), kp0)
    expect = oracle.verify_attention(bits(inp["q"].cpu()), kp0, vp0, inp["page_table"].cpu().numpy(),
                                     inp["ctx_lens"].cpu().numpy(), k)
    got = out.float().cpu().numpy().astype(np.float64)
    assert (np.abs(got - expect) <= 2e-3 + 1e-2 * np.abs(expect)).all()
    eo, en, am, dm = oracle.spec_accept(bits(acc["target"].cpu()), bits(acc["draft"].cpu()),
                                        acc["draft_tokens"].cpu().numpy(), acc["uniforms"].cpu().numpy(), 0.7,
                                        with_draw_margin=True)
    n_gpu = n_acc.cpu().numpy()
    tie = am < 1e-5                              # accept tests within the near-tie band
    assert (n_gpu[~tie] == en[~tie]).all()
    np.testing.assert_array_equal(lens.cpu().numpy(), oracle.kv_commit(inp["ctx_lens"].cpu().numpy(), n_gpu, k))
