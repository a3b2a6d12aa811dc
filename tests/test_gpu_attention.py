"""GPU parity of cs_verify_attention against the fp64 oracle (through the C ABI).

Tolerance (stated for the attention output): |gpu - oracle| <= 2e-3 + 1e-2 * |oracle|
element by element.  Sizes span several 64-key tiles, ragged tails, every
supported page size, the serving workloads (all requests where the oracle
finishes in seconds, seeded request samples at the largest sizes) and the
degenerate cases the method has.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_20507_gb300 import binding
from paper_2607_20507_gb300 import workloads as W

pytestmark = pytest.mark.gpu

ATOL, RTOL = 2e-3, 1e-2
DEV = "cuda:0"


def gpu(inp, sm_scale=0.0, workspace=None):
    out = binding.cs_verify_attention(inp["q"], inp["k_pages"], inp["v_pages"], inp["page_table"],
                                      inp["ctx_lens"], inp["n_draft"], sm_scale=sm_scale,
                                      workspace=workspace)
    torch.cuda.synchronize()
    return out


def ref(inp, sm_scale=0.0):
    return oracle.verify_attention(W.host_bits(inp["q"]), W.host_bits(inp["k_pages"]),
                                   W.host_bits(inp["v_pages"]), inp["page_table"].cpu().numpy(),
                                   inp["ctx_lens"].cpu().numpy(), inp["n_draft"], sm_scale)


def assert_parity(out, expect, what=""):
    got = out.float().cpu().numpy().astype(np.float64)
    err = np.abs(got - expect)
    tol = ATOL + RTOL * np.abs(expect)
    bad = err > tol
    assert np.isfinite(got).all(), f"{what}: non-finite output"
    assert not bad.any(), (f"{what}: {int(bad.sum())} of {bad.size} elements outside "
                           f"2e-3 + 1e-2|ref|; worst excess {float((err - tol).max()):.3e}")


def small(B=3, k=3, Hq=8, Hkv=2, ps=16, lo=70, hi=300, wid=90, cell=0, contiguous=False):
    return W.Workload(wid, "small", batch=B, n_draft=k, vocab=64, logit_dtype="bf16",
                      draft_sigma=1.0, temperatures=(1.0,), n_q_heads=Hq, n_kv_heads=Hkv,
                      head_dim=128, ctx=("uniform", lo, hi), page_size=ps, contiguous=contiguous,
                      cell=cell)


@pytest.mark.parametrize("ps", [8, 16, 32, 64, 128, 256])
def test_small_all_page_sizes(ps):
    inp = W.attention_inputs(small(ps=ps, cell=ps), DEV)
    assert_parity(gpu(inp), ref(inp), f"ps={ps}")


@pytest.mark.parametrize("k,Hq,Hkv", [(1, 4, 4), (2, 28, 4), (4, 32, 8), (8, 64, 8), (16, 64, 8),
                                       (16, 32, 8), (5, 12, 12)])
def test_row_packing_shapes(k, Hq, Hkv):
    inp = W.attention_inputs(small(B=2, k=k, Hq=Hq, Hkv=Hkv, lo=k + 1, hi=700, cell=k * 100 + Hq), DEV)
    assert_parity(gpu(inp), ref(inp), f"k={k} G={Hq // Hkv}")


@pytest.mark.parametrize("wid", [1, 2, 3])
def test_serving_workloads_all_requests(wid):
    inp = W.attention_inputs(W.WORKLOADS[wid], DEV)
    assert_parity(gpu(inp), ref(inp), W.WORKLOADS[wid].name)


def test_workload_4_sampled_requests():
    # B=256, contexts 2K-16K: the launch runs at full size, the oracle checks a
    # seeded sample of requests one by one
    w = W.WORKLOADS[4]
    inp = W.attention_inputs(w, DEV)
    out = gpu(inp)
    idx = sorted(np.random.default_rng(4).choice(w.batch, 24, replace=False).tolist())
    sub = W.attention_subset(inp, idx)
    assert_parity(out[idx], ref(sub), "workload 4 sample")


@pytest.mark.parametrize("k,B", [(k, B) for k in W.SWEEP_KS for B in W.SWEEP_BATCHES])
def test_sweep_attention_cells_sampled(k, B):
    """Every attention cell of the sweep (context 4096): the launch at full
    size, the oracle on a seeded sample of up to 3 requests."""
    w = next(c for c in W.sweep_attention_cells() if c.n_draft == k and c.batch == B)
    inp = W.attention_inputs(w, DEV)
    out = gpu(inp)
    n = min(3, B)
    idx = sorted(np.random.default_rng(k * 1000 + B).choice(B, n, replace=False).tolist())
    assert_parity(out[idx], ref(W.attention_subset(inp, idx)), w.name)


def test_min_and_degenerate_context_lengths():
    w = small(B=6, k=4, lo=5, hi=5, cell=7)
    inp = W.attention_inputs(w, DEV)
    # L = k+1 (row 0 sees one key), L < k+1 (rows without keys are zero), L = 0
    inp["ctx_lens"] = torch.tensor([5, 3, 1, 0, 5, 2], dtype=torch.int32, device=DEV)
    out = gpu(inp)
    expect = ref(inp)
    assert_parity(out, expect, "degenerate lengths")
    assert float(out[3].abs().max()) == 0.0


def test_context_longer_than_the_page_table_is_clamped():
    inp = W.attention_inputs(small(B=2, k=2, lo=40, hi=40, cell=8), DEV)
    cap = inp["page_table"].shape[1] * 16
    base = gpu(inp).clone()
    inp["ctx_lens"] = torch.tensor([cap + 100, 40], dtype=torch.int32, device=DEV)
    inp["page_table"][0, :] = inp["page_table"][0, 0]
    clamped = inp["ctx_lens"].clone()
    clamped[0] = cap
    got = gpu(inp)
    inp2 = dict(inp, ctx_lens=clamped)
    assert torch.equal(got, gpu(inp2))
    assert_parity(got, ref(inp2))
    assert torch.equal(got[1], base[1])


def test_out_of_range_page_ids_read_zeros():
    inp = W.attention_inputs(small(B=2, k=2, lo=100, hi=160, cell=9), DEV)
    P = inp["k_pages"].shape[0]
    inp["page_table"][0, 1] = P + 3
    inp["page_table"][1, 2] = -5
    assert_parity(gpu(inp), ref(inp), "bad page ids")


def test_garbage_past_the_context_never_reaches_the_output():
    # pool slots past L_b and unused pages hold NaN bit patterns
    w = small(B=3, k=3, lo=50, hi=200, cell=10)
    inp = W.attention_inputs(w, DEV)
    clean = gpu(inp).clone()
    kp, vp = inp["k_pages"], inp["v_pages"]
    nan = torch.tensor(float("nan"), dtype=torch.bfloat16, device=DEV)
    table = inp["page_table"].cpu()
    for b, L in enumerate(inp["ctx_lens"].cpu().tolist()):
        last = table[b, (L - 1) // 16].item()
        kp[last, :, (L - 1) % 16 + 1:] = nan
        vp[last, :, (L - 1) % 16 + 1:] = nan
    got = gpu(inp)
    assert torch.isfinite(got.float()).all()
    assert torch.equal(got, clean)


def test_page_permutation_is_bit_identical():
    inp = W.attention_inputs(small(B=4, k=3, lo=100, hi=500, cell=11), DEV)
    base = gpu(inp).clone()
    P = inp["k_pages"].shape[0]
    perm = torch.randperm(P, generator=torch.Generator().manual_seed(5))
    kp = torch.empty_like(inp["k_pages"])
    vp = torch.empty_like(inp["v_pages"])
    kp[perm.to(DEV)] = inp["k_pages"]
    vp[perm.to(DEV)] = inp["v_pages"]
    t = inp["page_table"].cpu()
    t = torch.where(t >= 0, perm[t.clamp(min=0).long()].to(torch.int32), t)
    got = gpu(dict(inp, k_pages=kp, v_pages=vp, page_table=t.to(DEV)))
    assert torch.equal(got, base)


def test_contiguous_and_paged_layouts_agree_bitwise():
    a = W.attention_inputs(small(B=2, k=2, lo=300, hi=300, cell=12, contiguous=True), DEV)
    b = W.attention_inputs(small(B=2, k=2, lo=300, hi=300, cell=12, contiguous=False), DEV)
    # same pages, scattered: rebuild b's pool from a's contiguous pool
    order = b["page_table"].cpu()
    kp = torch.empty_like(a["k_pages"])
    vp = torch.empty_like(a["v_pages"])
    src = a["page_table"].cpu()
    for r in range(2):
        n = (300 + 15) // 16
        kp[order[r, :n].long().to(DEV)] = a["k_pages"][src[r, :n].long().to(DEV)]
        vp[order[r, :n].long().to(DEV)] = a["v_pages"][src[r, :n].long().to(DEV)]
    got = gpu(dict(a, k_pages=kp, v_pages=vp, page_table=b["page_table"]))
    assert torch.equal(got, gpu(a))


def test_split_count_invariance_within_tolerance():
    # the same request alone and inside a large batch gets different split sizes
    big = W.attention_inputs(small(B=64, k=4, Hq=32, Hkv=8, lo=3000, hi=4096, cell=13), DEV)
    full = gpu(big)
    one = W.attention_subset(big, [17])
    alone = gpu(one)
    a, b = alone.float(), full[17:18].float()
    assert torch.allclose(a, b, atol=ATOL, rtol=RTOL)
    assert_parity(alone, ref(one))


def test_custom_scale():
    inp = W.attention_inputs(small(B=2, k=3, cell=14), DEV)
    assert_parity(gpu(inp, sm_scale=0.05), ref(inp, 0.05), "sm_scale")


def test_deterministic_and_status_clean():
    inp = W.attention_inputs(W.WORKLOADS[2], DEV)
    d = binding.attn_dims(inp["q"], inp["k_pages"], inp["page_table"])
    ws = torch.zeros(binding.load_library().cs_verify_attention_workspace_bytes(d, inp["n_draft"]),
                     dtype=torch.uint8, device=DEV)
    a = gpu(inp, workspace=ws).clone()
    b = gpu(inp, workspace=ws)
    assert torch.equal(a, b)
    assert binding.cs_read_device_status(ws) == 0


def test_empty_batch():
    inp = W.attention_inputs(small(B=1, k=2, cell=15), DEV)
    e = {k: (v[:0] if k in ("q", "page_table", "ctx_lens") else v) for k, v in inp.items()}
    out = gpu(e)
    assert out.shape[0] == 0


# ---- the tcgen05 form (33..128 query rows per KV head, pages of 16+ tokens)
@pytest.mark.parametrize("k,Hq,Hkv,ps", [(8, 64, 8, 16), (8, 64, 8, 32), (8, 64, 8, 64), (8, 64, 8, 128),
                                         (8, 64, 8, 256), (6, 28, 4, 16), (15, 64, 8, 32), (16, 32, 8, 16),
                                         (10, 24, 8, 16), (4, 28, 4, 16), (7, 48, 8, 32)])
def test_tcgen05_row_counts_and_page_sizes(k, Hq, Hkv, ps):
    """Boundary row counts (33, 128), the 33-48 band (33, 35, 48 rows), and
    every page size the form takes."""
    inp = W.attention_inputs(small(B=3, k=k, Hq=Hq, Hkv=Hkv, ps=ps, lo=k + 1, hi=900, cell=7000 + k * 10 + ps), DEV)
    assert_parity(gpu(inp), ref(inp), f"tc k={k} G={Hq // Hkv} ps={ps}")


@pytest.mark.parametrize("k,Hq,Hkv", [(4, 28, 4), (10, 24, 8), (7, 48, 8)])
def test_mma_sync_33_to_48_rows_on_8_token_pages(k, Hq, Hkv):
    """33-48 query rows on pages of 8 tokens take the mma.sync form without
    the key split (the tcgen05 form needs pages of 16+ tokens)."""
    inp = W.attention_inputs(small(B=3, k=k, Hq=Hq, Hkv=Hkv, ps=8, lo=k + 1, hi=800, cell=7300 + k * 10 + Hq), DEV)
    assert_parity(gpu(inp), ref(inp), f"mma.sync k={k} G={Hq // Hkv} ps=8")


def test_tcgen05_span_pieces_and_repeat_calls():
    """Many short spans (every CTA crosses spans and cut pieces) and the same
    workspace used for consecutive calls."""
    inp = W.attention_inputs(small(B=40, k=8, Hq=64, Hkv=8, ps=16, lo=9, hi=400, cell=7100), DEV)
    expect = ref(inp)
    for _ in range(3):
        assert_parity(gpu(inp), expect, "tc many spans")


def test_tcgen05_unaligned_query_falls_back():
    """A query base that is 4- but not 16-byte aligned cannot feed TMA: the call
    runs the other form on the same workspace and still matches."""
    inp = W.attention_inputs(small(B=2, k=8, Hq=64, Hkv=8, ps=16, lo=100, hi=600, cell=7200), DEV)
    q = inp["q"]
    buf = torch.empty(q.numel() + 2, dtype=torch.bfloat16, device=DEV)
    q2 = buf[2:].view(q.shape)
    q2.copy_(q)
    assert q2.data_ptr() % 16 != 0 and q2.data_ptr() % 4 == 0
    out = binding.cs_verify_attention(q2, inp["k_pages"], inp["v_pages"], inp["page_table"], inp["ctx_lens"],
                                      inp["n_draft"])
    torch.cuda.synchronize()
    assert_parity(out, ref(inp), "tc fallback")


@pytest.mark.parametrize("k,Hq,Hkv", [(2, 8, 2), (4, 16, 2)])
def test_batch_beyond_one_launch(k, Hq, Hkv):
    # more requests than one launch schedules (1024): the call runs two main
    # kernels (and merges) over the same workspace, the second on requests
    # 1024.. -- both attention forms (12 and 40 query rows per KV head)
    inp = W.attention_inputs(small(B=1030, k=k, Hq=Hq, Hkv=Hkv, lo=k + 1, hi=160, cell=7000 + k), DEV)
    assert_parity(gpu(inp), ref(inp), f"B=1030 k={k} G={Hq // Hkv}")
