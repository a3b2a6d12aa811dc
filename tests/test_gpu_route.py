"""GPU parity of cs_route / cs_route_norms against the fp64 routing oracle.

Tolerance (derived from the arithmetic): the kernel forms each dot product of
bf16 inputs with fp32 accumulation over d <= 384 terms, so its error is at
most about d * 2^-23 * |e| |c| (<= 4.6e-5 after normalisation, allowing a
truncating adder); each norm is an fp32 sum of d squares followed by rsqrtf
(relative error <= 2.4e-5 together).  Scores therefore agree within 1e-4.
Arg maxes are compared where the oracle's best-vs-second margin exceeds
2e-4, hit/miss decisions where |S - tau| exceeds 1e-4; inside those bands
the GPU's pick must still be a near-best group."""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_20507_gb300 import binding
from paper_2607_20507_gb300 import workloads as W

pytestmark = pytest.mark.gpu

DEV = "cuda:0"
TOL = 1e-4


def run_gpu(emb, cent, tau):
    e, c = emb.to(DEV), cent.to(DEV)
    inv = binding.cs_route_norms(c)
    g, b, s = binding.cs_route(e, c, inv, tau)
    torch.cuda.synchronize()
    return g.cpu().numpy(), b.cpu().numpy(), s.cpu().numpy()


def check(emb, cent, tau, rows=None):
    g, b, s = run_gpu(emb, cent, tau)
    e_bits, c_bits = W.host_bits(emb), W.host_bits(cent)
    if rows is not None:
        e_bits, g, b, s = e_bits[rows], g[rows], b[rows], s[rows]
    r = oracle.route(e_bits, c_bits, tau)
    N = cent.shape[0]
    if N == 0:
        np.testing.assert_array_equal(b, -1)
        np.testing.assert_array_equal(g, -1)
        assert np.all(np.isneginf(s))
        return r
    np.testing.assert_allclose(s, r["score"], rtol=0, atol=TOL)
    clear = r["margin"] > 2 * TOL
    np.testing.assert_array_equal(b[clear], r["best"][clear])
    # inside the band the GPU's group is still within the band of the best score
    assert np.all((b >= 0) & (b < N))
    if (~clear).any():
        cf = torch.from_numpy(c_bits.view(np.int16)).view(torch.bfloat16).double()
        ef = torch.from_numpy(e_bits.view(np.int16)).view(torch.bfloat16).double()
        idx = np.nonzero(~clear)[0]
        cs = torch.nn.functional.cosine_similarity(ef[idx], cf[torch.from_numpy(b[idx]).long()], dim=1).numpy()
        assert np.all(cs >= r["score"][idx] - 2 * TOL)
    sure = r["tau_margin"] > TOL
    np.testing.assert_array_equal(g[sure] >= 0, r["group"][sure] >= 0)
    hit = sure & clear & (r["group"] >= 0)
    np.testing.assert_array_equal(g[hit], r["group"][hit])
    assert np.all((g == -1) | (g == b))
    return r


@pytest.mark.parametrize("wid", [1, 2])
def test_workload_parity(wid):
    x = W.route_inputs(W.ROUTE_WORKLOADS[wid])
    r = check(x["emb"], x["centroids"], W.ROUTE_TAU)
    assert 0 < (r["group"] >= 0).sum() < len(r["group"])


def test_largest_workload_sampled_rows():
    w = W.ROUTE_WORKLOADS[3]
    x = W.route_inputs(w)
    rows = np.random.default_rng(5).choice(w.batch, 48, replace=False)
    rows = np.unique(np.concatenate([rows, [0, 127, 128, w.batch - 1]]))
    check(x["emb"], x["centroids"], W.ROUTE_TAU, rows)


@pytest.mark.parametrize("B,N,d", [(1, 1, 64), (1, 5, 384), (130, 1000, 384), (257, 129, 128),
                                   (64, 4096, 320), (300, 300, 192), (1000, 7, 64), (128, 128, 256)])
def test_ragged_shapes(B, N, d):
    x = W.route_inputs(W.RouteWorkload(0, "t", B, N, d), seed=B * 7919 + N * 31 + d)
    check(x["emb"], x["centroids"], 0.85)


def test_no_groups():
    x = W.route_inputs(W.RouteWorkload(0, "t", 20, 0, 128), seed=3)
    check(x["emb"], x["centroids"], 0.85)


def test_empty_batch():
    c = torch.randn(10, 64).bfloat16().to(DEV)
    e = torch.empty(0, 64, dtype=torch.bfloat16, device=DEV)
    g, b, s = binding.cs_route(e, c, binding.cs_route_norms(c), 0.85)
    assert g.numel() == b.numel() == s.numel() == 0


def test_planted_ties_and_zero_vectors():
    g_ = torch.Generator().manual_seed(17)
    N, d = 700, 384
    cent = torch.randn(N, d, generator=g_).bfloat16()
    cent[650] = cent[10]          # same centroid in another tile and split
    cent[200] = cent[199] * 2     # a scaled duplicate: same cosine after normalisation
    cent[300] = 0                 # a zero centroid scores 0
    emb = torch.randn(6, d, generator=g_).bfloat16()
    emb[0] = cent[650]
    emb[1] = 0                    # zero request: every score 0, lowest id wins
    emb[2] = cent[200]
    emb[3] = -cent[10]
    g, b, s = run_gpu(emb, cent, 0.85)
    assert b[0] == 10 and g[0] == 10 and abs(s[0] - 1) < TOL
    assert b[1] == 0 and s[1] == 0 and g[1] == -1
    assert b[2] in (199, 200) and abs(s[2] - 1) < TOL
    check(emb, cent, 0.85)


def test_norms_match_the_definition():
    c = torch.randn(1000, 384).bfloat16()
    c[5] = 0
    inv = binding.cs_route_norms(c.to(DEV)).cpu().double().numpy()
    ref = np.linalg.norm(c.double().numpy(), axis=1)
    np.testing.assert_allclose(inv[ref > 0] * ref[ref > 0], 1.0, rtol=0, atol=3e-5)
    assert inv[5] == 0


def test_device_status_is_clear_after_a_call():
    x = W.route_inputs(W.ROUTE_WORKLOADS[2])
    e, c = x["emb"].to(DEV), x["centroids"].to(DEV)
    inv = binding.cs_route_norms(c)
    dims = binding.RouteDims(e.shape[0], c.shape[0], e.shape[1])
    ws = torch.zeros(binding.load_library().cs_route_workspace_bytes(dims), dtype=torch.uint8, device=DEV)
    binding.cs_route(e, c, inv, 0.85, workspace=ws)
    assert binding.cs_read_device_status(ws) == 0
