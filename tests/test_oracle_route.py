"""Pins for the routing oracle (Sec. 3.1: cosine similarity of a request's
embedding with each group centroid, best group by arg max, cache miss below
the threshold tau).  Each pin comes from outside the oracle: scipy's cosine
distance, geometric special cases with closed-form cosines, and invariances
the definition implies."""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_20507_gb300 import workloads as W

scipy_distance = pytest.importorskip("scipy.spatial.distance")


def bf16(x):
    return W.host_bits(torch.as_tensor(np.asarray(x, dtype=np.float32)).bfloat16())


def as_f64(bits):
    return torch.from_numpy(bits.view(np.int16)).view(torch.bfloat16).double().numpy()


def rand_bits(shape, seed, scale=1.0):
    g = torch.Generator().manual_seed(seed)
    return W.host_bits((torch.randn(*shape, generator=g) * scale).bfloat16())


@pytest.mark.parametrize("B,N,d,seed", [(7, 13, 64, 1), (33, 200, 384, 2), (5, 1, 128, 3)])
def test_scores_match_scipy_cosine(B, N, d, seed):
    e, c = rand_bits((B, d), seed), rand_bits((N, d), seed + 100)
    r = oracle.route(e, c, 0.5)
    cos = 1.0 - scipy_distance.cdist(as_f64(e), as_f64(c), metric="cosine")
    np.testing.assert_allclose(r["score"], cos.max(axis=1), rtol=0, atol=1e-13)
    np.testing.assert_array_equal(r["best"], cos.argmax(axis=1))
    np.testing.assert_array_equal(r["group"], np.where(cos.max(axis=1) >= 0.5, cos.argmax(axis=1), -1))
    srt = np.sort(cos, axis=1)
    if N >= 2:
        np.testing.assert_allclose(r["margin"], srt[:, -1] - srt[:, -2], atol=1e-13)
    np.testing.assert_allclose(r["tau_margin"], np.abs(cos.max(axis=1) - 0.5), atol=1e-13)


def test_identical_and_antipodal_vectors():
    c = rand_bits((6, 64), 5)
    r = oracle.route(c, c, 0.999999)
    np.testing.assert_allclose(r["score"], 1.0, atol=1e-15)
    np.testing.assert_array_equal(r["best"], np.arange(6))
    np.testing.assert_array_equal(r["group"], np.arange(6))
    neg = c ^ np.uint16(0x8000)  # flip every sign bit
    r = oracle.route(neg[:1], c[:1], -2.0)
    np.testing.assert_allclose(r["score"], -1.0, atol=1e-15)


def test_orthogonal_axes_give_zero_and_the_lowest_id_wins_ties():
    d = 64
    eye = np.eye(d, dtype=np.float32)
    r = oracle.route(bf16(eye[:1]), bf16(eye[1:9]), 0.85)
    assert r["score"][0] == 0.0 and r["best"][0] == 0 and r["group"][0] == -1
    assert r["margin"][0] == 0.0
    # 45 degrees between e0 and e0 + e1: cos = 1 / sqrt(2)
    c = np.stack([eye[1], eye[0] + eye[1], eye[0] + eye[2]])
    r = oracle.route(bf16(eye[:1]), bf16(c), 0.7)
    assert r["best"][0] == 1 and abs(r["score"][0] - 2 ** -0.5) < 1e-15 and r["group"][0] == 1


def test_zero_vectors_score_zero():
    d = 128
    c = rand_bits((4, d), 9)
    c[2] = 0
    e = np.zeros((2, d), dtype=np.uint16)
    e[1] = c[3]
    r = oracle.route(e, c, 0.1)
    assert r["score"][0] == 0.0 and r["best"][0] == 0 and r["group"][0] == -1
    assert r["best"][1] == 3 and r["group"][1] == 3
    # a request with every centroid either zero or at a negative cosine picks the zero one (score 0)
    e2 = (c[3] ^ np.uint16(0x8000))[None]
    r = oracle.route(e2, c[2:4], -5.0)
    assert r["best"][0] == 0 and r["score"][0] == 0.0


def test_no_groups_is_a_miss():
    r = oracle.route(rand_bits((3, 64), 4), np.zeros((0, 64), dtype=np.uint16), -10.0)
    np.testing.assert_array_equal(r["best"], -1)
    np.testing.assert_array_equal(r["group"], -1)
    assert np.all(np.isneginf(r["score"]))


def test_scale_invariance():
    e, c = rand_bits((9, 192), 11), rand_bits((40, 192), 12)
    r = oracle.route(e, c, 0.2)
    # x 4 and x 0.25 are exact in bf16 (exponent shift) for these magnitudes
    e4 = W.host_bits(torch.from_numpy(e.view(np.int16)).view(torch.bfloat16) * 4)
    c4 = W.host_bits(torch.from_numpy(c.view(np.int16)).view(torch.bfloat16) * 0.25)
    r2 = oracle.route(e4, c4, 0.2)
    np.testing.assert_allclose(r2["score"], r["score"], atol=1e-15)
    np.testing.assert_array_equal(r2["best"], r["best"])


def test_centroid_permutation_maps_the_winner():
    e, c = rand_bits((20, 64), 21), rand_bits((50, 64), 22)
    perm = np.random.default_rng(3).permutation(50)
    r, rp = oracle.route(e, c, 0.0), oracle.route(e, c[perm], 0.0)
    np.testing.assert_array_equal(perm[rp["best"]], r["best"])
    np.testing.assert_allclose(rp["score"], r["score"], atol=0)


def test_planted_duplicate_goes_to_the_lower_id():
    c = rand_bits((30, 64), 31)
    c[17] = c[4]
    r = oracle.route(c[4:5], c, 0.9)
    assert r["best"][0] == 4 and r["group"][0] == 4 and r["margin"][0] == 0.0


def test_threshold_boundary_is_inclusive():
    e, c = rand_bits((1, 64), 41), rand_bits((5, 64), 42)
    s = oracle.route(e, c, 0.0)["score"][0]
    assert oracle.route(e, c, s)["group"][0] >= 0
    assert oracle.route(e, c, np.nextafter(s, np.inf))["group"][0] == -1


def test_workload_mix_has_hits_misses_and_near_threshold_requests():
    w = W.ROUTE_WORKLOADS[1]
    x = W.route_inputs(w)
    r = oracle.route(W.host_bits(x["emb"]), W.host_bits(x["centroids"]), W.ROUTE_TAU)
    hit = r["group"] >= 0
    assert 0.1 < hit.mean() < 0.9
    assert (np.abs(r["score"] - W.ROUTE_TAU) < 0.05).sum() >= 3
