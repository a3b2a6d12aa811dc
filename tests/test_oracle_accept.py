"""Pins for the fp64 speculative-acceptance oracle (CPU only).

The oracle is treated as a black box and checked against facts fixed by the
mathematics of speculative sampling, not against a retyped formula:

* exact enumeration on an 8-token vocabulary: the accept thresholds and the
  draw cells are located by bisection on the uniforms (the oracle takes fp64
  uniforms here), and the resulting emitted-token law at every position equals
  p_i = softmax(z_t,i / T) from scipy to 1e-12 -- the defining property of
  speculative sampling; the bonus draw equals p_k;
* the rejection mass equals the total-variation distance 1 - sum(min(p, q));
* special cases: p == q accepts everything; disjoint supports reject
  everything and then draw from p; a one-hot target always emits its token;
  ascending-id order of the inverse CDF;
* greedy mode equals numpy argmax (first occurrence) agreement;
* probabilities sum to one; hand-derived golden cases (tests/golden);
* Monte Carlo acceptance rate and emitted-token histogram.
"""
import json
import math
import os

import numpy as np
import pytest
import torch
from scipy.special import softmax

import oracle

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "accept_hand_v4.json")


def widen(z, dtype):
    """(array handed to the oracle, exact float64 values)."""
    z = np.asarray(z, dtype=np.float32)
    if dtype == "f32":
        return z, z.astype(np.float64)
    t = torch.from_numpy(z).to(torch.bfloat16)
    return t.view(torch.int16).numpy().view(np.uint16), t.to(torch.float64).numpy()


class OneRequest:
    """A single request of the acceptance step, evaluated through the oracle."""

    def __init__(self, zt, zd, T):
        self.zt, self.zd, self.T = zt, zd, T
        self.k = zt.shape[0] - 1
        self.V = zt.shape[1]

    def run(self, x, u):
        out, acc, _ = oracle.spec_accept(self.zt[None], self.zd[None],
                                         np.asarray(x, np.int32)[None],
                                         np.asarray(u, np.float64)[None], self.T)
        return out[0], int(acc[0])


def first_true(pred, lo=0.0, hi=1.0):
    """Boundary of a predicate that is False on [0, b) and True on [b, 1)."""
    top = np.nextafter(1.0, 0.0)
    if not pred(top):
        return 1.0
    if pred(0.0):
        return 0.0
    for _ in range(200):
        mid = 0.5 * (lo + hi)
        if mid <= lo or mid >= hi:
            break
        if pred(mid):
            hi = mid
        else:
            lo = mid
    return hi


def accept_threshold(req, x, i):
    """Measure of {u_i : position i accepted} with earlier positions accepted (u_j = 0)."""
    x = list(x)

    def rejected(ui):
        u = [0.0] * (req.k + 1)
        u[i] = ui
        return req.run(x, u)[1] <= i

    return first_true(rejected)


def draw_law(req, x, u_prefix, pos):
    """Law of the token emitted at `pos` as u_k sweeps [0, 1) (cells found by bisection)."""
    law = np.zeros(req.V)
    prev = 0.0
    for v in range(req.V):
        def beyond(uk, v=v):
            out, _ = req.run(x, list(u_prefix) + [uk])
            return out[pos] > v
        b = first_true(beyond)
        law[v] = b - prev
        prev = b
    return law


def make_rows(rng, k, V, dtype, scale=1.5):
    zt, zt64 = widen(rng.standard_normal((k + 1, V)) * scale, dtype)
    zd, zd64 = widen(zt64[:k] + rng.standard_normal((k, V)) * scale, dtype)
    return zt, zt64, zd, zd64


@pytest.mark.parametrize("k,T,dtype,seed", [
    (1, 1.0, "f32", 0), (2, 0.6, "f32", 1), (3, 1.7, "bf16", 2), (2, 1.0, "bf16", 3),
    (3, 0.9, "f32", 4),
])
def test_emitted_law_equals_target_at_every_position(k, T, dtype, seed):
    V = 8
    rng = np.random.default_rng(seed)
    zt, zt64, zd, zd64 = make_rows(rng, k, V, dtype)
    req = OneRequest(zt, zd, T)
    for i in range(k):
        p = softmax(zt64[i] / T)
        q = softmax(zd64[i] / T)
        theta = np.array([accept_threshold(req, [0] * i + [x] + [0] * (k - i - 1), i)
                          for x in range(V)])
        reject_mass = 1.0 - float(np.dot(q, theta))
        # rejection probability = total variation distance between p and q
        assert reject_mass == pytest.approx(1.0 - np.minimum(p, q).sum(), abs=1e-12)
        # residual law, reached through a draft token that can be rejected
        xr = int(np.argmin(theta))
        assert theta[xr] < 1.0
        u_prefix = [0.0] * i + [0.5 * (theta[xr] + 1.0)] + [0.0] * (k - i - 1)
        law = draw_law(req, [0] * i + [xr] + [0] * (k - i - 1), u_prefix, i)
        emitted = q * theta + reject_mass * law
        np.testing.assert_allclose(emitted, p, rtol=0, atol=1e-12)
    # bonus: all k accepted (u = 0) -> the token at position k follows p_k
    law = draw_law(req, [0] * k, [0.0] * k, k)
    np.testing.assert_allclose(law, softmax(zt64[k] / T), rtol=0, atol=1e-12)


def test_equal_distributions_accept_everything():
    rng = np.random.default_rng(5)
    k, V = 3, 8
    zt, zt64 = widen(rng.standard_normal((k + 1, V)) * 2, "f32")
    req = OneRequest(zt, zt[:k].copy(), 0.8)
    for i in range(k):
        for x in range(V):
            assert accept_threshold(req, [x] * k, i) == 1.0
    uu = rng.random((200, k + 1))
    for u in uu:
        out, a = req.run([int(v) for v in rng.integers(0, V, k)], u)
        assert a == k


def test_disjoint_supports_reject_and_draw_from_target():
    V, k, T = 8, 1, 1.0
    zt = np.full((2, V), -1.0e4, np.float32)
    zt[:, :4] = np.log([0.1, 0.2, 0.3, 0.4])
    zd = np.full((1, V), -1.0e4, np.float32)
    zd[0, 4:] = 0.0
    req = OneRequest(zt, zd, T)
    for x in range(4, 8):
        assert accept_threshold(req, [x], 0) == 0.0
    law = draw_law(req, [5], [0.5], 0)
    np.testing.assert_allclose(law, [0.1, 0.2, 0.3, 0.4, 0, 0, 0, 0], atol=1e-7)


def test_one_hot_target_always_emits_its_token():
    V, k = 8, 2
    rng = np.random.default_rng(6)
    zt = np.full((k + 1, V), -3.0e3, np.float32)
    zt[:, 6] = 0.0
    zd = rng.standard_normal((k, V)).astype(np.float32)
    req = OneRequest(zt, zd, 1.0)
    for _ in range(100):
        x = [int(v) for v in rng.integers(0, V, k)]
        out, a = req.run(x, rng.random(k + 1))
        assert out[a] == 6
        assert all(t == 6 for t in out[:a])


def test_inverse_cdf_ascends_token_ids():
    r = np.array([0, 0, 0.3, 0, 0, 0.7, 0, 0], float)
    assert oracle.inverse_cdf(r, 1.0, 0.0)[0] == 2
    assert oracle.inverse_cdf(r, 1.0, 0.29)[0] == 2
    assert oracle.inverse_cdf(r, 1.0, 0.31)[0] == 5
    assert oracle.inverse_cdf(r, 1.0, 0.999999)[0] == 5
    # u*Z at or beyond the total (rounding): the largest id with positive weight
    assert oracle.inverse_cdf(r, 1.0, 1.0)[0] == 5


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_greedy_equals_argmax_agreement(dtype):
    rng = np.random.default_rng(7)
    B, k, V = 64, 4, 50
    z = rng.standard_normal((B, k + 1, V)).astype(np.float32)
    # plant exact ties for the maximum in some rows (before rounding to the dtype)
    for b in range(0, B, 3):
        i = b % (k + 1)
        j1, j2 = sorted(rng.choice(V, 2, replace=False))
        z[b, i, j1] = z[b, i, j2] = z[b, i].max() + 1.0
    zt, zt64 = widen(z, dtype)
    g = np.argmax(zt64, axis=-1)                   # first occurrence
    x = g[:, :k].copy()
    # corrupt a random position in half the requests
    for b in range(0, B, 2):
        pos = b % k
        x[b, pos] = (x[b, pos] + 1 + b % (V - 1)) % V
    out, acc, margin = oracle.spec_accept(zt, None, x, rng.random((B, k + 1)).astype(np.float32), 0.0)
    for b in range(B):
        mism = [i for i in range(k) if x[b, i] != g[b, i]]
        a = mism[0] if mism else k
        assert acc[b] == a
        assert list(out[b, :a]) == list(x[b, :a])
        assert out[b, a] == g[b, a]
        assert all(out[b, a + 1:] == -1)
    assert np.all(np.isinf(margin))


def test_probabilities_sum_to_one():
    rng = np.random.default_rng(8)
    for V in (8, 1000, 32000):
        z = (rng.standard_normal(V) * 3).astype(np.float32)
        for T in (0.3, 0.7, 1.0, 2.0):
            p, S = oracle.row_probs(z, T)
            assert np.all(p >= 0)
            assert p.sum() == pytest.approx(1.0, abs=1e-12)
            np.testing.assert_allclose(p, softmax(z.astype(np.float64) / T), rtol=1e-12, atol=1e-300)
        q, _ = oracle.row_probs((z + rng.standard_normal(V)).astype(np.float32), 1.0)
        p, _ = oracle.row_probs(z, 1.0)
        r, Z = oracle.residual(p, q)
        assert np.all(r >= 0)
        assert (r / Z).sum() == pytest.approx(1.0, abs=1e-12)
        assert Z == pytest.approx(1.0 - np.minimum(p, q).sum(), abs=1e-12)
        assert np.all((r > 0) == (p > q))


def test_golden_hand_cases():
    g = json.load(open(GOLDEN))
    rows = {k: np.log(np.asarray(v, np.float64)).astype(np.float32) for k, v in g["rows"].items()}
    for c in g["cases"]:
        zt = np.stack([rows[n] for n in c["target"]])[None]
        zd = np.stack([rows[n] for n in c["draft"]])[None]
        out, acc, _ = oracle.spec_accept(zt, zd, np.asarray(c["x"], np.int32)[None],
                                         np.asarray(c["u"], np.float32)[None], c["T"])
        assert out[0].tolist() == c["out"], c["id"]
        assert int(acc[0]) == c["n_accepted"], c["id"]


def test_monte_carlo_acceptance_and_emitted_histogram():
    rng = np.random.default_rng(9)
    V, k, T, n = 8, 1, 1.0, 40000
    zt, zt64, zd, zd64 = make_rows(rng, k, V, "f32", scale=1.0)
    p0, q0 = softmax(zt64[0] / T), softmax(zd64[0] / T)
    x = rng.choice(V, size=(n, 1), p=q0).astype(np.int32)
    u = rng.random((n, k + 1)).astype(np.float32)
    out, acc, _ = oracle.spec_accept(np.repeat(zt[None], n, 0), np.repeat(zd[None], n, 0), x, u, T)
    alpha = np.minimum(p0, q0).sum()
    se = math.sqrt(alpha * (1 - alpha) / n)
    assert abs(acc.mean() - alpha) < 4 * se
    counts = np.bincount(out[:, 0], minlength=V)
    expected = n * p0
    chi2 = float(((counts - expected) ** 2 / expected).sum())
    assert chi2 < 30.0          # 7 dof: P(chi2 > 30) < 1e-4


def test_out_of_range_draft_token_is_rejected():
    rng = np.random.default_rng(10)
    zt, _, zd, _ = make_rows(rng, 2, 8, "f32")
    req = OneRequest(zt, zd, 1.0)
    for bad in (-1, 8, 1 << 30):
        out, a = req.run([bad, 0], [0.0, 0.0, 0.3])
        assert a == 0 and out[1] == -1 and 0 <= out[0] < 8


def test_margin_reports_threshold_distance():
    g = json.load(open(GOLDEN))
    rows = {k: np.log(np.asarray(v, np.float64)).astype(np.float32) for k, v in g["rows"].items()}
    zt = np.stack([rows["H"], rows["R"]])[None]
    zd = rows["U"][None, None]
    _, _, m, dm = oracle.spec_accept(zt, zd, np.array([[2]], np.int32),
                                     np.array([[0.49, 0.05]], np.float32), 1.0, with_draw_margin=True)
    # accept test: u_0 = 0.49 against the ratio 0.5; draw: u_1 = 0.05 inside the cell [0, 0.1)
    assert m[0] == pytest.approx(0.01, abs=1e-6)
    assert dm[0] == pytest.approx(0.05, abs=1e-6)
