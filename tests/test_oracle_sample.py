"""Pins for the fp64 draft-side sampling oracle (CPU only).

Checked against facts the mathematics fixes, not a retyped formula:

* exact law on an 8-token vocabulary: the cells of the inverse CDF are found
  by bisection on the (fp64) uniform, and their widths equal
  softmax(z / T) from scipy to 1e-12, for fp32 and bf16 logits;
* ascending-id order of the cells; u = 0 gives the smallest id of positive
  weight; masked (-inf) tokens have empty cells;
* closed forms: one finite logit always wins; equal logits split [0, 1)
  evenly;
* greedy mode equals numpy argmax (first occurrence on planted ties);
* the acceptance oracle with no drafted position draws the same token.
"""
import numpy as np
import pytest
import torch
from scipy.special import softmax

import oracle


def widen(z, dtype):
    z = np.asarray(z, dtype=np.float32)
    if dtype == "f32":
        return z, z.astype(np.float64)
    t = torch.from_numpy(z).to(torch.bfloat16)
    return t.view(torch.int16).numpy().view(np.uint16), t.to(torch.float64).numpy()


def first_true(pred):
    """Boundary b of a predicate False on [0, b) and True on [b, 1)."""
    top = np.nextafter(1.0, 0.0)
    if not pred(top):
        return 1.0
    if pred(0.0):
        return 0.0
    lo, hi = 0.0, 1.0
    for _ in range(200):
        mid = 0.5 * (lo + hi)
        if mid <= lo or mid >= hi:
            break
        if pred(mid):
            hi = mid
        else:
            lo = mid
    return hi


def law_of(z, T):
    """Widths of the inverse-CDF cells of every token of one row."""
    V = z.shape[-1]
    law, prev = np.zeros(V), 0.0
    for v in range(V):
        b = first_true(lambda u, v=v: oracle.sample(z[None], [u], T)[0] > v)
        law[v] = b - prev
        prev = b
    return law


@pytest.mark.parametrize("T,dtype,seed", [(1.0, "f32", 0), (0.6, "f32", 1), (1.7, "bf16", 2),
                                          (0.3, "bf16", 3), (2.5, "f32", 4)])
def test_law_equals_softmax(T, dtype, seed):
    rng = np.random.default_rng(seed)
    z, z64 = widen(rng.standard_normal(8) * 1.5, dtype)
    np.testing.assert_allclose(law_of(z, T), softmax(z64 / T), rtol=0, atol=1e-12)


def test_masked_tokens_have_empty_cells_and_u0_takes_the_first_live_id():
    z = np.array([-np.inf, -np.inf, 0.3, -np.inf, 1.2, 0.0, -np.inf, 2.0], dtype=np.float32)
    law = law_of(z, 1.0)
    assert (law[np.isinf(z)] == 0).all()
    live = np.isfinite(z)
    np.testing.assert_allclose(law[live], softmax(z[live].astype(np.float64)), rtol=0, atol=1e-12)
    assert oracle.sample(z[None], [0.0], 1.0)[0] == 2
    assert oracle.sample(z[None], [np.nextafter(1.0, 0.0)], 1.0)[0] == 7


def test_closed_forms():
    one = np.full(16, -np.inf, dtype=np.float32)
    one[11] = 0.5
    for u in (0.0, 0.3, 0.999999):
        assert oracle.sample(one[None], [u], 0.8)[0] == 11
    eq = np.zeros(4, dtype=np.float32)
    np.testing.assert_allclose(law_of(eq, 1.3), [0.25] * 4, rtol=0, atol=1e-12)


def test_greedy_is_first_argmax():
    rng = np.random.default_rng(5)
    z = rng.standard_normal((64, 300)).astype(np.float32)
    z[::3, 17] = z[::3].max(axis=1) + 1.0
    z[::3, 250] = z[::3, 17]          # planted tie: the lower id wins
    got = oracle.sample(z, np.zeros(64), 0.0)
    np.testing.assert_array_equal(got, np.argmax(z, axis=1))
    assert (got[::3] == 17).all()


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_matches_the_acceptance_oracle_with_no_drafts(dtype):
    rng = np.random.default_rng(6)
    z, _ = widen(rng.standard_normal((32, 1000)) * 2.0, dtype)
    u = rng.random(32)
    for T in (0.0, 0.7, 1.0):
        a = oracle.sample(z, u, T)
        z3 = np.ascontiguousarray(z[:, None, :])
        out, n, _ = oracle.spec_accept(z3, None if T == 0 else np.ascontiguousarray(z3[:, :0, :]),
                                       np.zeros((32, 0), np.int32), u[:, None], T)
        np.testing.assert_array_equal(a, out[:, 0])
        assert (n == 0).all()
