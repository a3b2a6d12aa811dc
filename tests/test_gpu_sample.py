"""GPU parity of cs_sample (the drafter's sampling step) against the fp64 oracle.

Tokens must equal the oracle's exactly, except draws whose uniform lies
within 1e-6 of either CDF edge of the drawn cell (near-ties, counted and
reported; the same band as the acceptance step's final draw).  Greedy mode
has no near-ties.  A chi-square test checks the sampled law.
"""
import math

import numpy as np
import pytest
import torch
from scipy.special import softmax

import oracle
from paper_2607_20507_gb300 import binding
from paper_2607_20507_gb300 import workloads as W

pytestmark = pytest.mark.gpu

DEV = "cuda:0"
from parity_bands import DRAW_TIE, check_band_mismatches


def logits_of(B, V, dtype, seed, scale=3.0):
    g = torch.Generator().manual_seed(seed)
    z = torch.randn(B, V, generator=g) * scale
    return z.to(torch.bfloat16 if dtype == "bf16" else torch.float32).to(DEV)


def uniforms_of(B, seed):
    return torch.rand(B, generator=torch.Generator().manual_seed(seed + 1)).to(DEV)


def check(z, u, T, what):
    got = binding.cs_sample(z, u, T)
    torch.cuda.synchronize()
    got = got.cpu().numpy()
    exp, margin = oracle.sample(W.host_bits(z), u.cpu().numpy(), T, with_margin=True)
    tie = margin < DRAW_TIE
    bad = (got != exp) & ~tie
    assert not bad.any(), f"{what}: {int(bad.sum())} rows differ outside the near-tie band"
    check_band_mismatches(int(((got != exp) & tie).sum()), len(got), what)
    V = z.shape[1]
    assert ((got >= 0) & (got < V)).all()
    print(f"{what}: {len(got)} rows, near-ties {int(tie.sum())}, of which differ {int(((got != exp) & tie).sum())}")


@pytest.mark.parametrize("B,V,dtype", [(40, 128256, "bf16"), (4, 32000, "f32"), (320, 151936, "bf16"),
                                       (1, 5, "f32"), (16, 4099, "bf16"), (16, 32001, "f32"),
                                       (2048, 32000, "bf16")])
@pytest.mark.parametrize("T", [0.0, 0.7, 1.0])
def test_parity(B, V, dtype, T):
    z = logits_of(B, V, dtype, seed=B * 7 + V % 1000)
    check(z, uniforms_of(B, B + V), T, f"B={B} V={V} {dtype} T={T}")


@pytest.mark.parametrize("T", [0.05, 2.5, 6.0])
def test_temperature_range(T):
    z = logits_of(64, 20000, "bf16", seed=int(T * 100))
    check(z, uniforms_of(64, 3), T, f"T={T}")


def test_masked_tokens_are_never_drawn():
    z = logits_of(64, 3000, "bf16", seed=11)
    mask = torch.rand(3000, generator=torch.Generator().manual_seed(12)) < 0.4
    z[:, mask.to(DEV)] = float("-inf")
    u = uniforms_of(64, 13)
    got = binding.cs_sample(z, u, 1.0).cpu()
    assert not mask[got.long()].any()
    check(z, u, 1.0, "-inf masked")


def test_top_of_the_cdf():
    # u just below 1: the draw is the last token of positive weight, whichever
    # of the crossing and the rounding fallback decides it
    V = 5000
    z = logits_of(24, V, "bf16", seed=14)
    z[:, V - 100:] = float("-inf")
    z[:, V - 101] = z.float().amax(dim=1).to(z.dtype) + 6.0
    u = torch.full((24,), float(np.nextafter(np.float32(1.0), np.float32(0.0))), device=DEV)
    got = binding.cs_sample(z, u, 1.0).cpu().numpy()
    assert (got == V - 101).all()


def test_law_chi_square():
    V, B, T = 8, 1 << 20, 0.9
    g = torch.Generator().manual_seed(21)
    row = torch.randn(V, generator=g) * 1.3
    z = row.expand(B, V).contiguous().to(DEV)
    u = torch.rand(B, generator=g).to(DEV)
    got = binding.cs_sample(z, u, T).cpu().numpy()
    p = softmax(row.double().numpy() / T)
    counts = np.bincount(got, minlength=V)
    chi2 = float(((counts - B * p) ** 2 / (B * p)).sum())
    assert chi2 < 35.0      # 7 dof; P(chi2 > 35) ~ 1e-5


def test_empty_batch():
    z = logits_of(1, 100, "bf16", seed=1)[:0]
    out = binding.cs_sample(z, torch.zeros(0, device=DEV), 1.0)
    assert out.shape == (0,)
