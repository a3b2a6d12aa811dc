"""GPU parity of cs_spec_accept against the fp64 oracle (through the C ABI).

Token ids and accepted counts must equal the oracle's exactly, except for
near-ties, which are counted and reported:
* an accept test with |u_i - p_i(x_i)/q_i(x_i)| < 1e-5;
* a draw with u_k within 1e-6 of either CDF value C(v-1)/Z, C(v)/Z that
  bracket the drawn token (the fp32 cumulative sums of the kernel resolve
  the CDF to ~1e-8 in practice; 1e-6 leaves a wide margin).
Greedy mode compares the stored logits themselves and has no near-ties.
Statistical tests check the GPU sampler against the laws speculative
sampling must produce.
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
from parity_bands import DRAW_TIE, NEAR_TIE, check_band_mismatches


def gpu(inp, T):
    d = inp["draft"] if T > 0 else None
    out, n = binding.cs_spec_accept(inp["target"], d, inp["draft_tokens"], inp["uniforms"], T)
    torch.cuda.synchronize()
    return out.cpu().numpy(), n.cpu().numpy()


def ref(inp, T):
    """(tokens, n_accepted, near_tie) from the oracle on the same inputs."""
    d = W.host_bits(inp["draft"]) if T > 0 else None
    eo, en, am, dm = oracle.spec_accept(W.host_bits(inp["target"]), d,
                                        inp["draft_tokens"].cpu().numpy(),
                                        inp["uniforms"].cpu().numpy(), T, with_draw_margin=True)
    return eo, en, (am < NEAR_TIE) | (dm < DRAW_TIE)


def assert_parity(inp, T, what=""):
    out, n = gpu(inp, T)
    eo, en, tie = ref(inp, T)
    mism = np.any(out != eo, axis=1) | (n != en)
    bad = mism & ~tie
    assert not bad.any(), (f"{what}: {int(bad.sum())} requests differ outside the near-tie band; "
                           f"first {np.nonzero(bad)[0][:5].tolist()}")
    print(f"{what}: {len(n)} requests, near-ties {int(tie.sum())}, of which differ {int((mism & tie).sum())}")
    check_band_mismatches(int((mism & tie).sum()), len(n), what)
    # structure of every GPU output, ties included
    k = out.shape[1] - 1
    V = inp["target"].shape[2]
    for b in range(out.shape[0]):
        a = int(n[b])
        assert 0 <= a <= k
        assert (out[b, a + 1:] == -1).all()
        assert 0 <= out[b, a] < V
    return int(tie.sum()), n


@pytest.mark.parametrize("wid,T", [(1, 1.0), (2, 0.0), (2, 0.7), (3, 1.0), (4, 0.8)])
def test_serving_workloads(wid, T):
    w = W.WORKLOADS[wid]
    inp = W.accept_inputs(w, T, DEV)
    ties, n = assert_parity(inp, T, f"{w.name} T={T}")
    print(f"  mean accepted {n.mean():.3f}")


@pytest.mark.parametrize("sigma,k,B,V", [(0.1, 4, 64, 256000), (4.0, 16, 8, 128256),
                                         (1.0, 1, 512, 32000), (0.5, 8, 256, 32000),
                                         (2.0, 2, 1, 256000), (0.1, 16, 64, 32000),
                                         (0.1, 8, 256, 128256), (0.1, 1, 512, 256000),
                                         (0.1, 2, 8, 32000), (4.0, 4, 64, 256000)])
def test_sweep_cells(sigma, k, B, V):
    w = next(c for c in W.sweep_accept_cells()
             if c.draft_sigma == sigma and c.n_draft == k and c.batch == B and c.vocab == V)
    inp = W.accept_inputs(w, W.SWEEP_TEMPERATURE, DEV)
    assert_parity(inp, W.SWEEP_TEMPERATURE, w.name)


def stratified_sweep_cells():
    """At each of B = 64, 256 and 512: five cells that between them take every
    k, every draft sigma and every vocabulary of the sweep once."""
    cells = []
    for bi, B in enumerate((64, 256, 512)):
        for i, k in enumerate(W.SWEEP_KS):
            sigma = W.SWEEP_SIGMAS[(i + bi) % 5]
            V = W.SWEEP_VOCABS[(i + bi) % 3]
            cells.append((sigma, k, B, V))
    return cells


@pytest.mark.parametrize("sigma,k,B,V", stratified_sweep_cells())
def test_sweep_stratified_at_serving_batches(sigma, k, B, V):
    """The launch at full size; the oracle on a seeded sample of 24 requests."""
    w = next(c for c in W.sweep_accept_cells()
             if c.draft_sigma == sigma and c.n_draft == k and c.batch == B and c.vocab == V)
    T = W.SWEEP_TEMPERATURE
    inp = W.accept_inputs(w, T, DEV)
    out, n = gpu(inp, T)
    idx = sorted(np.random.default_rng(w.cell).choice(B, 24, replace=False).tolist())
    sub = W.accept_subset(inp, idx)
    eo, en, tie = ref(sub, T)
    mism = np.any(out[idx] != eo, axis=1) | (n[idx] != en)
    assert not (mism & ~tie).any(), f"{w.name}: requests {np.nonzero(mism & ~tie)[0].tolist()} differ"
    check_band_mismatches(int((mism & tie).sum()), len(idx), w.name)
    assert (out[np.arange(B), n] >= 0).all() and (n >= 0).all() and (n <= k).all()


def custom(B, k, V, dtype, T, sigma=1.0, cell=0):
    w = W.Workload(91, "custom", batch=B, n_draft=k, vocab=V, logit_dtype=dtype,
                   draft_sigma=sigma, temperatures=(T,), n_q_heads=8, n_kv_heads=8, head_dim=128,
                   ctx=("const", 64), page_size=16, cell=cell)
    return W.accept_inputs(w, T, DEV)


@pytest.mark.parametrize("V", [8, 13, 1000, 4099, 32001])
@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_ragged_and_unaligned_vocabularies(V, dtype):
    for T in (0.0, 0.9):
        inp = custom(16, 3, V, dtype, T, cell=V % 97)
        assert_parity(inp, T, f"V={V} {dtype} T={T}")


@pytest.mark.parametrize("T", [0.05, 0.3, 2.5, 6.0])
def test_temperature_range(T):
    assert_parity(custom(32, 4, 5000, "bf16", T, cell=int(T * 100)), T, f"T={T}")


def test_equal_draft_accepts_everything():
    inp = custom(16, 6, 3000, "bf16", 1.0, cell=3)
    inp["draft"] = inp["target"][:, :6].contiguous()
    out, n = gpu(inp, 1.0)
    assert (n == 6).all()
    assert_parity(inp, 1.0, "p == q")


def test_out_of_range_draft_tokens_are_rejected():
    inp = custom(8, 3, 500, "f32", 1.0, cell=4)
    inp["draft_tokens"][:, 1] = torch.tensor([-1, 500, 1 << 30, -7, 501, 999, -100, 2 ** 31 - 1],
                                             dtype=torch.int32, device=DEV)
    out, n = gpu(inp, 1.0)
    assert (n <= 1).all()
    assert_parity(inp, 1.0, "bad tokens")
    inp0 = custom(8, 3, 500, "f32", 0.0, cell=4)
    inp0["draft_tokens"][:, 0] = -3
    out, n = gpu(inp0, 0.0)
    assert (n == 0).all()
    assert_parity(inp0, 0.0, "bad tokens greedy")


def test_masked_minus_inf_logits():
    inp = custom(16, 4, 2000, "bf16", 1.0, cell=5)
    mask = torch.rand(inp["target"].shape[-1], generator=torch.Generator().manual_seed(1)) < 0.3
    inp["target"][..., mask.to(DEV)] = float("-inf")
    inp["draft"][..., mask.to(DEV)] = float("-inf")
    # redraw draft tokens among unmasked ids
    allowed = torch.nonzero(~mask).flatten()
    pick = torch.randint(0, allowed.numel(), inp["draft_tokens"].shape, generator=torch.Generator().manual_seed(2))
    inp["draft_tokens"] = allowed[pick].to(torch.int32).to(DEV)
    out, n = gpu(inp, 1.0)
    assert not mask[torch.as_tensor(out[out >= 0])].any()
    assert_parity(inp, 1.0, "-inf masked")


@pytest.mark.parametrize("V,dtype", [(5000, "bf16"), (40000, "f32"), (300000, "bf16")])
def test_draw_at_the_top_of_the_cdf(V, dtype):
    # u_k just below 1 puts the draw at the end of the CDF, where the fp32
    # running sums may stop short of u_k * Z (the rounding fallback: the last
    # id with positive weight).  The last 100 ids are masked and the last
    # unmasked one carries most of the target's mass, so both paths must
    # emit exactly that id, for the residual and the bonus draw alike.
    B, k = 24, 3
    inp = custom(B, k, V, dtype, 1.0, cell=9)
    last = V - 101
    inp["target"][..., last + 1:] = float("-inf")
    inp["draft"][..., last + 1:] = float("-inf")
    inp["target"][..., last] = inp["target"].float().amax(dim=-1).to(inp["target"].dtype) + 6.0
    inp["draft_tokens"].clamp_(max=last)
    inp["uniforms"][:, k] = float(np.nextafter(np.float32(1.0), np.float32(0.0)))
    out, n = gpu(inp, 1.0)
    got = out[np.arange(B), n]
    assert (got == last).all(), got


def test_deterministic():
    inp = W.accept_inputs(W.WORKLOADS[3], 1.0, DEV)
    a = gpu(inp, 1.0)
    b = gpu(inp, 1.0)
    assert (a[0] == b[0]).all() and (a[1] == b[1]).all()


def test_rows_beyond_65535_requests():
    B = 65536 + 7
    inp = custom(B, 1, 8, "f32", 1.0, cell=6)
    out, n = gpu(inp, 1.0)
    sl = [0, 1, 65534, 65535, 65536, B - 1]
    sub = W.accept_subset(inp, sl)
    eo, en, tie = ref(sub, 1.0)
    ok = (out[sl] == eo).all(axis=1) & (n[sl] == en) | tie
    assert ok.all()


def test_statistics_emitted_law_and_acceptance_rate():
    # one fixed pair of rows, many requests with x ~ q and fresh uniforms:
    # the first emitted token must follow p, the acceptance rate sum(min(p, q))
    V, k, T, B = 8, 1, 1.0, 1 << 20
    g = torch.Generator().manual_seed(11)
    zt = (torch.randn(k + 1, V, generator=g) * 1.3).float()
    zd = (zt[:k] + torch.randn(k, V, generator=g)).float()
    p0 = softmax(zt[0].double().numpy() / T)
    q0 = softmax(zd[0].double().numpy() / T)
    x = torch.multinomial(torch.from_numpy(q0), B, replacement=True, generator=g).to(torch.int32)
    inp = dict(target=zt.expand(B, k + 1, V).contiguous().to(DEV),
               draft=zd.expand(B, k, V).contiguous().to(DEV),
               draft_tokens=x.view(B, 1).to(DEV),
               uniforms=torch.rand(B, k + 1, generator=g).to(DEV))
    out, n = gpu(inp, T)
    alpha = np.minimum(p0, q0).sum()
    se = math.sqrt(alpha * (1 - alpha) / B)
    assert abs(n.mean() - alpha) < 5 * se
    counts = np.bincount(out[:, 0], minlength=V)
    chi2 = float(((counts - B * p0) ** 2 / (B * p0)).sum())
    assert chi2 < 35.0      # 7 dof; P(chi2 > 35) ~ 1e-5
    # bonus draws (accepted requests) follow p_1
    p1 = softmax(zt[1].double().numpy() / T)
    acc = n == 1
    c1 = np.bincount(out[acc, 1], minlength=V)
    chi2b = float(((c1 - acc.sum() * p1) ** 2 / (acc.sum() * p1)).sum())
    assert chi2b < 35.0


def test_empty_batch():
    inp = custom(1, 2, 100, "bf16", 1.0, cell=7)
    e = {k: v[:0] for k, v in inp.items()}
    out, n = binding.cs_spec_accept(e["target"], e["draft"], e["draft_tokens"], e["uniforms"], 1.0)
    assert out.shape == (0, 3) and n.shape == (0,)
