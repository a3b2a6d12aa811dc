"""The seeded synthetic inputs: shapes, determinism and structure (CPU only)."""
import numpy as np
import torch

from paper_2607_20507_gb300 import workloads as W


def test_configs_match_the_serving_shapes():
    w1, w2, w3, w4 = (W.WORKLOADS[i] for i in (1, 2, 3, 4))
    assert (w1.batch, w1.n_draft, w1.vocab, w1.logit_dtype) == (1, 4, 32000, "f32")
    assert (w2.batch, w2.n_draft, w2.vocab, w2.temperatures) == (8, 5, 128256, (0.0, 0.7))
    assert (w3.batch, w3.n_q_heads, w3.n_kv_heads, w3.vocab) == (64, 28, 4, 151936)
    assert (w4.batch, w4.n_draft, w4.n_q_heads, w4.page_size) == (256, 8, 64, 32)
    assert len(list(W.sweep_accept_cells())) == 375
    assert len(list(W.sweep_attention_cells())) == 25


def test_context_lengths_follow_their_distribution():
    for wid, lo, hi in ((2, 1024, 4096), (3, 512, 8192), (4, 2048, 16384)):
        L = W.context_lengths(W.WORKLOADS[wid]).numpy()
        assert L.min() >= lo and L.max() <= hi
    L3 = W.context_lengths(W.WORKLOADS[3]).numpy()
    assert 1500 < np.median(L3) < 2800          # lognormal with median 2048
    assert (W.context_lengths(W.WORKLOADS[1]).numpy() == 512).all()


def test_attention_inputs_are_deterministic_and_paged():
    w = W.WORKLOADS[2].with_(batch=3, ctx=("uniform", 40, 100))
    a = W.attention_inputs(w)
    b = W.attention_inputs(w)
    for key in ("q", "k_pages", "v_pages", "page_table", "ctx_lens"):
        assert torch.equal(a[key], b[key])
    ps = w.page_size
    table, lens = a["page_table"].numpy(), a["ctx_lens"].numpy()
    used = []
    for r in range(w.batch):
        n = -(-int(lens[r]) // ps)
        assert (table[r, :n] >= 0).all() and (table[r, n:] == -1).all()
        used.extend(table[r, :n].tolist())
    assert sorted(used) == list(range(a["k_pages"].shape[0]))    # a permutation of the pool
    assert a["q"].shape == (3, w.n_draft + 1, w.n_q_heads, w.head_dim)
    assert a["q"].dtype == torch.bfloat16


def test_contiguous_workload_uses_identity_pages():
    a = W.attention_inputs(W.WORKLOADS[1])
    assert a["page_table"][0, :32].tolist() == list(range(32))


def test_accept_inputs_shapes_and_draft_noise():
    w = W.WORKLOADS[2].with_(batch=2, vocab=1000)
    for T in (0.0, 0.7):
        d = W.accept_inputs(w, T)
        assert d["target"].shape == (2, 6, 1000) and d["draft"].shape == (2, 5, 1000)
        assert d["draft_tokens"].dtype == torch.int32
        assert int(d["draft_tokens"].min()) >= 0 and int(d["draft_tokens"].max()) < 1000
        noise = (d["draft"].float() - d["target"][:, :5].float()).std().item()
        assert 0.4 < noise < 0.6
        assert 2.7 < d["target"].float().std().item() < 3.3
    d = W.accept_inputs(w, 0.0)
    assert torch.equal(d["draft_tokens"].long(), d["draft"].float().argmax(-1))


def test_subsets_keep_only_their_pages():
    w = W.WORKLOADS[3].with_(batch=5, ctx=("uniform", 30, 90))
    a = W.attention_inputs(w)
    s = W.attention_subset(a, [3, 1])
    assert torch.equal(s["ctx_lens"], a["ctx_lens"][[3, 1]])
    n = sum(-(-int(L) // w.page_size) for L in s["ctx_lens"].tolist())
    assert s["k_pages"].shape[0] == n
    assert torch.equal(s["k_pages"][int(s["page_table"][0, 0])], a["k_pages"][int(a["page_table"][3, 0])])
