"""Seeded synthetic inputs shaped like the serving workloads of the draft-and-verify step.

This module only draws random numbers and arranges them in the layouts the
library expects.  It holds none of the method's arithmetic (no attention, no
softmax, no acceptance test); both the CUDA path and the fp64 oracle receive
the tensors it produces.

The paper evaluates on request datasets (Shopping, WebShop, Formula,
CodeTAT-QA; Sec. 4.2) with Qwen3-32B as target and Qwen3-1.7B as drafter
(Sec. 4.1).  Neither the datasets nor the weights are used here: the tensors
below stand in for them, with the shapes of the serving workloads:

* Q, K, V ~ N(0, 1) in bf16;
* target logits ~ N(0, 3^2); draft logits = target + N(0, sigma^2), rounded to
  the logit dtype after adding the noise;
* draft tokens sampled from softmax(draft / T) by the Gumbel-max trick (the
  drafter's own sampling, upstream of the verified step), or argmax(draft)
  when T == 0;
* uniforms ~ U[0, 1) in fp32;
* context lengths constant, uniform, or lognormal-and-clipped per workload;
* paged KV: ceil(L_b / page_size) pages per request, drawn as a random
  permutation of the page pool (identity order for the contiguous workload).

Every tensor has its own seed: ``seed = 1_000_000*workload + 100*cell + tag``.
"""
from __future__ import annotations

import dataclasses
import itertools
import math

import numpy as np
import torch

# tensor tags used in the seed formula
TAG_CTX, TAG_PAGES, TAG_Q, TAG_K, TAG_V = 1, 2, 3, 4, 5
TAG_TARGET, TAG_NOISE, TAG_TOKENS, TAG_UNIFORM = 11, 12, 13, 14


@dataclasses.dataclass(frozen=True)
class Workload:
    """One serving-shaped configuration of the draft-and-verify step."""

    wid: int
    name: str
    batch: int
    n_draft: int
    vocab: int
    logit_dtype: str          # "f32" or "bf16"
    draft_sigma: float
    temperatures: tuple
    n_q_heads: int
    n_kv_heads: int
    head_dim: int
    ctx: tuple                # ("const", L) | ("uniform", lo, hi) | ("lognormal", median, log_sigma, lo, hi)
    page_size: int
    contiguous: bool = False
    cell: int = 0

    @property
    def max_ctx(self) -> int:
        kind = self.ctx[0]
        if kind == "const":
            return int(self.ctx[1])
        if kind == "uniform":
            return int(self.ctx[2])
        return int(self.ctx[4])

    @property
    def max_pages(self) -> int:
        return -(-self.max_ctx // self.page_size)

    def with_(self, **kw) -> "Workload":
        return dataclasses.replace(self, **kw)


WORKLOADS = {
    1: Workload(1, "b1-k4-v32000-f32-ctx512", batch=1, n_draft=4, vocab=32000,
                logit_dtype="f32", draft_sigma=1.0, temperatures=(1.0,),
                n_q_heads=32, n_kv_heads=8, head_dim=128, ctx=("const", 512),
                page_size=16, contiguous=True),
    2: Workload(2, "b8-k5-v128256-bf16-ctx1k-4k", batch=8, n_draft=5, vocab=128256,
                logit_dtype="bf16", draft_sigma=0.5, temperatures=(0.0, 0.7),
                n_q_heads=32, n_kv_heads=8, head_dim=128, ctx=("uniform", 1024, 4096),
                page_size=16),
    3: Workload(3, "b64-k4-v151936-bf16-ctxlognormal", batch=64, n_draft=4, vocab=151936,
                logit_dtype="bf16", draft_sigma=1.0, temperatures=(1.0,),
                n_q_heads=28, n_kv_heads=4, head_dim=128,
                ctx=("lognormal", 2048, 0.6, 512, 8192), page_size=16),
    4: Workload(4, "b256-k8-v128256-bf16-ctx2k-16k", batch=256, n_draft=8, vocab=128256,
                logit_dtype="bf16", draft_sigma=0.7, temperatures=(0.8,),
                n_q_heads=64, n_kv_heads=8, head_dim=128, ctx=("uniform", 2048, 16384),
                page_size=32),
}

SWEEP_SIGMAS = (0.1, 0.5, 1.0, 2.0, 4.0)
SWEEP_KS = (1, 2, 4, 8, 16)
SWEEP_BATCHES = (1, 8, 64, 256, 512)
SWEEP_VOCABS = (32000, 128256, 256000)
SWEEP_TEMPERATURE = 1.0   # the sweep states no temperature; 1.0 is the reading taken here


def sweep_accept_cells():
    """The 375 acceptance cells of the sweep: sigma x k x B x V."""
    cell = 0
    for sigma, k, b, v in itertools.product(SWEEP_SIGMAS, SWEEP_KS, SWEEP_BATCHES, SWEEP_VOCABS):
        yield Workload(5, f"sweep-s{sigma}-k{k}-b{b}-v{v}", batch=b, n_draft=k, vocab=v,
                       logit_dtype="bf16", draft_sigma=sigma,
                       temperatures=(SWEEP_TEMPERATURE,), n_q_heads=32, n_kv_heads=8,
                       head_dim=128, ctx=("const", 4096), page_size=16, cell=cell)
        cell += 1


def sweep_attention_cells():
    """The 25 attention cells of the sweep: k x B at context 4096."""
    cell = 1000
    for k, b in itertools.product(SWEEP_KS, SWEEP_BATCHES):
        yield Workload(5, f"sweep-attn-k{k}-b{b}", batch=b, n_draft=k, vocab=32000,
                       logit_dtype="bf16", draft_sigma=1.0, temperatures=(1.0,),
                       n_q_heads=32, n_kv_heads=8, head_dim=128, ctx=("const", 4096),
                       page_size=16, cell=cell)
        cell += 1


def seed_of(w: Workload, tag: int) -> int:
    return 1_000_000 * w.wid + 100 * w.cell + tag


def _gen(device, seed: int) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(seed)
    return g


def context_lengths(w: Workload, device="cpu") -> torch.Tensor:
    """int32 [B] context lengths L_b (each counts the k+1 verify positions)."""
    g = _gen("cpu", seed_of(w, TAG_CTX))
    kind = w.ctx[0]
    if kind == "const":
        lens = torch.full((w.batch,), int(w.ctx[1]), dtype=torch.int64)
    elif kind == "uniform":
        lens = torch.randint(int(w.ctx[1]), int(w.ctx[2]) + 1, (w.batch,), generator=g)
    elif kind == "lognormal":
        median, log_sigma, lo, hi = w.ctx[1:]
        z = torch.randn((w.batch,), generator=g, dtype=torch.float64)
        lens = torch.exp(math.log(median) + log_sigma * z).round().to(torch.int64).clamp(lo, hi)
    else:
        raise ValueError(kind)
    lens = lens.clamp(min=w.n_draft + 1)
    return lens.to(torch.int32).to(device)


def _randn_bf16(shape, device, seed: int, chunk_elems: int = 1 << 28) -> torch.Tensor:
    """N(0,1) bf16 tensor, generated in chunks so that no large fp32 temporary exists."""
    out = torch.empty(shape, dtype=torch.bfloat16, device=device)
    flat = out.view(-1)
    g = _gen(device, seed)
    for s in range(0, flat.numel(), chunk_elems):
        flat[s:s + chunk_elems].normal_(generator=g)
    return out


def attention_inputs(w: Workload, device="cpu", ctx_lens: torch.Tensor | None = None) -> dict:
    """Q, paged K/V pools, page table and context lengths for one workload.

    Layouts: q [B, k+1, Hq, D]; k_pages / v_pages [P, Hkv, ps, D];
    page_table [B, max_pages] int32 (unused slots -1); ctx_lens [B] int32.
    """
    lens = context_lengths(w) if ctx_lens is None else ctx_lens.to("cpu", torch.int32)
    ps = w.page_size
    n_pages = [(-(-int(L) // ps)) for L in lens.tolist()]
    P = int(sum(n_pages))
    max_pages = max(w.max_pages, max(n_pages) if n_pages else 1)
    if w.contiguous:
        perm = torch.arange(P, dtype=torch.int64)
    else:
        perm = torch.randperm(P, generator=_gen("cpu", seed_of(w, TAG_PAGES)))
    table = torch.full((w.batch, max_pages), -1, dtype=torch.int32)
    off = 0
    for b, n in enumerate(n_pages):
        table[b, :n] = perm[off:off + n].to(torch.int32)
        off += n
    rows = w.n_draft + 1
    q = _randn_bf16((w.batch, rows, w.n_q_heads, w.head_dim), device, seed_of(w, TAG_Q))
    kp = _randn_bf16((P, w.n_kv_heads, ps, w.head_dim), device, seed_of(w, TAG_K))
    vp = _randn_bf16((P, w.n_kv_heads, ps, w.head_dim), device, seed_of(w, TAG_V))
    return dict(q=q, k_pages=kp, v_pages=vp, page_table=table.to(device),
                ctx_lens=lens.to(device), n_draft=w.n_draft)


def _logit_torch_dtype(w: Workload):
    return torch.float32 if w.logit_dtype == "f32" else torch.bfloat16


def accept_inputs(w: Workload, temperature: float, device="cpu", sigma: float | None = None,
                  chunk_rows: int = 2048) -> dict:
    """Target / draft logits, draft tokens and uniforms for one workload.

    Layouts: target [B, k+1, V]; draft [B, k, V] (same dtype);
    draft_tokens [B, k] int32; uniforms [B, k+1] fp32.
    """
    sigma = w.draft_sigma if sigma is None else sigma
    B, k, V = w.batch, w.n_draft, w.vocab
    dt = _logit_torch_dtype(w)
    target = torch.empty((B, k + 1, V), dtype=dt, device=device)
    draft = torch.empty((B, k, V), dtype=dt, device=device)
    tokens = torch.empty((B, k), dtype=torch.int32, device=device)
    g_t = _gen(device, seed_of(w, TAG_TARGET))
    g_n = _gen(device, seed_of(w, TAG_NOISE))
    g_x = _gen(device, seed_of(w, TAG_TOKENS))
    # whole requests per chunk, so that each chunk is a few hundred MB at most
    per = max(1, chunk_rows // (k + 1))
    for b0 in range(0, B, per):
        b1 = min(B, b0 + per)
        zt = torch.randn((b1 - b0, k + 1, V), generator=g_t, device=device,
                         dtype=torch.float32).mul_(3.0)
        target[b0:b1] = zt.to(dt)
        zd = target[b0:b1, :k].float()
        zd.add_(torch.randn(zd.shape, generator=g_n, device=device, dtype=torch.float32), alpha=sigma)
        draft[b0:b1] = zd.to(dt)
        zd = draft[b0:b1].float()
        if temperature > 0:
            # Gumbel-max: argmax(z/T + G) with G = -log(-log(U)) samples softmax(z/T)
            uu = torch.rand(zd.shape, generator=g_x, device=device, dtype=torch.float32)
            uu.clamp_(min=1e-12, max=1.0 - 1e-7)
            zd.div_(temperature).sub_(uu.log_().neg_().log_())
        tokens[b0:b1] = torch.argmax(zd, dim=-1).to(torch.int32)
        del zt, zd
    uniforms = torch.rand((B, k + 1), generator=_gen(device, seed_of(w, TAG_UNIFORM)),
                          device=device, dtype=torch.float32)
    return dict(target=target, draft=draft, draft_tokens=tokens, uniforms=uniforms)


# ---------------------------------------------------------------------------
# host copies and request subsets (plumbing for comparisons at full sizes)
# ---------------------------------------------------------------------------

def host_bits(t: torch.Tensor) -> np.ndarray:
    """numpy copy of a tensor; bf16 becomes its uint16 bit patterns."""
    t = t.detach().contiguous()
    if t.dtype == torch.bfloat16:
        return t.view(torch.int16).cpu().numpy().view(np.uint16)
    return t.cpu().numpy()


def attention_subset(inp: dict, idx) -> dict:
    """The requests ``idx`` of an attention input, with only their pages, renumbered."""
    idx = torch.as_tensor(list(idx), dtype=torch.int64)
    dev = inp["q"].device
    table = inp["page_table"].cpu()[idx]
    lens = inp["ctx_lens"].cpu()[idx]
    ps = inp["k_pages"].shape[2]
    used = []
    new_table = torch.full_like(table, -1)
    for r in range(table.shape[0]):
        n = -(-int(lens[r]) // ps)
        for j in range(n):
            new_table[r, j] = len(used)
            used.append(int(table[r, j]))
    used_t = torch.as_tensor(used, dtype=torch.int64, device=dev)
    return dict(q=inp["q"][idx.to(dev)].contiguous(),
                k_pages=inp["k_pages"][used_t].contiguous(),
                v_pages=inp["v_pages"][used_t].contiguous(),
                page_table=new_table.to(dev), ctx_lens=lens.to(dev),
                n_draft=inp["n_draft"])


def accept_subset(inp: dict, idx) -> dict:
    idx = torch.as_tensor(list(idx), dtype=torch.int64, device=inp["target"].device)
    return {k: v[idx].contiguous() for k, v in inp.items()}


# --------------------------------------------------------------------------
# routing (the front end's semantic matching): synthetic embeddings
# --------------------------------------------------------------------------
ROUTE_TAU = 0.85   # the paper's semantic matching threshold


@dataclasses.dataclass(frozen=True)
class RouteWorkload:
    wid: int
    name: str
    batch: int          # requests per routing call
    n_groups: int       # existing request groups (centroids)
    dim: int = 384      # all-MiniLM-L6-v2 embedding width
    hit_fraction: float = 0.7


ROUTE_WORKLOADS = {
    1: RouteWorkload(1, "route-b64-g1000-d384", 64, 1000),
    2: RouteWorkload(2, "route-b1024-g16384-d384", 1024, 16384),
    3: RouteWorkload(3, "route-b4096-g100000-d384", 4096, 100000),
}


def route_inputs(w: RouteWorkload, device="cpu", seed: int | None = None) -> dict:
    """Centroids with random directions and scales; a `hit_fraction` of the
    requests are a centroid's direction plus isotropic noise of a spread that
    puts their cosine with it around the 0.85 threshold (about 0.75-0.93),
    the rest are random directions; request scales vary too.  bf16."""
    g = torch.Generator().manual_seed(seed if seed is not None else 7_000_000 + 1000 * w.wid)
    d, N, B = w.dim, w.n_groups, w.batch
    cent = torch.randn(N, d, generator=g) * (0.5 + 1.5 * torch.rand(N, 1, generator=g))
    hit = torch.rand(B, generator=g) < w.hit_fraction
    pick = torch.randint(0, max(N, 1), (B,), generator=g)
    sigma = 0.02 + 0.025 * torch.rand(B, 1, generator=g)
    unit = cent / cent.norm(dim=1, keepdim=True).clamp_min(1e-30) if N else torch.zeros(1, d)
    near = unit[pick] + sigma * torch.randn(B, d, generator=g)
    far = torch.randn(B, d, generator=g) / math.sqrt(d)
    emb = torch.where(hit[:, None], near, far) * (0.3 + 3.0 * torch.rand(B, 1, generator=g))
    return dict(emb=emb.to(torch.bfloat16).to(device), centroids=cent.to(torch.bfloat16).to(device))


# --------------------------------------------------------------------------
# token trees (multi-candidate verification): a static draft tree per
# workload, the same shape for every request, nodes in breadth-first order
# --------------------------------------------------------------------------

@dataclasses.dataclass(frozen=True)
class TreeWorkload:
    """A draft tree of `branching[d]` children per node at depth d, verified in
    one target pass; the attention geometry and logits of a serving workload."""

    wid: int
    name: str
    batch: int
    branching: tuple
    vocab: int
    logit_dtype: str
    draft_sigma: float
    temperatures: tuple
    n_q_heads: int
    n_kv_heads: int
    head_dim: int
    ctx: tuple
    page_size: int
    cell: int = 0

    @property
    def n_nodes(self) -> int:
        return len(tree_parents(self.branching))

    def chain_workload(self) -> Workload:
        """A chain-workload view with n_draft = nodes - 1 (for the shared generators)."""
        return Workload(self.wid, self.name, self.batch, self.n_nodes - 1, self.vocab, self.logit_dtype,
                        self.draft_sigma, self.temperatures, self.n_q_heads, self.n_kv_heads, self.head_dim,
                        self.ctx, self.page_size, cell=self.cell)


def tree_parents(branching) -> list:
    """Parent array of the tree with branching[d] children per node at depth d
    (breadth-first order; node 0, the root, has parent -1)."""
    parents = [-1]
    level = [0]
    for fan in branching:
        nxt = []
        for u in level:
            for _ in range(int(fan)):
                parents.append(u)
                nxt.append(len(parents) - 1)
        level = nxt
    return parents


TREE_WORKLOADS = {
    # the attention geometry and logits of the B = 8 serving workload, with a
    # 34-node tree (3, 2, 2, 1) in place of the 5-token chain
    2: TreeWorkload(12, "tree-b8-n34-v128256-bf16-ctx1k-4k", batch=8, branching=(3, 2, 2, 1), vocab=128256,
                    logit_dtype="bf16", draft_sigma=0.5, temperatures=(0.0, 0.7), n_q_heads=32, n_kv_heads=8,
                    head_dim=128, ctx=("uniform", 1024, 4096), page_size=16),
}


def tree_attention_inputs(w: TreeWorkload, device="cpu") -> dict:
    """q [B, n, Hq, D], paged K/V pools, page table, context lengths (counting the
    n tree positions) and parents [B, n] int32 for a tree workload."""
    inp = attention_inputs(w.chain_workload(), device)
    par = torch.tensor(tree_parents(w.branching), dtype=torch.int32)
    inp["parents"] = par.repeat(w.batch, 1).to(device)
    inp.pop("n_draft")
    return inp


def tree_accept_inputs(w: TreeWorkload, temperature: float, device="cpu") -> dict:
    """Target and draft logits [B, n, V] (target ~ N(0, 3^2), draft = target +
    N(0, sigma^2), rounded to the logit dtype), node tokens [B, n] and uniforms
    [B, n].  The children of a node are independent draws from the node's
    draft distribution softmax(draft / T) (Gumbel-max); at T == 0 they are the
    node's top draft tokens, best first."""
    par = tree_parents(w.branching)
    n, B, V = len(par), w.batch, w.vocab
    dt = _logit_torch_dtype(w)
    g_t = _gen(device, seed_of(w.chain_workload(), TAG_TARGET))
    g_n = _gen(device, seed_of(w.chain_workload(), TAG_NOISE))
    g_x = _gen(device, seed_of(w.chain_workload(), TAG_TOKENS))
    target = (torch.randn((B, n, V), generator=g_t, device=device, dtype=torch.float32) * 3.0).to(dt)
    zd = target.float() + w.draft_sigma * torch.randn((B, n, V), generator=g_n, device=device,
                                                      dtype=torch.float32)
    draft = zd.to(dt)
    tokens = torch.zeros((B, n), dtype=torch.int32, device=device)
    children = {}
    for c in range(1, n):
        children.setdefault(par[c], []).append(c)
    for u, kids in children.items():
        z = draft[:, u].float()
        if temperature > 0:
            uu = torch.rand((B, len(kids), V), generator=g_x, device=device, dtype=torch.float32)
            uu.clamp_(min=1e-12, max=1.0 - 1e-7)
            pick = torch.argmax(z[:, None, :] / temperature - uu.log_().neg_().log_(), dim=-1)
        else:
            pick = torch.topk(z, len(kids), dim=-1).indices
        tokens[:, kids] = pick.to(torch.int32)
    uniforms = torch.rand((B, n), generator=_gen(device, seed_of(w.chain_workload(), TAG_UNIFORM)),
                          device=device, dtype=torch.float32)
    return dict(target=target, draft=draft, parents=torch.tensor(par, dtype=torch.int32,
                                                                 device=device).repeat(B, 1),
                node_tokens=tokens, uniforms=uniforms)
