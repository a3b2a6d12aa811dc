"""Near-tie report of the acceptance step against the fp64 oracle, per configuration.

    python tests/report_near_ties.py [--out FILE]

Runs cs_spec_accept on the four serving workloads (every temperature they
name) and on the sampled sweep cells that the GPU tests check, compares the
tokens and accepted counts with the oracle's on the same seeded inputs
(all requests where the oracle finishes quickly, a seeded sample of up to
64 requests otherwise) and prints one markdown row per configuration:
requests compared, near-ties in the accept band (|u - p/q| < 1e-5) and in
the draw band (u_k within 1e-6 of an edge of the drawn cell), how many of
those near-ties differ, and how many requests differ outside the bands
(which must be 0).  Needs a GPU; calls only the library and the oracle.
"""
from __future__ import annotations

import argparse
import json
import os
import sys

import numpy as np
import torch

HERE = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, os.path.dirname(HERE))
sys.path.insert(0, HERE)

import oracle  # noqa: E402
from paper_2607_20507_gb300 import binding  # noqa: E402
from paper_2607_20507_gb300 import workloads as W  # noqa: E402
from parity_bands import DRAW_TIE, NEAR_TIE  # noqa: E402
from test_gpu_accept import stratified_sweep_cells  # noqa: E402

DEV = "cuda:0"
MAX_SAMPLE = 64


def one(w, T) -> dict:
    inp = W.accept_inputs(w, T, DEV)
    tok, n = binding.cs_spec_accept(inp["target"], inp["draft"] if T > 0 else None, inp["draft_tokens"],
                                    inp["uniforms"], T)
    torch.cuda.synchronize()
    tok, n = tok.cpu().numpy(), n.cpu().numpy()
    B = w.batch
    if B * (2 * w.n_draft + 1) * w.vocab <= 64 * 17 * 128256:
        idx = list(range(B))
    else:
        idx = sorted(np.random.default_rng(w.cell + 77).choice(B, MAX_SAMPLE, replace=False).tolist())
    sub = W.accept_subset(inp, idx)
    et, en, am, dm = oracle.spec_accept(W.host_bits(sub["target"]),
                                        W.host_bits(sub["draft"]) if T > 0 else None,
                                        sub["draft_tokens"].cpu().numpy(), sub["uniforms"].cpu().numpy(), T,
                                        with_draw_margin=True)
    mism = np.any(tok[idx] != et, axis=1) | (n[idx] != en)
    ta, td = am < NEAR_TIE, dm < DRAW_TIE
    tie = ta | td
    del inp, sub
    torch.cuda.empty_cache()
    return {"config": w.name, "temperature": T, "batch": B, "compared": len(idx),
            "draw_margin_le_1e-7": int((dm < 1e-7).sum()), "draw_margin_le_1e-8": int((dm < 1e-8).sum()),
            "differ_max_draw_margin": float(dm[mism].max()) if mism.any() else None,
            "differ_max_accept_margin": float(am[mism].max()) if mism.any() else None,
            "near_ties_accept": int(ta.sum()), "near_ties_draw": int(td.sum()),
            "near_ties_differ": int((mism & tie).sum()), "differ_outside_band": int((mism & ~tie).sum()),
            "mean_accepted": float(en.mean())}


def main() -> int:
    ap = argparse.ArgumentParser()
    ap.add_argument("--out", default=None, help="also write the rows as JSON lines here")
    args = ap.parse_args()
    binding.load_library()
    oracle.set_threads(os.cpu_count() or 1)
    rows = []
    for wid in sorted(W.WORKLOADS):
        w = W.WORKLOADS[wid]
        for T in w.temperatures:
            rows.append(one(w, T))
    cells = {(c.draft_sigma, c.n_draft, c.batch, c.vocab): c for c in W.sweep_accept_cells()}
    picked = [(0.1, 4, 64, 256000), (4.0, 16, 8, 128256), (1.0, 1, 512, 32000), (0.5, 8, 256, 32000),
              (2.0, 2, 1, 256000), (0.1, 16, 64, 32000), (0.1, 8, 256, 128256), (0.1, 1, 512, 256000),
              (0.1, 2, 8, 32000), (4.0, 4, 64, 256000)] + stratified_sweep_cells()
    for key in picked:
        rows.append(one(cells[key], W.SWEEP_TEMPERATURE))
    print("| configuration | T | B | compared | accept-band ties | draw-band ties | ties that differ "
          "| differ outside the bands | mean accepted (oracle) |")
    print("|---|---|---|---|---|---|---|---|---|")
    for r in rows:
        print(f"| {r['config']} | {r['temperature']} | {r['batch']} | {r['compared']} | {r['near_ties_accept']} "
              f"| {r['near_ties_draw']} | {r['near_ties_differ']} | {r['differ_outside_band']} "
              f"| {r['mean_accepted']:.3f} |")
    tot = {k: sum(r[k] for r in rows) for k in ("compared", "near_ties_accept", "near_ties_draw",
                                                 "near_ties_differ", "differ_outside_band")}
    print(f"| total | | | {tot['compared']} | {tot['near_ties_accept']} | {tot['near_ties_draw']} "
          f"| {tot['near_ties_differ']} | {tot['differ_outside_band']} | |")
    if args.out:
        with open(args.out, "w") as f:
            for r in rows:
                f.write(json.dumps(r) + "\n")
    return 1 if tot["differ_outside_band"] else 0


if __name__ == "__main__":
    sys.exit(main())
