#!/usr/bin/env python3
"""Benchmark of the draft-and-verify step on GB300.

One step = one pass of the whole hot path over one batch of synthetic input:
cs_verify_attention (one layer's verify attention over the paged KV cache)
followed by cs_spec_accept (the acceptance step at the workload's sampling
temperature).  The metric is verified draft tokens per second (B*k per step)
with the achieved HBM bandwidth of the dominant kernel against the measured
copy peak.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--workload 4] [--impl gb300|reference]

The headline workload is configuration 4 (B = 256, k = 8, V = 128256, 64 query
/ 8 KV heads, contexts 2K-16K, 32-token pages), the largest single-GPU
configuration; the other serving configurations are timed in the same run
and reported under ``per_workload``.

Under torchrun (N > 1) every rank runs an independent replica on its own GPU
with its own requests (the step shards by request; there is no collective on
the data path): value = requests*k over all ranks / max-over-ranks time.
``--impl reference`` times the fp64 CPU oracle on the host cores instead (a
deliberately slow baseline; rank 0 only).
"""
from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import statistics
import subprocess
import sys
import time

import numpy as np
import torch

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2607_20507_gb300 import workloads as W  # noqa: E402

METRIC = "verified draft tokens/sec and achieved HBM GB/s (fraction of ~8 TB/s) at 1 GB300"
UNIT = "verified draft tokens/s"
NOMINAL_HBM_GBS = 8000.0
FALLBACK_HBM_GBS = 6800.0
L2_FLUSH_BYTES = 512 << 20
ATT_ATOL, ATT_RTOL = 2e-3, 1e-2      # attention output tolerance against the oracle
NEAR_TIE_ACCEPT = 1e-5               # accept test: |u_i - p_i(x_i)/q_i(x_i)|
NEAR_TIE_DRAW = 1e-6                 # final draw: |u_k - C/Z| at an edge of the drawn cell
# the sources of each kernel pair whose DRAM traffic profiles/traffic.json records
KERNEL_SOURCES = {
    "verify_attention": ("paper_2607_20507_gb300/csrc/verify_attention.cu",
                         "paper_2607_20507_gb300/csrc/verify_attention_tc.cuh",
                         "paper_2607_20507_gb300/csrc/cs_device.cuh"),
    "spec_accept": ("paper_2607_20507_gb300/csrc/spec_accept.cu",
                    "paper_2607_20507_gb300/csrc/cs_device.cuh"),
}


# --------------------------------------------------------------------------
# helpers that need no GPU (covered by the CPU tests)
# --------------------------------------------------------------------------

def dist_env() -> tuple[int, int, int]:
    return (int(os.environ.get("RANK", "0")), int(os.environ.get("WORLD_SIZE", "1")),
            int(os.environ.get("LOCAL_RANK", "0")))


def replica_workload(w: W.Workload, rank: int) -> W.Workload:
    """Rank r's replica: same shapes, its own seeded requests."""
    return w if rank == 0 else w.with_(cell=w.cell + 7919 * rank)


def reduce_max(x: float, device) -> float:
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()):
        return x
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def aggregate_throughput(units_per_rank: float, seconds: float, world: int, device) -> tuple[float, float]:
    """(whole-job units/s, max-over-ranks seconds): every rank did `units_per_rank`."""
    t = reduce_max(seconds, device)
    return units_per_rank * world / t, t


def attention_bytes(ctx_lens: np.ndarray, w: W.Workload) -> int:
    """Algorithmic HBM bytes of one verify-attention call: every admissible K and
    V row once, Q read and out written once, the used page-table entries and
    the context lengths."""
    kv = int(ctx_lens.astype(np.int64).sum()) * 2 * w.n_kv_heads * w.head_dim * 2
    qo = 2 * w.batch * (w.n_draft + 1) * w.n_q_heads * w.head_dim * 2
    pages = int(np.ceil(ctx_lens / w.page_size).sum()) * 4
    return kv + qo + pages + 4 * w.batch


def attention_flops(ctx_lens: np.ndarray, w: W.Workload) -> int:
    k = w.n_draft
    keys = sum(int(L) * (k + 1) - k * (k + 1) // 2 for L in ctx_lens.tolist())
    return 4 * w.n_q_heads * w.head_dim * keys


def accept_bytes(n_accepted: np.ndarray, w: W.Workload, T: float) -> tuple[int, int]:
    """(bytes the method must read, bytes of every row) for one acceptance call.

    Sampling: target and draft rows 0..a, plus target row k when a == k.
    Greedy: target rows 0..a.  Rows after the first rejection cannot change
    the result.  Small per-request arrays (tokens, uniforms, outputs) added."""
    s = 4 if w.logit_dtype == "f32" else 2
    k, V, B = w.n_draft, w.vocab, w.batch
    a = n_accepted.astype(np.int64)
    if T > 0:
        rows = np.where(a < k, 2 * (a + 1), 2 * k + 1)
        full = B * (2 * k + 1)
    else:
        rows = a + 1
        full = B * (k + 1)
    small = B * k * 4 + B * (k + 1) * 4 + B * (k + 1) * 4 + B * 4
    return int(rows.sum()) * V * s + small, full * V * s + small


def measured_peaks() -> tuple[dict, str]:
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(p) as f:
            return json.load(f), "of measured"
    except Exception:
        return {"hbm_gbs": FALLBACK_HBM_GBS}, "of fallback"


def kernel_source_hash(kernel: str) -> str:
    h = hashlib.sha256()
    for rel in KERNEL_SOURCES[kernel]:
        with open(os.path.join(ROOT, rel), "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


def recorded_traffic(kernel: str, workload: str) -> int | None:
    """DRAM bytes per launch from the committed ncu summary, if it was taken on
    the current kernel sources; otherwise None."""
    p = os.path.join(ROOT, "profiles", "traffic.json")
    try:
        with open(p) as f:
            rec = json.load(f)
    except Exception:
        return None
    e = rec.get(kernel, {}).get(workload)
    if not e or e.get("source_hash") != kernel_source_hash(kernel):
        return None
    return int(e["dram_bytes_per_launch"])


def parse_clocks(lines: list[str]) -> dict:
    sm, mx, reasons = [], [], set()
    names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
    for ln in lines:
        f = [x.strip() for x in ln.split(",")]
        if len(f) < 9 or not f[1].replace(".", "").isdigit():
            continue
        sm.append(float(f[1]))
        mx.append(float(f[2]))
        for name, val in zip(names, f[5:9]):
            if val.lower() == "active":
                reasons.add(name)
    if not sm:
        return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
    return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
            "samples": len(sm)}


class ClockSampler:
    """nvidia-smi sampling of SM clock and throttle reasons while the GPU works."""

    QUERY = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index: int):
        self.proc = None
        self.lines: list[str] = []
        sel = []
        try:
            uuid = str(torch.cuda.get_device_properties(device_index).uuid)
            sel = ["-i", uuid if uuid.startswith("GPU-") else "GPU-" + uuid]
        except Exception:
            sel = []
        self.cmd = ["nvidia-smi", *sel, f"--query-gpu={self.QUERY}", "--format=csv,noheader,nounits",
                    "-lms", "100"]

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(self.cmd, stdout=subprocess.PIPE, stderr=subprocess.DEVNULL,
                                         text=True)
        except Exception:
            self.proc = None
        time.sleep(0.3)
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            time.sleep(0.25)
            self.proc.terminate()
            try:
                out, _ = self.proc.communicate(timeout=5)
                self.lines = out.splitlines()
            except Exception:
                self.proc.kill()
        return False

    def summary(self) -> dict:
        return parse_clocks(self.lines)


# --------------------------------------------------------------------------
# the GB300 arm
# --------------------------------------------------------------------------

def _events(n):
    return [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(n)]


def capture(fn):
    """fn run three times, then captured into a CUDA graph (host enqueue time
    -- Python, ctypes, tensor-map encoding -- stays out of the timed replays)."""
    for _ in range(3):
        fn()
    torch.cuda.synchronize()
    gr = torch.cuda.CUDAGraph()
    with torch.cuda.graph(gr):
        fn()
    torch.cuda.synchronize()
    return gr


def flushed_times(gr, steps, flush, stream) -> list[float]:
    """Seconds of `steps` replays of graph `gr`, the L2 flushed before each
    (outside the events)."""
    ev = _events(steps)
    for e0, e1 in ev:
        flush.zero_()
        e0.record(stream)
        gr.replay()
        e1.record(stream)
    torch.cuda.synchronize()
    return [e0.elapsed_time(e1) * 1e-3 for e0, e1 in ev]


def serving_calls(w, T, dev):
    """Inputs, output buffers and the two C-ABI calls of one workload's step."""
    from paper_2607_20507_gb300 import binding
    att = W.attention_inputs(w, dev)
    acc = W.accept_inputs(w, T, dev)
    k, B = w.n_draft, w.batch
    ws = binding.verify_attention_workspace(binding.attn_dims(att["q"], att["k_pages"], att["page_table"]),
                                            k, dev)
    bufs = {"out": torch.empty_like(att["q"]),
            "out_tok": torch.empty((B, k + 1), dtype=torch.int32, device=dev),
            "out_n": torch.empty((B,), dtype=torch.int32, device=dev)}

    def attention():
        binding.cs_verify_attention(att["q"], att["k_pages"], att["v_pages"], att["page_table"],
                                    att["ctx_lens"], k, out=bufs["out"], workspace=ws)

    def accept(inp=acc, temp=T):
        binding.cs_spec_accept(inp["target"], inp["draft"] if temp > 0 else None,
                               inp["draft_tokens"], inp["uniforms"], temp, bufs["out_tok"], bufs["out_n"])

    return att, acc, bufs, attention, accept


def kernel_figures(w, T, lens, n_acc, t_attn, t_acc, hbm_peak) -> dict:
    """Per-call time, algorithmic bytes and bandwidth of both calls of a step."""
    ab = attention_bytes(lens, w)
    acc_need, acc_full = accept_bytes(n_acc, w, T)
    m_attn, m_acc = statistics.mean(t_attn), statistics.mean(t_acc)
    return {
        "verify_attention": {"us": round(1e6 * m_attn, 2), "bytes": ab, "gbs": round(ab / m_attn / 1e9, 1),
                             "frac": round(ab / m_attn / 1e9 / hbm_peak, 4),
                             "frac_of_nominal_8tbs": round(ab / m_attn / 1e9 / NOMINAL_HBM_GBS, 4),
                             "tflops": round(attention_flops(lens, w) / m_attn / 1e12, 1)},
        # the acceptance kernels read every row once (all positions in parallel);
        # `needed_bytes` (rows 0..a) is what a rejection-ordered pass would touch
        "spec_accept": {"us": round(1e6 * m_acc, 2), "bytes": acc_full, "gbs": round(acc_full / m_acc / 1e9, 1),
                        "frac": round(acc_full / m_acc / 1e9 / hbm_peak, 4),
                        "frac_of_nominal_8tbs": round(acc_full / m_acc / 1e9 / NOMINAL_HBM_GBS, 4),
                        "needed_bytes": acc_need, "mean_accepted": round(float(n_acc.mean()), 4)},
    }


def other_workload(wid, steps, flush, stream, dev, hbm_peak) -> dict:
    """One serving workload besides the headline one: each call in its own
    graph, `steps` flushed replays each, and the step as one graph."""
    w = W.WORKLOADS[wid]
    T = max(w.temperatures)
    att, acc, bufs, attention, accept = serving_calls(w, T, dev)

    def step():
        attention()
        accept()

    g_a, g_c, g_s = capture(attention), capture(accept), capture(step)
    for _ in range(3):
        flush.zero_()
        g_s.replay()
    t_s = flushed_times(g_s, steps, flush, stream)
    t_a = flushed_times(g_a, steps, flush, stream)
    t_c = flushed_times(g_c, steps, flush, stream)
    lens = att["ctx_lens"].cpu().numpy()
    n_acc = bufs["out_n"].cpu().numpy()
    step_s = statistics.mean(t_s)
    res = {"temperature": T, "batch": w.batch, "n_draft": w.n_draft,
           "step_us": round(1e6 * step_s, 2),
           "verified_tokens_per_s": round(w.batch * w.n_draft / step_s, 1),
           "kernels": kernel_figures(w, T, lens, n_acc, t_a, t_c, hbm_peak)}
    if 0.0 in w.temperatures and T > 0:
        acc0 = W.accept_inputs(w, 0.0, dev)
        g0 = capture(lambda: accept(acc0, 0.0))
        t0 = flushed_times(g0, steps, flush, stream)
        ng = bufs["out_n"].cpu().numpy()
        res["greedy"] = kernel_figures(w, 0.0, lens, ng, t_a, t0, hbm_peak)["spec_accept"]
        del acc0, g0
    del att, acc, bufs, g_a, g_c, g_s
    torch.cuda.empty_cache()
    return res


def run_gb300(args) -> dict | None:
    import torch.distributed as dist
    from paper_2607_20507_gb300 import binding

    rank, world, local = dist_env()
    if world > 1:
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    binding.load_library()
    peaks, peak_src = measured_peaks()
    hbm_peak = float(peaks.get("hbm_gbs", FALLBACK_HBM_GBS))

    w = replica_workload(W.WORKLOADS[args.workload], rank)
    if args.batch:
        w = w.with_(batch=args.batch)
    T = args.temperature if args.temperature is not None else max(w.temperatures)
    att, acc, bufs, attention, accept = serving_calls(w, T, dev)
    k, B = w.n_draft, w.batch
    out, out_tok, out_n = bufs["out"], bufs["out_tok"], bufs["out_n"]
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream(dev)

    def step():
        attention()
        accept()

    # The step is captured once into a CUDA graph (both C-ABI calls, whose
    # kernels chain by programmatic dependent launch) and the timed steps
    # replay it.  Each call is also captured on its own, to time the two
    # calls' shares of the step.
    g_step, g_attn, g_acc = capture(step), capture(attention), capture(accept)

    # warm-up: at least W steps and about a second of work, with clocks sampled
    sampler = ClockSampler(local)
    with sampler:
        t0 = time.time()
        n = 0
        while n < args.warmup or time.time() - t0 < args.warmup_seconds:
            flush.zero_()
            g_step.replay()
            n += 1
            if n % 64 == 0:
                torch.cuda.synchronize()
        torch.cuda.synchronize()

        # timed region: exactly K steps, L2 flushed between steps (outside the events)
        evs = _events(args.steps)
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize()
        for e0, e1 in evs:
            flush.zero_()
            e0.record(stream)
            g_step.replay()
            e1.record(stream)
        torch.cuda.synchronize()
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize()
        # the two calls' shares: the same K steps with one graph per call
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True),
               torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]
        for e0, e1, e2 in ev:
            flush.zero_()
            e0.record(stream)
            g_attn.replay()
            e1.record(stream)
            g_acc.replay()
            e2.record(stream)
        torch.cuda.synchronize()
    # the same K steps through the direct API calls (host enqueue on the path)
    evd = _events(args.steps)
    for e0, e1 in evd:
        flush.zero_()
        e0.record(stream)
        step()
        e1.record(stream)
    torch.cuda.synchronize()
    direct_us = 1e6 * statistics.mean(e0.elapsed_time(e1) * 1e-3 for e0, e1 in evd)
    t_attn = [e0.elapsed_time(e1) * 1e-3 for e0, e1, _ in ev]
    t_acc = [e1.elapsed_time(e2) * 1e-3 for _, e1, e2 in ev]
    t_step = [e0.elapsed_time(e1) * 1e-3 for e0, e1 in evs]
    value, t_max = aggregate_throughput(float(B * k * args.steps), sum(t_step), world, dev)
    n_acc = out_n.cpu().numpy()
    lens = att["ctx_lens"].cpu().numpy()
    kernels = kernel_figures(w, T, lens, n_acc, t_attn, t_acc, hbm_peak)

    # hot-L2 times of the small workloads (inputs stay in the 129 MB L2)
    hot_l2 = None
    if w.wid in (1, 2):
        def hot_mean_us(gr):
            for _ in range(3):
                gr.replay()
            torch.cuda.synchronize()
            evh = _events(args.steps)
            for e0, e1 in evh:
                e0.record(stream)
                gr.replay()
                e1.record(stream)
            torch.cuda.synchronize()
            return 1e3 * statistics.mean(e0.elapsed_time(e1) for e0, e1 in evh)
        hot_l2 = {"step_us": round(hot_mean_us(g_step), 2), "attention_us": round(hot_mean_us(g_attn), 2),
                  "accept_us": round(hot_mean_us(g_acc), 2),
                  "note": "no L2 flush between replays: the inputs stay L2-resident; not the headline"}

    # the next rows of the path at the headline workload's shape: the KV
    # append of the k+1 verify rows and one drafter sampling step
    def timed_graph(fn):
        return statistics.mean(flushed_times(capture(fn), args.steps, flush, stream))

    # the append writes back the rows the pool already holds at the k+1
    # verify positions (the same bytes move; the pool, which the parity
    # sample below reads, stays as the timed steps saw it)
    Hkv_ = att["k_pages"].shape[1]
    pos = att["ctx_lens"].long()[:, None] - (k + 1) + torch.arange(k + 1, device=dev)[None, :]
    pg = att["page_table"].long().gather(1, pos // w.page_size)
    new_k = att["k_pages"][pg, :, pos % w.page_size, :].contiguous()
    new_v = att["v_pages"][pg, :, pos % w.page_size, :].contiguous()
    t_app = timed_graph(lambda: binding.cs_kv_append(new_k, new_v, att["k_pages"], att["v_pages"],
                                                     att["page_table"], att["ctx_lens"]))
    app_bytes = 2 * 2 * new_k.numel() * 2            # K and V, read the new rows and write the slots
    d_logits = acc["draft"][:, 0].contiguous() if acc["draft"] is not None else acc["target"][:, 0].contiguous()
    d_u = acc["uniforms"][:, 0].contiguous()
    d_out = torch.empty(B, dtype=torch.int32, device=dev)
    t_smp = timed_graph(lambda: binding.cs_sample(d_logits, d_u, T if T > 0 else 0.7, d_out))
    smp_bytes = d_logits.numel() * d_logits.element_size()
    next_rows = {"kv_append": {"us": round(1e6 * t_app, 2), "bytes": app_bytes,
                               "gbs": round(app_bytes / t_app / 1e9, 1), "rows": int(B * (k + 1) * Hkv_)},
                 "draft_sample": {"us": round(1e6 * t_smp, 2), "bytes": smp_bytes,
                                  "gbs": round(smp_bytes / t_smp / 1e9, 1), "rows": B,
                                  "vocab": int(d_logits.shape[1])}}
    del new_k, new_v, d_logits, d_u, d_out
    # the front end's semantic routing (one batch of request embeddings
    # against the group centroids), at two group-index sizes
    for rw in (W.ROUTE_WORKLOADS[2], W.ROUTE_WORKLOADS[3]):
        rx = W.route_inputs(rw, dev)
        r_inv = binding.cs_route_norms(rx["centroids"])
        r_out = [torch.empty(rw.batch, dtype=dt, device=dev) for dt in (torch.int32, torch.int32, torch.float32)]
        t_rt = timed_graph(lambda: binding.cs_route(rx["emb"], rx["centroids"], r_inv, W.ROUTE_TAU, *r_out))
        flops = 2.0 * rw.batch * rw.n_groups * rw.dim
        r_bytes = (rw.batch + rw.n_groups) * rw.dim * 2 + rw.n_groups * 4 + rw.batch * 12
        next_rows[f"route_b{rw.batch}_g{rw.n_groups}"] = {
            "us": round(1e6 * t_rt, 2), "tflops": round(flops / t_rt / 1e12, 1), "flops": flops, "bytes": r_bytes,
            "frac_of_bf16_peak": round(flops / t_rt / 1e12 / float(peaks.get("bf16_tflops", 1900.0)), 4),
            "hit_rate": float((r_out[0] >= 0).float().mean().item())}
        del rx, r_inv, r_out
    # token-tree verification at the B = 8 workload's attention geometry and
    # vocabulary: tree attention over the paged cache and the acceptance walk
    tw = W.TREE_WORKLOADS[2]
    ta = W.tree_attention_inputs(tw, dev)
    t_out = torch.empty_like(ta["q"])
    t_tat = timed_graph(lambda: binding.cs_tree_verify_attention(ta["q"], ta["k_pages"], ta["v_pages"],
                                                                 ta["page_table"], ta["ctx_lens"], ta["parents"],
                                                                 out=t_out))
    tlens = ta["ctx_lens"].cpu().numpy()
    tat_bytes = attention_bytes(tlens, tw.chain_workload())
    T_tree = max(tw.temperatures)
    tc = W.tree_accept_inputs(tw, T_tree, dev)
    t_bufs = [torch.empty((tw.batch, tw.n_nodes), dtype=torch.int32, device=dev) for _ in range(2)]
    t_na = torch.empty((tw.batch,), dtype=torch.int32, device=dev)
    t_tac = timed_graph(lambda: binding.cs_tree_accept(tc["target"], tc["draft"], tc["parents"], tc["node_tokens"],
                                                       tc["uniforms"], T_tree, *t_bufs, t_na))
    par = W.tree_parents(tw.branching)
    internal = len(set(u for u in par[1:]))
    s_log = 4 if tw.logit_dtype == "f32" else 2
    tac_bytes = tw.batch * (tw.n_nodes + internal) * tw.vocab * s_log
    next_rows[f"tree_{tw.name}"] = {
        "nodes": tw.n_nodes, "branching": list(tw.branching), "temperature": T_tree,
        "attention_us": round(1e6 * t_tat, 2), "attention_bytes": tat_bytes,
        "attention_gbs": round(tat_bytes / t_tat / 1e9, 1),
        "attention_frac": round(tat_bytes / t_tat / 1e9 / hbm_peak, 4),
        "accept_us": round(1e6 * t_tac, 2), "accept_bytes": tac_bytes,
        "accept_gbs": round(tac_bytes / t_tac / 1e9, 1),
        "mean_accepted": float(t_na.float().mean().item())}
    del ta, tc, t_out, t_bufs

    # end to end through the public API.  Every step's inputs -- the query
    # rows, the page table and context lengths, both logit tensors, the draft
    # tokens and the uniforms -- are copied from pinned host memory, and the
    # emitted tokens and counts are read back.  The paged KV cache stays
    # resident on the device (serving state that earlier steps wrote, not a
    # per-step input).
    step_inputs = {"q": att["q"], "page_table": att["page_table"], "ctx_lens": att["ctx_lens"],
                   "target": acc["target"], "draft_tokens": acc["draft_tokens"], "uniforms": acc["uniforms"]}
    if T > 0:
        step_inputs["draft"] = acc["draft"]
    host = {name: t.cpu().pin_memory() for name, t in step_inputs.items()}
    h2d = sum(t.numel() * t.element_size() for t in host.values())
    res_host = (torch.empty((B, k + 1), dtype=torch.int32).pin_memory(),
                torch.empty((B,), dtype=torch.int32).pin_memory())
    d2h = sum(t.numel() * t.element_size() for t in res_host)

    def e2e_step():
        for name, t in host.items():
            step_inputs[name].copy_(t, non_blocking=True)
        step()
        res_host[0].copy_(out_tok, non_blocking=True)
        res_host[1].copy_(out_n, non_blocking=True)

    for _ in range(max(3, args.warmup)):
        e2e_step()
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    e_start, e_end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e_start.record(stream)
    for _ in range(args.steps):
        e2e_step()
    e_end.record(stream)
    torch.cuda.synchronize()
    e2e_s = e_start.elapsed_time(e_end) * 1e-3
    e2e_value, _ = aggregate_throughput(float(B * k * args.steps), e2e_s, world, dev)

    # the other serving workloads, each timed the same way (not the headline)
    per_workload = {}
    if not args.no_per_workload:
        for wid in sorted(W.WORKLOADS):
            if wid != w.wid:
                per_workload[W.WORKLOADS[wid].name] = other_workload(wid, args.steps, flush, stream, dev, hbm_peak)

    # roofline of the dominant kernel (the one with the larger share of the step)
    dom = "verify_attention" if kernels["verify_attention"]["us"] >= kernels["spec_accept"]["us"] else "spec_accept"
    achieved = kernels[dom]["bytes"] / (kernels[dom]["us"] * 1e-6) / 1e9
    roofline = {"kernel": dom, "bound": "hbm", "achieved": round(achieved, 1), "peak": hbm_peak,
                "unit": "GB/s", "frac": round(achieved / hbm_peak, 4), "peak_source": peak_src,
                "frac_of_nominal_8tbs": round(achieved / NOMINAL_HBM_GBS, 4),
                "traffic": recorded_traffic(dom, w.name),
                "algorithmic_bytes_per_launch": kernels[dom]["bytes"],
                "us_per_launch": kernels[dom]["us"]}

    result = None
    if rank == 0:
        cpu, parity = (None, None)
        if not args.no_cpu_baseline:
            cpu, parity = oracle_baseline(w, T, att, acc, out, out_tok, out_n,
                                          seconds_budget=args.cpu_seconds)
        result = {
            "metric": METRIC, "value": round(value, 1), "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": round(1e3 * t_max / args.steps, 5), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
            "dtype_detail": "bf16 tensor-core attention with fp32 softmax and accumulation; fp32 acceptance arithmetic",
            "data": "synthetic (seeded; shapes of the serving workload, no dataset or weights)",
            "config": {"workload": w.name, "batch_per_gpu": B, "n_draft": k, "vocab": w.vocab,
                       "logit_dtype": w.logit_dtype, "temperature": T, "draft_sigma": w.draft_sigma,
                       "n_q_heads": w.n_q_heads, "n_kv_heads": w.n_kv_heads, "head_dim": w.head_dim,
                       "page_size": w.page_size, "ctx": list(w.ctx), "mean_ctx": float(lens.mean()),
                       "l2": "flushed between steps (512 MiB memset outside the timed events)",
                       "parallelism": f"replicas x{world} (requests shard; no collective)"},
            "kernels": kernels,
            "emitted_tokens_per_s": round(float((n_acc + 1).sum()) * args.steps / t_max, 1),
            "per_workload": per_workload,
            "next_rows": next_rows,
            "launch": {"timed_steps": "CUDA-graph replay of one step (both C-ABI calls in one graph; "
                                      "kernels chained by programmatic dependent launch)",
                       "kernel_times": "each C-ABI call in its own graph, the same K steps",
                       "per_call_graphs_step_us": round(1e6 * statistics.mean(a + b for a, b in zip(t_attn, t_acc)), 2),
                       "direct_call_step_us": round(direct_us, 2)},
            "hot_l2": hot_l2,
            "roofline": roofline,
            "cpu_baseline": cpu,
            "parity_sample": parity,
            "e2e": {"value": round(e2e_value, 1), "unit": UNIT, "h2d_bytes_per_step": h2d,
                    "d2h_bytes_per_step": d2h, "ms_per_step": round(1e3 * e2e_s / args.steps, 4),
                    "note": "per step: host->device copy from pinned memory of the query rows, page table, "
                            "context lengths, target and draft logits, draft tokens and uniforms; the two "
                            "C-ABI calls; device->host read of the emitted tokens and counts.  The paged KV "
                            "cache stays resident on the device (serving state, not a per-step input)"},
            # per step: the verify-attention kernel and its split merge (one pair per
            # 1024-request slice), the acceptance statistics kernel and the draw
            # kernel (one launch per 65535 requests)
            "gpu_launches": args.steps * (2 * math.ceil(B / 1024) + 1 + math.ceil(B / 65535)),
            "clocks": sampler.summary() | {"window": f"warm-up (>= {args.warmup_seconds:g} s) and the timed steps"},
        }
    if world > 1:
        dist.barrier()
        dist.destroy_process_group()
    return result


def parity_counts(out_tok, out_n, e_tok, e_n, accept_margin, draw_margin) -> dict:
    """Acceptance parity of GPU outputs against the oracle's on the same
    requests: near-ties (accept tests with |u - p/q| < 1e-5, draws with u_k
    within 1e-6 of an edge of the drawn cell) are counted, and so are the
    requests that differ inside and outside those bands."""
    mism = np.any(out_tok != e_tok, axis=1) | (out_n != e_n)
    tie_a = accept_margin < NEAR_TIE_ACCEPT
    tie_d = draw_margin < NEAR_TIE_DRAW
    tie = tie_a | tie_d
    return {"requests": int(len(e_n)), "near_ties_accept": int(tie_a.sum()), "near_ties_draw": int(tie_d.sum()),
            "near_ties_differ": int((mism & tie).sum()), "differ_outside_band": int((mism & ~tie).sum())}


def oracle_baseline(w, T, att, acc, out, out_tok, out_n, seconds_budget=15.0) -> tuple[dict, dict]:
    """The fp64 oracle on the host cores over a bounded, seeded request sample
    of the workload: its throughput (the cpu_baseline), and the GPU outputs of
    the same requests compared with its results (attention element by
    element against 2e-3 + 1e-2|ref|; tokens and counts exactly, near-ties
    counted)."""
    import oracle
    cores = os.cpu_count() or 1
    oracle.set_threads(cores)
    B = w.batch
    g_out = out.float().cpu().numpy()
    g_tok, g_n = out_tok.cpu().numpy(), out_n.cpu().numpy()
    n = 1
    spent = 0.0
    done = 0
    rng = np.random.default_rng(0)
    order = rng.permutation(B)
    att_bad = att_n = 0
    worst = 0.0
    cmp_tok, cmp_n, cmp_am, cmp_dm, cmp_et, cmp_en = [], [], [], [], [], []
    passes = 0
    while spent < seconds_budget and (done < B or passes == 0):
        take = order[done:done + n].tolist()
        sa = W.attention_subset(att, take)
        sc = W.accept_subset(acc, take)
        a_host = (W.host_bits(sa["q"]), W.host_bits(sa["k_pages"]), W.host_bits(sa["v_pages"]),
                  sa["page_table"].cpu().numpy(), sa["ctx_lens"].cpu().numpy())
        c_host = (W.host_bits(sc["target"]), W.host_bits(sc["draft"]) if T > 0 else None,
                  sc["draft_tokens"].cpu().numpy(), sc["uniforms"].cpu().numpy())
        t0 = time.perf_counter()
        e_out = oracle.verify_attention(*a_host, w.n_draft)
        e_tok, e_n, am, dm = oracle.spec_accept(*c_host, T, with_draw_margin=True)
        spent += time.perf_counter() - t0
        err = np.abs(g_out[take] - e_out)
        tol = ATT_ATOL + ATT_RTOL * np.abs(e_out)
        att_bad += int((err > tol).sum()) + int((~np.isfinite(g_out[take])).sum())
        att_n += err.size
        worst = max(worst, float((err / tol).max()) if err.size else 0.0)
        cmp_tok.append(g_tok[take])
        cmp_n.append(g_n[take])
        cmp_et.append(e_tok)
        cmp_en.append(e_n)
        cmp_am.append(am)
        cmp_dm.append(dm)
        done += len(take)
        if done >= B:
            # a workload the oracle finishes quickly is repeated until about
            # ten seconds of CPU work are measured
            passes += 1
            if spent >= 10.0:
                break
            done = 0
            n = B
        else:
            n = min(2 * n, B - done)
    n_req = sum(len(x) for x in cmp_n)
    value = n_req * w.n_draft / spent
    what = (f"{passes} passes over all {B} requests" if passes else
            f"a seeded sample of {n_req} of {B} requests")
    cpu = {"value": round(value, 2), "unit": UNIT, "cores": cores, "kind": "oracle",
           "sample": f"{what} of {w.name} (attention + acceptance, fp64, "
                     f"OpenMP over requests/heads), {spent:.2f} s"}
    acc_par = parity_counts(np.concatenate(cmp_tok), np.concatenate(cmp_n), np.concatenate(cmp_et),
                            np.concatenate(cmp_en), np.concatenate(cmp_am), np.concatenate(cmp_dm))
    parity = {"sample": what,
              "verify_attention": {"requests": n_req, "elements": att_n, "outside_tolerance": att_bad,
                                   "worst_err_over_tol": round(worst, 4),
                                   "tolerance": "|gpu - oracle| <= 2e-3 + 1e-2|oracle|"},
              "spec_accept": acc_par | {"bands": "accept |u - p/q| < 1e-5; draw |u_k - C/Z| < 1e-6"}}
    return cpu, parity


# --------------------------------------------------------------------------
# the reference arm: the oracle as it stands, on the host cores
# --------------------------------------------------------------------------

def run_reference(args) -> dict | None:
    rank, world, _ = dist_env()
    if rank != 0:
        return None
    import oracle
    w = W.WORKLOADS[args.workload]
    T = args.temperature if args.temperature is not None else max(w.temperatures)
    cores = os.cpu_count() or 1
    oracle.set_threads(cores)
    # inputs drawn where the GPU arm draws them (the same seeded values; on a
    # host without a GPU, the CPU generators); only the sampled requests are
    # copied to the host, and the timing covers the oracle alone
    gen_dev = "cuda" if torch.cuda.is_available() else "cpu"
    att = W.attention_inputs(w, gen_dev)
    acc = W.accept_inputs(w, T, gen_dev)
    # each step is a bounded sample: as many requests as fit about 2 s of oracle work
    take = np.random.default_rng(0).permutation(w.batch).tolist()
    probe = W.attention_subset(att, take[:1])
    ph = (W.host_bits(probe["q"]), W.host_bits(probe["k_pages"]), W.host_bits(probe["v_pages"]),
          probe["page_table"].cpu().numpy(), probe["ctx_lens"].cpu().numpy())
    t0 = time.perf_counter()
    oracle.verify_attention(*ph, w.n_draft)
    per_req = max(time.perf_counter() - t0, 1e-4)
    n_req = max(1, min(w.batch, int(2.0 / per_req)))
    sa = W.attention_subset(att, take[:n_req])
    sc = W.accept_subset(acc, take[:n_req])
    a_host = (W.host_bits(sa["q"]), W.host_bits(sa["k_pages"]), W.host_bits(sa["v_pages"]),
              sa["page_table"].cpu().numpy(), sa["ctx_lens"].cpu().numpy())
    c_host = (W.host_bits(sc["target"]), W.host_bits(sc["draft"]) if T > 0 else None,
              sc["draft_tokens"].cpu().numpy(), sc["uniforms"].cpu().numpy())
    del att, acc

    def step():
        oracle.verify_attention(*a_host, w.n_draft)
        oracle.spec_accept(*c_host, T)

    for _ in range(max(3, args.warmup)):
        step()
    times = []
    for _ in range(args.steps):
        t0 = time.perf_counter()
        step()
        times.append(time.perf_counter() - t0)
    total = sum(times)
    value = n_req * w.n_draft * args.steps / total
    sample = (f"a seeded sample of {n_req} of {w.batch} requests of {w.name} per step (attention + acceptance, fp64, "
              f"OpenMP on {cores} host threads)")
    return {"impl": "reference", "metric": METRIC, "value": round(value, 3), "unit": UNIT,
            "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": round(1e3 * total / args.steps, 3), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic (seeded; shapes of the serving workload)",
            "config": {"workload": w.name, "batch_per_gpu": w.batch, "n_draft": w.n_draft,
                       "vocab": w.vocab, "temperature": T},
            "cpu_baseline": {"value": round(value, 3), "unit": UNIT, "cores": cores, "kind": "oracle",
                             "sample": sample},
            "e2e": {"value": round(value, 3), "unit": UNIT, "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}


def run_sweep(args) -> None:
    """The sweep's cells at B >= 64 (one JSON line each): verify attention over
    k x B at context 4096, and the acceptance over k x B x V at draft sigma
    1.0 (the sigma changes how many positions are accepted, not the bytes the
    kernels read).  Each cell: inputs generated on the device, the C-ABI call
    captured in a CUDA graph, 5 untimed replays, then the median of `steps`
    replays with the L2 flushed before each (outside the events)."""
    from paper_2607_20507_gb300 import binding
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    binding.load_library()
    stream = torch.cuda.current_stream(dev)
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=dev)
    peaks, peak_src = measured_peaks()
    hbm_peak = float(peaks.get("hbm_gbs", FALLBACK_HBM_GBS))

    def median_us(fn):
        for _ in range(3):
            fn()
        torch.cuda.synchronize()
        gr = torch.cuda.CUDAGraph()
        with torch.cuda.graph(gr):
            fn()
        for _ in range(5):
            flush.zero_()
            gr.replay()
        ts = []
        for _ in range(args.steps):
            flush.zero_()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            gr.replay()
            e1.record(stream)
            torch.cuda.synchronize()
            ts.append(e0.elapsed_time(e1) * 1e3)
        return statistics.median(ts)

    def line(kind, w, us, nbytes, extra):
        gbs = nbytes / us / 1e3
        print(json.dumps({"sweep": kind, "cell": w.name, "batch": w.batch, "n_draft": w.n_draft,
                          "vocab": w.vocab if kind == "spec_accept" else None, "us": round(us, 2),
                          "bytes": nbytes, "gbs": round(gbs, 1), "frac_of_8tbs": round(gbs / NOMINAL_HBM_GBS, 4),
                          "frac_of_peak": round(gbs / hbm_peak, 4), "peak_source": peak_src} | extra), flush=True)

    for w in W.sweep_attention_cells():
        if w.batch < 64:
            continue
        att = W.attention_inputs(w, dev)
        ws = binding.verify_attention_workspace(binding.attn_dims(att["q"], att["k_pages"], att["page_table"]),
                                                w.n_draft, dev)
        out = torch.empty_like(att["q"])
        us = median_us(lambda: binding.cs_verify_attention(att["q"], att["k_pages"], att["v_pages"],
                                                           att["page_table"], att["ctx_lens"], w.n_draft,
                                                           out=out, workspace=ws))
        line("verify_attention", w, us, attention_bytes(att["ctx_lens"].cpu().numpy(), w), {})
        del att, ws, out
        torch.cuda.empty_cache()
    for w in W.sweep_accept_cells():
        if w.batch < 64 or w.draft_sigma != 1.0:
            continue
        T = W.SWEEP_TEMPERATURE
        acc = W.accept_inputs(w, T, dev)
        ot = torch.empty((w.batch, w.n_draft + 1), dtype=torch.int32, device=dev)
        on = torch.empty((w.batch,), dtype=torch.int32, device=dev)
        us = median_us(lambda: binding.cs_spec_accept(acc["target"], acc["draft"], acc["draft_tokens"],
                                                      acc["uniforms"], T, ot, on))
        n_acc = on.cpu().numpy()
        line("spec_accept", w, us, accept_bytes(n_acc, w, T)[1], {"mean_accepted": float(n_acc.mean())})
        del acc, ot, on
        torch.cuda.empty_cache()


def main(argv=None) -> int:
    ap = argparse.ArgumentParser(description=__doc__.splitlines()[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--workload", type=int, default=4, choices=sorted(W.WORKLOADS),
                    help="the headline workload (default 4: B = 256, the largest single-GPU configuration)")
    ap.add_argument("--temperature", type=float, default=None)
    ap.add_argument("--batch", type=int, default=0,
                    help="override the workload's batch (smaller cases for profiling)")
    ap.add_argument("--impl", choices=["gb300", "reference"], default="gb300")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-per-workload", action="store_true",
                    help="skip timing the other serving workloads")
    ap.add_argument("--cpu-seconds", type=float, default=15.0,
                    help="budget of the oracle's request sample (cpu_baseline and parity_sample)")
    ap.add_argument("--warmup-seconds", type=float, default=1.0,
                    help="keep warming up (and sampling clocks) for at least this long")
    ap.add_argument("--sweep", action="store_true",
                    help="time the sweep's cells at B >= 64 instead (one JSON line per cell)")
    args = ap.parse_args(argv)
    args.warmup = max(3, args.warmup)
    args.steps = max(1, args.steps)
    if args.sweep:
        run_sweep(args)
        return 0
    res = run_reference(args) if args.impl == "reference" else run_gb300(args)
    if res is not None:
        print(json.dumps(res), flush=True)
    return 0


if __name__ == "__main__":
    sys.exit(main())
