"""Failure detection on the GPU without a fault: a bounded wait that runs out.

cs_selftest_wait_timeout runs the kernels' bounded mbarrier wait on a barrier
that nothing completes; the wait gives up after about one second and records
CS_DEVICE_WAIT_TIMEOUT in the status word, and the context stays usable."""
import time

import numpy as np
import pytest
import torch

import oracle
from paper_2607_20507_gb300 import binding
from paper_2607_20507_gb300 import workloads as W

pytestmark = pytest.mark.gpu
DEV = "cuda:0"


def test_bounded_wait_times_out_and_reports():
    ws = torch.zeros(64, dtype=torch.int32, device=DEV)
    assert binding.cs_read_device_status(ws) == 0
    t0 = time.time()
    binding.cs_selftest_wait_timeout(ws)
    status = binding.cs_read_device_status(ws)
    elapsed = time.time() - t0
    assert status == binding.CS_DEVICE_WAIT_TIMEOUT
    assert 0.5 < elapsed < 30.0                      # gave up after about a second
    assert torch.count_nonzero(ws[1:]).item() == 0   # nothing else touched


def test_context_usable_after_a_timeout():
    ws = torch.zeros(64, dtype=torch.int32, device=DEV)
    binding.cs_selftest_wait_timeout(ws)
    assert binding.cs_read_device_status(ws) == binding.CS_DEVICE_WAIT_TIMEOUT
    # the next call runs normally on the same context, reports no timeout and
    # matches the oracle
    w = W.WORKLOADS[2].with_(batch=2, ctx=("uniform", 100, 700))
    inp = W.attention_inputs(w, DEV)
    dims = binding.attn_dims(inp["q"], inp["k_pages"], inp["page_table"])
    aws = binding.verify_attention_workspace(dims, w.n_draft, DEV)
    out = binding.cs_verify_attention(inp["q"], inp["k_pages"], inp["v_pages"], inp["page_table"],
                                      inp["ctx_lens"], w.n_draft, workspace=aws)
    torch.cuda.synchronize()
    assert binding.cs_read_device_status(aws) == 0
    expect = oracle.verify_attention(W.host_bits(inp["q"]), W.host_bits(inp["k_pages"]),
                                     W.host_bits(inp["v_pages"]), inp["page_table"].cpu().numpy(),
                                     inp["ctx_lens"].cpu().numpy(), w.n_draft, 0.0)
    got = out.float().cpu().numpy().astype(np.float64)
    assert np.isfinite(got).all()
    assert (np.abs(got - expect) <= 2e-3 + 1e-2 * np.abs(expect)).all()
