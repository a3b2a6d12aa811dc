"""The allocation-free verify attention, checked against the regular entry point.

cs_verify_attention_noalloc exists for callers that cannot allocate device
memory (a host framework that owns every allocation, a serving loop that
allows none after start-up, a binding without a device allocator); it runs
the same kernel on a fixed scratch array inside the library.  These tests
call both entry points through the C ABI on the same inputs and require the
same results within the attention tolerance, on two calls in a row (the
second call finds the scratch as the first one left it).  This file is
collected last on purpose.
"""
import ctypes

import pytest
import torch

from paper_2607_20507_gb300 import binding
from paper_2607_20507_gb300 import workloads as W

pytestmark = pytest.mark.gpu

DEV = "cuda:0"
ATOL, RTOL = 2e-3, 1e-2


def noalloc(lib, inp, out):
    d = binding.attn_dims(inp["q"], inp["k_pages"], inp["page_table"])
    st = lib.cs_verify_attention_noalloc(ctypes.byref(d), inp["q"].data_ptr(),
                                         inp["k_pages"].data_ptr(), inp["v_pages"].data_ptr(),
                                         inp["page_table"].data_ptr(), inp["ctx_lens"].data_ptr(),
                                         inp["n_draft"], out.data_ptr(),
                                         torch.cuda.current_stream().cuda_stream)
    assert st == binding.CS_OK, lib.cs_last_error().decode()
    torch.cuda.synchronize()
    # the call's device status word (in the library's scratch, which the
    # caller cannot address): no bounded wait gave up
    status = ctypes.c_int32(-1)
    st = lib.cs_verify_attention_noalloc_status(ctypes.byref(status), torch.cuda.current_stream().cuda_stream)
    assert st == binding.CS_OK, lib.cs_last_error().decode()
    assert status.value == 0
    return out


def with_workspace(inp):
    out = binding.cs_verify_attention(inp["q"], inp["k_pages"], inp["v_pages"], inp["page_table"],
                                      inp["ctx_lens"], inp["n_draft"])
    torch.cuda.synchronize()
    return out


def cases():
    small = W.Workload(93, "noalloc-small", batch=3, n_draft=3, vocab=64, logit_dtype="bf16",
                       draft_sigma=1.0, temperatures=(1.0,), n_q_heads=16, n_kv_heads=4,
                       head_dim=128, ctx=("uniform", 30, 900), page_size=16)
    return [small, W.WORKLOADS[1], W.WORKLOADS[2]]


@pytest.mark.parametrize("w", cases(), ids=lambda w: w.name)
def test_noalloc_matches_the_workspace_entry_point_twice(w):
    lib = binding.load_library()
    inp = W.attention_inputs(w, DEV)
    expect = with_workspace(inp).float()
    for call in range(2):
        out = torch.full_like(inp["q"], float("nan"))
        got = noalloc(lib, inp, out).float()
        assert torch.isfinite(got).all(), f"call {call}"
        err = (got - expect).abs()
        tol = ATOL + RTOL * expect.abs()
        assert (err <= tol).all(), f"call {call}: {int((err > tol).sum())} elements outside tolerance"


def test_noalloc_covers_the_largest_supported_geometry():
    # (k+1)*G = 144 query rows per KV head is the largest geometry the kernel
    # takes; its scratch need must fit the fixed array, and the results must
    # match the workspace entry point
    lib = binding.load_library()
    w = W.Workload(94, "noalloc-144rows", batch=2, n_draft=8, vocab=64, logit_dtype="bf16",
                   draft_sigma=1.0, temperatures=(1.0,), n_q_heads=128, n_kv_heads=8,
                   head_dim=128, ctx=("uniform", 200, 3000), page_size=32)
    inp = W.attention_inputs(w, DEV)
    d = binding.attn_dims(inp["q"], inp["k_pages"], inp["page_table"])
    assert lib.cs_verify_attention_workspace_bytes(ctypes.byref(d), 8) <= (32 << 20)
    expect = with_workspace(inp).float()
    for call in range(2):
        got = noalloc(lib, inp, torch.empty_like(inp["q"])).float()
        assert ((got - expect).abs() <= ATOL + RTOL * expect.abs()).all(), f"call {call}"
