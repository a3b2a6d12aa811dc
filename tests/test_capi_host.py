"""The C-ABI library on the host: it builds, loads, exports every symbol the
header declares, and rejects bad arguments before enqueuing anything.  No
call here reaches a kernel, so the file runs without a GPU."""
import ctypes
import os
import re

import pytest

from paper_2607_20507_gb300 import binding, build

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "cachespec.h")


@pytest.fixture(scope="module")
def lib():
    build.build()
    return binding.load_library()


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(cs_[a-z_]+)\s*\(", text)))


def test_header_declares_the_boundary():
    names = declared_functions()
    for must in ("cs_verify_attention", "cs_spec_accept", "cs_verify_attention_workspace_bytes",
                 "cs_spec_accept_workspace_bytes", "cs_last_error"):
        assert must in names


def test_library_exports_every_declared_symbol(lib):
    for name in declared_functions():
        assert hasattr(lib, name), name
    assert set(binding.EXPORTED_SYMBOLS) == set(declared_functions())
    assert lib.cs_abi_version() == 1


def test_library_is_built_for_sm_103a_only():
    # the build passes exactly one -gencode, for sm_103a
    assert build.ARCH == ["-gencode", "arch=compute_103a,code=sm_103a"]


FAKE = 0x10000  # a non-null, 256-byte aligned address that is never dereferenced


def attn(lib, dims, n_draft=4, q=FAKE, kp=FAKE, vp=FAKE, pt=FAKE, cl=FAKE, out=FAKE, ws=FAKE,
         ws_bytes=1 << 40):
    return lib.cs_verify_attention(ctypes.byref(dims), q, kp, vp, pt, cl, n_draft, out, ws,
                                   ws_bytes, None)


def good_attn_dims():
    return binding.AttnDims(4, 32, 8, 128, 16, 64, 256, 0.0)


@pytest.mark.parametrize("field,value,code", [
    ("batch", -1, binding.CS_ERR_INVALID_ARG),
    ("n_q_heads", 0, binding.CS_ERR_INVALID_ARG),
    ("n_kv_heads", 0, binding.CS_ERR_INVALID_ARG),
    ("n_q_heads", 30, binding.CS_ERR_INVALID_ARG),       # not a multiple of Hkv = 8
    ("head_dim", 64, binding.CS_ERR_UNSUPPORTED),
    ("page_size", 12, binding.CS_ERR_UNSUPPORTED),
    ("page_size", 0, binding.CS_ERR_INVALID_ARG),
    ("max_pages_per_seq", 0, binding.CS_ERR_INVALID_ARG),
    ("num_pages", 0, binding.CS_ERR_INVALID_ARG),
    ("sm_scale", float("nan"), binding.CS_ERR_INVALID_ARG),
])
def test_verify_attention_rejects_bad_dims(lib, field, value, code):
    d = good_attn_dims()
    setattr(d, field, value)
    assert attn(lib, d) == code
    assert lib.cs_last_error()


@pytest.mark.parametrize("n_draft", [0, -1, 17])
def test_verify_attention_rejects_bad_n_draft(lib, n_draft):
    assert attn(lib, good_attn_dims(), n_draft=n_draft) == binding.CS_ERR_INVALID_ARG


def test_verify_attention_rejects_too_many_rows(lib):
    d = binding.AttnDims(1, 128, 8, 128, 16, 8, 8, 0.0)     # G = 16, (k+1)*G = 272
    assert attn(lib, d, n_draft=16) == binding.CS_ERR_UNSUPPORTED


@pytest.mark.parametrize("arg", ["q", "kp", "vp", "pt", "cl", "out"])
def test_verify_attention_rejects_null_pointers(lib, arg):
    assert attn(lib, good_attn_dims(), **{arg: None}) == binding.CS_ERR_INVALID_ARG


def test_verify_attention_rejects_misaligned_pool(lib):
    assert attn(lib, good_attn_dims(), kp=FAKE + 8) == binding.CS_ERR_INVALID_ARG
    assert attn(lib, good_attn_dims(), ws=FAKE + 64) == binding.CS_ERR_INVALID_ARG


def test_verify_attention_workspace_is_checked(lib):
    d = good_attn_dims()
    need = lib.cs_verify_attention_workspace_bytes(ctypes.byref(d), 4)
    assert need >= 256
    assert attn(lib, d, ws=None) == binding.CS_ERR_WORKSPACE
    assert attn(lib, d, ws_bytes=need - 1) == binding.CS_ERR_WORKSPACE
    assert "needed" in lib.cs_last_error().decode()


def test_empty_batch_is_a_no_op(lib):
    d = good_attn_dims()
    d.batch = 0
    assert attn(lib, d, q=None, kp=None, vp=None, pt=None, cl=None, out=None, ws=None) == binding.CS_OK
    a = binding.AcceptDims(0, 32000, binding.CS_BF16)
    assert lib.cs_spec_accept(ctypes.byref(a), None, None, None, None, 4, 1.0, None, None, None, 0,
                              None) == binding.CS_OK


def accept(lib, dims, n_draft=4, T=1.0, t=FAKE, d=FAKE, x=FAKE, u=FAKE, out=FAKE, n=FAKE, ws=FAKE,
           ws_bytes=1 << 40):
    return lib.cs_spec_accept(ctypes.byref(dims), t, d, x, u, n_draft, T, out, n, ws, ws_bytes, None)


@pytest.mark.parametrize("field,value", [("batch", -2), ("vocab", 0), ("logit_dtype", 7)])
def test_spec_accept_rejects_bad_dims(lib, field, value):
    dims = binding.AcceptDims(4, 32000, binding.CS_BF16)
    setattr(dims, field, value)
    assert accept(lib, dims) == binding.CS_ERR_INVALID_ARG


def test_spec_accept_rejects_vocabularies_beyond_the_limit(lib):
    assert accept(lib, binding.AcceptDims(2, (1 << 22) + 1, binding.CS_BF16)) == binding.CS_ERR_UNSUPPORTED
    assert lib.cs_spec_accept_workspace_bytes(ctypes.byref(binding.AcceptDims(2, (1 << 22) + 1, binding.CS_BF16)), 4) == 0


@pytest.mark.parametrize("T", [-0.5, float("nan"), float("inf")])
def test_spec_accept_rejects_bad_temperature(lib, T):
    assert accept(lib, binding.AcceptDims(4, 32000, binding.CS_BF16), T=T) == binding.CS_ERR_INVALID_ARG


@pytest.mark.parametrize("n_draft", [0, 17])
def test_spec_accept_rejects_bad_n_draft(lib, n_draft):
    assert accept(lib, binding.AcceptDims(4, 32000, binding.CS_BF16), n_draft=n_draft) == binding.CS_ERR_INVALID_ARG


def test_spec_accept_null_and_alignment(lib):
    dims = binding.AcceptDims(4, 32000, binding.CS_F32)
    for arg in ("t", "x", "u", "out", "n"):
        assert accept(lib, dims, **{arg: None}) == binding.CS_ERR_INVALID_ARG
    assert accept(lib, dims, d=None) == binding.CS_ERR_INVALID_ARG            # T > 0 needs the draft
    assert accept(lib, dims, t=FAKE + 2) == binding.CS_ERR_INVALID_ARG        # fp32 logits, 2-byte offset
    need = lib.cs_spec_accept_workspace_bytes(ctypes.byref(dims), 4)
    assert need >= 4 * 9 * 4 * 8             # one (max, sum) pair per chunk of each row
    assert accept(lib, dims, ws=None) == binding.CS_ERR_WORKSPACE
    assert accept(lib, dims, ws_bytes=need - 1) == binding.CS_ERR_WORKSPACE


def sample(lib, dims, T=1.0, z=FAKE, u=FAKE, out=FAKE, ws=FAKE, ws_bytes=1 << 40):
    return lib.cs_sample(ctypes.byref(dims), z, u, T, out, ws, ws_bytes, None)


def test_sample_argument_checks(lib):
    dims = binding.AcceptDims(4, 32000, binding.CS_BF16)
    for arg in ("z", "u", "out"):
        assert sample(lib, dims, **{arg: None}) == binding.CS_ERR_INVALID_ARG
    for T in (-1.0, float("nan"), float("inf")):
        assert sample(lib, dims, T=T) == binding.CS_ERR_INVALID_ARG
    assert sample(lib, binding.AcceptDims(4, 32000, 9)) == binding.CS_ERR_INVALID_ARG
    assert sample(lib, binding.AcceptDims(4, (1 << 22) + 1, binding.CS_BF16)) == binding.CS_ERR_UNSUPPORTED
    need = lib.cs_sample_workspace_bytes(ctypes.byref(dims))
    assert need >= 4 * 16 * 8                 # one pair per 4 KB item of each row
    assert sample(lib, dims, ws=None) == binding.CS_ERR_WORKSPACE
    assert sample(lib, dims, ws_bytes=need - 1) == binding.CS_ERR_WORKSPACE
    assert sample(lib, dims, ws=FAKE + 64) == binding.CS_ERR_INVALID_ARG
    assert sample(lib, binding.AcceptDims(0, 100, binding.CS_F32), z=None, u=None, out=None, ws=None) == binding.CS_OK


def test_kv_argument_checks(lib):
    d = good_attn_dims()
    append = lambda dims=d, n=6, **kw: lib.cs_kv_append(ctypes.byref(dims), kw.get("nk", FAKE), kw.get("nv", FAKE),
                                                        kw.get("kp", FAKE), kw.get("vp", FAKE), kw.get("pt", FAKE),
                                                        kw.get("cl", FAKE), n, None)
    for arg in ("nk", "nv", "kp", "vp", "pt", "cl"):
        assert append(**{arg: None}) == binding.CS_ERR_INVALID_ARG
    assert append(nk=FAKE + 8) == binding.CS_ERR_INVALID_ARG
    assert append(n=0) == binding.CS_ERR_INVALID_ARG
    bad = good_attn_dims()
    bad.head_dim = 64
    assert append(dims=bad) == binding.CS_ERR_UNSUPPORTED
    empty = good_attn_dims()
    empty.batch = 0
    assert append(dims=empty, nk=None, nv=None, kp=None, vp=None, pt=None, cl=None) == binding.CS_OK
    assert lib.cs_kv_commit(4, None, FAKE, 5, None) == binding.CS_ERR_INVALID_ARG
    assert lib.cs_kv_commit(4, FAKE, FAKE, 17, None) == binding.CS_ERR_INVALID_ARG
    assert lib.cs_kv_commit(0, None, None, 5, None) == binding.CS_OK


def test_route_argument_checks(lib):
    def route(dims, e=FAKE, c=FAKE, inv=FAKE, tau=0.85, g=FAKE, b=FAKE, s=FAKE, ws=FAKE, ws_bytes=1 << 40):
        return lib.cs_route(ctypes.byref(dims), e, c, inv, tau, g, b, s, ws, ws_bytes, None)
    d = binding.RouteDims(1024, 16384, 384)
    for dim in (0, 100, 448, -64):
        assert route(binding.RouteDims(4, 10, dim)) == binding.CS_ERR_UNSUPPORTED
    assert route(binding.RouteDims(-1, 10, 64)) == binding.CS_ERR_INVALID_ARG
    assert route(binding.RouteDims(4, -1, 64)) == binding.CS_ERR_INVALID_ARG
    assert route(binding.RouteDims(128 * 65535 + 1, 10, 64)) == binding.CS_ERR_UNSUPPORTED
    for tau in (float("nan"), float("inf"), -float("inf")):
        assert route(d, tau=tau) == binding.CS_ERR_INVALID_ARG
    for arg in ("e", "c", "inv", "g", "b", "s"):
        assert route(d, **{arg: None}) == binding.CS_ERR_INVALID_ARG
    assert route(d, e=FAKE + 8) == binding.CS_ERR_INVALID_ARG
    assert route(d, c=FAKE + 2) == binding.CS_ERR_INVALID_ARG
    assert route(d, s=FAKE + 1) == binding.CS_ERR_INVALID_ARG
    need = lib.cs_route_workspace_bytes(ctypes.byref(d))
    assert need >= 256 + 1024 * 8             # status word + at least one partial per request
    assert lib.cs_route_workspace_bytes(ctypes.byref(binding.RouteDims(4, 10, 100))) == 0
    assert route(d, ws=None) == binding.CS_ERR_WORKSPACE
    assert route(d, ws_bytes=need - 1) == binding.CS_ERR_WORKSPACE
    assert route(d, ws=FAKE + 64) == binding.CS_ERR_INVALID_ARG
    assert route(binding.RouteDims(0, 10, 64), e=None, c=None, inv=None, g=None, b=None, s=None,
                 ws=None) == binding.CS_OK
    assert lib.cs_route_norms(5, 100, FAKE, FAKE, None) == binding.CS_ERR_UNSUPPORTED
    assert lib.cs_route_norms(-1, 64, FAKE, FAKE, None) == binding.CS_ERR_INVALID_ARG
    assert lib.cs_route_norms(5, 64, None, FAKE, None) == binding.CS_ERR_INVALID_ARG
    assert lib.cs_route_norms(5, 64, FAKE + 8, FAKE, None) == binding.CS_ERR_INVALID_ARG
    assert lib.cs_route_norms(0, 64, None, None, None) == binding.CS_OK


def test_tree_argument_checks(lib):
    d = good_attn_dims()

    def tattn(dims=d, n=8, par=FAKE, ws=FAKE, ws_bytes=1 << 40, **kw):
        return lib.cs_tree_verify_attention(ctypes.byref(dims), kw.get("q", FAKE), kw.get("kp", FAKE),
                                            kw.get("vp", FAKE), kw.get("pt", FAKE), kw.get("cl", FAKE), par, n,
                                            kw.get("out", FAKE), ws, ws_bytes, None)
    for n in (0, -1, 65):
        assert tattn(n=n) == binding.CS_ERR_INVALID_ARG
        assert lib.cs_tree_verify_attention_workspace_bytes(ctypes.byref(d), n) == 0
    for arg in ("q", "kp", "vp", "pt", "cl", "out"):
        assert tattn(**{arg: None}) == binding.CS_ERR_INVALID_ARG
    assert tattn(par=None) == binding.CS_ERR_INVALID_ARG
    assert tattn(par=FAKE + 2) == binding.CS_ERR_INVALID_ARG
    assert tattn(kp=FAKE + 8) == binding.CS_ERR_INVALID_ARG
    bad = good_attn_dims()
    bad.head_dim = 64
    assert tattn(dims=bad) == binding.CS_ERR_UNSUPPORTED
    # trees beyond 144 query rows per KV head are accepted (row blocks): G = 16, 64 nodes
    wide = binding.AttnDims(2, 128, 8, 128, 16, 8, 64, 0.0)
    need = lib.cs_tree_verify_attention_workspace_bytes(ctypes.byref(wide), 64)
    assert need >= 256
    assert tattn(dims=wide, n=64, ws=None) == binding.CS_ERR_WORKSPACE
    assert tattn(dims=wide, n=64, ws_bytes=need - 1) == binding.CS_ERR_WORKSPACE
    empty = good_attn_dims()
    empty.batch = 0
    assert tattn(dims=empty, par=None, ws=None, q=None, kp=None, vp=None, pt=None, cl=None, out=None) == binding.CS_OK

    a = binding.AcceptDims(4, 32000, binding.CS_BF16)

    def tacc(dims=a, n=8, T=1.0, ws=FAKE, ws_bytes=1 << 40, **kw):
        return lib.cs_tree_accept(ctypes.byref(dims), kw.get("t", FAKE), kw.get("dd", FAKE), kw.get("par", FAKE),
                                  kw.get("x", FAKE), kw.get("u", FAKE), n, T, kw.get("out", FAKE),
                                  kw.get("path", FAKE), kw.get("na", FAKE), ws, ws_bytes, None)
    for n in (0, 65):
        assert tacc(n=n) == binding.CS_ERR_INVALID_ARG
        assert lib.cs_tree_accept_workspace_bytes(ctypes.byref(a), n) == 0
    for T in (-1.0, float("nan"), float("inf")):
        assert tacc(T=T) == binding.CS_ERR_INVALID_ARG
    for arg in ("t", "par", "x", "u", "out", "path", "na"):
        assert tacc(**{arg: None}) == binding.CS_ERR_INVALID_ARG
    assert tacc(dd=None) == binding.CS_ERR_INVALID_ARG            # sampling needs the draft rows
    assert tacc(t=FAKE + 1) == binding.CS_ERR_INVALID_ARG
    assert tacc(path=FAKE + 2) == binding.CS_ERR_INVALID_ARG
    assert tacc(dims=binding.AcceptDims(2, (1 << 22) + 1, binding.CS_BF16)) == binding.CS_ERR_UNSUPPORTED
    need = lib.cs_tree_accept_workspace_bytes(ctypes.byref(a), 8)
    assert need >= 4 * 16 * 4                                     # at least a count per streamed row
    assert tacc(ws=None) == binding.CS_ERR_WORKSPACE
    assert tacc(ws_bytes=need - 1) == binding.CS_ERR_WORKSPACE
    assert tacc(ws=FAKE + 64) == binding.CS_ERR_INVALID_ARG
    assert tacc(dims=binding.AcceptDims(0, 100, binding.CS_F32), t=None, dd=None, par=None, x=None, u=None,
                out=None, path=None, na=None, ws=None) == binding.CS_OK

    def commit(dims=d, n=8, **kw):
        return lib.cs_kv_commit_tree(ctypes.byref(dims), kw.get("kp", FAKE), kw.get("vp", FAKE), kw.get("pt", FAKE),
                                     kw.get("cl", FAKE), kw.get("path", FAKE), kw.get("na", FAKE), n, None)
    for arg in ("kp", "vp", "pt", "cl", "path", "na"):
        assert commit(**{arg: None}) == binding.CS_ERR_INVALID_ARG
    assert commit(n=0) == binding.CS_ERR_INVALID_ARG
    assert commit(n=65) == binding.CS_ERR_INVALID_ARG
    assert commit(vp=FAKE + 4) == binding.CS_ERR_INVALID_ARG
    assert commit(dims=bad) == binding.CS_ERR_UNSUPPORTED
    assert commit(dims=empty, kp=None, vp=None, pt=None, cl=None, path=None, na=None) == binding.CS_OK


def test_binding_fails_loudly_without_library(tmp_path):
    with pytest.raises(RuntimeError, match="not found"):
        binding.load_library(str(tmp_path / "missing.so"))


def test_wait_selftest_argument_checks(lib):
    # rejected on the host before anything is enqueued
    assert lib.cs_selftest_wait_timeout(None, None) == binding.CS_ERR_INVALID_ARG
    assert lib.cs_selftest_wait_timeout(FAKE + 2, None) == binding.CS_ERR_INVALID_ARG


def test_noalloc_status_rejects_a_null_output(lib):
    assert lib.cs_verify_attention_noalloc_status(None, None) == binding.CS_ERR_INVALID_ARG
    assert b"NULL" in lib.cs_last_error()
