"""Python binding of libcachespec.so: the same entry points, argument marshalling only.

Every step of the draft-and-verify path runs in the library's CUDA kernels;
this module checks tensor dtypes, shapes and devices, passes raw device
pointers and the current CUDA stream through ctypes, and turns a non-OK
status into an exception.  It never computes any part of the method and has
no CPU fallback: if the library is missing, every call raises.
"""
from __future__ import annotations

import ctypes
import os
import threading

import torch

from . import build as _build

CS_OK, CS_ERR_INVALID_ARG, CS_ERR_UNSUPPORTED, CS_ERR_CUDA, CS_ERR_WORKSPACE = range(5)
CS_F32, CS_BF16 = 0, 1
CS_DEVICE_WAIT_TIMEOUT = 1   # device status bit: a bounded wait inside a kernel gave up
STATUS_NAMES = {0: "CS_OK", 1: "CS_ERR_INVALID_ARG", 2: "CS_ERR_UNSUPPORTED", 3: "CS_ERR_CUDA",
                4: "CS_ERR_WORKSPACE"}
EXPORTED_SYMBOLS = ("cs_abi_version", "cs_last_error", "cs_verify_attention_workspace_bytes",
                    "cs_verify_attention", "cs_spec_accept_workspace_bytes", "cs_spec_accept",
                    "cs_read_device_status", "cs_verify_attention_noalloc", "cs_verify_attention_noalloc_status",
                    "cs_sample_workspace_bytes",
                    "cs_sample", "cs_kv_append", "cs_kv_commit", "cs_route_workspace_bytes",
                    "cs_route_norms", "cs_route", "cs_tree_verify_attention_workspace_bytes",
                    "cs_tree_verify_attention", "cs_tree_accept_workspace_bytes", "cs_tree_accept",
                    "cs_kv_commit_tree", "cs_selftest_wait_timeout")


class RouteDims(ctypes.Structure):
    _fields_ = [("batch", ctypes.c_int32), ("n_groups", ctypes.c_int32), ("dim", ctypes.c_int32)]


class AttnDims(ctypes.Structure):
    _fields_ = [("batch", ctypes.c_int32), ("n_q_heads", ctypes.c_int32),
                ("n_kv_heads", ctypes.c_int32), ("head_dim", ctypes.c_int32),
                ("page_size", ctypes.c_int32), ("max_pages_per_seq", ctypes.c_int32),
                ("num_pages", ctypes.c_int32), ("sm_scale", ctypes.c_float)]


class AcceptDims(ctypes.Structure):
    _fields_ = [("batch", ctypes.c_int32), ("vocab", ctypes.c_int32),
                ("logit_dtype", ctypes.c_int32)]


class CacheSpecError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__(f"{STATUS_NAMES.get(status, status)}: {message}")
        self.status = status


_lib = None
_lock = threading.Lock()


def library_path() -> str:
    return _build.LIB


def load_library(path: str | None = None):
    """Load libcachespec.so (built in-tree by ``__graft_entry__.build()``).  Raises if absent."""
    global _lib
    with _lock:
        if _lib is not None and path is None:
            return _lib
        p = path or _build.LIB
        if not os.path.exists(p):
            raise RuntimeError(f"libcachespec.so not found at {p}; build it with "
                               "`python -c 'import __graft_entry__ as g; g.build()'`")
        lib = ctypes.CDLL(p)
        vp, i32, sz = ctypes.c_void_p, ctypes.c_int32, ctypes.c_size_t
        lib.cs_abi_version.restype = i32
        lib.cs_last_error.restype = ctypes.c_char_p
        lib.cs_verify_attention_workspace_bytes.restype = sz
        lib.cs_verify_attention_workspace_bytes.argtypes = [ctypes.POINTER(AttnDims), i32]
        lib.cs_verify_attention.restype = ctypes.c_int
        lib.cs_verify_attention.argtypes = [ctypes.POINTER(AttnDims), vp, vp, vp, vp, vp, i32, vp,
                                            vp, sz, vp]
        lib.cs_spec_accept_workspace_bytes.restype = sz
        lib.cs_spec_accept_workspace_bytes.argtypes = [ctypes.POINTER(AcceptDims), i32]
        lib.cs_spec_accept.restype = ctypes.c_int
        lib.cs_spec_accept.argtypes = [ctypes.POINTER(AcceptDims), vp, vp, vp, vp, i32,
                                       ctypes.c_float, vp, vp, vp, sz, vp]
        lib.cs_verify_attention_noalloc.restype = ctypes.c_int
        lib.cs_verify_attention_noalloc.argtypes = [ctypes.POINTER(AttnDims), vp, vp, vp, vp, vp,
                                                    i32, vp, vp]
        lib.cs_verify_attention_noalloc_status.restype = ctypes.c_int
        lib.cs_verify_attention_noalloc_status.argtypes = [ctypes.POINTER(ctypes.c_int32), vp]
        lib.cs_read_device_status.restype = ctypes.c_int
        lib.cs_read_device_status.argtypes = [vp, ctypes.POINTER(ctypes.c_int32), vp]
        lib.cs_selftest_wait_timeout.restype = ctypes.c_int
        lib.cs_selftest_wait_timeout.argtypes = [vp, vp]
        lib.cs_kv_append.restype = ctypes.c_int
        lib.cs_kv_append.argtypes = [ctypes.POINTER(AttnDims), vp, vp, vp, vp, vp, vp, i32, vp]
        lib.cs_kv_commit.restype = ctypes.c_int
        lib.cs_kv_commit.argtypes = [i32, vp, vp, i32, vp]
        lib.cs_route_workspace_bytes.restype = sz
        lib.cs_route_workspace_bytes.argtypes = [ctypes.POINTER(RouteDims)]
        lib.cs_route_norms.restype = ctypes.c_int
        lib.cs_route_norms.argtypes = [i32, i32, vp, vp, vp]
        lib.cs_route.restype = ctypes.c_int
        lib.cs_route.argtypes = [ctypes.POINTER(RouteDims), vp, vp, vp, ctypes.c_float, vp, vp, vp, vp, sz, vp]
        lib.cs_sample_workspace_bytes.restype = sz
        lib.cs_sample_workspace_bytes.argtypes = [ctypes.POINTER(AcceptDims)]
        lib.cs_sample.restype = ctypes.c_int
        lib.cs_sample.argtypes = [ctypes.POINTER(AcceptDims), vp, vp, ctypes.c_float, vp, vp, sz, vp]
        lib.cs_tree_verify_attention_workspace_bytes.restype = sz
        lib.cs_tree_verify_attention_workspace_bytes.argtypes = [ctypes.POINTER(AttnDims), i32]
        lib.cs_tree_verify_attention.restype = ctypes.c_int
        lib.cs_tree_verify_attention.argtypes = [ctypes.POINTER(AttnDims), vp, vp, vp, vp, vp, vp, i32, vp,
                                                 vp, sz, vp]
        lib.cs_tree_accept_workspace_bytes.restype = sz
        lib.cs_tree_accept_workspace_bytes.argtypes = [ctypes.POINTER(AcceptDims), i32]
        lib.cs_tree_accept.restype = ctypes.c_int
        lib.cs_tree_accept.argtypes = [ctypes.POINTER(AcceptDims), vp, vp, vp, vp, vp, i32, ctypes.c_float,
                                       vp, vp, vp, vp, sz, vp]
        lib.cs_kv_commit_tree.restype = ctypes.c_int
        lib.cs_kv_commit_tree.argtypes = [ctypes.POINTER(AttnDims), vp, vp, vp, vp, vp, vp, i32, vp]
        if path is None:
            _lib = lib
        return lib


def _check(lib, status: int) -> None:
    if status != CS_OK:
        raise CacheSpecError(status, lib.cs_last_error().decode(errors="replace"))


def _ptr(t: torch.Tensor | None) -> int | None:
    return None if t is None else t.data_ptr()


def _stream(device: torch.device) -> int:
    return torch.cuda.current_stream(device).cuda_stream


def _need(t: torch.Tensor, name: str, dtype: torch.dtype, ndim: int, device) -> None:
    if not isinstance(t, torch.Tensor):
        raise TypeError(f"{name} must be a torch.Tensor")
    if t.dtype != dtype:
        raise TypeError(f"{name} must be {dtype}, got {t.dtype}")
    if t.dim() != ndim:
        raise ValueError(f"{name} must have {ndim} dims, got shape {tuple(t.shape)}")
    if not t.is_cuda or (device is not None and t.device != device):
        raise ValueError(f"{name} must live on {device or 'a CUDA device'}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")


def attn_dims(q: torch.Tensor, k_pages: torch.Tensor, page_table: torch.Tensor,
              sm_scale: float = 0.0) -> AttnDims:
    B, _, Hq, D = q.shape
    P, Hkv, ps, _ = k_pages.shape
    return AttnDims(B, Hq, Hkv, D, ps, page_table.shape[1], P, float(sm_scale))


# Workspaces handed out by this module, one per (device, size).  The kernels
# leave a workspace ready for the next call, so calls ordered on one stream
# may share it.
_workspaces: dict = {}


def verify_attention_workspace(dims: AttnDims, n_draft: int, device) -> torch.Tensor:
    lib = load_library()
    n = lib.cs_verify_attention_workspace_bytes(ctypes.byref(dims), int(n_draft))
    key = (str(device), n)
    ws = _workspaces.get(key)
    if ws is None:
        ws = torch.zeros(max(n, 256), dtype=torch.uint8, device=device)
        _workspaces[key] = ws
    return ws


def cs_verify_attention_workspace_bytes(q, k_pages, page_table, n_draft, sm_scale=0.0) -> int:
    lib = load_library()
    d = attn_dims(q, k_pages, page_table, sm_scale)
    return int(lib.cs_verify_attention_workspace_bytes(ctypes.byref(d), int(n_draft)))


def cs_verify_attention(q, k_pages, v_pages, page_table, ctx_lens, n_draft, out=None,
                        workspace=None, sm_scale: float = 0.0, stream: int | None = None):
    """Verify attention; returns ``out`` (bf16 [B, k+1, Hq, D]).  See include/cachespec.h."""
    lib = load_library()
    dev = q.device
    _need(q, "q", torch.bfloat16, 4, dev)
    _need(k_pages, "k_pages", torch.bfloat16, 4, dev)
    _need(v_pages, "v_pages", torch.bfloat16, 4, dev)
    _need(page_table, "page_table", torch.int32, 2, dev)
    _need(ctx_lens, "ctx_lens", torch.int32, 1, dev)
    if v_pages.shape != k_pages.shape:
        raise ValueError("k_pages and v_pages must have the same shape")
    if q.shape[1] != n_draft + 1:
        raise ValueError(f"q has {q.shape[1]} rows per request, n_draft+1 = {n_draft + 1}")
    d = attn_dims(q, k_pages, page_table, sm_scale)
    if out is None:
        out = torch.empty_like(q)
    else:
        _need(out, "out", torch.bfloat16, 4, dev)
    if workspace is None:
        workspace = verify_attention_workspace(d, n_draft, dev)
    st = lib.cs_verify_attention(ctypes.byref(d), _ptr(q), _ptr(k_pages), _ptr(v_pages),
                                 _ptr(page_table), _ptr(ctx_lens), int(n_draft), _ptr(out),
                                 _ptr(workspace), workspace.numel() * workspace.element_size(),
                                 _stream(dev) if stream is None else stream)
    _check(lib, st)
    return out


def spec_accept_workspace(dims: AcceptDims, n_draft: int, device) -> torch.Tensor:
    lib = load_library()
    n = lib.cs_spec_accept_workspace_bytes(ctypes.byref(dims), int(n_draft))
    key = ("accept", str(device), n)
    ws = _workspaces.get(key)
    if ws is None:
        ws = torch.zeros(max(n, 256), dtype=torch.uint8, device=device)
        _workspaces[key] = ws
    return ws


def cs_spec_accept(target_logits, draft_logits, draft_tokens, uniforms, temperature,
                   out_tokens=None, out_n_accepted=None, workspace=None,
                   stream: int | None = None):
    """Speculative acceptance; returns (out_tokens [B, k+1], n_accepted [B]).  See include/cachespec.h."""
    lib = load_library()
    dev = target_logits.device
    if target_logits.dtype not in (torch.float32, torch.bfloat16):
        raise TypeError("logits must be float32 or bfloat16")
    dtype = target_logits.dtype
    _need(target_logits, "target_logits", dtype, 3, dev)
    B, rows, V = target_logits.shape
    k = rows - 1
    if draft_logits is not None:
        _need(draft_logits, "draft_logits", dtype, 3, dev)
        if tuple(draft_logits.shape) != (B, k, V):
            raise ValueError(f"draft_logits must be [{B}, {k}, {V}]")
    _need(draft_tokens, "draft_tokens", torch.int32, 2, dev)
    _need(uniforms, "uniforms", torch.float32, 2, dev)
    if out_tokens is None:
        out_tokens = torch.empty((B, k + 1), dtype=torch.int32, device=dev)
    if out_n_accepted is None:
        out_n_accepted = torch.empty((B,), dtype=torch.int32, device=dev)
    _need(out_tokens, "out_tokens", torch.int32, 2, dev)
    _need(out_n_accepted, "out_n_accepted", torch.int32, 1, dev)
    d = AcceptDims(B, V, CS_F32 if dtype == torch.float32 else CS_BF16)
    if workspace is None:
        workspace = spec_accept_workspace(d, k, dev)
    st = lib.cs_spec_accept(ctypes.byref(d), _ptr(target_logits), _ptr(draft_logits),
                            _ptr(draft_tokens), _ptr(uniforms), int(k), float(temperature),
                            _ptr(out_tokens), _ptr(out_n_accepted), _ptr(workspace),
                            workspace.numel() * workspace.element_size(),
                            _stream(dev) if stream is None else stream)
    _check(lib, st)
    return out_tokens, out_n_accepted


def cs_kv_append(new_k, new_v, k_pages, v_pages, page_table, ctx_lens, stream: int | None = None):
    """Append the K/V rows of the newest positions into the page pools (in place).
    new_k / new_v bf16 [B, n_new, Hkv, D]; pools [P, Hkv, ps, D].  See include/cachespec.h."""
    lib = load_library()
    dev = k_pages.device
    _need(new_k, "new_k", torch.bfloat16, 4, dev)
    _need(new_v, "new_v", torch.bfloat16, 4, dev)
    _need(k_pages, "k_pages", torch.bfloat16, 4, dev)
    _need(v_pages, "v_pages", torch.bfloat16, 4, dev)
    _need(page_table, "page_table", torch.int32, 2, dev)
    _need(ctx_lens, "ctx_lens", torch.int32, 1, dev)
    B, n_new, Hkv, D = new_k.shape
    P, Hkv2, ps, D2 = k_pages.shape
    if tuple(new_v.shape) != tuple(new_k.shape) or Hkv2 != Hkv or D2 != D or k_pages.shape != v_pages.shape:
        raise ValueError("new rows and pools do not match")
    d = AttnDims(B, Hkv, Hkv, D, ps, page_table.shape[1], P, 0.0)
    st = lib.cs_kv_append(ctypes.byref(d), _ptr(new_k), _ptr(new_v), _ptr(k_pages), _ptr(v_pages),
                          _ptr(page_table), _ptr(ctx_lens), int(n_new), _stream(dev) if stream is None else stream)
    _check(lib, st)


def cs_kv_commit(ctx_lens, n_accepted, n_draft: int, stream: int | None = None):
    """Keep the accepted prefix: ctx_lens <- max(0, ctx_lens - k + n_accepted), in place."""
    lib = load_library()
    dev = ctx_lens.device
    _need(ctx_lens, "ctx_lens", torch.int32, 1, dev)
    _need(n_accepted, "n_accepted", torch.int32, 1, dev)
    st = lib.cs_kv_commit(int(ctx_lens.shape[0]), _ptr(ctx_lens), _ptr(n_accepted), int(n_draft),
                          _stream(dev) if stream is None else stream)
    _check(lib, st)


def cs_route_norms(centroids, inv_norms=None, stream: int | None = None):
    """Inverse L2 norms of the group centroids (bf16 [N, d]); returns fp32 [N]."""
    lib = load_library()
    dev = centroids.device
    _need(centroids, "centroids", torch.bfloat16, 2, dev)
    N, d = centroids.shape
    if inv_norms is None:
        inv_norms = torch.empty((N,), dtype=torch.float32, device=dev)
    _need(inv_norms, "inv_norms", torch.float32, 1, dev)
    st = lib.cs_route_norms(int(N), int(d), _ptr(centroids) if N else None, _ptr(inv_norms) if N else None,
                            _stream(dev) if stream is None else stream)
    _check(lib, st)
    return inv_norms


def cs_route(emb, centroids, inv_norms, tau, out_group=None, out_best=None, out_score=None, workspace=None,
             stream: int | None = None):
    """Batched semantic routing; returns (group [B], best [B], score [B]).  See include/cachespec.h."""
    lib = load_library()
    dev = emb.device
    _need(emb, "emb", torch.bfloat16, 2, dev)
    _need(centroids, "centroids", torch.bfloat16, 2, dev)
    _need(inv_norms, "inv_norms", torch.float32, 1, dev)
    B, d = emb.shape
    N = centroids.shape[0]
    if N and centroids.shape[1] != d:
        raise ValueError("emb and centroids differ in width")
    out_group = torch.empty((B,), dtype=torch.int32, device=dev) if out_group is None else out_group
    out_best = torch.empty((B,), dtype=torch.int32, device=dev) if out_best is None else out_best
    out_score = torch.empty((B,), dtype=torch.float32, device=dev) if out_score is None else out_score
    dims = RouteDims(B, N, d)
    if workspace is None:
        n = lib.cs_route_workspace_bytes(ctypes.byref(dims))
        key = ("route", str(dev), n)
        workspace = _workspaces.get(key)
        if workspace is None:
            workspace = torch.zeros(max(n, 256), dtype=torch.uint8, device=dev)
            _workspaces[key] = workspace
    st = lib.cs_route(ctypes.byref(dims), _ptr(emb), _ptr(centroids) if N else None, _ptr(inv_norms) if N else None,
                      float(tau), _ptr(out_group), _ptr(out_best), _ptr(out_score), _ptr(workspace),
                      workspace.numel() * workspace.element_size(), _stream(dev) if stream is None else stream)
    _check(lib, st)
    return out_group, out_best, out_score


def cs_sample(logits, uniforms, temperature, out_tokens=None, workspace=None,
              stream: int | None = None):
    """Draft-side sampling, one token per row of ``logits`` [B, V]; returns out_tokens [B].
    See include/cachespec.h."""
    lib = load_library()
    dev = logits.device
    if logits.dtype not in (torch.float32, torch.bfloat16):
        raise TypeError("logits must be float32 or bfloat16")
    _need(logits, "logits", logits.dtype, 2, dev)
    B, V = logits.shape
    _need(uniforms, "uniforms", torch.float32, 1, dev)
    if out_tokens is None:
        out_tokens = torch.empty((B,), dtype=torch.int32, device=dev)
    _need(out_tokens, "out_tokens", torch.int32, 1, dev)
    d = AcceptDims(B, V, CS_F32 if logits.dtype == torch.float32 else CS_BF16)
    if workspace is None:
        n = lib.cs_sample_workspace_bytes(ctypes.byref(d))
        key = ("sample", str(dev), n)
        workspace = _workspaces.get(key)
        if workspace is None:
            workspace = torch.zeros(max(n, 256), dtype=torch.uint8, device=dev)
            _workspaces[key] = workspace
    st = lib.cs_sample(ctypes.byref(d), _ptr(logits), _ptr(uniforms), float(temperature), _ptr(out_tokens),
                       _ptr(workspace), workspace.numel() * workspace.element_size(),
                       _stream(dev) if stream is None else stream)
    _check(lib, st)
    return out_tokens


def _cached_workspace(kind: str, device, n: int) -> torch.Tensor:
    key = (kind, str(device), n)
    ws = _workspaces.get(key)
    if ws is None:
        ws = torch.zeros(max(n, 256), dtype=torch.uint8, device=device)
        _workspaces[key] = ws
    return ws


def cs_tree_verify_attention(q, k_pages, v_pages, page_table, ctx_lens, parents, out=None, workspace=None,
                             sm_scale: float = 0.0, stream: int | None = None):
    """Token-tree verify attention; q / out bf16 [B, n, Hq, D], parents int32 [B, n].
    Returns ``out``.  See include/cachespec.h."""
    lib = load_library()
    dev = q.device
    _need(q, "q", torch.bfloat16, 4, dev)
    _need(k_pages, "k_pages", torch.bfloat16, 4, dev)
    _need(v_pages, "v_pages", torch.bfloat16, 4, dev)
    _need(page_table, "page_table", torch.int32, 2, dev)
    _need(ctx_lens, "ctx_lens", torch.int32, 1, dev)
    _need(parents, "parents", torch.int32, 2, dev)
    if v_pages.shape != k_pages.shape:
        raise ValueError("k_pages and v_pages must have the same shape")
    B, n = q.shape[0], q.shape[1]
    if tuple(parents.shape) != (B, n):
        raise ValueError(f"parents must be [{B}, {n}]")
    d = attn_dims(q, k_pages, page_table, sm_scale)
    if out is None:
        out = torch.empty_like(q)
    _need(out, "out", torch.bfloat16, 4, dev)
    if workspace is None:
        workspace = _cached_workspace("tree_attn", dev,
                                      lib.cs_tree_verify_attention_workspace_bytes(ctypes.byref(d), int(n)))
    st = lib.cs_tree_verify_attention(ctypes.byref(d), _ptr(q), _ptr(k_pages), _ptr(v_pages), _ptr(page_table),
                                      _ptr(ctx_lens), _ptr(parents), int(n), _ptr(out), _ptr(workspace),
                                      workspace.numel() * workspace.element_size(),
                                      _stream(dev) if stream is None else stream)
    _check(lib, st)
    return out


def cs_tree_accept(target_logits, draft_logits, parents, node_tokens, uniforms, temperature, out_tokens=None,
                   out_path=None, out_n_accepted=None, workspace=None, stream: int | None = None):
    """Token-tree acceptance walk; target / draft logits [B, n, V], parents / node_tokens int32 [B, n],
    uniforms fp32 [B, n].  Returns (tokens [B, n], path [B, n], n_accepted [B]).  See include/cachespec.h."""
    lib = load_library()
    dev = target_logits.device
    if target_logits.dtype not in (torch.float32, torch.bfloat16):
        raise TypeError("logits must be float32 or bfloat16")
    dtype = target_logits.dtype
    _need(target_logits, "target_logits", dtype, 3, dev)
    B, n, V = target_logits.shape
    if draft_logits is not None:
        _need(draft_logits, "draft_logits", dtype, 3, dev)
        if tuple(draft_logits.shape) != (B, n, V):
            raise ValueError(f"draft_logits must be [{B}, {n}, {V}]")
    for name, t in (("parents", parents), ("node_tokens", node_tokens)):
        _need(t, name, torch.int32, 2, dev)
        if tuple(t.shape) != (B, n):
            raise ValueError(f"{name} must be [{B}, {n}]")
    _need(uniforms, "uniforms", torch.float32, 2, dev)
    out_tokens = torch.empty((B, n), dtype=torch.int32, device=dev) if out_tokens is None else out_tokens
    out_path = torch.empty((B, n), dtype=torch.int32, device=dev) if out_path is None else out_path
    out_n_accepted = torch.empty((B,), dtype=torch.int32, device=dev) if out_n_accepted is None else out_n_accepted
    _need(out_tokens, "out_tokens", torch.int32, 2, dev)
    _need(out_path, "out_path", torch.int32, 2, dev)
    _need(out_n_accepted, "out_n_accepted", torch.int32, 1, dev)
    d = AcceptDims(B, V, CS_F32 if dtype == torch.float32 else CS_BF16)
    if workspace is None:
        workspace = _cached_workspace("tree_accept", dev, lib.cs_tree_accept_workspace_bytes(ctypes.byref(d), int(n)))
    st = lib.cs_tree_accept(ctypes.byref(d), _ptr(target_logits), _ptr(draft_logits), _ptr(parents),
                            _ptr(node_tokens), _ptr(uniforms), int(n), float(temperature), _ptr(out_tokens),
                            _ptr(out_path), _ptr(out_n_accepted), _ptr(workspace),
                            workspace.numel() * workspace.element_size(), _stream(dev) if stream is None else stream)
    _check(lib, st)
    return out_tokens, out_path, out_n_accepted


def cs_kv_commit_tree(k_pages, v_pages, page_table, ctx_lens, path, n_accepted, stream: int | None = None):
    """Move the accepted tree path's K/V rows next to the root and shorten ctx_lens (in place);
    path int32 [B, n] and n_accepted [B] as returned by cs_tree_accept."""
    lib = load_library()
    dev = k_pages.device
    _need(k_pages, "k_pages", torch.bfloat16, 4, dev)
    _need(v_pages, "v_pages", torch.bfloat16, 4, dev)
    _need(page_table, "page_table", torch.int32, 2, dev)
    _need(ctx_lens, "ctx_lens", torch.int32, 1, dev)
    _need(path, "path", torch.int32, 2, dev)
    _need(n_accepted, "n_accepted", torch.int32, 1, dev)
    if k_pages.shape != v_pages.shape:
        raise ValueError("k_pages and v_pages must have the same shape")
    P, Hkv, ps, D = k_pages.shape
    B, n = path.shape
    d = AttnDims(B, Hkv, Hkv, D, ps, page_table.shape[1], P, 0.0)
    st = lib.cs_kv_commit_tree(ctypes.byref(d), _ptr(k_pages), _ptr(v_pages), _ptr(page_table), _ptr(ctx_lens),
                               _ptr(path), _ptr(n_accepted), int(n), _stream(dev) if stream is None else stream)
    _check(lib, st)


def cs_verify_attention_noalloc(q, k_pages, v_pages, page_table, ctx_lens, n_draft, out=None,
                                sm_scale: float = 0.0, stream: int | None = None):
    """Verify attention without a workspace, for callers that cannot allocate device
    memory (the library's own fixed scratch is used; see include/cachespec.h)."""
    lib = load_library()
    dev = q.device
    _need(q, "q", torch.bfloat16, 4, dev)
    _need(k_pages, "k_pages", torch.bfloat16, 4, dev)
    _need(v_pages, "v_pages", torch.bfloat16, 4, dev)
    _need(page_table, "page_table", torch.int32, 2, dev)
    _need(ctx_lens, "ctx_lens", torch.int32, 1, dev)
    d = attn_dims(q, k_pages, page_table, sm_scale)
    if out is None:
        out = torch.empty_like(q)
    _need(out, "out", torch.bfloat16, 4, dev)
    st = lib.cs_verify_attention_noalloc(ctypes.byref(d), _ptr(q), _ptr(k_pages), _ptr(v_pages),
                                         _ptr(page_table), _ptr(ctx_lens), int(n_draft), _ptr(out),
                                         _stream(dev) if stream is None else stream)
    _check(lib, st)
    return out


def cs_selftest_wait_timeout(workspace: torch.Tensor, stream: int | None = None) -> None:
    """Runs the kernels' bounded wait on a barrier nothing completes (about one
    second); it sets CS_DEVICE_WAIT_TIMEOUT in the workspace's status word."""
    lib = load_library()
    _check(lib, lib.cs_selftest_wait_timeout(_ptr(workspace),
                                             _stream(workspace.device) if stream is None else stream))


def cs_read_device_status(workspace: torch.Tensor, stream: int | None = None) -> int:
    """Status word of a verify-attention workspace (synchronises the stream)."""
    lib = load_library()
    v = ctypes.c_int32(0)
    _check(lib, lib.cs_read_device_status(_ptr(workspace), ctypes.byref(v),
                                          _stream(workspace.device) if stream is None else stream))
    return int(v.value)


def cs_verify_attention_noalloc_status(device=None, stream: int | None = None) -> int:
    """Status word of the allocation-free entry point on the current device: the
    CS_DEVICE_* bits of its latest call (synchronises the stream)."""
    lib = load_library()
    dev = torch.device("cuda", torch.cuda.current_device()) if device is None else torch.device(device)
    v = ctypes.c_int32(0)
    _check(lib, lib.cs_verify_attention_noalloc_status(ctypes.byref(v), _stream(dev) if stream is None else stream))
    return int(v.value)
