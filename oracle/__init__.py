"""fp64 CPU oracle for the draft-and-verify step (test infrastructure only).

Only ``tests/``, ``__graft_entry__.smoke()`` and the ``cpu_baseline`` /
``--impl reference`` leg of ``bench.py`` may import this package.  The CUDA
path never imports it and it never imports the CUDA path.

The arithmetic lives in ``cs_oracle.c`` (plain C, fp64, OpenMP over
independent requests); this module builds it with gcc and marshals numpy
arrays through ctypes.  What each routine computes and which passage of the
paper it follows is stated in ``cs_oracle.c``.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "cs_oracle.c")
_LIB_PATH = os.path.join(_HERE, "liboracle.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile ``cs_oracle.c`` into ``liboracle.so`` next to it (gcc, OpenMP)."""
    with _lock:
        if (not force and os.path.exists(_LIB_PATH)
                and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
            return _LIB_PATH
        tmp = _LIB_PATH + f".tmp{os.getpid()}"
        cmd = ["gcc", "-std=c11", "-O2", "-fno-fast-math", "-ffp-contract=off",
               "-fopenmp", "-fPIC", "-shared", "-o", tmp, _SRC, "-lm"]
        subprocess.run(cmd, check=True)
        os.replace(tmp, _LIB_PATH)
        return _LIB_PATH


def _load():
    global _lib
    if _lib is None:
        build()
        lib = ctypes.CDLL(_LIB_PATH)
        i32, f64, vp = ctypes.c_int32, ctypes.c_double, ctypes.c_void_p
        lib.oracle_verify_attention.restype = ctypes.c_int
        lib.oracle_verify_attention.argtypes = [i32] * 7 + [f64] + [vp] * 5 + [i32, vp]
        lib.oracle_spec_accept.restype = ctypes.c_int
        lib.oracle_spec_accept.argtypes = [i32, i32, i32, vp, vp, vp, vp, i32, f64, vp, vp, vp, vp]
        lib.oracle_spec_accept_f64u.restype = ctypes.c_int
        lib.oracle_spec_accept_f64u.argtypes = [i32, i32, i32, vp, vp, vp, vp, i32, f64, vp, vp, vp, vp]
        lib.oracle_row_probs.restype = f64
        lib.oracle_row_probs.argtypes = [vp, i32, i32, f64, vp]
        lib.oracle_residual.restype = f64
        lib.oracle_residual.argtypes = [vp, vp, i32, vp]
        lib.oracle_inverse_cdf.restype = i32
        lib.oracle_inverse_cdf.argtypes = [vp, f64, i32, f64, vp]
        lib.oracle_row_argmax.restype = i32
        lib.oracle_row_argmax.argtypes = [vp, i32, i32]
        lib.oracle_kv_append.restype = ctypes.c_int
        lib.oracle_kv_append.argtypes = [i32] * 6 + [vp] * 6 + [i32]
        lib.oracle_kv_commit.restype = ctypes.c_int
        lib.oracle_kv_commit.argtypes = [i32, vp, vp, i32]
        lib.oracle_route.restype = ctypes.c_int
        lib.oracle_route.argtypes = [i32, i32, i32, vp, vp, f64, vp, vp, vp, vp, vp]
        lib.oracle_sample.restype = ctypes.c_int
        lib.oracle_sample.argtypes = [i32, i32, i32, vp, vp, f64, vp, vp]
        lib.oracle_tree_attention.restype = ctypes.c_int
        lib.oracle_tree_attention.argtypes = [i32] * 7 + [f64] + [vp] * 6 + [i32, vp]
        lib.oracle_tree_accept.restype = ctypes.c_int
        lib.oracle_tree_accept.argtypes = [i32, i32, i32, vp, vp, vp, vp, vp, i32, f64] + [vp] * 5
        lib.oracle_tree_accept_f64u.restype = ctypes.c_int
        lib.oracle_tree_accept_f64u.argtypes = [i32, i32, i32, vp, vp, vp, vp, vp, i32, f64] + [vp] * 5
        lib.oracle_kv_commit_tree.restype = ctypes.c_int
        lib.oracle_kv_commit_tree.argtypes = [i32] * 6 + [vp] * 6 + [i32]
        lib.oracle_max_threads.restype = ctypes.c_int
        lib.oracle_set_threads.argtypes = [ctypes.c_int]
        _lib = lib
    return _lib


def _ptr(a: np.ndarray | None):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _logit_array(a: np.ndarray) -> tuple[np.ndarray, int]:
    """Return (contiguous array, dtype code): 0 = fp32, 1 = bf16 bit patterns (uint16)."""
    a = np.ascontiguousarray(a)
    if a.dtype == np.float32:
        return a, 0
    if a.dtype == np.uint16:
        return a, 1
    raise TypeError(f"logits must be float32 or bf16 bit patterns (uint16), got {a.dtype}")


def set_threads(n: int) -> None:
    _load().oracle_set_threads(int(n))


def max_threads() -> int:
    return int(_load().oracle_max_threads())


def verify_attention(q_bits, k_bits, v_bits, page_table, ctx_lens, n_draft, scale=0.0):
    """fp64 verify attention.

    q_bits [B, k+1, Hq, D] uint16 (bf16 bits); k_bits/v_bits [P, Hkv, ps, D]
    uint16; page_table [B, max_pages] int32; ctx_lens [B] int32.
    Returns fp64 [B, k+1, Hq, D].
    """
    lib = _load()
    q = np.ascontiguousarray(q_bits, dtype=np.uint16)
    kp = np.ascontiguousarray(k_bits, dtype=np.uint16)
    vp = np.ascontiguousarray(v_bits, dtype=np.uint16)
    pt = np.ascontiguousarray(page_table, dtype=np.int32)
    cl = np.ascontiguousarray(ctx_lens, dtype=np.int32)
    B, rows, Hq, D = q.shape
    assert rows == n_draft + 1
    P, Hkv, ps, D2 = kp.shape
    assert D2 == D and vp.shape == kp.shape and pt.shape[0] == B and cl.shape == (B,)
    out = np.zeros((B, rows, Hq, D), dtype=np.float64)
    rc = lib.oracle_verify_attention(B, Hq, Hkv, D, ps, pt.shape[1], P, float(scale),
                                     _ptr(q), _ptr(kp), _ptr(vp), _ptr(pt), _ptr(cl),
                                     int(n_draft), _ptr(out))
    if rc != 0:
        raise RuntimeError(f"oracle_verify_attention failed with status {rc}")
    return out


def spec_accept(target, draft, draft_tokens, uniforms, temperature, with_draw_margin=False):
    """fp64 speculative acceptance.

    target [B, k+1, V] (float32 or uint16 bf16 bits); draft [B, k, V] same dtype
    (None allowed when temperature == 0); draft_tokens [B, k] int32;
    uniforms [B, k+1] float32 (or float64, which the pins use to place u
    exactly on either side of a threshold).  Returns (out_tokens [B, k+1] int32,
    n_accepted [B] int32, margin [B] float64): margin is the smallest
    |u_i - p_i(x_i)/q_i(x_i)| over the deciding accept tests.  With
    ``with_draw_margin`` a fourth array gives |u_k - CDF| at the two edges of
    the drawn cell.
    """
    lib = _load()
    t, code = _logit_array(target)
    B, rows, V = t.shape
    k = rows - 1
    d = None
    if draft is not None:
        d, code_d = _logit_array(draft)
        assert code_d == code and d.shape == (B, k, V)
    x = np.ascontiguousarray(draft_tokens, dtype=np.int32).reshape(B, k)
    u = np.asarray(uniforms)
    if u.dtype == np.float64:          # fp64 uniforms: used by the oracle's own pins
        fn = lib.oracle_spec_accept_f64u
        u = np.ascontiguousarray(u).reshape(B, k + 1)
    else:                              # the library's uniform type
        fn = lib.oracle_spec_accept
        u = np.ascontiguousarray(u, dtype=np.float32).reshape(B, k + 1)
    out = np.zeros((B, k + 1), dtype=np.int32)
    acc = np.zeros((B,), dtype=np.int32)
    margin = np.zeros((B,), dtype=np.float64)
    draw_margin = np.zeros((B,), dtype=np.float64)
    rc = fn(B, V, code, _ptr(t), _ptr(d), _ptr(x), _ptr(u), k,
            float(temperature), _ptr(out), _ptr(acc), _ptr(margin), _ptr(draw_margin))
    if rc != 0:
        raise RuntimeError(f"oracle_spec_accept failed with status {rc}")
    if with_draw_margin:
        return out, acc, margin, draw_margin
    return out, acc, margin


def sample(logits, uniforms, temperature, with_margin=False):
    """Draft-side sampling oracle: one token per row of ``logits`` [B, V] (bf16 bit
    patterns or fp32); ``uniforms`` [B] (fp32 or fp64).  Returns tokens (and margins)."""
    lib = _load()
    z, code = _logit_array(np.asarray(logits))
    B, V = z.shape
    u = np.ascontiguousarray(np.asarray(uniforms, dtype=np.float64).reshape(B))
    out = np.zeros(B, dtype=np.int32)
    margin = np.zeros(B, dtype=np.float64)
    rc = lib.oracle_sample(B, V, code, _ptr(z), _ptr(u), float(temperature), _ptr(out), _ptr(margin))
    if rc != 0:
        raise RuntimeError(f"oracle_sample failed with status {rc}")
    return (out, margin) if with_margin else out


def kv_append(new_k, new_v, k_pages, v_pages, page_table, ctx_lens):
    """Paged append in place on numpy uint16 (bf16 bit) pools; new rows [B, n_new, Hkv, D]."""
    lib = _load()
    nk = np.ascontiguousarray(new_k, dtype=np.uint16)
    nv = np.ascontiguousarray(new_v, dtype=np.uint16)
    assert k_pages.dtype == np.uint16 and k_pages.flags.c_contiguous and v_pages.flags.c_contiguous
    B, n_new, Hkv, D = nk.shape
    P, _, ps, _ = k_pages.shape
    pt = np.ascontiguousarray(page_table, dtype=np.int32)
    cl = np.ascontiguousarray(ctx_lens, dtype=np.int32)
    rc = lib.oracle_kv_append(B, Hkv, D, ps, pt.shape[1], P, _ptr(nk), _ptr(nv), _ptr(k_pages),
                              _ptr(v_pages), _ptr(pt), _ptr(cl), n_new)
    if rc != 0:
        raise RuntimeError(f"oracle_kv_append failed with status {rc}")


def kv_commit(ctx_lens, n_accepted, n_draft):
    """New context lengths after the acceptance step (returns a new int32 array)."""
    lib = _load()
    cl = np.array(ctx_lens, dtype=np.int32)
    na = np.ascontiguousarray(n_accepted, dtype=np.int32)
    rc = lib.oracle_kv_commit(cl.shape[0], _ptr(cl), _ptr(na), int(n_draft))
    if rc != 0:
        raise RuntimeError(f"oracle_kv_commit failed with status {rc}")
    return cl


def route(emb_bits, centroid_bits, tau):
    """fp64 semantic routing.  emb [B, d] and centroids [N, d] as uint16 bf16 bits.
    Returns dict(group, best, score, margin, tau_margin)."""
    lib = _load()
    e = np.ascontiguousarray(emb_bits, dtype=np.uint16)
    c = np.ascontiguousarray(centroid_bits, dtype=np.uint16)
    B, d = e.shape
    N = c.shape[0] if c.size else 0
    if N:
        assert c.shape[1] == d
    out = {k: np.zeros(B, dtype=np.int32) for k in ("group", "best")}
    out.update({k: np.zeros(B, dtype=np.float64) for k in ("score", "margin", "tau_margin")})
    rc = lib.oracle_route(B, N, d, _ptr(e), _ptr(c) if N else None, float(tau), _ptr(out["group"]),
                          _ptr(out["best"]), _ptr(out["score"]), _ptr(out["margin"]), _ptr(out["tau_margin"]))
    if rc != 0:
        raise RuntimeError(f"oracle_route failed with status {rc}")
    return out


def row_probs(row, temperature):
    """p = softmax(row / T) in fp64 for one logit row; returns (p, normaliser)."""
    lib = _load()
    r, code = _logit_array(np.asarray(row).reshape(-1))
    p = np.zeros(r.shape[0], dtype=np.float64)
    S = lib.oracle_row_probs(_ptr(r), code, r.shape[0], float(temperature), _ptr(p))
    return p, S


def residual(p, q):
    """r = max(0, p - q) and Z = sum(r) in fp64."""
    lib = _load()
    p = np.ascontiguousarray(p, dtype=np.float64)
    q = np.ascontiguousarray(q, dtype=np.float64)
    r = np.zeros_like(p)
    Z = lib.oracle_residual(_ptr(p), _ptr(q), p.shape[0], _ptr(r))
    return r, Z


def inverse_cdf(r, Z, u):
    """Token drawn by the inverse CDF of weights r (total Z) at uniform u; (token, margin)."""
    lib = _load()
    r = np.ascontiguousarray(r, dtype=np.float64)
    m = ctypes.c_double(0.0)
    v = lib.oracle_inverse_cdf(_ptr(r), float(Z), r.shape[0], float(u), ctypes.byref(m))
    return int(v), float(m.value)


def row_argmax(row):
    lib = _load()
    r, code = _logit_array(np.asarray(row).reshape(-1))
    return int(lib.oracle_row_argmax(_ptr(r), code, r.shape[0]))


def tree_attention(q_bits, k_bits, v_bits, page_table, ctx_lens, parents, scale=0.0):
    """fp64 token-tree verify attention.

    q_bits [B, n, Hq, D] uint16 (bf16 bits), one query row per tree node;
    parents [B, n] int32 (node 0 is the root; parents[c] in [0, c)).  The other
    arguments as for ``verify_attention``.  Returns fp64 [B, n, Hq, D].
    """
    lib = _load()
    q = np.ascontiguousarray(q_bits, dtype=np.uint16)
    kp = np.ascontiguousarray(k_bits, dtype=np.uint16)
    vp = np.ascontiguousarray(v_bits, dtype=np.uint16)
    pt = np.ascontiguousarray(page_table, dtype=np.int32)
    cl = np.ascontiguousarray(ctx_lens, dtype=np.int32)
    B, n, Hq, D = q.shape
    par = np.ascontiguousarray(parents, dtype=np.int32).reshape(B, n)
    P, Hkv, ps, D2 = kp.shape
    assert D2 == D and vp.shape == kp.shape and pt.shape[0] == B and cl.shape == (B,)
    out = np.zeros((B, n, Hq, D), dtype=np.float64)
    rc = lib.oracle_tree_attention(B, Hq, Hkv, D, ps, pt.shape[1], P, float(scale), _ptr(q), _ptr(kp),
                                   _ptr(vp), _ptr(pt), _ptr(cl), _ptr(par), n, _ptr(out))
    if rc != 0:
        raise RuntimeError(f"oracle_tree_attention failed with status {rc}")
    return out


def tree_accept(target, draft, parents, node_tokens, uniforms, temperature):
    """fp64 token-tree acceptance (multi-candidate speculative sampling).

    target, draft [B, n, V] (float32 or uint16 bf16 bits; draft may be None when
    temperature == 0); parents, node_tokens [B, n] int32; uniforms [B, n]
    float32 (or float64 for the pins).  Returns dict(tokens [B, n], path [B, n],
    n_accepted [B], margin [B], draw_margin [B]).
    """
    lib = _load()
    t, code = _logit_array(target)
    B, n, V = t.shape
    d = None
    if draft is not None:
        d, code_d = _logit_array(draft)
        assert code_d == code and d.shape == (B, n, V)
    par = np.ascontiguousarray(parents, dtype=np.int32).reshape(B, n)
    x = np.ascontiguousarray(node_tokens, dtype=np.int32).reshape(B, n)
    u = np.asarray(uniforms)
    if u.dtype == np.float64:
        fn = lib.oracle_tree_accept_f64u
        u = np.ascontiguousarray(u).reshape(B, n)
    else:
        fn = lib.oracle_tree_accept
        u = np.ascontiguousarray(u, dtype=np.float32).reshape(B, n)
    res = {"tokens": np.zeros((B, n), np.int32), "path": np.zeros((B, n), np.int32),
           "n_accepted": np.zeros(B, np.int32), "margin": np.zeros(B), "draw_margin": np.zeros(B)}
    rc = fn(B, V, code, _ptr(t), _ptr(d), _ptr(par), _ptr(x), _ptr(u), n, float(temperature),
            _ptr(res["tokens"]), _ptr(res["path"]), _ptr(res["n_accepted"]), _ptr(res["margin"]),
            _ptr(res["draw_margin"]))
    if rc != 0:
        raise RuntimeError(f"oracle_tree_accept failed with status {rc}")
    return res


def kv_commit_tree(k_pages, v_pages, page_table, ctx_lens, path, n_accepted, n_nodes):
    """Moves the accepted path's K/V rows next to the root, in place on numpy uint16
    pools; returns the new context lengths (a new int32 array)."""
    lib = _load()
    assert k_pages.dtype == np.uint16 and k_pages.flags.c_contiguous and v_pages.flags.c_contiguous
    P, Hkv, ps, D = k_pages.shape
    pt = np.ascontiguousarray(page_table, dtype=np.int32)
    cl = np.array(ctx_lens, dtype=np.int32)
    B = cl.shape[0]
    pa = np.ascontiguousarray(path, dtype=np.int32).reshape(B, n_nodes)
    na = np.ascontiguousarray(n_accepted, dtype=np.int32)
    rc = lib.oracle_kv_commit_tree(B, Hkv, D, ps, pt.shape[1], P, _ptr(k_pages), _ptr(v_pages), _ptr(pt),
                                   _ptr(cl), _ptr(pa), _ptr(na), int(n_nodes))
    if rc != 0:
        raise RuntimeError(f"oracle_kv_commit_tree failed with status {rc}")
    return cl
