"""fp64 CPU oracle of the fused GEMM + tail path (test infrastructure only).

Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline / reference leg
of ``bench.py`` may import this package.  The product library never does, and
this package imports nothing from it: the two share no code.

Every function is the plain definition of the step it names, evaluated in
double precision by ``kf_oracle.c`` (compiled here with gcc, no fast-math, no
FP contraction):

* ``fused_gemm``   Y = chain(X W^T)  -- the GEMM + tail-op problems of the
  paper's B580 study (Sec. IV-B, Table 3: layer-wise fusion of the post-GEMM
  ops, fp32-or-wider post-processing).
* ``moe_route``    top-k routing + stable sort by expert (gpt-oss decode path,
  Sec. IV-A).
* ``moe_ffn``      per-token MoE expert FFN with SwiGLU and the routing-weighted
  sum (the "MoE finalize" step of Sec. IV-A, Table 1).
* ``grouped_gemm`` per-group GEMM + chain with optional row gather / scatter.

Chains are lists of ``(kind, params)``: kinds ``bias, scale, relu, gelu_tanh,
silu, sigmoid, residual_add, row_logsumexp, groupnorm, swiglu,
row_scale_scatter_add, mish, leaky_relu, mul, row_scale, row_sum``; params ``p0, p1`` (tensors),
``scalar, eps, groups``.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading
from typing import Dict, List, Optional, Sequence, Tuple

import numpy as np
import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
# KF_ORACLE_SRC / KF_ORACLE_BUILD let the mutation test build a deliberately
# broken copy of the oracle (in a temporary directory) and check that the pins fail.
_SRC = os.environ.get("KF_ORACLE_SRC", os.path.join(_HERE, "kf_oracle.c"))
_BUILD = os.environ.get("KF_ORACLE_BUILD", os.path.join(_HERE, "_build"))
_LIB_PATH = os.path.join(_BUILD, "libkf_oracle.so")
_lock = threading.Lock()
_lib = None

ORC_F32, ORC_BF16, ORC_F16 = 0, 1, 2
KINDS = {
    "bias": 0, "scale": 1, "relu": 2, "gelu_tanh": 3, "silu": 4, "sigmoid": 5,
    "residual_add": 6, "row_logsumexp": 7, "groupnorm": 8, "swiglu": 9,
    "row_scale_scatter_add": 10, "mish": 11, "leaky_relu": 12, "mul": 13, "row_scale": 14,
    "row_sum": 15,
}


class _Op(ctypes.Structure):
    _fields_ = [("kind", ctypes.c_int32), ("groups", ctypes.c_int32),
                ("scalar", ctypes.c_double), ("eps", ctypes.c_double),
                ("p0", ctypes.c_void_p), ("p1", ctypes.c_void_p),
                ("p_dtype", ctypes.c_int32), ("pad_", ctypes.c_int32), ("ld", ctypes.c_int64)]


def build(force: bool = False) -> str:
    """Compile kf_oracle.c into oracle/_build/libkf_oracle.so (gcc, -O2)."""
    os.makedirs(_BUILD, exist_ok=True)
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O2", "-std=c11", "-D_GNU_SOURCE", "-ffp-contract=off", "-fno-fast-math",
           "-fPIC", "-shared", "-pthread", _SRC, "-o", tmp, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(build())
            P, I64, I32, D = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int32, ctypes.c_double
            lib.orc_fused_gemm.argtypes = [P, ctypes.c_int, I64, P, ctypes.c_int, I64, I64, I64, I64,
                                           P, ctypes.c_int, P, I64, P, I64, ctypes.c_int]
            lib.orc_fused_gemm.restype = ctypes.c_int
            lib.orc_moe_route.argtypes = [P, I64, I32, I32, P, P, P, P, P, P]
            lib.orc_moe_route.restype = ctypes.c_int
            D = ctypes.c_double
            lib.orc_moe_ffn.argtypes = [P, P, P, P, P, I64, I64, I32, P, I64, ctypes.c_int, P, ctypes.c_int,
                                        P, P, D, D, D]
            lib.orc_moe_ffn.restype = ctypes.c_int
            lib.orc_grouped_gemm.argtypes = [P, ctypes.c_int, I64, P, P, ctypes.c_int, I64, I64, P, I32,
                                             I64, I64, P, ctypes.c_int, P, I64]
            lib.orc_grouped_gemm.restype = ctypes.c_int
            lib.orc_add_rmsnorm.argtypes = [P, P, ctypes.c_int, P, ctypes.c_int, D, I64, I64, P, P]
            lib.orc_add_rmsnorm.restype = ctypes.c_int
            lib.orc_qkv_rope_kv.argtypes = [P, P, ctypes.c_int, P, ctypes.c_int, P, P, P, P, I64, I64, I64, I32, I32,
                                            I32, I64, P, P, P]
            lib.orc_qkv_rope_kv.restype = ctypes.c_int
            lib.orc_round_bf16.argtypes = [D]
            lib.orc_round_bf16.restype = D
            _lib = lib
    return _lib


def _np(t) -> Tuple[np.ndarray, int]:
    """Contiguous numpy view of a tensor/array and the oracle dtype code.
    bf16 tensors are passed as their raw 16-bit patterns."""
    if isinstance(t, torch.Tensor):
        t = t.detach().cpu().contiguous()
        if t.dtype == torch.bfloat16:
            return t.view(torch.int16).numpy().view(np.uint16), ORC_BF16
        if t.dtype == torch.float16:
            return t.view(torch.int16).numpy().view(np.uint16), ORC_F16
        if t.dtype == torch.float32:
            return t.numpy(), ORC_F32
        if t.dtype == torch.int32:
            return t.numpy(), -1
        if t.dtype == torch.float64:
            return t.to(torch.float32).numpy(), ORC_F32
        raise TypeError(f"oracle: unsupported tensor dtype {t.dtype}")
    a = np.ascontiguousarray(t)
    if a.dtype == np.float32:
        return a, ORC_F32
    if a.dtype == np.uint16:
        return a, ORC_BF16
    if a.dtype == np.float16:
        return a.view(np.uint16), ORC_F16
    if a.dtype == np.int32:
        return a, -1
    raise TypeError(f"oracle: unsupported array dtype {a.dtype}")


def _ptr(a: np.ndarray) -> int:
    return a.ctypes.data


def _ops(chain: Sequence[Tuple[str, Dict]], keep: list):
    arr = (_Op * max(1, len(chain)))()
    for i, (kind, prm) in enumerate(chain):
        o = arr[i]
        o.kind = KINDS[kind]
        o.groups = int(prm.get("groups", 0))
        o.scalar = float(prm.get("scalar", 0.0 if kind != "leaky_relu" else 0.01))
        o.eps = float(prm.get("eps", 0.0))
        o.p_dtype = ORC_F32
        o.ld = 0
        for slot in ("p0", "p1"):
            v = prm.get(slot)
            if v is None:
                setattr(o, slot, None)
                continue
            a, dt = _np(v)
            keep.append(a)
            setattr(o, slot, _ptr(a))
            if slot == "p0" and dt >= 0:
                o.p_dtype = dt
                if a.ndim == 2:
                    o.ld = int(prm.get("ld", a.shape[1]))
    return arr


def fused_gemm(X, W, chain: Sequence[Tuple[str, Dict]], rows: Optional[Sequence[int]] = None,
               nthreads: int = 0) -> np.ndarray:
    """Y = chain(X W^T) in fp64.  X [M, K], W [N, K] (fp32 or bf16).

    Returns float64 [len(rows) or M, N] (or [.., 1] after a row log-sum-exp or
    a row sum);
    output row r is input row ``rows[r]``."""
    lib = _load()
    keep: list = []
    x, xt = _np(X)
    w, wt = _np(W)
    M, K = x.shape
    N = w.shape[0]
    assert w.shape[1] == K
    ops = _ops(chain, keep)
    rows_a = None
    n_rows = M
    if rows is not None:
        rows_a = np.ascontiguousarray(np.asarray(rows, dtype=np.int64))
        n_rows = len(rows_a)
    Y = np.zeros((n_rows, N), dtype=np.float64)
    lib.orc_fused_gemm(_ptr(x), xt, K, _ptr(w), wt, K, M, N, K, ctypes.cast(ops, ctypes.c_void_p),
                       len(chain), None if rows_a is None else _ptr(rows_a), n_rows, _ptr(Y), N,
                       int(nthreads))
    if any(k in ("row_logsumexp", "row_sum") for k, _ in chain):
        return Y[:, :1].copy()
    return Y


def moe_route(logits, k: int):
    """Top-k routing + stable counting sort.  Returns a dict of numpy arrays:
    topk_ids int32 [T,k], topk_w f64 [T,k], offsets int32 [E+1],
    sorted_token int32 [T*k], sorted_w f64 [T*k], sorted_pair int32 [T*k]."""
    lib = _load()
    l, dt = _np(logits)
    assert dt == ORC_F32
    T, E = l.shape
    ids = np.zeros((T, k), np.int32)
    w = np.zeros((T, k), np.float64)
    off = np.zeros(E + 1, np.int32)
    st = np.zeros(T * k, np.int32)
    sw = np.zeros(T * k, np.float64)
    sp = np.zeros(T * k, np.int32)
    rc = lib.orc_moe_route(_ptr(l), T, E, k, _ptr(ids), _ptr(w), _ptr(off), _ptr(st), _ptr(sw), _ptr(sp))
    if rc != 0:
        raise ValueError("oracle moe_route: bad arguments")
    return dict(topk_ids=ids, topk_w=w, offsets=off, sorted_token=st, sorted_w=sw, sorted_pair=sp)


def moe_ffn(X, W_gu, W_down, topk_ids, topk_w, tokens: Optional[Sequence[int]] = None,
            round_h: bool = True, nthreads: int = 0, b_gu=None, b_down=None, alpha: float = 1.0,
            limit: float = 0.0, linear_offset: float = 0.0) -> np.ndarray:
    """Per-token MoE expert FFN in fp64 (h rounded to bf16 unless round_h=False).
    The expert activation is g' sigmoid(alpha g') (u' + linear_offset) with g, u
    clamped to (-inf, limit] / [-limit, limit] when limit > 0, after the optional
    per-expert biases b_gu [E, 2I] (gate then up, bf16); b_down [E, H] (bf16) is
    added to each expert's output before its routing weight.  The defaults are the
    plain SwiGLU.  Returns float64 [len(tokens), H]."""
    lib = _load()
    x, _ = _np(X)
    wg, _ = _np(W_gu)
    wd, _ = _np(W_down)
    T, H = x.shape
    I = wg.shape[1] // 2
    k = int(np.asarray(topk_ids).shape[1])
    ids = np.ascontiguousarray(np.asarray(topk_ids, dtype=np.int32))
    w = np.ascontiguousarray(np.asarray(topk_w, dtype=np.float64))
    toks = np.ascontiguousarray(np.arange(T, dtype=np.int64) if tokens is None
                                else np.asarray(tokens, dtype=np.int64))
    Y = np.zeros((len(toks), H), np.float64)
    bg = bd = None
    if b_gu is not None:
        bg, t1 = _np(b_gu)
        if t1 != ORC_BF16:
            raise TypeError("moe_ffn: b_gu must be bf16")
    if b_down is not None:
        bd, t2 = _np(b_down)
        if t2 != ORC_BF16:
            raise TypeError("moe_ffn: b_down must be bf16")
    lib.orc_moe_ffn(_ptr(x), _ptr(wg), _ptr(wd), _ptr(ids), _ptr(w), H, I, k, _ptr(toks), len(toks),
                    1 if round_h else 0, _ptr(Y), int(nthreads), None if bg is None else _ptr(bg),
                    None if bd is None else _ptr(bd), float(alpha), float(limit), float(linear_offset))
    return Y


def grouped_gemm(A, B, offsets, N: int, chain: Sequence[Tuple[str, Dict]], row_index=None,
                 out_rows: Optional[int] = None) -> np.ndarray:
    """Per-group GEMM + chain.  A [R_src, K]; B [G, nb, K] with nb = N (or 2N for
    SwiGLU); offsets int32 [G+1].  Returns float64 [rows_total, N], or the
    scatter target [out_rows, N] when the chain ends in row_scale_scatter_add."""
    lib = _load()
    keep: list = []
    a, at = _np(A)
    b, bt = _np(B)
    G = b.shape[0]
    K = a.shape[1]
    off = np.ascontiguousarray(np.asarray(offsets, dtype=np.int32))
    ri = None if row_index is None else np.ascontiguousarray(np.asarray(row_index, dtype=np.int32))
    ops = _ops(chain, keep)
    scatter = any(k == "row_scale_scatter_add" for k, _ in chain)
    rows = int(off[-1])
    out = np.zeros(((out_rows if scatter else rows), N), np.float64)
    lib.orc_grouped_gemm(_ptr(a), at, K, None if ri is None else _ptr(ri), _ptr(b), bt, K,
                         b.shape[1] * K, _ptr(off), G, N, K, ctypes.cast(ops, ctypes.c_void_p),
                         len(chain), _ptr(out), N)
    return out


def add_rmsnorm(Y, R, gamma, eps: float) -> Tuple[np.ndarray, np.ndarray]:
    """Block tail after the MoE FFN (Sec. IV-A, Fused Add + RMSNorm with the MoE
    finalize): R_out = bf16(R + Y); normed = R_out / sqrt(mean(R_out^2) + eps) *
    gamma per row.  Y float64 [T, H] (the unrounded MoE output), R [T, H] and
    gamma [H] at their stored dtype.  Returns (R_out, normed), float64."""
    lib = _load()
    y = np.ascontiguousarray(np.asarray(Y, dtype=np.float64))
    r, rt = _np(R)
    g, gt = _np(gamma)
    T, H = y.shape
    r_out = np.zeros((T, H), np.float64)
    normed = np.zeros((T, H), np.float64)
    st = lib.orc_add_rmsnorm(_ptr(y), _ptr(r), rt, _ptr(g), gt, float(eps), T, H, _ptr(r_out), _ptr(normed))
    if st != 0:
        raise ValueError("orc_add_rmsnorm: bad arguments")
    return r_out, normed


def qkv_rope_kv(X, W, bias, positions, cache_rows, cos_t, sin_t, nq: int, nkv: int, d: int, rows: int,
                k_cache=None, v_cache=None):
    """Bias + RoPE + KV-cache update of the QKV projection (Sec. IV-A) in fp64.
    X [T, H] and W [(nq + 2 nkv) d, H] of one dtype; bias or None; positions and
    cache_rows int32 [T]; cos_t / sin_t fp32 [max_pos, d/2].  Returns (q_out
    [T, nq d], k_cache [rows, nkv d], v_cache [rows, nkv d]) as float64; the
    caches start from the given arrays (NaN when None) and only the rows named
    by cache_rows change."""
    lib = _load()
    x, xt = _np(X)
    w, wt = _np(W)
    if xt != wt:
        raise TypeError("qkv_rope_kv: X and W must share one dtype")
    b, bt = (None, 0) if bias is None else _np(bias)
    T, H = x.shape
    pos = np.ascontiguousarray(np.asarray(positions, dtype=np.int32))
    crow = np.ascontiguousarray(np.asarray(cache_rows, dtype=np.int32))
    c, _ = _np(cos_t)
    sn, _ = _np(sin_t)
    max_pos = c.shape[0]
    q = np.zeros((T, nq * d), np.float64)
    kc = np.full((rows, nkv * d), np.nan) if k_cache is None else np.array(k_cache, dtype=np.float64, copy=True)
    vc = np.full((rows, nkv * d), np.nan) if v_cache is None else np.array(v_cache, dtype=np.float64, copy=True)
    st = lib.orc_qkv_rope_kv(_ptr(x), _ptr(w), xt, None if b is None else _ptr(b), bt, _ptr(pos), _ptr(crow), _ptr(c),
                             _ptr(sn), max_pos, T, H, nq, nkv, d, rows, _ptr(q), _ptr(kc), _ptr(vc))
    if st != 0:
        raise ValueError(f"orc_qkv_rope_kv: status {st}")
    return q, kc, vc


def round_bf16(x: float) -> float:
    """Nearest bf16 value of a double (ties to even)."""
    return _load().orc_round_bf16(float(x))
