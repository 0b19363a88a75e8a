"""Thin Python binding of the sm_103a fused GEMM + tail library (``libkf.so``).

Every function here only marshals arguments (device pointers, sizes, the
current CUDA stream) into the C ABI of ``include/kf.h``; all arithmetic runs in
the library's CUDA kernels.  PyTorch provides device memory and streams.  There
is no fallback: if ``libkf.so`` is missing the import of the library raises.

Tail chains are lists of ``(kind, params)``; kinds are the lower-case names of
``kf_op_kind`` (``bias, scale, relu, gelu_tanh, silu, sigmoid, residual_add,
row_logsumexp, groupnorm, swiglu, row_scale_scatter_add, mish, leaky_relu,
mul, row_scale, row_sum``); params ``p0, p1`` (device tensors), ``scalar, eps,
groups, ld``.

Workspaces start with a ``KF_WORKSPACE_HEADER_BYTES`` header holding the error
word of the calls given that workspace (``check_device_error``); the header must
be zero before first use: ``new_workspace`` allocates one that way, and the
workspaces the functions here allocate themselves are zeroed the same way.
"""
from __future__ import annotations

import ctypes
import os
from typing import Dict, Optional, Sequence, Tuple

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libkf.so")

KF_OK, KF_ERR_INVALID_ARG, KF_ERR_UNSUPPORTED, KF_ERR_MISALIGNED = 0, 1, 2, 3
KF_ERR_WORKSPACE, KF_ERR_CUDA, KF_ERR_DEVICE_TIMEOUT, KF_ERR_DEVICE_BOUNDS = 4, 5, 6, 7
KF_F32, KF_BF16, KF_I32, KF_F16 = 0, 1, 2, 3
OPS = {
    "bias": 0, "scale": 1, "relu": 2, "gelu_tanh": 3, "silu": 4, "sigmoid": 5,
    "residual_add": 6, "row_logsumexp": 7, "groupnorm": 8, "swiglu": 9,
    "row_scale_scatter_add": 10, "mish": 11, "leaky_relu": 12, "mul": 13, "row_scale": 14,
    "row_sum": 15,
}
ROW_REDUCTIONS = ("row_logsumexp", "row_sum")
KF_WORKSPACE_HEADER_BYTES = 256
KF_MOE_DETERMINISTIC = 1
# every entry point declared in include/kf.h
ABI_SYMBOLS = (
    "kf_fused_gemm", "kf_fused_gemm_workspace", "kf_moe_route", "kf_grouped_gemm",
    "kf_grouped_gemm_workspace", "kf_moe_ffn", "kf_moe_ffn_workspace", "kf_get_device_error",
    "kf_set_wait_timeout_ns", "kf_status_string", "kf_abi_version", "kf_fused_gemm_lse_noalloc",
    "kf_fused_gemm_lse_noalloc_max_bytes", "kf_moe_ffn_ex", "kf_moe_ffn_workspace_ex", "kf_moe_ffn_add_rmsnorm",
    "kf_qkv_rope_kv", "kf_moe_ffn_act", "kf_fused_gemm_ex", "kf_check_device_error", "kf_workspace_init",
)
KF_GEMM_F32_FFMA, KF_GEMM_F32_TF32X3 = 1, 2


class KfError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__(f"{where}: {status_string(status)} (status {status})")


class EpilogueOp(ctypes.Structure):
    _fields_ = [("kind", ctypes.c_int32), ("scalar", ctypes.c_float), ("eps", ctypes.c_float),
                ("groups", ctypes.c_int32), ("p0", ctypes.c_void_p), ("p1", ctypes.c_void_p),
                ("p_dtype", ctypes.c_int32), ("ld", ctypes.c_int64)]


class MoeAct(ctypes.Structure):
    _fields_ = [("alpha", ctypes.c_float), ("limit", ctypes.c_float), ("linear_offset", ctypes.c_float),
                ("b_gu", ctypes.c_void_p), ("b_down", ctypes.c_void_p)]


class Epilogue(ctypes.Structure):
    _fields_ = [("num_ops", ctypes.c_int32), ("ops", ctypes.POINTER(EpilogueOp))]


_lib = None


def lib() -> ctypes.CDLL:
    """The loaded C library with argument types set.  Raises if it is not built."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise ImportError(f"{LIB_PATH} is not built; run paper_2606_02963_gb300.build.build()")
    L = ctypes.CDLL(LIB_PATH)
    P, I32, I64, SZ = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_size_t
    EP = ctypes.POINTER(Epilogue)
    L.kf_fused_gemm.argtypes = [P, I32, I64, P, I32, I64, P, I32, I64, I64, I64, I64, EP, P, SZ, P]
    L.kf_fused_gemm_ex.argtypes = [P, I32, I64, P, I32, I64, P, I32, I64, I64, I64, I64, EP, P, SZ, ctypes.c_uint32, P]
    L.kf_fused_gemm_ex.restype = I32
    L.kf_fused_gemm_workspace.argtypes = [I64, I64, I64, EP]
    L.kf_fused_gemm_workspace.restype = SZ
    L.kf_moe_route.argtypes = [P, I64, I32, I32, P, P, P, P, P, P]
    L.kf_grouped_gemm.argtypes = [P, I32, I64, I64, P, P, I32, I64, I64, P, I32, I64, I64, I64, P, I32, I64,
                                  EP, P, SZ, P]
    L.kf_grouped_gemm_workspace.argtypes = [I64, I64, I64, I32, I32, EP]
    L.kf_grouped_gemm_workspace.restype = SZ
    L.kf_moe_ffn.argtypes = [P, P, P, P, P, I64, I64, I64, I32, I32, P, SZ, P, P, P]
    L.kf_moe_ffn_workspace.argtypes = [I64, I64, I64, I32, I32]
    L.kf_moe_ffn_workspace.restype = SZ
    L.kf_moe_ffn_ex.argtypes = [P, P, P, P, P, I64, I64, I64, I32, I32, ctypes.c_uint32, P, SZ, P, P, P]
    L.kf_moe_ffn_ex.restype = I32
    L.kf_moe_ffn_act.argtypes = [P, P, P, P, ctypes.POINTER(MoeAct), P, I64, I64, I64, I32, I32, ctypes.c_uint32, P,
                                 SZ, P, P, P]
    L.kf_moe_ffn_act.restype = I32
    L.kf_moe_ffn_add_rmsnorm.argtypes = [P, P, P, P, P, P, ctypes.c_float, P, P, I64, I64, I64, I32, I32,
                                         ctypes.c_uint32, P, SZ, P, P, P]
    L.kf_moe_ffn_add_rmsnorm.restype = I32
    L.kf_qkv_rope_kv.argtypes = [P, P, I32, I64, I64, P, I32, P, P, P, P, I64, I64, I64, I32, I32, I32, P, I64,
                                 P, P, I64, I64, I32, P]
    L.kf_qkv_rope_kv.restype = I32
    L.kf_moe_ffn_workspace_ex.argtypes = [I64, I64, I64, I32, I32, ctypes.c_uint32]
    L.kf_moe_ffn_workspace_ex.restype = SZ
    L.kf_get_device_error.argtypes = [P, ctypes.POINTER(ctypes.c_uint32)]
    L.kf_check_device_error.argtypes = [P, P, ctypes.POINTER(ctypes.c_uint32)]
    L.kf_check_device_error.restype = I32
    L.kf_workspace_init.argtypes = [P, SZ, P]
    L.kf_workspace_init.restype = I32
    L.kf_set_wait_timeout_ns.argtypes = [ctypes.c_uint64]
    L.kf_fused_gemm_lse_noalloc.argtypes = [P, I32, I64, P, I32, I64, P, I32, I64, I64, I64, EP, P]
    L.kf_fused_gemm_lse_noalloc.restype = I32
    L.kf_fused_gemm_lse_noalloc_max_bytes.restype = SZ
    L.kf_status_string.argtypes = [I32]
    L.kf_status_string.restype = ctypes.c_char_p
    L.kf_abi_version.restype = I32
    for f in ("kf_fused_gemm", "kf_moe_route", "kf_grouped_gemm", "kf_moe_ffn", "kf_get_device_error",
              "kf_set_wait_timeout_ns"):
        getattr(L, f).restype = I32
    _lib = L
    return L


def status_string(s: int) -> str:
    return lib().kf_status_string(int(s)).decode()


def _check(status: int, where: str):
    if status != KF_OK:
        raise KfError(status, where)


def _dt(t: torch.Tensor) -> int:
    if t.dtype == torch.bfloat16:
        return KF_BF16
    if t.dtype == torch.float32:
        return KF_F32
    if t.dtype == torch.int32:
        return KF_I32
    if t.dtype == torch.float16:
        return KF_F16
    raise TypeError(f"unsupported dtype {t.dtype}")


def _ptr(t: Optional[torch.Tensor]) -> Optional[int]:
    return None if t is None else t.data_ptr()


def _stream(stream=None) -> int:
    if stream is None:
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, torch.cuda.Stream):
        return stream.cuda_stream
    return int(stream)


def _rows(t: torch.Tensor, name: str):
    if t.dim() != 2 or t.stride(1) != 1:
        raise ValueError(f"{name} must be 2-D with unit column stride")
    return t.stride(0)


def make_epilogue(chain: Sequence[Tuple[str, Dict]], keep: list, default_ld: int = 0) -> Epilogue:
    """Build the C epilogue descriptor; tensors are kept alive in ``keep``."""
    arr = (EpilogueOp * max(1, len(chain)))()
    for i, (kind, prm) in enumerate(chain):
        o = arr[i]
        o.kind = OPS[kind]
        o.scalar = float(prm.get("scalar", 0.01 if kind == "leaky_relu" else 0.0))
        o.eps = float(prm.get("eps", 0.0))
        o.groups = int(prm.get("groups", 0))
        o.p_dtype = KF_F32
        o.ld = int(prm.get("ld", 0))
        for slot in ("p0", "p1"):
            v = prm.get(slot)
            if v is None:
                continue
            keep.append(v)
            setattr(o, slot, v.data_ptr())
            if slot == "p0" or (kind == "groupnorm" and prm.get("p0") is None):
                o.p_dtype = _dt(v)
            if slot == "p0" and kind == "residual_add" and "ld" not in prm:
                o.ld = v.stride(0)
        if kind == "row_scale_scatter_add" and "ld" not in prm:
            o.ld = default_ld
    keep.append(arr)
    return Epilogue(len(chain), ctypes.cast(arr, ctypes.POINTER(EpilogueOp)))


def new_workspace(nbytes: int, device, stream=None) -> torch.Tensor:
    """A workspace of ``nbytes`` (at least the header) with its header zeroed
    (kf_workspace_init on ``stream``)."""
    ws = torch.empty(max(int(nbytes), KF_WORKSPACE_HEADER_BYTES), dtype=torch.uint8, device=device)
    _check(lib().kf_workspace_init(ws.data_ptr(), ws.numel(), _stream(stream)), "kf_workspace_init")
    return ws


def _workspace(nbytes: int, device, workspace: Optional[torch.Tensor]) -> Tuple[Optional[torch.Tensor], int]:
    if workspace is None:
        if nbytes == 0:
            return None, 0
        workspace = new_workspace(nbytes, device)
    if workspace.numel() * workspace.element_size() < nbytes:
        raise ValueError("workspace too small")
    return workspace, workspace.numel() * workspace.element_size()


def fused_gemm(X: torch.Tensor, W: torch.Tensor, chain: Sequence[Tuple[str, Dict]] = (),
               out: Optional[torch.Tensor] = None, out_dtype: Optional[torch.dtype] = None,
               workspace: Optional[torch.Tensor] = None, f32_mode: Optional[str] = None, stream=None) -> torch.Tensor:
    """Y = chain(X W^T) on the GPU (kf_fused_gemm_ex).  Y is [M, N], or [M] after a
    row log-sum-exp (fp32 unless ``out_dtype`` says otherwise).  fp32 operands:
    ``f32_mode`` "ffma" or "tf32x3" forces a path (default: by problem size)."""
    M, K = X.shape
    N = W.shape[0]
    lse = any(k in ROW_REDUCTIONS for k, _ in chain)
    if out is None:
        dt = out_dtype or (torch.float32 if (lse or X.dtype == torch.float32) else X.dtype)
        out = torch.empty((M,) if lse else (M, N), dtype=dt, device=X.device)
    keep: list = []
    epi = make_epilogue(chain, keep)
    L = lib()
    ws_need = L.kf_fused_gemm_workspace(M, N, K, ctypes.byref(epi))
    ws, ws_bytes = _workspace(ws_need, X.device, workspace)
    ldy = out.stride(0) if out.dim() == 2 else 1
    flags = {None: 0, "ffma": KF_GEMM_F32_FFMA, "tf32x3": KF_GEMM_F32_TF32X3}[f32_mode]
    st = L.kf_fused_gemm_ex(X.data_ptr(), _dt(X), _rows(X, "X"), W.data_ptr(), _dt(W), _rows(W, "W"),
                            out.data_ptr(), _dt(out), ldy, M, N, K, ctypes.byref(epi), _ptr(ws), ws_bytes, flags,
                            _stream(stream))
    _check(st, "kf_fused_gemm_ex")
    return out


def moe_route(logits: torch.Tensor, k: int, stream=None) -> Dict[str, torch.Tensor]:
    """Top-k routing + stable sort by expert (kf_moe_route)."""
    T, E = logits.shape
    dev = logits.device
    r = dict(topk_ids=torch.empty(T, k, dtype=torch.int32, device=dev),
             topk_w=torch.empty(T, k, dtype=torch.float32, device=dev),
             offsets=torch.empty(E + 1, dtype=torch.int32, device=dev),
             sorted_token=torch.empty(T * k, dtype=torch.int32, device=dev),
             sorted_w=torch.empty(T * k, dtype=torch.float32, device=dev))
    st = lib().kf_moe_route(logits.data_ptr(), T, E, k, r["topk_ids"].data_ptr(), r["topk_w"].data_ptr(),
                            r["offsets"].data_ptr(), r["sorted_token"].data_ptr(), r["sorted_w"].data_ptr(),
                            _stream(stream))
    _check(st, "kf_moe_route")
    return r


def grouped_gemm(A: torch.Tensor, B: torch.Tensor, offsets: torch.Tensor, N: int,
                 chain: Sequence[Tuple[str, Dict]] = (), row_index: Optional[torch.Tensor] = None,
                 rows_total: Optional[int] = None, out: Optional[torch.Tensor] = None,
                 out_dtype: torch.dtype = torch.bfloat16, workspace: Optional[torch.Tensor] = None,
                 stream=None) -> torch.Tensor:
    """Per-group C rows = chain(A rows B[g]^T) (kf_grouped_gemm).  B is [G, nb, K]
    with nb = N (or 2N for SwiGLU); offsets int32 [G+1] on the device."""
    G, nb, K = B.shape
    if rows_total is None:
        rows_total = row_index.numel() if row_index is not None else A.shape[0]
    scatter = any(k == "row_scale_scatter_add" for k, _ in chain)
    if out is None:
        if scatter:
            raise ValueError("scatter-add needs the fp32 target `out`")
        out = torch.empty(rows_total, N, dtype=out_dtype, device=A.device)
    keep: list = []
    epi = make_epilogue(chain, keep, default_ld=out.shape[0])
    L = lib()
    ws_need = L.kf_grouped_gemm_workspace(rows_total, N, K, G, 1 if row_index is not None else 0,
                                          ctypes.byref(epi))
    ws, ws_bytes = _workspace(ws_need, A.device, workspace)
    st = L.kf_grouped_gemm(A.data_ptr(), _dt(A), _rows(A, "A"), A.shape[0], _ptr(row_index),
                           B.data_ptr(), _dt(B), B.stride(1), B.stride(0), offsets.data_ptr(), G, rows_total, N, K,
                           out.data_ptr(), _dt(out), out.stride(0), ctypes.byref(epi), _ptr(ws), ws_bytes,
                           _stream(stream))
    _check(st, "kf_grouped_gemm")
    return out


def moe_ffn_workspace_bytes(T: int, H: int, I: int, E: int, k: int, deterministic: bool = False) -> int:
    return lib().kf_moe_ffn_workspace_ex(T, H, I, E, k, KF_MOE_DETERMINISTIC if deterministic else 0)


def moe_ffn(X: torch.Tensor, logits: torch.Tensor, W_gu: torch.Tensor, W_down: torch.Tensor, k: int,
            out: Optional[torch.Tensor] = None, workspace: Optional[torch.Tensor] = None,
            return_routing: bool = False, deterministic: bool = False, act: Optional[Dict] = None, stream=None):
    """Routed MoE expert FFN (kf_moe_ffn_ex): route, gate/up + SwiGLU, down +
    scale + scatter-add (or, deterministic, per-row outputs summed in slot order),
    bf16 output.  With ``return_routing`` also returns (ids, w).  ``act`` (keys
    alpha, limit, linear_offset, b_gu [E, 2I], b_down [E, H]; kf_moe_ffn_act)
    selects the gated-expert activation with per-expert biases."""
    T, H = X.shape
    E, I2, _ = W_gu.shape
    I = I2 // 2
    for t, nm in ((X, "X"), (logits, "logits"), (W_gu, "W_gu"), (W_down, "W_down")):
        if not t.is_contiguous():
            raise ValueError(f"{nm} must be contiguous")
    if out is None:
        out = torch.empty(T, H, dtype=torch.bfloat16, device=X.device)
    L = lib()
    flags = KF_MOE_DETERMINISTIC if deterministic else 0
    ws, ws_bytes = _workspace(L.kf_moe_ffn_workspace_ex(T, H, I, E, k, flags), X.device, workspace)
    ids = w = None
    if return_routing:
        ids = torch.empty(T, k, dtype=torch.int32, device=X.device)
        w = torch.empty(T, k, dtype=torch.float32, device=X.device)
    if act is None:
        st = L.kf_moe_ffn_ex(X.data_ptr(), logits.data_ptr(), W_gu.data_ptr(), W_down.data_ptr(), out.data_ptr(), T,
                             H, I, E, k, flags, _ptr(ws), ws_bytes, _ptr(ids), _ptr(w), _stream(stream))
        _check(st, "kf_moe_ffn_ex")
    else:
        for nm in ("b_gu", "b_down"):
            b = act.get(nm)
            if b is not None and (b.dtype != torch.bfloat16 or not b.is_contiguous()):
                raise ValueError(f"{nm} must be contiguous bf16")
        a = MoeAct(float(act.get("alpha", 1.0)), float(act.get("limit", 0.0)), float(act.get("linear_offset", 0.0)),
                   _ptr(act.get("b_gu")), _ptr(act.get("b_down")))
        st = L.kf_moe_ffn_act(X.data_ptr(), logits.data_ptr(), W_gu.data_ptr(), W_down.data_ptr(), ctypes.byref(a),
                              out.data_ptr(), T, H, I, E, k, flags, _ptr(ws), ws_bytes, _ptr(ids), _ptr(w),
                              _stream(stream))
        _check(st, "kf_moe_ffn_act")
    return (out, ids, w) if return_routing else out


def moe_ffn_add_rmsnorm(X: torch.Tensor, logits: torch.Tensor, W_gu: torch.Tensor, W_down: torch.Tensor, k: int,
                        R: torch.Tensor, gamma: torch.Tensor, eps: float, out: Optional[torch.Tensor] = None,
                        r_out: Optional[torch.Tensor] = None, workspace: Optional[torch.Tensor] = None,
                        deterministic: bool = False, stream=None) -> Tuple[torch.Tensor, torch.Tensor]:
    """MoE block tail fused into the finalize (kf_moe_ffn_add_rmsnorm): returns
    (Y, R_out) with R_out = bf16(R + MoE(X)) and Y = bf16(rmsnorm(R_out) * gamma).
    ``r_out`` may be ``R`` (in-place residual update)."""
    T, H = X.shape
    E, I2, _ = W_gu.shape
    I = I2 // 2
    for t, nm in ((X, "X"), (logits, "logits"), (W_gu, "W_gu"), (W_down, "W_down"), (R, "R"), (gamma, "gamma")):
        if not t.is_contiguous():
            raise ValueError(f"{nm} must be contiguous")
    if out is None:
        out = torch.empty(T, H, dtype=torch.bfloat16, device=X.device)
    if r_out is None:
        r_out = torch.empty(T, H, dtype=torch.bfloat16, device=X.device)
    L = lib()
    flags = KF_MOE_DETERMINISTIC if deterministic else 0
    ws, ws_bytes = _workspace(L.kf_moe_ffn_workspace_ex(T, H, I, E, k, flags), X.device, workspace)
    st = L.kf_moe_ffn_add_rmsnorm(X.data_ptr(), logits.data_ptr(), W_gu.data_ptr(), W_down.data_ptr(), R.data_ptr(),
                                  gamma.data_ptr(), float(eps), r_out.data_ptr(), out.data_ptr(), T, H, I, E, k, flags,
                                  _ptr(ws), ws_bytes, None, None, _stream(stream))
    _check(st, "kf_moe_ffn_add_rmsnorm")
    return out, r_out


def qkv_rope_kv(X: torch.Tensor, W: torch.Tensor, bias: Optional[torch.Tensor], positions: torch.Tensor,
                cache_rows: torch.Tensor, cos_t: torch.Tensor, sin_t: torch.Tensor, nq: int, nkv: int, d: int,
                k_cache: torch.Tensor, v_cache: torch.Tensor, q_out: Optional[torch.Tensor] = None,
                stream=None) -> torch.Tensor:
    """QKV projection with bias, rotary embedding and key / value cache write
    (kf_qkv_rope_kv).  Writes rows ``cache_rows`` of ``k_cache`` / ``v_cache``
    ([rows, nkv d], their dtype is the output dtype) and returns the rotated
    queries [T, nq d]."""
    T, H = X.shape
    if q_out is None:
        q_out = torch.empty(T, nq * d, dtype=k_cache.dtype, device=X.device)
    if k_cache.dtype != v_cache.dtype or q_out.dtype != k_cache.dtype:
        raise TypeError("q_out, k_cache and v_cache must share one dtype")
    if k_cache.stride() != v_cache.stride() or k_cache.shape[0] != v_cache.shape[0]:
        raise ValueError("k_cache and v_cache must have one shape and row stride")
    for t, nm in ((positions, "positions"), (cache_rows, "cache_rows")):
        if t.dtype != torch.int32 or not t.is_contiguous() or t.numel() != T:
            raise ValueError(f"{nm} must be contiguous int32 [T]")
    for t, nm in ((cos_t, "cos_t"), (sin_t, "sin_t")):
        if t.dtype != torch.float32 or not t.is_contiguous() or t.shape[1] != d // 2:
            raise ValueError(f"{nm} must be contiguous fp32 [max_pos, d/2]")
    if bias is not None and not bias.is_contiguous():
        raise ValueError("bias must be contiguous")
    if _dt(X) != _dt(W):
        raise TypeError("X and W must share one dtype")
    L = lib()
    st = L.kf_qkv_rope_kv(X.data_ptr(), W.data_ptr(), _dt(X), _rows(X, "X"), _rows(W, "W"), _ptr(bias),
                              _dt(bias) if bias is not None else KF_BF16, positions.data_ptr(), cache_rows.data_ptr(),
                              cos_t.data_ptr(), sin_t.data_ptr(), cos_t.shape[0], T, H, nq, nkv, d,
                              q_out.data_ptr(), _rows(q_out, "q_out"), k_cache.data_ptr(), v_cache.data_ptr(),
                              _rows(k_cache, "k_cache"), k_cache.shape[0], _dt(k_cache), _stream(stream))
    _check(st, "kf_qkv_rope_kv")
    return q_out


def get_device_error(stream=None) -> Tuple[int, int]:
    """(status, raw bits) of this device's error word (every call on the
    device); synchronizes the stream and clears the word."""
    raw = ctypes.c_uint32(0)
    st = lib().kf_get_device_error(_stream(stream), ctypes.byref(raw))
    return st, raw.value


def check_device_error(workspace: torch.Tensor, stream=None) -> Tuple[int, int]:
    """(status, raw bits) of the error word in ``workspace``'s header (only the
    calls given that workspace); synchronizes the stream and clears the word."""
    raw = ctypes.c_uint32(0)
    st = lib().kf_check_device_error(workspace.data_ptr(), _stream(stream), ctypes.byref(raw))
    return st, raw.value


def set_wait_timeout_ns(ns: int) -> None:
    _check(lib().kf_set_wait_timeout_ns(int(ns)), "kf_set_wait_timeout_ns")
