"""Seeded synthetic workloads shared by the CUDA path's tests/bench and the oracle.

This module only draws random inputs and describes shapes; it holds none of the
arithmetic of the fused GEMM + tail path (no GEMM, no activation, no reduction).
Both sides receive exactly the tensors produced here: values are drawn in fp32
from one ``torch.Generator('cpu')`` per workload, in the order the workload lists
them, then rounded (round-to-nearest-even) to the workload dtype *before* either
side sees them, so the oracle and the kernels read identical operand values.

The workloads stand in for the GEMM + tail-op problems of the paper's Intel Arc
B580 study (Sec. IV-B, Table 3) and the gpt-oss-20b decode-path MoE of its B200
study (Sec. IV-A). Neither benchmark suite nor the model weights are available,
so shapes and distributions are synthetic.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field
from typing import Callable, Dict, List, Optional, Tuple

import torch

__all__ = ["Workload", "WORKLOADS", "generate", "chain_spec", "moe_generate", "MOE_SHAPE", "qkv_generate", "QKV_SHAPE"]


@dataclass(frozen=True)
class Workload:
    name: str
    M: int
    N: int
    K: int
    dtype: str                      # "f32" or "bf16": operand and output dtype
    # Tail chain as pure data: (kind, {param-name: tensor-key or scalar}).
    chain: Tuple[Tuple[str, Tuple[Tuple[str, object], ...]], ...]
    description: str = ""


def _ch(*ops):
    return tuple((k, tuple(sorted(p.items()))) for k, p in ops)


WORKLOADS: Dict[str, Workload] = {
    # fp32 ReLU linear, 128x256x512; X, W, b ~ U(-1, 1)
    "fp32_relu_linear": Workload(
        "fp32_relu_linear", 128, 256, 512, "f32",
        _ch(("bias", {"p0": "b"}), ("relu", {})),
        "fp32 Y = ReLU(X W^T + b), X[128x512], W[256x512], b[256] ~ U(-1,1)"),
    # bf16 GELU_tanh * 2 + R, 1024x4096x4096; all ~ N(0,1)/sqrt(K)
    "bf16_gelu_scale_residual": Workload(
        "bf16_gelu_scale_residual", 1024, 4096, 4096, "bf16",
        _ch(("bias", {"p0": "b"}), ("gelu_tanh", {}), ("scale", {"scalar": 2.0}),
            ("residual_add", {"p0": "R"})),
        "bf16 Y = GELU_tanh(X W^T + b) * 2 + R, 1024x4096x4096"),
    # bf16 GEMM * 0.125 -> row logsumexp, 2048x8192x8192
    "bf16_scale_rowlse": Workload(
        "bf16_scale_rowlse", 2048, 8192, 8192, "bf16",
        _ch(("scale", {"scalar": 0.125}), ("row_logsumexp", {})),
        "bf16 out[i] = logsumexp_j (X W^T)[i,j] * 0.125, fp32 [2048]"),
    # bf16 GEMM + b -> GroupNorm(16 x 512, eps 1e-5) -> Swish, 4096x8192x2048
    "bf16_groupnorm_swish": Workload(
        "bf16_groupnorm_swish", 4096, 8192, 2048, "bf16",
        _ch(("bias", {"p0": "b"}), ("groupnorm", {"groups": 16, "eps": 1e-5, "p0": "gamma", "p1": "beta"}),
            ("silu", {})),
        "bf16 Y = Swish(GroupNorm16(X W^T + b)), 4096x8192x2048"),
}


def chain_spec(wl: Workload) -> List[Tuple[str, Dict[str, object]]]:
    """The tail chain as a list of (kind, params) with params as a plain dict."""
    return [(k, dict(p)) for k, p in wl.chain]


def _round(t: torch.Tensor, dtype: str) -> torch.Tensor:
    if dtype == "bf16":
        return t.to(torch.bfloat16)
    if dtype == "f16":
        return t.to(torch.float16)
    return t.to(torch.float32)


def generate(name: str, seed: int = 0, M: Optional[int] = None, N: Optional[int] = None,
             K: Optional[int] = None, dist: str = "default", dtype: Optional[str] = None) -> Dict[str, torch.Tensor]:
    """Draw the inputs of workload ``name`` (optionally at another M/N/K).

    ``dist`` selects the distribution sweep used for parity only:
      "default"  the workload's own recipe,
      "unscaled" N(0,1) operands (no 1/sqrt(K)),
      "uniform"  U(-1,1) operands,
      "offset"   the default recipe plus a large constant (+8) on the bias / first
                 operand column, which stresses max-subtraction and cancellation.
    ``dtype`` ("bf16", "f16" or "f32") overrides the workload's dtype: the same
    fp32 draws, rounded (RNE) to that dtype instead.
    Returns CPU tensors in the workload dtype (fp32 for fp32 workloads).
    """
    wl = WORKLOADS[name]
    M = wl.M if M is None else M
    N = wl.N if N is None else N
    K = wl.K if K is None else K
    g = torch.Generator("cpu").manual_seed(seed)
    dt = wl.dtype if dtype is None else dtype
    out: Dict[str, torch.Tensor] = {}

    def normal(*shape, std=1.0):
        return torch.randn(*shape, generator=g, dtype=torch.float32) * std

    def uniform(*shape, lo=-1.0, hi=1.0):
        return torch.rand(*shape, generator=g, dtype=torch.float32) * (hi - lo) + lo

    s = 1.0 / math.sqrt(K)
    if dist == "unscaled":
        draw = lambda *sh: normal(*sh)
    elif dist == "uniform":
        draw = lambda *sh: uniform(*sh)
    else:
        draw = lambda *sh: normal(*sh, std=s)

    if name == "fp32_relu_linear":
        d = (lambda *sh: uniform(*sh)) if dist == "default" else draw
        out["X"] = d(M, K)
        out["W"] = d(N, K)
        out["b"] = d(N)
    elif name == "bf16_gelu_scale_residual":
        out["X"] = draw(M, K)
        out["W"] = draw(N, K)
        out["b"] = draw(N)
        out["R"] = draw(M, N)
    elif name == "bf16_scale_rowlse":
        out["X"] = draw(M, K)
        out["W"] = draw(N, K)
    elif name == "bf16_groupnorm_swish":
        out["X"] = draw(M, K)
        out["W"] = draw(N, K)
        out["b"] = draw(N)
        out["gamma"] = uniform(N, lo=0.5, hi=1.5)
        out["beta"] = uniform(N, lo=-0.1, hi=0.1)
    else:  # pragma: no cover
        raise KeyError(name)
    if dist == "offset":
        if "b" in out:
            out["b"] = out["b"] + 8.0
        else:
            out["X"][:, 0] += 8.0
    return {k: _round(v, dt) for k, v in out.items()}


# ---------------------------------------------------------------------------
# MoE expert FFN (gpt-oss-20b-shaped decode / prefill): hidden 2880, 32 experts,
# top-4 routing; W_gu[e] holds the gate rows (0..I-1) then the up rows (I..2I-1).
# ---------------------------------------------------------------------------
MOE_SHAPE = dict(H=2880, I=2880, E=32, k=4)


def moe_generate(T: int, seed: int = 0, H: int = 2880, I: int = 2880, E: int = 32,
                 k: int = 4, w_std: float = 0.02, device: str = "cpu") -> Dict[str, torch.Tensor]:
    """Draw X[T,H] ~ N(0,1), logits[T,E] ~ N(0,1) (fp32), W_gu[E,2I,H] and
    W_down[E,H,I] ~ N(0, w_std), all bf16 except the logits.

    ``device="cuda"`` draws the weights with a seeded CUDA generator (used only by
    the benchmark for speed; parity tests use the CPU generator)."""
    g = torch.Generator("cpu").manual_seed(seed)
    X = torch.randn(T, H, generator=g, dtype=torch.float32).to(torch.bfloat16)
    logits = torch.randn(T, E, generator=g, dtype=torch.float32)
    if device == "cpu":
        W_gu = (torch.randn(E, 2 * I, H, generator=g, dtype=torch.float32) * w_std).to(torch.bfloat16)
        W_down = (torch.randn(E, H, I, generator=g, dtype=torch.float32) * w_std).to(torch.bfloat16)
    else:
        gd = torch.Generator(device).manual_seed(seed + 1)
        W_gu = (torch.randn(E, 2 * I, H, generator=gd, device=device) * w_std).to(torch.bfloat16)
        W_down = (torch.randn(E, H, I, generator=gd, device=device) * w_std).to(torch.bfloat16)
    return dict(X=X, logits=logits, W_gu=W_gu, W_down=W_down)


QKV_SHAPE = dict(H=2880, nq=64, nkv=8, d=64)  # gpt-oss-20b attention input projection


def qkv_generate(T: int, seed: int = 0, H: int = 2880, nq: int = 64, nkv: int = 8, d: int = 64,
                 max_pos: int = 4096, cache_rows: Optional[int] = None, prefill: bool = False,
                 theta: float = 150000.0, w_std: float = 0.02, dtype: str = "bf16") -> Dict[str, torch.Tensor]:
    """Inputs of the QKV projection tail: X[T,H] ~ N(0,1); W[(nq+2nkv)d, H] ~
    N(0, w_std); bias ~ N(0, 0.1); fp32 rotary tables cos / sin(p * theta^(-2i/d))
    for p < max_pos, i < d/2 (the caller's tables; any frequency scaling would
    live here).  Decode (default): T sequences, each adding one token at a random
    position, into distinct random rows of a cache of ``cache_rows`` rows
    (default max(4096, 2T)).  Prefill: one sequence, positions 0..T-1, cache rows
    r0..r0+T-1."""
    g = torch.Generator("cpu").manual_seed(seed)
    N = (nq + 2 * nkv) * d
    rows = cache_rows if cache_rows is not None else max(4096, 2 * T)
    X = _round(torch.randn(T, H, generator=g, dtype=torch.float32), dtype)
    W = _round(torch.randn(N, H, generator=g, dtype=torch.float32) * w_std, dtype)
    b = _round(torch.randn(N, generator=g, dtype=torch.float32) * 0.1, dtype)
    if prefill:
        if T > max_pos or T > rows:
            raise ValueError("prefill longer than the tables or the cache")
        positions = torch.arange(T, dtype=torch.int32)
        r0 = int(torch.randint(0, rows - T + 1, (1,), generator=g))
        crow = torch.arange(r0, r0 + T, dtype=torch.int32)
    else:
        if T > rows:
            raise ValueError("more tokens than cache rows")
        positions = torch.randint(0, max_pos, (T,), generator=g, dtype=torch.int32)
        crow = torch.randperm(rows, generator=g)[:T].to(torch.int32)
    inv = theta ** (-torch.arange(0, d // 2, dtype=torch.float64) * 2.0 / d)
    ang = torch.arange(max_pos, dtype=torch.float64)[:, None] * inv[None, :]
    return dict(X=X, W=W, b=b, positions=positions, cache_rows=crow, cos=torch.cos(ang).float(),
                sin=torch.sin(ang).float(), rows=torch.tensor(rows))


# gpt-oss expert activation: sigmoid slope, clamp limit, offset on the linear branch
GPT_OSS_ACT = dict(alpha=1.702, limit=7.0, linear_offset=1.0)


def moe_bias_generate(E: int, H: int, I: int, seed: int = 0, std_gu: float = 0.5,
                      std_down: float = 0.1) -> Dict[str, torch.Tensor]:
    """Per-expert biases of the gated expert MLP: b_gu [E, 2I] (gate then up)
    ~ N(0, std_gu), b_down [E, H] ~ N(0, std_down), bf16."""
    g = torch.Generator("cpu").manual_seed(seed)
    return dict(b_gu=(torch.randn(E, 2 * I, generator=g) * std_gu).to(torch.bfloat16),
                b_down=(torch.randn(E, H, generator=g) * std_down).to(torch.bfloat16))
