"""GPU parity of the tail-chain shapes of the paper's GEMM + tail problems
(Sec. IV-B, Table 3): element-wise ops before a GroupNorm, element-wise ops and a
per-column multiply after it, and a scalar op after the row log-sum-exp -- at
ragged sizes, through the paths the chain selects (interpreter chains, couples
of CTA pairs for 512-column groups, whole groups per tile for narrower ones)."""
import pytest
import torch

import kf_workloads
import oracle
import paper_2606_02963_gb300 as kf
from tests._util import check_bf16, check_f32, chain_to

pytestmark = pytest.mark.gpu
DEV = "cuda"


def _inputs(seed, M, N, K):
    inp = kf_workloads.generate("bf16_groupnorm_swish", seed=seed, M=M, N=N, K=K, dist="unscaled")
    g = torch.Generator().manual_seed(seed + 100)
    inp["v"] = (torch.rand(N, generator=g) + 0.5).to(torch.bfloat16)  # per-column multiplier
    return inp


def _chains(inp, groups):
    gn = ("groupnorm", {"groups": groups, "eps": 1e-5, "p0": inp["gamma"], "p1": inp["beta"]})
    return {
        # Swish, then a bias sum, then GroupNorm
        "swish_bias_gn": [("silu", {}), ("bias", {"p0": inp["b"]}), gn],
        # GroupNorm, Swish, per-column multiply, Swish
        "gn_swish_mul_swish": [("bias", {"p0": inp["b"]}), gn, ("silu", {}), ("mul", {"p0": inp["v"]}), ("silu", {})],
        # GroupNorm, LeakyReLU, then the sum of the result with itself
        "gn_lrelu_sum": [gn, ("leaky_relu", {"scalar": 0.01}), ("scale", {"scalar": 2.0})],
    }


@pytest.mark.parametrize("N,groups", [(1536, 3), (1024, 4), (768, 6)])  # 512-, 256-, 128-column groups
@pytest.mark.parametrize("pattern", ["swish_bias_gn", "gn_swish_mul_swish", "gn_lrelu_sum"])
@pytest.mark.parametrize("out_dtype", [torch.bfloat16, torch.float32])
def test_groupnorm_chain_patterns(N, groups, pattern, out_dtype):
    M, K = 300, 200
    inp = _inputs(31, M, N, K)
    chain = _chains(inp, groups)[pattern]
    Y = kf.fused_gemm(inp["X"].to(DEV), inp["W"].to(DEV), chain_to(chain, DEV), out_dtype=out_dtype)
    ref = oracle.fused_gemm(inp["X"], inp["W"], chain)
    if out_dtype == torch.float32:
        check_f32(Y, ref, f"{pattern} gs={N // groups}")
    else:
        check_bf16(Y, ref, f"{pattern} gs={N // groups}")
    assert kf.get_device_error()[0] == kf.KF_OK


@pytest.mark.parametrize("post", [("mish", {}), ("leaky_relu", {"scalar": 0.2}), ("scale", {"scalar": -0.5})])
def test_scale_lse_then_scalar_op(post):
    inp = kf_workloads.generate("bf16_scale_rowlse", seed=33, M=300, N=1000, K=200, dist="unscaled")
    chain = [("scale", {"scalar": 0.125}), ("row_logsumexp", {}), post]
    Y = kf.fused_gemm(inp["X"].to(DEV), inp["W"].to(DEV), chain)
    check_f32(Y, oracle.fused_gemm(inp["X"], inp["W"], chain)[:, 0], f"lse + {post[0]}")
    assert kf.get_device_error()[0] == kf.KF_OK
