"""GPU parity of the row sum (KF_OP_ROW_SUM): the 'Sum' that ends the paper's
Table 3 chains (Sec. IV-B), read as a reduction over each row.  It runs in the
GEMM's epilogue (per-tile row partials, then a fixed-order combine) after a
pointwise chain, or after a GroupNorm and its post chain (Matmul, GroupNorm,
LeakyReLU, Sum).  Integer operands make every partial sum exact, so those cases
must match the oracle bit for bit; the others hold the fp32 / bf16 tolerances."""
import numpy as np
import pytest
import torch

import kf_workloads
import oracle
import paper_2606_02963_gb300 as kf
from tests._util import check_bf16, check_f32, chain_to, to_np

pytestmark = pytest.mark.gpu
DEV = "cuda"


def _ints(shape, lo, hi, g):
    return torch.randint(lo, hi + 1, shape, generator=g).float().to(torch.bfloat16)


def _no_device_error():
    st, raw = kf.get_device_error()
    assert st == kf.KF_OK, f"device error word {raw:#x}"


@pytest.mark.parametrize("M,N,K", [(1, 16, 8), (100, 300, 64), (200, 300, 136), (384, 4480, 64), (129, 257, 72)])
def test_row_sum_integer_is_bit_exact(M, N, K):
    # |x w| <= 16 and K <= 136: each product sum and each row sum stay below 2^24
    g = torch.Generator().manual_seed(M + 7 * N + 13 * K)
    X, W = _ints((M, K), -4, 4, g), _ints((N, K), -4, 4, g)
    b = _ints((N,), -8, 8, g)
    chain = [("bias", {"p0": b}), ("relu", {}), ("row_sum", {})]
    Y = kf.fused_gemm(X.to(DEV), W.to(DEV), chain_to(chain, DEV))
    assert Y.shape == (M,) and Y.dtype == torch.float32
    ref = oracle.fused_gemm(X, W, chain)[:, 0]
    assert np.array_equal(to_np(Y), ref)
    _no_device_error()


@pytest.mark.parametrize("M,N,K,dist", [(200, 1000, 136, "default"), (300, 2500, 264, "unscaled"),
                                        (130, 300, 64, "offset"), (64, 33, 40, "uniform")])
def test_row_sum_after_pointwise_chain(M, N, K, dist):
    inp = kf_workloads.generate("bf16_gelu_scale_residual", seed=41, M=M, N=N, K=K, dist=dist)
    chain = [("bias", {"p0": inp["b"]}), ("leaky_relu", {"scalar": 0.01}), ("row_sum", {}), ("scale", {"scalar": 0.5})]
    Y = kf.fused_gemm(inp["X"].to(DEV), inp["W"].to(DEV), chain_to(chain, DEV))
    check_f32(Y, oracle.fused_gemm(inp["X"], inp["W"], chain)[:, 0], f"row sum {dist}")
    Yb = kf.fused_gemm(inp["X"].to(DEV), inp["W"].to(DEV), chain_to(chain, DEV), out_dtype=torch.bfloat16)
    check_bf16(Yb, oracle.fused_gemm(inp["X"], inp["W"], chain)[:, 0], f"row sum {dist} bf16")
    # the combine adds the partials in a fixed order: repeated calls agree bit for bit
    Y2 = kf.fused_gemm(inp["X"].to(DEV), inp["W"].to(DEV), chain_to(chain, DEV))
    assert torch.equal(Y, Y2)
    _no_device_error()


def test_row_sum_full_size_sampled_rows():
    # the row log-sum-exp workload's shape (2048 x 8192 x 8192) with the row sum
    inp = kf_workloads.generate("bf16_scale_rowlse", seed=0)
    chain = [("scale", {"scalar": 0.125}), ("row_sum", {})]
    Y = kf.fused_gemm(inp["X"].to(DEV), inp["W"].to(DEV), chain)
    rows = [0, 1, 127, 128, 255, 256, 1023, 1500, 2046, 2047]
    ref = oracle.fused_gemm(inp["X"], inp["W"], chain, rows=rows)[:, 0]
    # fp32 tolerance against the sampled rows' own scale (their rms)
    check_f32(to_np(Y)[rows], ref, "row sum 2048x8192x8192")
    _no_device_error()


def _gn_chain(inp, groups):
    return [("bias", {"p0": inp["b"]}),
            ("groupnorm", {"groups": groups, "eps": 1e-5, "p0": inp["gamma"], "p1": inp["beta"]}),
            ("leaky_relu", {"scalar": 0.01}), ("row_sum", {})]


# 512-column groups on clusters of four (M > 128) or one CTA with two
# accumulators (M <= 128); 256-column groups one per tile; 128-column groups
# several per tile
@pytest.mark.parametrize("M,N,groups", [(300, 1536, 3), (100, 1024, 2), (300, 1024, 4), (257, 768, 6)])
@pytest.mark.parametrize("out_dtype", [torch.float32, torch.bfloat16])
def test_groupnorm_lrelu_row_sum(M, N, groups, out_dtype):
    inp = kf_workloads.generate("bf16_groupnorm_swish", seed=43, M=M, N=N, K=200, dist="unscaled")
    chain = _gn_chain(inp, groups)
    Y = kf.fused_gemm(inp["X"].to(DEV), inp["W"].to(DEV), chain_to(chain, DEV), out_dtype=out_dtype)
    assert Y.shape == (M,)
    ref = oracle.fused_gemm(inp["X"], inp["W"], chain)[:, 0]
    if out_dtype == torch.float32:
        check_f32(Y, ref, f"gn sum gs={N // groups}")
    else:
        check_bf16(Y, ref, f"gn sum gs={N // groups}")
    _no_device_error()


def test_groupnorm_lrelu_row_sum_scalar_after_and_integer_exactness():
    # constant groups normalise to beta exactly: with gamma = 1 and integer beta
    # every value after the GroupNorm is beta_j, so each row sums to sum_j
    # lrelu(beta_j) * 3 exactly (the scale follows the sum)
    M, N, K = 260, 1024, 64
    X = torch.ones(M, K).to(torch.bfloat16)
    W = torch.zeros(N, K).to(torch.bfloat16)
    beta = torch.randint(-4, 5, (N,), generator=torch.Generator().manual_seed(44)).float()
    chain = [("groupnorm", {"groups": 2, "eps": 1e-5, "p1": beta}), ("leaky_relu", {"scalar": 0.25}),
             ("row_sum", {}), ("scale", {"scalar": 3.0})]
    Y = kf.fused_gemm(X.to(DEV), W.to(DEV), chain_to(chain, DEV))
    want = float(torch.where(beta > 0, beta, 0.25 * beta).sum()) * 3.0
    assert np.all(to_np(Y) == want)
    assert np.all(oracle.fused_gemm(X, W, chain)[:, 0] == want)
    _no_device_error()


def test_groupnorm_lrelu_row_sum_full_size_sampled_rows():
    # the GroupNorm workload's shape (4096 x 8192 x 2048, 16 groups of 512)
    inp = kf_workloads.generate("bf16_groupnorm_swish", seed=0)
    chain = _gn_chain(inp, 16)
    Y = kf.fused_gemm(inp["X"].to(DEV), inp["W"].to(DEV), chain_to(chain, DEV))
    rows = [0, 1, 255, 256, 2047, 2048, 4094, 4095]
    ref = oracle.fused_gemm(inp["X"], inp["W"], chain, rows=rows)[:, 0]
    check_f32(to_np(Y)[rows], ref, "gn sum 4096x8192x2048")
    _no_device_error()
