"""GPU parity of the fp16-operand path (the paper's B580 kernels ran their
matmuls in fp16 with fp32 accumulation and post-processing, Sec. IV-B):
tcgen05 kind::f16 with fp16 A and B, fp16 / bf16 / fp32 outputs and fp16
epilogue operands, against the oracle reading the same fp16 values."""
import numpy as np
import pytest
import torch

import kf_workloads
import oracle
import paper_2606_02963_gb300 as kf
from tests._util import check_bf16, check_f32, chain_to, wl_chain

pytestmark = pytest.mark.gpu
DEV = "cuda"


def _err_ok():
    assert kf.get_device_error()[0] == kf.KF_OK


@pytest.mark.parametrize("M,N,K", [(128, 256, 64), (300, 520, 136), (1, 16, 8)])
def test_f16_integer_gemm_is_bit_exact(M, N, K):
    # small integers are exact in fp16 and every partial sum is exact in fp32
    g = torch.Generator().manual_seed(M + N)
    X = torch.randint(-4, 5, (M, K), generator=g).to(torch.float16)
    W = torch.randint(-4, 5, (N, K), generator=g).to(torch.float16)
    Y = kf.fused_gemm(X.to(DEV), W.to(DEV), [], out_dtype=torch.float32)
    assert np.array_equal(Y.cpu().numpy().astype(np.float64), oracle.fused_gemm(X, W, []))
    _err_ok()


@pytest.mark.parametrize("out_dtype", [torch.float16, torch.bfloat16, torch.float32])
@pytest.mark.parametrize("dist", ["default", "unscaled"])
def test_f16_gelu_chain(out_dtype, dist):
    inp = kf_workloads.generate("bf16_gelu_scale_residual", seed=41, M=300, N=520, K=264, dist=dist, dtype="f16")
    chain = wl_chain("bf16_gelu_scale_residual", inp)
    Y = kf.fused_gemm(inp["X"].to(DEV), inp["W"].to(DEV), chain_to(chain, DEV), out_dtype=out_dtype)
    ref = oracle.fused_gemm(inp["X"], inp["W"], chain)
    if out_dtype == torch.float32:
        check_f32(Y, ref, f"f16 gelu {dist}")
    else:
        check_bf16(Y, ref, f"f16 gelu {dist} -> {out_dtype}")
    _err_ok()


@pytest.mark.parametrize("out_dtype", [torch.float32, torch.float16])
def test_f16_row_logsumexp(out_dtype):
    inp = kf_workloads.generate("bf16_scale_rowlse", seed=42, M=300, N=1000, K=200, dist="unscaled", dtype="f16")
    chain = [("scale", {"scalar": 0.125}), ("row_logsumexp", {})]
    Y = kf.fused_gemm(inp["X"].to(DEV), inp["W"].to(DEV), chain, out_dtype=out_dtype)
    ref = oracle.fused_gemm(inp["X"], inp["W"], chain)[:, 0]
    if out_dtype == torch.float32:
        check_f32(Y, ref, "f16 lse")
    else:
        check_bf16(Y, ref, "f16 lse -> f16")
    _err_ok()


@pytest.mark.parametrize("N,groups", [(1536, 3), (1024, 4), (768, 6)])
def test_f16_groupnorm_swish(N, groups):
    inp = kf_workloads.generate("bf16_groupnorm_swish", seed=43, M=300, N=N, K=200, dtype="f16")
    chain = [("bias", {"p0": inp["b"]}),
             ("groupnorm", {"groups": groups, "eps": 1e-5, "p0": inp["gamma"], "p1": inp["beta"]}),
             ("silu", {})]
    Y = kf.fused_gemm(inp["X"].to(DEV), inp["W"].to(DEV), chain_to(chain, DEV))
    assert Y.dtype == torch.float16
    check_bf16(Y, oracle.fused_gemm(inp["X"], inp["W"], chain), f"f16 gn gs={N // groups}")
    _err_ok()


def test_f16_full_size_headline_sampled_rows():
    inp = kf_workloads.generate("bf16_gelu_scale_residual", seed=44, dtype="f16")
    d = {k: v.to(DEV) for k, v in inp.items()}
    Y = kf.fused_gemm(d["X"], d["W"], wl_chain("bf16_gelu_scale_residual", d))
    torch.cuda.synchronize()
    rows = [0, 1, 255, 256, 1023]
    ref = oracle.fused_gemm(inp["X"], inp["W"], wl_chain("bf16_gelu_scale_residual", inp), rows=rows)
    check_bf16(Y[rows], ref, "f16 headline")
    _err_ok()
