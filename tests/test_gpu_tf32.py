"""GPU parity of the fp32 GEMM + tail on the tensor cores (3xTF32: each fp32
operand split into a tf32 high part and an fp32 remainder, three products
accumulated in fp32) against the fp64 oracle, within the fp32 tolerance, on
ragged shapes, both tile widths, fp32 / bf16 / fp16 outputs, and at the size
where the automatic choice takes it."""
import numpy as np
import pytest
import torch

import oracle
import paper_2606_02963_gb300 as kf
from tests._util import check_bf16, check_f32

pytestmark = pytest.mark.gpu
DEV = "cuda"


def _case(M, N, K, seed, scale=1.0):
    g = torch.Generator().manual_seed(seed)
    X = torch.randn(M, K, generator=g) * scale
    W = torch.randn(N, K, generator=g) / np.sqrt(K)
    b = torch.randn(N, generator=g)
    return X, W, b


@pytest.mark.parametrize("M,N,K", [(300, 200, 100), (129, 257, 72), (1, 64, 32), (1000, 1000, 1024),
                                   (640, 4096, 512)])
@pytest.mark.parametrize("chain_name", ["plain", "bias_relu", "bias_gelu_scale"])
def test_tf32x3_matches_oracle(M, N, K, chain_name):
    X, W, b = _case(M, N, K, seed=M + N + K)
    chains = {"plain": [], "bias_relu": [("bias", {"p0": b}), ("relu", {})],
              "bias_gelu_scale": [("bias", {"p0": b}), ("gelu_tanh", {}), ("scale", {"scalar": 0.5})]}
    chain = chains[chain_name]
    dchain = [(k, {kk: (v.to(DEV) if isinstance(v, torch.Tensor) else v) for kk, v in p.items()}) for k, p in chain]
    Y = kf.fused_gemm(X.to(DEV), W.to(DEV), dchain, f32_mode="tf32x3")
    ref = oracle.fused_gemm(X, W, chain)
    check_f32(Y, ref, f"3xTF32 {M}x{N}x{K} {chain_name}")
    assert kf.get_device_error()[0] == kf.KF_OK


@pytest.mark.parametrize("out_dtype", [torch.bfloat16, torch.float16])
def test_tf32x3_narrow_outputs(out_dtype):
    X, W, b = _case(300, 520, 256, seed=7)
    Y = kf.fused_gemm(X.to(DEV), W.to(DEV), [("bias", {"p0": b.to(DEV)})], out_dtype=out_dtype, f32_mode="tf32x3")
    check_bf16(Y, oracle.fused_gemm(X, W, [("bias", {"p0": b})]), f"3xTF32 -> {out_dtype}")
    assert kf.get_device_error()[0] == kf.KF_OK


def test_tf32x3_error_is_fp32_class_not_tf32_class():
    # large-magnitude inputs: one tf32 product (cuBLAS with TF32 allowed) is off
    # by ~1e-3 of the rms; the three-product split stays within the fp32
    # tolerance and at least 10x below the single product
    X, W, _ = _case(256, 384, 1024, seed=8, scale=100.0)
    Xd, Wd = X.to(DEV), W.to(DEV)
    y3 = kf.fused_gemm(Xd, Wd, [], f32_mode="tf32x3").double().cpu().numpy()
    yf = kf.fused_gemm(Xd, Wd, [], f32_mode="ffma").double().cpu().numpy()
    prev = torch.backends.cuda.matmul.allow_tf32
    torch.backends.cuda.matmul.allow_tf32 = True
    try:
        y1 = torch.mm(Xd, Wd.t()).double().cpu().numpy()
    finally:
        torch.backends.cuda.matmul.allow_tf32 = prev
    ref = oracle.fused_gemm(X, W, [])
    rms = np.sqrt(np.mean(ref ** 2))
    e3, ef, e1 = (np.abs(y - ref).max() / rms for y in (y3, yf, y1))
    assert e3 < 1e-4 and e3 < e1 / 10, (e3, ef, e1)
    assert kf.get_device_error()[0] == kf.KF_OK


def test_large_fp32_gemm_takes_tensor_cores_and_matches_sampled_rows():
    # 2 M N K = 34 GFLOP: the default path is 3xTF32 with 256-column tiles
    M = N = K = 2048
    X, W, b = _case(M, N, K, seed=9)
    Y = kf.fused_gemm(X.to(DEV), W.to(DEV), [("bias", {"p0": b.to(DEV)})])
    rows = [0, 1, 127, 128, 1000, M - 1]
    ref = oracle.fused_gemm(X, W, [("bias", {"p0": b})], rows=rows)
    check_f32(Y[rows], ref, "3xTF32 default 2048^3")
    Yf = kf.fused_gemm(X.to(DEV), W.to(DEV), [("bias", {"p0": b.to(DEV)})], f32_mode="ffma")
    check_f32(Yf[rows], ref, "FFMA 2048^3")
    assert kf.get_device_error()[0] == kf.KF_OK
