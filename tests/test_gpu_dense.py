"""GPU parity of kf_fused_gemm against the fp64 oracle (element by element at
sizes spanning several tiles with ragged tails; sampled rows at the full
workload sizes, in the launch configuration the benchmark times)."""
import numpy as np
import pytest
import torch

import kf_workloads
import oracle
import paper_2606_02963_gb300 as kf
from tests._util import check_bf16, check_f32, chain_to, to_np, wl_chain

pytestmark = pytest.mark.gpu
DEV = "cuda"


def _ints(shape, lo, hi, g):
    return torch.randint(lo, hi + 1, shape, generator=g).float().to(torch.bfloat16)


def _no_device_error():
    st, raw = kf.get_device_error()
    assert st == kf.KF_OK, f"device error word {raw:#x}"


# ------------------------------------------------------------- exact GEMM core
@pytest.mark.parametrize("M,N,K", [(128, 256, 64), (256, 512, 128), (200, 300, 136), (1, 16, 8),
                                   (129, 257, 72), (384, 448, 256)])
def test_integer_gemm_is_bit_exact(M, N, K):
    """Small-integer bf16 operands make every product and partial sum exact in
    fp32 (|sum| < 2^24), so the tensor-core result must equal the oracle exactly:
    this pins the tile layout, swizzle, descriptors and ragged-edge masking."""
    g = torch.Generator().manual_seed(M * 7 + N * 3 + K)
    X, W = _ints((M, K), -4, 4, g), _ints((N, K), -4, 4, g)
    Y = kf.fused_gemm(X.to(DEV), W.to(DEV), [], out_dtype=torch.float32)
    torch.cuda.synchronize()
    ref = oracle.fused_gemm(X, W, [])
    assert np.array_equal(to_np(Y), ref)
    _no_device_error()


def test_integer_gemm_bf16_output_is_rne_of_exact():
    g = torch.Generator().manual_seed(5)
    X, W = _ints((160, 192), -8, 8, g), _ints((288, 192), -8, 8, g)
    Y = kf.fused_gemm(X.to(DEV), W.to(DEV), [])
    ref = torch.from_numpy(oracle.fused_gemm(X, W, [])).float().to(torch.bfloat16)
    assert torch.equal(Y.cpu(), ref)


def test_strided_operands_and_output():
    g = torch.Generator().manual_seed(6)
    Xb = _ints((150, 136), -3, 3, g)
    Wb = _ints((90, 200), -3, 3, g)
    X, W = Xb[:, :128], Wb[:, :128]
    out = torch.zeros(150, 104, dtype=torch.float32, device=DEV)
    kf.fused_gemm(Xb.to(DEV)[:, :128], Wb.to(DEV)[:, :128], [], out=out[:, :90])
    ref = oracle.fused_gemm(X.contiguous(), W.contiguous(), [])
    assert np.array_equal(to_np(out[:, :90]), ref)
    assert torch.count_nonzero(out[:, 90:]) == 0


# --------------------------------------------------------- element-wise tails
OPS_ALONE = [
    [("bias", {"p0": "b"})],
    [("scale", {"scalar": -1.5})],
    [("relu", {})],
    [("gelu_tanh", {})],
    [("silu", {})],
    [("sigmoid", {})],
    [("residual_add", {"p0": "R"})],
    [("mish", {})],
    [("leaky_relu", {"scalar": 0.1})],
    [("mul", {"p0": "b"})],
]


@pytest.mark.parametrize("ops", OPS_ALONE, ids=lambda o: o[0][0])
@pytest.mark.parametrize("out_dtype", [torch.bfloat16, torch.float32])
def test_each_tail_op(ops, out_dtype):
    inp = kf_workloads.generate("bf16_gelu_scale_residual", seed=3, M=200, N=300, K=136, dist="unscaled")
    chain = [(k, {kk: (inp[v] if kk == "p0" else v) for kk, v in p.items()}) for k, p in ops]
    Y = kf.fused_gemm(inp["X"].to(DEV), inp["W"].to(DEV), chain_to(chain, DEV), out_dtype=out_dtype)
    ref = oracle.fused_gemm(inp["X"], inp["W"], chain)
    if out_dtype == torch.float32:
        check_f32(Y, ref, str(ops))
    else:
        check_bf16(Y, ref, str(ops))


@pytest.mark.parametrize("dist", ["default", "unscaled", "uniform", "offset"])
def test_gelu_scale_residual_chain_sweep(dist):
    inp = kf_workloads.generate("bf16_gelu_scale_residual", seed=4, M=300, N=520, K=264, dist=dist)
    chain = wl_chain("bf16_gelu_scale_residual", inp)
    Y = kf.fused_gemm(inp["X"].to(DEV), inp["W"].to(DEV), chain_to(chain, DEV))
    check_bf16(Y, oracle.fused_gemm(inp["X"], inp["W"], chain), dist)
    _no_device_error()


@pytest.mark.parametrize("path", ["interpreter", "residual_tile"])
def test_gelu_far_outside_fp16_range(path):
    """Pre-activations of +-1e3, +-7e4 and +-3e5 (bf16-exact) among ordinary
    ones: GELU gives x above zero and ~0 below, never inf or NaN, on the packed
    fp16 path bf16 outputs take.  X = I makes X W^T = W^T exactly."""
    g = torch.Generator().manual_seed(31)
    M = K = 256
    N = 512
    big = torch.tensor([1e3, -1e3, 7e4, -7e4, 3e5, -3e5]).to(torch.bfloat16).float()
    vals = torch.randn(M, N, generator=g) * 3
    idx = torch.randperm(M * N, generator=g)[:M * N // 7]
    vals.view(-1)[idx] = big[torch.arange(idx.numel()) % big.numel()]
    vals = vals.to(torch.bfloat16)
    X = torch.eye(K).to(torch.bfloat16)
    W = vals.t().contiguous()
    if path == "interpreter":
        chain = [("gelu_tanh", {})]
    else:  # the headline's compiled chain on CTA pairs (residual tile in shared memory)
        chain = [("bias", {"p0": torch.zeros(N).to(torch.bfloat16)}), ("gelu_tanh", {}), ("scale", {"scalar": 2.0}),
                 ("residual_add", {"p0": torch.zeros(M, N).to(torch.bfloat16)})]
    Y = kf.fused_gemm(X.to(DEV), W.to(DEV), chain_to(chain, DEV))
    ref = oracle.fused_gemm(X, W, chain)
    y = to_np(Y)
    assert np.isfinite(y).all()
    check_bf16(Y, ref, path)
    f = 1.0 if path == "interpreter" else 2.0
    x = vals.double().numpy()
    hi, lo = x >= 1e3, x <= -1e3
    assert np.all(np.abs(y[hi] - f * x[hi]) <= 1e-2 * f * x[hi])
    assert np.all(np.abs(y[lo]) <= 1e-2)
    _no_device_error()


@pytest.mark.parametrize("in_place", [False, True])
def test_gelu_chain_more_tiles_than_cta_pairs(in_place):
    # 4 ragged 256-row tiles x 20 column tiles of 224 = 80 tiles: more than the
    # CTA pairs of the grid, so pairs run a second tile and reload their
    # residual tile in shared memory after the first tile's stores
    inp = kf_workloads.generate("bf16_gelu_scale_residual", seed=14, M=1000, N=4480, K=136, dist="unscaled")
    chain = wl_chain("bf16_gelu_scale_residual", inp)
    ref = oracle.fused_gemm(inp["X"], inp["W"], chain)
    gchain = chain_to(chain, DEV)
    if in_place:
        R = inp["R"].to(DEV).clone()
        gchain[-1] = ("residual_add", {"p0": R})
        Y = kf.fused_gemm(inp["X"].to(DEV), inp["W"].to(DEV), gchain, out=R)
    else:
        Y = kf.fused_gemm(inp["X"].to(DEV), inp["W"].to(DEV), gchain)
    check_bf16(Y, ref, f"80 tiles, in place {in_place}")
    _no_device_error()


def test_residual_in_place():
    inp = kf_workloads.generate("bf16_gelu_scale_residual", seed=8, M=256, N=256, K=128)
    chain = wl_chain("bf16_gelu_scale_residual", inp)
    ref = oracle.fused_gemm(inp["X"], inp["W"], chain)
    R = inp["R"].to(DEV).clone()
    gchain = chain_to(chain, DEV)
    gchain[-1] = ("residual_add", {"p0": R})
    kf.fused_gemm(inp["X"].to(DEV), inp["W"].to(DEV), gchain, out=R)
    check_bf16(R, ref, "in place")


def test_empty_problem_is_noop():
    X = torch.zeros(0, 64, dtype=torch.bfloat16, device=DEV)
    W = torch.zeros(32, 64, dtype=torch.bfloat16, device=DEV)
    assert kf.fused_gemm(X, W, []).shape == (0, 32)


# -------------------------------------------------------------- fp32 FFMA path
def test_fp32_relu_linear_workload_full():
    inp = kf_workloads.generate("fp32_relu_linear", seed=0)
    chain = wl_chain("fp32_relu_linear", inp)
    Y = kf.fused_gemm(inp["X"].to(DEV), inp["W"].to(DEV), chain_to(chain, DEV))
    check_f32(Y, oracle.fused_gemm(inp["X"], inp["W"], chain), "fp32 relu linear")


def test_fp32_ragged_chain():
    inp = kf_workloads.generate("fp32_relu_linear", seed=1, M=77, N=45, K=101)
    R = torch.randn(77, 45, generator=torch.Generator().manual_seed(2))
    chain = [("bias", {"p0": inp["b"]}), ("silu", {}), ("residual_add", {"p0": R}), ("scale", {"scalar": 0.5})]
    Y = kf.fused_gemm(inp["X"].to(DEV), inp["W"].to(DEV), chain_to(chain, DEV))
    check_f32(Y, oracle.fused_gemm(inp["X"], inp["W"], chain), "fp32 ragged")


# ----------------------------------------------------------- row log-sum-exp
@pytest.mark.parametrize("M,N,K,dist", [(200, 1000, 136, "default"), (300, 2500, 264, "unscaled"),
                                        (130, 300, 64, "offset"), (64, 33, 40, "uniform")])
def test_row_logsumexp(M, N, K, dist):
    inp = kf_workloads.generate("bf16_scale_rowlse", seed=5, M=M, N=N, K=K, dist=dist)
    chain = wl_chain("bf16_scale_rowlse", inp)
    Y = kf.fused_gemm(inp["X"].to(DEV), inp["W"].to(DEV), chain_to(chain, DEV))
    assert Y.shape == (M,) and Y.dtype == torch.float32
    ref = oracle.fused_gemm(inp["X"], inp["W"], chain)[:, 0]
    check_f32(Y, ref, f"lse {dist}")
    _no_device_error()


def test_row_logsumexp_then_scalar_op():
    inp = kf_workloads.generate("bf16_scale_rowlse", seed=6, M=150, N=700, K=128, dist="unscaled")
    chain = [("scale", {"scalar": 0.125}), ("row_logsumexp", {}), ("mish", {})]
    Y = kf.fused_gemm(inp["X"].to(DEV), inp["W"].to(DEV), chain)
    check_f32(Y, oracle.fused_gemm(inp["X"], inp["W"], chain)[:, 0], "lse+mish")


# ------------------------------------------------------------------ GroupNorm
@pytest.mark.parametrize("N,groups", [(1024, 2), (768, 3), (512, 8), (1280, 5)])
def test_groupnorm_swish(N, groups):
    inp = kf_workloads.generate("bf16_groupnorm_swish", seed=7, M=200, N=N, K=136)
    chain = [("bias", {"p0": inp["b"]}),
             ("groupnorm", {"groups": groups, "eps": 1e-5, "p0": inp["gamma"], "p1": inp["beta"]}),
             ("silu", {})]
    Y = kf.fused_gemm(inp["X"].to(DEV), inp["W"].to(DEV), chain_to(chain, DEV))
    check_bf16(Y, oracle.fused_gemm(inp["X"], inp["W"], chain), f"gn gs={N // groups}")
    _no_device_error()


@pytest.mark.parametrize("post", ["silu", "gelu_tanh"])  # compiled program / interpreter
def test_groupnorm_512_many_units_per_cluster(post):
    # 4 ragged 256-row tiles x 24 groups of 512 = 96 units: more than the clusters
    # of four that fit at once, so every cluster reuses its statistics slots
    inp = kf_workloads.generate("bf16_groupnorm_swish", seed=17, M=1000, N=12288, K=136)
    chain = [("bias", {"p0": inp["b"]}),
             ("groupnorm", {"groups": 24, "eps": 1e-5, "p0": inp["gamma"], "p1": inp["beta"]}),
             (post, {})]
    Y = kf.fused_gemm(inp["X"].to(DEV), inp["W"].to(DEV), chain_to(chain, DEV))
    check_bf16(Y, oracle.fused_gemm(inp["X"], inp["W"], chain), f"gn 512 x96 {post}")
    _no_device_error()


@pytest.mark.parametrize("M,N,groups", [(200, 1024, 2), (1000, 12288, 24)])
def test_groupnorm_512_without_workspace(M, N, groups):
    # no workspace: the statistics of a 512-column group are exchanged on chip
    # by clusters of four; with one (the binding's default) by couples of CTA
    # pairs through global memory -- both must match the oracle
    import ctypes
    inp = kf_workloads.generate("bf16_groupnorm_swish", seed=19, M=M, N=N, K=136)
    chain = [("bias", {"p0": inp["b"]}),
             ("groupnorm", {"groups": groups, "eps": 1e-5, "p0": inp["gamma"], "p1": inp["beta"]}),
             ("silu", {})]
    X, W = inp["X"].to(DEV), inp["W"].to(DEV)
    keep = []
    epi = kf.make_epilogue(chain_to(chain, DEV), keep)
    L = kf.lib()
    assert L.kf_fused_gemm_workspace(M, N, 136, ctypes.byref(epi)) > 0
    Y = torch.empty(M, N, dtype=torch.bfloat16, device=DEV)
    st = L.kf_fused_gemm(X.data_ptr(), kf.KF_BF16, 136, W.data_ptr(), kf.KF_BF16, 136, Y.data_ptr(), kf.KF_BF16, N,
                         M, N, 136, ctypes.byref(epi), None, 0, None)
    assert st == kf.KF_OK, kf.status_string(st)
    torch.cuda.synchronize()
    ref = oracle.fused_gemm(inp["X"], inp["W"], chain)
    check_bf16(Y, ref, "gn 512, clusters of four")
    Y2 = kf.fused_gemm(X, W, chain_to(chain, DEV))
    check_bf16(Y2, ref, "gn 512, couples")
    _no_device_error()


def test_groupnorm_no_affine_unit_moments():
    inp = kf_workloads.generate("bf16_groupnorm_swish", seed=9, M=130, N=1024, K=64, dist="unscaled")
    chain = [("groupnorm", {"groups": 2, "eps": 1e-5})]
    Y = kf.fused_gemm(inp["X"].to(DEV), inp["W"].to(DEV), chain, out_dtype=torch.float32)
    ref = oracle.fused_gemm(inp["X"], inp["W"], chain)
    check_f32(Y, ref, "gn no affine")
    y = to_np(Y).reshape(130, 2, 512)
    assert np.allclose(y.mean(-1), 0, atol=1e-3)


# --------------------------------------------- full-size workloads, sampled rows
FULL = ["bf16_gelu_scale_residual", "bf16_scale_rowlse", "bf16_groupnorm_swish"]


@pytest.mark.parametrize("name", FULL)
def test_full_size_workload_sampled_rows(name):
    inp = kf_workloads.generate(name, seed=0)
    chain = wl_chain(name, inp)
    dinp = {k: v.to(DEV) for k, v in inp.items()}
    Y = kf.fused_gemm(dinp["X"], dinp["W"], wl_chain(name, dinp))
    torch.cuda.synchronize()
    M = inp["X"].shape[0]
    rows = sorted(set([0, 1, 127, 128, M - 1] + list(np.random.default_rng(0).choice(M, 11, replace=False))))
    ref = oracle.fused_gemm(inp["X"], inp["W"], chain, rows=rows)
    got = Y[rows]
    if name == "bf16_scale_rowlse":
        check_f32(got, ref[:, 0], name)
    else:
        check_bf16(got, ref, name)
    _no_device_error()
    # whole-output invariants at full size
    if name == "bf16_scale_rowlse":
        assert torch.isfinite(Y).all()
    else:
        assert torch.isfinite(Y.float()).all()
