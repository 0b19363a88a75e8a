"""Pins of the fp64 oracle against facts that do not come from the oracle itself:
closed forms, library routines for special cases, exact rational brute force and
invariants.  Each test is chosen so that a plausible slip in the oracle (a dropped
term, a wrong sign, a swapped index, a transposed operand) fails at least one."""
import math
from fractions import Fraction

import numpy as np
import pytest
import scipy.special
import torch
import torch.nn.functional as F

import oracle

pytestmark = pytest.mark.filterwarnings("ignore")


def bf16(a):
    return torch.as_tensor(a, dtype=torch.float32).to(torch.bfloat16)


def f64(t):
    return t.to(torch.float64).numpy()


# --------------------------------------------------------------------- GEMM core
def test_gemm_identity_gives_transposed_rows():
    g = torch.Generator().manual_seed(1)
    K, N = 24, 40
    W = bf16(torch.randint(-4, 5, (N, K), generator=g).float())
    X = bf16(torch.eye(K))
    Y = oracle.fused_gemm(X, W, [])
    assert np.array_equal(Y, f64(W).T)


def test_gemm_rank1_closed_form():
    g = torch.Generator().manual_seed(2)
    M, N, K = 7, 11, 33
    u = torch.randint(-3, 4, (M, 1), generator=g).float()
    a = torch.randint(-3, 4, (1, K), generator=g).float()
    v = torch.randint(-3, 4, (N, 1), generator=g).float()
    c = torch.randint(-3, 4, (1, K), generator=g).float()
    X, W = bf16(u @ a), bf16(v @ c)
    Y = oracle.fused_gemm(X, W, [])
    ref = (u.double() @ v.double().T) * float((a.double() * c.double()).sum())
    assert np.array_equal(Y, ref.numpy())


@pytest.mark.parametrize("M,N,K", [(1, 1, 1), (2, 3, 5), (6, 4, 6), (5, 6, 3)])
def test_gemm_bruteforce_fractions(M, N, K):
    g = torch.Generator().manual_seed(M * 100 + N * 10 + K)
    X = bf16(torch.randn(M, K, generator=g) * 3)
    W = bf16(torch.randn(N, K, generator=g) * 3)
    xs = [[Fraction(float(v)) for v in row] for row in X.float().tolist()]
    ws = [[Fraction(float(v)) for v in row] for row in W.float().tolist()]
    Y = oracle.fused_gemm(X, W, [])
    for i in range(M):
        for j in range(N):
            exact = sum(xs[i][k] * ws[j][k] for k in range(K))
            assert abs(Fraction(Y[i, j]) - exact) <= abs(exact) * Fraction(1, 2**50) + Fraction(1, 2**200)


def test_gemm_fp32_operands_and_row_subset():
    g = torch.Generator().manual_seed(3)
    X = torch.rand(9, 17, generator=g) * 2 - 1
    W = torch.rand(5, 17, generator=g) * 2 - 1
    Y = oracle.fused_gemm(X, W, [])
    ref = X.double().numpy() @ W.double().numpy().T
    assert np.allclose(Y, ref, rtol=1e-14, atol=1e-14)
    Ys = oracle.fused_gemm(X, W, [], rows=[8, 0, 3])
    assert np.array_equal(Ys, Y[[8, 0, 3]])


# ------------------------------------------------------ elementwise tail ops
def _through_identity(vals, chain, extra=None):
    """Make s = vals exactly: X = I, W = vals^T (vals must be bf16-exact)."""
    vals = bf16(vals)
    M, N = vals.shape
    X = bf16(torch.eye(M))
    W = vals.T.contiguous()
    return oracle.fused_gemm(X, W, chain), f64(vals)


def _grid(M=8, N=64, lo=-6, hi=6):
    return torch.linspace(lo, hi, M * N).reshape(M, N)


@pytest.mark.parametrize("kind,fn", [
    ("gelu_tanh", lambda t: F.gelu(t, approximate="tanh")),
    ("silu", F.silu),
    ("sigmoid", torch.sigmoid),
    ("relu", F.relu),
    ("mish", F.mish),
])
def test_activation_matches_library_fp64(kind, fn):
    Y, s = _through_identity(_grid(), [(kind, {})])
    ref = fn(torch.from_numpy(s)).numpy()
    assert np.allclose(Y, ref, rtol=1e-14, atol=1e-15)


def test_leaky_relu_slope():
    Y, s = _through_identity(_grid(), [("leaky_relu", {"scalar": 0.2})])
    assert np.allclose(Y, F.leaky_relu(torch.from_numpy(s), 0.2).numpy(), rtol=0, atol=0)


def test_gelu_odd_part_identity_and_limits():
    Y, s = _through_identity(_grid(4, 32, -9, 9), [("gelu_tanh", {})])
    Yn, _ = _through_identity(-_grid(4, 32, -9, 9), [("gelu_tanh", {})])
    assert np.allclose(Y - Yn, s, atol=1e-13)          # gelu(x) - gelu(-x) = x
    Y0, _ = _through_identity(torch.zeros(2, 8), [("gelu_tanh", {})])
    assert np.all(Y0 == 0)
    Yb, sb = _through_identity(torch.full((1, 8), 40.0), [("gelu_tanh", {})])
    assert np.allclose(Yb, sb, rtol=1e-15)             # -> x for large x


def test_sigmoid_silu_symmetries():
    Y, s = _through_identity(_grid(), [("sigmoid", {})])
    Yn, _ = _through_identity(-_grid(), [("sigmoid", {})])
    assert np.allclose(Y + Yn, 1.0, atol=1e-15)
    S, _ = _through_identity(_grid(), [("silu", {})])
    Sn, _ = _through_identity(-_grid(), [("silu", {})])
    assert np.allclose(S - Sn, s, atol=1e-13)


def test_bias_scale_residual_chain_order():
    g = torch.Generator().manual_seed(4)
    M, N, K = 6, 10, 12
    X = bf16(torch.randint(-3, 4, (M, K), generator=g).float())
    W = bf16(torch.randint(-3, 4, (N, K), generator=g).float())
    b = bf16(torch.randint(-5, 6, (N,), generator=g).float())
    R = bf16(torch.randint(-5, 6, (M, N), generator=g).float())
    s = f64(X) @ f64(W).T
    Y = oracle.fused_gemm(X, W, [("bias", {"p0": b}), ("scale", {"scalar": 2.0}),
                                 ("residual_add", {"p0": R})])
    assert np.array_equal(Y, (s + f64(b)[None, :]) * 2.0 + f64(R))
    # a different order is a different function
    Y2 = oracle.fused_gemm(X, W, [("scale", {"scalar": 2.0}), ("bias", {"p0": b}),
                                  ("residual_add", {"p0": R})])
    assert np.array_equal(Y2, s * 2.0 + f64(b)[None, :] + f64(R))
    Ym = oracle.fused_gemm(X, W, [("mul", {"p0": b})])
    assert np.array_equal(Ym, s * f64(b)[None, :])


def test_residual_uses_true_row_under_subset():
    g = torch.Generator().manual_seed(5)
    X = bf16(torch.randn(8, 16, generator=g))
    W = bf16(torch.randn(4, 16, generator=g))
    R = bf16(torch.randn(8, 4, generator=g))
    full = oracle.fused_gemm(X, W, [("residual_add", {"p0": R})])
    sub = oracle.fused_gemm(X, W, [("residual_add", {"p0": R})], rows=[7, 2])
    assert np.array_equal(sub, full[[7, 2]])


# ------------------------------------------------------------- row logsumexp
def test_row_lse_matches_scipy_and_bounds():
    g = torch.Generator().manual_seed(6)
    M, N, K = 5, 300, 64
    X = bf16(torch.randn(M, K, generator=g))
    W = bf16(torch.randn(N, K, generator=g))
    Y = oracle.fused_gemm(X, W, [("scale", {"scalar": 0.125}), ("row_logsumexp", {})])
    S = 0.125 * (f64(X) @ f64(W).T)
    ref = scipy.special.logsumexp(S, axis=1)
    assert Y.shape == (M, 1)
    assert np.allclose(Y[:, 0], ref, rtol=1e-14, atol=1e-13)
    m = S.max(axis=1)
    assert np.all(Y[:, 0] >= m) and np.all(Y[:, 0] <= m + math.log(N) + 1e-12)
    assert np.allclose(np.exp(S - Y).sum(axis=1), 1.0, atol=1e-12)


def test_row_lse_constant_row_and_shift():
    c = 3.0
    Y, _ = _through_identity(torch.full((3, 64), c), [("row_logsumexp", {})])
    assert np.allclose(Y[:, 0], c + math.log(64), atol=1e-14)
    base = torch.round(_grid(2, 64, -4, 4) * 8) / 8   # bf16-exact before and after +16
    Y1, _ = _through_identity(base, [("row_logsumexp", {})])
    Y2, _ = _through_identity(base + 16.0, [("row_logsumexp", {})])
    assert np.allclose(Y2 - Y1, 16.0, atol=1e-12)
    # huge offsets must not overflow (max subtraction)
    Y3, _ = _through_identity(torch.full((1, 16), 1000.0), [("row_logsumexp", {})])
    assert np.isfinite(Y3).all() and abs(Y3[0, 0] - (1000.0 + math.log(16))) < 1e-10


# ----------------------------------------------------------------- GroupNorm
def test_groupnorm_matches_torch_fp64():
    g = torch.Generator().manual_seed(7)
    M, N, K, G = 6, 96, 40, 4
    X = bf16(torch.randn(M, K, generator=g))
    W = bf16(torch.randn(N, K, generator=g))
    b = bf16(torch.randn(N, generator=g))
    gam = torch.rand(N, generator=g) + 0.5
    bet = torch.rand(N, generator=g) * 0.2 - 0.1
    chain = [("bias", {"p0": b}), ("groupnorm", {"groups": G, "eps": 1e-5, "p0": gam, "p1": bet}),
             ("silu", {})]
    Y = oracle.fused_gemm(X, W, chain)
    Z = torch.from_numpy(f64(X) @ f64(W).T + f64(b)[None, :])
    ref = F.silu(F.group_norm(Z, G, gam.double(), bet.double(), 1e-5)).numpy()
    assert np.allclose(Y, ref, rtol=1e-12, atol=1e-13)


def test_groupnorm_unit_affine_moments():
    g = torch.Generator().manual_seed(8)
    M, N, K, G, eps = 4, 64, 32, 2, 1e-5
    X = bf16(torch.randn(M, K, generator=g) * 0.05)
    W = bf16(torch.randn(N, K, generator=g) * 0.05)
    Y = oracle.fused_gemm(X, W, [("groupnorm", {"groups": G, "eps": eps})])
    Z = f64(X) @ f64(W).T
    for gi in range(G):
        sl = slice(gi * N // G, (gi + 1) * N // G)
        var = Z[:, sl].var(axis=1)
        assert np.allclose(Y[:, sl].mean(axis=1), 0.0, atol=1e-12)
        assert np.allclose(Y[:, sl].var(axis=1), var / (var + eps), rtol=1e-10)
    # constant group -> beta
    bet = torch.linspace(-1, 1, 16)
    Yc, _ = _through_identity(torch.full((2, 16), 5.0),
                              [("groupnorm", {"groups": 2, "eps": eps, "p0": torch.ones(16), "p1": bet})])
    assert np.allclose(Yc, bet.double().numpy()[None, :], atol=1e-12)


# ------------------------------------------------------------------- routing
def test_route_matches_torch_topk_and_softmax():
    g = torch.Generator().manual_seed(9)
    T, E, k = 50, 32, 4
    logits = torch.randn(T, E, generator=g)
    r = oracle.moe_route(logits, k)
    v, idx = torch.topk(logits, k, dim=1)
    assert np.array_equal(r["topk_ids"], idx.int().numpy())
    ref_w = torch.softmax(v.double(), dim=1).numpy()
    assert np.allclose(r["topk_w"], ref_w, rtol=1e-15, atol=1e-16)
    assert np.allclose(r["topk_w"].sum(1), 1.0, atol=1e-15)
    flat = r["topk_ids"].reshape(-1)
    order = np.argsort(flat, kind="stable")
    assert np.array_equal(r["sorted_pair"], order)
    assert np.array_equal(r["sorted_token"], order // k)
    assert np.array_equal(r["offsets"], np.concatenate([[0], np.cumsum(np.bincount(flat, minlength=E))]))
    assert np.array_equal(r["sorted_w"], r["topk_w"].reshape(-1)[order])


def test_route_ties_take_lower_index():
    logits = torch.zeros(2, 8)
    logits[0, 5] = 1.0
    logits[1] = torch.tensor([0.0, 2.0, 2.0, 1.0, 2.0, 0.0, 1.0, 1.0])
    r = oracle.moe_route(logits, 3)
    assert r["topk_ids"][0].tolist() == [5, 0, 1]
    assert r["topk_ids"][1].tolist() == [1, 2, 4]
    assert np.allclose(r["topk_w"][1], 1 / 3, atol=1e-15)


# ------------------------------------------------------------------ bf16 round
def test_round_bf16_matches_torch_on_fp32_values():
    g = torch.Generator().manual_seed(10)
    x = torch.cat([torch.randn(4000, generator=g) * 10 ** torch.randint(-30, 30, (4000,), generator=g).float(),
                   # exact ties between two bf16 neighbours
                   (torch.arange(1, 200).float() * 2 + 1) * 2.0 ** -8 + 1.0 - 2.0 ** -8])
    ref = x.to(torch.bfloat16).double().numpy()
    got = np.array([oracle.round_bf16(float(v)) for v in x.tolist()])
    assert np.array_equal(got, ref)


# ------------------------------------------------------------------------ MoE
def _moe_small(T=6, H=24, I=16, E=4, k=2, seed=11):
    g = torch.Generator().manual_seed(seed)
    X = bf16(torch.randn(T, H, generator=g))
    Wgu = bf16(torch.randn(E, 2 * I, H, generator=g) * 0.2)
    Wd = bf16(torch.randn(E, H, I, generator=g) * 0.2)
    logits = torch.randn(T, E, generator=g)
    return X, Wgu, Wd, logits


def _ffn_numpy(x, wgu, wd, round_h):
    I = wgu.shape[0] // 2
    gt, up = wgu[:I] @ x, wgu[I:] @ x
    h = gt / (1 + np.exp(-gt)) * up
    if round_h:
        h = torch.from_numpy(h).float().to(torch.bfloat16).double().numpy()
    return wd @ h


def test_moe_ffn_matches_numpy_definition():
    X, Wgu, Wd, logits = _moe_small()
    r = oracle.moe_route(logits, 2)
    Y = oracle.moe_ffn(X, Wgu, Wd, r["topk_ids"], r["topk_w"], round_h=False)
    x, wgu, wd = f64(X), f64(Wgu), f64(Wd)
    for t in range(X.shape[0]):
        ref = sum(r["topk_w"][t, j] * _ffn_numpy(x[t], wgu[r["topk_ids"][t, j]], wd[r["topk_ids"][t, j]], False)
                  for j in range(2))
        assert np.allclose(Y[t], ref, rtol=1e-12, atol=1e-13)
    Yr = oracle.moe_ffn(X, Wgu, Wd, r["topk_ids"], r["topk_w"], round_h=True)
    t = 3
    ref = sum(r["topk_w"][t, j] * _ffn_numpy(x[t], wgu[r["topk_ids"][t, j]], wd[r["topk_ids"][t, j]], True)
              for j in range(2))
    assert np.allclose(Yr[t], ref, rtol=1e-9, atol=1e-9)
    assert not np.allclose(Yr, Y, rtol=0, atol=0)  # the rounding point is live


def test_moe_identical_experts_ignore_routing():
    X, Wgu, Wd, logits = _moe_small(E=3, k=2)
    Wgu = Wgu[:1].repeat(3, 1, 1)
    Wd = Wd[:1].repeat(3, 1, 1)
    r = oracle.moe_route(logits, 2)
    Y = oracle.moe_ffn(X, Wgu, Wd, r["topk_ids"], r["topk_w"])
    ids = np.zeros_like(r["topk_ids"])
    Y0 = oracle.moe_ffn(X, Wgu, Wd, ids, r["topk_w"])
    assert np.allclose(Y, Y0, rtol=1e-13, atol=1e-14)
    dense = np.stack([_ffn_numpy(f64(X)[t], f64(Wgu)[0], f64(Wd)[0], True) for t in range(X.shape[0])])
    assert np.allclose(Y, dense, rtol=1e-9, atol=1e-9)


def test_grouped_gemm_composition_equals_moe_ffn():
    X, Wgu, Wd, logits = _moe_small(T=9, E=4, k=2)
    T, H = X.shape
    I = Wgu.shape[1] // 2
    r = oracle.moe_route(logits, 2)
    h = oracle.grouped_gemm(X, Wgu, r["offsets"], I, [("swiglu", {})], row_index=r["sorted_token"])
    # gate/up from numpy for one routed row
    row = 5
    e = int(np.searchsorted(r["offsets"], row, side="right") - 1)
    x = f64(X)[r["sorted_token"][row]]
    g = f64(Wgu)[e, :I] @ x
    u = f64(Wgu)[e, I:] @ x
    assert np.allclose(h[row], g / (1 + np.exp(-g)) * u, rtol=1e-12, atol=1e-13)
    hb = torch.from_numpy(h).float().to(torch.bfloat16)
    sw = torch.from_numpy(r["sorted_w"]).float()
    st = torch.from_numpy(r["sorted_token"]).int()
    Y = oracle.grouped_gemm(hb, Wd, r["offsets"], H,
                            [("row_scale_scatter_add", {"p0": sw, "p1": st})], out_rows=T)
    w32 = torch.from_numpy(r["topk_w"]).float().double().numpy()
    Yref = oracle.moe_ffn(X, Wgu, Wd, r["topk_ids"], w32)
    assert np.allclose(Y, Yref, rtol=1e-5, atol=1e-5)


def test_grouped_single_group_equals_dense():
    g = torch.Generator().manual_seed(12)
    X = bf16(torch.randn(7, 20, generator=g))
    W = bf16(torch.randn(9, 20, generator=g))
    b = bf16(torch.randn(9, generator=g))
    chain = [("bias", {"p0": b}), ("gelu_tanh", {})]
    dense = oracle.fused_gemm(X, W, chain)
    grp = oracle.grouped_gemm(X, W[None], np.array([0, 7], np.int32), 9, chain)
    assert np.array_equal(dense, grp)


def test_grouped_f16_groups_equal_dense_calls():
    """fp16 experts: every group of a grouped GEMM reads its own weights, so G
    groups equal G dense products (this fails if the group stride were taken in
    the wrong element size)."""
    g = torch.Generator().manual_seed(21)
    K, N = 24, 6
    A = torch.randint(-4, 5, (9, K), generator=g).float().to(torch.float16)
    B = torch.randint(-4, 5, (2, N, K), generator=g).float().to(torch.float16)
    off = np.array([0, 4, 9], np.int32)
    grp = oracle.grouped_gemm(A, B, off, N, [])
    for e in range(2):
        dense = oracle.fused_gemm(A[off[e]:off[e + 1]], B[e], [])
        assert np.array_equal(grp[off[e]:off[e + 1]], dense)
        exact = A[off[e]:off[e + 1]].double().numpy() @ B[e].double().numpy().T
        assert np.array_equal(dense, exact)
    # the same integers in bf16 give the same products
    grp_bf = oracle.grouped_gemm(A.float().to(torch.bfloat16), B.float().to(torch.bfloat16), off, N, [])
    assert np.array_equal(grp, grp_bf)


# ------------------------------------------------------------------ row sum
def test_row_sum_closed_forms():
    # constant row c over N columns sums to N c; rank-1 s_ij = u_i v_j (a.c)
    # sums to u_i (a.c) sum_j v_j (small integers: exact in fp64)
    Y, _ = _through_identity(torch.full((3, 64), 1.5), [("row_sum", {})])
    assert Y.shape == (3, 1) and np.all(Y[:, 0] == 96.0)
    g = torch.Generator().manual_seed(22)
    M, N, K = 5, 37, 19
    u = torch.randint(-3, 4, (M, 1), generator=g).float()
    a = torch.randint(-3, 4, (1, K), generator=g).float()
    v = torch.randint(-3, 4, (N, 1), generator=g).float()
    c = torch.randint(-3, 4, (1, K), generator=g).float()
    Y = oracle.fused_gemm(bf16(u @ a), bf16(v @ c), [("row_sum", {})])
    ref = u.double()[:, 0] * float((a.double() * c.double()).sum()) * float(v.double().sum())
    assert np.array_equal(Y[:, 0], ref.numpy())


def test_row_sum_bruteforce_and_linearity():
    g = torch.Generator().manual_seed(23)
    M, N, K = 4, 6, 5
    X = bf16(torch.randn(M, K, generator=g) * 3)
    W = bf16(torch.randn(N, K, generator=g) * 3)
    b = bf16(torch.randn(N, generator=g))
    Y = oracle.fused_gemm(X, W, [("bias", {"p0": b}), ("row_sum", {}), ("scale", {"scalar": 0.5})])
    xs = [[Fraction(float(t)) for t in row] for row in X.float().tolist()]
    ws = [[Fraction(float(t)) for t in row] for row in W.float().tolist()]
    bs = [Fraction(float(t)) for t in b.float().tolist()]
    for i in range(M):
        exact = sum(sum(xs[i][k] * ws[j][k] for k in range(K)) + bs[j] for j in range(N)) / 2
        assert abs(Fraction(Y[i, 0]) - exact) <= abs(exact) * Fraction(1, 2**48) + Fraction(1, 2**200)
    # linearity: the sum of 2W is twice the sum of W; X W^T summed over j equals
    # X (sum_j W_j)^T, a matrix-vector product
    Y1 = oracle.fused_gemm(X, W, [("row_sum", {})])
    Y2 = oracle.fused_gemm(X, bf16(W.float() * 2), [("row_sum", {})])
    assert np.allclose(Y2, 2 * Y1, rtol=1e-14, atol=1e-14)
    mv = f64(X) @ f64(W).sum(axis=0)
    assert np.allclose(Y1[:, 0], mv, rtol=1e-13, atol=1e-13)


def test_row_scale_multiplies_each_row():
    g = torch.Generator().manual_seed(13)
    X = bf16(torch.randint(-3, 4, (5, 8), generator=g).float())
    W = bf16(torch.randint(-3, 4, (6, 8), generator=g).float())
    sc = torch.tensor([1.0, -2.0, 0.5, 0.0, 3.0])
    Y = oracle.fused_gemm(X, W, [("row_scale", {"p0": sc})])
    assert np.array_equal(Y, (f64(X) @ f64(W).T) * sc.double().numpy()[:, None])


# ------------------------------------------- residual add + RMSNorm (block tail)
def test_add_rmsnorm_matches_torch_rms_norm():
    # R + Y chosen exactly representable in fp32, so torch's fp32 -> bf16 rounding
    # gives the exact bf16 residual independently of the oracle's own rounding
    g = torch.Generator().manual_seed(21)
    T, H = 6, 40
    R = bf16(torch.randn(T, H, generator=g))
    Y = (torch.randint(-512, 513, (T, H), generator=g).double() / 256.0).numpy()
    gamma = bf16(torch.rand(H, generator=g) + 0.5)
    eps = 1e-5
    r_out, normed = oracle.add_rmsnorm(Y, R, gamma, eps)
    r_ref = (R.double() + torch.from_numpy(Y)).float().to(torch.bfloat16).double()
    assert np.array_equal(r_out, r_ref.numpy())
    ref = F.rms_norm(r_ref, (H,), weight=gamma.double(), eps=eps)
    assert np.allclose(normed, ref.numpy(), rtol=1e-12, atol=1e-12)


def test_add_rmsnorm_constant_row_and_moments():
    T, H = 3, 16
    R = bf16(torch.zeros(T, H))
    Y = np.array([[1.5] * H, [-3.0] * H, [0.25] * H])
    gamma = bf16(torch.ones(H))
    eps = 0.01
    r_out, normed = oracle.add_rmsnorm(Y, R, gamma, eps)
    for t, c in enumerate((1.5, -3.0, 0.25)):
        assert np.all(r_out[t] == c)
        assert np.allclose(normed[t], c / math.sqrt(c * c + eps), rtol=1e-14)
    # unit gamma: mean of normed^2 = ms / (ms + eps) exactly
    g = torch.Generator().manual_seed(22)
    Yr = torch.randn(4, 64, generator=g).double().numpy()
    r_out, normed = oracle.add_rmsnorm(Yr, bf16(torch.zeros(4, 64)), bf16(torch.ones(64)), eps)
    ms = (r_out ** 2).mean(axis=1)
    assert np.allclose((normed ** 2).mean(axis=1), ms / (ms + eps), rtol=1e-12)


def test_add_rmsnorm_scale_invariant_without_eps():
    g = torch.Generator().manual_seed(23)
    Yr = (torch.randint(-64, 65, (3, 32), generator=g).double() / 16.0).numpy()
    gamma = bf16(torch.rand(32, generator=g) + 0.5)
    R0 = bf16(torch.zeros(3, 32))
    _, n1 = oracle.add_rmsnorm(Yr, R0, gamma, 0.0)
    _, n2 = oracle.add_rmsnorm(Yr * 8.0, R0, gamma, 0.0)  # power of two: rounding commutes
    assert np.allclose(n1, n2, rtol=1e-14, atol=1e-14)


def test_f16_operands_read_exactly():
    # every finite binary16 value, read through a K = 1 GEMM against 1.0,
    # equals numpy's own float16 -> float64 conversion
    bits = np.arange(0, 1 << 16, dtype=np.uint32).astype(np.uint16)
    f = bits.view(np.float16)
    v = f[np.isfinite(f)]
    X = torch.ones(1, 1, dtype=torch.float16)
    W = torch.from_numpy(v.copy()).reshape(-1, 1)
    Y = oracle.fused_gemm(X, W, [])
    assert np.array_equal(Y[0], v.astype(np.float64))


# ---- QKV projection tail: bias, rotary embedding of query / key heads, cache rows
def _qkv_case(seed, T=5, H=24, nq=3, nkv=2, d=8, max_pos=16, rows=12):
    g = torch.Generator().manual_seed(seed)
    N = (nq + 2 * nkv) * d
    # small integers: every product and sum is exact in fp64
    X = torch.randint(-4, 5, (T, H), generator=g).to(torch.bfloat16)
    W = torch.randint(-4, 5, (N, H), generator=g).to(torch.bfloat16)
    b = torch.randint(-8, 9, (N,), generator=g).to(torch.bfloat16)
    pos = torch.randperm(max_pos, generator=g)[:T].to(torch.int32)      # positions != token index
    crow = torch.randperm(rows, generator=g)[:T].to(torch.int32)        # distinct cache rows
    s = X.double().numpy() @ W.double().numpy().T + b.double().numpy()
    return X, W, b, pos, crow, s, dict(nq=nq, nkv=nkv, d=d, rows=rows, max_pos=max_pos)


def test_qkv_identity_tables_route_plain_projection():
    X, W, b, pos, crow, s, c = _qkv_case(41)
    nq, nkv, d, half = c["nq"], c["nkv"], c["d"], c["d"] // 2
    cos_t = torch.ones(c["max_pos"], half)
    sin_t = torch.zeros(c["max_pos"], half)
    k0 = np.arange(c["rows"] * nkv * d, dtype=np.float64).reshape(c["rows"], nkv * d)
    q, kc, vc = oracle.qkv_rope_kv(X, W, b, pos, crow, cos_t, sin_t, nq, nkv, d, c["rows"], k_cache=k0, v_cache=-k0)
    assert np.array_equal(q, s[:, :nq * d])
    assert np.array_equal(kc[crow.numpy()], s[:, nq * d:(nq + nkv) * d])
    assert np.array_equal(vc[crow.numpy()], s[:, (nq + nkv) * d:])
    untouched = np.setdiff1d(np.arange(c["rows"]), crow.numpy())
    assert np.array_equal(kc[untouched], k0[untouched]) and np.array_equal(vc[untouched], -k0[untouched])
    # no bias: the projection alone
    q0, _, _ = oracle.qkv_rope_kv(X, W, None, pos, crow, cos_t, sin_t, nq, nkv, d, c["rows"])
    assert np.array_equal(q0, s[:, :nq * d] - b.double().numpy()[:nq * d])


def test_qkv_rotation_is_complex_multiplication():
    # the pair (s_i, s_{i+d/2}) as the complex number s_i + j s_{i+d/2}, turned by
    # the angle theta[pos, i]: numpy's complex product, not the oracle's formula
    X, W, b, pos, crow, s, c = _qkv_case(42, d=16)
    nq, nkv, d, half = c["nq"], c["nkv"], c["d"], c["d"] // 2
    g = torch.Generator().manual_seed(43)
    theta = (torch.rand(c["max_pos"], half, generator=g, dtype=torch.float64) * 12.0 - 6.0)
    cos_t, sin_t = torch.cos(theta).float(), torch.sin(theta).float()
    q, kc, vc = oracle.qkv_rope_kv(X, W, b, pos, crow, cos_t, sin_t, nq, nkv, d, c["rows"])
    rot = cos_t.double().numpy() + 1j * sin_t.double().numpy()  # the stored fp32 pair
    heads = s.reshape(s.shape[0], nq + 2 * nkv, d)
    z = heads[:, :nq + nkv, :half] + 1j * heads[:, :nq + nkv, half:]
    z = z * rot[pos.numpy()][:, None, :]
    ref = np.concatenate([z.real, z.imag], axis=2)
    assert np.allclose(q.reshape(-1, nq, d), ref[:, :nq], rtol=1e-12, atol=1e-9)
    assert np.allclose(kc[crow.numpy()].reshape(-1, nkv, d), ref[:, nq:], rtol=1e-12, atol=1e-9)
    assert np.array_equal(vc[crow.numpy()], s[:, (nq + nkv) * d:])  # value heads are not rotated
    # a rotation keeps each pair's length
    assert np.allclose(np.abs(z), np.abs(heads[:, :nq + nkv, :half] + 1j * heads[:, :nq + nkv, half:]), rtol=1e-6)


def test_qkv_quarter_turn_swaps_halves():
    # cos = 0, sin = 1: (a, b) -> (-b, a) for every pair of a query or key head
    X, W, b, pos, crow, s, c = _qkv_case(44)
    nq, nkv, d, half = c["nq"], c["nkv"], c["d"], c["d"] // 2
    q, kc, _ = oracle.qkv_rope_kv(X, W, b, pos, crow, torch.zeros(c["max_pos"], half),
                                  torch.ones(c["max_pos"], half), nq, nkv, d, c["rows"])
    heads = s.reshape(s.shape[0], nq + 2 * nkv, d)
    ref = np.concatenate([-heads[:, :, half:], heads[:, :, :half]], axis=2)
    assert np.array_equal(q.reshape(-1, nq, d), ref[:, :nq])
    assert np.array_equal(kc[crow.numpy()].reshape(-1, nkv, d), ref[:, nq:nq + nkv])


def test_qkv_scores_depend_on_relative_position():
    # with tables cos / sin(p * w_i), a query at position m and a key at position
    # n score q . k as a function of m - n only (the point of the embedding)
    T, H, d = 2, 16, 8
    half = d // 2
    g = torch.Generator().manual_seed(45)
    X = torch.randint(-4, 5, (T, H), generator=g).to(torch.bfloat16)
    W = torch.randint(-4, 5, (3 * d, H), generator=g).to(torch.bfloat16)
    P = 40
    w = 10000.0 ** (-np.arange(half) / half)
    ang = np.arange(P)[:, None] * w[None, :]
    cos_t = torch.from_numpy(np.cos(ang)).float()
    sin_t = torch.from_numpy(np.sin(ang)).float()

    def score(m, n):
        q, kc, _ = oracle.qkv_rope_kv(X, W, None, [m, n], [0, 1], cos_t, sin_t, 1, 1, d, 2)
        return float(q[0] @ kc[1])

    for m, n, sh in [(3, 1, 7), (10, 20, 5), (0, 0, 31)]:
        assert math.isclose(score(m, n), score(m + sh, n + sh), rel_tol=1e-5, abs_tol=1e-4)
    assert not math.isclose(score(3, 1), score(4, 1), rel_tol=1e-3)


def test_qkv_rejects_out_of_range_position_or_row():
    X, W, b, pos, crow, s, c = _qkv_case(46)
    half = c["d"] // 2
    cs = torch.ones(c["max_pos"], half), torch.zeros(c["max_pos"], half)
    bad = pos.clone()
    bad[2] = c["max_pos"]
    with pytest.raises(ValueError):
        oracle.qkv_rope_kv(X, W, b, bad, crow, *cs, c["nq"], c["nkv"], c["d"], c["rows"])
    badr = crow.clone()
    badr[0] = -1
    with pytest.raises(ValueError):
        oracle.qkv_rope_kv(X, W, b, pos, badr, *cs, c["nq"], c["nkv"], c["d"], c["rows"])


def test_qkv_fp16_operands_read_like_bf16_ones():
    # small integers are exact in both 16-bit formats: the same projection
    X, W, b, pos, crow, s, c = _qkv_case(47)
    half = c["d"] // 2
    cs = torch.ones(c["max_pos"], half), torch.zeros(c["max_pos"], half)
    args = (pos, crow, *cs, c["nq"], c["nkv"], c["d"], c["rows"])
    q16, k16, v16 = oracle.qkv_rope_kv(X.half(), W.half(), b.float(), *args)
    assert np.array_equal(q16, s[:, :c["nq"] * c["d"]])
    assert np.array_equal(k16[crow.numpy()], s[:, c["nq"] * c["d"]:(c["nq"] + c["nkv"]) * c["d"]])
    assert np.array_equal(v16[crow.numpy()], s[:, (c["nq"] + c["nkv"]) * c["d"]:])


# ---- gpt-oss expert activation: per-expert biases, clamp, sigmoid slope, +c on the linear branch
def _gate_case(bg, bu, alpha, limit, c, I=4, H=6, E=3, seed=51):
    """X = 0, so g and u are the biases exactly; k = 1 (weight 1); W_down maps h[n]
    to output column n; returns the output row of the token routed to expert 1."""
    T = 2
    X = bf16(torch.zeros(T, H))
    Wgu = bf16(torch.zeros(E, 2 * I, H))
    Wd = torch.zeros(E, H, I)
    for n in range(I):
        Wd[:, n, n] = 1.0
    Wd = bf16(Wd)
    b_gu = torch.zeros(E, 2 * I)
    b_gu[1, :I] = torch.tensor(bg, dtype=torch.float32)
    b_gu[1, I:] = torch.tensor(bu, dtype=torch.float32)
    b_gu = bf16(b_gu)
    logits = torch.tensor([[0.0, 5.0, 0.0], [5.0, 0.0, 0.0]])[:T, :E]
    r = oracle.moe_route(logits, 1)
    assert r["topk_ids"][0, 0] == 1 and r["topk_w"][0, 0] == 1.0
    Y = oracle.moe_ffn(X, Wgu, Wd, r["topk_ids"], r["topk_w"], round_h=False, b_gu=b_gu, alpha=alpha,
                       limit=limit, linear_offset=c)
    return Y[0, :I]


def test_moe_gate_activation_at_exact_sigmoid_points():
    # sigmoid(ln 3) = 3/4 and sigmoid(-ln 3) = 1/4 exactly; biases are exact in bf16
    l3 = math.log(3.0)
    # slope: g = 1, alpha = ln 3 -> 1 * 3/4 * (u + 1) with u = 2 -> 2.25
    # gate clamp from above: g = 12 -> 8 with alpha = ln 3 / 8 -> 8 * 3/4 * 3 = 18
    y = _gate_case([1.0, 12.0, 0.0, -1.0], [2.0, 2.0, 5.0, -1.0], alpha=l3, limit=8.0, c=1.0)
    assert math.isclose(y[0], 2.25, rel_tol=1e-14)
    y = _gate_case([12.0, 0.0, 0.0, 0.0], [2.0, 0.0, 0.0, 0.0], alpha=l3 / 8, limit=8.0, c=1.0)
    assert math.isclose(y[0], 18.0, rel_tol=1e-14)
    # no clamp below on the gate: g = -12, alpha = ln 3 / 12 -> -12 * 1/4 * (2 + 1) = -9
    y = _gate_case([-12.0, 0.0, 0.0, 0.0], [2.0, 0.0, 0.0, 0.0], alpha=l3 / 12, limit=8.0, c=1.0)
    assert math.isclose(y[0], -9.0, rel_tol=1e-14)
    # the linear branch is clamped on both sides: u = -20 -> -8, u = 20 -> 8
    y = _gate_case([1.0, 1.0, 0.0, 0.0], [-20.0, 20.0, 0.0, 0.0], alpha=l3, limit=8.0, c=1.0)
    assert math.isclose(y[0], 0.75 * -7.0, rel_tol=1e-14) and math.isclose(y[1], 0.75 * 9.0, rel_tol=1e-14)
    # g = 0 or u + c = 0 give exactly zero; without a limit nothing is clamped
    y = _gate_case([0.0, 1.0, 0.0, 0.0], [7.0, -1.0, 0.0, 0.0], alpha=l3, limit=8.0, c=1.0)
    assert y[0] == 0.0 and y[1] == 0.0
    y = _gate_case([12.0, 0.0, 0.0, 0.0], [20.0, 0.0, 0.0, 0.0], alpha=l3 / 12, limit=0.0, c=0.0)
    assert math.isclose(y[0], 12.0 * 0.75 * 20.0, rel_tol=1e-14)


def test_moe_down_bias_is_weighted_per_expert():
    # X = 0 and W_down = 0: the output is the routing-weighted sum of the chosen
    # experts' down biases, whatever the activation does
    T, H, I, E, k = 5, 8, 4, 4, 2
    g = torch.Generator().manual_seed(52)
    X = bf16(torch.zeros(T, H))
    Wgu = bf16(torch.randn(E, 2 * I, H, generator=g))
    Wd = bf16(torch.zeros(E, H, I))
    b_gu = bf16(torch.randn(E, 2 * I, generator=g))
    b_down = bf16(torch.randn(E, H, generator=g))
    r = oracle.moe_route(torch.randn(T, E, generator=g), k)
    Y = oracle.moe_ffn(X, Wgu, Wd, r["topk_ids"], r["topk_w"], b_gu=b_gu, b_down=b_down, alpha=1.702, limit=7.0,
                       linear_offset=1.0)
    bd = f64(b_down)
    ref = np.stack([sum(r["topk_w"][t, j] * bd[r["topk_ids"][t, j]] for j in range(k)) for t in range(T)])
    assert np.allclose(Y, ref, rtol=1e-14, atol=1e-15)


def test_moe_gate_defaults_are_the_plain_swiglu():
    X, Wgu, Wd, logits = _moe_small()
    r = oracle.moe_route(logits, 2)
    E, I2, H = Wgu.shape
    Y0 = oracle.moe_ffn(X, Wgu, Wd, r["topk_ids"], r["topk_w"])
    Y1 = oracle.moe_ffn(X, Wgu, Wd, r["topk_ids"], r["topk_w"], b_gu=bf16(torch.zeros(E, I2)),
                        b_down=bf16(torch.zeros(E, H)), alpha=1.0, limit=0.0, linear_offset=0.0)
    assert np.array_equal(Y0, Y1)
