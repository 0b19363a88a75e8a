"""GPU parity of the MoE path (routing, grouped GEMMs, full expert FFN) against
the fp64 oracle: index work bit-exact, floating outputs within tolerance."""
import numpy as np
import pytest
import torch

import kf_workloads
import oracle
import paper_2606_02963_gb300 as kf
from tests._util import check_bf16, check_f32, to_np

pytestmark = pytest.mark.gpu
DEV = "cuda"


def _no_device_error():
    st, raw = kf.get_device_error()
    assert st == kf.KF_OK, f"device error word {raw:#x}"


@pytest.mark.parametrize("T,E,k", [(1, 32, 4), (64, 32, 4), (4096, 32, 4), (333, 8, 2), (50, 256, 8),
                                   (17, 40, 40)])
def test_route_bit_exact(T, E, k):
    logits = torch.randn(T, E, generator=torch.Generator().manual_seed(T + E))
    r = kf.moe_route(logits.to(DEV), k)
    ref = oracle.moe_route(logits, k)
    assert np.array_equal(r["topk_ids"].cpu().numpy(), ref["topk_ids"])
    assert np.array_equal(r["offsets"].cpu().numpy(), ref["offsets"])
    assert np.array_equal(r["sorted_token"].cpu().numpy(), ref["sorted_token"])
    assert np.allclose(r["topk_w"].cpu().numpy(), ref["topk_w"], rtol=1e-5, atol=1e-7)
    assert np.allclose(r["sorted_w"].cpu().numpy(), ref["sorted_w"], rtol=1e-5, atol=1e-7)


def test_route_ties_lower_index():
    logits = torch.zeros(3, 16)
    logits[1, 7] = 1.0
    logits[2] = torch.tensor([0., 2, 2, 1, 2, 0, 1, 1, 0, 0, 0, 0, 0, 0, 0, 2])
    r = kf.moe_route(logits.to(DEV), 4)
    ref = oracle.moe_route(logits, 4)
    assert np.array_equal(r["topk_ids"].cpu().numpy(), ref["topk_ids"])
    assert np.array_equal(r["sorted_token"].cpu().numpy(), ref["sorted_token"])


def _groups(sizes, K, nb, seed, w_std=0.05):
    g = torch.Generator().manual_seed(seed)
    rows = sum(sizes)
    off = torch.tensor(np.concatenate([[0], np.cumsum(sizes)]), dtype=torch.int32)
    B = (torch.randn(len(sizes), nb, K, generator=g) * w_std).to(torch.bfloat16)
    return rows, off, B, g


@pytest.mark.parametrize("sizes", [[0, 1, 7, 129, 0, 300], [8] * 32, [0, 0, 5], [256]])
def test_grouped_swiglu_with_gather(sizes):
    N, K = 288, 200
    rows, off, B, g = _groups(sizes, K, 2 * N, seed=len(sizes))
    T = 97
    A = torch.randn(T, K, generator=g).to(torch.bfloat16)
    idx = torch.randint(0, T, (rows,), generator=g, dtype=torch.int32)
    h = kf.grouped_gemm(A.to(DEV), B.to(DEV), off.to(DEV), N, [("swiglu", {})], row_index=idx.to(DEV))
    ref = oracle.grouped_gemm(A, B, off.numpy(), N, [("swiglu", {})], row_index=idx.numpy())
    check_bf16(h, ref, f"swiglu {sizes}")
    _no_device_error()


@pytest.mark.parametrize("sizes", [[0, 1, 7, 129, 0, 300], [3] * 20])
def test_grouped_scale_scatter_add(sizes):
    N, K = 384, 136
    rows, off, B, g = _groups(sizes, K, N, seed=11 + len(sizes))
    A = torch.randn(rows, K, generator=g).to(torch.bfloat16)
    T = 50
    dst = torch.randint(0, T, (rows,), generator=g, dtype=torch.int32)
    scale = torch.rand(rows, generator=g)
    C = torch.zeros(T, N, dtype=torch.float32, device=DEV)
    chain = [("row_scale_scatter_add", {"p0": scale, "p1": dst})]
    kf.grouped_gemm(A.to(DEV), B.to(DEV), off.to(DEV), N,
                    [("row_scale_scatter_add", {"p0": scale.to(DEV), "p1": dst.to(DEV)})], out=C)
    ref = oracle.grouped_gemm(A, B, off.numpy(), N, chain, out_rows=T)
    check_f32(C, ref, "scatter")
    _no_device_error()


def test_grouped_store_chain_equals_dense_per_group():
    sizes = [130, 0, 64]
    N, K = 256, 128
    rows, off, B, g = _groups(sizes, K, N, seed=21)
    A = torch.randn(rows, K, generator=g).to(torch.bfloat16)
    bias = torch.randn(N, generator=g).to(torch.bfloat16)
    chain = [("bias", {"p0": bias}), ("gelu_tanh", {})]
    C = kf.grouped_gemm(A.to(DEV), B.to(DEV), off.to(DEV), N, [("bias", {"p0": bias.to(DEV)}), ("gelu_tanh", {})])
    ref = oracle.grouped_gemm(A, B, off.numpy(), N, chain)
    check_bf16(C, ref, "grouped store")


def test_grouped_bad_offsets_reported_not_faulted():
    N, K = 128, 64
    A = torch.zeros(10, K, dtype=torch.bfloat16, device=DEV)
    B = torch.zeros(2, N, K, dtype=torch.bfloat16, device=DEV)
    off = torch.tensor([0, 8, 4], dtype=torch.int32, device=DEV)  # decreasing
    kf.grouped_gemm(A, B, off, N, [], rows_total=10)
    st, raw = kf.get_device_error()
    assert st == kf.KF_ERR_DEVICE_BOUNDS and raw & 8


@pytest.mark.parametrize("T,H,I,E,k", [(24, 64, 96, 8, 2), (100, 256, 320, 16, 4), (7, 2880, 2880, 32, 4)])
def test_moe_ffn_small(T, H, I, E, k):
    m = kf_workloads.moe_generate(T, seed=T, H=H, I=I, E=E, k=k, w_std=0.05)
    out, ids, w = kf.moe_ffn(m["X"].to(DEV), m["logits"].to(DEV), m["W_gu"].to(DEV), m["W_down"].to(DEV), k,
                             return_routing=True)
    r = oracle.moe_route(m["logits"], k)
    assert np.array_equal(ids.cpu().numpy(), r["topk_ids"])
    ref = oracle.moe_ffn(m["X"], m["W_gu"], m["W_down"], r["topk_ids"], r["topk_w"])
    check_bf16(out, ref, "moe small")
    _no_device_error()


@pytest.mark.parametrize("T,n_check", [(64, 64), (4096, 24)])
def test_moe_ffn_full_size(T, n_check):
    m = kf_workloads.moe_generate(T, seed=0)
    d = {k: v.to(DEV) for k, v in m.items()}
    out, ids, w = kf.moe_ffn(d["X"], d["logits"], d["W_gu"], d["W_down"], 4, return_routing=True)
    torch.cuda.synchronize()
    r = oracle.moe_route(m["logits"], 4)
    assert np.array_equal(ids.cpu().numpy(), r["topk_ids"])
    toks = sorted(set([0, T - 1] + list(np.random.default_rng(1).choice(T, n_check, replace=False))))
    ref = oracle.moe_ffn(m["X"], m["W_gu"], m["W_down"], r["topk_ids"], r["topk_w"], tokens=toks)
    check_bf16(out[toks], ref, f"moe T={T}")
    assert torch.isfinite(out.float()).all()
    _no_device_error()


@pytest.mark.parametrize("T", [64, 500, 1000])  # 1000 tokens: 4000 pairs, the multi-block routing sort
def test_moe_ffn_deterministic_mode(T):
    """Fixed-order finalize: bit-identical across runs, and within tolerance of
    the oracle (the atomic scatter-add mode is checked above)."""
    m = kf_workloads.moe_generate(T, seed=T + 7, H=2880, I=2880, E=32, k=4)
    d = {k: v.to(DEV) for k, v in m.items()}
    y1 = kf.moe_ffn(d["X"], d["logits"], d["W_gu"], d["W_down"], 4, deterministic=True)
    y2 = kf.moe_ffn(d["X"], d["logits"], d["W_gu"], d["W_down"], 4, deterministic=True)
    torch.cuda.synchronize()
    assert torch.equal(y1, y2)
    r = oracle.moe_route(m["logits"], 4)
    toks = sorted(set([0, T - 1] + list(np.random.default_rng(2).choice(T, 12, replace=False))))
    ref = oracle.moe_ffn(m["X"], m["W_gu"], m["W_down"], r["topk_ids"], r["topk_w"], tokens=toks)
    check_bf16(y1[toks], ref, f"deterministic moe T={T}")
    _no_device_error()


def test_grouped_row_scale_store():
    sizes = [5, 0, 70]
    N, K = 256, 64
    rows, off, B, g = _groups(sizes, K, N, seed=31)
    A = torch.randn(rows, K, generator=g).to(torch.bfloat16)
    sc = torch.rand(rows, generator=g)
    C = kf.grouped_gemm(A.to(DEV), B.to(DEV), off.to(DEV), N, [("row_scale", {"p0": sc.to(DEV)})],
                        out_dtype=torch.float32)
    ref = oracle.grouped_gemm(A, B, off.numpy(), N, [("row_scale", {"p0": sc})])
    check_f32(C, ref, "row scale")


# ------------------------------------------------- MoE block tail: add + RMSNorm
def _block_inputs(T, H, seed):
    g = torch.Generator().manual_seed(seed)
    R = torch.randn(T, H, generator=g).to(torch.bfloat16)
    gamma = (torch.rand(H, generator=g) + 0.5).to(torch.bfloat16)
    return R, gamma


@pytest.mark.parametrize("T,H,I,E,k,det", [(37, 256, 128, 8, 2, False), (37, 256, 128, 8, 2, True),
                                           (64, 2880, 2880, 32, 4, False), (300, 2880, 2880, 32, 4, True)])
def test_moe_add_rmsnorm(T, H, I, E, k, det):
    m = kf_workloads.moe_generate(T, seed=T + 91, H=H, I=I, E=E, k=k)
    d = {kk: v.to(DEV) for kk, v in m.items()}
    R, gamma = _block_inputs(T, H, seed=T)
    eps = 1e-5
    Y, R_out = kf.moe_ffn_add_rmsnorm(d["X"], d["logits"], d["W_gu"], d["W_down"], k, R.to(DEV), gamma.to(DEV), eps,
                                      deterministic=det)
    torch.cuda.synchronize()
    r = oracle.moe_route(m["logits"], k)
    toks = list(range(T)) if T <= 64 else sorted(set([0, T - 1] + list(np.random.default_rng(3).choice(T, 14, replace=False))))
    y = oracle.moe_ffn(m["X"], m["W_gu"], m["W_down"], r["topk_ids"], r["topk_w"], tokens=toks)
    r_ref, n_ref = oracle.add_rmsnorm(y, R[toks], gamma, eps)
    check_bf16(R_out[toks], r_ref, f"residual T={T} det={det}")
    check_bf16(Y[toks], n_ref, f"normed T={T} det={det}")
    _no_device_error()


def test_moe_add_rmsnorm_in_place_and_consistent_with_moe_ffn():
    T, H, I, E, k = 64, 512, 256, 16, 4
    m = kf_workloads.moe_generate(T, seed=5, H=H, I=I, E=E, k=k)
    d = {kk: v.to(DEV) for kk, v in m.items()}
    R, gamma = _block_inputs(T, H, seed=6)
    Rd = R.to(DEV)
    Y1, R1 = kf.moe_ffn_add_rmsnorm(d["X"], d["logits"], d["W_gu"], d["W_down"], k, Rd, gamma.to(DEV), 1e-6,
                                    deterministic=True)
    Rin = Rd.clone()
    Y2, R2 = kf.moe_ffn_add_rmsnorm(d["X"], d["logits"], d["W_gu"], d["W_down"], k, Rin, gamma.to(DEV), 1e-6,
                                    r_out=Rin, deterministic=True)
    torch.cuda.synchronize()
    assert R2.data_ptr() == Rin.data_ptr()
    assert torch.equal(Y1, Y2) and torch.equal(R1, R2)
    # the residual equals R + the plain MoE output up to the bf16 rounding of that output
    y = kf.moe_ffn(d["X"], d["logits"], d["W_gu"], d["W_down"], k, deterministic=True)
    diff = (R1.float() - (Rd.float() + y.float())).abs()
    assert diff.max().item() <= 2e-2 * (Rd.float() + y.float()).abs().max().item()
    _no_device_error()


def _act(b, dev=None, **over):
    a = dict(kf_workloads.GPT_OSS_ACT)
    a.update(over)
    if b is not None:
        a["b_gu"], a["b_down"] = (b["b_gu"].to(dev), b["b_down"].to(dev)) if dev else (b["b_gu"], b["b_down"])
    return a


@pytest.mark.parametrize("det", [False, True])
@pytest.mark.parametrize("T,H,I,E,k,w_std", [(24, 64, 96, 8, 2, 0.3), (100, 256, 320, 16, 4, 0.15),
                                             (7, 2880, 2880, 32, 4, 0.02)])
def test_moe_gated_expert_activation_with_biases(T, H, I, E, k, w_std, det):
    # weights large enough that many gate / linear values pass the clamp limit
    m = kf_workloads.moe_generate(T, seed=T + 3, H=H, I=I, E=E, k=k, w_std=w_std)
    b = kf_workloads.moe_bias_generate(E, H, I, seed=T)
    out = kf.moe_ffn(m["X"].to(DEV), m["logits"].to(DEV), m["W_gu"].to(DEV), m["W_down"].to(DEV), k,
                     deterministic=det, act=_act(b, DEV))
    r = oracle.moe_route(m["logits"], k)
    ref = oracle.moe_ffn(m["X"], m["W_gu"], m["W_down"], r["topk_ids"], r["topk_w"], **_act(b))
    check_bf16(out, ref, f"gated moe T={T} det={det}")
    _no_device_error()
    if w_std >= 0.15:  # the clamp is live: without it the result differs
        no_clamp = oracle.moe_ffn(m["X"], m["W_gu"], m["W_down"], r["topk_ids"], r["topk_w"], **_act(b, limit=0.0))
        assert np.abs(no_clamp - ref).max() > 0.1


@pytest.mark.parametrize("T,n_check", [(64, 64), (4096, 16)])
def test_moe_gated_full_size(T, n_check):
    m = kf_workloads.moe_generate(T, seed=1)
    b = kf_workloads.moe_bias_generate(32, 2880, 2880, seed=2)
    d = {k2: v.to(DEV) for k2, v in m.items()}
    out = kf.moe_ffn(d["X"], d["logits"], d["W_gu"], d["W_down"], 4, act=_act(b, DEV))
    torch.cuda.synchronize()
    r = oracle.moe_route(m["logits"], 4)
    toks = sorted(set([0, T - 1] + list(np.random.default_rng(3).choice(T, n_check, replace=False))))
    ref = oracle.moe_ffn(m["X"], m["W_gu"], m["W_down"], r["topk_ids"], r["topk_w"], tokens=toks, **_act(b))
    check_bf16(out[toks], ref, f"gated moe T={T}")
    _no_device_error()


def test_moe_act_plain_parameters_equal_plain_swiglu_bitwise():
    # alpha 1, no clamp, offset 0, no biases: the same arithmetic as kf_moe_ffn_ex
    m = kf_workloads.moe_generate(300, seed=9, H=512, I=384, E=16, k=4, w_std=0.05)
    d = {k2: v.to(DEV) for k2, v in m.items()}
    y0 = kf.moe_ffn(d["X"], d["logits"], d["W_gu"], d["W_down"], 4, deterministic=True)
    y1 = kf.moe_ffn(d["X"], d["logits"], d["W_gu"], d["W_down"], 4, deterministic=True,
                    act=dict(alpha=1.0, limit=0.0, linear_offset=0.0))
    torch.cuda.synchronize()
    assert torch.equal(y0, y1)
    _no_device_error()
