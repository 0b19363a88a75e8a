"""Repeat-run checks on the GPU: every path whose arithmetic order is fixed must
give bitwise-identical results call after call (a race between warps, CTAs,
clusters or consecutive launches shows up as a difference), and one call of
each is checked against the oracle on sampled rows.  The default MoE finalize
adds with fp32 atomics (order free); its deterministic mode is checked here."""
import numpy as np
import pytest
import torch

import kf_workloads
import oracle
import paper_2606_02963_gb300 as kf
from tests._util import check_bf16, check_f32, wl_chain

pytestmark = pytest.mark.gpu
DEV = "cuda"
REPS = 8


def _same(outs, what):
    ref = outs[0]
    for i, o in enumerate(outs[1:], 1):
        assert torch.equal(o, ref), f"{what}: call {i} differs from call 0"


@pytest.mark.parametrize("name", ["bf16_gelu_scale_residual", "bf16_groupnorm_swish", "bf16_scale_rowlse"])
def test_dense_workload_repeats_bitwise(name):
    inp = kf_workloads.generate(name, seed=5)
    d = {k: v.to(DEV) for k, v in inp.items()}
    chain = wl_chain(name, d)
    outs = [kf.fused_gemm(d["X"], d["W"], chain).clone() for _ in range(REPS)]
    torch.cuda.synchronize()
    _same(outs, name)
    rows = [0, 1, 255, 256, 777, inp["X"].shape[0] - 1]
    ref = oracle.fused_gemm(inp["X"], inp["W"], wl_chain(name, inp), rows=rows)
    if name == "bf16_scale_rowlse":
        check_f32(outs[0][rows], ref[:, 0], name)
    else:
        check_bf16(outs[0][rows], ref, name)
    assert kf.get_device_error()[0] == kf.KF_OK


def test_moe_deterministic_prefill_repeats_bitwise():
    T, E, k, H, I = 1024, 32, 4, 2880, 2880
    g = torch.Generator("cpu").manual_seed(11)
    X = torch.randn(T, H, generator=g).to(torch.bfloat16).to(DEV)
    logits = torch.randn(T, E, generator=g).to(DEV)
    gd = torch.Generator(DEV).manual_seed(12)
    Wgu = (torch.randn(E, 2 * I, H, generator=gd, device=DEV) * 0.02).to(torch.bfloat16)
    Wd = (torch.randn(E, H, I, generator=gd, device=DEV) * 0.02).to(torch.bfloat16)
    outs = [kf.moe_ffn(X, logits, Wgu, Wd, k, deterministic=True).clone() for _ in range(REPS // 2)]
    torch.cuda.synchronize()
    _same(outs, "moe deterministic")
    # the atomic (default) mode agrees with it to fp32 summation order
    y = kf.moe_ffn(X, logits, Wgu, Wd, k)
    diff = (y.float() - outs[0].float()).abs().max().item()
    assert diff <= 2e-2 * outs[0].float().abs().max().item(), diff
    assert kf.get_device_error()[0] == kf.KF_OK
