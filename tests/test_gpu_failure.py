"""Failure detection without a GPU fault: every device-side wait of the tensor-core
kernels has a wall-clock limit.  With the limit set to 1 ns the first wait that
is not already satisfied gives up; the kernel records a timeout bit in the
device error word, drains its in-flight copies and MMAs, frees tensor memory and
returns.  The host reads KF_ERR_DEVICE_TIMEOUT, and the context stays usable: the
next (normal) call is correct."""
import ctypes

import numpy as np
import pytest
import torch

import kf_workloads
import oracle
import paper_2606_02963_gb300 as kf
from tests._util import check_bf16, wl_chain, chain_to

pytestmark = pytest.mark.gpu
DEV = "cuda"


def _problem():
    # K = 2048 (32 k-blocks): the epilogue's wait for the accumulator outlasts
    # the hardware's own suspension inside one mbarrier try_wait (with 8
    # k-blocks a single try_wait could see the whole mainloop finish)
    inp = kf_workloads.generate("bf16_gelu_scale_residual", seed=21, M=512, N=1024, K=2048)
    return inp, {k: v.to(DEV) for k, v in inp.items()}


@pytest.mark.parametrize("M", [100, 512])  # single-CTA tiles and CTA pairs
def test_wait_timeout_is_reported_and_context_survives(M):
    inp, d = _problem()
    X, R = d["X"][:M], d["R"][:M]
    chain = chain_to(wl_chain("bf16_gelu_scale_residual", inp), DEV)
    chain[-1] = ("residual_add", {"p0": R})
    assert kf.get_device_error()[0] == kf.KF_OK
    try:
        kf.set_wait_timeout_ns(1)
        kf.fused_gemm(X, d["W"], chain)
        st, raw = kf.get_device_error()
    finally:
        kf.set_wait_timeout_ns(0)
    assert st == kf.KF_ERR_DEVICE_TIMEOUT, (st, hex(raw))
    assert raw & 0x7
    # the error word was cleared by the read, and the next call is correct
    assert kf.get_device_error()[0] == kf.KF_OK
    Y = kf.fused_gemm(X, d["W"], chain)
    torch.cuda.synchronize()
    ref_chain = wl_chain("bf16_gelu_scale_residual", inp)
    ref = oracle.fused_gemm(inp["X"][:M], inp["W"], ref_chain)
    check_bf16(Y, ref, "after timeout")
    assert kf.get_device_error()[0] == kf.KF_OK


def test_grouped_wait_timeout_is_reported():
    # K = 2048 (32 k-blocks): the epilogue's wait for the accumulator outlasts
    # the hardware's own suspension inside one mbarrier try_wait, so at least
    # one wait must give up (with two k-blocks every wait could be satisfied
    # within a single try_wait)
    g = torch.Generator().manual_seed(3)
    A = torch.randn(300, 2048, generator=g).to(torch.bfloat16).to(DEV)
    B = (torch.randn(3, 256, 2048, generator=g) * 0.02).to(torch.bfloat16).to(DEV)
    off = torch.tensor([0, 100, 100, 300], dtype=torch.int32, device=DEV)
    try:
        kf.set_wait_timeout_ns(1)
        kf.grouped_gemm(A, B, off, 256, [])
        st, raw = kf.get_device_error()
    finally:
        kf.set_wait_timeout_ns(0)
    assert st == kf.KF_ERR_DEVICE_TIMEOUT, (st, hex(raw))
    C = kf.grouped_gemm(A, B, off, 256, [])
    ref = oracle.grouped_gemm(A.cpu(), B.cpu(), off.cpu().numpy(), 256, [])
    check_bf16(C, ref, "grouped after timeout")


def test_error_words_are_per_workspace():
    """Two streams, two workspaces: the call whose waits are limited to 1 ns
    reports the timeout in its own workspace's error word; the other call's
    word stays clean (the device-wide word sees the timeout as well).  A store
    chain needs no scratch, so each call is given a header-only workspace for
    its error word (the same problem as the timeout test above)."""
    inp, d = _problem()
    chain = chain_to(wl_chain("bf16_gelu_scale_residual", inp), DEV)
    wa = kf.new_workspace(kf.KF_WORKSPACE_HEADER_BYTES, DEV)
    wb = kf.new_workspace(kf.KF_WORKSPACE_HEADER_BYTES, DEV)
    sa, sb = torch.cuda.Stream(), torch.cuda.Stream()
    torch.cuda.synchronize()
    assert kf.get_device_error()[0] == kf.KF_OK
    try:
        kf.set_wait_timeout_ns(1)
        kf.fused_gemm(d["X"], d["W"], chain, workspace=wa, stream=sa)
    finally:
        kf.set_wait_timeout_ns(0)
    yb = kf.fused_gemm(d["X"], d["W"], chain, workspace=wb, stream=sb)
    stb, rawb = kf.check_device_error(wb, sb)
    sta, rawa = kf.check_device_error(wa, sa)
    assert stb == kf.KF_OK, ("other stream", stb, hex(rawb))
    assert sta == kf.KF_ERR_DEVICE_TIMEOUT and rawa & 0x7, ("timed-out stream", sta, hex(rawa))
    assert kf.check_device_error(wa, sa)[0] == kf.KF_OK  # cleared by the read
    dst, draw = kf.get_device_error()
    assert dst == kf.KF_ERR_DEVICE_TIMEOUT, ("device word", dst, hex(draw))
    assert kf.get_device_error()[0] == kf.KF_OK
    torch.cuda.synchronize()
    check_bf16(yb, oracle.fused_gemm(inp["X"], inp["W"], wl_chain("bf16_gelu_scale_residual", inp)),
               "the other stream's call")


def test_bounds_errors_are_per_workspace():
    """The same isolation with a deterministic error: a gathered grouped GEMM
    whose row index points outside A sets the bounds bit in its own
    workspace's word only; a correct call on another stream reports KF_OK."""
    g = torch.Generator().manual_seed(4)
    A = torch.randn(64, 128, generator=g).to(torch.bfloat16).to(DEV)
    B = (torch.randn(2, 256, 128, generator=g) * 0.1).to(torch.bfloat16).to(DEV)
    off = torch.tensor([0, 40, 96], dtype=torch.int32, device=DEV)
    good = torch.randint(0, 64, (96,), generator=g, dtype=torch.int32)
    bad = good.clone()
    bad[17] = 1 << 20
    need = kf.lib().kf_grouped_gemm_workspace(96, 256, 128, 2, 1, None)
    wa, wb = kf.new_workspace(need, DEV), kf.new_workspace(need, DEV)
    sa, sb = torch.cuda.Stream(), torch.cuda.Stream()
    gi, bi = good.to(DEV), bad.to(DEV)
    torch.cuda.synchronize()
    kf.get_device_error()
    kf.grouped_gemm(A, B, off, 256, [], row_index=bi, workspace=wa, stream=sa)
    C = kf.grouped_gemm(A, B, off, 256, [], row_index=gi, workspace=wb, stream=sb)
    stb, rawb = kf.check_device_error(wb, sb)
    sta, rawa = kf.check_device_error(wa, sa)
    assert stb == kf.KF_OK, hex(rawb)
    assert sta == kf.KF_ERR_DEVICE_BOUNDS and rawa == 0x8, (sta, hex(rawa))
    assert kf.get_device_error()[0] == kf.KF_ERR_DEVICE_BOUNDS
    torch.cuda.synchronize()
    ref = oracle.grouped_gemm(A.cpu(), B.cpu(), off.cpu().numpy(), 256, [], row_index=good.numpy())
    check_bf16(C, ref, "the other stream's grouped call")


@pytest.mark.parametrize("T", [1, 32, 64])  # token boxes of 32 and 64 rows, direct and staged partial rows
def test_qkv_decode_wait_timeout_is_reported_and_context_survives(T):
    s = kf_workloads.QKV_SHAPE
    inp = kf_workloads.qkv_generate(T, seed=400 + T, cache_rows=512)
    g = {k: v.to(DEV) for k, v in inp.items() if k != "rows"}
    rows = int(inp["rows"])

    def run():
        kc = torch.zeros(rows, s["nkv"] * s["d"], dtype=torch.bfloat16, device=DEV)
        vc = torch.zeros_like(kc)
        q = kf.qkv_rope_kv(g["X"], g["W"], g["b"], g["positions"], g["cache_rows"], g["cos"], g["sin"], s["nq"],
                           s["nkv"], s["d"], kc, vc)
        return q, kc, vc

    assert kf.get_device_error()[0] == kf.KF_OK
    try:
        kf.set_wait_timeout_ns(1)
        run()
        st, raw = kf.get_device_error()
    finally:
        kf.set_wait_timeout_ns(0)
    # the epilogue warps wait for the accumulator through the whole mainloop
    assert st == kf.KF_ERR_DEVICE_TIMEOUT, (st, hex(raw))
    q, kc, vc = run()
    assert kf.get_device_error()[0] == kf.KF_OK
    rq, rk, rv = oracle.qkv_rope_kv(inp["X"], inp["W"], inp["b"], inp["positions"], inp["cache_rows"], inp["cos"],
                                    inp["sin"], s["nq"], s["nkv"], s["d"], rows)
    check_bf16(q, rq, f"qkv after timeout T={T}")
    named = np.flatnonzero(~np.isnan(rk[:, 0]))
    check_bf16(kc[torch.as_tensor(named, device=DEV)], rk[named], f"k after timeout T={T}")
