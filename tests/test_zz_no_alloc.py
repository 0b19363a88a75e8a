"""The allocation-free row log-sum-exp entry point (kf_fused_gemm_lse_noalloc).

It serves callers that cannot allocate device memory (code hosted by another
runtime that owns all device memory, loops that must not call cudaMalloc because
it can synchronize the device): its scratch is a fixed device array inside the
library.  Called through the C ABI, its output must match the workspace-taking
kf_fused_gemm on two calls in a row (the second on a different problem, so stale
scratch contents from the first would show), within the fp32 tolerance used by
the other tests.  Kept in a file that is collected last."""
import ctypes

import pytest
import torch

import kf_workloads
import paper_2606_02963_gb300 as kf
from tests._util import check_f32

pytestmark = pytest.mark.gpu
DEV = "cuda"


def _noalloc(X, W, chain, out):
    keep = []
    epi = kf.make_epilogue(chain, keep)
    M, K = X.shape
    N = W.shape[0]
    dt = kf.KF_F16 if X.dtype == torch.float16 else kf.KF_BF16
    return kf.lib().kf_fused_gemm_lse_noalloc(
        X.data_ptr(), dt, X.stride(0), W.data_ptr(), dt, W.stride(0), out.data_ptr(),
        kf.KF_F32, M, N, K, ctypes.byref(epi), torch.cuda.current_stream().cuda_stream)


@pytest.mark.parametrize("op_dtype", [torch.bfloat16, torch.float16])
def test_noalloc_lse_matches_workspace_entry_point_on_two_calls(op_dtype):
    problems = [dict(seed=1, M=300, N=2500, K=264, dist="unscaled"),
                dict(seed=2, M=2048, N=8192, K=8192, dist="default")]
    for pr in problems:
        inp = kf_workloads.generate("bf16_scale_rowlse", **pr)
        X, W = inp["X"].to(op_dtype).to(DEV), inp["W"].to(op_dtype).to(DEV)
        chain = [("scale", {"scalar": 0.125}), ("row_logsumexp", {})]
        ref = kf.fused_gemm(X, W, chain)                       # caller-provided workspace
        out = torch.full((X.shape[0],), float("nan"), dtype=torch.float32, device=DEV)
        st = _noalloc(X, W, chain, out)
        assert st == kf.KF_OK, kf.status_string(st)
        torch.cuda.synchronize()
        check_f32(out, ref.double().cpu().numpy(), f"noalloc M={pr['M']}")
        st, raw = kf.get_device_error()
        assert st == kf.KF_OK, hex(raw)


def test_noalloc_rejects_problems_beyond_the_fixed_scratch():
    L = kf.lib()
    cap = L.kf_fused_gemm_lse_noalloc_max_bytes()
    assert cap == 4 << 20
    X = torch.zeros(8, 64, dtype=torch.bfloat16, device=DEV)
    W = torch.zeros(8, 64, dtype=torch.bfloat16, device=DEV)
    out = torch.zeros(8, dtype=torch.float32, device=DEV)
    chain = [("row_logsumexp", {})]
    keep = []
    epi = kf.make_epilogue(chain, keep)
    M = cap // 8 + 1          # one column tile of partials per row: just over the cap
    st = L.kf_fused_gemm_lse_noalloc(X.data_ptr(), kf.KF_BF16, 64, W.data_ptr(), kf.KF_BF16, 64, out.data_ptr(),
                                     kf.KF_F32, M, 8, 64, ctypes.byref(epi), None)
    assert st == kf.KF_ERR_WORKSPACE
    no_lse = kf.make_epilogue([("relu", {})], keep)
    st = L.kf_fused_gemm_lse_noalloc(X.data_ptr(), kf.KF_BF16, 64, W.data_ptr(), kf.KF_BF16, 64, out.data_ptr(),
                                     kf.KF_F32, 8, 8, 64, ctypes.byref(no_lse), None)
    assert st == kf.KF_ERR_INVALID_ARG
