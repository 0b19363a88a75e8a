"""CPU tests of the C-ABI boundary: the library builds and loads, exports every
entry point include/kf.h declares, and rejects bad arguments on the host with a
status code before any CUDA call (no GPU needed: every call below returns during
argument checking)."""
import ctypes
import os
import re
import subprocess

import pytest

import paper_2606_02963_gb300 as kf
from paper_2606_02963_gb300 import build as kbuild

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def L():
    kbuild.build()
    return kf.lib()


def header_symbols():
    src = open(os.path.join(ROOT, "include", "kf.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(kf_[a-z_0-9]+)\s*\(", src)))


def test_header_declares_the_binding_symbols():
    assert header_symbols() == sorted(kf.ABI_SYMBOLS)


def test_library_exports_every_declared_symbol(L):
    out = subprocess.run(["nm", "-D", "--defined-only", kf.LIB_PATH], capture_output=True, text=True).stdout
    exported = set(re.findall(r" T (kf_\w+)", out))
    missing = [s for s in header_symbols() if s not in exported]
    assert not missing, missing
    for s in header_symbols():
        assert hasattr(L, s)


def test_status_strings(L):
    assert L.kf_abi_version() == 2
    for s in range(8):
        assert len(kf.status_string(s)) > 0
    assert "unknown" in kf.status_string(99)


A16, B16, C16 = 0x10000, 0x20000, 0x30000  # aligned fake device addresses, never dereferenced


def fused(L, X=A16, xt=1, ldx=64, W=B16, wt=1, ldw=64, Y=C16, yt=1, ldy=64, M=10, N=10, K=64, epi=None,
          ws=None, wsb=0):
    return L.kf_fused_gemm(X, xt, ldx, W, wt, ldw, Y, yt, ldy, M, N, K,
                           None if epi is None else ctypes.byref(epi), ws, wsb, None)


def epi_of(chain, keep):
    return kf.make_epilogue(chain, keep)


def test_fused_gemm_argument_errors(L):
    assert fused(L, X=None) == kf.KF_ERR_INVALID_ARG
    assert fused(L, W=None) == kf.KF_ERR_INVALID_ARG
    assert fused(L, Y=None) == kf.KF_ERR_INVALID_ARG
    assert fused(L, M=-1) == kf.KF_ERR_INVALID_ARG
    assert fused(L, K=0) == kf.KF_ERR_INVALID_ARG
    assert fused(L, ldx=32) == kf.KF_ERR_INVALID_ARG        # ld < K
    assert fused(L, ldy=5) == kf.KF_ERR_INVALID_ARG         # ldy < N
    assert fused(L, xt=7) == kf.KF_ERR_INVALID_ARG          # unknown dtype
    assert fused(L, xt=0, wt=1) == kf.KF_ERR_UNSUPPORTED    # mixed f32 x bf16
    assert fused(L, xt=0, wt=0, yt=1) == kf.KF_ERR_UNSUPPORTED  # fp32 path writes fp32
    # TMA alignment: base pointers and row strides
    assert fused(L, X=A16 + 2) == kf.KF_ERR_MISALIGNED
    assert fused(L, W=B16 + 8) == kf.KF_ERR_MISALIGNED
    assert fused(L, ldx=68) == kf.KF_ERR_MISALIGNED
    assert fused(L, ldw=66) == kf.KF_ERR_MISALIGNED
    # fp32 path has no alignment rule (checked up to the launch, which needs a GPU)
    # empty problems are no-ops
    assert fused(L, M=0) == kf.KF_OK
    assert fused(L, N=0) == kf.KF_OK


def test_fused_gemm_chain_errors(L):
    keep = []
    assert fused(L, epi=epi_of([("bias", {})], keep)) == kf.KF_ERR_INVALID_ARG  # bias needs p0
    bad = kf.Epilogue(1, ctypes.cast((kf.EpilogueOp * 1)(kf.EpilogueOp(kind=99)), ctypes.POINTER(kf.EpilogueOp)))
    assert fused(L, epi=bad) == kf.KF_ERR_INVALID_ARG
    too_many = kf.Epilogue(9, ctypes.cast((kf.EpilogueOp * 9)(), ctypes.POINTER(kf.EpilogueOp)))
    assert fused(L, epi=too_many) == kf.KF_ERR_INVALID_ARG
    # swiglu / scatter are grouped-only
    assert fused(L, epi=epi_of([("swiglu", {})], keep)) == kf.KF_ERR_INVALID_ARG
    # two reductions in one chain
    two = (kf.EpilogueOp * 2)(kf.EpilogueOp(kind=7), kf.EpilogueOp(kind=7))
    assert fused(L, epi=kf.Epilogue(2, ctypes.cast(two, ctypes.POINTER(kf.EpilogueOp)))) == kf.KF_ERR_UNSUPPORTED
    # only scalar ops may follow a row log-sum-exp
    lb = (kf.EpilogueOp * 2)(kf.EpilogueOp(kind=7), kf.EpilogueOp(kind=0, p0=B16, p_dtype=1))
    e = kf.Epilogue(2, ctypes.cast(lb, ctypes.POINTER(kf.EpilogueOp)))
    assert fused(L, epi=e, ws=A16, wsb=1 << 20) == kf.KF_ERR_INVALID_ARG
    # row log-sum-exp needs its workspace
    lse = kf.Epilogue(1, ctypes.cast((kf.EpilogueOp * 1)(kf.EpilogueOp(kind=7)), ctypes.POINTER(kf.EpilogueOp)))
    need = L.kf_fused_gemm_workspace(1000, 1000, 64, ctypes.byref(lse))
    assert need >= 1000 * 8 * 8
    assert fused(L, epi=lse, M=1000, N=1000, ldy=1000) == kf.KF_ERR_WORKSPACE
    assert fused(L, epi=lse, M=1000, N=1000, ws=A16, wsb=need - 1) == kf.KF_ERR_WORKSPACE
    # row sum: needs the workspace, only scalar ops after it, may follow a
    # GroupNorm (with pointwise ops between) but nothing else special
    op = lambda k, **kw: kf.EpilogueOp(kind=k, **kw)
    ep = lambda *ops: kf.Epilogue(len(ops), ctypes.cast((kf.EpilogueOp * len(ops))(*ops), ctypes.POINTER(kf.EpilogueOp)))
    rs = ep(op(15))
    need_rs = L.kf_fused_gemm_workspace(1000, 1000, 64, ctypes.byref(rs))
    assert need_rs == need and need_rs >= 256 + 1000 * 8 * 8
    assert fused(L, epi=rs, M=1000, N=1000, ldy=1) == kf.KF_ERR_WORKSPACE
    assert fused(L, epi=rs, M=1000, N=1000, ws=A16, wsb=need_rs - 1) == kf.KF_ERR_WORKSPACE
    assert fused(L, epi=ep(op(15), op(0, p0=B16, p_dtype=1)), ws=A16, wsb=1 << 20) == kf.KF_ERR_INVALID_ARG
    assert fused(L, epi=ep(op(15), op(15))) == kf.KF_ERR_UNSUPPORTED
    assert fused(L, epi=ep(op(7), op(15))) == kf.KF_ERR_UNSUPPORTED
    assert fused(L, epi=ep(op(15), op(8, groups=2, eps=1e-5))) == kf.KF_ERR_UNSUPPORTED
    gn_sum = ep(op(8, groups=2, eps=1e-5), op(12, scalar=0.1), op(15), op(1, scalar=2.0))
    assert fused(L, epi=gn_sum, N=64, ldy=1) == kf.KF_ERR_WORKSPACE   # planned; needs its partials
    assert L.kf_fused_gemm_workspace(1000, 1024, 64, ctypes.byref(gn_sum)) >= 256 + 1000 * 8 * 4
    assert fused(L, epi=ep(op(8, groups=2, eps=1e-5), op(15), op(0, p0=B16, p_dtype=1)), N=64, ldy=1,
                 ws=A16, wsb=1 << 20) == kf.KF_ERR_INVALID_ARG
    # GroupNorm: N % groups, group size rules
    gn = lambda g: kf.Epilogue(1, ctypes.cast((kf.EpilogueOp * 1)(kf.EpilogueOp(kind=8, groups=g, eps=1e-5)),
                                              ctypes.POINTER(kf.EpilogueOp)))
    assert fused(L, epi=gn(3), N=64, ldy=64) == kf.KF_ERR_INVALID_ARG     # 64 % 3
    assert fused(L, epi=gn(4), N=64, ldy=64) == kf.KF_ERR_UNSUPPORTED     # group of 16 columns
    assert fused(L, epi=gn(0), N=64, ldy=64) == kf.KF_ERR_INVALID_ARG


def test_workspace_header_calls_check_arguments(L):
    # the error-word calls refuse a missing or misaligned workspace before any
    # device access; the size queries include the header
    raw = ctypes.c_uint32(0)
    assert L.kf_check_device_error(None, None, ctypes.byref(raw)) == kf.KF_ERR_INVALID_ARG
    assert L.kf_check_device_error(A16 + 4, None, ctypes.byref(raw)) == kf.KF_ERR_INVALID_ARG
    assert L.kf_workspace_init(None, 1 << 20, None) == kf.KF_ERR_INVALID_ARG
    assert L.kf_workspace_init(A16, 255, None) == kf.KF_ERR_INVALID_ARG
    assert L.kf_grouped_gemm_workspace(100, 64, 64, 4, 0, None) == 0
    assert L.kf_grouped_gemm_workspace(100, 64, 64, 4, 1, None) == 256 + 100 * 64 * 2
    assert L.kf_moe_ffn_workspace(64, 2880, 2880, 32, 4) % 256 == 0


def grouped(L, A=A16, at=1, lda=64, a_rows=0, idx=None, B=B16, bt=1, ldb=64, bgs=64 * 64, off=C16, G=4,
            rows=100, N=64, K=64, C=0x40000, ct=1, ldc=64, epi=None, ws=None, wsb=0):
    return L.kf_grouped_gemm(A, at, lda, a_rows, idx, B, bt, ldb, bgs, off, G, rows, N, K, C, ct, ldc,
                             None if epi is None else ctypes.byref(epi), ws, wsb, None)


def test_grouped_gemm_argument_errors(L):
    assert grouped(L, off=None) == kf.KF_ERR_INVALID_ARG
    assert grouped(L, G=0) == kf.KF_ERR_INVALID_ARG
    assert grouped(L, G=5000) == kf.KF_ERR_INVALID_ARG
    assert grouped(L, at=0) == kf.KF_ERR_UNSUPPORTED
    assert grouped(L, bgs=64 * 63) == kf.KF_ERR_INVALID_ARG       # groups of B overlap
    assert grouped(L, B=B16 + 4) == kf.KF_ERR_MISALIGNED
    assert grouped(L, bgs=64 * 64 + 4) == kf.KF_ERR_MISALIGNED
    assert grouped(L, idx=0x50000, a_rows=0) == kf.KF_ERR_INVALID_ARG
    assert grouped(L, idx=0x50000, a_rows=10) == kf.KF_ERR_WORKSPACE  # gather needs workspace
    keep = []
    lse = kf.Epilogue(1, ctypes.cast((kf.EpilogueOp * 1)(kf.EpilogueOp(kind=7)), ctypes.POINTER(kf.EpilogueOp)))
    assert grouped(L, epi=lse) == kf.KF_ERR_UNSUPPORTED
    sc = kf.Epilogue(1, ctypes.cast((kf.EpilogueOp * 1)(kf.EpilogueOp(kind=10, p0=A16, p1=B16, ld=10)),
                                    ctypes.POINTER(kf.EpilogueOp)))
    assert grouped(L, epi=sc, ct=1) == kf.KF_ERR_UNSUPPORTED        # scatter target must be fp32
    sc0 = kf.Epilogue(1, ctypes.cast((kf.EpilogueOp * 1)(kf.EpilogueOp(kind=10, p0=A16, p1=B16, ld=0)),
                                     ctypes.POINTER(kf.EpilogueOp)))
    assert grouped(L, epi=sc0, ct=0) == kf.KF_ERR_INVALID_ARG       # destination row count
    assert grouped(L, rows=0) == kf.KF_OK


def test_moe_argument_errors(L):
    f = L.kf_moe_ffn
    ok = dict(X=A16, lg=B16, wgu=C16, wd=0x40000, Y=0x50000, T=8, H=64, I=64, E=4, k=2)

    def call(**kw):
        a = dict(ok, **kw)
        return f(a["X"], a["lg"], a["wgu"], a["wd"], a["Y"], a["T"], a["H"], a["I"], a["E"], a["k"],
                 None, 0, None, None, None)
    assert call(k=5) == kf.KF_ERR_INVALID_ARG
    assert call(E=300) == kf.KF_ERR_INVALID_ARG
    assert call(X=None) == kf.KF_ERR_INVALID_ARG
    assert call(H=60) == kf.KF_ERR_MISALIGNED
    assert call() == kf.KF_ERR_WORKSPACE
    assert call(T=0) == kf.KF_OK
    assert L.kf_moe_ffn_workspace(4096, 2880, 2880, 32, 4) > 4096 * 4 * 2880 * 4
    r = L.kf_moe_route
    assert r(A16, 8, 4, 5, B16, C16, 0x40000, 0x50000, 0x60000, None) == kf.KF_ERR_INVALID_ARG
    assert r(A16, 8, 4, 2, B16, C16, None, 0x50000, 0x60000, None) == kf.KF_ERR_INVALID_ARG


def test_product_path_does_not_touch_the_oracle():
    """The library and its binding never import or link the oracle."""
    pkg = os.path.join(ROOT, "paper_2606_02963_gb300")
    for dirpath, _, files in os.walk(pkg):
        for fn in files:
            if fn.endswith((".py", ".cu", ".cuh", ".h")):
                src = open(os.path.join(dirpath, fn)).read()
                assert "oracle" not in src.replace("oracle-free", ""), fn
    out = subprocess.run(["ldd", kf.LIB_PATH], capture_output=True, text=True).stdout
    assert "oracle" not in out


def test_moe_add_rmsnorm_argument_errors_before_any_launch():
    L = kf.lib()
    fake = 1 << 20  # aligned, never dereferenced: the checks come first
    def call(H=2880, eps=1e-5, R=fake):
        return L.kf_moe_ffn_add_rmsnorm(fake, fake, fake, fake, R, fake, eps, fake, fake, 4, H, 2880, 32, 4, 0,
                                        fake, 1 << 30, None, None, None)
    assert call(H=16384) == kf.KF_ERR_UNSUPPORTED
    assert call(eps=-1.0) == kf.KF_ERR_INVALID_ARG
    assert call(R=None) == kf.KF_ERR_INVALID_ARG
    assert call(R=fake + 4) == kf.KF_ERR_MISALIGNED


def test_mixed_f16_bf16_operands_are_refused(L):
    # one operand format per tcgen05 MMA: fp16 with bf16 is refused before any launch
    assert fused(L, xt=kf.KF_F16, wt=kf.KF_BF16) == kf.KF_ERR_UNSUPPORTED
    assert fused(L, xt=kf.KF_BF16, wt=kf.KF_F16) == kf.KF_ERR_UNSUPPORTED


def test_qkv_rope_kv_argument_errors_before_any_launch(L):
    fake = 1 << 20  # aligned, never dereferenced: the checks come first

    def call(T=4, H=2880, nq=64, nkv=8, d=64, xw=kf.KF_BF16, out=kf.KF_BF16, ldx=None, ldq=None, ldc=None,
             X=fake, cos=fake, max_pos=4096, rows=256, bias=None, bdt=kf.KF_BF16, kc=fake):
        return L.kf_qkv_rope_kv(X, fake, xw, H if ldx is None else ldx, H, bias, bdt, fake, fake, cos, fake,
                                max_pos, T, H, nq, nkv, d, fake, nq * d if ldq is None else ldq, kc, fake,
                                nkv * d if ldc is None else ldc, rows, out, None)
    assert call(d=96) == kf.KF_ERR_UNSUPPORTED          # half a head is not whole 32-column chunks
    assert call(d=512) == kf.KF_ERR_UNSUPPORTED
    assert call(xw=kf.KF_F32) == kf.KF_ERR_UNSUPPORTED  # tensor-core operands only
    assert call(out=kf.KF_I32) == kf.KF_ERR_INVALID_ARG
    assert call(nkv=0) == kf.KF_ERR_INVALID_ARG
    assert call(T=-1) == kf.KF_ERR_INVALID_ARG
    assert call(max_pos=0) == kf.KF_ERR_INVALID_ARG
    assert call(rows=0) == kf.KF_ERR_INVALID_ARG
    assert call(ldq=64 * 64 - 8) == kf.KF_ERR_INVALID_ARG
    assert call(ldc=8 * 64 - 8) == kf.KF_ERR_INVALID_ARG
    assert call(ldx=2000) == kf.KF_ERR_INVALID_ARG
    assert call(kc=None) == kf.KF_ERR_INVALID_ARG
    assert call(X=fake + 2) == kf.KF_ERR_MISALIGNED
    assert call(ldx=2884) == kf.KF_ERR_MISALIGNED
    assert call(cos=fake + 4) == kf.KF_ERR_MISALIGNED
    assert call(bias=fake, bdt=kf.KF_I32) == kf.KF_ERR_INVALID_ARG
    assert call(T=0, X=None, kc=None) == kf.KF_OK       # empty: nothing read or written


def test_moe_ffn_act_argument_errors_before_any_launch(L):
    fake = 1 << 20

    def call(alpha=1.702, limit=7.0, off=1.0, b_gu=fake, b_down=fake, act=True):
        a = kf.MoeAct(alpha, limit, off, b_gu, b_down)
        return L.kf_moe_ffn_act(fake, fake, fake, fake, ctypes.byref(a) if act else None, fake, 4, 2880, 2880, 32, 4,
                                0, fake, 1 << 30, None, None, None)
    assert call(act=False) == kf.KF_ERR_INVALID_ARG
    assert call(limit=-1.0) == kf.KF_ERR_INVALID_ARG
    assert call(alpha=float("nan")) == kf.KF_ERR_INVALID_ARG
    assert call(off=float("inf")) == kf.KF_ERR_INVALID_ARG
    assert call(b_gu=fake + 2) == kf.KF_ERR_MISALIGNED
    assert call(b_down=fake + 8) == kf.KF_ERR_MISALIGNED


def test_fused_gemm_ex_flags_checked_before_any_launch(L):
    fake = 1 << 20
    op = kf.EpilogueOp()
    epi = kf.Epilogue(0, ctypes.cast(ctypes.pointer(op), ctypes.POINTER(kf.EpilogueOp)))

    def call(flags, ldx=64, X=fake):
        return L.kf_fused_gemm_ex(X, kf.KF_F32, ldx, fake, kf.KF_F32, 64, fake, kf.KF_F32, 64, 64, 64, 64,
                                  ctypes.byref(epi), None, 0, flags, None)
    assert call(kf.KF_GEMM_F32_FFMA | kf.KF_GEMM_F32_TF32X3) == kf.KF_ERR_INVALID_ARG
    assert call(4) == kf.KF_ERR_INVALID_ARG
    assert call(kf.KF_GEMM_F32_TF32X3, ldx=66) == kf.KF_ERR_MISALIGNED
    assert call(kf.KF_GEMM_F32_TF32X3, X=fake + 4) == kf.KF_ERR_MISALIGNED
