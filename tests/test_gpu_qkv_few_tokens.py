"""GPU parity of the QKV projection tail for one to eight tokens (clusters of
CTAs splitting K over 256-column tiles, partial rows pushed to their owning
CTA through distributed shared memory, bias, rotary embedding, key / value
cache rows; the gpt-oss decode kernel "Bias + RoPE + KV update" of Sec. IV-A)
against the oracle: the gpt-oss shape, 128- and 256-column heads, K of one
partial k-block and of four k-blocks, many heads, fp16 operands, fp32 / fp16
outputs, fp32 and absent bias, strided weight rows, out-of-range positions and
cache rows, repeats."""
import numpy as np
import pytest
import torch

import kf_workloads
import oracle
import paper_2606_02963_gb300 as kf
from tests._util import check_bf16, check_f32

pytestmark = pytest.mark.gpu
DEV = "cuda"
SENT = -7.0  # cache rows no token names keep this value


def _run(inp, nq, nkv, d, out_dtype=torch.bfloat16, bias=True, W=None, bias_f32=False):
    rows = int(inp["rows"])
    kc = torch.full((rows, nkv * d), SENT, dtype=out_dtype, device=DEV)
    vc = torch.full((rows, nkv * d), SENT, dtype=out_dtype, device=DEV)
    g = {k: v.to(DEV) for k, v in inp.items() if k != "rows"}
    b = None
    if bias:
        b = g["b"].float() if bias_f32 else g["b"]
    q = kf.qkv_rope_kv(g["X"], g["W"] if W is None else W, b, g["positions"], g["cache_rows"], g["cos"], g["sin"],
                       nq, nkv, d, kc, vc)
    assert kf.get_device_error()[0] == kf.KF_OK
    rq, rk, rv = oracle.qkv_rope_kv(inp["X"], inp["W"], inp["b"] if bias else None, inp["positions"],
                                    inp["cache_rows"], inp["cos"], inp["sin"], nq, nkv, d, rows)
    return (q, kc, vc), (rq, rk, rv)


def _check(got, ref, what, out_dtype=torch.bfloat16):
    q, kc, vc = got
    rq, rk, rv = ref
    chk = check_f32 if out_dtype == torch.float32 else check_bf16
    chk(q, rq, what + " q")
    named = np.flatnonzero(~np.isnan(rk[:, 0]))
    chk(kc[torch.as_tensor(named, device=DEV)], rk[named], what + " k")
    chk(vc[torch.as_tensor(named, device=DEV)], rv[named], what + " v")
    other = np.setdiff1d(np.arange(kc.shape[0]), named)
    o = torch.as_tensor(other, device=DEV)
    assert bool((kc[o] == SENT).all()) and bool((vc[o] == SENT).all()), f"{what}: unnamed rows written"


@pytest.mark.parametrize("T", [1, 2, 3, 8])
def test_gpt_oss_shape(T):
    s = kf_workloads.QKV_SHAPE
    inp = kf_workloads.qkv_generate(T, seed=300 + T, cache_rows=4096)
    got, ref = _run(inp, s["nq"], s["nkv"], s["d"])
    _check(got, ref, f"few T={T}")


@pytest.mark.parametrize("T", [1, 8])
@pytest.mark.parametrize("nq,nkv,d,H", [(8, 2, 128, 640), (2, 1, 256, 512), (32, 8, 128, 4096), (3, 2, 64, 8),
                                         (64, 8, 128, 512), (72, 4, 256, 256)])
def test_head_sizes_row_widths(nq, nkv, d, H, T):
    # 128- and 256-column heads; K of 8 (one partial k-block: clusters of one
    # CTA) and 256 (four k-blocks: clusters of at most four); 48 heads of 128
    # at H = 4096 (24 tiles); 80 heads of 128 and of 256 (40 and 80 tiles)
    inp = kf_workloads.qkv_generate(T, seed=310 + d + nq + T + H, H=H, nq=nq, nkv=nkv, d=d, cache_rows=64)
    got, ref = _run(inp, nq, nkv, d)
    _check(got, ref, f"few nq={nq} nkv={nkv} d={d} H={H} T={T}")


@pytest.mark.parametrize("out_dtype", [torch.float32, torch.float16])
def test_fp16_operands_and_wide_outputs(out_dtype):
    inp = kf_workloads.qkv_generate(5, seed=320, H=2880, nq=16, nkv=4, d=64, dtype="f16", cache_rows=300)
    got, ref = _run(inp, 16, 4, 64, out_dtype=out_dtype)
    _check(got, ref, f"few f16 -> {out_dtype}", out_dtype=out_dtype)


def test_no_bias_fp32_output_and_fp32_bias():
    inp = kf_workloads.qkv_generate(1, seed=321, H=384, nq=4, nkv=1, d=128, cache_rows=64)
    got, ref = _run(inp, 4, 1, 128, out_dtype=torch.float32, bias=False)
    _check(got, ref, "few no bias", out_dtype=torch.float32)
    got, ref = _run(inp, 4, 1, 128, bias_f32=True)
    _check(got, ref, "few fp32 bias")


def test_strided_weight_rows():
    # W rows 8 elements apart from the next row's start (the tensor map's row
    # stride)
    s = kf_workloads.QKV_SHAPE
    inp = kf_workloads.qkv_generate(4, seed=322, cache_rows=128)
    N, H = inp["W"].shape
    big = torch.zeros(N, H + 8, dtype=inp["W"].dtype)
    big[:, :H] = inp["W"]
    big[:, H:] = 1e4  # never read
    Wd = big.to(DEV)[:, :H]
    assert Wd.stride(0) == H + 8
    got, ref = _run(inp, s["nq"], s["nkv"], s["d"], W=Wd)
    _check(got, ref, "few strided W")


@pytest.mark.parametrize("bad_field", ["position", "cache_row"])
def test_out_of_range_token_skips_only_that_token(bad_field):
    nq, nkv, d = 4, 2, 64
    T = 6
    inp = kf_workloads.qkv_generate(T, seed=323, H=256, nq=nq, nkv=nkv, d=d, max_pos=512, cache_rows=128)
    bad = 3
    if bad_field == "position":
        inp["positions"][bad] = 512  # one past the tables
    else:
        inp["cache_rows"][bad] = -1
    rows = int(inp["rows"])
    kc = torch.full((rows, nkv * d), SENT, dtype=torch.bfloat16, device=DEV)
    vc = torch.full((rows, nkv * d), SENT, dtype=torch.bfloat16, device=DEV)
    q = torch.full((T, nq * d), SENT, dtype=torch.bfloat16, device=DEV)
    g = {k: v.to(DEV) for k, v in inp.items() if k != "rows"}
    kf.qkv_rope_kv(g["X"], g["W"], g["b"], g["positions"], g["cache_rows"], g["cos"], g["sin"], nq, nkv, d, kc, vc,
                   q_out=q)
    st, raw = kf.get_device_error()
    assert st == kf.KF_ERR_DEVICE_BOUNDS and raw & 8
    assert bool((q[bad] == SENT).all())
    if bad_field == "position":
        r = int(inp["cache_rows"][bad])
        assert bool((kc[r] == SENT).all()) and bool((vc[r] == SENT).all())
    good = torch.tensor([t for t in range(T) if t != bad])
    rq, rk, rv = oracle.qkv_rope_kv(inp["X"][good], inp["W"], inp["b"], inp["positions"][good],
                                    inp["cache_rows"][good], inp["cos"], inp["sin"], nq, nkv, d, rows)
    check_bf16(q[good.to(DEV)], rq, "few good tokens q")
    named = np.flatnonzero(~np.isnan(rk[:, 0]))
    check_bf16(kc[torch.as_tensor(named, device=DEV)], rk[named], "few good tokens k")
    check_bf16(vc[torch.as_tensor(named, device=DEV)], rv[named], "few good tokens v")
    assert kf.get_device_error()[0] == kf.KF_OK  # the read cleared the word


@pytest.mark.parametrize("T", [1, 8])
def test_repeats_bitwise(T):
    # each output's sum has a fixed order (k-blocks within a CTA, then the
    # CTAs' partials in cluster-rank order)
    s = kf_workloads.QKV_SHAPE
    inp = kf_workloads.qkv_generate(T, seed=324 + T)
    g = {k: v.to(DEV) for k, v in inp.items() if k != "rows"}
    outs = []
    for _ in range(3):
        kc = torch.zeros(int(inp["rows"]), s["nkv"] * s["d"], dtype=torch.bfloat16, device=DEV)
        vc = torch.zeros_like(kc)
        q = kf.qkv_rope_kv(g["X"], g["W"], g["b"], g["positions"], g["cache_rows"], g["cos"], g["sin"], s["nq"],
                           s["nkv"], s["d"], kc, vc)
        outs.append((q, kc, vc))
    torch.cuda.synchronize()
    for o in outs[1:]:
        assert all(torch.equal(x, y) for x, y in zip(o, outs[0]))
    assert kf.get_device_error()[0] == kf.KF_OK
