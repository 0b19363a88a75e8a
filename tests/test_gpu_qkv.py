"""GPU parity of the QKV projection tail (bias, rotary embedding of query and key
heads, key / value cache rows; the gpt-oss decode kernel "Bias + RoPE + KV
update" of Sec. IV-A, here fused with the projection GEMM) against the oracle:
few-token calls (clusters splitting K, partials reduced in shared memory; token
boxes of 32 and 64 rows; clusters of one to three CTAs owning many rows), decode batches up to 128 tokens (one 128-row tile,
narrow tiles), prefill (CTA
pairs, ragged last row tile), 128- and 256-column heads, ragged last column
tile, fp16 operands, fp32 / fp16 outputs, outputs at odd offsets and strides,
no bias, out-of-range positions, untouched cache rows, repeat runs."""
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


def _run(inp, nq, nkv, d, out_dtype=torch.bfloat16, bias=True, sub=None):
    """The library's outputs and the oracle's, on the tokens `sub` (all if None)."""
    rows = int(inp["rows"])
    kc = torch.full((rows, nkv * d), SENT, dtype=out_dtype, device=DEV)
    vc = torch.full((rows, nkv * d), SENT, dtype=out_dtype, device=DEV)
    g = {k: v.to(DEV) for k, v in inp.items() if k != "rows"}
    q = kf.qkv_rope_kv(g["X"], g["W"], g["b"] if bias else None, g["positions"], g["cache_rows"], g["cos"],
                       g["sin"], nq, nkv, d, kc, vc)
    assert kf.get_device_error()[0] == kf.KF_OK
    idx = torch.arange(inp["X"].shape[0]) if sub is None else torch.as_tensor(sub)
    rq, rk, rv = oracle.qkv_rope_kv(inp["X"][idx], inp["W"], inp["b"] if bias else None, inp["positions"][idx],
                                    inp["cache_rows"][idx], inp["cos"], inp["sin"], nq, nkv, d, rows)
    return (q, kc, vc), (rq, rk, rv), idx


def _check(got, ref, idx, what, out_dtype=torch.bfloat16, all_tokens=True):
    q, kc, vc = got
    rq, rk, rv = ref
    chk = check_f32 if out_dtype == torch.float32 else check_bf16
    chk(q[idx.to(DEV)], rq, what + " q")
    named = np.flatnonzero(~np.isnan(rk[:, 0]))
    chk(kc[torch.as_tensor(named, device=DEV)], rk[named], what + " k")
    chk(vc[torch.as_tensor(named, device=DEV)], rv[named], what + " v")
    if all_tokens:
        other = np.setdiff1d(np.arange(kc.shape[0]), named)
        if other.size:
            o = torch.as_tensor(other, device=DEV)
            assert bool((kc[o] == SENT).all()) and bool((vc[o] == SENT).all()), f"{what}: unnamed rows written"


@pytest.mark.parametrize("T", [1, 16, 32, 33, 48, 49, 64, 65, 128])
def test_decode_gpt_oss_shape(T):
    # <= 64 tokens: clusters splitting K (32-row token boxes up to 32 tokens,
    # 64-row ones above); 65..128: one 128-row tile per CTA
    s = kf_workloads.QKV_SHAPE
    inp = kf_workloads.qkv_generate(T, seed=60 + T)
    got, ref, idx = _run(inp, s["nq"], s["nkv"], s["d"])
    _check(got, ref, idx, f"decode T={T}")


@pytest.mark.parametrize("T", [20, 45])
@pytest.mark.parametrize("nq,nkv,d", [(8, 2, 128), (2, 1, 256), (3, 2, 64)])
def test_few_tokens_other_head_sizes_and_ragged_tile(nq, nkv, d, T):
    # 128- and 256-column heads (two / four pairs per lane), and 7 heads of 64
    # (the last 256-column tile holds three heads)
    inp = kf_workloads.qkv_generate(T, seed=90 + d + nq + T, H=640, nq=nq, nkv=nkv, d=d, cache_rows=100)
    got, ref, idx = _run(inp, nq, nkv, d)
    _check(got, ref, idx, f"few tokens nq={nq} nkv={nkv} d={d}")


@pytest.mark.parametrize("T", [7, 45])
def test_few_token_path_repeats_bitwise(T):
    # the cluster reduction sums the partials in a fixed order
    s = kf_workloads.QKV_SHAPE
    inp = kf_workloads.qkv_generate(T, seed=95 + T)
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


@pytest.mark.parametrize("T", [129, 300])
def test_prefill_ragged_rows_on_cta_pairs(T):
    s = kf_workloads.QKV_SHAPE
    inp = kf_workloads.qkv_generate(T, seed=70 + T, H=512, prefill=True, cache_rows=1000)
    got, ref, idx = _run(inp, s["nq"], s["nkv"], s["d"])
    _check(got, ref, idx, f"prefill T={T}")


@pytest.mark.parametrize("T", [50, 200])
def test_head_dim_128(T):
    inp = kf_workloads.qkv_generate(T, seed=80 + T, H=256, nq=8, nkv=2, d=128, cache_rows=512)
    got, ref, idx = _run(inp, 8, 2, 128)
    _check(got, ref, idx, f"d=128 T={T}")


def test_ragged_last_column_tile():
    # nq + 2 nkv = 7 heads of 64: wide tiles end part-way (whole heads only)
    T = 300
    inp = kf_workloads.qkv_generate(T, seed=85, H=192, nq=3, nkv=2, d=64, cache_rows=700)
    got, ref, idx = _run(inp, 3, 2, 64)
    _check(got, ref, idx, "7 heads")


@pytest.mark.parametrize("T", [8, 64])
@pytest.mark.parametrize("out_dtype", [torch.float32, torch.float16])
def test_fp16_operands_and_wide_outputs(out_dtype, T):
    inp = kf_workloads.qkv_generate(T, seed=90, H=2880, nq=16, nkv=4, d=64, dtype="f16", cache_rows=300)
    got, ref, idx = _run(inp, 16, 4, 64, out_dtype=out_dtype)
    _check(got, ref, idx, f"f16 -> {out_dtype}", out_dtype=out_dtype)


def test_no_bias_fp32_output():
    inp = kf_workloads.qkv_generate(10, seed=91, H=384, nq=4, nkv=1, d=128, cache_rows=64)
    got, ref, idx = _run(inp, 4, 1, 128, out_dtype=torch.float32, bias=False)
    _check(got, ref, idx, "no bias", out_dtype=torch.float32)


@pytest.mark.parametrize("nq,nkv,d,H,T", [(3, 2, 64, 8, 45), (3, 2, 64, 8, 64), (8, 2, 64, 128, 64),
                                           (8, 2, 128, 192, 33), (4, 4, 64, 64, 17)])
def test_few_k_blocks_many_rows_per_cta(nq, nkv, d, H, T):
    # K of one to three k-blocks: clusters of one to three CTAs, so a CTA owns
    # up to 64 of the tile's token rows and an epilogue warp reduces up to 8 of
    # them (positions of all, table rows two ahead), staged and direct
    inp = kf_workloads.qkv_generate(T, seed=70 + H + T, H=H, nq=nq, nkv=nkv, d=d, cache_rows=256)
    got, ref, idx = _run(inp, nq, nkv, d)
    _check(got, ref, idx, f"H={H} T={T}")


@pytest.mark.parametrize("T", [3, 20, 64, 100])
@pytest.mark.parametrize("out_dtype", [torch.bfloat16, torch.float32])
def test_outputs_at_odd_offsets_and_strides(out_dtype, T):
    # q_out and the caches one element past an aligned start, rows an odd number
    # of elements apart: no vector store is legal, every output goes through
    # the element-wise stores (clusters with direct and with staged partial
    # rows, one tcgen05 tile)
    s = kf_workloads.QKV_SHAPE
    nq, nkv, d = s["nq"], s["nkv"], s["d"]
    inp = kf_workloads.qkv_generate(T, seed=95 + T, cache_rows=256)
    rows = int(inp["rows"])
    qb = torch.full((T, nq * d + 3), SENT, dtype=out_dtype, device=DEV)
    kb = torch.full((rows, nkv * d + 3), SENT, dtype=out_dtype, device=DEV)
    vb = torch.full((rows, nkv * d + 3), SENT, dtype=out_dtype, device=DEV)
    q, kc, vc = qb[:, 1:1 + nq * d], kb[:, 1:1 + nkv * d], vb[:, 1:1 + nkv * d]
    g = {k: v.to(DEV) for k, v in inp.items() if k != "rows"}
    kf.qkv_rope_kv(g["X"], g["W"], g["b"], g["positions"], g["cache_rows"], g["cos"], g["sin"], nq, nkv, d, kc, vc,
                   q_out=q)
    assert kf.get_device_error()[0] == kf.KF_OK
    for buf in (qb, kb, vb):  # the columns around the views stay untouched
        assert bool((buf[:, 0] == SENT).all()) and bool((buf[:, -2:] == SENT).all())
    rq, rk, rv = oracle.qkv_rope_kv(inp["X"], inp["W"], inp["b"], inp["positions"], inp["cache_rows"], inp["cos"],
                                    inp["sin"], nq, nkv, d, rows)
    _check((q, kc, vc), (rq, rk, rv), torch.arange(T), f"odd offsets T={T}", out_dtype=out_dtype)


@pytest.mark.parametrize("T", [12, 40, 100])
def test_out_of_range_position_skips_only_that_token(T):
    nq, nkv, d = 4, 2, 64
    inp = kf_workloads.qkv_generate(T, seed=92, H=256, nq=nq, nkv=nkv, d=d, max_pos=512, cache_rows=128)
    bad = 7
    inp["positions"][bad] = 512  # one past the tables
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
    r = int(inp["cache_rows"][bad])
    assert bool((kc[r] == SENT).all()) and bool((vc[r] == SENT).all())
    good = torch.tensor([t for t in range(T) if t != bad])
    rq, rk, rv = oracle.qkv_rope_kv(inp["X"][good], inp["W"], inp["b"], inp["positions"][good],
                                    inp["cache_rows"][good], inp["cos"], inp["sin"], nq, nkv, d, rows)
    _check((q, kc, vc), (rq, rk, rv), good, "bad position")
    assert kf.get_device_error()[0] == kf.KF_OK  # the read cleared the word


def test_full_size_prefill_sampled_tokens_and_repeats():
    # 4096-token prefill at the gpt-oss shape, checked on sampled tokens; the
    # path's arithmetic order is fixed, so repeated calls agree bit for bit
    s = kf_workloads.QKV_SHAPE
    T = 4096
    inp = kf_workloads.qkv_generate(T, seed=93, prefill=True, cache_rows=8192)
    sub = [0, 1, 127, 128, 255, 256, 2047, 3001, T - 1]
    got, ref, idx = _run(inp, s["nq"], s["nkv"], s["d"], sub=sub)
    _check(got, ref, idx, "prefill 4096 sampled", all_tokens=False)
    g = {k: v.to(DEV) for k, v in inp.items() if k != "rows"}
    for _ in range(3):
        kc = torch.full_like(got[1], SENT)
        vc = torch.full_like(got[2], SENT)
        q = kf.qkv_rope_kv(g["X"], g["W"], g["b"], g["positions"], g["cache_rows"], g["cos"], g["sin"],
                           s["nq"], s["nkv"], s["d"], kc, vc)
        assert torch.equal(q, got[0]) and torch.equal(kc, got[1]) and torch.equal(vc, got[2])
    assert kf.get_device_error()[0] == kf.KF_OK
