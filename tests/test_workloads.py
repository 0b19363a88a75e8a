"""The seeded input generators both sides read (kf_workloads): the same seed gives
the same tensors and another seed others, shapes and dtypes follow each
workload's recipe, the distributions are the stated ones, and the rotary tables
and cache rows of the QKV inputs are well formed.  CPU only."""
import math

import pytest
import torch

import kf_workloads as kw


def _same(a, b):
    return a.keys() == b.keys() and all(torch.equal(a[k], b[k]) for k in a)


@pytest.mark.parametrize("name", sorted(kw.WORKLOADS))
def test_generate_is_seeded(name):
    small = dict(M=64, N=96, K=80)
    a = kw.generate(name, seed=3, **small)
    assert _same(a, kw.generate(name, seed=3, **small))
    b = kw.generate(name, seed=4, **small)
    assert not torch.equal(a["X"], b["X"])


@pytest.mark.parametrize("name", sorted(kw.WORKLOADS))
def test_generate_shapes_and_dtypes(name):
    wl = kw.WORKLOADS[name]
    M, N, K = 64, 96, 80
    d = kw.generate(name, seed=0, M=M, N=N, K=K)
    dt = torch.float32 if wl.dtype == "f32" else torch.bfloat16
    assert d["X"].shape == (M, K) and d["W"].shape == (N, K)
    assert all(v.dtype == dt for v in d.values())
    for kind, prm in kw.chain_spec(wl):  # every tensor the chain names exists, with its shape
        for slot in ("p0", "p1"):
            key = prm.get(slot)
            if isinstance(key, str):
                assert d[key].shape == ((M, N) if kind == "residual_add" else (N,)), (kind, slot)


def test_headline_full_size_recipe():
    wl = kw.WORKLOADS["bf16_gelu_scale_residual"]
    assert (wl.M, wl.N, wl.K) == (1024, 4096, 4096)
    d = kw.generate("bf16_gelu_scale_residual", seed=0)
    assert d["X"].shape == (1024, 4096) and d["W"].shape == (4096, 4096)
    assert d["b"].shape == (4096,) and d["R"].shape == (1024, 4096)
    s = 1.0 / math.sqrt(4096)
    for k in ("X", "W", "R"):
        x = d[k].float()
        assert abs(float(x.mean())) < 0.02 * s and abs(float(x.std()) / s - 1.0) < 0.01, k


def test_distributions():
    d = kw.generate("fp32_relu_linear", seed=1)
    for k in ("X", "W", "b"):
        assert float(d[k].min()) >= -1.0 and float(d[k].max()) < 1.0
    g = kw.generate("bf16_groupnorm_swish", seed=1, M=32, N=1024, K=64)
    assert 0.5 <= float(g["gamma"].float().min()) and float(g["gamma"].float().max()) <= 1.5
    lim = float(torch.tensor(0.1).to(torch.bfloat16))  # the bound as rounded to bf16
    assert -lim <= float(g["beta"].float().min()) and float(g["beta"].float().max()) <= lim
    u = kw.generate("bf16_gelu_scale_residual", seed=1, M=64, N=64, K=64, dist="unscaled")
    assert abs(float(u["W"].float().std()) - 1.0) < 0.05
    o = kw.generate("bf16_gelu_scale_residual", seed=1, M=64, N=64, K=64, dist="offset")
    base = kw.generate("bf16_gelu_scale_residual", seed=1, M=64, N=64, K=64)
    # +8 is added to the fp32 draw before rounding: within one bf16 step of [8, 16)
    assert torch.allclose(o["b"].float(), base["b"].float() + 8.0, rtol=0.0, atol=2.0 ** -4)


def test_moe_generators():
    a = kw.moe_generate(8, seed=2, H=64, I=32, E=4)
    assert _same(a, kw.moe_generate(8, seed=2, H=64, I=32, E=4))
    assert a["X"].shape == (8, 64) and a["logits"].shape == (8, 4) and a["logits"].dtype == torch.float32
    assert a["W_gu"].shape == (4, 64, 64) and a["W_down"].shape == (4, 64, 32)
    assert abs(float(a["W_gu"].float().std()) - 0.02) < 0.003
    b = kw.moe_bias_generate(4, 64, 32, seed=2)
    assert b["b_gu"].shape == (4, 64) and b["b_down"].shape == (4, 64) and b["b_gu"].dtype == torch.bfloat16


def test_qkv_generator_decode_and_prefill():
    nq, nkv, d = 4, 2, 64
    dec = kw.qkv_generate(50, seed=5, H=128, nq=nq, nkv=nkv, d=d, max_pos=512, cache_rows=300)
    assert _same(dec, kw.qkv_generate(50, seed=5, H=128, nq=nq, nkv=nkv, d=d, max_pos=512, cache_rows=300))
    assert dec["W"].shape == ((nq + 2 * nkv) * d, 128) and dec["b"].shape == ((nq + 2 * nkv) * d,)
    assert int(dec["rows"]) == 300
    assert dec["positions"].dtype == torch.int32 and dec["cache_rows"].dtype == torch.int32
    assert int(dec["positions"].min()) >= 0 and int(dec["positions"].max()) < 512
    crow = dec["cache_rows"]
    assert int(crow.min()) >= 0 and int(crow.max()) < 300 and crow.unique().numel() == 50
    pre = kw.qkv_generate(40, seed=6, H=128, nq=nq, nkv=nkv, d=d, max_pos=512, cache_rows=300, prefill=True)
    assert torch.equal(pre["positions"], torch.arange(40, dtype=torch.int32))
    r = pre["cache_rows"]
    assert torch.equal(r, torch.arange(int(r[0]), int(r[0]) + 40, dtype=torch.int32)) and int(r[-1]) < 300
    # tables: unit circle; row 1 holds the per-pair frequencies theta^(-2i/d)
    c, s = dec["cos"].double(), dec["sin"].double()
    assert c.shape == (512, d // 2) and torch.allclose(c * c + s * s, torch.ones_like(c), atol=1e-6)
    i = torch.arange(d // 2, dtype=torch.float64)
    want = 150000.0 ** (-2.0 * i / d)
    assert torch.allclose(torch.atan2(s[1], c[1]), want, atol=1e-6)
    with pytest.raises(ValueError):
        kw.qkv_generate(20, H=64, nq=1, nkv=1, d=64, cache_rows=10)
