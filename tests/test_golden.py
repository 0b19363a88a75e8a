"""Pins of the fp64 oracle against hand-worked examples (tests/golden/worked_examples.json).

Each case is a tiny input whose result follows from the definition of the step
by a few lines of arithmetic, written out in the fixture's 'derivation' and
stored as closed-form expressions; the section of the paper that defines the
step is in 'cite'.  The expected values never come from the oracle or from the
CUDA path."""
import json
import math
import os

import numpy as np
import pytest
import torch

import oracle

HERE = os.path.dirname(os.path.abspath(__file__))
FIXTURE = os.path.join(HERE, "golden", "worked_examples.json")

DTYPES = {"bf16": torch.bfloat16, "f32": torch.float32, "f16": torch.float16, "i32": torch.int32}


def load_cases():
    with open(FIXTURE) as f:
        return json.load(f)["cases"]


def tensor(spec):
    """A fixture tensor; its data must be exact in the stated dtype unless the
    fixture marks them 'rounded'."""
    if not isinstance(spec, dict):
        return spec
    t64 = torch.tensor(spec["data"], dtype=torch.float64)
    t = t64.to(DTYPES[spec["dtype"]])
    if not spec.get("rounded", False):
        assert torch.equal(t.to(torch.float64), t64), f"fixture data not exact in {spec['dtype']}"
    return t


def namespace(case):
    ns = {"sqrt": math.sqrt, "exp": math.exp, "log": math.log, "tanh": math.tanh, "pi": math.pi,
          "e": math.e, "nan": math.nan, "f32": lambda x: float(np.float32(x))}
    for k, expr in case.get("defs", {}).items():
        ns[k] = eval(expr, {"__builtins__": {}}, ns)
    return ns


def expected(tree, ns):
    if isinstance(tree, list):
        return [expected(x, ns) for x in tree]
    return float(eval(tree, {"__builtins__": {}}, ns))


def run(case):
    c = case["call"]
    if c == "fused_gemm":
        chain = [(kind, {k: tensor(v) for k, v in prm.items()}) for kind, prm in case["chain"]]
        return {"Y": oracle.fused_gemm(tensor(case["X"]), tensor(case["W"]), chain)}
    if c == "grouped_gemm":
        chain = [(kind, {k: tensor(v) for k, v in prm.items()}) for kind, prm in case["chain"]]
        return {"C": oracle.grouped_gemm(tensor(case["A"]), tensor(case["B"]), case["offsets"], case["N"], chain,
                                         row_index=case.get("row_index"), out_rows=case.get("out_rows"))}
    if c == "moe_route":
        return oracle.moe_route(tensor(case["logits"]), case["k"])
    if c == "moe_ffn":
        kw = {k: case[k] for k in ("alpha", "limit", "linear_offset") if k in case}
        for k in ("b_gu", "b_down"):
            if k in case:
                kw[k] = tensor(case[k])
        Y = oracle.moe_ffn(tensor(case["X"]), tensor(case["W_gu"]), tensor(case["W_down"]),
                           np.asarray(case["topk_ids"], np.int32), np.asarray(case["topk_w"], np.float64),
                           round_h=case["round_h"], **kw)
        return {"Y": Y}
    if c == "qkv_rope_kv":
        q, kc, vc = oracle.qkv_rope_kv(tensor(case["X"]), tensor(case["W"]), tensor(case["bias"]),
                                        case["positions"], case["cache_rows"], tensor(case["cos_t"]),
                                        tensor(case["sin_t"]), case["nq"], case["nkv"], case["d"], case["rows"])
        return {"q_out": q, "k_cache": kc, "v_cache": vc}
    if c == "add_rmsnorm":
        r_out, normed = oracle.add_rmsnorm(np.asarray(case["Y"], np.float64), tensor(case["R"]),
                                           tensor(case["gamma"]), case["eps"])
        return {"R_out": r_out, "normed": normed}
    raise AssertionError(f"unknown call {c}")


CASES = load_cases()


def test_fixture_is_complete():
    steps = {c["call"] for c in CASES}
    assert steps == {"fused_gemm", "grouped_gemm", "moe_route", "moe_ffn", "qkv_rope_kv", "add_rmsnorm"}
    for c in CASES:
        assert c["cite"].startswith("Sec. ") and c["derivation"] and c["expect"]


@pytest.mark.parametrize("case", CASES, ids=[c["name"] for c in CASES])
def test_worked_example(case):
    got = run(case)
    ns = namespace(case)
    for name, tree in case["expect"].items():
        want = np.asarray(expected(tree, ns), np.float64)
        have = np.asarray(got[name], np.float64)
        assert have.shape == want.shape, (name, have.shape, want.shape)
        nan = np.isnan(want)
        assert np.array_equal(np.isnan(have), nan), name
        np.testing.assert_allclose(have[~nan], want[~nan], rtol=case["rtol"], atol=case["atol"], err_msg=name)
