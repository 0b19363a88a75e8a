"""Plant one mistake at a time in a copy of the oracle (on the CPU) and check that
the pins in test_oracle_pins.py catch it, and, on their own, the hand-worked
examples of test_golden.py.  This shows both constrain every part of the oracle
the parity tests rely on."""
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRC = os.path.join(ROOT, "oracle", "kf_oracle.c")

MUTATIONS = {
    "bias_sign": ("case ORC_BIAS: return v + orc_load", "case ORC_BIAS: return v - orc_load"),
    "gelu_cubic": ("0.044715 * v * v * v", "0.04715 * v * v * v"),
    "gemm_k_index": ("orc_load(jb->W, jb->wt, j * jb->ldw + k)",
                     "orc_load(jb->W, jb->wt, j * jb->ldw + (jb->K - 1 - k))"),
    "gn_unbiased_var": ("    var /= (double)gs;", "    var /= (double)(gs > 1 ? gs - 1 : 1);"),
    "gn_no_eps": ("sqrt(var + op->eps)", "sqrt(var)"),
    "lse_drop_max": ("return m + log(acc);", "return log(acc);"),
    "route_tie_upper": ("l[e] > l[best]", "l[e] >= l[best]"),
    "route_unstable": ("  for (int64_t p = 0; p < P; ++p) {\n    int32_t e = topk_ids[p];",
                       "  for (int64_t p = P - 1; p >= 0; --p) {\n    int32_t e = topk_ids[p];"),
    "swiglu_swap": ("s[j] = g * orc_sigmoid(g) * u;", "s[j] = u * orc_sigmoid(u) * g;"),
    "moe_drop_weight": ("y[c] += wt * acc;", "y[c] += acc;"),
    "bf16_round_bits": ("ldexp(1.0, e - 8)", "ldexp(1.0, e - 9)"),
    "scale_ignored": ("case ORC_SCALE: return v * op->scalar;", "case ORC_SCALE: return v;"),
    "rmsnorm_no_eps": ("sqrt(ss / (double)H + eps)", "sqrt(ss / (double)H)"),
    "rmsnorm_sum_not_mean": ("sqrt(ss / (double)H + eps)", "sqrt(ss + eps)"),
    "rmsnorm_unrounded_residual": ("const double h = orc_round_bf16(orc_load(R, rt, t * H + j) + Y[t * H + j]);",
                                   "const double h = orc_load(R, rt, t * H + j) + Y[t * H + j];"),
    "f16_exponent_bias": ("v = ldexp((double)(1024 + fr), ex - 25);", "v = ldexp((double)(1024 + fr), ex - 24);"),
    "f16_subnormal_scale": ("v = ldexp((double)fr, -24);", "v = ldexp((double)fr, -25);"),
    "rope_sin_sign": ("h[i] = a * c - b * v;", "h[i] = a * c + b * v;"),
    "rope_keys_unrotated": ("if (hd < nq + nkv) /* query and key heads", "if (hd < nq) /* query and key heads"),
    "rope_values_rotated": ("if (hd < nq + nkv) /* query and key heads", "if (hd < nq + 2 * nkv) /* query and key heads"),
    "rope_token_not_position": ("(double)cos_t[pos * half + i]", "(double)cos_t[t * half + i]"),
    "rope_adjacent_partner": ("const double a = h[i], b = h[i + half];", "const double a = h[i], b = h[i ^ 1];"),
    "kv_row_is_token": ("k_cache + (int64_t)row * nkv * d", "k_cache + t * nkv * d"),
    "moe_alpha_ignored": ("orc_sigmoid(jb->alpha * g)", "orc_sigmoid(g)"),
    "moe_gate_clamp_symmetric": ("g = fmin(g, jb->limit);", "g = fmax(fmin(g, jb->limit), -jb->limit);"),
    "moe_linear_offset_dropped": ("* (u + jb->c);", "* u;"),
    "moe_down_bias_outside_weight": ("if (jb->bd) acc += orc_load(jb->bd, ORC_BF16, e * H + c);\n        y[c] += wt * acc;",
                                     "y[c] += wt * acc;\n        if (jb->bd) y[c] += orc_load(jb->bd, ORC_BF16, e * H + c);"),
    "moe_up_bias_from_gate": ("u += orc_load(jb->bgu, ORC_BF16, e * 2 * I + I + n);",
                              "u += orc_load(jb->bgu, ORC_BF16, e * 2 * I + n);"),
    "grouped_f16_stride": ("static size_t orc_elt_size(int dt) { return dt == ORC_F32 ? 4 : 2; }",
                           "static size_t orc_elt_size(int dt) { return dt == ORC_BF16 ? 2 : 4; }"),
    "row_sum_drops_last": ("for (int64_t j = 0; j < n; ++j) acc += s[j];\n  return acc;",
                           "for (int64_t j = 0; j + 1 < n; ++j) acc += s[j];\n  return acc;"),
    "row_sum_is_mean": ("for (int64_t j = 0; j < n; ++j) acc += s[j];\n  return acc;",
                        "for (int64_t j = 0; j < n; ++j) acc += s[j];\n  return acc / (double)n;"),
    "residual_dropped": ("case ORC_RESIDUAL_ADD: return v + orc_load", "case ORC_RESIDUAL_ADD: return v + 0 * orc_load"),
}


@pytest.mark.parametrize("name", sorted(MUTATIONS))
def test_pins_catch_planted_mistake(name, tmp_path):
    old, new = MUTATIONS[name]
    src = open(SRC).read()
    assert src.count(old) == 1, f"mutation anchor for {name} not unique/found"
    mpath = tmp_path / "kf_oracle.c"
    mpath.write_text(src.replace(old, new))
    env = dict(os.environ, KF_ORACLE_SRC=str(mpath), KF_ORACLE_BUILD=str(tmp_path / "_build"))
    r = subprocess.run([sys.executable, "-m", "pytest", "-q", "-rf", "-p", "no:cacheprovider",
                        os.path.join(ROOT, "tests", "test_oracle_pins.py"),
                        os.path.join(ROOT, "tests", "test_golden.py")],
                       cwd=ROOT, env=env, capture_output=True, text=True, timeout=600)
    assert r.returncode != 0, f"nothing caught mutation {name}:\n{r.stdout[-2000:]}"
    for f in ("test_oracle_pins.py", "test_golden.py"):
        assert f"FAILED tests/{f}" in r.stdout, f"{f} did not catch mutation {name}:\n{r.stdout[-2000:]}"
