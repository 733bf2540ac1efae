"""Each planted mistake in the oracle must trip at least one pin.

The mutants are built from a copy of oracle/fusion_oracle.c with one textual change
each (a dropped term, a wrong sign or index, a flipped comparison, a wrong tie rule),
compiled with gcc into a temporary directory, and run on the CPU only.
"""
import ctypes
import os
import subprocess
import sys

import pytest

sys.path.insert(0, os.path.dirname(os.path.abspath(__file__)))

import oracle  # noqa: E402
from oracle_pins import ALL_PINS  # noqa: E402

MUTANTS = {
    "bf16_round_half_up": ("frac > 0.5 || (frac == 0.5 && fmod(whole, 2.0) == 1.0)", "frac >= 0.5"),
    "bf16_subnormal_spacing": ("lead = -126;", "lead = -127;"),
    "argmax_ties_to_last": ("if (s > bv) {", "if (s >= bv) {"),
    "b_index_off_by_one": ("khat[(int64_t)pb * dk + j]", "khat[(int64_t)(pb + 1 < N ? pb + 1 : pb) * dk + j]"),
    "no_key_normalisation": ("double inv = 1.0 / (nrm > 1e-12 ? nrm : 1e-12);", "double inv = 1.0;"),
    "sort_ties_to_last": ("(val[idx[j]] == val[cur] && idx[j] > cur)", "(val[idx[j]] == val[cur] && idx[j] < cur)"),
    "unweighted_size_sum": ("wsum += sizes[ra];", "wsum += 1.0;"),
    "unweighted_mean": ("num[j] += (double)sizes[ra] * load_elem", "num[j] += load_elem"),
    "dropped_score_sum": ("ssum += scores[ra];", ";"),
    "a_match_wrong_row": ("(int32_t)(base + 1 + 2 * match[(p - 2) / 2])", "(int32_t)(base + 2 * match[(p - 2) / 2])"),
    "unbiased_variance": ("var /= d;", "var /= (d - 1);"),
    "ln_without_eps": ("1.0 / sqrt(var + eps)", "1.0 / sqrt(var)"),
    "ln_no_bf16_rounding": ("v = bf16_to_double(double_to_bf16(v));", "v = v;"),
    "dropped_bias": ("l[k] = acc + (double)bias[k];", "l[k] = acc;"),
    "softmax_no_shift": ("S += exp(l[k] - lmax);", "S += exp(l[k]);"),
    "exit_strict_compare": ("(c >= tau) ? 1 : 0", "(c > tau) ? 1 : 0"),
    "prune_floor": ("double kk = ceil((double)rho[i] * (double)P);", "double kk = floor((double)rho[i] * (double)P);"),
    "prune_drops_cls": ("if (p > 0 && !kept[p - 1])", "if (p == 0 || !kept[p - 1])"),
    "compact_keeps_exited": ("if (exit_mask[i])\n            continue;", "if (0)\n            continue;"),
    "router_no_profile_scale": ("double mt = m * scale;", "double mt = m;"),
    "router_ceil": ("const double r = floor(v);", "const double r = ceil(v);"),
    "router_sigmoid_sign": ("exp(-(z + beta))", "exp(z + beta)"),
    "router_drops_beta": ("exp(-(z + beta))", "exp(-z)"),
    "router_patch_count": ("mt * (0.5 * (double)N)", "mt * (0.5 * (double)(N - 1))"),
    "router_no_clamp": ("if (mt > 1.0)\n            mt = 1.0;", "if (0)\n            mt = 1.0;"),
    "router_scale_inverted": ("(1.0 - tau_tgt) / (1.0 - tau_ref)", "(1.0 - tau_ref) / (1.0 - tau_tgt)"),
    "scores_dropped_bias": ("scores_out[t] = (float)(acc + b);", "scores_out[t] = (float)acc;"),
    "scores_reversed_weights": ("acc += load_elem(dtype, w, j) * load_elem(dtype, x, t * d + j);",
                                "acc += load_elem(dtype, w, d - 1 - j) * load_elem(dtype, x, t * d + j);"),
    "scores_float_accumulator": ("acc += load_elem(dtype, w, j) * load_elem(dtype, x, t * d + j);",
                                 "acc = (float)(acc + load_elem(dtype, w, j) * load_elem(dtype, x, t * d + j));"),
    "mlp_pool_unweighted": ("z[j] += (double)sizes[t] * load_elem(dtype, x, t * d + j);",
                            "z[j] += load_elem(dtype, x, t * d + j);"),
    "mlp_pool_weight_sum": ("wsum += (double)sizes[t];", "wsum += 1.0;"),
    "mlp_pool_includes_cls": ("for (int64_t t = o + 1; t < o + n; ++t) {\n                wsum",
                              "for (int64_t t = o; t < o + n; ++t) {\n                wsum"),
    "mlp_gelu_relu": ("double g = 0.5 * a * (1.0 + erf(a / sqrt(2.0)));", "double g = a > 0.0 ? a : 0.0;"),
    "mlp_gelu_tanh": ("double g = 0.5 * a * (1.0 + erf(a / sqrt(2.0)));",
                      "double g = 0.5 * a * (1.0 + tanh(0.7978845608 * (a + 0.044715 * a * a * a)));"),
    "mlp_no_hidden_rounding": ("g = bf16_to_double(double_to_bf16(g));", "g = g;"),
    "mlp_dropped_b1": ("a += (double)b1[k];", ";"),
    "mlp_w1_transposed": ("load_elem(dtype, W1, (int64_t)k * d + j)", "load_elem(dtype, W1, (int64_t)j * H + k)"),
    "mlp_w2_transposed": ("load_elem(dtype, W2, (int64_t)c * H + k)", "load_elem(dtype, W2, (int64_t)k * C + c)"),
    "attn_no_scale": ("l[j] = dot * scale + ", "l[j] = dot + "),
    "attn_size_not_log": ("(sizes ? log((double)sizes[o + j]) : 0.0)", "(sizes ? (double)sizes[o + j] : 0.0)"),
    "attn_k_from_q": ("ko = (int64_t)(H + h) * dh", "ko = (int64_t)h * dh"),
    "attn_v_from_k": ("vo = (int64_t)(2 * H + h) * dh", "vo = (int64_t)(H + h) * dh"),
    "attn_not_normalised": ("dst[e] = acc / S;", "dst[e] = acc;"),
    "scores_skip_last_row": ("for (int64_t t = offsets[i]; t < offsets[i + 1]; ++t) {",
                             "for (int64_t t = offsets[i]; t < offsets[i + 1] - 1; ++t) {"),
}


def _build_mutant(tmp_path, name, old, new):
    with open(os.path.join(os.path.dirname(oracle.__file__), "fusion_oracle.c")) as f:
        src = f.read()
    assert src.count(old) >= 1, f"mutation site for {name} not found"
    src = src.replace(old, new)
    c = tmp_path / f"{name}.c"
    so = tmp_path / f"lib{name}.so"
    c.write_text(src)
    subprocess.check_call(["gcc", "-O1", "-std=c11", "-fPIC", "-shared", "-o", str(so), str(c), "-lm"])
    return oracle.configure(ctypes.CDLL(str(so)))


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_mutant_is_caught(name, tmp_path):
    old, new = MUTANTS[name]
    lib = _build_mutant(tmp_path, name, old, new)
    saved = oracle._load()
    oracle._lib = lib
    caught = None
    try:
        for pin in ALL_PINS:
            try:
                pin()
            except (AssertionError, RuntimeError) as e:
                caught = (pin.__name__, str(e)[:120])
                break
    finally:
        oracle._lib = saved
    assert caught is not None, f"no pin caught the planted mistake {name}"
