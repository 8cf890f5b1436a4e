"""Planted mistakes in the oracle are caught by the pins (no GPU).

Each mutant is a copy of ``oracle/fasgd_oracle.c`` with one plausible slip
(a dropped term, a wrong sign, a swapped operand or index, an off-by-one),
built on the CPU into a temporary directory.  Every mutant must fail at
least one check of ``pins.ALL_CHECKS``; a mutant that passes them all would
show a hole in the pins.
"""

import os
import subprocess

import pytest

import oracle
import pins

MUTANTS = {
    "n_drops_one_minus_gamma": ("(1 - gamma) * (g * g)", "(g * g)"),
    "n_uses_g_not_g2": ("(1 - gamma) * (g * g)", "(1 - gamma) * g"),
    "b_swaps_gamma": ("*b = gamma * *b + (1 - gamma) * g", "*b = (1 - gamma) * *b + gamma * g"),
    "var_sign": ("*n - *b * *b", "*n + *b * *b"),
    "var_drops_b2": ("ora_max0(*n - *b * *b)", "ora_max0(*n)"),
    "eps_dropped": ("ora_sqrt(var + eps)", "ora_sqrt(var)"),
    "r_not_inverted": ("REAL r = 1 / ora_sqrt(var + eps);", "REAL r = ora_sqrt(var + eps);"),
    "v_swaps_beta": ("*v = beta * *v + (1 - beta) * r", "*v = (1 - beta) * *v + beta * r"),
    "step_times_v": ("coef * g / *v", "coef * g * *v"),
    "step_sign": ("*theta = *theta - coef * g / *v", "*theta = *theta + coef * g / *v"),
    "step_uses_old_v": (
        "*v = beta * *v + (1 - beta) * r;                  /* Eq. 6 */\n"
        "        *theta = *theta - coef * g / *v;                  /* Eq. 7-8 */",
        "*theta = *theta - coef * g / (*v == 0 ? 1 : *v);\n"
        "        *v = beta * *v + (1 - beta) * r;"),
    "sgd_sign": ("*theta = *theta - coef * g;", "*theta = *theta + coef * g;"),
    "tau_not_clamped_at_1": ("int64_t t = tau < 1 ? 1 : tau;", "int64_t t = tau < 1 ? 2 : tau;"),
    "sasgd_multiplies": ("(double)alpha / (double)t", "(double)alpha * (double)t"),
    "asgd_divides_too": ("    if (variant == ORA_ASGD)\n        return (REAL)alpha;\n", ""),
    "philox_swaps_lo": ("uint32_t y1 = lo1;", "uint32_t y1 = lo0;"),
    "philox_bumps_first": ("if (round > 0) {", "if (round >= 0) {"),
    "philox_mult_constant": ("mult1 = 0xCD9E8D57u", "mult1 = 0xCD9E8D55u"),
    "draw_wrong_word": ("out[p & 3] >> 8", "out[(p + 1) & 3] >> 8"),
    "draw_low_bits": ("out[p & 3] >> 8", "out[p & 3] & 0xFFFFFFu"),
    "draw_counter_no_client": ("client | (stream << 31)", "0u | (stream << 31)"),
    "draw_streams_collide": ("client | (stream << 31)", "client"),
    "fetch_uses_push_stream": ("return ora_select_stream(P, theta, v, c, eps_b, seed, 1,",
                               "return ora_select_stream(P, theta, v, c, eps_b, seed, 0,"),
    "fetch_apply_wrong_slot": ("theta_client[idx[i]] = val[i];", "theta_client[i] = val[i];"),
    "mean_v_wrong_divisor": ("return ora_sum_mean(&s, P);", "return ora_sum_mean(&s, P + 1);"),
    "mean_v_first_only": ("for (int64_t p = 0; p < P; p++)\n        ora_sum_add(&s, (double)v[p]);",
                          "for (int64_t p = 0; p < 1; p++)\n        ora_sum_add(&s, (double)v[p]);"),
    "mean_v_fp64_sequential": ("return ora_sum_mean(&s, P);",
                               "{ double t = 0; for (int64_t p = 0; p < P; p++) t += (double)v[p];"
                               " return (float)(t / (double)P); }"),
    "mean_ties_away": ("if (guard && (sticky || (mant & 1u)))", "if (guard)"),
    "mean_truncates": ("if (guard && (sticky || (mant & 1u)))\n        mant++;",
                       "if (guard && (sticky || (mant & 1u)))\n        mant += 0;"),
    "mean_drops_remainder": ("int sticky = r != 0;", "int sticky = 0;"),
    "mean_drops_low_bits": ("sticky = (q[bit / 32] >> (bit % 32)) & 1u;", "sticky = 0;"),
    "mean_ignores_sign": ("ora_acc_add(neg ? s->neg : s->pos, m,", "ora_acc_add(s->pos, m,"),
    "mean_exponent_off_by_one": ("E == 0 ? 0 : E - 1", "E == 0 ? 0 : E"),
    "mean_carry_dropped": ("c = (c >> 32) + (uint64_t)w[i + 2] + (hi >> 32);",
                           "c = (uint64_t)w[i + 2] + (hi >> 32);"),
    "decide_not_strict": ("< (double)a * 16777216.0", "<= (double)a * 16777216.0"),
    "decide_product_in_fp32": ("(double)u * (double)d <", "(double)((float)u * d) <"),
    "decide_threshold_scale": ("(double)a * 16777216.0", "(double)a * 8388608.0"),
    "tensor_mean_divisor": ("vbar[t] = ora_sum_mean(&s, sizes[t]);",
                            "vbar[t] = ora_sum_mean(&s, sizes[t] + 1);"),
    "tensor_mean_no_offset": ("vbar[t] = ora_sum_mean(&s, sizes[t]);\n        off += sizes[t];",
                              "vbar[t] = ora_sum_mean(&s, sizes[t]);"),
    "message_draw_collides": ("uint32_t ctr[4] = {0xFFFFFFFFu,", "uint32_t ctr[4] = {0u,"),
    "message_draw_ignores_stream": ("{0xFFFFFFFFu, client | (stream << 31),", "{0xFFFFFFFFu, client,"),
    "std_variant_inverts": ("REAL r = ora_sqrt(var + eps);\n        *v = beta", "REAL r = 1 / ora_sqrt(var + eps);\n        *v = beta"),
    "sim_noise_half_range": ("(1.0f / 8388608.0f) - 0.5f", "(1.0f / 16777216.0f) - 0.5f"),
    "sim_grad_sign": ("float d = theta[p] - star[p];\n        g[p]", "float d = star[p] - theta[p];\n        g[p]"),
    "sim_loss_no_half": ("return 0.5 * s;", "return s;"),
    "decide_drops_eps": ("float a = v + eps_b;", "float a = v;"),
    "select_val_index": ("val[m] = g[p];", "val[m] = g[m];"),
    "select_idx_off_by_one": ("idx[m] = (int32_t)p;", "idx[m] = (int32_t)(p + 1);"),
    "sparse_val_reversed": ("(REAL)val[i], coef,", "(REAL)val[count - 1 - i], coef,"),
    "sparse_no_order_check": ("if (i > 0 && idx[i] <= idx[i - 1])\n            return -1;\n", ""),
    "budget_term_scale": ("int shift = e - 24 + 32;", "int shift = e - 24 + 31;"),
    "budget_ignores_size": ("int64_t prod = size * M;", "int64_t prod = M;"),
    "budget_drops_eps": ("float a = vbar + eps_b;\n    if (!(a > 0.0f)",
                         "float a = vbar;\n    if (!(a > 0.0f)"),
    "budget_returns_lo": ("    return ora_float_of_bits(hi);\n}", "    return ora_float_of_bits(lo);\n}"),
    "budget_no_zero_shortcut": ("vbar, eps_b, 0.0f) <= limit)\n        return 0.0f;",
                                "vbar, eps_b, 0.0f) < limit)\n        return 0.0f;"),
    "tensor_draw_word": ("return out[t & 3] >> 8;", "return out[(t + 1) & 3] >> 8;"),
    "tensor_draw_param_domain": ("0x80000000u + ((uint32_t)t >> 2)", "((uint32_t)t >> 2)"),
    "tensor_select_counts_tensors": ("m += sizes[t];\n    }\n    return m;",
                                     "m += 1;\n    }\n    return m;"),
    "apply_tensors_offset": ("gamma, beta, eps);\n        off += sizes[t];",
                             "gamma, beta, eps);\n        off += sent[t] ? sizes[t] : 0;"),
    "dense_skips_last": ("for (int64_t p = 0; p < P; p++)\n        ora_update_one",
                         "for (int64_t p = 0; p < P - 1; p++)\n        ora_update_one"),
}


def _build_mutant(tmp_path, name, old, new):
    src = open(oracle._SRC).read()
    assert old in src, f"mutant {name}: pattern no longer in the oracle source"
    mutated = src.replace(old, new, 1)
    cpath = tmp_path / f"{name}.c"
    cpath.write_text(mutated)
    libs = {}
    for real, ctype in (("f32", "float"), ("f64", "double")):
        out = tmp_path / f"lib{name}_{real}.so"
        subprocess.run(["gcc", *oracle._CFLAGS, "-w", f"-DREAL={ctype}", str(cpath),
                        "-o", str(out), "-lm"], check=True)
        libs[real] = oracle.load_library(str(out), real)
    return pins.Libs(libs["f32"], libs["f64"])


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_mutant_is_caught(tmp_path, name):
    old, new = MUTANTS[name]
    libs = _build_mutant(tmp_path, name, old, new)
    caught = None
    for check in pins.ALL_CHECKS:   # the first pin that fails catches the mutant
        try:
            check(libs)
        except Exception as e:      # any failure of a pin counts as a catch
            caught = f"{check.__name__}: {type(e).__name__}"
            break
    assert caught is not None, f"mutant {name} passed every pin"
