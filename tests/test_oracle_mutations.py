"""Plant plausible mistakes in a copy of the oracle (on the CPU) and check that
the pins catch every one: a dropped term, a wrong sign, a wrong index, a wrong
exponent bias, a reversed bit order, a dropped path, a wrong chain step."""
import os
import subprocess

import pytest

import oracle
from tests import oracle_pins

SRC = os.path.join(os.path.dirname(oracle.__file__), "lb_oracle.c")

# (name, text in lb_oracle.c, replacement)
MUTATIONS = [
    ("u_sign_polarity", "return ((word >> (j % 32)) & 1u) ? -1 : 1;",
     "return ((word >> (j % 32)) & 1u) ? 1 : -1;"),
    ("v_bit_index", "return ((word >> (i % 32)) & 1u) ? -1 : 1;",
     "return ((word >> (j % 32)) & 1u) ? -1 : 1;"),
    ("v_word_index", "uint32_t word = words[(i / 32) * r + j];",
     "uint32_t word = words[(i / 32) * r + (r - 1 - j)];"),
    ("factored_drops_g", "a[tt * din + i] = X[tt * din + i] * lbo_half_to_double(P->g[i]);",
     "a[tt * din + i] = X[tt * din + i];"),
    ("factored_drops_l", "t[tj] *= lbo_half_to_double(P->l[tj % r]);", "t[tj] *= 1.0;"),
    ("factored_h_index", "y[to] += s * lbo_half_to_double(P->h[o]);",
     "y[to] += s * lbo_half_to_double(P->h[tt]);"),
    ("factored_one_path", "    int64_t t_off = 0;\n    for (int p = 0; p < L->n_paths; p++) {",
     "    int64_t t_off = 0;\n    for (int p = 0; p < 1; p++) {"),
    ("dense_drops_g", "W[o * din + i] += ho * s * gi;", "W[o * din + i] += ho * s;"),
    ("half_bias", "v = ldexp((double)(1024 + f), e - 25);", "v = ldexp((double)(1024 + f), e - 24);"),
    ("half_subnormal", "v = ldexp((double)f, -24);", "v = ldexp((double)f, -25);"),
    ("bf16_bias", "v = ldexp((double)(128 + f), e - 134);", "v = ldexp((double)(128 + f), e - 133);"),
    ("pack_bit_order", "word |= (uint32_t)1 << k;\n                else if (v != 1)\n                    return -1;\n            }\n            out[o * nw + w] = word;",
     "word |= (uint32_t)1 << (31 - k);\n                else if (v != 1)\n                    return -1;\n            }\n            out[o * nw + w] = word;"),
    ("rms_not_mean", "double inv = 1.0 / sqrt(ss / (double)n);", "double inv = 1.0 / sqrt(ss);"),
    ("chain_no_silu", "gt[i] = silu(gt[i]) * up[i];", "gt[i] = gt[i] * up[i];"),
    ("chain_gqa_index", "attn[j] = v[(hq / group) * head_dim + c];",
     "attn[j] = v[(hq % (dkv / head_dim)) * head_dim + c];"),
    ("chain_no_attn_residual", "a[i] += o[i];                       /* h = a + o */",
     "a[i] = o[i];"),
    ("chain_no_mlp_residual", "a[i] += dn[i];", "a[i] = dn[i];"),
    ("chain_silu_sign", "return x / (1.0 + exp(-x));", "return x / (1.0 + exp(x));"),
    ("bpw_drops_latent_scale", "+ 16.0 * (double)(d_out + d_in + r);", "+ 16.0 * (double)(d_out + d_in);"),
    ("rank_solve_one_path", "(n_paths * s + n_paths * 16.0);", "(s + n_paths * 16.0);"),
    ("latent_drops_l", "z[tt * n1 + off + j] = lbo_half_to_double(P->l[j]) * s;",
     "z[tt * n1 + off + j] = s;"),
    ("latent_drops_g",
     "s += X[tt * din + i] * lbo_half_to_double(P->g[i]) * sign_v(P->v_words, r, i, j);",
     "s += X[tt * din + i] * sign_v(P->v_words, r, i, j);"),
    ("latent_path_offset", "        off += r;\n    }\n    free(X);", "        off += 1;\n    }\n    free(X);"),
    ("expand_drops_h", "acc += lbo_half_to_double(P->h[o]) * s;", "acc += s;"),
    ("expand_path_offset", "            off += P->r;", "            off += 0;"),
    ("expand_u_transposed", "s += z[tt * n1 + off + j] * sign_u(P->u_words, P->r, o, j);",
     "s += z[tt * n1 + off + j] * sign_u(P->u_words, P->r, j % L->d_out, o % P->r);"),
    ("dsvid_no_sqrt_split", "double q = sqrt(s[j]);", "double q = s[j];"),
    ("dsvid_latent_lu_only", "l[j] = lu[j] * lv[j];", "l[j] = lu[j];"),
    ("dsvid_sign_of_zero", "usign[k] = U[k] < 0 ? -1 : 1;", "usign[k] = U[k] <= 0 ? -1 : 1;"),
    ("dsvid_no_abs", "        U[k] = fabs(U[k]);", "        U[k] = U[k];"),
    ("jacobi_rotation_sign", "y[i] = sn * a + c * b;", "y[i] = -sn * a + c * b;"),
    ("svd_sign_convention", "double sg = J[best * n + imax] < 0 ? -1.0 : 1.0;",
     "double sg = J[best * n + imax] > 0 ? -1.0 : 1.0;"),
    ("path_weight_drops_g", "What[o * d_in + i] = h[o] * acc * g[i];", "What[o * d_in + i] = h[o] * acc;"),
    ("qat_du_drops_h", "s += dY[tt * dout + o] * P->h[o] * z[tt * r + j];",
     "s += dY[tt * dout + o] * z[tt * r + j];"),
    ("qat_tanh_sign", "D->du[oj] = relaxed ? s : s * k * (1.0 - th * th);",
     "D->du[oj] = relaxed ? s : s * k * (1.0 + th * th);"),
    ("qat_dt_drops_l", "dz[tj] *= P->l[tj % r]; /* dz now holds dt */", "dz[tj] *= 1.0;"),
    ("qat_dg_drops_x", "s += da[tt * din + i] * X[tt * din + i];", "s += da[tt * din + i];"),
    ("qat_dx_drops_g", "dX[ti] += da[ti] * P->g[ti % din];", "dX[ti] += da[ti];"),
    ("qat_dl_index", "s += dz[tt * r + j] * t[tt * r + j];", "s += dz[tt * r + j] * t[tt * r + (r - 1 - j)];"),
    ("flops_factor", "return (double)n_paths * 2.0 * (double)T", "return (double)n_paths * 1.0 * (double)T"),
    ("bf16_ties_away", "if (rem > 0.5 || (rem == 0.5 && fmod(f, 2.0) != 0.0))", "if (rem >= 0.5)"),
    ("bf16_one_bit_short", "double q = ldexp(1.0, e - 8);", "double q = ldexp(1.0, e - 7);"),
    ("rope_frequency", "double th = (double)p * pow(base, -2.0 * (double)i / (double)D);",
     "double th = (double)p * pow(base, -1.0 * (double)i / (double)D);"),
    ("rope_rotation_sign", "x[i] = a * c - b * sn;", "x[i] = a * c + b * sn;"),
    ("rope_interleaved", "double c = cos(th), sn = sin(th), a = x[i], b = x[i + h];",
     "double c = cos(th), sn = sin(th), a = x[i], b = x[(i + 1) % D];"),
    ("attn_no_scale", "w[t] = s / sqrt((double)head_dim);", "w[t] = s;"),
    ("attn_group_index", "int64_t g = h / group;", "int64_t g = h % n_kv_heads;"),
    ("attn_not_normalised", "attn[(int64_t)h * head_dim + c] = acc / sum;",
     "attn[(int64_t)h * head_dim + c] = acc;"),
    ("attn_skips_new_row", "for (int64_t t = 0; t <= pos; t++) {\n                double s = 0.0;",
     "for (int64_t t = 0; t < pos; t++) {\n                double s = 0.0;"),
    ("decoder_cache_row", "memcpy(Kc + pos * dkv, k, (size_t)dkv * sizeof(double));",
     "memcpy(Kc + 0 * dkv, k, (size_t)dkv * sizeof(double));"),
    ("decoder_unrounded_attn", "                attn[i] = lbo_round_bf16(attn[i]);",
     "                attn[i] = attn[i];"),
    ("decoder_no_silu", "gt[i] = up[i] * silu(gt[i]);", "gt[i] = up[i] * gt[i];"),
    ("decoder_k_not_rotated", "            lbo_rope(k + (int64_t)g * head_dim, head_dim, pos, rope_base);",
     "            (void)g;"),
]


@pytest.mark.parametrize("name,old,new", MUTATIONS, ids=[m[0] for m in MUTATIONS])
def test_pins_catch_planted_mistake(tmp_path, name, old, new):
    src = open(SRC).read()
    assert src.count(old) == 1, f"mutation anchor for {name} not unique"
    mutated = tmp_path / "lb_oracle.c"
    mutated.write_text(src.replace(old, new))
    (tmp_path / "lb_oracle.h").write_text(open(SRC[:-1] + "h").read())
    so = tmp_path / f"liblboracle_{name}.so"
    subprocess.run(["gcc", "-std=c11", "-O2", "-fPIC", "-shared", "-fopenmp", "-ffp-contract=off",
                    "-o", str(so), str(mutated), "-lm"], check=True)
    bad = oracle.Oracle(str(so))
    caught = []
    for pin in oracle_pins.ALL_PINS:
        try:
            pin(bad)
        except (AssertionError, ValueError, MemoryError):
            caught.append(pin.__name__)
    assert caught, f"no pin caught the planted mistake {name}"
