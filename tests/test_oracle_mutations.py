"""Plants plausible mistakes in a copy of the oracle and checks the pins catch each.

Each mutation edits one line of ``oracle/rola_oracle.c`` (a sign, an index, a
divisor, a dropped factor, a swapped order), compiles it to a temporary
library and runs the pin suite against it in a subprocess: the suite must
fail.  CPU only; nothing here touches the CUDA library.
"""
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRC = os.path.join(ROOT, "oracle", "rola_oracle.c")

MUTATIONS = {
    "rotation_sign": ("out[2 * m] = x * ca - y * sa;", "out[2 * m] = x * ca + y * sa;"),
    "rotation_pair_swap": ("out[2 * m + 1] = x * sa + y * ca;", "out[2 * m + 1] = y * sa + x * ca;"),
    "frequency_exponent": ("pow(c->theta, -2.0 * (double)i / (double)d_axis)",
                           "pow(c->theta, -1.0 * (double)i / (double)d_axis)"),
    "axis_boundary": ("if (m < pt) { axis = 0;", "if (m <= pt) { axis = 0;"),
    "position_row_index": ("int x = (n / c->Ww) % c->Hh;", "int x = (n / c->Hh) % c->Ww;"),
    "silu_sign": ("return x / (1.0 + exp(-x));", "return x / (1.0 + exp(x));"),
    "truncation_pairs": ("rotate_pairs(r / 2, cs, u, feat, r);\n    } else if",
                         "rotate_pairs(r / 2 - 1, cs, u, feat, r);\n    } else if"),
    "summary_transposed": ("Cb[(size_t)a * dh + d] += kt[a] * (double)vn[d];",
                           "Cb[(size_t)a * dh + d] += kt[a] * (double)vn[(d + 1) % dh];"),
    "mask_tie_order": ("return (x->j < y->j) ? -1 : (x->j > y->j);",
                       "return (x->j > y->j) ? -1 : (x->j < y->j);"),
    "pool_divisor": ("mean[(size_t)blk * dh + d] /= (double)cnt;", "mean[(size_t)blk * dh + d] /= (double)bs;"),
    "pool_unrotated": ("mean[(size_t)blk * dh + d] += xr[d];", "mean[(size_t)blk * dh + d] += xi[d];"),
    "softmax_scale": ("double isd = 1.0 / sqrt((double)dh);\n    int ntask",
                      "double isd = 1.0;\n    int ntask"),
    "ragged_keys_padded": ("for (int t = 0; t < nkeys; ++t) { s[t] = exp(s[t] - mx); den += s[t]; }",
                           "for (int t = 0; t < nkeys; ++t) { s[t] = exp(s[t] - mx); den += s[t]; } "
                           "den += (double)((64 - nkeys % 64) % 64) * exp(-mx);"),
    "qblock_pool_divisor": ("const int* cntv = which == 0 ? qcount : count;",
                            "const int* cntv = which == 0 ? count : count;"),
    "qblock_sparse_rows": ("for (int mi = 0; mi < qcount[i]; ++mi) {\n            int p = qmembers",
                           "for (int mi = 0; mi < qcount[i] && mi < bs; ++mi) {\n            int p = qmembers"),
    "qblock_backward_rows": ("for (int mi = 0; mi < qcount[i]; ++mi) {\n                int p = qmembers",
                             "for (int mi = 0; mi < qcount[i] && mi < bs; ++mi) {\n                int p = qmembers"),
    "tau_fp64_roundoff": ("const double u = ldexp(1.0, -24);", "const double u = ldexp(1.0, -53);"),
    "cube_axis_stride": ("return ((t / CUBE) * nx + x / CUBE) * ny + y / CUBE;",
                         "return ((t / CUBE) * ny + x / CUBE) * nx + y / CUBE;"),
    "cube_grid_rounding": ("int nx = (c->Hh + CUBE - 1) / CUBE, ny = (c->Ww + CUBE - 1) / CUBE;",
                           "int nx = c->Hh / CUBE + 1, ny = c->Ww / CUBE + 1;"),
    "fusion_norm": ("out[d] = (os[d] / rp + g * olr[d]) * rp;", "out[d] = (os[d] + g * olr[d]) * rp;"),
    "rmsnorm_mean": ("double inv = 1.0 / sqrt(ss / (double)dh + c->eps_lr);",
                     "double inv = 1.0 / sqrt(ss + c->eps_lr);"),
    "gate_bias_dropped": ("double logit = b;", "double logit = 0.0;"),
    "gate_sigmoid_sign": ("g[p] = 1.0 / (1.0 + exp(-logit));", "g[p] = 1.0 / (1.0 + exp(logit));"),
    "gate_last_feature": ("for (int d = 0; d < D; ++d) logit +=", "for (int d = 0; d < D - 1; ++d) logit +="),
    "gelu_scale": ("return 0.5 * x * (1.0 + erf(x / sqrt(2.0)));", "return 0.5 * x * (1.0 + erf(x / 2.0));"),
    "tanh_for_identity": ("case 1: return x;", "case 1: return tanh(x);"),
    "relu_leaky": ("case 3: return x > 0.0 ? x : 0.0;", "case 3: return x > 0.0 ? x : 0.01 * x;"),
    "activation_before_rotation_only": ("for (int a = 0; a < r; ++a) u[a] = orc_activation(c, u[a]);",
                                        "for (int a = 0; a < r; ++a) u[a] = silu(u[a]);"),
    "bwd_softmax_no_centering": ("double dsv = pr[t] * (dpr[t] - Dp) * isd;", "double dsv = pr[t] * dpr[t] * isd;"),
    "bwd_rope_not_transposed": ("out[2 * m] = x * ca + y * sa;\n        out[2 * m + 1] = -x * sa + y * ca;",
                                "out[2 * m] = x * ca - y * sa;\n        out[2 * m + 1] = x * sa + y * ca;"),
    "bwd_fusion_rms_term": ("dOs[(size_t)p * dh + d] = (double)dop[d] + dr * osp[d] / ((double)dh * rp);",
                            "dOs[(size_t)p * dh + d] = (double)dop[d];"),
    "bwd_rmsnorm_projection": ("dy[d] = (g * rp * (double)dop[d] - olr[d] * od / (double)dh) / rho;",
                               "dy[d] = g * rp * (double)dop[d] / rho;"),
    "bwd_silu_derivative": ("return sg * (1.0 + x * (1.0 - sg));", "return sg;"),
    "bwd_summary_value_grad": ("dv[head + (size_t)j * dh + d] += ft[aa] * dC[(size_t)aa * dh + d];",
                               "dv[head + (size_t)j * dh + d] += ft[aa] * dC[(size_t)aa * dh + (d + 1) % dh];"),
    "bwd_inside_activation_point": ("w[a] = orc_activation_grad(c, w[a]) * df[a];",
                                    "w[a] = orc_activation_grad(c, u[a]) * df[a];"),
    "bwd_projection_grad_input": ("dP[(size_t)a * dh + d] += du[a] * (double)x[d];",
                                  "dP[(size_t)a * dh + d] += du[a] * (double)x[(d + 1) % dh];"),
    "bwd_key_grad_operand": ("dkr[(size_t)j * dh + d] += dsv * qp[d];", "dkr[(size_t)j * dh + d] += dsv * kq[d];"),
    "bwd_gate_grad_rms": ("dg_bh[(size_t)bh * N + p] = rp * a;", "dg_bh[(size_t)bh * N + p] = a;"),
    "f32_pool_sequential": ("return pairwise_f32(x, n / 2) + pairwise_f32(x + n / 2, n - n / 2);",
                            "return x[0] + pairwise_f32(x + 1, n - 1);"),
    "f32_rotation_sign": ("yr[2 * m] = fmaf(x0, cm, -p1);", "yr[2 * m] = fmaf(x0, cm, p1);"),
    "f32_pool_divisor": ("pairwise_f32(vals, slots) / (float)cnt;", "pairwise_f32(vals, slots) / (float)slots;"),
    "f32_query_chunk_slots": ("int qslots = c->geometry == 1 ? kslots : qblock_size(c);", "int qslots = kslots;"),
    "f32_tie_order": ("return (x->j > y->j) - (x->j < y->j);", "return (x->j < y->j) - (x->j > y->j);"),
    "f32_scale_dropped": ("row[j].s = acc * scale;", "row[j].s = acc;"),
    "f32_cube_slot_order": ("x = CUBE * cx + (i / CUBE) % CUBE, y = CUBE * cy + i % CUBE;",
                            "x = CUBE * cx + i % CUBE, y = CUBE * cy + (i / CUBE) % CUBE;"),
    "out_proj_concat_order": ("cat[h * dh + d] = O[", "cat[d * H + h] = O["),
    "out_proj_transposed_weight": ("y += cat[k] * (double)W[(size_t)f * K + k];",
                                   "y += cat[k] * (double)W[((size_t)k * d_model + f) % ((size_t)K * d_model)];"),
    "out_proj_bias_dropped": ("double y = bias ? (double)bias[f] : 0.0;", "double y = 0.0;"),
    "readout_index": ("s += qt[a] * Cb[(size_t)a * dh + d];", "s += qt[a] * Cb[(size_t)d * c->r % (c->r * dh) + a];"),
}


@pytest.mark.parametrize("name", sorted(MUTATIONS))
def test_pins_catch_planted_mistake(name, tmp_path):
    old, new = MUTATIONS[name]
    src = open(SRC).read()
    assert src.count(old) == 1, f"mutation anchor for {name} not unique"
    mutated = tmp_path / "mut.c"
    mutated.write_text(src.replace(old, new))
    lib = tmp_path / "libmut.so"
    subprocess.check_call(["gcc", "-O2", "-fopenmp", "-fPIC", "-shared", "-std=c99", "-ffp-contract=off", "-o", str(lib),
                           str(mutated), "-lm"])
    env = dict(os.environ, ORACLE_LIB=str(lib), OMP_NUM_THREADS="4")
    res = subprocess.run([sys.executable, "-m", "pytest", "-x", "-q", "-p", "no:cacheprovider",
                          os.path.join(ROOT, "tests", "test_oracle_pins.py"),
                          os.path.join(ROOT, "tests", "test_oracle_backward_pins.py")],
                         cwd=ROOT, env=env, capture_output=True, text=True, timeout=600)
    assert res.returncode != 0, f"mutation {name} survived the pins:\n{res.stdout[-2000:]}"
