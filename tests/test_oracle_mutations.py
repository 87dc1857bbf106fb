"""Each plausible mistake, planted in a scratch copy of the oracle's C source,
must make the pin tests fail. This checks that the pins constrain the oracle;
the mistakes are planted on the CPU only."""
import os
import shutil
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
PINS = os.path.join(ROOT, "tests", "test_oracle_pins.py")
BT_PINS = os.path.join(ROOT, "tests", "test_oracle_bt_pins.py")

MUTATIONS = {
    "drop_b1": ("h[j] = oracle_gelu(dot(row, z, Ds) + ld(w, dt, o_b1 + j));",
                "h[j] = oracle_gelu(dot(row, z, Ds));"),
    "drop_b2": ("ym[i] = dot(row, h, H) + ld(w, dt, o_b2 + i);", "ym[i] = dot(row, h, H);"),
    "drop_bg": ("logit[m] = dot(row, z, Ds) + ld(w, dt, off_bg + m);", "logit[m] = dot(row, z, Ds);"),
    "gelu_sign": ("return 0.5 * x * (1.0 + erf(x / sqrt(2.0)));",
                  "return 0.5 * x * (1.0 - erf(x / sqrt(2.0)));"),
    "gelu_tanh_form": ("return 0.5 * x * (1.0 + erf(x / sqrt(2.0)));",
                       "return 0.5 * x * (1.0 + tanh(0.7978845608028654 * (x + 0.044715 * x * x * x)));"),
    "src_head_dim_swapped": ("const int64_t hs = c / d->d_s, i = c % d->d_s;",
                             "const int64_t hs = c % d->H_s, i = c / d->H_s;"),
    "dst_head_dim_swapped": ("const int64_t ht = c / d->d_t, i = c % d->d_t;",
                             "const int64_t ht = c % d->H_t, i = c / d->H_t;"),
    "W1_transposed": ("ld_row(w, dt, o_w1 + j * Ds, Ds, row);",
                      "for (int64_t k = 0; k < Ds; ++k) row[k] = ld(w, dt, o_w1 + k * H + j);"),
    "softmax_no_max_subtraction": ("g[m] = exp(logit[m] - mx);", "g[m] = exp(logit[m]);"),
    "topk_not_renormalised": ("g[m] = keep[m] ? g[m] / ks : 0.0;", "g[m] = keep[m] ? g[m] : 0.0;"),
    "topk_ties_to_higher_index": ("if (!keep[m] && (best < 0 || g[m] > g[best])) best = m;",
                                  "if (!keep[m] && (best < 0 || g[m] >= g[best])) best = m;"),
    "map_floor": ("out[l] = (int32_t)((2 * num + den) / (2 * den));", "out[l] = (int32_t)(num / den);"),
    "map_half_down": ("out[l] = (int32_t)((2 * num + den) / (2 * den));",
                      "out[l] = (int32_t)((2 * num + den - 1) / (2 * den));"),
    "blob_group_ignores_X": ("const char* w = (const char*)blob + (r * 2 + X) * gsz * esz;",
                             "const char* w = (const char*)blob + (r * 2) * gsz * esz;"),
    "blob_group_by_target_layer": ("const char* w = (const char*)blob + (r * 2 + X) * gsz * esz;",
                                   "const char* w = (const char*)blob + (l * 2 + X) * gsz * esz;"),
    "combine_ignores_gate": ("for (int64_t i = 0; i < Dt; ++i) y[i] += g[m] * ym[i];",
                             "for (int64_t i = 0; i < Dt; ++i) y[i] += ym[i] / E;"),
}


# Mistakes in the backbone-translator oracle (App. C.2), caught by its own pins.
BT_MUTATIONS = {
    "bt_drop_ln_in": ("ln_blob(w, dt, o_lnin, ds, x + (r * P + p) * ds, s->vec, s);",
                      "memcpy(s->vec, x + (r * P + p) * ds, sizeof(double) * (size_t)ds);"),
    "bt_h0_from_last_slot": ("memcpy(s->h, s->z, sizeof(double) * (size_t)Pd);",
                             "memcpy(s->h, s->z + (L->N - 1) * Pd, sizeof(double) * (size_t)Pd);"),
    "bt_attn_unscaled": ("sc[j] = s * scale;", "sc[j] = s;"),
    "bt_attn_one_head": ("oracle_bt_attention((int)P, (int)d, (int)L->na, s->q, s->k, s->v, s->o);",
                         "oracle_bt_attention((int)P, (int)d, 1, s->q, s->k, s->v, s->o);"),
    "bt_keys_from_state": ("ln_blob(w, dt, o_lnc, d, zr + p * d, s->nc + p * d, s);",
                           "ln_blob(w, dt, o_lnc, d, s->h + p * d, s->nc + p * d, s);"),
    "bt_no_attn_residual": ("s->ht[p * d + i] = s->h[p * d + i] + s->a[p * d + i];",
                            "s->ht[p * d + i] = s->a[p * d + i];"),
    "bt_ffn_no_gelu": ("for (int64_t j = 0; j < df; ++j) s->f[j] = oracle_gelu(s->f[j]);", ""),
    "bt_ln_out_per_row": ("ln_blob(w, dt, o_lnout, Pd, s->h, s->nF, s);",
                          "for (int64_t p = 0; p < P; ++p) "
                          "oracle_layernorm(s->h + p * d, d, NULL, NULL, s->nF + p * d);"),
    "bt_no_output_gelu": ("for (int64_t i = 0; i < L->Dt; ++i) yr[i] = oracle_gelu(yr[i]);", ""),
    "bt_gate_no_bias": ("logit[m] = sdot + bld(blob, d->dtype, gbase + E * WD + m);",
                        "logit[m] = sdot;"),
    "bt_ln_eps": ("static const double kLnEps = 1e-5;", "static const double kLnEps = 1e-3;"),
    "bt_ln_unbiased": ("  var /= (double)n;", "  var /= (double)(n - 1);"),
    "bt_window_ignores_map": ("const int64_t sl = map[bt->win_start + r];",
                              "const int64_t sl = bt->win_start + r;"),
    "bt_slots_reversed": ("for (int64_t i = 0; i < Dt; ++i) o[i] = acc[r * Dt + i];",
                          "for (int64_t i = 0; i < Dt; ++i) o[i] = acc[(N - 1 - r) * Dt + i];"),
}

# Mistakes in the replay-attention oracle (App. C.4), caught by its own pins.
REPLAY_PINS = os.path.join(ROOT, "tests", "test_oracle_replay_pins.py")
REPLAY_MUTATIONS = {
    "replay_ties_to_higher_position": ("if (best < 0 || v > bv) { best = j; bv = v; }",
                                       "if (best < 0 || v >= bv) { best = j; bv = v; }"),
    "replay_not_causal": ("  const uint16_t* row = guide + ((int64_t)b * d->N + u) * d->N;",
                          "  n = d->N;\n  const uint16_t* row = guide + ((int64_t)b * d->N + u) * d->N;"),
    "replay_previous_row": ("  const uint16_t* row = guide + ((int64_t)b * d->N + u) * d->N;",
                            "  const uint16_t* row = guide + ((int64_t)b * d->N + (u > 0 ? u - 1 : 0)) * d->N;"),
    "replay_unscaled": ("s[t] = acc * scale;", "s[t] = acc;"),
    "replay_gqa_interleaved": ("const int hk = h / (d->Hq / d->Hkv);", "const int hk = h % d->Hkv;"),
    "replay_full_layer_boundary": ("const int sparse = layer >= d->n_full;",
                                   "const int sparse = layer > d->n_full;"),
}

CASES = ([(n, "mot_oracle.c", PINS, MUTATIONS[n]) for n in sorted(MUTATIONS)] +
         [(n, "bt_oracle.c", BT_PINS, BT_MUTATIONS[n]) for n in sorted(BT_MUTATIONS)] +
         [(n, "replay_oracle.c", REPLAY_PINS, REPLAY_MUTATIONS[n])
          for n in sorted(REPLAY_MUTATIONS)])


@pytest.mark.parametrize("name,src_name,pins,change", CASES, ids=[c[0] for c in CASES])
def test_planted_mistake_is_caught(name, src_name, pins, change, tmp_path):
    before, after = change
    src = open(os.path.join(ROOT, "oracle", src_name)).read()
    assert src.count(before) == 1, "mutation anchor not found: the oracle source changed"
    dst = tmp_path / "oracle"
    shutil.copytree(os.path.join(ROOT, "oracle"), dst,
                    ignore=shutil.ignore_patterns("*.so", "*.tmp", "__pycache__"))
    (dst / src_name).write_text(src.replace(before, after))
    env = dict(os.environ, PYTHONPATH=f"{tmp_path}{os.pathsep}{ROOT}")
    r = subprocess.run([sys.executable, "-m", "pytest", "-q", "-x", "-p", "no:cacheprovider",
                        "--rootdir", str(tmp_path), pins], cwd=tmp_path, env=env,
                       capture_output=True, text=True, timeout=300)
    assert r.returncode != 0, f"pins did not catch '{name}':\n{r.stdout[-2000:]}"
    assert "failed" in r.stdout
