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


@pytest.mark.parametrize("name", sorted(MUTATIONS))
def test_planted_mistake_is_caught(name, tmp_path):
    before, after = MUTATIONS[name]
    src = open(os.path.join(ROOT, "oracle", "mot_oracle.c")).read()
    assert src.count(before) == 1, "mutation anchor not found: the oracle source changed"
    dst = tmp_path / "oracle"
    shutil.copytree(os.path.join(ROOT, "oracle"), dst,
                    ignore=shutil.ignore_patterns("*.so", "*.tmp", "__pycache__"))
    (dst / "mot_oracle.c").write_text(src.replace(before, after))
    env = dict(os.environ, PYTHONPATH=f"{tmp_path}{os.pathsep}{ROOT}")
    r = subprocess.run([sys.executable, "-m", "pytest", "-q", "-x", "-p", "no:cacheprovider",
                        "--rootdir", str(tmp_path), PINS], cwd=tmp_path, env=env,
                       capture_output=True, text=True, timeout=300)
    assert r.returncode != 0, f"pins did not catch '{name}':\n{r.stdout[-2000:]}"
    assert "failed" in r.stdout
