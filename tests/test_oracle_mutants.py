"""The oracle's pins must catch plausible mistakes.  Each case plants one
mistake in a copy of the oracle's C source (on the CPU, in a temporary
directory), builds it, and runs the pin suite against it: the suite must
fail.  The committed oracle is never modified."""
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRC = os.path.join(ROOT, "oracle", "eqb_oracle.c")

MUTANTS = {
    "cutoff_is_Kth_not_K+1th": ("tau[i] = buf[K].s;", "tau[i] = buf[K - 1].s;"),
    "ties_to_higher_index": ("return (a->e < b->e) ? -1 : (a->e > b->e) ? 1 : 0;",
                             "return (a->e > b->e) ? -1 : (a->e < b->e) ? 1 : 0;"),
    "margin_sign_flipped": ("float d = tau[t] - bf16_bits_to_f32(z[t * E + e]);",
                            "float d = bf16_bits_to_f32(z[t * E + e]) - tau[t];"),
    "quantile_rank_off_by_one": ("uint16_t q = m[r - 1];", "uint16_t q = m[r < T ? r : r - 1];"),
    "rank_floor_not_ceil": ("return (num + E - 1) / E;", "return num / E;"),
    "centering_sign": ("b_next[e] = (float)((double)bf16_bits_to_f32(qhat[e]) - mean);",
                       "b_next[e] = (float)((double)bf16_bits_to_f32(qhat[e]) + mean);"),
    "lei_norm_inverted": ("sigma = (xi == 0.0) ? 1.0 : tanh(xi) / xi;",
                          "sigma = (xi == 0.0) ? 1.0 : xi / tanh(xi);"),
    "lei_target_drops_K": ("double fbar = (double)K * (double)n / (double)E;",
                           "double fbar = (double)n / (double)E;"),
    "bf16_truncates": ("u += 0x7fffu + lsb;", "u += 0u * lsb;"),
    "kappa_negative_wrong": ("if (x & 0x8000u) return (uint16_t)(~x & 0xffffu);",
                             "if (x & 0x8000u) return (uint16_t)(x & 0x7fffu);"),
    "rho_off_by_one": ("rho[e] = (int32_t)(r - below);", "rho[e] = (int32_t)(r - below + 1);"),
    "loads_ignore_microbatch": ("loads[(int64_t)l * E + buf[k].e] += 1;", "loads[buf[k].e] += 1;"),
    "score_drops_bias": ("buf[e].s = zf + b[e];", "buf[e].s = zf;"),
    "maxvio_local_counts_empty": ("*local = sum / (double)count;", "*local = sum / (double)M;"),
    "maxvio_drops_K": ("const double fbar_l = (double)K * (double)n / (double)E;",
                       "const double fbar_l = (double)n / (double)E;"),
    "maxvio_global_is_max_local": ("  *global = g;", "  *global = sum > g ? sum : g;"),
    "gshard_drops_mean": ("g_out[t * E + j] = (float)((double)g[t * E + j] + scale * (R[j] - m));",
                          "g_out[t * E + j] = (float)((double)g[t * E + j] + scale * R[j]);"),
    "gshard_batch_is_step": ("const double scale = (double)alpha / ((double)n * d);",
                             "const double scale = (double)alpha / ((double)T * d);"),
    "gshard_drops_score_sum": ("for (int32_t e = 0; e < E; ++e) m += (s[e] / d) * R[e];",
                               "for (int32_t e = 0; e < E; ++e) m += s[e] * R[e];"),
    "lei_not_all_experts": ("for (int32_t e = 0; e < E; ++e)\n          g_out[t * E + e] = (float)((double)g[t * E + e] + a[e]);",
                            "for (int32_t e = 0; e < E; ++e)\n          g_out[t * E + e] = (loads[(int64_t)l * E + e] > 0) ? (float)((double)g[t * E + e] + a[e]) : g[t * E + e];"),
}


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_pins_catch_planted_mistake(name, tmp_path):
    old, new = MUTANTS[name]
    src = open(SRC).read()
    assert src.count(old) == 1, f"mutation site for {name} not found exactly once"
    mutant = tmp_path / "mutant.c"
    mutant.write_text(src.replace(old, new))
    lib = tmp_path / "libmutant.so"
    subprocess.run(["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-ffp-contract=off",
                    "-o", str(lib), str(mutant), "-lm"], check=True)
    env = dict(os.environ, EQB_ORACLE_LIB=str(lib))
    r = subprocess.run([sys.executable, "-m", "pytest", "-x", "-q", "-p", "no:cacheprovider",
                        os.path.join(ROOT, "tests", "test_oracle_pins.py")],
                       env=env, cwd=ROOT, capture_output=True, text=True, timeout=600)
    assert r.returncode != 0, f"planted mistake {name} was not caught:\n{r.stdout[-2000:]}"
