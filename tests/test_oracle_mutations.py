"""Each plausible mistake planted in a copy of the oracle fails at least one
pin.  The copies are compiled with gcc into a temporary directory; the oracle
in the repository is never modified."""
import os
import subprocess

import pytest

import oracle
from tests import oracle_pins

SRC = os.path.join(os.path.dirname(oracle.__file__), "moe_oracle.c")

# (name, original text, mutated text)
MUTATIONS = [
    ("silu_on_v1", "h[f] = a / (1.0 + exp(-a)) * b;", "h[f] = b / (1.0 + exp(-b)) * a;"),
    ("sigmoid_sign", "h[f] = a / (1.0 + exp(-a)) * b;", "h[f] = a / (1.0 + exp(a)) * b;"),
    ("no_silu", "h[f] = a / (1.0 + exp(-a)) * b;", "h[f] = a * b;"),
    ("w2_transposed", "h[f] * orc_load(w2e, wdt, (size_t)d * F + f)",
     "h[f] * orc_load(w2e, wdt, (size_t)f * D + d)"),
    ("w1_dropped_term", "for (int d = 0; d < D; ++d) {\n            a +=",
     "for (int d = 1; d < D; ++d) {\n            a +="),
    ("router_transposed", "orc_load(wr, wdt, (size_t)d * E + e)",
     "orc_load(wr, wdt, (size_t)e * D + d)"),
    ("tie_to_higher_index", "if (best < 0 || l[e] > l[best]) best = e;",
     "if (best < 0 || l[e] >= l[best]) best = e;"),
    ("no_renormalisation", "gate[(size_t)t * K + k] = p[idx[(size_t)t * K + k]] / psel;",
     "gate[(size_t)t * K + k] = p[idx[(size_t)t * K + k]];"),
    ("softmax_sign", "p[e] = exp(l[e] - m);", "p[e] = exp(m - l[e]);"),
    ("dispatch_reversed", "for (int s = 0; s < S; ++s)\n            if (idx[s] == e) {",
     "for (int s = S - 1; s >= 0; --s)\n            if (idx[s] == e) {"),
    ("offsets_not_scanned", "offsets[e + 1] = offsets[e] + counts[e];",
     "offsets[e + 1] = counts[e];"),
    ("combine_ungated", "o[d] += g[k] * y[d];\n        }\n        if (idx_out)",
     "o[d] += y[d];\n        }\n        if (idx_out)"),
    ("dense_mask_ungated", "mask[idx[k]] = g[k];", "mask[idx[k]] = 1.0;"),
    ("experts_range_upper_inclusive", "if (e < e_begin || e >= e_end) continue;",
     "if (e < e_begin || e > e_end) continue;"),
    ("experts_range_ignored", "if (e < e_begin || e >= e_end) continue;", "(void)e_begin;"),
    ("experts_share_ungated", "o[d] += g[k] * y[d];\n        }\n    }\n    free(",
     "o[d] += y[d];\n        }\n    }\n    free("),
    ("bf16_round_to_9_bits", "const double ulp = ldexp(1.0, e - 8);",
     "const double ulp = ldexp(1.0, e - 9);"),
    ("bf16_round_truncates", "out[i] = nearbyint(v / ulp) * ulp;",
     "out[i] = trunc(v / ulp) * ulp;"),
    ("rmsnorm_no_sqrt", "const double s = 1.0 / sqrt(ss / D + eps);",
     "const double s = 1.0 / (ss / D + eps);"),
    ("rmsnorm_sum_not_mean", "const double s = 1.0 / sqrt(ss / D + eps);",
     "const double s = 1.0 / sqrt(ss + eps);"),
    ("rope_turns_backwards", "r[i] = a * c - b * s;\n                r[i + half] = b * c + a * s;",
     "r[i] = a * c + b * s;\n                r[i + half] = b * c - a * s;"),
    ("rope_frequency", "pow(base, -2.0 * i / dh)", "pow(base, -1.0 * i / dh)"),
    ("rope_adjacent_pairs", "const double a = r[i], b = r[i + half];",
     "const double a = r[2 * (i % (half / 2 + 1))], b = r[i + half];"),
    ("attention_unscaled", "sc[j] = dot * scale;", "sc[j] = dot;"),
    ("attention_misses_own_position", "n = pos[t] + 1;", "n = pos[t] + (pos[t] == 0);"),
    ("gqa_interleaved", "g = h / group,", "g = h % Hkv,"),
    ("wo_transposed", "orc_load(wo, wdt, (size_t)d * nq + c)", "orc_load(wo, wdt, (size_t)c * D + d)"),
    ("keys_not_rotated", "    orc_rope(T, Hkv, dh, base, pos, k);\n", "\n"),
    ("values_from_keys", "qkv + (size_t)t * nr + nq + nkv, sizeof(double) * nkv);",
     "qkv + (size_t)t * nr + nq, sizeof(double) * nkv);"),
    ("cache_not_rounded", "        orc_round_bf16((size_t)T * nkv, v, v);\n", "\n"),
    ("queries_not_rounded", "        orc_round_bf16((size_t)T * nq, q, q);\n", "\n"),
]


@pytest.mark.parametrize("name,old,new", MUTATIONS, ids=[m[0] for m in MUTATIONS])
def test_mutation_is_caught(tmp_path, name, old, new):
    src = open(SRC).read()
    assert src.count(old) == 1, f"mutation site for {name} not unique"
    mutated = tmp_path / "moe_oracle_mut.c"
    mutated.write_text(src.replace(old, new))
    so = tmp_path / f"libmut_{name}.so"
    subprocess.check_call(["gcc", "-O2", "-fopenmp", "-fPIC", "-shared", "-std=c11",
                           "-o", str(so), str(mutated), "-lm"])
    orc = oracle.OracleLib(str(so))
    failed = []
    for pin in oracle_pins.ALL_PINS:
        try:
            pin(orc)
        except AssertionError:
            failed.append(pin.__name__)
    assert failed, f"mutation {name} passed every pin"
