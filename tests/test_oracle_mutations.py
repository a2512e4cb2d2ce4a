"""The oracle's pins are strong enough to catch plausible mistakes (CPU only).

Each case plants one mistake in a private copy of the C oracle (a transposed operand, a
dropped term, a wrong index, a wrong sign ...), builds it in a temporary directory, and
checks that at least one pin from ``test_oracle.py``'s families fails against it. The
committed oracle is never modified.
"""
from __future__ import annotations

import ctypes
import os
import subprocess

import numpy as np
import pytest

import oracle
from oracle import dense
from tests import test_oracle as pins
from tests import test_oracle_fp8 as fp8_pins
from tests import test_oracle_latent as latent_pins
from tests import test_oracle_prefill as prefill_pins
from tests._inputs import bits, default_scale, tiny

SRC = os.path.join(os.path.dirname(oracle.__file__), "keyless_oracle.c")

MUTATIONS = {
    "transposed_wr": ("W[(size_t)k * D + j]", "W[(size_t)j * D + k]"),
    "dropped_first_term": ("for (int k = 0; k < D; ++k) {\n        double qk",
                           "for (int k = 1; k < D; ++k) {\n        double qk"),
    "wrong_group_map": ("        int g = h / G;\n        double *qv",
                        "        int g = h % Hkv;\n        double *qv"),
    "row_off_by_one": ("(size_t)(t % P)) * D;", "(size_t)((t + 1) % P)) * D;"),
    "missing_scale": ("s[t - t0] = scale * dot;", "s[t - t0] = dot;"),
    "flipped_exponent": ("double e = exp(s[t - t0] - m);", "double e = exp(m - s[t - t0]);"),
    "combine_drops_l": ("double w = ml[2 * s + 1] * exp(ml[2 * s] - M);",
                        "double w = exp(ml[2 * s] - M);"),
    # prefill: the causal limit of a chunk row
    "prefill_mask_off_by_one": ("int p = seq_lens[b] - n + (r - cu_q[b]);",
                                "int p = seq_lens[b] - n + (r - cu_q[b]) - 1;"),
    "prefill_ignores_prefix": ("int p = seq_lens[b] - n + (r - cu_q[b]);",
                               "int p = r - cu_q[b];"),
    "prefill_not_causal": ("int p = seq_lens[b] - n + (r - cu_q[b]);",
                           "int p = seq_lens[b] - 1;"),
    # latent cache: the absorbed query, the output expansion, the latent group
    "latent_no_absorb": ("            qs[k] = acc;\n", "            qs[k] = qr[k];\n"),
    "latent_no_up_projection": ("            o[j] = acc;\n        }\n        free(s);\n        free(os);",
                                "            o[j] = j < r ? os[j] : 0.0;\n        }\n        free(s);\n        free(os);"),
    "latent_wrong_group": ("        int g = h / G, w = wr_per_query_head ? h : g;\n        const uint16_t *Wp",
                           "        int g = h % Hl, w = wr_per_query_head ? h : g;\n        const uint16_t *Wp"),
    # FP8 cache: the exponent bias, the tie rule, the per-row scale
    "e4m3_wrong_bias": ("v = (1.0 + (double)m / 8.0) * ldexp(1.0, e - 7);",
                        "v = (1.0 + (double)m / 8.0) * ldexp(1.0, e - 8);"),
    "e4m3_ties_away": ("pick = (lo & 1) ? lo + 1 : lo;    /* tie: even mantissa */",
                       "pick = lo + 1;"),
    "fp8_drops_scale": ("rows[(size_t)t * D + j] = (double)scales[row] * e4m3_value(codes[row * D + j]);",
                        "rows[(size_t)t * D + j] = e4m3_value(codes[row * D + j]);"),
    "prefill_wrong_row_base": ("route_row(D, q + ((size_t)r * Hq + h) * D, w_r + (size_t)w * D * D, qr);",
                               "route_row(D, q + ((size_t)(r - cu_q[b]) * Hq + h) * D, w_r + (size_t)w * D * D, qr);"),
}


def _pin_results():
    """Run a cross-section of the pins; return {name: passed}."""
    res = {}

    def run(name, fn, *a):
        try:
            fn(*a)
            res[name] = True
        except (AssertionError, ValueError):
            res[name] = False

    run("dense_gqa", pins.test_paged_oracle_equals_dense_bruteforce,
        dict(B=3, Hq=8, Hkv=2, D=64, P=16, lens=(1, 37, 100)))
    run("theorem1", pins.test_theorem1_keyless_equals_standard_attention_with_k_equal_v_wr_transposed)
    run("group_map", pins.test_group_mapping_reads_value_head_h_over_g)
    run("dominant", pins.test_dominant_score_selects_that_row)
    run("split_merge", pins.test_split_merge_identity, 33)
    run("route", pins.test_route_matches_row_times_matrix)
    run("prefill_dense", prefill_pins.test_paged_prefill_equals_dense_causal_bruteforce,
        dict(B=3, Hq=8, Hkv=2, D=64, P=16, lens=(5, 37, 100), q_lens=(5, 12, 1)))
    run("prefill_sdpa", prefill_pins.test_full_causal_prefill_equals_sdpa_with_k_equal_v_wr_transposed)
    run("latent_expand", latent_pins.test_absorbed_query_equals_expanded_values,
        dict(B=3, Hq=8, Hl=2, D=128, r=64, P=16, lens=(1, 37, 100)))
    run("latent_identity", latent_pins.test_identity_expansion_is_the_plain_keyless_decode)
    run("e4m3_torch", fp8_pins.test_every_code_decodes_like_torch_float8_e4m3fn)
    run("e4m3_encode", fp8_pins.test_encoding_matches_torch_rounding_in_range)
    run("fp8_dense", fp8_pins.test_fp8_decode_equals_dense_over_dequantized_rows)
    return res


@pytest.mark.parametrize("name", sorted(MUTATIONS))
def test_planted_mistake_is_caught(name, tmp_path, monkeypatch):
    before, after = MUTATIONS[name]
    src = open(SRC).read()
    assert src.count(before) == 1, f"mutation anchor for {name} not unique"
    mutated = tmp_path / "mutated.c"
    mutated.write_text(src.replace(before, after))
    so = tmp_path / f"libmut_{name}.so"
    subprocess.run(["gcc", "-O1", "-fPIC", "-shared", "-std=c11", str(mutated), "-o", str(so),
                    "-lm"], check=True, capture_output=True)
    lib = ctypes.CDLL(str(so))
    real = oracle._load()
    for f in ("ko_route", "ko_decode", "ko_standard_decode", "ko_attention_weights",
              "ko_decode_partial", "ko_combine", "ko_append", "ko_prefill", "ko_append_chunk",
              "ko_latent_decode", "ko_quantize_rows", "ko_append_fp8", "ko_decode_fp8",
              "ko_e4m3_from_f32", "ko_e4m3_value"):
        getattr(lib, f).argtypes = getattr(real, f).argtypes
        getattr(lib, f).restype = getattr(real, f).restype
    monkeypatch.setattr(oracle, "_lib", lib)
    res = _pin_results()
    assert not all(res.values()), f"mutation {name} survived every pin: {res}"


def test_unmutated_oracle_passes_the_same_pins():
    assert all(_pin_results().values())
