"""Pin strength: plant plausible mistakes in copies of the oracle (on the
CPU) and check that the independent pins of ``test_oracle_pins`` catch each
one.  The stored golden outputs are left out on purpose: they are a
regression record of the oracle itself, not an independent pin."""
from __future__ import annotations

import os

import pytest

import oracle
from tests import test_oracle_pins as pins

SRC = os.path.join(os.path.dirname(oracle.__file__), "oracle.c")

# (name, original text, planted mistake)
MUTANTS = [
    ("rope-sign", "v[j] = a * c - b * s;", "v[j] = a * c + b * s;"),
    ("rope-pairing", "double a = v[j], b = v[j + half];", "double a = v[2 * j], b = v[2 * j + 1];"),
    ("concat-order", "u[t] = load_el(embed, (int64_t)prev * d + t, bf);\n                    u[d + t] = hhat[t];",
     "u[d + t] = load_el(embed, (int64_t)prev * d + t, bf);\n                    u[t] = hhat[t];"),
    ("causal-window", "orc_attend(q + h * D, kb, vb, bf, D, pos + 1,", "orc_attend(q + h * D, kb, vb, bf, D, pos + 2,"),
    ("gqa-mapping", "int64_t g = h / group;", "int64_t g = h % Hkv;"),
    ("softmax-scale", "double scale = 1.0 / sqrt((double)D);", "double scale = 1.0 / (double)D;"),
    ("attn-residual", "w->a[i] += w->x0[i];", "w->a[i] += 0.0 * w->x0[i];"),
    ("mlp-residual", "w->y[i] += w->a[i];", "w->y[i] += w->x0[i];"),
    ("gate-up-swap", "silu(w->gu[j]) * w->gu[F + j]", "silu(w->gu[F + j]) * w->gu[j]"),
    ("decode-position", "layer_row(c, m, u, L + n + k - 2,", "layer_row(c, m, u, L + n + k - 1,"),
    ("hhat-chain", "u[d + t] = hhat[t];", "u[d + t] = w.x0[t];"),
    ("rmsnorm-mean", "double inv = 1.0 / sqrt(ss / (double)n + eps);", "double inv = 1.0 / sqrt(ss + eps);"),
    ("final-gain", "orc_rmsnorm(h, w->g_final, d, c->rms_eps, nf);", "orc_rmsnorm(h, w->g_mlp, d, c->rms_eps, nf);"),
    ("prefill-last-row", "memcpy(hhat, w.y, sizeof(double) * (size_t)d);",
     "if (k > 1 || n == 1) memcpy(hhat, w.y, sizeof(double) * (size_t)d); else if (hhat[0] == 0.0) memcpy(hhat, w.y, sizeof(double) * (size_t)d);"),
    ("argmax-tie", "return (a > b) - (a < b);", "return (a < b) - (a > b);"),
    ("accept-commit", "kv_len[b] += n_new[b];", "kv_len[b] += n_new[b] + a;"),
    ("accept-bonus", "else if (j == a) v = target[b * (K + 1) + a];", "else if (j == a) v = draft[b * K + (a < K ? a : K - 1)];"),
    ("silu-sign", "return t / (1.0 + exp(-t));", "return t / (1.0 + exp(t));"),
    ("rmsnorm-eps-outside", "double inv = 1.0 / sqrt(ss / (double)n + eps);", "double inv = 1.0 / (sqrt(ss / (double)n) + eps);"),
    ("value-split", "*v = w->qkv + (Hq + Hkv) * D;", "*v = w->qkv + Hq * D;"),
    ("cache-store-swap", "store_el(kc_b, idx, bf, k[g * D + t]);", "store_el(kc_b, idx, bf, v[g * D + t]);"),
    ("attend-with-keys", "o[t] += s[j] * load_el(vc, j * row_stride + t, bf16);",
     "o[t] += s[j] * load_el(kc, j * row_stride + t, bf16);"),
    ("key-rope-position", "orc_rope(k + g * D, (int32_t)D, pos, c->rope_theta);",
     "orc_rope(k + g * D, (int32_t)D, pos + 1, c->rope_theta);"),
    ("prefill-hidden-shift", "\n                        u[d + t] = load_el(hidden, ((int64_t)b * max_new + i) * d + t, bf);",
     "\n                        u[d + t] = i > 0 ? load_el(hidden, ((int64_t)b * max_new + i - 1) * d + t, bf) : 0.0;"),
    ("hhat-normed", "prev = tid[0];\n            if (tau > 0.0) {", "prev = tid[0];\n            memcpy(hhat, w.n1, sizeof(double) * (size_t)d);\n            if (tau > 0.0) {"),
    ("topk-order", "top_vals[r] = z[order[r]];", "top_vals[r] = z[order[c->topk - 1 - r]];"),
    # the bf16 contract: each projection operand is rounded right before its product
    ("round-n1", "round_vec(w->n1, d, ra);", "(void)0;"),
    ("round-o", "round_vec(w->o, Hq * D, ra);", "(void)0;"),
    ("round-n2", "round_vec(w->n2, d, ra);", "(void)0;"),
    ("round-m", "round_vec(w->mm, F, ra);", "(void)0;"),
    ("round-final", "round_vec(nf, d, c->round_acts);", "(void)0;"),
    ("round-decode-input", "round_vec(u, 2 * d, c->round_acts);\n                layer_row(c, m, u, L + n + k - 2,",
     "layer_row(c, m, u, L + n + k - 2,"),
]

PINS = [
    lambda: pins.test_round_matches_library_reference((0, 1, 2)),
    lambda: pins.test_round_matches_library_reference((0, 1, 1)),
    pins.test_round_without_final_norm_matches_reference,
    pins.test_bf16_contract_matches_reference,
    pins.test_prefill_equals_sequential_decode,
    pins.test_closed_form_draft_repeats_last_token,
    pins.test_closed_form_hidden_passthrough,
    pins.test_closed_form_uniform_attention,
    pins.test_accept_exhaustive_patterns,
    pins.test_greedy_acceptance_is_the_zero_temperature_rule,
    pins.test_topk_lists_are_the_sorted_logits,
]


def _caught() -> bool:
    for pin in PINS:
        try:
            pin()
        except (AssertionError, ValueError, FloatingPointError):
            return True
    return False


def _argmax_tie_caught() -> bool:
    try:
        pins.test_argmax_ties_go_to_lowest_id()
    except AssertionError:
        return True
    return False


def test_unmutated_oracle_passes_every_pin():
    assert not _caught() and not _argmax_tie_caught()


@pytest.mark.parametrize("name,orig,mut", MUTANTS, ids=[m[0] for m in MUTANTS])
def test_planted_mistake_is_caught(tmp_path, name, orig, mut):
    src = open(SRC).read()
    assert src.count(orig) == 1, f"mutation anchor for {name} not found exactly once"
    p = tmp_path / "mutant.c"
    p.write_text(src.replace(orig, mut))
    # a unique, undeleted file per mutant: dlopen matches already-loaded
    # libraries by (device, inode), and a deleted file's inode can be reused
    lib = oracle.compile_source(str(p), str(tmp_path / f"libmutant_{name}.so"))
    with oracle.variant(lib):
        caught = _argmax_tie_caught() if name == "argmax-tie" else _caught()
    assert caught, f"planted mistake '{name}' was not caught by any pin"
