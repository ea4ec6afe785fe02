"""The oracle's pins catch plausible mistakes planted in the oracle itself.

Each case copies the oracle package to a temporary directory, changes one
expression in its source (the C attention kernel, core.py or dit.py: a
transposed operand, a dropped term, a wrong sign, an off-by-one range, a
strict instead of a non-strict comparison ...), imports the copy under a
fresh name, points the pin modules at it and requires that at least one of
the pins named for that case fails with an AssertionError. A control run of
the unchanged copy passes every pin used here, so a failure is the planted
mistake's doing. Everything runs on the CPU; the C mutants are compiled with
gcc into the temporary copy.
"""
import importlib.util
import itertools
import os
import shutil
import sys

import pytest

import test_oracle_dit_pins as dit_pins
import test_oracle_pins as pins

ORACLE_DIR = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "oracle")
_count = itertools.count()

# (id, file, old, new, pins that must notice); a pin is (module, name, args).
P, DP = pins, dit_pins
MUTATIONS = [
    # attention by its definition (attn_oracle.c)
    ("logits_from_v", "attn_oracle.c", "dot += qi[c] * kh[j * J->d + c]", "dot += qi[c] * vh[j * J->d + c]",
     [(P, "test_attention_brute_force_tiny", (False,)), (P, "test_attention_matches_library_softmax", ())]),
    ("output_from_k", "attn_oracle.c", "oi[c] += p * vh[j * J->d + c]", "oi[c] += p * kh[j * J->d + c]",
     [(P, "test_attention_matches_library_softmax", ()), (P, "test_rows_sum_to_one", ())]),
    ("softmax_sign", "attn_oracle.c", "exp(s[j] - smax)", "exp(smax - s[j])",
     [(P, "test_attention_matches_library_softmax", ())]),
    ("scale_dropped", "attn_oracle.c", "double sj = J->scale * dot;", "double sj = dot;",
     [(P, "test_attention_brute_force_tiny", (False,)), (P, "test_attention_matches_library_softmax", ())]),
    ("bias_on_every_row", "attn_oracle.c", "if (biased && j >= J->r0", "if (J->bias && j >= J->r0",
     [(P, "test_attention_brute_force_tiny", (True,)), (P, "test_bias_closed_form_mass", ())]),
    ("bias_range_one_past", "attn_oracle.c", "j < J->r1) sj += J->bias[h]", "j <= J->r1) sj += J->bias[h]",
     [(P, "test_attention_brute_force_tiny", (True,)), (P, "test_bias_closed_form_mass", ())]),
    ("mass_range_skips_first", "attn_oracle.c", "if (j >= J->r0 && j < J->r1) m += p;",
     "if (j > J->r0 && j < J->r1) m += p;",
     [(P, "test_equal_logits_give_mean_value_and_share_mass", ()),
      (P, "test_reference_and_complement_mass_partition", ())]),
    ("normaliser_drops_last_key", "attn_oracle.c", "for (int64_t j = 0; j < J->nk; ++j) { s[j] = exp",
     "for (int64_t j = 0; j < J->nk - 1; ++j) { s[j] = exp",
     [(P, "test_rows_sum_to_one", ()), (P, "test_attention_matches_library_softmax", ())]),
    ("query_layout_transposed", "attn_oracle.c", "J->q + (h * J->nq + i) * J->d", "J->q + (h + i * J->H) * J->d",
     [(P, "test_attention_brute_force_tiny", (False,)), (P, "test_attention_matches_library_softmax", ())]),
    # Eq. 1 (core.py)
    ("q_change_no_sqrt", "core.py", "den = np.sqrt(np.sum(qp ** 2, axis=(-2, -1))) + eps",
     "den = np.sum(qp ** 2, axis=(-2, -1)) + eps",
     [(P, "test_q_change_closed_forms", ()), (P, "test_q_change_brute_force", ())]),
    ("q_change_normalised_by_current", "core.py", "den = np.sqrt(np.sum(qp ** 2", "den = np.sqrt(np.sum(qc ** 2",
     [(P, "test_q_change_closed_forms", ()), (P, "test_q_change_brute_force", ())]),
    ("q_change_eps_inside_sqrt", "core.py", "den = np.sqrt(np.sum(qp ** 2, axis=(-2, -1))) + eps",
     "den = np.sqrt(np.sum(qp ** 2, axis=(-2, -1)) + eps)",
     [(P, "test_q_change_brute_force", ())]),
    ("bf16_shift", "core.py", "<< np.uint32(16)", "<< np.uint32(15)",
     [(P, "test_bf16_widening_known_patterns", ())]),
    # Eqs. 5-6, the exposure summaries (core.py)
    ("eq5_drops_last_head", "core.py", "for h in range(M.shape[-1]):", "for h in range(M.shape[-1] - 1):",
     [(P, "test_head_mean_exposure_eq5", ())]),
    ("eq6_divides_by_T", "core.py", "return 100.0 * total / (T - 1)", "return 100.0 * total / T",
     [(P, "test_adjacent_ref_mass_change_eq6", ())]),
    ("eq6_signed_change", "core.py", "total = total + np.abs(Mbar[t] - Mbar[t - 1])",
     "total = total + (Mbar[t] - Mbar[t - 1])",
     [(P, "test_adjacent_ref_mass_change_eq6", ())]),
    ("eq6_fraction_not_points", "core.py", "return 100.0 * total / (T - 1)", "return total / (T - 1)",
     [(P, "test_adjacent_ref_mass_change_eq6", ())]),
    # gate, Eqs. 12-13 and the bounded-age refresh (core.py)
    ("gate_mean_then_product", "core.py",
     "g = [float(D[s][h]) * float(M_prev[s][h]) for h in range(len(D[s]))]",
     "g = [float(np.mean(D[s])) * float(np.mean(M_prev[s])) for h in range(len(D[s]))]",
     [(P, "test_gate_head_mean_of_products", ())]),
    ("gate_strict_threshold", "core.py", "cross = gbar >= self.theta", "cross = gbar > self.theta",
     [(P, "test_gate_first_crossing_table", ()), (P, "test_gate_head_mean_of_products", ())]),
    ("gate_age_strict", "core.py", "elif t - self.a_full >= self.delta_max:", "elif t - self.a_full > self.delta_max:",
     [(P, "test_gate_bounded_age_refresh", ())]),
    ("gate_no_latch", "core.py", "self.reactivated[s] = True", "self.reactivated[s] = False",
     [(P, "test_gate_first_crossing_table", ()), (P, "test_gate_monotone_suffix_invariant", ())]),
    # Algorithm 1's cache semantics (core.py)
    ("boundary_reads_fresh_reference", "core.py", "if mode == REUSE or mode == BOUNDARY:", "if mode == REUSE:",
     [(P, "test_boundary_uses_cached_reference_kv", ())]),
    ("cache_stamp_off_by_one", "core.py", "a_b[b][s] = t\n", "a_b[b][s] = t - 1\n",
     [(P, "test_zero_threshold_puts_boundary_at_block_zero", ())]),
    # DiT block (dit.py)
    ("round_bf16_truncates", "dit.py", "np.rint(m * 256.0)", "np.floor(m * 256.0)",
     [(DP, "test_round_bf16_ties_and_known_values", ()), (DP, "test_round_bf16_matches_torch_on_fp32_values", ())]),
    ("adaln_scale_without_one", "dit.py", "* (1.0 + np.asarray(scale, np.float64))", "* (np.asarray(scale, np.float64))",
     [(DP, "test_layer_norm_modulate_closed_forms", ())]),
    ("rope_rotation_sign", "dit.py", "out[..., 0::2] = x0 * c - x1 * s", "out[..., 0::2] = x0 * c + x1 * s",
     [(DP, "test_rope_rotation_properties", ()), (DP, "test_rope_scores_depend_on_relative_position_only", ())]),
    ("gelu_square_term", "dit.py", "0.044715 * x ** 3", "0.044715 * x ** 2",
     [(DP, "test_gelu_tanh_against_exact_gelu", ())]),
]


def _import_copy(tmp_path, file=None, old=None, new=None):
    name = "oracle_copy_%d" % next(_count)
    dst = tmp_path / name
    shutil.copytree(ORACLE_DIR, dst, ignore=shutil.ignore_patterns("*.so", "*.so.tmp*", "__pycache__"))
    if file is not None:
        src = (dst / file).read_text()
        assert src.count(old) == 1, "the planted expression must occur exactly once in %s: %r" % (file, old)
        (dst / file).write_text(src.replace(old, new))
    spec = importlib.util.spec_from_file_location(name, dst / "__init__.py", submodule_search_locations=[str(dst)])
    mod = importlib.util.module_from_spec(spec)
    sys.modules[name] = mod
    spec.loader.exec_module(mod)
    return mod


def _point_pins_at(monkeypatch, mod):
    monkeypatch.setattr(pins, "oracle", mod)
    monkeypatch.setattr(dit_pins, "oracle", mod)
    monkeypatch.setattr(dit_pins, "dit", sys.modules[mod.__name__ + ".dit"])
    for n in ("REUSE", "BOUNDARY", "COMPUTE", "FULL"):
        monkeypatch.setattr(pins, n, getattr(mod, n))
        monkeypatch.setattr(dit_pins, n, getattr(mod, n))


def _fails(module, name, args):
    try:
        getattr(module, name)(*args)
    except AssertionError:
        return True
    return False


def test_unchanged_copy_passes_every_pin_used(tmp_path, monkeypatch):
    mod = _import_copy(tmp_path)
    importlib.import_module(mod.__name__ + ".dit")
    _point_pins_at(monkeypatch, mod)
    used = {(m.__name__, n, a) for *_, cases in MUTATIONS for (m, n, a) in cases}
    for mname, n, a in sorted(used):
        assert not _fails(sys.modules[mname], n, a), "%s%r fails on the unchanged oracle" % (n, a)


@pytest.mark.parametrize("case", MUTATIONS, ids=[m[0] for m in MUTATIONS])
def test_planted_mistake_is_caught(tmp_path, monkeypatch, case):
    _, file, old, new, cases = case
    mod = _import_copy(tmp_path, file, old, new)
    importlib.import_module(mod.__name__ + ".dit")
    _point_pins_at(monkeypatch, mod)
    caught = [n for (m, n, a) in cases if _fails(m, n, a)]
    assert caught, "no pin noticed %s: %r -> %r" % (file, old, new)
