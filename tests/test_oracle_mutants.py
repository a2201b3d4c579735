"""The oracle's pins must catch plausible mistakes (planted in a copy, on the CPU).

Each case applies one source edit to a private copy of the oracle -- a dropped
term, a wrong sign or index, an inverted ratio -- and requires that at least one
pin of ``oracle_pins`` fails on the mutant.  The real oracle is untouched.
"""
import inspect
import types

import pytest

import oracle.spade_oracle as O
from tests import oracle_pins as pins

MUTANTS = {
    "dropped_score_scale": ("s = K @ qv / math.sqrt(qv.shape[-1])", "s = K @ qv"),
    "mask_off_by_one": ("last = int(ctx_lens[b]) + int(row_pos[r])",
                        "last = int(ctx_lens[b]) + int(row_pos[r]) - 1"),
    "gqa_modulo": ("kvh = h // G", "kvh = h % Hkv"),
    "inverted_ratio": ("ratio = p[d] / qd", "ratio = qd / p[d]"),
    "non_strict_accept": ("ok = u < ratio", "ok = u <= ratio"),
    "residual_sign": ("r = np.maximum(0.0, _f64(p) - _f64(q))",
                      "r = np.maximum(0.0, _f64(q) - _f64(p))"),
    "sample_wrong_row": ("lr = _f64(logits[r0 + a])", "lr = _f64(logits[r0 + k])"),
    "bonus_from_residual": ("r, Z, fb = p, p.sum(), False",
                            "r, Z, fb = residual_distribution(p, draft_probs[d0 + a - 1])"),
    "cdf_non_strict": ("hit = np.nonzero(c > T)[0]", "hit = np.nonzero(c >= T)[0]"),
    "cdf_descending": ("c = np.cumsum(r)", "c = np.cumsum(r[::-1])[::-1]"),
    "commit_keeps_correction_slot": ("lo = int(ctx[b]) + a + 1", "lo = int(ctx[b]) + a + 2"),
    "temperature_2": ("e = np.exp(l - l.max(axis=-1, keepdims=True))",
                      "e = np.exp(2.0 * (l - l.max(axis=-1, keepdims=True)))"),
    "greedy_uses_draft_row_shift": ("l = _f64(logits[r0 + i])", "l = _f64(logits[r0 + i + 1])"),
    "uniform_of_wrong_row": ("u = float(uniforms[r0 + i])", "u = float(uniforms[r0 + k])"),
    # Mistakes in the margins and flags that decide which GPU mismatches are excused.
    "top2_margin_always_inf": ("return float(top[1] - top[0])", "return float('inf')"),
    "top2_margin_always_zero": ("return float(top[1] - top[0])", "return 0.0"),
    "sample_margin_over_Z": ("margin = min(T - lo, c[x] - T) / r[x] if r[x] > 0 else 0.0",
                             "margin = min(T - lo, c[x] - T) / Z if r[x] > 0 else 0.0"),
    "sample_margin_always_zero": ("margin = min(T - lo, c[x] - T) / r[x] if r[x] > 0 else 0.0",
                                  "margin = 0.0"),
    "sample_spread_dropped": ("if m < margin or m * r[x] < spread:", "if m < margin:"),
    "sample_spread_over_every_token": ("terms = np.where(r > 0, p * logit_rel_err * np.maximum(1.0, np.abs(lt)), 0.0)",
                                       "terms = logit_rel_err * np.maximum(1.0, np.abs(lt))"),
    "sample_spread_without_magnitude": ("terms = np.where(r > 0, p * logit_rel_err * np.maximum(1.0, np.abs(lt)), 0.0)",
                                        "terms = np.where(r > 0, p * logit_rel_err, 0.0)"),
    "flag_every_sequence": ("flag_dec = np.zeros(B, dtype=bool)", "flag_dec = np.ones(B, dtype=bool)"),
    "flag_every_sample": ("flag_smp = np.zeros(B, dtype=bool)", "flag_smp = np.ones(B, dtype=bool)"),
    "greedy_draft_rows_never_flag": ("                if _top2_margin(l) < margin:",
                                     "                if _top2_margin(l) < 0.0:"),
    "stochastic_never_flags": ("if abs(u - ratio) < margin:", "if abs(u - ratio) < 0.0:"),
    "flag_rows_after_rejection": ("            if not ok:\n                break",
                                  "            if not ok:\n                flag_dec[b] |= any(abs(float(uniforms[r0 + j]) - 0.5) "
                                  "< margin for j in range(i + 1, k))\n                break"),
    # Rotary embedding and the QKV projection of the verify block.
    "rope_interleaved_pairs": ("a, b = x[..., :h], x[..., h:]", "a, b = x[..., 0::2], x[..., 1::2]"),
    "rope_clockwise": ("return np.concatenate([a * c - b * s, b * c + a * s], axis=-1)",
                       "return np.concatenate([a * c + b * s, b * c - a * s], axis=-1)"),
    "rope_exponent_j_over_D": ("return float(theta) ** (-2.0 * np.arange(D // 2) / D)",
                               "return float(theta) ** (-1.0 * np.arange(D // 2) / D)"),
    "rope_position_off_by_one": ("pos[int(cu_q[b]) + i] = int(ctx_lens[b]) + i",
                                 "pos[int(cu_q[b]) + i] = int(ctx_lens[b]) + i + 1"),
    "qkv_split_k_before_q": ("q = y[:, :Hq * D].reshape(R, Hq, D)", "q = y[:, Hkv * D:(Hq + Hkv) * D].reshape(R, Hq, D)"),
    "values_rotated": ("return rope(q, pos[:, None], theta), rope(k, pos[:, None], theta), v",
                       "return rope(q, pos[:, None], theta), rope(k, pos[:, None], theta), rope(v, pos[:, None], theta)"),
    "keys_not_rotated": ("return rope(q, pos[:, None], theta), rope(k, pos[:, None], theta), v",
                         "return rope(q, pos[:, None], theta), k, v"),
    "kv_write_wrong_slot": ("kc[seq[r], :, pos[r]] = k[r]", "kc[seq[r], :, pos[r] - 1] = k[r]"),
    # Temperature of p.
    "temperature_multiplies": ("nucleus(softmax(l_row / t_b), tp_b)", "nucleus(softmax(l_row * t_b), tp_b)"),
    "temperature_ignored": ("nucleus(softmax(l_row / t_b), tp_b)", "nucleus(softmax(l_row), tp_b)"),
    # Top-p truncation.
    "nucleus_ascending": ("order = np.argsort(-p, kind=\"stable\")", "order = np.argsort(p, kind=\"stable\")"),
    "nucleus_strict_reach": ("j = int(np.nonzero(c >= top_p)[0][0])", "j = int(np.nonzero(c > top_p)[0][0])"),
    "nucleus_not_renormalised": ("    pt = pt / pt.sum()\n", ""),
    "nucleus_drops_ties": ("keep = p >= tau", "keep = p > tau"),
    # Paged cache addressing.
    "paged_row_from_page_index": ("return int(block_table[b][s // page]), s % page",
                                  "return int(block_table[b][s // page]), s // page"),
    "paged_table_transposed": ("return int(block_table[b][s // page]), s % page",
                               "return int(block_table[s // page][b]), s % page"),
    "paged_commit_off_by_one": ("        lo = int(ctx[b]) + int(accepted_len[b]) + 1\n        for s in range(lo,",
                                "        lo = int(ctx[b]) + int(accepted_len[b]) + 1\n        for s in range(lo + 1,"),
}


def _mutant(old, new):
    src = inspect.getsource(O)
    assert src.count(old) == 1, old
    mod = types.ModuleType("spade_oracle_mutant")
    exec(compile(src.replace(old, new), "<mutant>", "exec"), mod.__dict__)
    return mod


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_pins_catch_mutant(name):
    mod = _mutant(*MUTANTS[name])
    caught = []
    for check in pins.ALL_CHECKS:
        try:
            check(mod)
        except Exception as e:  # AssertionError or a crash both count as caught
            caught.append((check.__name__, type(e).__name__))
            break
    assert caught, f"no pin catches mutant {name}"
