"""Plant plausible mistakes in a copy of the oracle; each must fail at least one pin.

This checks that the pins in ``pins.py`` would notice a dropped term, a wrong
sign, a wrong index or a reversed tie-break anywhere in the oracle. Mutants are
compiled from a patched copy of ``oracle/rps_oracle.c`` in a temporary folder,
on the CPU only.
"""
import pytest

import pins
from oracle.build import SOURCE, build_oracle
from oracle.oracle import Oracle

# (name, original text, replacement). The original must occur exactly once.
MUTANTS = [
    ("entropy sign", "if (p > 0.0) h -= p * (z - l);", "if (p > 0.0) h += p * (z - l);"),
    ("entropy drops lse", "if (p > 0.0) h -= p * (z - l);", "if (p > 0.0) h -= p * (z - m);"),
    ("lse drops the shift", "const double l = m + log(sum);", "const double l = log(sum);"),
    ("pmax sign", "pmax[n] = exp(m - l);", "pmax[n] = exp(l - m);"),
    ("argmax keeps last tie", "if (z > m) { m = z; am = v; }", "if (z >= m) { m = z; am = v; }"),
    ("rank ties reversed", "if (a->v < b->v) return -1;\n    if (a->v > b->v) return 1;",
     "if (a->v > b->v) return -1;\n    if (a->v < b->v) return 1;"),
    ("rank by lower logit", "if (a->z > b->z) return -1;\n    if (a->z < b->z) return 1;",
     "if (a->z < b->z) return -1;\n    if (a->z > b->z) return 1;"),
    ("mu drops the first token", "mass += p;", "if (t > 0) mass += p;"),
    ("truncated entropy vs max", "if (p > 0.0) ht -= p * (order[t].z - l);",
     "if (p > 0.0) ht -= p * (order[t].z - m);"),
    ("bf16 decode shift", "(uint32_t)((const uint16_t *)row)[v] << 16", "(uint32_t)((const uint16_t *)row)[v] << 15"),
    ("commit threshold strict", "in_S[k] = pmax[base + k] >= tau;", "in_S[k] = pmax[base + k] > tau;"),
    ("fallback takes min", "if (a > b || (a == b && mask_pos[base + k] < mask_pos[base + best])) best = k;",
     "if (a < b || (a == b && mask_pos[base + k] < mask_pos[base + best])) best = k;"),
    ("fallback tie to higher", "if (a > b || (a == b && mask_pos[base + k] < mask_pos[base + best])) best = k;",
     "if (a > b || (a == b && mask_pos[base + k] > mask_pos[base + best])) best = k;"),
    ("feasibility strict", "if (!(mu[base + k] >= tau_pivot)) continue;",
     "if (!(mu[base + k] > tau_pivot)) continue;"),
    ("pivot by min truncated entropy",
     "if (best < 0 || v > bv || (v == bv && rem_pos[base + i] < rem_pos[base + best])) {",
     "if (best < 0 || v < bv || (v == bv && rem_pos[base + i] < rem_pos[base + best])) {"),
    ("pivot tie to higher", "if (best < 0 || v > bv || (v == bv && rem_pos[base + i] < rem_pos[base + best])) {",
     "if (best < 0 || v > bv || (v == bv && rem_pos[base + i] > rem_pos[base + best])) {"),
    ("top-k commit takes the smallest",
     "if (best < 0 || v > bv || (v == bv && mask_pos[base + k] < mask_pos[base + best])) {",
     "if (best < 0 || v < bv || (v == bv && mask_pos[base + k] < mask_pos[base + best])) {"),
    ("lowest-entropy commit takes the highest", "pmax[base + k] : -H[base + k];", "pmax[base + k] : H[base + k];"),
    ("max-entropy pivot uses truncated entropy",
     "v = pivot_rule == PIVOT_MAX_CONFIDENCE ? pmax[base + k] : H[base + k];\n                    if (v != v) continue;",
     "v = pivot_rule == PIVOT_MAX_CONFIDENCE ? pmax[base + k] : htrunc[base + k];\n                    if (v != v) continue;"),
    ("max-confidence pivot keeps the mass constraint",
     "v = pivot_rule == PIVOT_MAX_CONFIDENCE ? pmax[base + k] : H[base + k];\n                    if (v != v) continue;",
     "v = pivot_rule == PIVOT_MAX_CONFIDENCE ? pmax[base + k] : H[base + k];\n                    if (v != v || !(mu[base + k] >= tau_pivot)) continue;"),
    ("candidate test absolute", "if (zt - zmax[base + k] >= log_r)", "if (zt >= log_r)"),
    ("candidate test strict", "if (zt - zmax[base + k] >= log_r)", "if (zt - zmax[base + k] > log_r)"),
    ("one candidate suffices", "if (nc >= 2) searchable = 1;", "if (nc >= 1) searchable = 1;"),
    ("branch rows keep the pivot", "if (rem_k[base + i] == kp) continue;\n                    rows[used * 3 + 0] = q;",
     "rows[used * 3 + 0] = q;"),
    ("mean over |M'|", "const int32_t n = rem_cnt[q] - 1;", "const int32_t n = rem_cnt[q];"),
    ("lambda sign", "score[o] = -h_bar + (lambda != 0.0 ? lambda * la : 0.0);",
     "score[o] = -h_bar - (lambda != 0.0 ? lambda * la : 0.0);"),
    ("score drops entropy", "score[o] = -h_bar + (lambda != 0.0 ? lambda * la : 0.0);",
     "score[o] = (lambda != 0.0 ? lambda * la : 0.0);"),
    ("N_tau strict", "if (branch_pmax[first + i] >= tau) count++;", "if (branch_pmax[first + i] > tau) count++;"),
    ("MASK plausibility zero", "la = anchor_zmax[base + kp] - anchor_lse[base + kp];", "la = 0.0;"),
    ("MASK keeps the pivot row", "if (k == kp) continue;\n                        sum_H += anchor_H[base + k];",
     "sum_H += anchor_H[base + k];"),
    ("candidate plausibility vs max", "la = logit_at(row, dtype, tok) - anchor_lse[base + kp];",
     "la = logit_at(row, dtype, tok) - anchor_zmax[base + kp];"),
    ("ties favour the token", "if (s[c] > s[best]) best = c;", "if (s[c] >= s[best]) best = c;"),
    ("winner takes smallest gain", "gain[q * P + j] > gain[q * P + win_j] ||",
     "gain[q * P + j] < gain[q * P + win_j] ||"),
    ("mask keeps committed pivot", "if (rem_pos[base + i] == commit_pos[q]) continue;\n", ""),
]


@pytest.mark.parametrize("name,old,new", MUTANTS, ids=[m[0] for m in MUTANTS])
def test_mutant_is_caught(tmp_path, name, old, new):
    src = SOURCE.read_text()
    assert src.count(old) == 1, f"mutant '{name}': the original text must occur exactly once"
    mutated = tmp_path / "rps_oracle_mutant.c"
    mutated.write_text(src.replace(old, new))
    lib = build_oracle(out=tmp_path / "liboracle_mutant.so", src=mutated)
    o = Oracle(lib)
    for pin in pins.ALL_PINS:
        try:
            pin(o)
        except AssertionError:
            return
    pytest.fail(f"mutant '{name}' passed every pin")


# Plausible mistakes in the LM-head oracle's contraction (its statistics are the
# row-statistics oracle's, mutated above): each must fail an LM-head pin.
def _lm_mutants():
    import numpy as np
    import oracle.lmhead as lm
    orig = lm.lmhead_logits
    return {
        "negated product": lambda h, w: -orig(h, w),
        "tokens reversed": lambda h, w: orig(h, w)[:, ::-1].copy(),
        "last weight dropped": lambda h, w: (lm.bf16_to_f64(h)[:, :-1] @ lm.bf16_to_f64(w)[:, :-1].T).astype(np.float32),
        "product doubled": lambda h, w: 2 * orig(h, w),
        "first row for every row": lambda h, w: np.repeat(orig(h, w)[:1], len(h), axis=0),
    }


@pytest.mark.parametrize("name", ["negated product", "tokens reversed", "last weight dropped", "product doubled",
                                  "first row for every row"])
def test_lmhead_mutant_is_caught(oracle, monkeypatch, name):
    import oracle.lmhead as lm
    monkeypatch.setattr(lm, "lmhead_logits", _lm_mutants()[name])
    caught = False
    for pin in (p for p in pins.ALL_PINS if p.__name__.startswith("pin_lmhead")):
        try:
            pin(oracle)
        except Exception:
            caught = True
            break
    assert caught, f"no LM-head pin catches '{name}'"


# Planted mistakes in the packed-attention oracle: each must fail an attention pin.
def _attn_mutants():
    import numpy as np
    import oracle.attention as at
    keys, soft = at.allowed_keys, at.softmax_attention
    return {
        "context sees every branch": ("allowed_keys", lambda C, NB, G, s: np.arange(C + NB * G) if s == 0 else keys(C, NB, G, s)),
        "branch sees the next branch": ("allowed_keys", lambda C, NB, G, s: keys(C, NB, G, s if s in (0, NB) else s + 1)),
        "last context key dropped": ("allowed_keys", lambda C, NB, G, s: keys(C, NB, G, s)[1:]),
        "scale dropped": ("softmax_attention", lambda q, k, v, scale: soft(q, k, v, 1.0)),
        "keys for values": ("softmax_attention", lambda q, k, v, scale: soft(q, k, k, scale)),
    }


@pytest.mark.parametrize("name", ["context sees every branch", "branch sees the next branch", "last context key dropped",
                                  "scale dropped", "keys for values"])
def test_attention_mutant_is_caught(oracle, monkeypatch, name):
    import oracle.attention as at
    attr, fn = _attn_mutants()[name]
    monkeypatch.setattr(at, attr, fn)
    caught = False
    for pin in (p for p in pins.ALL_PINS if p.__name__.startswith("pin_attention")):
        try:
            pin(oracle)
        except Exception:
            caught = True
            break
    assert caught, f"no attention pin catches '{name}'"
