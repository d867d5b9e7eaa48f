"""Planted-mistake tests for the oracle's pins (CPU only).

Each case copies oracle/hla_oracle.c, plants one plausible mistake (a dropped
term, a wrong sign, a wrong time index, a swapped operand, an off-by-one in
the scan), builds the copy with gcc into a temporary directory and runs the
pins against it.  At least one pin must fail for every mutant; otherwise the
pins would not protect the oracle against that kind of mistake.  The mistakes
are planted only in temporary copies, never in the oracle itself.
"""
import os
import subprocess

import pytest

import oracle
import pins

SRC = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "oracle", "hla_oracle.c")

# (id, text in the source, replacement, which occurrence to replace)
MUTANTS = [
    ("hla2_drop_G_correction", "double num = uC[c] - (a->masked ? qG[c] : 0.0);", "double num = uC[c];", 0),
    ("hla2_G_sign", "double num = uC[c] - (a->masked ? qG[c] : 0.0);",
     "double num = uC[c] + (a->masked ? qG[c] : 0.0);", 0),
    ("hla2_G_uses_C_t", "for (int c = 0; c < dv; ++c) G[(size_t)r * dv + c] += kt[r] * kC[c];",
     "for (int c = 0; c < dv; ++c) G[(size_t)r * dv + c] += kt[r] * (kC[c] + dot(kt, qt, d) * vt[c]);", 0),
    ("hla2_h_uses_m_t", "h[r] += kt[r] * km;", "h[r] += kt[r] * (km + dot(kt, qt, d));", 0),
    ("hla2_den_sign", "den -= dot(qt, h, d);", "den += dot(qt, h, d);", 0),
    ("hla2_S_wrong_operand", " S[(size_t)r * d + c] += kt[r] * kt[c];", " S[(size_t)r * d + c] += kt[r] * qt[c];", 0),
    ("hla2_eps_dropped", "a->normalized ? num / (den + a->eps) : num;", "a->normalized ? num / den : num;", 0),
    ("combine_cross_term_swapped", "mat_mul(B + oS, A + oC, d, d, dv, SC);", "mat_mul(A + oS, B + oC, d, d, dv, SC);", 0),
    ("blelloch_operand_order", "hla2_combine_f64(r, old_left, tmp, d, dv, masked);",
     "hla2_combine_f64(old_left, r, tmp, d, dv, masked);", 0),
    ("chunk_carry_off_by_one", "const double *carry = summ + len * (size_t)(c + 1);",
     "const double *carry = summ + len * (size_t)c;", 0),
    ("hla3_G2_uses_P_t", "rowvec_mat(qt, Pp, d, dv, rowP);", "rowvec_mat(qt, P, d, dv, rowP);", 0),
    ("hla3_drop_G3", "G3[(size_t)r * dv + c] += a3[r] * vt[c];", "G3[(size_t)r * dv + c] += 0.0 * a3[r] * vt[c];", 0),
    ("hla3_eps_dropped", "a->normalized ? num / (den + a->eps) : num;", "a->normalized ? num / den : num;", 1),
    ("hla3_concat_drop_map_term", "out->F[i] = A->F[i] + B->F[i] + t1[i] + t2[i] + t3[i];",
     "out->F[i] = A->F[i] + B->F[i] + t1[i] + t3[i];", 0),
    ("hla3_map_of_wrong_segment", "seg3_apply_maps(tk, B->t0, B->t1, A->SQ, t2, e2);",
     "seg3_apply_maps(tk, A->t0, A->t1, A->SQ, t2, e2);", 0),
]


def _replace_nth(text, old, new, which):
    idx = -1
    for _ in range(which + 1):
        idx = text.find(old, idx + 1)
        assert idx >= 0, (old, which)
    return text[:idx] + new + text[idx + len(old):]


@pytest.mark.parametrize("name,old,new,which", MUTANTS, ids=[m[0] for m in MUTANTS])
def test_pins_catch_planted_mistake(name, old, new, which, tmp_path, monkeypatch):
    src = open(SRC).read()
    assert src.count(old) >= which + 1, "mutation anchor not found: " + name
    mutated = tmp_path / (name + ".c")
    mutated.write_text(_replace_nth(src, old, new, which))
    lib_path = str(tmp_path / ("lib" + name + ".so"))
    subprocess.run(["gcc", "-O2", "-std=c99", "-shared", "-fPIC", "-pthread", "-o", lib_path, str(mutated), "-lm"],
                   check=True)
    monkeypatch.setattr(oracle, "_lib", oracle.load(lib_path))
    failed = []
    for pin in pins.ALL_PINS:
        try:
            pin()
        except AssertionError:
            failed.append(pin.__name__)
            break
    assert failed, "no pin caught the planted mistake " + name
