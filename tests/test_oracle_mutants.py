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
    ("sde_G_sign", "for (size_t i = 0; i < (size_t)d * dv; ++i) oD[i] -= G[i];",
     "for (size_t i = 0; i < (size_t)d * dv; ++i) oD[i] += G[i];", 0),
    ("sde_e_uses_m_only", "mat_vec(S, m, d, d, oe);", "memcpy(oe, m, sizeof(double) * d);", 0),
    ("ahla_E_uses_exclusive_P", "rowvec_mat(qt, P, d, dv, r);       /* r = q_t^T P_t  */",
     "rowvec_mat(qt, P, d, dv, r); for (int c = 0; c < dv; ++c) r[c] -= dot(qt, kt, d) * vt[c];", 0),
    ("ahla_n_dropped_self_term", "const double s = dot(qt, m, d);    /* s = q_t^T m_t  */",
     "const double s = dot(qt, m, d) - dot(qt, kt, d);", 0),
    ("ahla_combine_cross_swapped", "mat_mul(B + oR, A + oP, d, d, dv, RP);   /* R_B P_A */",
     "mat_mul(A + oR, B + oP, d, d, dv, RP);", 0),
    ("ahla_combine_drop_Rm", "for (int i = 0; i < d; ++i) out[on + i] += Rm[i];",
     "for (int i = 0; i < d; ++i) out[on + i] += 0.0 * Rm[i];", 0),
    ("bwd_drop_G_adjoint_on_C", "for (int c = 0; c < dv; ++c) dC[(size_t)r * dv + c] += kt[r] * kdG[c];",
     "for (int c = 0; c < dv; ++c) dC[(size_t)r * dv + c] += 0.0 * kdG[c];", 0),
    ("bwd_drop_Cprev_term", "dkt[r] += s1 + s2 + dh[r] * kmp + mp[r] * kdh;", "dkt[r] += s1 + dh[r] * kmp + mp[r] * kdh;",
     0),
    ("bwd_gden_sign", "gden = -go / (den + a->eps);", "gden = go / (den + a->eps);", 0),
    ("bwd_S_adjoint_not_symmetrised", "s += (dS[(size_t)r * d + c] + dS[(size_t)c * d + r]) * kt[c];",
     "s += 2.0 * dS[(size_t)r * d + c] * kt[c];", 0),
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
