"""Records of how ambiguous or erroneous passages of the paper are read.

Each test shows, on small fp64 inputs, that the reading the build takes is the
one that agrees with the paper's own serial definitions, and that the literal
alternative does not.
"""
import numpy as np

import oracle
from pins import rand_qkv, relerr


def _chunks(n, C):
    return [(c, min(c + C, n)) for c in range(0, n, C)]


def test_fig1c_literal_chunk_formula_misses_cross_term():
    """Fig. 1(C) writes O_t = q_t^T(S_p C_p - G_p) + [(W W^T) . L] V inside a
    chunk.  That drops q_t^T S_p C_loc,t = [(Q S_p Q^T) . L] V, the cross term
    between the carried key moment and the chunk's own query-value pairs; with
    it added the chunk form equals the serial recurrence (Eq. semidirect)."""
    n, d, dv, C = 16, 4, 3, 4
    q, k, v = rand_qkv(n, d, dv, seed=2)
    ref, st = oracle.hla2_serial(q, k, v, masked=True, return_state=True)
    Q, K, V = q[0], k[0], v[0]
    lit = np.zeros((n, dv))
    fixed = np.zeros((n, dv))
    for t0, t1 in _chunks(n, C):
        Sp = K[:t0].T @ K[:t0]
        Cp = Q[:t0].T @ V[:t0]
        Gp = sum((np.outer(K[i], K[i]) @ (Q[:i].T @ V[:i]) for i in range(t0)), np.zeros((d, dv)))
        Qc, Kc, Vc = Q[t0:t1], K[t0:t1], V[t0:t1]
        W = np.tril(Qc @ Kc.T)
        intra = np.tril(W @ W.T) @ Vc
        carry = Qc @ (Sp @ Cp - Gp)
        lit[t0:t1] = carry + intra
        fixed[t0:t1] = carry + intra + np.tril(Qc @ Sp @ Qc.T) @ Vc
    assert relerr(fixed, ref[0]) < 1e-12
    assert relerr(lit, ref[0]) > 1e-2


def test_hla3_operator_is_tied_max_triple_set():
    """Third order: Algorithm 3 / Theorem 3 compute the triples whose largest
    index occurs at least twice.  Two other natural readings of the masked
    third-order matrix differ: ((W W^T) . L) W V and ((W W^T W) . L) V."""
    n, d, dv = 7, 3, 2
    q, k, v = rand_qkv(n, d, dv, seed=9)
    ref = oracle.hla3_serial(q, k, v, masked=True)[0]
    Q, K, V = q[0], k[0], v[0]
    W = np.tril(Q @ K.T)
    alt1 = np.tril(W @ W.T) @ W @ V
    alt2 = np.tril(W @ W.T @ W) @ V
    assert relerr(alt1, ref) > 1e-3
    assert relerr(alt2, ref) > 1e-3


def test_unmasked_is_prefix_causal_not_full_tensor_attention():
    """Eq. hla-unnorm: o_t = q_t^T S_t C_t uses prefix sums up to t (causal in t,
    with i and j each running to t), not the non-causal T_2 = (QK^T)(QK^T)^T V."""
    n, d, dv = 8, 3, 2
    q, k, v = rand_qkv(n, d, dv, seed=10)
    ou = oracle.hla2_serial(q, k, v, masked=False)[0]
    A = q[0] @ k[0].T
    full = (A @ A.T) @ v[0]
    assert relerr(ou[-1], full[-1]) < 1e-12   # the last row sees every token
    assert relerr(ou[:-1], full[:-1]) > 1e-3  # earlier rows do not see the future
