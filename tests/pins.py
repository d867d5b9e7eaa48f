"""Pins for the fp64 oracle: checks against what the paper and mathematics fix.

Every pin is a plain function that raises AssertionError when the oracle is
wrong, so that the mutation tests can run the same pins against oracle builds
with a planted mistake.  The references here are written independently of the
oracle's recurrence: the defining sums of the operators (numpy matrix forms and
pure-Python loops), exact integer arithmetic, closed forms for special cases,
and algebraic invariants stated in the paper.
"""
from __future__ import annotations

import itertools
import json
import os

import numpy as np

import oracle

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def rand_qkv(n, d, dv, seed, BH=1):
    """fp64 inputs with the workload recipe (unit-norm Gaussian q, k rows; N(0,1) v)."""
    rng = np.random.default_rng(seed)
    q = rng.standard_normal((BH, n, d))
    k = rng.standard_normal((BH, n, d))
    q /= np.linalg.norm(q, axis=-1, keepdims=True)
    k /= np.linalg.norm(k, axis=-1, keepdims=True)
    v = rng.standard_normal((BH, n, dv))
    return q, k, v


def relerr(a, b):
    """max |a-b| / max(|b|, tiny): scale-aware comparison for fp64 pins."""
    a, b = np.asarray(a, float), np.asarray(b, float)
    return float(np.max(np.abs(a - b)) / max(np.max(np.abs(b)), 1e-300)) if b.size else 0.0


# --------------------------------------------------------------------------
# independent references (defining sums)
# --------------------------------------------------------------------------

def brute2(q, k, v, masked):
    """Second order from the defining sums, one head (q,k: [n,d], v: [n,dv]).

    masked  (Theorem 1, Fig. 1(B)): T = [(L.QK^T)(L.QK^T)^T] . L,  o = T V, den = T 1
    unmasked (Eq. hla-unnorm):       o_t = sum_{j<=t} sum_{i<=t} (q_t.k_i)(q_j.k_i) v_j
    """
    n = q.shape[0]
    A = q @ k.T
    if masked:
        W = np.tril(A)
        T = np.tril(W @ W.T)
        return T @ v, T.sum(axis=1)
    out = np.zeros((n, v.shape[1]))
    den = np.zeros(n)
    for t in range(n):
        w = A[: t + 1, : t + 1] @ A[t, : t + 1]  # w_j = sum_{i<=t} A[t,i] A[j,i], j <= t
        out[t] = w @ v[: t + 1]
        den[t] = w.sum()
    return out, den


def brute2_loops(q, k, v, masked):
    """The same defining sums with pure-Python scalar loops (tiny n only)."""
    n, d, dv = len(q), len(q[0]), len(v[0])

    def dotp(a, b):
        return sum(a[x] * b[x] for x in range(d))

    out = [[0.0] * dv for _ in range(n)]
    den = [0.0] * n
    for t in range(n):
        for j in range(t + 1):
            w = 0.0
            for i in range((j if masked else t) + 1):
                w += dotp(q[t], k[i]) * dotp(q[j], k[i])
            den[t] += w
            for c in range(dv):
                out[t][c] += w * v[j][c]
    return out, den


def brute3(q, k, v, masked):
    """Third order from index triples, one head (tiny n).

    term(i,u,j) = (q_t.k_i)(q_u.k_i)(q_u.k_j) v_j over (i,u,j) in [1..t]^3.
    unmasked (Sec. 7.1): all triples (= q_t^T S^K S^Q P^KV).
    masked (Theorem 3): the triples whose largest index occurs at least twice,
    i.e. all triples minus those with a unique maximum in position i (G1),
    u (G2) or j (G3).
    """
    n, dv = q.shape[0], v.shape[1]
    A = q @ k.T
    out = np.zeros((n, dv))
    den = np.zeros(n)
    for t in range(n):
        for i, u, j in itertools.product(range(t + 1), repeat=3):
            if masked:
                mx = max(i, u, j)
                if (i, u, j).count(mx) < 2:
                    continue
            w = A[t, i] * A[u, i] * A[u, j]
            out[t] += w * v[j]
            den[t] += w
    return out, den


# --------------------------------------------------------------------------
# second-order pins
# --------------------------------------------------------------------------

CASES2 = [(1, 1, 1), (2, 3, 2), (5, 4, 3), (17, 3, 5), (33, 8, 4)]


def pin_hla2_bruteforce(tol=1e-12):
    """Serial recurrence == defining sums (Theorem 1; Eq. hla-unnorm; v -> 1 for den)."""
    for (n, d, dv), masked, normalized in itertools.product(CASES2, (True, False), (False, True)):
        q, k, v = rand_qkv(n, d, dv, seed=n * 100 + d * 10 + dv, BH=2)
        eps = 0.5
        got, den = oracle.hla2_serial(q, k, v, masked=masked, normalized=normalized, eps=eps, return_den=True)
        for hd in range(2):
            o_ref, den_ref = brute2(q[hd], k[hd], v[hd], masked)
            if normalized:
                o_ref = o_ref / (den_ref + eps)[:, None]
            assert relerr(got[hd], o_ref) < tol, ("out", n, d, dv, masked, normalized, relerr(got[hd], o_ref))
            assert relerr(den[hd], den_ref) < tol, ("den", n, d, dv, masked)


def pin_hla2_python_loops(tol=1e-12):
    """Serial recurrence == the double sum evaluated with scalar Python loops."""
    for masked in (True, False):
        q, k, v = rand_qkv(6, 3, 2, seed=7)
        got, den = oracle.hla2_serial(q, k, v, masked=masked, return_den=True)
        o_ref, den_ref = brute2_loops(q[0].tolist(), k[0].tolist(), v[0].tolist(), masked)
        assert relerr(got[0], o_ref) < tol, masked
        assert relerr(den[0], den_ref) < tol, masked


def pin_hla2_golden():
    """Hand-worked integer example (tests/golden/hla2_hand_example.json): exact."""
    g = json.load(open(os.path.join(GOLDEN, "hla2_hand_example.json")))
    q, k, v = (np.array(g[x], dtype=float) for x in ("q", "k", "v"))
    o, den, st = oracle.hla2_serial(q, k, v, masked=True, return_den=True, return_state=True)
    assert np.array_equal(o[0], np.array(g["masked_out"], float)), o
    assert np.array_equal(den[0], np.array(g["masked_den"], float)), den
    parts = oracle.split_state2(st[0], 2, 1)
    assert np.array_equal(parts["G"], np.array(g["G_final"], float)), parts["G"]
    assert np.array_equal(parts["h"], np.array(g["h_final"], float)), parts["h"]
    o, den = oracle.hla2_serial(q, k, v, masked=False, return_den=True)
    assert np.array_equal(o[0], np.array(g["unmasked_out"], float)), o
    assert np.array_equal(den[0], np.array(g["unmasked_den"], float)), den


def pin_hla2_exact_integers():
    """Small-integer inputs: fp64 arithmetic is exact, so the oracle must equal
    the defining sum evaluated in Python integers bit for bit."""
    rng = np.random.default_rng(11)
    n, d, dv = 7, 3, 2
    q = rng.integers(-2, 3, (n, d))
    k = rng.integers(-2, 3, (n, d))
    v = rng.integers(-3, 4, (n, dv))
    for masked in (True, False):
        ref, rden = brute2_loops(q.tolist(), k.tolist(), v.tolist(), masked)  # Python ints: exact
        got, den = oracle.hla2_serial(q, k, v, masked=masked, return_den=True)
        assert np.array_equal(got[0], np.array(ref, float)), masked
        assert np.array_equal(den[0], np.array(rden, float)), masked


def pin_hla2_masked_vs_unmasked():
    """unmasked - masked = q_t^T G_t and den: q_t^T h_t, for every t (Theorem 1
    vs Eq. hla-unnorm: the masked numerator subtracts exactly G_t)."""
    n, d, dv = 9, 4, 3
    q, k, v = rand_qkv(n, d, dv, seed=5)
    om, dm = oracle.hla2_serial(q, k, v, masked=True, return_den=True)
    ou, du = oracle.hla2_serial(q, k, v, masked=False, return_den=True)
    for t in range(n):
        st = oracle.hla2_serial(q[:, : t + 1], k[:, : t + 1], v[:, : t + 1], masked=True, return_state=True)[1]
        parts = oracle.split_state2(st[0], d, dv)
        assert relerr(ou[0, t] - om[0, t], q[0, t] @ parts["G"]) < 1e-10, t
        assert abs((du[0, t] - dm[0, t]) - q[0, t] @ parts["h"]) < 1e-10 * max(1.0, abs(du[0, t])), t


def pin_hla2_state_definitions():
    """Final state equals the definitions: S = sum k k^T, C = sum q v^T, m = sum q,
    G = sum_i k_i k_i^T C_{i-1}, h = sum_i k_i k_i^T m_{i-1} (Sec. 3 and 3.2)."""
    n, d, dv = 8, 3, 2
    q, k, v = rand_qkv(n, d, dv, seed=8)
    st = oracle.hla2_serial(q, k, v, masked=True, return_state=True)[1]
    p = oracle.split_state2(st[0], d, dv)
    Q, K, V = q[0], k[0], v[0]
    assert relerr(p["S"], K.T @ K) < 1e-13
    assert relerr(p["C"], Q.T @ V) < 1e-13
    assert relerr(p["m"], Q.sum(0)) < 1e-13
    G = np.zeros((d, dv))
    h = np.zeros(d)
    for i in range(n):
        Cp = Q[:i].T @ V[:i]
        mp = Q[:i].sum(0)
        G += np.outer(K[i], K[i]) @ Cp
        h += np.outer(K[i], K[i]) @ mp
    assert relerr(p["G"], G) < 1e-13
    assert relerr(p["h"], h) < 1e-13


def pin_hla2_chunked_equals_serial():
    """Theorem 2: the two-level exclusive scan equals the serial loop, for every
    chunk size (ragged last chunk included), with and without an initial state."""
    n, d, dv = 13, 3, 2
    q, k, v = rand_qkv(n, d, dv, seed=13)
    st0 = oracle.hla2_serial(*rand_qkv(4, d, dv, seed=99), masked=True, return_state=True)[1]
    for masked, normalized in itertools.product((True, False), (False, True)):
        for init in (None, st0):
            ref, rden, rst = oracle.hla2_serial(q, k, v, masked=masked, normalized=normalized, eps=0.25,
                                               state_in=init, return_den=True, return_state=True)
            for chunk in range(1, n + 2):
                got, den, st = oracle.hla2_chunked(q, k, v, chunk, masked=masked, normalized=normalized, eps=0.25,
                                                   state_in=init, return_den=True, return_state=True)
                assert relerr(got, ref) < 1e-11, (masked, normalized, chunk)
                assert relerr(den, rden) < 1e-11, (masked, chunk)
                assert relerr(st, rst) < 1e-11, (masked, chunk)


def pin_hla2_combine_algebra():
    """Eq. semidirect is associative; zero is its identity; and folding a
    single-token segment into a state is one step of the serial recurrence
    (proof of Theorem 2: Phi(X, T_t) = X (+) T_t)."""
    d, dv = 3, 2
    L = oracle.hla2_state_len(d, dv)
    rng = np.random.default_rng(3)
    for masked in (True, False):
        A, B, C = (rng.standard_normal(L) for _ in range(3))
        left = oracle.hla2_combine(oracle.hla2_combine(A, B, d, dv, masked), C, d, dv, masked)
        right = oracle.hla2_combine(A, oracle.hla2_combine(B, C, d, dv, masked), d, dv, masked)
        assert relerr(left, right) < 1e-13, masked
        Z = np.zeros(L)
        assert relerr(oracle.hla2_combine(Z, A, d, dv, masked), A) == 0.0
        assert relerr(oracle.hla2_combine(A, Z, d, dv, masked), A) == 0.0
    # non-commutativity of the masked product (the cross term depends on order)
    AB = oracle.hla2_combine(A, B, d, dv, True)
    BA = oracle.hla2_combine(B, A, d, dv, True)
    assert relerr(AB, BA) > 1e-6
    # one serial step == state (+) token segment, token segment has G = h = 0
    q, k, v = rand_qkv(6, d, dv, seed=4)
    st5 = oracle.hla2_serial(q[:, :5], k[:, :5], v[:, :5], masked=True, return_state=True)[1][0]
    st6 = oracle.hla2_serial(q, k, v, masked=True, return_state=True)[1][0]
    qt, kt, vt = q[0, 5], k[0, 5], v[0, 5]
    T = oracle.pack_state2(np.outer(kt, kt), np.outer(qt, vt), qt, np.zeros((d, dv)), np.zeros(d))
    assert relerr(oracle.hla2_combine(st5, T, d, dv, True), st6) < 1e-13


def pin_hla2_special_cases():
    """n = 1: o = (q.k)^2 v, den = (q.k)^2 (masked = unmasked at t = 1);
    d = dv = 1: masked o_t = q_t sum_{j<=t} q_j v_j s_j with s_j = sum_{i<=j} k_i^2,
    unmasked o_t = q_t s_t sum_{j<=t} q_j v_j."""
    q, k, v = rand_qkv(1, 5, 3, seed=1)
    for masked in (True, False):
        o, den = oracle.hla2_serial(q, k, v, masked=masked, return_den=True)
        a = float(q[0, 0] @ k[0, 0])
        assert relerr(o[0, 0], a * a * v[0, 0]) < 1e-14
        assert abs(den[0, 0] - a * a) < 1e-15
    rng = np.random.default_rng(2)
    n = 11
    q = rng.standard_normal((1, n, 1))
    k = rng.standard_normal((1, n, 1))
    v = rng.standard_normal((1, n, 1))
    s = np.cumsum(k[0, :, 0] ** 2)
    qv = q[0, :, 0] * v[0, :, 0]
    om = oracle.hla2_serial(q, k, v, masked=True)[0, :, 0]
    ou = oracle.hla2_serial(q, k, v, masked=False)[0, :, 0]
    assert relerr(om, q[0, :, 0] * np.cumsum(qv * s)) < 1e-12
    assert relerr(ou, q[0, :, 0] * s * np.cumsum(qv)) < 1e-12


def pin_hla2_causality():
    """Changing tokens after t leaves outputs up to t bit-identical."""
    n, d, dv, t = 12, 4, 3, 6
    q, k, v = rand_qkv(n, d, dv, seed=21)
    q2, k2, v2 = q.copy(), k.copy(), v.copy()
    rng = np.random.default_rng(0)
    q2[:, t + 1:] = rng.standard_normal(q2[:, t + 1:].shape)
    k2[:, t + 1:] = rng.standard_normal(k2[:, t + 1:].shape)
    v2[:, t + 1:] = rng.standard_normal(v2[:, t + 1:].shape)
    for masked in (True, False):
        a = oracle.hla2_serial(q, k, v, masked=masked, normalized=True)
        b = oracle.hla2_serial(q2, k2, v2, masked=masked, normalized=True)
        assert np.array_equal(a[:, : t + 1], b[:, : t + 1])
        assert not np.array_equal(a[:, t + 1:], b[:, t + 1:])


def pin_hla2_state_handoff():
    """Resuming from a saved state equals the uninterrupted run (streaming form):
    forward(n1) -> state -> forward(n2) == forward(n1 + n2); a chain of
    single-token calls (decode steps) == forward over the concatenation."""
    n, d, dv = 14, 4, 3
    q, k, v = rand_qkv(n, d, dv, seed=31, BH=2)
    for masked, normalized in itertools.product((True, False), (False, True)):
        ref, rst = oracle.hla2_serial(q, k, v, masked=masked, normalized=normalized, return_state=True)
        o1, st = oracle.hla2_serial(q[:, :9], k[:, :9], v[:, :9], masked=masked, normalized=normalized,
                                    return_state=True)
        o2, st2 = oracle.hla2_serial(q[:, 9:], k[:, 9:], v[:, 9:], masked=masked, normalized=normalized,
                                     state_in=st, return_state=True)
        assert relerr(np.concatenate([o1, o2], axis=1), ref) < 1e-12
        assert relerr(st2, rst) < 1e-12
        st = None
        outs = []
        for t in range(n):
            o, st = oracle.hla2_serial(q[:, t:t + 1], k[:, t:t + 1], v[:, t:t + 1], masked=masked,
                                       normalized=normalized, state_in=st, return_state=True)
            outs.append(o)
        assert relerr(np.concatenate(outs, axis=1), ref) < 1e-12
        assert relerr(st, rst) < 1e-12


# --------------------------------------------------------------------------
# third-order pins
# --------------------------------------------------------------------------

CASES3 = [(1, 1, 1), (2, 2, 1), (5, 3, 2), (9, 2, 3)]


def pin_hla3_bruteforce(tol=1e-11):
    """Algorithm 3 (gamma = 1) == the sum over index triples (Theorem 3); the
    unmasked factorisation == all triples (Sec. 7.1)."""
    for (n, d, dv), masked, normalized in itertools.product(CASES3, (True, False), (False, True)):
        q, k, v = rand_qkv(n, d, dv, seed=3 * n + d, BH=2)
        eps = 0.5
        got, den = oracle.hla3_serial(q, k, v, masked=masked, normalized=normalized, eps=eps, return_den=True)
        for hd in range(2):
            o_ref, den_ref = brute3(q[hd], k[hd], v[hd], masked)
            if normalized:
                o_ref = o_ref / (den_ref + eps)[:, None]
            assert relerr(got[hd], o_ref) < tol, (n, d, dv, masked, normalized, relerr(got[hd], o_ref))
            assert relerr(den[hd], den_ref) < tol, (n, d, dv, masked)


def pin_hla3_golden():
    """Hand-worked scalar example (tests/golden/hla3_hand_example.json): exact."""
    g = json.load(open(os.path.join(GOLDEN, "hla3_hand_example.json")))
    q, k, v = (np.array(g[x], dtype=float) for x in ("q", "k", "v"))
    assert np.array_equal(oracle.hla3_serial(q, k, v, masked=True)[0], np.array(g["masked_out"], float))
    assert np.array_equal(oracle.hla3_serial(q, k, v, masked=False)[0], np.array(g["unmasked_out"], float))


def pin_hla3_chunked_equals_serial():
    """Theorem 4: exclusive scans under the third-order concatenation (with the
    segment maps) reproduce Algorithm 3 for every chunk size."""
    n, d, dv = 10, 2, 2
    q, k, v = rand_qkv(n, d, dv, seed=17)
    for normalized in (False, True):
        ref, rden = oracle.hla3_serial(q, k, v, masked=True, normalized=normalized, eps=0.25, return_den=True)
        for chunk in range(1, n + 2):
            got, den = oracle.hla3_chunked(q, k, v, chunk, normalized=normalized, eps=0.25, return_den=True)
            assert relerr(got, ref) < 1e-11, (chunk, normalized, relerr(got, ref))
            assert relerr(den, rden) < 1e-11, chunk


def pin_hla3_state_handoff():
    """Third-order streaming resumes exactly from a saved state."""
    n, d, dv = 9, 3, 2
    q, k, v = rand_qkv(n, d, dv, seed=41)
    for masked in (True, False):
        ref, rst = oracle.hla3_serial(q, k, v, masked=masked, return_state=True)
        o1, st = oracle.hla3_serial(q[:, :4], k[:, :4], v[:, :4], masked=masked, return_state=True)
        o2, st2 = oracle.hla3_serial(q[:, 4:], k[:, 4:], v[:, 4:], masked=masked, state_in=st, return_state=True)
        assert relerr(np.concatenate([o1, o2], axis=1), ref) < 1e-12
        assert relerr(st2, rst) < 1e-12


# --------------------------------------------------------------------------
# (S, D, e) state, AHLA, gradients
# --------------------------------------------------------------------------

def pin_sde_definition():
    """The (S, D, e) fold of the masked tuple: D_t = sum_{j<=t} x_j v_j^T and
    e_t = sum_{j<=t} x_j with x_j = S_j q_j (proof of Theorem 1: num_t =
    q_t^T sum_j S_j q_j v_j^T), built here token by token from the definitions
    of S; and q_t^T D_t, q_t^T e_t are Theorem 1's num_t, den_t."""
    n, d, dv = 9, 4, 3
    q, k, v = rand_qkv(n, d, dv, seed=17)
    st0 = oracle.hla2_serial(*rand_qkv(5, d, dv, seed=18), masked=True, return_state=True)[1]
    for init in (None, st0):
        out, den, st = oracle.hla2_serial(q, k, v, masked=True, state_in=init, return_state=True, return_den=True)
        sde = oracle.hla2_state_to_sde(st[0], d, dv)
        p0 = oracle.split_state2(st0[0], d, dv) if init is not None else None
        S = p0["S"].copy() if p0 else np.zeros((d, d))
        D = (p0["S"] @ p0["C"] - p0["G"]) if p0 else np.zeros((d, dv))
        e = (p0["S"] @ p0["m"] - p0["h"]) if p0 else np.zeros(d)
        for t in range(n):
            S = S + np.outer(k[0, t], k[0, t])
            x = S @ q[0, t]
            D = D + np.outer(x, v[0, t])
            e = e + x
        assert relerr(sde[: d * d], S.ravel()) < 1e-13
        assert relerr(sde[d * d: d * d + d * dv], D.ravel()) < 1e-12
        assert relerr(sde[d * d + d * dv:], e) < 1e-12
        assert relerr(q[0, -1] @ sde[d * d: d * d + d * dv].reshape(d, dv), out[0, -1]) < 1e-12
        assert abs(q[0, -1] @ sde[d * d + d * dv:] - den[0, -1]) < 1e-12 * max(1.0, abs(den[0, -1]))


def brute_ahla(q, k, v):
    """AHLA from its definition (Eq. AHLA-explicit), one head: with A = L . (Q K^T),
    (A A)_{tj} = sum_{i=j..t} (q_t.k_i)(q_i.k_j), o = (A A) V, den = (A A) 1."""
    A = np.tril(q @ k.T)
    AA = A @ A
    return AA @ v, AA.sum(axis=1)


def brute_ahla_loops(q, k, v):
    """Eq. AHLA-explicit as nested loops over Python numbers (exact for integers)."""
    n, d, dv = len(q), len(q[0]), len(v[0])
    dotp = lambda a, b: sum(x * y for x, y in zip(a, b))
    out, den = [], []
    for t in range(n):
        o = [0] * dv
        s = 0
        for j in range(t + 1):
            w = sum(dotp(q[t], k[i]) * dotp(q[i], k[j]) for i in range(j, t + 1))
            for c in range(dv):
                o[c] += w * v[j][c]
            s += w
        out.append(o)
        den.append(s)
    return out, den


def pin_ahla_bruteforce():
    """The AHLA recurrence (Theorem AHLA) equals its defining sum, unnormalised
    and ratio-normalised (v -> 1 gives the denominator)."""
    n, d, dv = 10, 3, 2
    q, k, v = rand_qkv(n, d, dv, seed=51, BH=2)
    out, den = oracle.ahla_serial(q, k, v, return_den=True)
    outn = oracle.ahla_serial(q, k, v, normalized=True, eps=0.3)
    for h in range(2):
        ref, rden = brute_ahla(q[h], k[h], v[h])
        assert relerr(out[h], ref) < 1e-12
        assert relerr(den[h], rden) < 1e-12
        assert relerr(outn[h], ref / (rden + 0.3)[:, None]) < 1e-12


def pin_ahla_exact_integers():
    """Small-integer inputs: the fp64 recurrence equals the defining sum in Python integers bit for bit."""
    rng = np.random.default_rng(52)
    n, d, dv = 6, 3, 2
    q, k, v = rng.integers(-2, 3, (n, d)), rng.integers(-2, 3, (n, d)), rng.integers(-3, 4, (n, dv))
    ref, rden = brute_ahla_loops(q.tolist(), k.tolist(), v.tolist())
    got, den = oracle.ahla_serial(q, k, v, return_den=True)
    assert np.array_equal(got[0], np.array(ref, float))
    assert np.array_equal(den[0], np.array(rden, float))


def pin_ahla_scan_equals_serial():
    """Scan equivalence for AHLA: exclusive Blelloch scans under Eq. AHLA-semidirect,
    then local inclusion, reproduce the serial recurrence for every chunk size; and a
    serial run resumed from a saved state equals one run over the concatenation."""
    n, d, dv = 11, 3, 2
    q, k, v = rand_qkv(n, d, dv, seed=53)
    for normalized in (False, True):
        ref, rden = oracle.ahla_serial(q, k, v, normalized=normalized, eps=0.25, return_den=True)
        for chunk in range(1, n + 2):
            got, den = oracle.ahla_chunked(q, k, v, chunk, normalized=normalized, eps=0.25, return_den=True)
            assert relerr(got, ref) < 1e-11, (normalized, chunk)
            assert relerr(den, rden) < 1e-11, chunk
    ref, rst = oracle.ahla_serial(q, k, v, return_state=True)
    o1, st = oracle.ahla_serial(q[:, :5], k[:, :5], v[:, :5], return_state=True)
    o2, st2 = oracle.ahla_serial(q[:, 5:], k[:, 5:], v[:, 5:], state_in=st, return_state=True)
    assert relerr(np.concatenate([o1, o2], axis=1), ref) < 1e-12
    assert relerr(st2, rst) < 1e-12


def pin_ahla_combine_algebra():
    """Eq. AHLA-semidirect is associative with zero as identity, not commutative;
    and the fold of single-token summaries (R = k q^T, P = k v^T, m = k,
    E = (q.k) k v^T, n = (q.k) k) is the serial state (its P, m, E, n)."""
    d, dv = 3, 2
    L = oracle.ahla_summary_len(d, dv)
    rng = np.random.default_rng(54)
    A, B, C = (rng.standard_normal(L) for _ in range(3))
    left = oracle.ahla_combine(oracle.ahla_combine(A, B, d, dv), C, d, dv)
    right = oracle.ahla_combine(A, oracle.ahla_combine(B, C, d, dv), d, dv)
    assert relerr(left, right) < 1e-13
    Z = np.zeros(L)
    assert relerr(oracle.ahla_combine(Z, A, d, dv), A) == 0.0 and relerr(oracle.ahla_combine(A, Z, d, dv), A) == 0.0
    assert relerr(oracle.ahla_combine(A, B, d, dv), oracle.ahla_combine(B, A, d, dv)) > 1e-6
    q, k, v = rand_qkv(7, d, dv, seed=55)
    acc = np.zeros(L)
    for t in range(7):
        qt, kt, vt = q[0, t], k[0, t], v[0, t]
        a = qt @ kt
        T = np.concatenate([np.outer(kt, qt).ravel(), np.outer(kt, vt).ravel(), kt, a * np.outer(kt, vt).ravel(),
                            a * kt])
        acc = oracle.ahla_combine(acc, T, d, dv)
    st = oracle.ahla_serial(q, k, v, return_state=True)[1][0]
    assert relerr(acc[d * d:], st) < 1e-12


def _loss2(q, k, v, g, masked, normalized, eps):
    return float((oracle.hla2_serial(q, k, v, masked=masked, normalized=normalized, eps=eps) * g).sum())


def pin_hla2_backward_finite_differences():
    """Gradients of L = sum_t g_t . o_t from the reverse sweep equal central finite
    differences of the forward (fp64, step 1e-6), masked and unmasked, plain and
    ratio-normalised, for every entry of q, k and v."""
    n, d, dv = 7, 3, 2
    q, k, v = rand_qkv(n, d, dv, seed=61)
    g = np.random.default_rng(62).standard_normal((1, n, dv))
    hstep = 1e-6
    for masked, normalized in itertools.product((True, False), (False, True)):
        eps = 0.5
        grads = oracle.hla2_backward(q, k, v, g, masked=masked, normalized=normalized, eps=eps, ckpt=3)
        for x, gx in zip((q, k, v), grads):
            fd = np.zeros_like(x)
            for idx in np.ndindex(x.shape):
                xp, xm = x.copy(), x.copy()
                xp[idx] += hstep
                xm[idx] -= hstep
                args_p = [xp if y is x else y for y in (q, k, v)]
                args_m = [xm if y is x else y for y in (q, k, v)]
                fd[idx] = (_loss2(*args_p, g, masked, normalized, eps) - _loss2(*args_m, g, masked, normalized,
                                                                               eps)) / (2 * hstep)
            assert relerr(gx, fd) < 1e-6, (masked, normalized)


def pin_hla2_backward_exact_integers():
    """Integer inputs: L is a polynomial of degree at most 2 in each input entry
    (each q_t, k_i occurs in at most two factors of the defining sums of Theorem 1 /
    Eq. hla-unnorm), so the central difference with step 1 of the defining sum in
    Python integers is the exact derivative; the reverse sweep must equal it bit for bit."""
    rng = np.random.default_rng(63)
    n, d, dv = 5, 2, 2
    q, k, v = rng.integers(-2, 3, (n, d)), rng.integers(-2, 3, (n, d)), rng.integers(-2, 3, (n, dv))
    g = rng.integers(-2, 3, (n, dv))
    for masked in (True, False):
        def loss(qq, kk, vv):
            o, _ = brute2_loops(qq, kk, vv, masked)
            return sum(o[t][c] * int(g[t, c]) for t in range(n) for c in range(dv))
        grads = oracle.hla2_backward(q, k, v, g, masked=masked, ckpt=2)
        for which, gx in enumerate(grads):
            base = [q.tolist(), k.tolist(), v.tolist()]
            for idx in np.ndindex(gx.shape[1:]):
                plus = [list(map(list, a)) for a in base]
                minus = [list(map(list, a)) for a in base]
                plus[which][idx[0]][idx[1]] += 1
                minus[which][idx[0]][idx[1]] -= 1
                diff = loss(*plus) - loss(*minus)
                assert diff % 2 == 0
                assert gx[0][idx] == diff // 2, (masked, which, idx)


def pin_hla2_backward_checkpoints():
    """The reverse sweep does not depend on where the forward states are checkpointed."""
    n, d, dv = 10, 3, 2
    q, k, v = rand_qkv(n, d, dv, seed=64)
    g = np.random.default_rng(65).standard_normal((1, n, dv))
    for masked, normalized in ((True, False), (True, True), (False, True)):
        ref = oracle.hla2_backward(q, k, v, g, masked=masked, normalized=normalized, eps=0.5, ckpt=1)
        for ck in (3, 4, 10, 64):
            got = oracle.hla2_backward(q, k, v, g, masked=masked, normalized=normalized, eps=0.5, ckpt=ck)
            for a, b in zip(got, ref):
                assert relerr(a, b) < 1e-13, ck


ALL_PINS = [
    pin_hla2_bruteforce, pin_hla2_python_loops, pin_hla2_golden, pin_hla2_exact_integers,
    pin_hla2_masked_vs_unmasked, pin_hla2_state_definitions, pin_hla2_chunked_equals_serial,
    pin_hla2_combine_algebra, pin_hla2_special_cases, pin_hla2_causality, pin_hla2_state_handoff,
    pin_hla3_bruteforce, pin_hla3_golden, pin_hla3_chunked_equals_serial, pin_hla3_state_handoff,
    pin_sde_definition, pin_ahla_bruteforce, pin_ahla_exact_integers, pin_ahla_scan_equals_serial,
    pin_ahla_combine_algebra, pin_hla2_backward_finite_differences, pin_hla2_backward_exact_integers,
    pin_hla2_backward_checkpoints,
]
