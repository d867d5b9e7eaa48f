"""Where the factor K of the fp32 bound in tests/parity.py comes from.

tests/den_model.py repeats in float32 the stages by which the fused kernel forms
the denominator of the ratio-normalised output (Theorem 1, Eq. masked).  Check 3
of tests/parity.py allows the implied denominator an absolute error of
max(bar |den_t + eps|, K u sqrt(t+1) s_t); only rows whose error exceeds
bar |den_t + eps| depend on K.  The K such a row needs is
err_t / (u sqrt(t+1) s_t); its maximum over the rows of the cases the GPU tests
run is the envelope that K must cover.  These tests compute that envelope from
the model (no GPU) and check that K_FP32 covers it without exceeding it by more
than a factor of two (the margin for the tensor cores' accumulation order,
which the model does not reproduce).
"""
import numpy as np
import pytest

import hla_inputs
import oracle
from den_model import fused_den
from parity import K_FP32, TOL, U32, local_rms


def _k_needed(qf, kf, seg_tiles, tol=TOL["bf16"], eps=hla_inputs.EPS):
    """(K needed, rows whose model denominator misses tol |den + eps|, the oracle's denominators) for
    heads [h, n, d]."""
    vf = np.zeros(qf.shape[:2] + (1,), np.float32)
    _, den = oracle.hla2_serial(qf, kf, vf, masked=True, normalized=False, return_den=True, nthreads=8)
    n = qf.shape[1]
    scale = U32 * np.sqrt(np.arange(n) + 1.0) * local_rms(den)
    k_need, rows = 0.0, 0
    for h in range(qf.shape[0]):
        dm = fused_den(qf[h], kf[h], seg_tiles)
        err = np.abs(dm - den[h])
        miss = err > tol * np.abs(den[h] + eps)
        rows += int(miss.sum())
        if miss.any():
            k_need = max(k_need, float((err[miss] / scale[h][miss]).max()))
    return k_need, rows, den


def test_model_matches_oracle_where_well_conditioned():
    """The model computes the paper's denominator: on rows far from a zero of den it agrees with the
    fp64 oracle to the precision of its bf16 hi + lo operands, with one segment per head and with the
    carried e prefix of later segments (2 and 6 tiles per segment)."""
    q, k, _ = hla_inputs.make_qkv(1, 2, 700, 128, 128, seed=5, dtype="bf16")
    qf, kf = q.reshape(2, 700, 128), k.reshape(2, 700, 128)
    _, den = oracle.hla2_serial(qf, kf, np.zeros((2, 700, 1)), masked=True, return_den=True)
    s = local_rms(den)
    for h in range(2):
        for seg in (1, 2, 6):
            dm = fused_den(qf[h], kf[h], seg)
            well = np.abs(den[h]) > 0.1 * s[h]
            assert np.abs(dm - den[h])[well].max() <= 1e-4 * np.abs(den[h][well]).max()


@pytest.fixture(scope="module")
def envelopes():
    out = {}
    # the 80-head case of the fused tests (one segment per head: 3 tiles)
    for d in (64, 128):
        q, k, _ = hla_inputs.make_qkv(2, 40, 300, d, d, seed=77 + d, dtype="bf16")
        out["80x300 d%d" % d] = _k_needed(q.reshape(80, 300, d), k.reshape(80, 300, d), 3)[:2]
    # the long workload's sampled heads (segments of 7 tiles on 152 SMs)
    w = hla_inputs.WORKLOADS["long_bf16_norm"]
    q, k, _ = hla_inputs.make_workload(w)
    heads = [0, w.BH // 2 + 1, w.BH - 1]
    out["long sampled"] = _k_needed(q.reshape(w.BH, w.n, w.d)[heads], k.reshape(w.BH, w.n, w.d)[heads], 7)[:2]
    return out


def test_k_is_the_model_envelope(envelopes):
    k_env = max(v[0] for v in envelopes.values())
    print("model envelope of K:", {k: round(v[0], 3) for k, v in envelopes.items()},
          "rows beyond the bar:", {k: v[1] for k, v in envelopes.items()})
    assert k_env <= K_FP32, envelopes
    assert K_FP32 <= 2.0 * k_env, (K_FP32, envelopes)


def test_rows_beyond_the_bar_are_rare(envelopes):
    """Rows whose fp32 denominator misses the bar are those with den within about u sqrt(t) s_t / bar
    of zero: a few in tens of thousands."""
    for name, (_, rows) in envelopes.items():
        assert rows <= 5, (name, rows)
