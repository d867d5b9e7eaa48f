"""fp32 model of how the fused second-order kernel forms the denominator of the
ratio-normalised output -- TEST INFRASTRUCTURE (numpy; shares nothing with the
CUDA library and is not the oracle).

The denominator of Theorem 1 (Eq. masked), den_t = q_t . e_t with
e_t = sum_{j<=t} x_j and x_j = S_j q_j, is a sum whose terms are much larger
than the sum itself on some rows, so its rounding error decides which rows an
fp32 evaluation can resolve.  This module repeats, in float32 numpy with
explicit bf16 roundings, the arithmetic the fused kernel performs for it, in
the kernel's order of stages:

* per 128-token tile, the S carry S_p (fp32, accumulated tile by tile from
  K^T K products) is shifted by c I with c = bf16(trace / d) of the carry one
  tile back (the carry-in for the first two tiles of a segment), and
  R = S_p - c I is split into bf16 hi + lo;
* W = L . (Q K^T) (fp32 products) is split into bf16 hi + lo;
* X = Q R_hi + Q R_lo + W_hi K + W_lo K (fp32 accumulation), then x = X + c q;
* x is split into bf16 hi + lo and T = L . (Q X_hi^T + Q X_lo^T) (fp32);
* per row, each of the four 32-column quarters sums q . e_p over its columns
  (fused multiply-adds in column order) and then its T entries; the four
  partials are added in the order ((q0 + q1) + q2) + q3;
* the segment-local e carry gains the column sums of x of each tile (sums of
  32-row quarters, combined as (E0 + E1) + (E2 + E3));
* segments after the first keep that local denominator and later add
  q_t . e_prefix (e_prefix = the fp32 sum of the earlier segments' local e
  carries, in order), again per quarter: (((den_loc + qe0) + qe1) + qe2) + qe3.

Matrix products are float32 numpy products (fp32 accumulation with the
library's own blocking); the tensor cores accumulate in another order, so the
model reproduces the size of the rounding errors, not their bits.
"""
from __future__ import annotations

import numpy as np

TILE = 128


def bf16(x):
    """Round float32 values to bfloat16 (nearest, ties to even), returned as float32."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    b = x.view(np.uint32).astype(np.uint64)
    b = ((b + np.uint64(0x7FFF) + ((b >> np.uint64(16)) & np.uint64(1))) >> np.uint64(16)) << np.uint64(16)
    return b.astype(np.uint32).view(np.float32)


def split(x, exact=False):
    """bf16 hi + lo of fp32 values (hi + lo = x within 2^-16 |x|); with exact, x itself and zeros."""
    if exact:
        return np.float32(x), np.zeros_like(x, dtype=np.float32)
    hi = bf16(x)
    return hi, bf16(np.float32(x) - hi)


def _quarter_dot(q, e):
    """Per row, the four 32-column partial sums of q . e, as fused multiply-adds
    in column order (one rounding per step: the product of a bf16 and an fp32
    value is exact in fp64, and so is its sum with the fp32 partial)."""
    n = q.shape[0]
    parts = np.zeros((n, 4), np.float32)
    for c in range(q.shape[1]):
        parts[:, c // 32] = (parts[:, c // 32].astype(np.float64)
                             + q[:, c].astype(np.float64) * np.float64(e[c])).astype(np.float32)
    return parts


def _quarter_add_rows(parts, T):
    """Add each row's T entries to the partial of the quarter they belong to, in column order."""
    for c in range(T.shape[1]):
        parts[:, c // 32] = np.float32(parts[:, c // 32] + T[:, c])
    return parts


def _colsum_quarters(x):
    """e increment of a tile: column sums of x over four 32-row quarters, combined (E0 + E1) + (E2 + E3)."""
    E = [x[32 * i:32 * (i + 1)].astype(np.float32).sum(axis=0, dtype=np.float32) for i in range(4)]
    return np.float32(np.float32(E[0] + E[1]) + np.float32(E[2] + E[3]))


def fused_den(q, k, seg_tiles, exact_splits=False):
    """Denominator (without eps) of one head as the fused kernel forms it.

    q, k: [n, d] float32 with bf16-exact values (d <= 128; zero-padded to 128).
    seg_tiles: tiles of 128 tokens per segment (the kernel's work item).
    exact_splits: use the fp32 operands themselves where the kernel uses bf16
    hi + lo pairs (the same stages with fp32 operands throughout).
    Returns float64 [n].
    """
    n, d = q.shape
    D = 128
    Q = np.zeros((n, D), np.float32)
    K = np.zeros((n, D), np.float32)
    Q[:, :d] = q
    K[:, :d] = k
    M = (n + TILE - 1) // TILE
    L = max(1, min(seg_tiles, M))
    G = (M + L - 1) // L
    den = np.zeros(n, np.float64)
    lower = np.tril(np.ones((TILE, TILE), bool))
    S_prefix = np.zeros((D, D), np.float32)   # inclusive S prefix published by the previous segment
    e_prefix = np.zeros(D, np.float32)        # inclusive e prefix published by the previous segment
    for sg in range(G):
        t0 = sg * L
        nt = min(L, M - t0)
        S_in = S_prefix.copy()
        # segment aggregate of K^T K (the pre-pass), published as S_in + agg
        agg = np.zeros((D, D), np.float32)
        for j in range(nt):
            a, b = (t0 + j) * TILE, min(n, (t0 + j + 1) * TILE)
            agg = np.float32(agg + K[a:b].T @ K[a:b])
        S_next = np.float32(S_in + agg)
        S = S_in.copy()                       # the S carry of the sweep
        e_loc = np.zeros(D, np.float32)
        tr = [np.float32(np.trace(S_in))]     # traces of the carry at each tile start
        den_loc = np.zeros(nt * TILE, np.float32)
        for j in range(nt):
            a, b = (t0 + j) * TILE, min(n, (t0 + j + 1) * TILE)
            Qt = np.zeros((TILE, D), np.float32)
            Kt = np.zeros((TILE, D), np.float32)
            Qt[: b - a] = Q[a:b]
            Kt[: b - a] = K[a:b]
            c = bf16(np.float32(tr[max(0, j - 1)] / np.float32(D)))
            R_hi, R_lo = split(S - c * np.eye(D, dtype=np.float32), exact_splits)
            A = Qt @ Kt.T
            W = np.where(lower, A, np.float32(0))
            W_hi, W_lo = split(W, exact_splits)
            X = np.float32(np.float32(np.float32(Qt @ R_hi + Qt @ R_lo) + W_hi @ Kt) + W_lo @ Kt)
            x = np.float32(X + c * Qt)
            X_hi, X_lo = split(x, exact_splits)
            T = np.where(lower, np.float32(Qt @ X_hi.T + Qt @ X_lo.T), np.float32(0))
            parts = _quarter_add_rows(_quarter_dot(Qt, e_loc), T)
            dl = np.float32(np.float32(np.float32(parts[:, 0] + parts[:, 1]) + parts[:, 2]) + parts[:, 3])
            den_loc[j * TILE:(j + 1) * TILE] = dl
            e_loc = np.float32(e_loc + _colsum_quarters(x))
            S = np.float32(S + Kt.T @ Kt)
            tr.append(np.float32(np.trace(S)))
        a, b = t0 * TILE, min(n, (t0 + nt) * TILE)
        if sg == 0:
            den[a:b] = den_loc[: b - a]
        else:
            parts = _quarter_dot(Q[a:b], e_prefix)
            dfix = np.float32(np.float32(np.float32(np.float32(den_loc[: b - a] + parts[:, 0]) + parts[:, 1])
                                         + parts[:, 2]) + parts[:, 3])
            den[a:b] = dfix
        e_prefix = np.float32(e_prefix + e_loc)
        S_prefix = S_next
    return den
