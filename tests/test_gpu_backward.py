"""Gradients of masked second-order HLA on the GPU (hla2_backward, the reverse
chunk scan) against the oracle's reverse sweep of the serial recurrence
(itself pinned by finite differences and exact integer derivatives).  Error per
row of dq, dk, dv: max_c |g_gpu - g_ref| / ||g_ref row||_2, bars 1e-4 (fp32
tokens) and 2e-2 (bf16 tokens)."""
import numpy as np
import pytest
import torch

import hla_inputs
import oracle
from parity import TOL, rowerr, rowerr_stats

pytestmark = pytest.mark.gpu
DEV = "cuda:0"


@pytest.fixture(scope="module")
def hla():
    from paper_2510_27258_gb300 import build
    build.build()
    from paper_2510_27258_gb300 import hla as binding
    return binding


def _grads(hla, q, k, v, g, dtype, normalized, eps, chunk):
    tq, tk, tv, tg = (hla_inputs.as_torch(x, dtype, DEV) for x in (q, k, v, g))
    out = hla.hla2_backward(tq, tk, tv, tg, normalized=normalized, eps=eps, chunk=chunk)
    torch.cuda.synchronize()
    return [x.float().cpu().numpy() for x in out]


def _check(hla, B, H, n, d, dv, chunk, dtype, normalized, eps, seed, heads=None):
    q, k, v = hla_inputs.make_qkv(B, H, n, d, dv, seed=seed, dtype=dtype)
    g = hla_inputs.round_to(np.random.default_rng(seed + 1).standard_normal((B, H, n, dv)), dtype)
    got = _grads(hla, q, k, v, g, dtype, normalized, eps, chunk)
    BH = B * H
    heads = list(range(BH)) if heads is None else heads
    flat = lambda x: x.reshape(BH, n, -1)[heads]
    ref = oracle.hla2_backward(flat(q), flat(k), flat(v), flat(g), masked=True, normalized=normalized, eps=eps,
                               ckpt=64, nthreads=8)
    errs = [rowerr(flat(a), b) for a, b in zip(got, ref)]
    for name, e in zip(("dq", "dk", "dv"), errs):
        assert e < TOL[dtype], (name, e)
    _check.stats = [rowerr_stats(flat(a), b)[0] for a, b in zip(got, ref)]
    return errs


SHAPES = [
    # (B, H, n, d, dv, chunk, dtype)
    (1, 1, 1, 16, 16, 16, "f32"),
    (1, 2, 37, 16, 32, 16, "f32"),
    (1, 1, 300, 32, 128, 100, "f32"),
    (1, 3, 96, 64, 16, 32, "f32"),
    (1, 2, 257, 128, 128, 128, "f32"),
    (2, 1, 200, 64, 64, 64, "bf16"),
    (1, 1, 130, 128, 64, 7, "bf16"),
]


@pytest.mark.parametrize("shape", SHAPES, ids=lambda s: "B%dH%dn%dd%ddv%dC%d%s" % s)
def test_backward_small(hla, shape):
    B, H, n, d, dv, chunk, dtype = shape
    _check(hla, B, H, n, d, dv, chunk, dtype, False, hla_inputs.EPS, seed=3000 + n)


@pytest.mark.parametrize("shape", SHAPES[:5], ids=lambda s: "B%dH%dn%dd%ddv%dC%d%s" % s)
def test_backward_normalized(hla, shape):
    """Ratio-normalised output with eps chosen from the oracle's denominators so that
    den_t + eps >= 1 on every row: there the gradient of num / (den + eps) is well
    conditioned, and fp32 must meet the 1e-4 bar (near a zero of den + eps it is not:
    its relative error is that of den + eps itself)."""
    B, H, n, d, dv, chunk, dtype = shape
    seed = 3100 + n
    q, k, _ = hla_inputs.make_qkv(B, H, n, d, dv, seed=seed, dtype=dtype)
    _, den = oracle.hla2_serial(q.reshape(B * H, n, d), k.reshape(B * H, n, d), np.zeros((B * H, n, 1)),
                                masked=True, return_den=True)
    eps = 1.0 + max(0.0, -float(den.min()))
    _check(hla, B, H, n, d, dv, chunk, dtype, True, eps, seed=seed)


def test_backward_chunk_sizes_agree(hla):
    q, k, v = hla_inputs.make_qkv(1, 2, 333, 32, 32, seed=31, dtype="f32")
    g = hla_inputs.round_to(np.random.default_rng(32).standard_normal((1, 2, 333, 32)), "f32")
    ref = _grads(hla, q, k, v, g, "f32", False, 1e-6, 1)
    for chunk in (5, 16, 64, 128):
        got = _grads(hla, q, k, v, g, "f32", False, 1e-6, chunk)
        for a, b in zip(got, ref):
            assert rowerr(a.reshape(2, 333, -1), b.reshape(2, 333, -1)) < 1e-5, chunk


def test_backward_mid_workload_sampled(hla):
    """The mid workload's shapes (B8 H16 n2048 d64 bf16, chunk 64); the oracle
    checks every position of sampled heads."""
    w = hla_inputs.WORKLOADS["mid_bf16"]
    errs = _check(hla, w.B, w.H, w.n, w.d, w.dv, w.chunk, w.dtype, False, hla_inputs.EPS, seed=w.seed,
                  heads=[0, 65, w.BH - 1])
    print("\nbackward on mid_bf16 sampled heads: dq %s; dk %s; dv %s" % tuple(_check.stats))


# ----------------------------------------------------------------------------
# the tensor-core kernel (bf16 tokens, d = dv = 64, plain output)
# ----------------------------------------------------------------------------

TC_SHAPES = [(1, 1, 1), (1, 2, 127), (1, 2, 128), (2, 1, 129), (1, 3, 300), (1, 2, 700)]


@pytest.mark.parametrize("shape", TC_SHAPES, ids=lambda s: "B%dH%dn%d" % s)
def test_backward_tensor_core_path(hla, shape, monkeypatch):
    """Every head against the oracle, and against the CUDA-core kernels on the same inputs."""
    B, H, n = shape
    assert hla.hla2_backward_path(B, H, n, 64, 64) == 1
    q, k, v = hla_inputs.make_qkv(B, H, n, 64, 64, seed=6000 + n, dtype="bf16")
    g = hla_inputs.round_to(np.random.default_rng(6001 + n).standard_normal((B, H, n, 64)), "bf16")
    got = _grads(hla, q, k, v, g, "bf16", False, hla_inputs.EPS, 64)
    flat = lambda x: x.reshape(B * H, n, -1)
    ref = oracle.hla2_backward(flat(q), flat(k), flat(v), flat(g), masked=True, ckpt=64, nthreads=8)
    for name, a, b in zip(("dq", "dk", "dv"), got, ref):
        assert rowerr(flat(a), b) < TOL["bf16"], (name, rowerr(flat(a), b))
    monkeypatch.setenv("HLA_DISABLE_FUSED", "1")
    assert hla.hla2_backward_path(B, H, n, 64, 64) == 0
    cc = _grads(hla, q, k, v, g, "bf16", False, hla_inputs.EPS, 64)
    for name, a, b in zip(("dq", "dk", "dv"), got, cc):
        assert rowerr(flat(a), flat(b)) < TOL["bf16"], (name, rowerr(flat(a), flat(b)))


def test_backward_tensor_core_more_heads_than_sms(hla):
    """200 heads: a CTA takes several heads in turn (both sweeps restart per head)."""
    B, H, n = 2, 100, 260
    errs = _check(hla, B, H, n, 64, 64, 64, "bf16", False, hla_inputs.EPS, seed=6100, heads=[0, 1, 151, 152, 199])
    print("\nbackward, 200 heads: dq %.3g dk %.3g dv %.3g" % tuple(errs))


def test_backward_tensor_core_deterministic(hla):
    q, k, v = hla_inputs.make_qkv(1, 2, 500, 64, 64, seed=6200, dtype="bf16")
    g = hla_inputs.round_to(np.random.default_rng(6201).standard_normal((1, 2, 500, 64)), "bf16")
    a = _grads(hla, q, k, v, g, "bf16", False, hla_inputs.EPS, 64)
    b = _grads(hla, q, k, v, g, "bf16", False, hla_inputs.EPS, 64)
    for x, y in zip(a, b):
        assert np.array_equal(x, y)
