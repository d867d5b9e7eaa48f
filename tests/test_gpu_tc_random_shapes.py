"""Randomised shapes for the tensor-core paths that have no fp32 fallback inside them:
the third-order forward (fp32, d = dv = 32), the backward (bf16, d = dv = 64) and the
AHLA forward (bf16, d and dv in {64, 128}).  Lengths around tile boundaries and head
counts around the SM count, drawn from a fixed seed; every head against the oracle."""
import numpy as np
import pytest
import torch

import hla_inputs
import oracle
from parity import TOL, rowerr

pytestmark = pytest.mark.gpu
DEV = "cuda:0"
# tile boundaries (128 tokens) and their neighbours, then lengths drawn from a fixed seed
LENGTHS = [1, 127, 128, 129, 257] + sorted(int(x) for x in np.random.default_rng(20261202).integers(2, 2049, size=5))
HEADS = [(1, 1), (1, 3), (2, 5), (3, 7)]


@pytest.fixture(scope="module")
def hla():
    from paper_2510_27258_gb300 import build
    build.build()
    from paper_2510_27258_gb300 import hla as binding
    return binding


@pytest.mark.parametrize("n", LENGTHS)
@pytest.mark.parametrize("bh", HEADS, ids=lambda x: "B%dH%d" % x)
def test_third_order_tensor_cores(hla, n, bh, monkeypatch):
    B, H = bh
    seg = 1 + (n + 7 * H) % 4
    monkeypatch.setenv("HLA3_SEGMENT_TILES", str(seg))  # segments of 1..4 tiles
    assert hla.hla3_forward_path(B, H, n, 32, 32)[0] == 2
    q, k, v = hla_inputs.make_qkv(B, H, n, 32, 32, seed=7000 + n + 31 * H, dtype="f32")
    out = hla.hla3_forward(*(hla_inputs.as_torch(x, "f32", DEV) for x in (q, k, v)), masked=True, chunk=32)
    torch.cuda.synchronize()
    ref = oracle.hla3_serial(q.reshape(B * H, n, 32), k.reshape(B * H, n, 32), v.reshape(B * H, n, 32), masked=True,
                             nthreads=8)
    assert rowerr(out.cpu().numpy().reshape(B * H, n, 32), ref) < TOL["f32"]


@pytest.mark.parametrize("n", LENGTHS)
@pytest.mark.parametrize("bh", HEADS, ids=lambda x: "B%dH%d" % x)
def test_backward_tensor_cores(hla, n, bh):
    B, H = bh
    assert hla.hla2_backward_path(B, H, n, 64, 64) == 1
    q, k, v = hla_inputs.make_qkv(B, H, n, 64, 64, seed=8000 + n + 31 * H, dtype="bf16")
    g = hla_inputs.round_to(np.random.default_rng(8001 + n).standard_normal((B, H, n, 64)), "bf16")
    got = hla.hla2_backward(*(hla_inputs.as_torch(x, "bf16", DEV) for x in (q, k, v, g)), chunk=64)
    torch.cuda.synchronize()
    flat = lambda x: x.reshape(B * H, n, -1)
    ref = oracle.hla2_backward(flat(q), flat(k), flat(v), flat(g), masked=True, nthreads=8)
    for name, a, b in zip(("dq", "dk", "dv"), got, ref):
        e = rowerr(flat(a.float().cpu().numpy()), b)
        assert e < TOL["bf16"], (name, e)


@pytest.mark.parametrize("n", LENGTHS)
@pytest.mark.parametrize("dims", [(64, 64), (128, 64), (64, 128), (128, 128)], ids=lambda x: "d%ddv%d" % x)
def test_ahla_tensor_cores(hla, n, dims):
    d, dv = dims
    B, H = 1, 3
    assert hla.ahla_forward_path(B, H, n, d, dv) == 1
    q, k, v = hla_inputs.make_qkv(B, H, n, d, dv, seed=9000 + n + d + dv, dtype="bf16")
    out = hla.ahla_forward(*(hla_inputs.as_torch(x, "bf16", DEV) for x in (q, k, v)), chunk=64)
    torch.cuda.synchronize()
    ref = oracle.ahla_serial(q.reshape(B * H, n, d), k.reshape(B * H, n, d), v.reshape(B * H, n, dv), nthreads=3)
    assert rowerr(out.float().cpu().numpy().reshape(B * H, n, dv), ref) < TOL["bf16"]


# ---------------------------------------------------------------------------------------------
# the fused second-order forward (bf16, masked; plain and ratio-normalised; d, dv in {64, 128}),
# at the same lengths and head counts, with segment lengths of 1..4 tiles or the planner's
# ---------------------------------------------------------------------------------------------

def _fused(hla, q, k, v, normalized):
    tq, tk, tv = (hla_inputs.as_torch(x, "bf16", DEV) for x in (q, k, v))
    ws = hla.alloc_workspace(hla.hla2_workspace_bytes(*q.shape, v.shape[-1], 128, torch.bfloat16), DEV)
    out = hla.hla2_forward(tq, tk, tv, masked=True, normalized=normalized, eps=hla_inputs.EPS, chunk=128,
                           workspace=ws)
    torch.cuda.synchronize()
    assert hla.hla_poll_error(ws) == 0
    B, H, n, _ = q.shape
    return out.float().cpu().numpy().reshape(B * H, n, -1)


@pytest.mark.parametrize("n", LENGTHS)
@pytest.mark.parametrize("bh", HEADS, ids=lambda x: "B%dH%d" % x)
@pytest.mark.parametrize("dims", [(64, 64), (128, 128), (64, 128)], ids=lambda x: "d%ddv%d" % x)
def test_fused_forward(hla, n, bh, dims, monkeypatch):
    from parity import check_normalized
    B, H = bh
    d, dv = dims
    seg = (n + 3 * H + d) % 5  # 0: the planner's segments, else segments of 1..4 tiles
    if seg:
        monkeypatch.setenv("HLA_FUSED_SEGMENT_TILES", str(seg))
    assert hla.hla2_forward_path(B, H, n, d, dv, chunk=128)[0] == 1
    q, k, v = hla_inputs.make_qkv(B, H, n, d, dv, seed=11000 + n + 17 * H + d + dv, dtype="bf16")
    flat = lambda x: x.reshape(B * H, n, -1)
    num_ref, den_ref = oracle.hla2_serial(flat(q), flat(k), flat(v), masked=True, normalized=False, return_den=True,
                                          nthreads=8)
    num = _fused(hla, q, k, v, False)
    assert rowerr(num, num_ref) < TOL["bf16"], rowerr(num, num_ref)
    o = _fused(hla, q, k, v, True)
    check_normalized(o, num, num_ref, den_ref, hla_inputs.EPS, TOL["bf16"])


@pytest.mark.parametrize("n", LENGTHS)
@pytest.mark.parametrize("bh", HEADS, ids=lambda x: "B%dH%d" % x)
@pytest.mark.parametrize("dims", [(64, 64), (128, 128)], ids=lambda x: "d%ddv%d" % x)
def test_fused_forward_unmasked(hla, n, bh, dims):
    """The unmasked operator: the plain output on the fused kernel (one segment per head), the
    ratio-normalised one on the fp32 path."""
    from parity import check_normalized
    B, H = bh
    d, dv = dims
    assert hla.hla2_forward_path(B, H, n, d, dv, masked=False, chunk=128)[0] == 1
    q, k, v = hla_inputs.make_qkv(B, H, n, d, dv, seed=12000 + n + 17 * H + d, dtype="bf16")
    flat = lambda x: x.reshape(B * H, n, -1)
    num_ref, den_ref = oracle.hla2_serial(flat(q), flat(k), flat(v), masked=False, normalized=False,
                                          return_den=True, nthreads=8)

    def fused(normalized):
        tq, tk, tv = (hla_inputs.as_torch(x, "bf16", DEV) for x in (q, k, v))
        ws = hla.alloc_workspace(hla.hla2_workspace_bytes(B, H, n, d, dv, 128, torch.bfloat16), DEV)
        out = hla.hla2_forward(tq, tk, tv, masked=False, normalized=normalized, eps=hla_inputs.EPS, chunk=128,
                               workspace=ws)
        torch.cuda.synchronize()
        assert hla.hla_poll_error(ws) == 0
        return out.float().cpu().numpy().reshape(B * H, n, -1)

    num = fused(False)
    assert rowerr(num, num_ref) < TOL["bf16"], rowerr(num, num_ref)
    check_normalized(fused(True), num, num_ref, den_ref, hla_inputs.EPS, TOL["bf16"])
