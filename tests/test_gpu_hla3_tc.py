"""The tensor-core path of the masked third-order forward (fp32 tokens, d = dv = 32,
plain output, no states), through the C ABI, against the fp64 oracle (Algorithm 3
at gamma = 1) and against the chunk-parallel CUDA-core kernels on the same inputs.
Segments of a head run on different SMs; HLA3_SEGMENT_TILES forces their length
so that the pre-pass sums, the segment starts and the fix-up all run."""
import numpy as np
import pytest
import torch

import hla_inputs
import oracle
from parity import rowerr_stats

pytestmark = pytest.mark.gpu
DEV = "cuda:0"
TOL = 1e-4


@pytest.fixture(scope="module")
def hla():
    from paper_2510_27258_gb300 import build
    build.build()
    from paper_2510_27258_gb300 import hla as binding
    return binding


def rowerr(got, ref):
    nrm = np.linalg.norm(ref, axis=-1, keepdims=True)
    return float(np.max(np.abs(got - ref) / np.maximum(nrm, 1e-30)))


def run(hla, q, k, v):
    B, H, n, d = q.shape
    tq, tk, tv = (hla_inputs.as_torch(x, "f32", DEV) for x in (q, k, v))
    out = hla.hla3_forward(tq, tk, tv, masked=True, normalized=False, chunk=32)
    torch.cuda.synchronize()
    return out.cpu().numpy().reshape(B * H, n, -1)


def ref(q, k, v, heads=None):
    B, H, n, d = q.shape
    qf, kf, vf = (x.reshape(B * H, n, -1) for x in (q, k, v))
    if heads is not None:
        qf, kf, vf = qf[heads], kf[heads], vf[heads]
    return oracle.hla3_serial(qf, kf, vf, masked=True, normalized=False, nthreads=8)


SHAPES = [(1, 1, 1), (1, 2, 127), (1, 2, 128), (2, 1, 129), (1, 3, 300), (1, 2, 1000)]


@pytest.mark.parametrize("shape", SHAPES, ids=lambda s: "B%dH%dn%d" % s)
def test_tc_path_against_oracle_and_cuda_cores(hla, shape, monkeypatch):
    B, H, n = shape
    assert hla.hla3_forward_path(B, H, n, 32, 32)[0] == 2
    q, k, v = hla_inputs.make_qkv(B, H, n, 32, 32, seed=5000 + n, dtype="f32")
    r = ref(q, k, v)
    got = run(hla, q, k, v)
    err = rowerr(got, r)
    assert err < TOL, err
    monkeypatch.setenv("HLA_DISABLE_FUSED", "1")
    assert hla.hla3_forward_path(B, H, n, 32, 32)[0] == 1
    assert rowerr(run(hla, q, k, v), r) < TOL


@pytest.mark.parametrize("seg_tiles", [1, 2, 3, 6])
def test_tc_segments(hla, seg_tiles, monkeypatch):
    """A head of 6 tiles (the last ragged) cut into segments of 1, 2, 3 and 6 tiles."""
    monkeypatch.setenv("HLA3_SEGMENT_TILES", str(seg_tiles))
    B, H, n = 1, 2, 700
    q, k, v = hla_inputs.make_qkv(B, H, n, 32, 32, seed=5100, dtype="f32")
    expected_launches = 1 if seg_tiles >= 6 else 3
    assert hla.hla3_forward_path(B, H, n, 32, 32) == (2, expected_launches)
    got = run(hla, q, k, v)
    err = rowerr(got, ref(q, k, v))
    print("\nsegments of %d tiles: max row error %.3g" % (seg_tiles, err))
    assert err < TOL, err


def test_tc_more_heads_than_sms(hla):
    """200 heads of 3 tiles: one segment per head, CTAs take several heads in turn."""
    B, H, n = 2, 100, 260
    q, k, v = hla_inputs.make_qkv(B, H, n, 32, 32, seed=5200, dtype="f32")
    got = run(hla, q, k, v)
    heads = [0, 1, 151, 152, 153, 199]
    assert rowerr(got[heads], ref(q, k, v, heads)) < TOL


def test_tc_causality_and_determinism(hla):
    B, H, n, t = 1, 2, 600, 333
    q, k, v = hla_inputs.make_qkv(B, H, n, 32, 32, seed=5300, dtype="f32")
    a = run(hla, q, k, v)
    assert np.array_equal(a, run(hla, q, k, v))
    q2, k2, v2 = q.copy(), k.copy(), v.copy()
    rng = np.random.default_rng(9)
    for x in (q2, k2, v2):
        x[:, :, t + 1:] = rng.standard_normal(x[:, :, t + 1:].shape).astype(np.float32)
    b = run(hla, q2, k2, v2)
    assert np.array_equal(a[:, : t + 1], b[:, : t + 1])
    assert not np.array_equal(a[:, t + 1:], b[:, t + 1:])


def test_tc_workload_full_size_sampled(hla, monkeypatch):
    """The hla3_f32 workload (B4 H8 n4096 d32, the configuration the bench times), four
    heads against the oracle; every head against the CUDA-core kernels."""
    w = hla_inputs.WORKLOADS["hla3_f32"]
    assert hla.hla3_forward_path(w.B, w.H, w.n, w.d, w.dv)[0] == 2
    q, k, v = hla_inputs.make_workload(w)
    got = run(hla, q, k, v)
    heads = [0, 9, 22, w.BH - 1]
    err = rowerr(got[heads], ref(q, k, v, heads))
    monkeypatch.setenv("HLA_DISABLE_FUSED", "1")
    cuda_cores = run(hla, q, k, v)
    err_all = rowerr(got, cuda_cores)
    print("\nhla3_f32 heads %s: row error %s against the oracle; all heads %.3g against the CUDA-core path"
          % (heads, rowerr_stats(got[heads], ref(q, k, v, heads))[0], err_all))
    assert err < TOL, err
    assert err_all < TOL, err_all
