"""Third-order HLA on the GPU (through the C ABI) against the fp64 oracle
(Algorithm 3 at gamma = 1; unmasked factorisation of Sec. 7.1).  Calls without
state_out take the chunk-parallel path (Theorem 4), calls with it the serial
kernel."""
import numpy as np
import pytest
import torch

import hla_inputs
import oracle
from parity import check_normalized

pytestmark = pytest.mark.gpu
DEV = "cuda:0"


@pytest.fixture(scope="module")
def hla():
    from paper_2510_27258_gb300 import build
    build.build()
    from paper_2510_27258_gb300 import hla as binding
    return binding


def rowerr(got, ref):
    nrm = np.linalg.norm(ref, axis=-1, keepdims=True)
    return float(np.max(np.abs(got - ref) / np.maximum(nrm, 1e-30)))


def run(hla, q, k, v, dtype, masked, normalized, state_in=None, want_state=False, chunk=32):
    B, H, n, d = q.shape
    dv = v.shape[-1]
    tq, tk, tv = (hla_inputs.as_torch(x, dtype, DEV) for x in (q, k, v))
    sin = None if state_in is None else torch.from_numpy(np.ascontiguousarray(state_in, np.float32)).to(DEV)
    sout = torch.zeros((B, H, hla.hla3_state_floats(d, dv)), dtype=torch.float32, device=DEV) if want_state else None
    out = hla.hla3_forward(tq, tk, tv, masked=masked, normalized=normalized, eps=hla_inputs.EPS, chunk=chunk,
                           state_in=sin, state_out=sout)
    torch.cuda.synchronize()
    o = out.float().cpu().numpy().reshape(B * H, n, dv)
    return (o, sout.cpu().numpy().reshape(B * H, -1)) if want_state else o


@pytest.mark.parametrize("d,dv", [(16, 16), (32, 32), (64, 32), (128, 128)])
@pytest.mark.parametrize("masked,normalized", [(True, False), (True, True), (False, False)])
def test_hla3_small(hla, d, dv, masked, normalized):
    B, H, n = 1, 2, 70
    q, k, v = hla_inputs.make_qkv(B, H, n, d, dv, seed=d * 3 + dv, dtype="f32")
    got = run(hla, q, k, v, "f32", masked, normalized)
    ref = oracle.hla3_serial(q.reshape(B * H, n, d), k.reshape(B * H, n, d), v.reshape(B * H, n, dv), masked=masked,
                             normalized=normalized, eps=hla_inputs.EPS)
    assert rowerr(got, ref) < 1e-4


def test_hla3_state_handoff(hla):
    B, H, n, d, dv = 1, 2, 40, 32, 32
    q, k, v = hla_inputs.make_qkv(B, H, n, d, dv, seed=5, dtype="f32")
    o1, st = run(hla, q[:, :, :25], k[:, :, :25], v[:, :, :25], "f32", True, False, want_state=True)
    o2 = run(hla, q[:, :, 25:], k[:, :, 25:], v[:, :, 25:], "f32", True, False, state_in=st)
    ref = oracle.hla3_serial(q.reshape(B * H, n, d), k.reshape(B * H, n, d), v.reshape(B * H, n, dv), masked=True)
    assert rowerr(np.concatenate([o1, o2], axis=1), ref) < 1e-4


def test_hla3_workload_sampled(hla):
    w = hla_inputs.WORKLOADS["hla3_f32"]
    q, k, v = hla_inputs.make_workload(w)
    got = run(hla, q, k, v, w.dtype, w.masked, w.normalized)
    heads = [0, w.BH - 1]
    qf, kf, vf = (x.reshape(w.BH, w.n, -1)[heads] for x in (q, k, v))
    ref = oracle.hla3_serial(qf, kf, vf, masked=True, normalized=w.normalized, eps=hla_inputs.EPS, nthreads=2)
    assert rowerr(got[heads], ref) < 1e-4


@pytest.mark.parametrize("n,d,dv,chunk", [(1, 16, 16, 32), (33, 32, 32, 32), (257, 16, 32, 7), (130, 64, 64, 100),
                                          (200, 128, 64, 128), (97, 32, 16, 1)])
@pytest.mark.parametrize("masked,normalized", [(True, False), (True, True), (False, False), (False, True)])
def test_hla3_chunked_shapes(hla, n, d, dv, chunk, masked, normalized):
    """Chunk-parallel path: ragged lengths, chunk sizes 1..128 (internal chunk capped at 64 / 32)."""
    B, H = 1, 2
    q, k, v = hla_inputs.make_qkv(B, H, n, d, dv, seed=n + d + chunk, dtype="f32")
    num = run(hla, q, k, v, "f32", masked, False, chunk=chunk)
    num_ref, den_ref = oracle.hla3_serial(q.reshape(B * H, n, d), k.reshape(B * H, n, d), v.reshape(B * H, n, dv),
                                          masked=masked, normalized=False, return_den=True)
    if not normalized:
        assert rowerr(num, num_ref) < 1e-4
        return
    # the ratio is ill-conditioned where the denominator nears zero: numerator on every row,
    # the ratio on rows fp32 can resolve, the implied denominator bounded on every row
    o = run(hla, q, k, v, "f32", masked, True, chunk=chunk)
    check_normalized(o, num, num_ref, den_ref, hla_inputs.EPS, 1e-4)


@pytest.mark.parametrize("masked", [True, False])
def test_hla3_chunked_initial_state(hla, masked):
    """state_in on the chunk-parallel path (state_out computed by the serial kernel on the prefix)."""
    B, H, n, d, dv = 1, 3, 150, 32, 32
    q, k, v = hla_inputs.make_qkv(B, H, n, d, dv, seed=21, dtype="f32")
    _, st = run(hla, q[:, :, :60], k[:, :, :60], v[:, :, :60], "f32", masked, False, want_state=True)
    o2 = run(hla, q[:, :, 60:], k[:, :, 60:], v[:, :, 60:], "f32", masked, True, state_in=st)
    ref = oracle.hla3_serial(q.reshape(B * H, n, d), k.reshape(B * H, n, d), v.reshape(B * H, n, dv), masked=masked,
                             normalized=True, eps=hla_inputs.EPS)
    assert rowerr(o2, ref[:, 60:]) < 1e-4


def test_hla3_chunked_bf16(hla):
    B, H, n, d, dv = 2, 2, 300, 32, 32
    q, k, v = hla_inputs.make_qkv(B, H, n, d, dv, seed=22, dtype="bf16")
    got = run(hla, q, k, v, "bf16", True, False, chunk=32)
    ref = oracle.hla3_serial(q.reshape(B * H, n, d), k.reshape(B * H, n, d), v.reshape(B * H, n, dv), masked=True)
    assert rowerr(got, ref) < 2e-2


def test_hla3_chunked_equals_serial_closely(hla):
    """The two CUDA third-order paths on the same inputs (serial: asked for state_out)."""
    B, H, n, d, dv = 1, 4, 500, 32, 32
    q, k, v = hla_inputs.make_qkv(B, H, n, d, dv, seed=23, dtype="f32")
    a = run(hla, q, k, v, "f32", True, False)
    b, _ = run(hla, q, k, v, "f32", True, False, want_state=True)
    assert rowerr(a, b) < 1e-4


def test_hla3_chunked_deterministic(hla):
    q, k, v = hla_inputs.make_qkv(2, 2, 400, 32, 32, seed=24, dtype="f32")
    assert np.array_equal(run(hla, q, k, v, "f32", True, True), run(hla, q, k, v, "f32", True, True))
