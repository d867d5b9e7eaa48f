"""hla2_forward_noalloc, the entry point for callers that cannot allocate device
memory (they cannot call cudaMalloc or hand over a workspace, e.g. code running
under someone else's memory pool or budget).  Its outputs must match the fp64
oracle within the bf16 bar and be bit-identical to hla2_forward with a caller
workspace (the same kernel on the same inputs), on consecutive calls that reuse
the library's own scratch array, also when a call of another shape has left
its contents there.  Kept in the last test file so that a run stopping at its
first failure has already run everything else."""
import ctypes

import numpy as np
import pytest
import torch

import hla_inputs
import oracle
from parity import TOL, check_normalized, rowerr

pytestmark = pytest.mark.gpu
DEV = "cuda:0"


@pytest.fixture(scope="module")
def hla():
    from paper_2510_27258_gb300 import build
    build.build()
    from paper_2510_27258_gb300 import hla as binding
    return binding


def _noalloc(hla, q, k, v, out, normalized, state_in=None):
    """The C entry point through ctypes (no Python wrapper)."""
    B, H, n, d = q.shape
    L = hla.lib()
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    return L.hla2_forward_noalloc(ctypes.c_void_p(q.data_ptr()), ctypes.c_void_p(k.data_ptr()),
                                  ctypes.c_void_p(v.data_ptr()), ctypes.c_void_p(out.data_ptr()), hla.HLA_BF16,
                                  B, H, n, d, v.shape[-1], 1, int(normalized), ctypes.c_float(hla_inputs.EPS), 128,
                                  None if state_in is None else ctypes.c_void_p(state_in.data_ptr()), stream)


def _foreign_call(hla):
    """A call of another shape, so that the scratch holds its counters, ring and denominators."""
    q, k, v = hla_inputs.make_qkv(1, 3, 900, 64, 64, seed=5, dtype="bf16")
    tq, tk, tv = (hla_inputs.as_torch(x, "bf16", DEV) for x in (q, k, v))
    out = torch.empty((1, 3, 900, 64), dtype=torch.bfloat16, device=DEV)
    assert _noalloc(hla, tq, tk, tv, out, True) == hla.HLA_OK, hla.lib().hla_last_error()


def _check_oracle(q, k, v, got, normalized, state_in=None):
    B, H, n, d = q.shape
    dv = v.shape[-1]
    qf, kf, vf = q.reshape(B * H, n, d), k.reshape(B * H, n, d), v.reshape(B * H, n, dv)
    sin = None if state_in is None else state_in.reshape(B * H, -1).astype(np.float64)
    num, den = oracle.hla2_serial(qf, kf, vf, masked=True, normalized=False, eps=hla_inputs.EPS, state_in=sin,
                                  return_den=True, nthreads=4)
    got = got.reshape(B * H, n, dv)
    if not normalized:
        assert rowerr(got, num) < TOL["bf16"]
        return None
    return num, den


@pytest.mark.parametrize("d", [64, 128])
@pytest.mark.parametrize("normalized", [False, True])
def test_noalloc_matches_oracle_and_workspace_forward_on_two_calls(hla, d, normalized):
    B, H, n = 1, 4, 1000
    q, k, v = hla_inputs.make_qkv(B, H, n, d, d, seed=77 + d, dtype="bf16")
    tq, tk, tv = (hla_inputs.as_torch(x, "bf16", DEV) for x in (q, k, v))
    ref = hla.hla2_forward(tq, tk, tv, masked=True, normalized=normalized, eps=hla_inputs.EPS, chunk=128)
    num_gpu = hla.hla2_forward(tq, tk, tv, masked=True, normalized=False, eps=hla_inputs.EPS, chunk=128)
    torch.cuda.synchronize()
    ref = ref.float().cpu().numpy()
    num_gpu = num_gpu.float().cpu().numpy().reshape(B * H, n, d)
    for call in range(2):  # the second call reuses the scratch left by a call of another shape
        if call == 1:
            _foreign_call(hla)
        out = torch.zeros((B, H, n, d), dtype=torch.bfloat16, device=DEV)
        assert _noalloc(hla, tq, tk, tv, out, normalized) == hla.HLA_OK, hla.lib().hla_last_error()
        assert hla.hla_poll_error_noalloc() == hla.HLA_OK
        got = out.float().cpu().numpy()
        assert np.array_equal(got, ref), call
        nd = _check_oracle(q, k, v, got, normalized)
        if nd is not None:
            check_normalized(got.reshape(B * H, n, d), num_gpu, nd[0], nd[1], hla_inputs.EPS, TOL["bf16"])


def test_noalloc_python_wrapper_with_initial_state(hla):
    """The Python wrapper with an initial state (d = dv = 128), twice in a row."""
    B, H, n, d = 1, 2, 700, 128
    pq, pk, pv = hla_inputs.make_qkv(B, H, 300, d, d, seed=31, dtype="bf16")
    _, st0 = oracle.hla2_serial(pq.reshape(B * H, 300, d), pk.reshape(B * H, 300, d), pv.reshape(B * H, 300, d),
                                masked=True, return_state=True)
    st0 = st0.astype(np.float32)
    q, k, v = hla_inputs.make_qkv(B, H, n, d, d, seed=32, dtype="bf16")
    tq, tk, tv = (hla_inputs.as_torch(x, "bf16", DEV) for x in (q, k, v))
    tst = torch.from_numpy(st0).to(DEV)
    ref = hla.hla2_forward(tq, tk, tv, masked=True, normalized=False, eps=hla_inputs.EPS, chunk=128, state_in=tst)
    torch.cuda.synchronize()
    ref = ref.float().cpu().numpy()
    for _ in range(2):
        got = hla.hla2_forward_noalloc(tq, tk, tv, masked=True, normalized=False, eps=hla_inputs.EPS, chunk=128,
                                       state_in=tst)
        torch.cuda.synchronize()
        got = got.float().cpu().numpy()
        assert np.array_equal(got, ref)
        _check_oracle(q, k, v, got, False, state_in=st0)


def test_noalloc_wait_timeout_is_reported(hla, monkeypatch):
    """A segment that never publishes its S prefix (injected on the host side, as in
    the fused tests): the next segment's 20 ms wait runs out, the call finishes,
    hla_poll_error_noalloc reports HLA_ERR_TIMEOUT and clears it, and the next call
    on the same scratch is correct."""
    monkeypatch.setenv("HLA_FUSED_SEGMENT_TILES", "1")
    monkeypatch.setenv("HLA_TEST_WAIT_NS", "20000000")
    monkeypatch.setenv("HLA_TEST_SKIP_PUBLISH_ITEM", "0")
    B, H, n, d = 1, 1, 512, 128
    q, k, v = hla_inputs.make_qkv(B, H, n, d, d, seed=51, dtype="bf16")
    tq, tk, tv = (hla_inputs.as_torch(x, "bf16", DEV) for x in (q, k, v))
    out = torch.zeros((B, H, n, d), dtype=torch.bfloat16, device=DEV)
    assert _noalloc(hla, tq, tk, tv, out, False) == hla.HLA_OK
    assert hla.hla_poll_error_noalloc() == hla.HLA_ERR_TIMEOUT
    assert hla.hla_poll_error_noalloc() == hla.HLA_OK  # cleared
    monkeypatch.delenv("HLA_TEST_SKIP_PUBLISH_ITEM")
    assert _noalloc(hla, tq, tk, tv, out, False) == hla.HLA_OK
    assert hla.hla_poll_error_noalloc() == hla.HLA_OK
    _check_oracle(q, k, v, out.float().cpu().numpy(), False)


def test_noalloc_empty_problem_is_ok(hla):
    t = torch.zeros((1, 0, 256, 128), dtype=torch.bfloat16, device=DEV)
    assert _noalloc(hla, t, t, t, t, False) == hla.HLA_OK
    assert hla.lib().hla_last_error() == b""


def test_noalloc_rejects_sizes_beyond_its_scratch(hla):
    # 128 heads need about 33 MiB of scratch (> 16 MiB): refused before any launch
    B, H, n, d = 1, 128, 256, 128
    t = torch.zeros((B, H, n, d), dtype=torch.bfloat16, device=DEV)
    assert _noalloc(hla, t, t, t, t, False) == hla.HLA_ERR_WORKSPACE
    assert b"scratch" in hla.lib().hla_last_error()
