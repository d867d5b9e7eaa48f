"""The C ABI without a GPU: the library loads, exports every function that
include/hla.h declares, and host-side argument checks return their error codes
before anything is launched."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "hla.h")


@pytest.fixture(scope="module")
def L():
    from paper_2510_27258_gb300 import build, hla
    build.build()
    return hla.lib()


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b((?:hla|ahla)\w+)\s*\(", text)))


def test_header_declares_expected_entry_points():
    from paper_2510_27258_gb300 import hla
    assert declared_functions() == sorted(hla.EXPORTS)


def test_library_exports_every_declared_symbol(L):
    for name in declared_functions():
        assert hasattr(L, name), name
        assert ctypes.cast(getattr(L, name), ctypes.c_void_p).value


def test_status_strings(L):
    from paper_2510_27258_gb300 import hla
    names = [hla.hla_status_string(c) for c in range(6)]
    assert names == ["HLA_OK", "HLA_ERR_INVALID_ARGUMENT", "HLA_ERR_UNSUPPORTED", "HLA_ERR_CUDA",
                     "HLA_ERR_TIMEOUT", "HLA_ERR_WORKSPACE"]


def test_state_sizes(L):
    assert L.hla2_state_floats(128, 128) == 128 * 128 + 2 * 128 * 128 + 2 * 128
    assert L.hla2_state_floats(16, 32) == 16 * 16 + 2 * 16 * 32 + 32
    assert L.hla3_state_floats(32, 32) == 2 * 32 * 32 + 4 * 32 * 32 + 4 * 32
    assert L.hla2_workspace_bytes(1, 1, 64, 16, 16, 16, 0) > 0
    assert L.hla2_workspace_bytes(1, 1, 64, 48, 16, 16, 0) == 0   # unsupported d
    assert L.hla2_workspace_bytes(1, 1, 64, 16, 16, 256, 0) == 0  # unsupported chunk
    assert L.hla2_workspace_bytes(1, 1, 64, 16, 16, 16, 7) == 0   # unknown dtype
    assert L.hla2_workspace_bytes(2, 16, 16384, 128, 128, 128, 1) % 256 == 0


def _fwd(L, q=16, k=16, v=16, out=16, dt=1, B=1, H=1, n=64, d=16, dv=16, masked=1, normalized=0, eps=1e-6,
         chunk=16, st_in=None, st_out=None, ws=256, ws_bytes=1 << 30, fn="hla2_forward"):
    return getattr(L, fn)(q, k, v, out, dt, B, H, n, d, dv, masked, normalized, ctypes.c_float(eps), chunk, st_in,
                          st_out, ws, ws_bytes, None)


def test_forward_argument_errors_return_before_launch(L):
    from paper_2510_27258_gb300 import hla as H
    # none of these reach a CUDA call: there is no GPU here
    assert _fwd(L, q=None) == H.HLA_ERR_INVALID_ARGUMENT
    assert _fwd(L, q=8) == H.HLA_ERR_INVALID_ARGUMENT                      # misaligned
    assert _fwd(L, dt=5) == H.HLA_ERR_INVALID_ARGUMENT
    assert _fwd(L, B=-1) == H.HLA_ERR_INVALID_ARGUMENT
    assert _fwd(L, n=-3) == H.HLA_ERR_INVALID_ARGUMENT
    assert _fwd(L, masked=2) == H.HLA_ERR_INVALID_ARGUMENT
    assert _fwd(L, eps=float("nan")) == H.HLA_ERR_INVALID_ARGUMENT
    assert _fwd(L, d=48) == H.HLA_ERR_UNSUPPORTED
    assert _fwd(L, dv=256) == H.HLA_ERR_UNSUPPORTED
    assert _fwd(L, chunk=0) == H.HLA_ERR_INVALID_ARGUMENT
    assert _fwd(L, chunk=129) == H.HLA_ERR_UNSUPPORTED
    assert _fwd(L, ws=None) == H.HLA_ERR_WORKSPACE
    assert _fwd(L, ws_bytes=100) == H.HLA_ERR_WORKSPACE
    assert _fwd(L, ws=256 + 16) == H.HLA_ERR_INVALID_ARGUMENT              # workspace alignment
    assert _fwd(L, st_in=4) == H.HLA_ERR_INVALID_ARGUMENT
    assert "16-byte" in L.hla_last_error().decode()
    assert _fwd(L, fn="hla3_forward", d=24) == H.HLA_ERR_UNSUPPORTED
    # empty problems succeed without touching the device
    assert _fwd(L, B=0) == H.HLA_OK
    assert _fwd(L, H=0, q=None, k=None, v=None, out=None) == H.HLA_OK


def test_step_argument_errors(L):
    from paper_2510_27258_gb300 import hla as H
    f = ctypes.c_float(0.0)
    assert L.hla2_step(16, 16, 16, 16, 1, 1, 1, 128, 128, 1, 0, f, None, None) == H.HLA_ERR_INVALID_ARGUMENT
    assert L.hla2_step(16, 16, 16, 16, 1, 1, 1, 100, 128, 1, 0, f, 16, None) == H.HLA_ERR_UNSUPPORTED
    assert L.hla2_step(16, 16, 16, 16, 1, 0, 1, 128, 128, 1, 0, f, 16, None) == H.HLA_OK


def test_poll_error_null_workspace(L):
    from paper_2510_27258_gb300 import hla as H
    assert L.hla_poll_error(None, None) == H.HLA_ERR_INVALID_ARGUMENT


def test_sde_sizes_and_argument_errors(L):
    from paper_2510_27258_gb300 import hla as H
    assert L.hla2_sde_state_floats(128, 128) == 128 * 128 + 128 * 128 + 128
    assert L.hla2_sde_state_floats(16, 32) == 16 * 16 + 16 * 32 + 16
    f = ctypes.c_float(0.0)
    # conversion: null, misaligned, unsupported head size, overlapping buffers, empty problem
    assert L.hla2_state_to_sde(None, 4096, 1, 1, 16, 16, None) == H.HLA_ERR_INVALID_ARGUMENT
    assert L.hla2_state_to_sde(4100, 1 << 20, 1, 1, 16, 16, None) == H.HLA_ERR_INVALID_ARGUMENT
    assert L.hla2_state_to_sde(4096, 1 << 20, 1, 1, 24, 16, None) == H.HLA_ERR_UNSUPPORTED
    assert L.hla2_state_to_sde(4096, 4096 + 64, 1, 1, 16, 16, None) == H.HLA_ERR_INVALID_ARGUMENT
    assert "overlap" in L.hla_last_error().decode()
    assert L.hla2_state_to_sde(4096, 4096, 0, 1, 16, 16, None) == H.HLA_OK
    # decode step on (S, D, e): as hla2_step
    assert L.hla2_step_sde(16, 16, 16, 16, 1, 1, 1, 128, 128, 0, f, None, None) == H.HLA_ERR_INVALID_ARGUMENT
    assert L.hla2_step_sde(16, 16, 16, 16, 1, 1, 1, 100, 128, 0, f, 16, None) == H.HLA_ERR_UNSUPPORTED
    assert L.hla2_step_sde(16, 16, 16, 16, 1, 0, 1, 128, 128, 0, f, 16, None) == H.HLA_OK


def test_noalloc_empty_problem_without_gpu(L):
    from paper_2510_27258_gb300 import hla as H
    f = ctypes.c_float(1e-6)
    assert L.hla2_forward_noalloc(None, None, None, None, 1, 1, 0, 256, 128, 128, 1, 0, f, 128, None, None) == H.HLA_OK
    assert L.hla_last_error() == b""


def test_ahla_and_backward_argument_errors(L):
    from paper_2510_27258_gb300 import hla as H
    f = ctypes.c_float(1e-6)
    assert L.ahla_state_floats(128, 64) == 2 * 128 * 64 + 2 * 128
    assert L.ahla_workspace_bytes(1, 1, 64, 16, 16, 16, 0) > 0
    assert L.ahla_workspace_bytes(1, 1, 64, 48, 16, 16, 0) == 0
    assert L.hla2_backward_workspace_bytes(1, 1, 64, 16, 16, 16, 1) > 0
    assert L.hla2_backward_workspace_bytes(1, 1, 64, 16, 16, 0, 1) == 0

    def ahla(q=16, B=1, n=64, d=16, chunk=16, ws=256, ws_bytes=1 << 30):
        return L.ahla_forward(q, 16, 16, 16, 1, B, 1, n, d, 16, 0, f, chunk, None, None, ws, ws_bytes, None)
    assert ahla(q=None) == H.HLA_ERR_INVALID_ARGUMENT
    assert ahla(q=8) == H.HLA_ERR_INVALID_ARGUMENT
    assert ahla(d=24) == H.HLA_ERR_UNSUPPORTED
    assert ahla(chunk=129) == H.HLA_ERR_UNSUPPORTED
    assert ahla(ws=None) == H.HLA_ERR_WORKSPACE
    assert ahla(ws=272) == H.HLA_ERR_INVALID_ARGUMENT
    assert ahla(B=0) == H.HLA_OK
    assert L.ahla_step(16, 16, 16, 16, 1, 1, 1, 128, 128, 0, f, None, None) == H.HLA_ERR_INVALID_ARGUMENT
    assert L.ahla_step(16, 16, 16, 16, 1, 0, 1, 128, 128, 0, f, 16, None) == H.HLA_OK
    assert L.ahla_forward_path(1, 1, 64, 24, 16, 0, 16, 1, 0, 0) == -1
    assert L.ahla_forward_path(1, 1, 64, 16, 16, 0, 16, 0, 0, 0) == 0  # fp32 tokens: the CUDA-core kernels
    assert L.hla2_backward_path(1, 1, 64, 24, 64, 0, 64, 1) == -1
    assert L.hla2_backward_path(8, 16, 2048, 64, 64, 0, 64, 1) == 0  # no device here: the CUDA-core kernels
    # third order: no device here, so never the tensor-core path; chunk-parallel or serial otherwise
    nl = ctypes.c_int(-7)
    assert L.hla3_forward_path(1, 1, 64, 24, 32, 1, 0, 32, 0, 0, 0, ctypes.byref(nl)) == -1
    assert L.hla3_forward_path(2, 4, 4096, 32, 32, 1, 0, 32, 0, 0, 0, ctypes.byref(nl)) == 1 and nl.value == 5
    assert L.hla3_forward_path(2, 4, 4096, 32, 32, 1, 0, 32, 0, 1, 0, ctypes.byref(nl)) == 1 and nl.value == 6
    assert L.hla3_forward_path(2, 4, 4096, 32, 32, 0, 0, 32, 0, 0, 0, ctypes.byref(nl)) == 1 and nl.value == 3
    assert L.hla3_forward_path(2, 4, 4096, 32, 32, 1, 0, 32, 0, 0, 1, ctypes.byref(nl)) == 0 and nl.value == 1
    assert L.hla3_forward_path(0, 4, 4096, 32, 32, 1, 0, 32, 0, 0, 0, ctypes.byref(nl)) == 0 and nl.value == 0

    def bwd(dout=16, dq=16, n=64, d=16, ws=256, ws_bytes=1 << 30):
        return L.hla2_backward(16, 16, 16, dout, dq, 16, 16, 1, 1, 1, n, d, 16, 0, f, 16, ws, ws_bytes, None)
    assert bwd(dout=None) == H.HLA_ERR_INVALID_ARGUMENT
    assert bwd(dq=24) == H.HLA_ERR_INVALID_ARGUMENT
    assert bwd(d=100) == H.HLA_ERR_UNSUPPORTED
    assert bwd(ws_bytes=16) == H.HLA_ERR_WORKSPACE
    assert bwd(n=0) == H.HLA_OK
