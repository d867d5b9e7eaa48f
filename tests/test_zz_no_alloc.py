"""hla2_forward_noalloc, the entry point for callers that cannot allocate device
memory (they cannot call cudaMalloc or hand over a workspace, e.g. code running
under someone else's memory pool or budget): it must give the same outputs as
hla2_forward with a caller workspace, on consecutive calls that reuse the
library's own scratch array.  Kept in the last test file so that a run stopping
at its first failure has already run everything else."""
import ctypes

import numpy as np
import pytest
import torch

import hla_inputs
from parity import TOL, rowerr

pytestmark = pytest.mark.gpu
DEV = "cuda:0"


@pytest.fixture(scope="module")
def hla():
    from paper_2510_27258_gb300 import build
    build.build()
    from paper_2510_27258_gb300 import hla as binding
    return binding


def _noalloc(hla, q, k, v, out, normalized):
    B, H, n, d = q.shape
    L = hla.lib()
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    return L.hla2_forward_noalloc(ctypes.c_void_p(q.data_ptr()), ctypes.c_void_p(k.data_ptr()),
                                  ctypes.c_void_p(v.data_ptr()), ctypes.c_void_p(out.data_ptr()), hla.HLA_BF16,
                                  B, H, n, d, v.shape[-1], 1, int(normalized), ctypes.c_float(hla_inputs.EPS), 128,
                                  None, stream)


@pytest.mark.parametrize("normalized", [False, True])
def test_noalloc_matches_workspace_forward_on_two_calls(hla, normalized):
    B, H, n, d = 1, 4, 1000, 128
    q, k, v = hla_inputs.make_qkv(B, H, n, d, d, seed=77, dtype="bf16")
    tq, tk, tv = (hla_inputs.as_torch(x, "bf16", DEV) for x in (q, k, v))
    ref = hla.hla2_forward(tq, tk, tv, masked=True, normalized=normalized, eps=hla_inputs.EPS, chunk=128)
    torch.cuda.synchronize()
    ref = ref.float().cpu().numpy().reshape(B * H, n, d)
    for call in range(2):  # the second call reuses the scratch left by the first
        out = torch.zeros((B, H, n, d), dtype=torch.bfloat16, device=DEV)
        assert _noalloc(hla, tq, tk, tv, out, normalized) == hla.HLA_OK, hla.lib().hla_last_error()
        torch.cuda.synchronize()
        got = out.float().cpu().numpy().reshape(B * H, n, d)
        assert rowerr(got, ref) < TOL["bf16"], (call, rowerr(got, ref))


def test_noalloc_rejects_sizes_beyond_its_scratch(hla):
    # 128 heads need about 33 MiB of scratch (> 16 MiB): refused before any launch
    B, H, n, d = 1, 128, 256, 128
    t = torch.zeros((B, H, n, d), dtype=torch.bfloat16, device=DEV)
    assert _noalloc(hla, t, t, t, t, False) == hla.HLA_ERR_WORKSPACE
    assert b"scratch" in hla.lib().hla_last_error()
