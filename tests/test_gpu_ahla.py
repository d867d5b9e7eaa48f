"""AHLA (asymmetric second order) on the GPU, through the C ABI, against the
fp64 oracle (Theorem AHLA's recurrence, itself pinned by Eq. AHLA-explicit and
the scan equivalence).  Error metric and bars as for second order."""
import numpy as np
import pytest
import torch

import hla_inputs
import oracle
from parity import TOL, check_normalized, rowerr, rowerr_stats

pytestmark = pytest.mark.gpu
DEV = "cuda:0"


@pytest.fixture(scope="module")
def hla():
    from paper_2510_27258_gb300 import build
    build.build()
    from paper_2510_27258_gb300 import hla as binding
    return binding


def gpu_ahla(hla, q, k, v, dtype, normalized, chunk, state_in=None, want_state=False):
    B, H, n, d = q.shape
    tq, tk, tv = (hla_inputs.as_torch(x, dtype, DEV) for x in (q, k, v))
    sin = None if state_in is None else torch.from_numpy(np.ascontiguousarray(state_in, np.float32)).to(DEV)
    sout = (torch.zeros((B, H, hla.ahla_state_floats(d, v.shape[-1])), dtype=torch.float32, device=DEV)
            if want_state else None)
    out = hla.ahla_forward(tq, tk, tv, normalized=normalized, eps=hla_inputs.EPS, chunk=chunk, state_in=sin,
                           state_out=sout)
    torch.cuda.synchronize()
    res = out.float().cpu().numpy().reshape(B * H, n, -1)
    return (res, sout.cpu().numpy().reshape(B * H, -1)) if want_state else res


def ref_ahla(q, k, v, state_in=None):
    B, H, n, d = q.shape
    sin = None if state_in is None else np.asarray(state_in, np.float64).reshape(B * H, -1)
    return oracle.ahla_serial(q.reshape(B * H, n, d), k.reshape(B * H, n, d), v.reshape(B * H, n, -1),
                              normalized=False, state_in=sin, return_den=True, return_state=True, nthreads=8)


SHAPES = [
    # (B, H, n, d, dv, chunk, dtype)
    (1, 1, 1, 16, 16, 16, "f32"),
    (1, 2, 37, 16, 32, 16, "f32"),
    (2, 1, 200, 64, 64, 64, "bf16"),
    (1, 2, 257, 128, 128, 128, "bf16"),
    (1, 1, 300, 32, 128, 100, "f32"),
    (1, 1, 130, 128, 64, 7, "bf16"),
    (1, 3, 96, 64, 16, 32, "f32"),
]


@pytest.mark.parametrize("shape", SHAPES, ids=lambda s: "B%dH%dn%dd%ddv%dC%d%s" % s)
@pytest.mark.parametrize("normalized", [False, True])
def test_ahla_forward_small(hla, shape, normalized):
    B, H, n, d, dv, chunk, dtype = shape
    q, k, v = hla_inputs.make_qkv(B, H, n, d, dv, seed=2000 + n, dtype=dtype)
    num_ref, den_ref, _ = ref_ahla(q, k, v)
    num_gpu = gpu_ahla(hla, q, k, v, dtype, False, chunk)
    assert rowerr(num_gpu, num_ref) < TOL[dtype]
    if normalized:
        o_gpu = gpu_ahla(hla, q, k, v, dtype, True, chunk)
        assert np.isfinite(o_gpu).all()
        check_normalized(o_gpu, num_gpu, num_ref, den_ref, hla_inputs.EPS, TOL[dtype])


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_ahla_state_in_out(hla, dtype):
    B, H, n, d, dv = 1, 3, 150, 64, 32
    pq, pk, pv = hla_inputs.make_qkv(B, H, 40, d, dv, seed=21, dtype=dtype)
    _, _, st0 = ref_ahla(pq, pk, pv)
    st0 = st0.astype(np.float32)
    q, k, v = hla_inputs.make_qkv(B, H, n, d, dv, seed=22, dtype=dtype)
    got, gst = gpu_ahla(hla, q, k, v, dtype, False, 32, state_in=st0, want_state=True)
    ref, _, rst = ref_ahla(q, k, v, state_in=st0)
    assert rowerr(got, ref) < TOL[dtype]
    scale = np.abs(rst).max()
    assert np.abs(gst - rst).max() <= 2e-5 * scale


def test_ahla_chunk_sizes_agree(hla):
    """The chunk argument is the scan granularity: fp32 results agree across chunk sizes."""
    q, k, v = hla_inputs.make_qkv(1, 2, 333, 32, 32, seed=23, dtype="f32")
    ref = gpu_ahla(hla, q, k, v, "f32", False, 1)
    for chunk in (5, 16, 64, 128):
        assert rowerr(gpu_ahla(hla, q, k, v, "f32", False, chunk), ref) < 1e-5, chunk


def test_ahla_causality_bit_exact(hla):
    B, H, n, d, dv, t = 1, 2, 256, 64, 64, 100
    q, k, v = hla_inputs.make_qkv(B, H, n, d, dv, seed=24, dtype="bf16")
    a = gpu_ahla(hla, q, k, v, "bf16", True, 64)
    q2, k2, v2 = q.copy(), k.copy(), v.copy()
    rng = np.random.default_rng(1)
    for x in (q2, k2, v2):
        x[:, :, t + 1:] = hla_inputs.round_to(rng.standard_normal(x[:, :, t + 1:].shape), "bf16")
    b = gpu_ahla(hla, q2, k2, v2, "bf16", True, 64)
    assert np.array_equal(a[:, : t + 1], b[:, : t + 1])


def test_ahla_workload_sampled(hla):
    """The AHLA bench workload (B8 H16 n2048 d64 bf16, chunk 64); sampled heads."""
    w = hla_inputs.WORKLOADS["ahla_bf16"]
    q, k, v = hla_inputs.make_workload(w)
    got = gpu_ahla(hla, q, k, v, w.dtype, False, w.chunk)
    heads = [0, 40, w.BH - 1]
    ref = oracle.ahla_serial(q.reshape(w.BH, w.n, w.d)[heads], k.reshape(w.BH, w.n, w.d)[heads],
                             v.reshape(w.BH, w.n, w.dv)[heads], nthreads=3)
    err = rowerr(got[heads], ref)
    print("\nahla_bf16 sampled heads %s: row error %s" % (heads, rowerr_stats(got[heads], ref)[0]))
    assert err < TOL["bf16"], err


@pytest.mark.parametrize("d,dv", [(16, 16), (64, 32), (128, 128), (32, 64)])
@pytest.mark.parametrize("normalized", [False, True])
def test_ahla_step(hla, d, dv, normalized):
    """Prefix by ahla_forward (state_out), then single-token steps; the oracle runs prefix and
    steps as one sequence."""
    B, H, prefix, steps = 2, 3, 50, 6
    w = hla_inputs.Workload("t", B, H, 0, d, dv, 64, "f32", True, normalized, d + dv, decode_prefix=prefix,
                            decode_steps=steps)
    (qp, kp, vp), (qs, ks, vs) = hla_inputs.make_decode(w)
    st = torch.zeros((B, H, hla.ahla_state_floats(d, dv)), dtype=torch.float32, device=DEV)
    tq, tk, tv = (hla_inputs.as_torch(x, "f32", DEV) for x in (qp, kp, vp))
    hla.ahla_forward(tq, tk, tv, chunk=64, state_out=st)
    outs = []
    for s in range(steps):
        o = hla.ahla_step(*(hla_inputs.as_torch(x[s], "f32", DEV) for x in (qs, ks, vs)), st, normalized=normalized,
                          eps=hla_inputs.EPS)
        outs.append(o.cpu().numpy().reshape(B * H, dv))
    torch.cuda.synchronize()
    got = np.stack(outs, axis=1)
    cat = [np.concatenate([p.reshape(B * H, prefix, -1), np.moveaxis(x.reshape(steps, B * H, -1), 0, 1)], axis=1)
           for p, x in ((qp, qs), (kp, ks), (vp, vs))]
    num, den, rst = oracle.ahla_serial(*cat, return_den=True, return_state=True)
    if normalized:
        st2 = torch.zeros_like(st)
        hla.ahla_forward(tq, tk, tv, chunk=64, state_out=st2)
        nums = [hla.ahla_step(*(hla_inputs.as_torch(x[s], "f32", DEV) for x in (qs, ks, vs)), st2).cpu().numpy()
                .reshape(B * H, dv) for s in range(steps)]
        check_normalized(got, np.stack(nums, axis=1), num[:, prefix:], den[:, prefix:], hla_inputs.EPS, TOL["f32"])
    else:
        assert rowerr(got, num[:, prefix:]) < TOL["f32"]
    assert np.abs(st.cpu().numpy().reshape(B * H, -1) - rst).max() <= 2e-5 * np.abs(rst).max()



@pytest.mark.parametrize("dtype", ["bf16", "f32"])
@pytest.mark.parametrize("normalized", [False, True])
def test_ahla_step_more_heads_than_sms(hla, dtype, normalized):
    """320 heads (more than the SMs): a block of the staged step works through two or three heads,
    refilling its buffers a pass ahead; three steps after a random state, every head against the
    oracle's single-token updates."""
    B, H, d, dv, steps = 2, 160, 128, 64, 3
    BH = B * H
    L = hla.ahla_state_floats(d, dv)
    # a state as ahla_forward leaves it: [P | m | E | n] of a 40-token prefix, from the oracle
    w = hla_inputs.Workload("t", B, H, 0, d, dv, 64, dtype, True, normalized, 17, decode_prefix=40,
                            decode_steps=steps)
    (qp, kp, vp), (qs, ks, vs) = hla_inputs.make_decode(w)
    flat = lambda x: x.reshape(BH, x.shape[-2], -1).astype(np.float64)
    _, _, st0 = oracle.ahla_serial(flat(qp), flat(kp), flat(vp), return_den=True, return_state=True)
    def steps_from(state0, norm):
        st = torch.from_numpy(np.ascontiguousarray(state0.reshape(B, H, L), np.float32)).to(DEV)
        outs = []
        for s_ in range(steps):
            o = hla.ahla_step(*(hla_inputs.as_torch(x[s_], dtype, DEV) for x in (qs, ks, vs)), st, normalized=norm,
                              eps=hla_inputs.EPS)
            outs.append(o.float().cpu().numpy().reshape(BH, dv))
        torch.cuda.synchronize()
        return np.stack(outs, axis=1), st.cpu().numpy().reshape(BH, -1)

    got, st_got = steps_from(st0, normalized)
    seq = lambda x: np.moveaxis(x.reshape(steps, BH, -1), 0, 1).astype(np.float64)
    num, den, rst = oracle.ahla_serial(seq(qs), seq(ks), seq(vs), state_in=st0.astype(np.float64), return_den=True,
                                       return_state=True)
    if normalized:  # outputs in the token type (bf16 rounds them: its bar)
        nums, _ = steps_from(st0, False)
        check_normalized(got, nums, num, den, hla_inputs.EPS, TOL[dtype])
    else:
        assert rowerr(got, num) < TOL[dtype]
    assert np.abs(st_got - rst).max() <= 2e-5 * np.abs(rst).max()

# ----------------------------------------------------------------------------
# the tensor-core path (bf16, d and dv in {64, 128}, plain output, no states)
# ----------------------------------------------------------------------------

TC_SHAPES = [
    # (B, H, n, d, dv)
    (1, 1, 1, 128, 128),
    (1, 2, 127, 128, 128),
    (2, 3, 300, 64, 64),
    (1, 2, 700, 64, 128),
    (1, 1, 1000, 128, 64),
]


@pytest.mark.parametrize("shape", TC_SHAPES, ids=lambda s: "B%dH%dn%dd%ddv%d" % s)
def test_ahla_tensor_core_path(hla, shape, monkeypatch):
    """Every head against the oracle, and against the CUDA-core path on the same inputs."""
    B, H, n, d, dv = shape
    q, k, v = hla_inputs.make_qkv(B, H, n, d, dv, seed=4000 + n + d, dtype="bf16")
    ref, _, _ = ref_ahla(q, k, v)
    got = gpu_ahla(hla, q, k, v, "bf16", False, 64)
    assert rowerr(got, ref) < TOL["bf16"]
    monkeypatch.setenv("HLA_DISABLE_FUSED", "1")
    generic = gpu_ahla(hla, q, k, v, "bf16", False, 64)
    assert rowerr(generic, ref) < TOL["bf16"]


def test_ahla_tensor_core_more_heads_than_sms(hla):
    """200 heads: a CTA sweeps several heads one after the other (carries restarted per head)."""
    B, H, n, d = 2, 100, 260, 128
    q, k, v = hla_inputs.make_qkv(B, H, n, d, d, seed=4100, dtype="bf16")
    got = gpu_ahla(hla, q, k, v, "bf16", False, 64)
    heads = [0, 1, 151, 152, 153, 199]
    ref = oracle.ahla_serial(q.reshape(B * H, n, d)[heads], k.reshape(B * H, n, d)[heads],
                             v.reshape(B * H, n, d)[heads], nthreads=6)
    assert rowerr(got[heads], ref) < TOL["bf16"]


def test_ahla_tensor_core_causality_and_determinism(hla):
    B, H, n, d, t = 1, 2, 512, 128, 300
    q, k, v = hla_inputs.make_qkv(B, H, n, d, d, seed=4200, dtype="bf16")
    a = gpu_ahla(hla, q, k, v, "bf16", False, 64)
    assert np.array_equal(a, gpu_ahla(hla, q, k, v, "bf16", False, 64))
    q2, k2, v2 = q.copy(), k.copy(), v.copy()
    rng = np.random.default_rng(3)
    for x in (q2, k2, v2):
        x[:, :, t + 1:] = hla_inputs.round_to(rng.standard_normal(x[:, :, t + 1:].shape), "bf16")
    b = gpu_ahla(hla, q2, k2, v2, "bf16", False, 64)
    assert np.array_equal(a[:, : t + 1], b[:, : t + 1])
    assert not np.array_equal(a[:, t + 1:], b[:, t + 1:])
