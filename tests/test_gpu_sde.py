"""The (S, D, e) decode state on the GPU (through the C ABI) against the fp64
oracle: the conversion of paper tuples (D = S C - G, e = S m - h) and the
decode step on (S, D, e) states, whose outputs must equal the oracle's serial
recurrence over the prefix and the decoded tokens as one sequence."""
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


def _sde_close(got, ref, d, dv, tol=2e-5):
    """Parts S, D, e within tol of max(|part|, |S| |D| / |D|-free scale)."""
    parts = ((0, d * d), (d * d, d * d + d * dv), (d * d + d * dv, d * d + d * dv + d))
    for lo, hi in parts:
        g, r = got[..., lo:hi], ref[..., lo:hi]
        scale = max(np.abs(r).max(), 1.0)
        assert np.abs(g - r).max() <= tol * scale, (lo, hi, np.abs(g - r).max(), scale)


@pytest.mark.parametrize("d,dv", [(16, 16), (64, 32), (128, 128), (32, 64)])
def test_state_to_sde_matches_oracle(hla, d, dv):
    B, H = 2, 3
    q, k, v = hla_inputs.make_qkv(B, H, 90, d, dv, seed=300 + d + dv, dtype="f32")
    _, st = oracle.hla2_serial(q.reshape(B * H, 90, d), k.reshape(B * H, 90, d), v.reshape(B * H, 90, dv),
                               masked=True, return_state=True)
    st32 = st.astype(np.float32)
    ref = oracle.hla2_state_to_sde(st32.astype(np.float64), d, dv)
    tst = torch.from_numpy(st32).reshape(B, H, -1).to(DEV)
    got = hla.hla2_state_to_sde(tst, d, dv)
    torch.cuda.synchronize()
    _sde_close(got.cpu().numpy().reshape(B * H, -1), ref, d, dv, tol=1e-5)


def _run(hla, B, H, d, dv, prefix, steps, dtype, normalized, seed, heads=None):
    w = hla_inputs.Workload("t", B, H, 0, d, dv, 64, dtype, True, normalized, seed, decode_prefix=prefix,
                            decode_steps=steps)
    (qp, kp, vp), (qs, ks, vs) = hla_inputs.make_decode(w)
    st = torch.zeros((B, H, hla.hla2_state_floats(d, dv)), dtype=torch.float32, device=DEV)
    tq, tk, tv = (hla_inputs.as_torch(x, dtype, DEV) for x in (qp, kp, vp))
    hla.hla2_forward(tq, tk, tv, masked=True, normalized=False, eps=hla_inputs.EPS, chunk=64, state_out=st)
    del tq, tk, tv
    sde = hla.hla2_state_to_sde(st, d, dv)
    del st
    outs = []
    for s in range(steps):
        o = hla.hla2_step_sde(hla_inputs.as_torch(qs[s], dtype, DEV), hla_inputs.as_torch(ks[s], dtype, DEV),
                              hla_inputs.as_torch(vs[s], dtype, DEV), sde, normalized=normalized, eps=hla_inputs.EPS)
        outs.append(o.float().cpu().numpy().reshape(B * H, dv))
    torch.cuda.synchronize()
    got = np.stack(outs, axis=1)
    gsde = sde.cpu().numpy().reshape(B * H, -1)
    heads = list(range(B * H)) if heads is None else heads
    cat = [np.concatenate([p.reshape(B * H, prefix, -1)[heads], np.moveaxis(x.reshape(steps, B * H, -1), 0, 1)[heads]],
                          axis=1) for p, x in ((qp, qs), (kp, ks), (vp, vs))]
    num, den, rst = oracle.hla2_serial(*cat, masked=True, normalized=False, return_den=True, return_state=True,
                                       nthreads=4)
    return got[heads], gsde[heads], num[:, prefix:], den[:, prefix:], oracle.hla2_state_to_sde(rst, d, dv), cat


@pytest.mark.parametrize("d,dv", [(16, 16), (64, 32), (128, 128), (32, 64)])
@pytest.mark.parametrize("normalized", [False, True])
def test_step_sde_matches_oracle(hla, d, dv, normalized):
    got, gsde, num, den, rsde, _ = _run(hla, 2, 3, d, dv, 50, 6, "f32", normalized, seed=d + 2 * dv)
    if normalized:
        num_gpu = _run(hla, 2, 3, d, dv, 50, 6, "f32", False, seed=d + 2 * dv)[0]
        check_normalized(got, num_gpu, num, den, hla_inputs.EPS, TOL["f32"])
    else:
        assert rowerr(got, num) < TOL["f32"]
    _sde_close(gsde, rsde, d, dv)


@pytest.mark.parametrize("d,dv,dtype", [(32, 64, "f32"), (64, 64, "bf16"), (128, 32, "f32")])
def test_step_sde_more_heads_than_sms(hla, d, dv, dtype):
    """320 heads: a block of the decode kernel works through several heads."""
    got, gsde, num, _, rsde, _ = _run(hla, 4, 80, d, dv, 20, 3, dtype, False, seed=11 + d + dv)
    assert rowerr(got, num) < TOL[dtype]
    _sde_close(gsde, rsde, d, dv)


def test_step_sde_equals_tuple_step(hla):
    """Both decode formats give the same outputs on the same tokens (fp32 tokens)."""
    B, H, d, dv, steps = 2, 4, 64, 64, 5
    w = hla_inputs.Workload("t", B, H, 0, d, dv, 64, "f32", True, False, 5, decode_prefix=40, decode_steps=steps)
    (qp, kp, vp), (qs, ks, vs) = hla_inputs.make_decode(w)
    st = torch.zeros((B, H, hla.hla2_state_floats(d, dv)), dtype=torch.float32, device=DEV)
    tq, tk, tv = (hla_inputs.as_torch(x, "f32", DEV) for x in (qp, kp, vp))
    hla.hla2_forward(tq, tk, tv, masked=True, chunk=64, state_out=st)
    sde = hla.hla2_state_to_sde(st, d, dv)
    for s in range(steps):
        toks = [hla_inputs.as_torch(x[s], "f32", DEV) for x in (qs, ks, vs)]
        a = hla.hla2_step(*toks, st, masked=True)
        b = hla.hla2_step_sde(*toks, sde)
        torch.cuda.synchronize()
        a, b = a.cpu().numpy().reshape(B * H, dv), b.cpu().numpy().reshape(B * H, dv)
        assert rowerr(b, a) < 1e-5, s


def test_step_sde_decode_workload_full_depth_sampled(hla):
    """The decode workload's shape (B64 H32 d128, bf16 tokens) at its full
    4096-token prefix, 16 steps on (S, D, e) states; sampled heads checked."""
    w = hla_inputs.WORKLOADS["decode_bf16"]
    heads = [0, 700, 1300, w.BH - 1]
    got, gsde, num, _, rsde, _ = _run(hla, w.B, w.H, w.d, w.dv, w.decode_prefix, 16, w.dtype, w.normalized, w.seed,
                                      heads=heads)
    err = rowerr(got, num)
    print("\ndecode on (S, D, e) at depth %d, 16 steps, heads %s: row error %s" % (w.decode_prefix, heads,
                                                                                rowerr_stats(got, num)[0]))
    assert err < TOL["bf16"], err
    _sde_close(gsde, rsde, w.d, w.dv)
