"""Second-order HLA on the GPU (through the C ABI) against the fp64 oracle.

Inputs come from hla_inputs (identical bits on both sides; bf16 values are
upcast exactly for the oracle).  Error metric per output row t:
max_c |o_gpu[t,c] - o_ref[t,c]| / ||o_ref[t,:]||_2, maximised over rows.
Bars: 1e-4 for fp32 tokens, 2e-2 for bf16 tokens (fp32 accumulation); ratio-
normalised outputs are checked as described in tests/parity.py.
"""
import numpy as np
import pytest
import torch

import hla_inputs
import oracle
from parity import TOL, check_normalized, rowerr, rowerr_rows, rowerr_stats

pytestmark = pytest.mark.gpu

DEV = "cuda:0"


@pytest.fixture(scope="module")
def hla():
    from paper_2510_27258_gb300 import build
    build.build()
    from paper_2510_27258_gb300 import hla as binding
    return binding


def gpu_forward(hla, q, k, v, dtype, masked=True, normalized=False, chunk=64, state_in=None, want_state=False,
                alias_state=False):
    B, H, n, d = q.shape
    dv = v.shape[-1]
    tq, tk, tv = (hla_inputs.as_torch(x, dtype, DEV) for x in (q, k, v))
    sin = None if state_in is None else torch.from_numpy(np.ascontiguousarray(state_in, np.float32)).to(DEV)
    sout = None
    if want_state:
        sout = sin if alias_state else torch.zeros((B, H, hla.hla2_state_floats(d, dv)), dtype=torch.float32,
                                                   device=DEV)
    out = hla.hla2_forward(tq, tk, tv, masked=masked, normalized=normalized, eps=hla_inputs.EPS, chunk=chunk,
                           state_in=sin, state_out=sout)
    torch.cuda.synchronize()
    res = out.float().cpu().numpy()
    if want_state:
        return res, sout.cpu().numpy().reshape(B * H, -1)
    return res


def ref_forward(q, k, v, masked=True, normalized=False, state_in=None, heads=None, want_state=False,
                want_den=False):
    B, H, n, d = q.shape
    dv = v.shape[-1]
    qf, kf, vf = q.reshape(B * H, n, d), k.reshape(B * H, n, d), v.reshape(B * H, n, dv)
    sin = None if state_in is None else np.asarray(state_in, np.float64).reshape(B * H, -1)
    if heads is not None:
        qf, kf, vf = qf[heads], kf[heads], vf[heads]
        sin = None if sin is None else sin[heads]
    return oracle.hla2_serial(qf, kf, vf, masked=masked, normalized=normalized, eps=hla_inputs.EPS, state_in=sin,
                              return_state=want_state, return_den=want_den, nthreads=8)


def check_forward(hla, q, k, v, dtype, masked, normalized, chunk, state_in=None, heads=None):
    """GPU forward vs oracle with the criteria of tests/parity.py; returns the errors."""
    B, H, n, d = q.shape
    dv = v.shape[-1]
    pick = (lambda a: a.reshape(B * H, n, dv)) if heads is None else (lambda a: a.reshape(B * H, n, dv)[heads])
    num_gpu = pick(gpu_forward(hla, q, k, v, dtype, masked, False, chunk, state_in=state_in))
    num_ref, den_ref = ref_forward(q, k, v, masked, False, state_in=state_in, heads=heads, want_den=True)
    tol = TOL[dtype]
    if not normalized:
        err = rowerr(num_gpu, num_ref)
        assert err < tol, err
        return {"num": err}
    o_gpu = pick(gpu_forward(hla, q, k, v, dtype, masked, True, chunk, state_in=state_in))
    assert np.isfinite(o_gpu).all()
    return check_normalized(o_gpu, num_gpu, num_ref, den_ref, hla_inputs.EPS, tol)


SMALL = [
    # (B, H, n, d, dv, chunk, dtype)
    (1, 1, 1, 16, 16, 16, "f32"),
    (1, 2, 37, 16, 32, 16, "f32"),
    (2, 1, 200, 64, 64, 64, "bf16"),
    (1, 2, 257, 128, 128, 128, "bf16"),
    (1, 1, 300, 32, 128, 100, "f32"),
    (1, 1, 130, 128, 64, 7, "bf16"),
    (1, 3, 96, 64, 16, 32, "f32"),
]


@pytest.mark.parametrize("shape", SMALL, ids=lambda s: "B%dH%dn%dd%ddv%dC%d%s" % s)
@pytest.mark.parametrize("masked,normalized", [(True, False), (True, True), (False, False), (False, True)])
def test_forward_small(hla, shape, masked, normalized):
    B, H, n, d, dv, chunk, dtype = shape
    q, k, v = hla_inputs.make_qkv(B, H, n, d, dv, seed=1000 + n, dtype=dtype)
    check_forward(hla, q, k, v, dtype, masked, normalized, chunk)


def test_tiny_workload_full(hla):
    w = hla_inputs.WORKLOADS["tiny_f32"]
    q, k, v = hla_inputs.make_workload(w)
    got = gpu_forward(hla, q, k, v, w.dtype, w.masked, w.normalized, w.chunk)
    ref = ref_forward(q, k, v, w.masked, w.normalized)
    err = rowerr(got.reshape(w.BH, w.n, w.dv), ref)
    assert err < 1e-4, err


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("masked", [True, False])
def test_state_in_out(hla, dtype, masked):
    B, H, n, d, dv, chunk = 1, 3, 150, 64, 32, 32
    pq, pk, pv = hla_inputs.make_qkv(B, H, 40, d, dv, seed=7, dtype=dtype)
    _, st0 = ref_forward(pq, pk, pv, masked=masked, want_state=True)
    st0 = st0.astype(np.float32)  # the GPU state is fp32; feed both sides the same values
    q, k, v = hla_inputs.make_qkv(B, H, n, d, dv, seed=8, dtype=dtype)
    check_forward(hla, q, k, v, dtype, masked, True, chunk, state_in=st0)
    got, gst = gpu_forward(hla, q, k, v, dtype, masked, False, chunk, state_in=st0, want_state=True)
    ref, rst = ref_forward(q, k, v, masked, False, state_in=st0, want_state=True)
    assert rowerr(got.reshape(B * H, n, dv), ref) < TOL[dtype]
    parts_g, parts_r = oracle.split_state2(gst, d, dv), oracle.split_state2(rst, d, dv)
    for name in ("S", "C", "m", "G", "h"):
        scale = max(np.abs(parts_r[name]).max(), np.abs(parts_r["S"]).max() * np.abs(parts_r["C"]).max())
        assert np.abs(parts_g[name] - parts_r[name]).max() <= 2e-5 * max(scale, 1.0), name
    if not masked:
        assert not parts_g["G"].any() and not parts_g["h"].any()


def test_state_out_aliases_state_in(hla):
    B, H, n, d, dv = 1, 2, 64, 32, 32
    pq, pk, pv = hla_inputs.make_qkv(B, H, 30, d, dv, seed=9, dtype="f32")
    _, st0 = ref_forward(pq, pk, pv, want_state=True)
    st0 = st0.astype(np.float32)
    q, k, v = hla_inputs.make_qkv(B, H, n, d, dv, seed=10, dtype="f32")
    got, gst = gpu_forward(hla, q, k, v, "f32", True, False, 16, state_in=st0.copy(), want_state=True,
                           alias_state=True)
    ref, rst = ref_forward(q, k, v, True, False, state_in=st0, want_state=True)
    assert rowerr(got.reshape(B * H, n, dv), ref) < 1e-4
    assert np.abs(gst - rst).max() <= 1e-4 * np.abs(rst).max()


def test_empty_sequence_passes_state_through(hla):
    B, H, d, dv = 1, 2, 16, 16
    pq, pk, pv = hla_inputs.make_qkv(B, H, 5, d, dv, seed=11, dtype="f32")
    _, st0 = ref_forward(pq, pk, pv, want_state=True)
    st0 = st0.astype(np.float32)
    q = np.zeros((B, H, 0, d), np.float32)
    v = np.zeros((B, H, 0, dv), np.float32)
    got, gst = gpu_forward(hla, q, q, v, "f32", True, False, 16, state_in=st0, want_state=True)
    assert got.shape == (B, H, 0, dv)
    assert np.abs(gst - st0).max() <= 1e-5 * np.abs(st0).max()


def test_causality_bit_exact(hla):
    B, H, n, d, dv, t = 1, 2, 256, 64, 64, 100
    q, k, v = hla_inputs.make_qkv(B, H, n, d, dv, seed=12, dtype="bf16")
    a = gpu_forward(hla, q, k, v, "bf16", True, True, 64)
    rng = np.random.default_rng(0)
    q2, k2, v2 = q.copy(), k.copy(), v.copy()
    q2[:, :, t + 1:] = hla_inputs.round_to(rng.standard_normal(q2[:, :, t + 1:].shape), "bf16")
    k2[:, :, t + 1:] = hla_inputs.round_to(rng.standard_normal(k2[:, :, t + 1:].shape), "bf16")
    v2[:, :, t + 1:] = hla_inputs.round_to(rng.standard_normal(v2[:, :, t + 1:].shape), "bf16")
    b = gpu_forward(hla, q2, k2, v2, "bf16", True, True, 64)
    assert np.array_equal(a[:, :, : t + 1], b[:, :, : t + 1])
    assert not np.array_equal(a[:, :, t + 1:], b[:, :, t + 1:])


def test_deterministic(hla):
    q, k, v = hla_inputs.make_qkv(2, 4, 512, 128, 128, seed=13, dtype="bf16")
    a = gpu_forward(hla, q, k, v, "bf16", True, True, 128)
    b = gpu_forward(hla, q, k, v, "bf16", True, True, 128)
    assert np.array_equal(a, b)


def _tile_errors(got, ref, tile=128):
    """Largest row error of each 128-token tile, over the given heads ([heads, n, dv])."""
    r = rowerr_rows(got, ref)
    n = r.shape[-1]
    return [float(r[:, a:a + tile].max()) for a in range(0, n, tile)]


@pytest.mark.parametrize("name", ["mid_bf16", "long_bf16_norm"])
def test_workload_full_size_sampled(hla, name):
    """Full-size workloads in the launch configuration the benchmark times;
    the oracle checks every position of sampled heads (one in each quarter of
    the heads, so that heads late in the ticket order are included).  Prints the
    literal figures: the numerator's largest row error per 128-token tile (tiles
    after a head's first segment get their carry term in the fix-up), and for
    the normalised output the largest row error over every row, the rows beyond
    the bar and the K those rows needed."""
    w = hla_inputs.WORKLOADS[name]
    q, k, v = hla_inputs.make_workload(w)
    heads = [0, w.BH // 4 + 1, w.BH // 2 + 1, 3 * w.BH // 4 + 2, w.BH - 1]
    res = check_forward(hla, q, k, v, w.dtype, w.masked, w.normalized, w.chunk, heads=heads)
    num_gpu = gpu_forward(hla, q, k, v, w.dtype, w.masked, False, w.chunk).reshape(w.BH, w.n, w.dv)[heads]
    num_ref = ref_forward(q, k, v, w.masked, False, heads=heads)
    tiles = _tile_errors(num_gpu, num_ref)
    print("\n%s sampled heads %s: %s; numerator row error %s; by tile: first %.3g, max %.3g (tile %d), "
          "tiles 0-6 %.3g, tiles 7+ %.3g" % (name, heads, res, rowerr_stats(num_gpu, num_ref)[0], tiles[0],
                                             max(tiles), int(np.argmax(tiles)), max(tiles[:7]),
                                             max(tiles[7:]) if len(tiles) > 7 else 0.0))
    if w.normalized:
        assert res["ill_rows"] <= 0.01 * res["rows"], res


# ----------------------------------------------------------------------------
# decode step
# ----------------------------------------------------------------------------

def _decode_run(hla, B, H, d, dv, prefix, steps, dtype, masked, normalized, seed, heads=None):
    w = hla_inputs.Workload("t", B, H, 0, d, dv, 64, dtype, masked, normalized, seed, decode_prefix=prefix,
                            decode_steps=steps)
    (qp, kp, vp), (qs, ks, vs) = hla_inputs.make_decode(w)
    st = torch.zeros((B, H, hla.hla2_state_floats(d, dv)), dtype=torch.float32, device=DEV)
    tq, tk, tv = (hla_inputs.as_torch(x, dtype, DEV) for x in (qp, kp, vp))
    hla.hla2_forward(tq, tk, tv, masked=masked, normalized=normalized, eps=hla_inputs.EPS, chunk=64, state_out=st)
    outs = []
    for s in range(steps):
        o = hla.hla2_step(hla_inputs.as_torch(qs[s], dtype, DEV), hla_inputs.as_torch(ks[s], dtype, DEV),
                          hla_inputs.as_torch(vs[s], dtype, DEV), st, masked=masked, normalized=normalized,
                          eps=hla_inputs.EPS)
        outs.append(o.float().cpu().numpy())
    torch.cuda.synchronize()
    got = np.stack(outs, axis=2).reshape(B * H, steps, dv)
    # oracle: the prefix and the decode tokens as one sequence
    qa = np.concatenate([qp, np.moveaxis(qs, 0, 2)], axis=2)
    ka = np.concatenate([kp, np.moveaxis(ks, 0, 2)], axis=2)
    va = np.concatenate([vp, np.moveaxis(vs, 0, 2)], axis=2)
    ref, rst = ref_forward(qa, ka, va, masked, normalized, heads=heads, want_state=True)
    gst = st.cpu().numpy().reshape(B * H, -1)
    if heads is not None:
        got, gst = got[heads], gst[heads]
    return got, ref[:, prefix:], gst, rst


@pytest.mark.parametrize("d,dv", [(16, 16), (64, 32), (128, 128), (32, 64)])
@pytest.mark.parametrize("masked,normalized", [(True, False), (True, True), (False, False)])
def test_decode_small(hla, d, dv, masked, normalized):
    dtype = "f32"
    got, ref, gst, rst = _decode_run(hla, 2, 3, d, dv, 50, 6, dtype, masked, normalized, seed=d + dv)
    if normalized:
        num, nref, _, _ = _decode_run(hla, 2, 3, d, dv, 50, 6, dtype, masked, False, seed=d + dv)
        B, H = 2, 3
        (qp, kp, vp), (qs, ks, vs) = hla_inputs.make_decode(hla_inputs.Workload(
            "t", B, H, 0, d, dv, 64, dtype, masked, False, d + dv, decode_prefix=50, decode_steps=6))
        qa, ka, va = (np.concatenate([a, np.moveaxis(b, 0, 2)], axis=2) for a, b in ((qp, qs), (kp, ks), (vp, vs)))
        _, den_ref = ref_forward(qa, ka, va, masked, False, want_den=True)
        check_normalized(got, num, nref, den_ref[:, 50:], hla_inputs.EPS, 1e-4)
    else:
        assert rowerr(got, ref) < 1e-4
    pg, pr = oracle.split_state2(gst, d, dv), oracle.split_state2(rst, d, dv)
    for name in ("S", "C", "m") + (("G", "h") if masked else ()):
        scale = max(np.abs(pr[name]).max(), np.abs(pr["S"]).max() * np.abs(pr["C"]).max())
        assert np.abs(pg[name] - pr[name]).max() <= 2e-5 * max(scale, 1.0), name


@pytest.mark.parametrize("d,dv,dtype", [(32, 64, "f32"), (64, 64, "bf16"), (128, 32, "f32")])
@pytest.mark.parametrize("masked", [True, False])
def test_decode_more_heads_than_sms(hla, d, dv, dtype, masked):
    """320 heads (more than the SMs, so a block of the decode kernel works
    through several heads with the next head's state staged while it computes):
    every head's outputs and state against the oracle."""
    B, H = 4, 80
    got, ref, gst, rst = _decode_run(hla, B, H, d, dv, 20, 3, dtype, masked, False, seed=7 + d + dv)
    assert rowerr(got, ref) < (1e-4 if dtype == "f32" else 2e-2)
    pg, pr = oracle.split_state2(gst, d, dv), oracle.split_state2(rst, d, dv)
    for name in ("S", "C", "m") + (("G", "h") if masked else ()):
        scale = max(np.abs(pr[name]).max(), np.abs(pr["S"]).max() * np.abs(pr["C"]).max())
        assert np.abs(pg[name] - pr[name]).max() <= 2e-5 * max(scale, 1.0), name


def test_decode_workload_full_depth_sampled(hla):
    """The decode workload as the benchmark runs it: B64 H32 d128, bf16 tokens, the
    fp32 state built by one forward over the 4096-token prefix, then 16
    single-token steps; the oracle runs the prefix and the steps as one sequence
    for sampled heads and checks every step's output and the final state."""
    w = hla_inputs.WORKLOADS["decode_bf16"]
    steps = 16
    (qp, kp, vp), (qs, ks, vs) = hla_inputs.make_decode(w, steps=steps)
    st = torch.zeros((w.B, w.H, hla.hla2_state_floats(w.d, w.dv)), dtype=torch.float32, device=DEV)
    tq, tk, tv = (hla_inputs.as_torch(x, w.dtype, DEV) for x in (qp, kp, vp))
    hla.hla2_forward(tq, tk, tv, masked=w.masked, normalized=w.normalized, eps=hla_inputs.EPS, chunk=w.chunk,
                     state_out=st)
    del tq, tk, tv
    outs = []
    for s in range(steps):
        o = hla.hla2_step(hla_inputs.as_torch(qs[s], w.dtype, DEV), hla_inputs.as_torch(ks[s], w.dtype, DEV),
                          hla_inputs.as_torch(vs[s], w.dtype, DEV), st, masked=w.masked, normalized=w.normalized,
                          eps=hla_inputs.EPS)
        outs.append(o.float().cpu().numpy().reshape(w.BH, w.dv))
    torch.cuda.synchronize()
    heads = [0, 700, 1300, w.BH - 1]
    got = np.stack(outs, axis=1)[heads]
    gst = st.cpu().numpy().reshape(w.BH, -1)[heads]
    cat = [np.concatenate([p.reshape(w.BH, w.decode_prefix, -1)[heads],
                           np.moveaxis(x.reshape(steps, w.BH, -1), 0, 1)[heads]], axis=1) for p, x in
           ((qp, qs), (kp, ks), (vp, vs))]
    ref, rst = oracle.hla2_serial(*cat, masked=w.masked, normalized=w.normalized, eps=hla_inputs.EPS,
                                  return_state=True, nthreads=4)
    err = rowerr(got, ref[:, w.decode_prefix:])
    print("\ndecode at depth %d, %d steps, heads %s: row error %s" % (w.decode_prefix, steps, heads,
                                                                      rowerr_stats(got, ref[:, w.decode_prefix:])[0]))
    assert err < TOL["bf16"], err
    pg, pr = oracle.split_state2(gst, w.d, w.dv), oracle.split_state2(rst, w.d, w.dv)
    for name in ("S", "C", "m", "G", "h"):
        scale = max(np.abs(pr[name]).max(), np.abs(pr["S"]).max() * np.abs(pr["C"]).max())
        assert np.abs(pg[name] - pr[name]).max() <= 2e-5 * max(scale, 1.0), name


def test_decode_workload_shape_sampled(hla):
    """The decode workload's shape (B64 H32 d128, bf16 tokens, fp32 state) with
    a shortened prefix; the oracle checks sampled heads."""
    w = hla_inputs.WORKLOADS["decode_bf16"]
    heads = [0, 1000, w.BH - 1]
    got, ref, _, _ = _decode_run(hla, w.B, w.H, w.d, w.dv, 256, 4, w.dtype, w.masked, w.normalized, seed=w.seed,
                                 heads=heads)
    assert rowerr(got, ref) < 2e-2
