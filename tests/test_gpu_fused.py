"""The fused tcgen05 forward (bf16, masked; d and dv in {64, 128}, 64 running as
zero-padded 128; 128-token tiles for any requested chunk) against the fp64
oracle, including its cross-SM chained scans (forced short segments), ragged
tails, an initial state, and the device-side timeout path."""
import numpy as np
import pytest
import torch

import hla_inputs
import oracle
from parity import check_normalized, rowerr

pytestmark = pytest.mark.gpu
DEV = "cuda:0"


@pytest.fixture(scope="module")
def hla():
    from paper_2510_27258_gb300 import build
    build.build()
    from paper_2510_27258_gb300 import hla as binding
    return binding


def run(hla, q, k, v, normalized, state_in=None, chunk=128, masked=True):
    tq, tk, tv = (hla_inputs.as_torch(x, "bf16", DEV) for x in (q, k, v))
    sin = None if state_in is None else torch.from_numpy(np.ascontiguousarray(state_in, np.float32)).to(DEV)
    ws = hla.alloc_workspace(hla.hla2_workspace_bytes(*q.shape, v.shape[-1], chunk, torch.bfloat16), DEV)
    out = hla.hla2_forward(tq, tk, tv, masked=masked, normalized=normalized, eps=hla_inputs.EPS, chunk=chunk,
                           state_in=sin, workspace=ws)
    torch.cuda.synchronize()
    assert hla.hla_poll_error(ws) == 0
    B, H, n, _ = q.shape
    return out.float().cpu().numpy().reshape(B * H, n, -1)


def check(hla, q, k, v, normalized, state_in=None, chunk=128):
    B, H, n, d = q.shape
    dv = v.shape[-1]
    assert hla.hla2_forward_path(B, H, n, d, dv, normalized=normalized, chunk=chunk,
                                 has_state_in=state_in is not None)[0] == 1
    sin = None if state_in is None else np.asarray(state_in, np.float64).reshape(B * H, -1)
    num_ref, den_ref = oracle.hla2_serial(q.reshape(B * H, n, d), k.reshape(B * H, n, d), v.reshape(B * H, n, dv),
                                          masked=True, normalized=False, state_in=sin, return_den=True, nthreads=8)
    num = run(hla, q, k, v, False, state_in, chunk)
    if not normalized:
        err = rowerr(num, num_ref)
        assert err < 2e-2, err
        return err
    o = run(hla, q, k, v, True, state_in, chunk)
    return check_normalized(o, num, num_ref, den_ref, hla_inputs.EPS, 2e-2)


def test_fused_path_selected(hla):
    assert hla.hla2_forward_path(2, 16, 16384, 128, 128, normalized=True) == (1, 1)
    assert hla.hla2_forward_path(2, 16, 16384, 128, 128, normalized=True, has_state_out=True) == (1, 3)
    assert hla.hla2_forward_path(2, 16, 16384, 128, 128, has_state_in=True, has_state_out=True) == (1, 4)
    # unmasked: plain output, one segment per head, no state
    assert hla.hla2_forward_path(2, 16, 16384, 128, 128, masked=False) == (1, 1)
    assert hla.hla2_forward_path(2, 16, 16384, 128, 128, masked=False, normalized=True)[0] == 0
    assert hla.hla2_forward_path(2, 16, 16384, 128, 128, masked=False, has_state_out=True)[0] == 0
    assert hla.hla2_forward_path(2, 16, 16384, 128, 128, masked=False, has_state_in=True)[0] == 0
    # d, dv of 64 as zero-padded 128, any chunk; an initial state only in the 128 x 128 layout
    assert hla.hla2_forward_path(8, 16, 2048, 64, 64, chunk=64) == (1, 1)
    assert hla.hla2_forward_path(1, 1, 100, 64, 128, chunk=7)[0] == 1
    assert hla.hla2_forward_path(1, 1, 100, 128, 64, chunk=128)[0] == 1
    assert hla.hla2_forward_path(1, 1, 100, 128, 128, chunk=32, has_state_in=True)[0] == 1
    assert hla.hla2_forward_path(1, 1, 100, 64, 64, has_state_in=True)[0] == 0
    assert hla.hla2_forward_path(1, 1, 100, 32, 32)[0] == 0
    assert hla.hla2_forward_path(1, 1, 100, 128, 128, dtype=torch.float32)[0] == 0


@pytest.mark.parametrize("d,dv", [(64, 64), (64, 128), (128, 64)])
@pytest.mark.parametrize("B,H,n,chunk", [(1, 1, 1, 64), (1, 2, 129, 64), (2, 3, 600, 128), (1, 1, 1000, 32)])
@pytest.mark.parametrize("seg", ["1", "default"])
@pytest.mark.parametrize("normalized", [False, True])
def test_fused_head_size_64(hla, monkeypatch, d, dv, B, H, n, chunk, seg, normalized):
    """Head sizes of 64: d = dv = 64 has its own instantiation (products over 64 features), mixes run as
    128 with zero features; the requested chunk changes nothing but rounding."""
    if seg != "default":
        monkeypatch.setenv("HLA_FUSED_SEGMENT_TILES", seg)
    q, k, v = hla_inputs.make_qkv(B, H, n, d, dv, seed=n + 31 * d + dv, dtype="bf16")
    check(hla, q, k, v, normalized, chunk=chunk)


@pytest.mark.parametrize("B,H,n", [(1, 1, 1), (1, 2, 127), (1, 2, 128), (1, 3, 129), (2, 2, 600), (1, 1, 2000)])
@pytest.mark.parametrize("seg", ["1", "2", "3", "default"])
@pytest.mark.parametrize("normalized", [False, True])
def test_fused_matches_oracle(hla, monkeypatch, B, H, n, seg, normalized):
    if seg != "default":
        monkeypatch.setenv("HLA_FUSED_SEGMENT_TILES", seg)
    q, k, v = hla_inputs.make_qkv(B, H, n, 128, 128, seed=n + 17 * H, dtype="bf16")
    check(hla, q, k, v, normalized)


@pytest.mark.parametrize("seg", ["1", "default"])
def test_fused_initial_state(hla, monkeypatch, seg):
    if seg != "default":
        monkeypatch.setenv("HLA_FUSED_SEGMENT_TILES", seg)
    B, H, d = 1, 2, 128
    pq, pk, pv = hla_inputs.make_qkv(B, H, 300, d, d, seed=5, dtype="bf16")
    _, st0 = oracle.hla2_serial(pq.reshape(B * H, 300, d), pk.reshape(B * H, 300, d), pv.reshape(B * H, 300, d),
                                masked=True, return_state=True)
    st0 = st0.astype(np.float32)
    q, k, v = hla_inputs.make_qkv(B, H, 400, d, d, seed=6, dtype="bf16")
    check(hla, q, k, v, True, state_in=st0)
    check(hla, q, k, v, False, state_in=st0)


@pytest.mark.parametrize("d", [64, 128])
@pytest.mark.parametrize("normalized", [False, True])
def test_fused_one_segment_per_head(hla, d, normalized):
    """80 heads (at least half the SMs): the kernel gives each head one segment (no chains, no
    fix-up), including the ragged last tile; every head against the oracle."""
    q, k, v = hla_inputs.make_qkv(2, 40, 300, d, d, seed=77 + d, dtype="bf16")
    check(hla, q, k, v, normalized)


def test_fused_deterministic(hla, monkeypatch):
    monkeypatch.setenv("HLA_FUSED_SEGMENT_TILES", "2")
    q, k, v = hla_inputs.make_qkv(2, 3, 1500, 128, 128, seed=21, dtype="bf16")
    a = run(hla, q, k, v, True)
    b = run(hla, q, k, v, True)
    assert np.array_equal(a, b)


def test_fused_equals_generic_closely(hla, monkeypatch):
    """Both CUDA paths on the same inputs (the generic one in fp32 SIMT)."""
    q, k, v = hla_inputs.make_qkv(1, 2, 700, 128, 128, seed=31, dtype="bf16")
    a = run(hla, q, k, v, False)
    monkeypatch.setenv("HLA_DISABLE_FUSED", "1")
    b = run(hla, q, k, v, False)
    assert rowerr(a, b) < 2e-2


def test_fused_causality_bit_exact(hla):
    B, H, n, t = 1, 2, 700, 300
    q, k, v = hla_inputs.make_qkv(B, H, n, 128, 128, seed=40, dtype="bf16")
    a = run(hla, q, k, v, True)
    rng = np.random.default_rng(1)
    q2, k2, v2 = q.copy(), k.copy(), v.copy()
    for x in (q2, k2, v2):
        x[:, :, t + 1:] = hla_inputs.round_to(rng.standard_normal(x[:, :, t + 1:].shape), "bf16")
    b = run(hla, q2, k2, v2, True)
    assert np.array_equal(a[:, : t + 1], b[:, : t + 1])


def test_fused_wait_timeout_is_reported_not_hung(hla, monkeypatch):
    """A segment that never publishes its S prefix (injected on the host side):
    the next segment's bounded wait runs out, the kernel finishes, and
    hla_poll_error reports HLA_ERR_TIMEOUT; the workspace then works again."""
    monkeypatch.setenv("HLA_FUSED_SEGMENT_TILES", "1")
    monkeypatch.setenv("HLA_TEST_WAIT_NS", "20000000")     # 20 ms budget
    monkeypatch.setenv("HLA_TEST_SKIP_PUBLISH_ITEM", "0")  # (head 0, segment 0) skips its publish
    q, k, v = hla_inputs.make_qkv(1, 1, 512, 128, 128, seed=50, dtype="bf16")
    tq, tk, tv = (hla_inputs.as_torch(x, "bf16", DEV) for x in (q, k, v))
    ws = hla.alloc_workspace(hla.hla2_workspace_bytes(1, 1, 512, 128, 128, 128, torch.bfloat16), DEV)
    hla.hla2_forward(tq, tk, tv, masked=True, normalized=False, chunk=128, workspace=ws)
    assert hla.hla_poll_error(ws) == hla.HLA_ERR_TIMEOUT
    monkeypatch.delenv("HLA_TEST_SKIP_PUBLISH_ITEM")
    out = hla.hla2_forward(tq, tk, tv, masked=True, normalized=False, chunk=128, workspace=ws)
    assert hla.hla_poll_error(ws) == hla.HLA_OK
    ref = oracle.hla2_serial(q.reshape(1, 512, 128), k.reshape(1, 512, 128), v.reshape(1, 512, 128), masked=True)
    assert rowerr(out.float().cpu().numpy().reshape(1, 512, 128), ref) < 2e-2


@pytest.mark.parametrize("d,dv", [(128, 128), (64, 64), (64, 128)])
@pytest.mark.parametrize("n,seg", [(1, "default"), (200, "1"), (700, "2"), (1000, "default")])
@pytest.mark.parametrize("normalized", [False, True])
def test_fused_state_out(hla, monkeypatch, d, dv, n, seg, normalized):
    """The final state tuple written by the fused path against the oracle's (parts S, C, m, G, h)."""
    if seg != "default":
        monkeypatch.setenv("HLA_FUSED_SEGMENT_TILES", seg)
    B, H = 1, 2
    q, k, v = hla_inputs.make_qkv(B, H, n, d, dv, seed=n + d + dv, dtype="bf16")
    assert hla.hla2_forward_path(B, H, n, d, dv, normalized=normalized, has_state_out=True)[0] == 1
    tq, tk, tv = (hla_inputs.as_torch(x, "bf16", DEV) for x in (q, k, v))
    st = torch.zeros((B, H, hla.hla2_state_floats(d, dv)), dtype=torch.float32, device=DEV)
    out = hla.hla2_forward(tq, tk, tv, masked=True, normalized=normalized, eps=hla_inputs.EPS, chunk=128, state_out=st)
    torch.cuda.synchronize()
    num_ref, rst = oracle.hla2_serial(q.reshape(B * H, n, d), k.reshape(B * H, n, d), v.reshape(B * H, n, dv),
                                      masked=True, normalized=False, return_state=True, nthreads=4)
    if not normalized:
        assert rowerr(out.float().cpu().numpy().reshape(B * H, n, dv), num_ref) < 2e-2
    gst = st.cpu().numpy().reshape(B * H, -1)
    parts_g, parts_r = oracle.split_state2(gst, d, dv), oracle.split_state2(rst, d, dv)
    for name in ("S", "C", "m", "G", "h"):
        scale = max(np.abs(parts_r[name]).max(), np.abs(parts_r["S"]).max() * np.abs(parts_r["C"]).max())
        err = np.abs(parts_g[name] - parts_r[name]).max()
        assert err <= 2e-5 * max(scale, 1.0), (name, err, scale)


@pytest.mark.parametrize("alias", [False, True])
def test_fused_state_in_out(hla, monkeypatch, alias):
    """state_in -> forward -> state_out on the fused path (state_out may be state_in), and the
    next chunk of the sequence from that state equals the whole sequence at once."""
    monkeypatch.setenv("HLA_FUSED_SEGMENT_TILES", "1")
    B, H, n1, n2, d = 1, 2, 300, 260, 128
    q, k, v = hla_inputs.make_qkv(B, H, n1 + n2, d, d, seed=77, dtype="bf16")
    tq, tk, tv = (hla_inputs.as_torch(x, "bf16", DEV) for x in (q, k, v))
    st1 = torch.zeros((B, H, hla.hla2_state_floats(d, d)), dtype=torch.float32, device=DEV)
    hla.hla2_forward(tq[:, :, :n1].contiguous(), tk[:, :, :n1].contiguous(), tv[:, :, :n1].contiguous(),
                     masked=True, chunk=128, state_out=st1)
    st2 = st1 if alias else torch.zeros_like(st1)
    out2 = hla.hla2_forward(tq[:, :, n1:].contiguous(), tk[:, :, n1:].contiguous(), tv[:, :, n1:].contiguous(),
                            masked=True, chunk=128, state_in=st1, state_out=st2)
    torch.cuda.synchronize()
    num_ref, rst = oracle.hla2_serial(q.reshape(B * H, -1, d), k.reshape(B * H, -1, d), v.reshape(B * H, -1, d),
                                      masked=True, normalized=False, return_state=True, nthreads=4)
    assert rowerr(out2.float().cpu().numpy().reshape(B * H, n2, d), num_ref[:, n1:]) < 2e-2
    parts_g, parts_r = oracle.split_state2(st2.cpu().numpy().reshape(B * H, -1), d, d), oracle.split_state2(rst, d, d)
    for name in ("S", "C", "m", "G", "h"):
        scale = max(np.abs(parts_r[name]).max(), np.abs(parts_r["S"]).max() * np.abs(parts_r["C"]).max())
        assert np.abs(parts_g[name] - parts_r[name]).max() <= 2e-5 * max(scale, 1.0), name


@pytest.mark.parametrize("d,dv", [(64, 64), (128, 128), (64, 128), (128, 64)])
@pytest.mark.parametrize("B,H,n", [(1, 1, 1), (1, 2, 129), (2, 3, 600), (1, 1, 1000)])
@pytest.mark.parametrize("normalized", [False, True])
def test_fused_unmasked(hla, d, dv, B, H, n, normalized):
    """The unmasked operator (online updates after Theorem 1 without G, h): the plain output on the
    fused kernel (T = L . (X Q^T), O = T V + X C_p, one segment per head), the ratio-normalised one
    on the fp32 path."""
    assert hla.hla2_forward_path(B, H, n, d, dv, masked=False, chunk=128) == (1, 1)
    assert hla.hla2_forward_path(B, H, n, d, dv, masked=False, normalized=True, chunk=128)[0] == 0
    q, k, v = hla_inputs.make_qkv(B, H, n, d, dv, seed=7700 + n + d + 3 * dv, dtype="bf16")
    flat = lambda x: x.reshape(B * H, n, -1)
    num_ref, den_ref = oracle.hla2_serial(flat(q), flat(k), flat(v), masked=False, normalized=False,
                                          return_den=True, nthreads=8)
    num = run(hla, q, k, v, False, masked=False)
    err = rowerr(num, num_ref)
    assert err < 2e-2, err
    if normalized:
        o = run(hla, q, k, v, True, masked=False)
        check_normalized(o, num, num_ref, den_ref, hla_inputs.EPS, 2e-2)
