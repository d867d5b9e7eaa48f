"""fp64 CPU oracle for Higher-order Linear Attention -- TEST INFRASTRUCTURE.

The oracle is the plain, slow, obviously-correct reference that the CUDA path
is checked against.  Only the test suite, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` may import it; the library in
``paper_2510_27258_gb300`` never does, and this package never imports that
library.  The two share no code.

The arithmetic lives in ``hla_oracle.c`` (C99, fp64, POSIX threads over heads);
this module only builds it with gcc and marshals numpy arrays.  Each function
names the passage of the paper it follows:

* :func:`hla2_serial`   -- online updates after Theorem 1 and the outputs of
  Theorem 1 (masked) / Eq. hla-unnorm, Eq. hla-row (unmasked).
* :func:`hla2_combine`  -- the masked semidirect product, Eq. semidirect
  (unmasked: the additive monoid of Sec. 4.1).
* :func:`hla2_chunked`  -- Theorem 2: exclusive Blelloch scans within and
  across chunks, then local inclusion of the token segment.
* :func:`hla3_serial`   -- Algorithm 3 at gamma = 1 (masked) and the unmasked
  third-order factorisation of Sec. 7.1.
* :func:`hla3_chunked`  -- Theorem 4 / Algorithm 4 with the segment maps
  applied by contraction.
* :func:`hla2_state_to_sde` -- the masked tuple folded to (S, D = SC - G,
  e = Sm - h), the quantities Theorem 1's outputs read.
* :func:`ahla_serial`   -- the AHLA online updates (Theorem AHLA, Algorithm
  AHLA-stream at gamma = 1).
* :func:`ahla_combine`  -- Eq. AHLA-semidirect on (R, P, m, E, n).
* :func:`ahla_chunked`  -- the AHLA scan route (exclusive Blelloch scans
  under the AHLA product, then local inclusion; scan equivalence).
* :func:`hla2_backward` -- gradients of second-order HLA by a reverse sweep
  over the online updates, forward states checkpointed at tile boundaries
  (Sec. "Chunk-parallel training via associative scans").

Array conventions: q, k are ``[BH, n, d]``, v is ``[BH, n, dv]``; outputs are
``[BH, n, dv]``; the state tuple of one head is laid out as in
:func:`hla2_state_len`.  Inputs are converted to C-contiguous float64.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "hla_oracle.c")
_LIB_PATH = os.path.join(_HERE, "libhla_oracle.so")
_lock = threading.Lock()
_lib = None

_dp = ctypes.POINTER(ctypes.c_double)


def build(force: bool = False, src: str = _SRC, out: str = _LIB_PATH) -> str:
    """Compile the oracle with gcc (-O2, no fast-math: plain IEEE fp64)."""
    if (not force and os.path.exists(out)
            and os.path.getmtime(out) >= os.path.getmtime(src)):
        return out
    tmp = out + ".tmp%d" % os.getpid()
    cmd = ["gcc", "-O2", "-std=c99", "-fno-fast-math", "-ffp-contract=off", "-shared", "-fPIC",
           "-pthread", "-o", tmp, src, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, out)
    return out


def load(path: str | None = None):
    """Load (building first if needed) the oracle shared library."""
    global _lib
    with _lock:
        if path is not None:
            return _bind(ctypes.CDLL(path))
        if _lib is None:
            _lib = _bind(ctypes.CDLL(build()))
        return _lib


def _bind(lib):
    i, d = ctypes.c_int, ctypes.c_double
    lib.hla2_serial_f64.argtypes = [_dp, _dp, _dp, _dp, _dp, i, i, i, i, i, i, d, _dp, _dp, i]
    lib.hla2_serial_f64.restype = i
    lib.hla2_chunked_f64.argtypes = [_dp, _dp, _dp, _dp, _dp, i, i, i, i, i, i, d, i, _dp, _dp, i]
    lib.hla2_chunked_f64.restype = i
    lib.hla2_combine_f64.argtypes = [_dp, _dp, _dp, i, i, i]
    lib.hla2_combine_f64.restype = None
    lib.hla2_state_len_f64.argtypes = [i, i]
    lib.hla2_state_len_f64.restype = ctypes.c_size_t
    lib.hla3_serial_f64.argtypes = [_dp, _dp, _dp, _dp, _dp, i, i, i, i, i, i, d, _dp, _dp, i]
    lib.hla3_serial_f64.restype = i
    lib.hla3_chunked_f64.argtypes = [_dp, _dp, _dp, _dp, _dp, i, i, i, i, i, d, i, i]
    lib.hla3_chunked_f64.restype = i
    lib.hla3_state_len_f64.argtypes = [i, i]
    lib.hla3_state_len_f64.restype = ctypes.c_size_t
    lib.hla2_state_to_sde_f64.argtypes = [_dp, _dp, i, i, i]
    lib.hla2_state_to_sde_f64.restype = None
    lib.ahla_serial_f64.argtypes = [_dp, _dp, _dp, _dp, _dp, i, i, i, i, i, d, _dp, _dp, i]
    lib.ahla_serial_f64.restype = i
    lib.ahla_chunked_f64.argtypes = [_dp, _dp, _dp, _dp, _dp, i, i, i, i, i, i, d, i]
    lib.ahla_chunked_f64.restype = i
    lib.ahla_combine_f64.argtypes = [_dp, _dp, _dp, i, i]
    lib.ahla_combine_f64.restype = None
    lib.hla2_backward_f64.argtypes = [_dp, _dp, _dp, _dp, _dp, _dp, _dp, i, i, i, i, i, i, d, i, i]
    lib.hla2_backward_f64.restype = i
    return lib


def _f64(x):
    return np.ascontiguousarray(np.asarray(x, dtype=np.float64))


def _ptr(x):
    return None if x is None else x.ctypes.data_as(_dp)


def _shapes(q, k, v):
    q, k, v = _f64(q), _f64(k), _f64(v)
    if q.ndim == 2:
        q, k, v = q[None], k[None], v[None]
    BH, n, d = q.shape
    dv = v.shape[2]
    assert k.shape == (BH, n, d) and v.shape == (BH, n, dv)
    return q, k, v, BH, n, d, dv


def hla2_state_len(d: int, dv: int) -> int:
    """Length of one head's second-order state tuple ``[S | C | m | G | h]``:
    d*d + d*dv + d + d*dv + d (Fig. 1(A))."""
    return d * d + 2 * d * dv + 2 * d


def hla3_state_len(d: int, dv: int) -> int:
    """Length of ``[SK | SQ | P | mK | G1 | G2 | G3 | h1 | h2 | h3]`` (Theorem 3)."""
    return 2 * d * d + 4 * d * dv + 4 * d


def split_state2(st, d: int, dv: int) -> dict:
    """View a (..., hla2_state_len) array as its named parts S, C, m, G, h."""
    st = np.asarray(st)
    o = 0
    parts = {}
    for name, size, shape in (("S", d * d, (d, d)), ("C", d * dv, (d, dv)), ("m", d, (d,)),
                              ("G", d * dv, (d, dv)), ("h", d, (d,))):
        parts[name] = st[..., o:o + size].reshape(st.shape[:-1] + shape)
        o += size
    return parts


def pack_state2(S, C, m, G, h):
    """Inverse of :func:`split_state2` for one or more heads."""
    lead = np.asarray(m).shape[:-1]
    return np.concatenate([np.reshape(S, lead + (-1,)), np.reshape(C, lead + (-1,)), np.reshape(m, lead + (-1,)),
                           np.reshape(G, lead + (-1,)), np.reshape(h, lead + (-1,))], axis=-1)


def hla2_serial(q, k, v, masked=True, normalized=False, eps=1e-6, state_in=None, return_state=False,
                return_den=False, nthreads=1):
    """Serial fp64 second-order HLA (online updates after Theorem 1).

    Returns ``out`` (and, as requested, ``den`` of shape [BH, n] and the final
    state tuple of shape [BH, hla2_state_len]).  ``den`` is the masked (or
    unmasked) denominator WITHOUT eps.
    """
    q, k, v, BH, n, d, dv = _shapes(q, k, v)
    out = np.zeros((BH, n, dv))
    den = np.zeros((BH, n)) if return_den else None
    st_in = None if state_in is None else _f64(state_in).reshape(BH, hla2_state_len(d, dv))
    st_out = np.zeros((BH, hla2_state_len(d, dv))) if return_state else None
    rc = load().hla2_serial_f64(_ptr(q), _ptr(k), _ptr(v), _ptr(out), _ptr(den), BH, n, d, dv, int(masked),
                                int(normalized), float(eps), _ptr(st_in), _ptr(st_out), int(nthreads))
    assert rc == 0
    res = [out]
    if return_den:
        res.append(den)
    if return_state:
        res.append(st_out)
    return res[0] if len(res) == 1 else tuple(res)


def hla2_chunked(q, k, v, chunk, masked=True, normalized=False, eps=1e-6, state_in=None, return_state=False,
                 return_den=False, nthreads=1):
    """fp64 second-order HLA through the two-level exclusive scan of Theorem 2."""
    q, k, v, BH, n, d, dv = _shapes(q, k, v)
    out = np.zeros((BH, n, dv))
    den = np.zeros((BH, n)) if return_den else None
    st_in = None if state_in is None else _f64(state_in).reshape(BH, hla2_state_len(d, dv))
    st_out = np.zeros((BH, hla2_state_len(d, dv))) if return_state else None
    rc = load().hla2_chunked_f64(_ptr(q), _ptr(k), _ptr(v), _ptr(out), _ptr(den), BH, n, d, dv, int(masked),
                                 int(normalized), float(eps), int(chunk), _ptr(st_in), _ptr(st_out),
                                 int(nthreads))
    assert rc == 0
    res = [out]
    if return_den:
        res.append(den)
    if return_state:
        res.append(st_out)
    return res[0] if len(res) == 1 else tuple(res)


def hla2_combine(A, B, d, dv, masked=True):
    """``A (+) B`` for adjacent segments, A first (Eq. semidirect)."""
    A, B = _f64(A), _f64(B)
    out = np.zeros(hla2_state_len(d, dv))
    load().hla2_combine_f64(_ptr(A), _ptr(B), _ptr(out), d, dv, int(masked))
    return out


def hla3_serial(q, k, v, masked=True, normalized=False, eps=1e-6, state_in=None, return_state=False,
                return_den=False, nthreads=1):
    """Serial fp64 third-order HLA (Algorithm 3 at gamma = 1; unmasked: Sec. 7.1)."""
    q, k, v, BH, n, d, dv = _shapes(q, k, v)
    out = np.zeros((BH, n, dv))
    den = np.zeros((BH, n)) if return_den else None
    st_in = None if state_in is None else _f64(state_in).reshape(BH, hla3_state_len(d, dv))
    st_out = np.zeros((BH, hla3_state_len(d, dv))) if return_state else None
    rc = load().hla3_serial_f64(_ptr(q), _ptr(k), _ptr(v), _ptr(out), _ptr(den), BH, n, d, dv, int(masked),
                                int(normalized), float(eps), _ptr(st_in), _ptr(st_out), int(nthreads))
    assert rc == 0
    res = [out]
    if return_den:
        res.append(den)
    if return_state:
        res.append(st_out)
    return res[0] if len(res) == 1 else tuple(res)


def hla3_chunked(q, k, v, chunk, normalized=False, eps=1e-6, return_den=False, nthreads=1):
    """fp64 masked third-order HLA through the scan of Theorem 4 / Algorithm 4."""
    q, k, v, BH, n, d, dv = _shapes(q, k, v)
    out = np.zeros((BH, n, dv))
    den = np.zeros((BH, n)) if return_den else None
    rc = load().hla3_chunked_f64(_ptr(q), _ptr(k), _ptr(v), _ptr(out), _ptr(den), BH, n, d, dv, int(normalized),
                                 float(eps), int(chunk), int(nthreads))
    assert rc == 0
    return (out, den) if return_den else out


def hla2_sde_len(d: int, dv: int) -> int:
    """Length of one head's (S, D, e) state: d*d + d*dv + d."""
    return d * d + d * dv + d


def hla2_state_to_sde(st, d: int, dv: int):
    """(S, C, m, G, h) tuples [..., hla2_state_len] -> (S, D = S C - G, e = S m - h) [..., hla2_sde_len]."""
    st = _f64(st)
    lead = st.shape[:-1]
    flat = np.ascontiguousarray(st.reshape(-1, hla2_state_len(d, dv)))
    out = np.zeros((flat.shape[0], hla2_sde_len(d, dv)))
    load().hla2_state_to_sde_f64(_ptr(flat), _ptr(out), flat.shape[0], d, dv)
    return out.reshape(lead + (hla2_sde_len(d, dv),))


def ahla_state_len(d: int, dv: int) -> int:
    """Length of one head's AHLA streaming state [P | m | E | n]: 2 d dv + 2 d."""
    return 2 * d * dv + 2 * d


def ahla_summary_len(d: int, dv: int) -> int:
    """Length of an AHLA segment summary [R | P | m | E | n]: d*d + 2 d dv + 2 d."""
    return d * d + ahla_state_len(d, dv)


def ahla_serial(q, k, v, normalized=False, eps=1e-6, state_in=None, return_state=False, return_den=False,
                nthreads=1):
    """Serial fp64 AHLA (Theorem AHLA online updates): out [BH, n, dv] (and, as requested, den [BH, n]
    without eps and the final state [BH, ahla_state_len])."""
    q, k, v, BH, n, d, dv = _shapes(q, k, v)
    out = np.zeros((BH, n, dv))
    den = np.zeros((BH, n)) if return_den else None
    sin = None if state_in is None else _f64(state_in).reshape(BH, ahla_state_len(d, dv))
    sout = np.zeros((BH, ahla_state_len(d, dv))) if return_state else None
    rc = load().ahla_serial_f64(_ptr(q), _ptr(k), _ptr(v), _ptr(out), _ptr(den), BH, n, d, dv, int(normalized),
                                float(eps), _ptr(sin), _ptr(sout), int(nthreads))
    assert rc == 0
    res = (out,)
    if return_den:
        res += (den,)
    if return_state:
        res += (sout,)
    return res[0] if len(res) == 1 else res


def ahla_chunked(q, k, v, chunk, normalized=False, eps=1e-6, return_den=False, nthreads=1):
    """AHLA by exclusive scans under Eq. AHLA-semidirect (scan equivalence)."""
    q, k, v, BH, n, d, dv = _shapes(q, k, v)
    out = np.zeros((BH, n, dv))
    den = np.zeros((BH, n)) if return_den else None
    rc = load().ahla_chunked_f64(_ptr(q), _ptr(k), _ptr(v), _ptr(out), _ptr(den), BH, n, d, dv, int(chunk),
                                 int(normalized), float(eps), int(nthreads))
    assert rc == 0
    return (out, den) if return_den else out


def ahla_combine(A, B, d, dv):
    """A (+)_AHLA B on summaries [R | P | m | E | n] (Eq. AHLA-semidirect)."""
    A, B = _f64(A), _f64(B)
    out = np.zeros(ahla_summary_len(d, dv))
    load().ahla_combine_f64(_ptr(A), _ptr(B), _ptr(out), d, dv)
    return out


def hla2_backward(q, k, v, dout, masked=True, normalized=False, eps=1e-6, ckpt=64, nthreads=1):
    """Gradients (dq, dk, dv) of L = sum_t dout_t . o_t for second-order HLA from a zero state, by the
    reverse sweep of the online updates with checkpoints every `ckpt` tokens."""
    q, k, v, BH, n, d, dv = _shapes(q, k, v)
    g = _f64(dout).reshape(BH, n, dv)
    dq, dk, dvv = np.zeros((BH, n, d)), np.zeros((BH, n, d)), np.zeros((BH, n, dv))
    rc = load().hla2_backward_f64(_ptr(q), _ptr(k), _ptr(v), _ptr(g), _ptr(dq), _ptr(dk), _ptr(dvv), BH, n, d, dv,
                                  int(masked), int(normalized), float(eps), int(ckpt), int(nthreads))
    assert rc == 0
    return dq, dk, dvv
