"""CPU oracle for the Ember optimizer step (numpy front end to ember_oracle.c).

TEST INFRASTRUCTURE ONLY.  Only tests/, __graft_entry__.smoke() and the CPU
baseline leg of bench.py may import this package.  It shares no code with the
CUDA library and never imports it.

Every function follows Algorithm 1 ("Ember") of "Token Geometry"
(arXiv 2607.01455, Section 2.1) and, for the sparse step, Section 2.2.
Arrays are numpy and are updated in place:

* ``W``: V x D, ``np.float32`` or bfloat16 bit patterns as ``np.uint16``;
* ``G``: V x D ``np.float32``; ``rows``: N x D ``np.float32``;
* ``ids``: N ``np.int64`` token ids;
* ``r``: V ``np.float32``; ``c``: D ``np.float32`` (the whole optimizer state);
* ``dlogits``: T x V and ``hidden``: T x D, bfloat16 bit patterns (``np.uint16``),
  the two factors of an LM head's gradient.

Parity status: every function is pinned by tests/test_oracle_pins.py except
the behaviour of gradients so small that g^2 or the fp32 state underflows,
which is "parity unpinned".
"""
import ctypes
import os

import numpy as np

from .build import build_oracle

_VARIANTS = {"full": 0, "row": 1, "col": 2}
_lib = None


_lib_omp = None


def _load():
    global _lib
    if _lib is None:
        # EMBER_ORACLE_LIB lets the mutation test load a deliberately broken copy.
        _lib = _bind(ctypes.CDLL(os.environ.get("EMBER_ORACLE_LIB") or build_oracle()))
    return _lib


def _load_omp():
    """The same source built with -fopenmp (for the all-cores CPU baseline)."""
    global _lib_omp
    if _lib_omp is None:
        _lib_omp = _bind(ctypes.CDLL(build_oracle(openmp=True)))
    return _lib_omp


def _bind(lib):
    i64, dbl, vp, ip = ctypes.c_int64, ctypes.c_double, ctypes.c_void_p, ctypes.c_int
    lib.ember_oracle_step_dense.argtypes = [
        i64, i64, ip, vp, vp, vp, vp, dbl, i64, dbl, dbl, ip, ip, ip, vp]
    lib.ember_oracle_step_dense.restype = ip
    lib.ember_oracle_step_sparse.argtypes = [
        i64, i64, ip, vp, i64, vp, vp, vp, vp, dbl, i64, dbl, dbl, ip, ip, ip, vp]
    lib.ember_oracle_step_sparse.restype = ip
    lib.ember_oracle_dedup.argtypes = [i64, vp, i64, vp, vp]
    lib.ember_oracle_dedup.restype = i64
    lib.ember_oracle_round_bf16.argtypes = [i64, vp, vp]
    lib.ember_oracle_round_bf16.restype = None
    lib.ember_oracle_bf16_to_double.argtypes = [i64, vp, vp]
    lib.ember_oracle_bf16_to_double.restype = None
    lib.ember_oracle_lmhead_grad.argtypes = [i64, i64, i64, vp, vp, i64, vp, vp, vp]
    lib.ember_oracle_lmhead_grad.restype = ip
    lib.ember_oracle_threads.argtypes = [ip]
    lib.ember_oracle_threads.restype = ip
    return lib


def _ptr(a):
    return a.ctypes.data_as(ctypes.c_void_p)


def _check_state(W, r, c):
    if W.ndim != 2:
        raise ValueError("W must be V x D")
    V, D = W.shape
    if W.dtype not in (np.float32, np.uint16):
        raise TypeError("W must be float32 or bfloat16 bits (uint16)")
    for name, a, n in (("r", r, V), ("c", c, D)):
        if a.dtype != np.float32 or a.shape != (n,):
            raise ValueError(f"{name} must be float32 of length {n}")
    for a in (W, r, c):
        if not a.flags.c_contiguous or not a.flags.writeable:
            raise ValueError("W, r, c must be writeable C-contiguous arrays")
    return V, D


def _diag(d):
    return {"bc": d[0], "rbar": d[1], "cbar": d[2], "s": d[3], "zero_rows": int(d[4])}


def threads(n=0):
    """Threads of the all-cores build: n > 0 sets the count; returns it."""
    return _load_omp().ember_oracle_threads(int(n))


def step_dense(W, G, r, c, lr, t, beta2=0.999, eps=1e-8, maximize=False,
               bias_correction=True, variant="full", all_cores=False):
    """One dense Ember step (Algorithm 1) in place on W, r, c; returns the
    step's scalars (1-beta2^t, mean rhat, mean chat, s, zero rows).
    all_cores=True runs the OpenMP build of the same source (see threads());
    it gives the same bits."""
    V, D = _check_state(W, r, c)
    G = np.ascontiguousarray(G, dtype=np.float32)
    if G.shape != (V, D):
        raise ValueError("G must have W's shape")
    d = np.zeros(5, np.float64)
    lib = _load_omp() if all_cores else _load()
    rc = lib.ember_oracle_step_dense(
        V, D, int(W.dtype == np.uint16), _ptr(W), _ptr(G), _ptr(r), _ptr(c),
        float(lr), int(t), float(beta2), float(eps), int(bool(maximize)),
        int(bool(bias_correction)), _VARIANTS[variant], _ptr(d))
    if rc != 0:
        raise ValueError(f"oracle dense step rejected its arguments (code {rc})")
    return _diag(d)


def step_sparse(W, ids, rows, r, c, lr, t, beta2=0.999, eps=1e-8,
                maximize=False, bias_correction=True, variant="full"):
    """One sparse Ember step (Section 2.2): Algorithm 1 on the gradient whose
    row u is the sum, in occurrence order, of every row k with ids[k] == u."""
    V, D = _check_state(W, r, c)
    ids = np.ascontiguousarray(ids, dtype=np.int64)
    rows = np.ascontiguousarray(rows, dtype=np.float32)
    N = ids.shape[0]
    if rows.shape != (N, D):
        raise ValueError("rows must be N x D")
    d = np.zeros(5, np.float64)
    rc = _load().ember_oracle_step_sparse(
        V, D, int(W.dtype == np.uint16), _ptr(W), N, _ptr(ids), _ptr(rows),
        _ptr(r), _ptr(c), float(lr), int(t), float(beta2), float(eps),
        int(bool(maximize)), int(bool(bias_correction)), _VARIANTS[variant], _ptr(d))
    if rc != 0:
        raise ValueError(f"oracle sparse step rejected its arguments (code {rc})")
    return _diag(d)


def dedup(ids, V):
    """Distinct ids in [0, V), ascending, and the number of times each occurs."""
    ids = np.ascontiguousarray(ids, dtype=np.int64)
    N = ids.shape[0]
    uniq = np.zeros(max(N, 1), np.int64)
    counts = np.zeros(max(N, 1), np.int64)
    U = _load().ember_oracle_dedup(N, _ptr(ids), int(V), _ptr(uniq), _ptr(counts))
    if U < 0:
        raise ValueError("oracle dedup rejected its arguments")
    return uniq[:U].copy(), counts[:U].copy()


def round_bf16(x):
    """Round float64 values to bfloat16 (nearest, ties to even); uint16 bits."""
    x = np.ascontiguousarray(x, dtype=np.float64)
    out = np.zeros(x.shape, np.uint16)
    _load().ember_oracle_round_bf16(x.size, _ptr(x), _ptr(out))
    return out


def bf16_to_float64(bits):
    """Exact values of bfloat16 bit patterns."""
    bits = np.ascontiguousarray(bits, dtype=np.uint16)
    out = np.zeros(bits.shape, np.float64)
    _load().ember_oracle_bf16_to_double(bits.size, _ptr(bits), _ptr(out))
    return out


def lmhead_grad(dlogits, hidden, rows=None):
    """The LM-head gradient G = dlogits^T hidden (appendix "Decomposing the
    Squared Gradient": a sum over tokens of the outer product of the softmax
    error and the hidden state), in fp64, summed in token order.

    ``dlogits`` (T x V) and ``hidden`` (T x D) are bfloat16 bit patterns.
    ``rows``: the row indices v to compute (default: all).  Returns
    ``(G, absG)``, both len(rows) x D float64; ``absG`` is sum_t |delta h|."""
    dlogits = np.ascontiguousarray(dlogits, dtype=np.uint16)
    hidden = np.ascontiguousarray(hidden, dtype=np.uint16)
    if dlogits.ndim != 2 or hidden.ndim != 2 or dlogits.shape[0] != hidden.shape[0]:
        raise ValueError("dlogits must be T x V and hidden T x D")
    T, V = dlogits.shape
    D = hidden.shape[1]
    if rows is None:
        nrows, rp = V, None
    else:
        rows = np.ascontiguousarray(rows, dtype=np.int64)
        nrows, rp = rows.shape[0], _ptr(rows)
    G = np.zeros((nrows, D), np.float64)
    A = np.zeros((nrows, D), np.float64)
    rc = _load().ember_oracle_lmhead_grad(T, V, D, _ptr(dlogits), _ptr(hidden), nrows, rp,
                                           _ptr(G), _ptr(A))
    if rc != 0:
        raise ValueError(f"oracle LM-head gradient rejected its arguments (code {rc})")
    return G, A
