"""Plain fp64 CPU oracle of the MoE-ViE fine-grained MoE FFN layer (forward, bias
update and backward).

TEST INFRASTRUCTURE, NOT PRODUCT CODE.  Only the tests, ``__graft_entry__.smoke()``
and the CPU-baseline leg of ``bench.py`` may import this package.  It shares no
code with the CUDA library in ``paper_2608_17402_gb300``; the two meet only in the
seeded input generator (``workloads``), which holds none of the method's
arithmetic.

The arithmetic lives in ``moevie_oracle.c`` (plain C, fp64, pthreads over tokens);
this module builds it with gcc and marshals numpy arrays through ctypes.  What it
computes, with the paper's equations:

* :func:`logits`        Eq. (1), ``s = x . W_r`` (W_r stored ``[d, E]``)
* :func:`select`        Eq. (7) selection by ``top-k(sigmoid(s) + b)``, ties to the
  lower id, ids ascending; Eqs. (4)-(5) gates ``sigmoid(s)`` renormalised over the
  selected experts (the bias only selects)
* :func:`permute`       App. B, Algorithm 1 phase 1: BinCount, CumSum offsets and a
  stable sort of the flat slots by expert
* :func:`expert_rows`   ``E_e(x) = GELU(x W1[e]) W2[e]`` for expert-major rows
* :func:`combine`       Eq. (6) gate-weighted sum plus ``lambda`` times the shared
  expert
* :func:`forward_tokens` the whole layer, token by token (Eqs. 1, 7, 4-6)
* :func:`update_bias`   the loss-free bias update, z-score (Eq. 9) or sign (Eq. 8)
* :func:`backward`      the training path: gradients of ``sum dy . y`` with the
  selection held fixed (through the gates of Eqs. 4-5 into ``W_r`` and ``x``, and
  through the experts), the bias getting none
* :func:`backward_rows` its routed-expert part per expert-major row: the gradients
  at the hidden pre-activations and ``dy . E_e(x)``
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "moevie_oracle.c")
_LIB = os.path.join(_HERE, "liboracle.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile ``moevie_oracle.c`` into ``oracle/liboracle.so`` with gcc."""
    if not force and os.path.exists(_LIB) and os.path.getmtime(_LIB) >= os.path.getmtime(_SRC):
        return _LIB
    cmd = ["gcc", "-O2", "-std=c11", "-ffp-contract=off", "-fno-fast-math", "-fPIC",
           "-shared", "-pthread", _SRC, "-o", _LIB + ".tmp", "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(_LIB + ".tmp", _LIB)
    return _LIB


def default_threads() -> int:
    return max(1, os.cpu_count() or 1)


def _load():
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        build()
        lib = ctypes.CDLL(_LIB)
        P = ctypes.c_void_p
        I64 = ctypes.c_int64
        lib.oracle_logits.argtypes = [P, P, I64, I64, I64, P, ctypes.c_int]
        lib.oracle_select.argtypes = [P, P, I64, I64, I64, P, P, P, ctypes.c_int]
        lib.oracle_permute.argtypes = [P, I64, I64, I64, P, P, P, P]
        lib.oracle_expert_rows.argtypes = [P, P, P, P, P, I64, I64, I64, I64, I64, P, I64,
                                           ctypes.c_int, P, ctypes.c_int]
        lib.oracle_combine.argtypes = [P, P, P, P, ctypes.c_double, I64, I64, I64, P]
        lib.oracle_update_bias.argtypes = [P, I64, ctypes.c_float, ctypes.c_int, P]
        lib.oracle_forward_tokens.argtypes = [P, P, P, P, P, P, P, P, P, ctypes.c_double,
                                              I64, I64, I64, I64, I64, I64, P, I64,
                                              P, P, P, P, P, ctypes.c_int]
        lib.oracle_backward.argtypes = [P, P, P, P, P, P, P, P, P, ctypes.c_double,
                                        I64, I64, I64, I64, I64, I64, P, P, P, P, P, P, P, P, P]
        lib.oracle_backward_rows.argtypes = [P, P, P, P, P, P, P, P, I64, I64, I64, I64, I64, P, I64,
                                             P, P, P]
        for fn in (lib.oracle_logits, lib.oracle_select, lib.oracle_permute,
                   lib.oracle_expert_rows, lib.oracle_combine, lib.oracle_forward_tokens,
                   lib.oracle_update_bias, lib.oracle_backward, lib.oracle_backward_rows):
            fn.restype = ctypes.c_int
        _lib = lib
        return lib


def _ptr(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _c(a, dtype):
    """C-contiguous array of ``dtype``; bf16 data travels as uint16 bit patterns."""
    return np.ascontiguousarray(a, dtype=dtype)


def _check(rc, what):
    if rc != 0:
        raise RuntimeError(f"oracle {what} failed with code {rc}")


def logits(x_bf16, Wr, nthreads=None):
    """Eq. (1): ``s[t, e] = sum_i x[t, i] W_r[i, e]`` in fp64.  ``x_bf16`` uint16 [T, d]."""
    x = _c(x_bf16, np.uint16)
    Wr = _c(Wr, np.float32)
    T, d = x.shape
    E = Wr.shape[1]
    assert Wr.shape[0] == d
    s = np.empty((T, E), np.float64)
    _check(_load().oracle_logits(_ptr(x), _ptr(Wr), T, d, E, _ptr(s), nthreads or default_threads()),
           "logits")
    return s


def select(s, b, k, nthreads=None):
    """Eqs. (7), (4), (5): returns ``(idx int32 [T,k], gate fp64 [T,k], margin fp64 [T])``."""
    s = _c(s, np.float64)
    b = _c(b, np.float32)
    T, E = s.shape
    idx = np.empty((T, k), np.int32)
    gate = np.empty((T, k), np.float64)
    margin = np.empty((T,), np.float64)
    _check(_load().oracle_select(_ptr(s), _ptr(b), T, E, k, _ptr(idx), _ptr(gate), _ptr(margin),
                                 nthreads or default_threads()), "select")
    return idx, gate, margin


def route(x_bf16, Wr, b, k, nthreads=None):
    """Logits then selection: ``(idx, gate, margin)``."""
    return select(logits(x_bf16, Wr, nthreads), b, k, nthreads)


def permute(idx, E):
    """Algorithm 1 phase 1: ``(counts [E], offsets [E+1], perm [T*k], inv [T*k])`` int32."""
    idx = _c(idx, np.int32)
    T, k = idx.shape
    counts = np.empty((E,), np.int32)
    offsets = np.empty((E + 1,), np.int32)
    perm = np.empty((T * k,), np.int32)
    inv = np.empty((T * k,), np.int32)
    _check(_load().oracle_permute(_ptr(idx), T, k, E, _ptr(counts), _ptr(offsets), _ptr(perm),
                                  _ptr(inv)), "permute")
    return counts, offsets, perm, inv


def update_bias(counts, b, alpha, rule="zscore"):
    """Loss-free bias update (Sec. 2.2.2): z-score (Eq. 9) or sign (Eq. 8) rule; returns the new b (fp32)."""
    counts = _c(counts, np.int32)
    out = np.array(b, dtype=np.float32, copy=True)
    r = {"zscore": 0, "sign": 1}[rule]
    _check(_load().oracle_update_bias(_ptr(counts), counts.size, ctypes.c_float(alpha), r, _ptr(out)),
           "update_bias")
    return out


def expert_rows(x_bf16, perm, offsets, W1, W2, k, rows, hidden=False, nthreads=None):
    """Un-gated ``E_e(x_t)`` (or ``GELU(x_t W1[e])`` when ``hidden``) for expert-major ``rows``."""
    x = _c(x_bf16, np.uint16)
    perm = _c(perm, np.int32)
    offsets = _c(offsets, np.int32)
    W1 = _c(W1, np.uint16)
    W2 = None if W2 is None else _c(W2, np.uint16)
    rows = _c(rows, np.int32)
    T, d = x.shape
    E, d1, h = W1.shape
    assert d1 == d
    width = h if hidden else d
    out = np.empty((rows.size, width), np.float64)
    _check(_load().oracle_expert_rows(_ptr(x), _ptr(perm), _ptr(offsets), _ptr(W1), _ptr(W2),
                                      T, d, h, E, k, _ptr(rows), rows.size, 1 if hidden else 0,
                                      _ptr(out), nthreads or default_threads()), "expert_rows")
    return out


def combine(rows_out, inv, gate, shared=None, lam=1.0):
    """Eq. (6): ``y[t] = sum_j gate[t,j] rows_out[inv[t*k+j]] + lam * shared[t]`` (fp64)."""
    rows_out = _c(rows_out, np.float64)
    gate = _c(gate, np.float64)
    inv = _c(inv, np.int32)
    T, k = gate.shape
    d = rows_out.shape[1]
    sh = None if shared is None else _c(shared, np.float64)
    y = np.empty((T, d), np.float64)
    _check(_load().oracle_combine(_ptr(rows_out), _ptr(inv), _ptr(gate), _ptr(sh), float(lam),
                                  T, k, d, _ptr(y)), "combine")
    return y


def forward_tokens(x_bf16, Wr, b, W1, W2, k, Ws1=None, Ws2=None, lam=1.0, tokens=None,
                   nthreads=None, want_shared=False, W3=None, Ws3=None):
    """The whole layer for ``tokens`` (all tokens when None); SwiGLU experts
    ``(SiLU(x W1[e]) * (x W3[e])) W2[e]`` when ``W3`` is given, else GELU experts.

    Returns ``(y fp64 [n, d], idx int32 [n, k], gate fp64 [n, k], margin fp64 [n])`` and,
    with ``want_shared``, the un-weighted shared expert output as a fifth item.
    """
    x = _c(x_bf16, np.uint16)
    Wr = _c(Wr, np.float32)
    b = _c(b, np.float32)
    W1 = _c(W1, np.uint16)
    W2 = _c(W2, np.uint16)
    W3 = None if W3 is None else _c(W3, np.uint16)   # SwiGLU experts when given
    T, d = x.shape
    E, _, h = W1.shape
    assert W3 is None or W3.shape == W1.shape
    hs = 0
    if Ws1 is not None:
        Ws1 = _c(Ws1, np.uint16)
        Ws2 = _c(Ws2, np.uint16)
        hs = Ws1.shape[1]
        Ws3 = None if Ws3 is None else _c(Ws3, np.uint16)   # SwiGLU shared expert when given
        assert Ws3 is None or Ws3.shape == Ws1.shape
    toks = None if tokens is None else _c(tokens, np.int32)
    n = T if toks is None else toks.size
    y = np.empty((n, d), np.float64)
    idx = np.empty((n, k), np.int32)
    gate = np.empty((n, k), np.float64)
    margin = np.empty((n,), np.float64)
    shared = np.empty((n, d), np.float64) if (want_shared and hs > 0) else None
    _check(_load().oracle_forward_tokens(_ptr(x), _ptr(Wr), _ptr(b), _ptr(W1), _ptr(W2), _ptr(W3),
                                         _ptr(Ws1), _ptr(Ws2), _ptr(Ws3), float(lam), T, d, E, k, h, hs,
                                         _ptr(toks), n, _ptr(y), _ptr(idx), _ptr(gate),
                                         _ptr(margin), _ptr(shared),
                                         nthreads or default_threads()), "forward_tokens")
    if want_shared:
        return y, idx, gate, margin, shared
    return y, idx, gate, margin


def backward(x_bf16, Wr, b, W1, W2, k, dy, Ws1=None, Ws2=None, lam=1.0, W3=None, Ws3=None):
    """Gradients of ``L = sum_t dy[t] . y[t]`` (``dy`` fp64 [T, d]) for the layer of
    :func:`forward_tokens`, with the top-k selection held fixed and no gradient for
    the bias (it only selects).  Returns a dict of fp64 arrays: ``dx`` [T, d], ``dWr``
    [d, E], ``dW1`` [E, d, h], ``dW2`` [E, h, d], and ``dW3``, ``dWs1``, ``dWs2``,
    ``dWs3`` when those weights are given.  One thread, tokens in ascending order."""
    x = _c(x_bf16, np.uint16)
    Wr = _c(Wr, np.float32)
    b = _c(b, np.float32)
    W1 = _c(W1, np.uint16)
    W2 = _c(W2, np.uint16)
    W3 = None if W3 is None else _c(W3, np.uint16)
    dy = _c(dy, np.float64)
    T, d = x.shape
    E, _, h = W1.shape
    assert dy.shape == (T, d) and (W3 is None or W3.shape == W1.shape)
    hs = 0
    if Ws1 is not None:
        Ws1 = _c(Ws1, np.uint16)
        Ws2 = _c(Ws2, np.uint16)
        hs = Ws1.shape[1]
        Ws3 = None if Ws3 is None else _c(Ws3, np.uint16)
        assert Ws3 is None or Ws3.shape == Ws1.shape
    out = {"dx": np.empty((T, d)), "dWr": np.empty((d, E)), "dW1": np.empty((E, d, h)),
           "dW2": np.empty((E, h, d))}
    if W3 is not None:
        out["dW3"] = np.empty((E, d, h))
    if hs > 0:
        out["dWs1"] = np.empty((d, hs))
        out["dWs2"] = np.empty((hs, d))
        if Ws3 is not None:
            out["dWs3"] = np.empty((d, hs))
    _check(_load().oracle_backward(_ptr(x), _ptr(Wr), _ptr(b), _ptr(W1), _ptr(W2), _ptr(W3),
                                   _ptr(Ws1), _ptr(Ws2), _ptr(Ws3), float(lam), T, d, E, k, h, hs,
                                   _ptr(dy), _ptr(out["dx"]), _ptr(out["dWr"]), _ptr(out["dW1"]),
                                   _ptr(out["dW2"]), _ptr(out.get("dW3")), _ptr(out.get("dWs1")),
                                   _ptr(out.get("dWs2")), _ptr(out.get("dWs3"))), "backward")
    return out


def backward_rows(x_bf16, perm, offsets, gate_rows, W1, W2, k, dy, rows, W3=None):
    """Per expert-major row r = rows[i] (token perm[r] // k, gate gate_rows[r]): the
    gradients at the hidden pre-activations, ``du`` [n, h] (and ``dv`` [n, h] with SwiGLU
    experts), and ``dg`` [n] = dy[t] . E_e(x_t), the un-gated expert output.  Returns a
    dict of fp64 arrays."""
    x = _c(x_bf16, np.uint16)
    perm = _c(perm, np.int32)
    offsets = _c(offsets, np.int32)
    gate_rows = _c(gate_rows, np.float64)
    W1 = _c(W1, np.uint16)
    W2 = _c(W2, np.uint16)
    W3 = None if W3 is None else _c(W3, np.uint16)
    dy = _c(dy, np.float64)
    rows = _c(rows, np.int32)
    T, d = x.shape
    E, _, h = W1.shape
    n = rows.size
    out = {"du": np.empty((n, h)), "dg": np.empty((n,))}
    if W3 is not None:
        out["dv"] = np.empty((n, h))
    _check(_load().oracle_backward_rows(_ptr(x), _ptr(perm), _ptr(offsets), _ptr(gate_rows), _ptr(W1),
                                        _ptr(W2), _ptr(W3), _ptr(dy), T, d, h, E, k, _ptr(rows), n,
                                        _ptr(out["du"]), _ptr(out.get("dv")), _ptr(out["dg"])),
           "backward_rows")
    return out
