"""fp64 CPU oracle for the causal Self-Exchange Relation operator (ctypes binding).

TEST INFRASTRUCTURE ONLY.  Only the test suite, ``__graft_entry__.smoke()`` and the
benchmark's CPU-baseline leg may import this package.  The CUDA library never uses
it, and it uses nothing from the CUDA library: the two share no code.

The arithmetic lives in ``relation_oracle.c`` (plain C, fp64), which follows the
paper's definitions: Eq. (causal-relation) and Eq. (relation-flow) for the
materialised forward, App. A.1.2-A.1.8 for the factorised form, App. A.3 for the
tiled Exchange scan and App. A.1.7 for the two backward derivations.
``linear_oracle.c`` (plain C, fp64) holds Linear Relation (Sec. 5.2, App. A.4): the
recurrent step, its unrolled form and the reverse-mode backward of the recurrence.
``linear_chunked.py`` (plain numpy, fp64) evaluates the same Linear Relation forward and
backward block by block (the form a block-parallel kernel computes), pinned to the
recurrence.
``layer.py`` (plain numpy, fp64) holds the layer's transforms around the operator: RoPE
on P1, P2 and the Givens mixing of the information states, with their gradients.
This module only marshals numpy arrays.

``Oracle(path)`` binds one compiled copy of the C file; the module-level functions
use the default copy built from ``relation_oracle.c`` by :func:`build`.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
SOURCE = os.path.join(_HERE, "relation_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD, "liboracle.so")
LINEAR_SOURCE = os.path.join(_HERE, "linear_oracle.c")
_LINEAR_LIB_PATH = os.path.join(_BUILD, "liblinear_oracle.so")
_linear = None
_lock = threading.Lock()
_default = None

TAU_S = 2.0  # Self temperature fixed by the paper (Sec. 3.1)

_dp = ctypes.POINTER(ctypes.c_double)


def compile_source(src: str, out: str) -> str:
    """Compile one C source file of the oracle into a shared library at ``out``."""
    os.makedirs(os.path.dirname(out), exist_ok=True)
    tmp = out + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fopenmp", src, "-o", tmp, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, out)
    return out


def build(force: bool = False) -> str:
    """Compile relation_oracle.c into oracle/_build/liboracle.so and linear_oracle.c into
    oracle/_build/liblinear_oracle.so (gcc, -fopenmp); returns the first."""
    for src, out in ((SOURCE, _LIB_PATH), (LINEAR_SOURCE, _LINEAR_LIB_PATH)):
        if (force or not os.path.exists(out)
                or os.path.getmtime(out) < os.path.getmtime(src)):
            compile_source(src, out)
    return _LIB_PATH


def _in(a) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(a, dtype=np.float64))


def _p(a):
    return None if a is None else a.ctypes.data_as(_dp)


def _check(rc: int, name: str):
    if rc != 0:
        raise ValueError(f"oracle {name} rejected its arguments (rc={rc})")


def _head_args(q, k, v):
    q, k, v = _in(q), _in(k), _in(v)
    if q.ndim != 2 or q.shape != k.shape or q.shape != v.shape:
        raise ValueError("one head: q, k, v must all be [T, d]")
    return q, k, v, q.shape[0], q.shape[1]


def _mhr_args(q, k, v):
    q, k, v = _in(q), _in(k), _in(v)
    if q.ndim != 4 or q.shape != k.shape or q.shape != v.shape:
        raise ValueError("multi-head: q, k, v must all be [B, T, H, d]")
    B, T, H, d = q.shape
    return q, k, v, B, T, H, d


class Oracle:
    """One loaded copy of the compiled oracle."""

    def __init__(self, path: str):
        lib = ctypes.CDLL(path)
        i, ll, d = ctypes.c_int, ctypes.c_longlong, ctypes.c_double
        sig = {
            "rel_oracle_fwd": [i, i, _dp, _dp, _dp, d, d, _dp, _dp, _dp, _dp],
            "rel_oracle_fwd_rows": [i, i, _dp, _dp, _dp, d, d, i, ctypes.POINTER(ctypes.c_int),
                                    _dp, _dp],
            "rel_oracle_fwd_factorized": [i, i, _dp, _dp, _dp, d, d, _dp, _dp, _dp, _dp, _dp, _dp,
                                          _dp, _dp, _dp],
            "rel_oracle_fwd_scan": [i, i, _dp, _dp, _dp, d, d, i, i, _dp, _dp],
            "rel_oracle_bwd": [i, i, _dp, _dp, _dp, _dp, d, d, _dp, _dp, _dp, _dp],
            "rel_oracle_bwd_tail": [i, i, _dp, _dp, _dp, _dp, d, d, i, _dp, _dp, _dp, _dp],
            "rel_oracle_bwd_credit": [i, i, _dp, _dp, _dp, _dp, d, d, _dp, _dp, _dp, _dp],
            "rel_oracle_mhr_fwd": [i, i, i, i, ll, ll, ll, _dp, _dp, _dp, d, d, _dp, _dp, i],
            "rel_oracle_mhr_bwd": [i, i, i, i, ll, ll, ll, _dp, _dp, _dp, _dp, d, d, _dp, _dp,
                                   _dp, _dp, i],
            "rel_oracle_max_threads": [],
        }
        for name, args in sig.items():
            fn = getattr(lib, name)
            fn.argtypes = args
            fn.restype = ctypes.c_int
        self.lib = lib
        self.path = path

    def fwd(self, q, k, v, lam: float, tau_s: float = TAU_S, want_matrices: bool = False):
        """Materialised forward of one head.  Returns (Y [T,d], logZ [T]) or, with
        ``want_matrices``, (Y, logZ, R [T,T], F [T,T])."""
        q, k, v, T, d = _head_args(q, k, v)
        y = np.empty((T, d)); lz = np.empty(T)
        R = np.empty((T, T)) if want_matrices else None
        F = np.empty((T, T)) if want_matrices else None
        _check(self.lib.rel_oracle_fwd(T, d, _p(q), _p(k), _p(v), lam, tau_s, _p(y), _p(lz),
                                       _p(R), _p(F)), "fwd")
        return (y, lz, R, F) if want_matrices else (y, lz)

    def fwd_rows(self, q, k, v, rows, lam: float, tau_s: float = TAU_S):
        """Materialised forward of one head restricted to the given (zero-based) rows."""
        q, k, v, T, d = _head_args(q, k, v)
        rows = np.ascontiguousarray(np.asarray(rows, dtype=np.int32))
        y = np.empty((len(rows), d)); lz = np.empty(len(rows))
        _check(self.lib.rel_oracle_fwd_rows(T, d, _p(q), _p(k), _p(v), lam, tau_s, len(rows),
                                            rows.ctypes.data_as(ctypes.POINTER(ctypes.c_int)),
                                            _p(y), _p(lz)), "fwd_rows")
        return y, lz

    def fwd_factorized(self, q, k, v, lam: float, tau_s: float = TAU_S):
        """Factorised Self-Exchange forward of one head.  Returns a dict with
        Y, logZ, S, LE, A, g, Fii, Ibar and pi ([T,T], zero for j >= i)."""
        q, k, v, T, d = _head_args(q, k, v)
        out = {"Y": np.empty((T, d)), "logZ": np.empty(T), "S": np.empty(T), "LE": np.empty(T),
               "A": np.empty(T), "g": np.empty(T), "Fii": np.empty(T),
               "Ibar": np.empty((T, d)), "pi": np.empty((T, T))}
        _check(self.lib.rel_oracle_fwd_factorized(
            T, d, _p(q), _p(k), _p(v), lam, tau_s, _p(out["Y"]), _p(out["logZ"]),
            _p(out["S"]), _p(out["LE"]), _p(out["A"]), _p(out["g"]), _p(out["Fii"]),
            _p(out["Ibar"]), _p(out["pi"])), "fwd_factorized")
        return out

    def fwd_scan(self, q, k, v, lam: float, tile: int, reverse: bool = False,
                 tau_s: float = TAU_S):
        """FlashRelation tiled Exchange scan of one head in fp64.  Returns (Y, logZ)."""
        q, k, v, T, d = _head_args(q, k, v)
        y = np.empty((T, d)); lz = np.empty(T)
        _check(self.lib.rel_oracle_fwd_scan(T, d, _p(q), _p(k), _p(v), lam, tau_s, int(tile),
                                            int(bool(reverse)), _p(y), _p(lz)), "fwd_scan")
        return y, lz

    def bwd(self, q, k, v, dy, lam: float, tau_s: float = TAU_S):
        """Backward of one head via the generic softmax gradient.
        Returns (dq, dk, dv, dlambda)."""
        q, k, v, T, d = _head_args(q, k, v)
        dy = _in(dy)
        dq = np.empty((T, d)); dk = np.empty((T, d)); dv = np.empty((T, d))
        dl = np.empty(1)
        _check(self.lib.rel_oracle_bwd(T, d, _p(q), _p(k), _p(v), _p(dy), lam, tau_s, _p(dq),
                                       _p(dk), _p(dv), _p(dl)), "bwd")
        return dq, dk, dv, float(dl[0])

    def bwd_tail(self, q, k, v, dy, lam: float, row_begin: int, tau_s: float = TAU_S):
        """Backward of one head restricted to rows r >= row_begin: exact dq rows
        >= row_begin and dk, dv rows >= row_begin (dq rows below are 0; dlambda sums
        the processed rows).  Returns (dq, dk, dv, dlambda)."""
        q, k, v, T, d = _head_args(q, k, v)
        dy = _in(dy)
        dq = np.empty((T, d)); dk = np.empty((T, d)); dv = np.empty((T, d))
        dl = np.empty(1)
        _check(self.lib.rel_oracle_bwd_tail(T, d, _p(q), _p(k), _p(v), _p(dy), lam, tau_s,
                                            int(row_begin), _p(dq), _p(dk), _p(dv), _p(dl)),
               "bwd_tail")
        return dq, dk, dv, float(dl[0])

    def bwd_credit(self, q, k, v, dy, lam: float, tau_s: float = TAU_S):
        """Backward of one head via the Self-Exchange credit decomposition.
        Returns (dq, dk, dv, dlambda)."""
        q, k, v, T, d = _head_args(q, k, v)
        dy = _in(dy)
        dq = np.empty((T, d)); dk = np.empty((T, d)); dv = np.empty((T, d))
        dl = np.empty(1)
        _check(self.lib.rel_oracle_bwd_credit(T, d, _p(q), _p(k), _p(v), _p(dy), lam, tau_s,
                                              _p(dq), _p(dk), _p(dv), _p(dl)), "bwd_credit")
        return dq, dk, dv, float(dl[0])

    def mhr_fwd(self, q, k, v, lam: float, tau_s: float = TAU_S, nthreads: int = 0):
        """Multi-head forward on [B,T,H,d] arrays.  Returns (Y [B,T,H,d], logZ [B,H,T])."""
        q, k, v, B, T, H, d = _mhr_args(q, k, v)
        y = np.empty_like(q); lz = np.empty((B, H, T))
        _check(self.lib.rel_oracle_mhr_fwd(B, T, H, d, T * H * d, H * d, d, _p(q), _p(k), _p(v),
                                           lam, tau_s, _p(y), _p(lz), int(nthreads)), "mhr_fwd")
        return y, lz

    def mhr_bwd(self, q, k, v, dy, lam: float, tau_s: float = TAU_S, nthreads: int = 0):
        """Multi-head backward on [B,T,H,d] arrays.  Returns (dq, dk, dv, dlambda)."""
        q, k, v, B, T, H, d = _mhr_args(q, k, v)
        dy = _in(dy)
        dq = np.empty_like(q); dk = np.empty_like(q); dv = np.empty_like(q)
        dl = np.empty(1)
        _check(self.lib.rel_oracle_mhr_bwd(B, T, H, d, T * H * d, H * d, d, _p(q), _p(k), _p(v),
                                           _p(dy), lam, tau_s, _p(dq), _p(dk), _p(dv), _p(dl),
                                           int(nthreads)), "mhr_bwd")
        return dq, dk, dv, float(dl[0])

    def max_threads(self) -> int:
        """OpenMP threads the oracle's parallel loops use by default."""
        return int(self.lib.rel_oracle_max_threads())


def default() -> Oracle:
    """The oracle compiled from relation_oracle.c (built on first use)."""
    global _default
    with _lock:
        if _default is None:
            _default = Oracle(build())
        return _default


def fwd(*a, **kw):
    return default().fwd(*a, **kw)


def fwd_rows(*a, **kw):
    return default().fwd_rows(*a, **kw)


def fwd_factorized(*a, **kw):
    return default().fwd_factorized(*a, **kw)


def fwd_scan(*a, **kw):
    return default().fwd_scan(*a, **kw)


def bwd(*a, **kw):
    return default().bwd(*a, **kw)


def bwd_tail(*a, **kw):
    return default().bwd_tail(*a, **kw)


def bwd_credit(*a, **kw):
    return default().bwd_credit(*a, **kw)


def mhr_fwd(*a, **kw):
    return default().mhr_fwd(*a, **kw)


def mhr_bwd(*a, **kw):
    return default().mhr_bwd(*a, **kw)


def max_threads() -> int:
    return default().max_threads()


# --- Linear Relation (linear_oracle.c) ---------------------------------------------

class LinearOracle:
    """One loaded copy of the compiled Linear Relation oracle (one head per call,
    [T, d] arrays: p1, p2 after RoPE, information v, retention alpha in (0, 1])."""

    def __init__(self, path: str):
        lib = ctypes.CDLL(path)
        i, d = ctypes.c_int, ctypes.c_double
        sig = {
            "rel_linear_fwd": [i, i, _dp, _dp, _dp, _dp, d, _dp, _dp, _dp],
            "rel_linear_fwd_unrolled": [i, i, _dp, _dp, _dp, _dp, d, _dp],
            "rel_linear_bwd": [i, i, _dp, _dp, _dp, _dp, _dp, d, _dp, _dp, _dp, _dp],
        }
        for name, args in sig.items():
            fn = getattr(lib, name)
            fn.argtypes = args
            fn.restype = ctypes.c_int
        self.lib = lib

    @staticmethod
    def _args(p1, p2, v, alpha):
        p1, p2, v, alpha = _in(p1), _in(p2), _in(v), _in(alpha)
        if p1.ndim != 2 or not (p1.shape == p2.shape == v.shape == alpha.shape):
            raise ValueError("one head: p1, p2, v, alpha must all be [T, d]")
        return p1, p2, v, alpha, p1.shape[0], p1.shape[1]

    def fwd(self, p1, p2, v, alpha, tau_s: float = TAU_S, want_states: bool = False):
        """Recurrent forward (App. A.4.2).  Returns (Y [T, d], S [T]) or, with
        ``want_states``, (Y, S, C [T + 1, d, d]) with C[0] = 0."""
        p1, p2, v, alpha, T, d = self._args(p1, p2, v, alpha)
        y = np.empty((T, d)); S = np.empty(T)
        C = np.empty((T + 1, d, d)) if want_states else None
        _check(self.lib.rel_linear_fwd(T, d, _p(p1), _p(p2), _p(v), _p(alpha), tau_s, _p(y),
                                       _p(S), _p(C)), "linear_fwd")
        return (y, S, C) if want_states else (y, S)

    def fwd_unrolled(self, p1, p2, v, alpha, tau_s: float = TAU_S):
        """Unrolled forward (App. A.4.4-A.4.5), for tiny T.  Returns Y [T, d]."""
        p1, p2, v, alpha, T, d = self._args(p1, p2, v, alpha)
        y = np.empty((T, d))
        _check(self.lib.rel_linear_fwd_unrolled(T, d, _p(p1), _p(p2), _p(v), _p(alpha), tau_s,
                                                _p(y)), "linear_fwd_unrolled")
        return y

    def bwd(self, p1, p2, v, alpha, dy, tau_s: float = TAU_S):
        """Reverse-mode backward of the recurrence.  Returns (dp1, dp2, dv, dalpha)."""
        p1, p2, v, alpha, T, d = self._args(p1, p2, v, alpha)
        dy = _in(dy)
        if dy.shape != (T, d):
            raise ValueError("dy must be [T, d]")
        out = [np.empty((T, d)) for _ in range(4)]
        _check(self.lib.rel_linear_bwd(T, d, _p(p1), _p(p2), _p(v), _p(alpha), _p(dy), tau_s,
                                       *(_p(o) for o in out)), "linear_bwd")
        return tuple(out)


def linear() -> LinearOracle:
    """The Linear Relation oracle compiled from linear_oracle.c (built on first use)."""
    global _linear
    with _lock:
        if _linear is None:
            build()
            _linear = LinearOracle(_LINEAR_LIB_PATH)
        return _linear


def linear_fwd(*a, **kw):
    return linear().fwd(*a, **kw)


def linear_fwd_unrolled(*a, **kw):
    return linear().fwd_unrolled(*a, **kw)


def linear_bwd(*a, **kw):
    return linear().bwd(*a, **kw)
