"""fp64 CPU oracle for block-hybrid attention -- TEST INFRASTRUCTURE ONLY.

Only the test suite, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import this package.  The CUDA library never imports, links
or calls it, and it shares no code with the CUDA library.

The arithmetic lives in ``hybrid_oracle.c`` (plain C, double precision, one
loop per definition of Section 3.1 / Eq. 1 of "Retrofitting Linear Attention
into Diffusion Language Models").  This module only compiles it with gcc and
marshals numpy float64 arrays in and out.

Logical layouts (row-major):
    Q, O   [n_req, B, Hq, d]       K, V  [n_req, T, Hkv, d]
    training form: Q, O, dO [n_seq, L, Hq, d], K, V [n_seq, L, Hkv, d]
    W      [Hkv, d, F]             alpha [Hq]
    S      [n_req, Hkv, 2F, d]     z     [n_req, Hkv, 2F]
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
SOURCE = os.path.join(_HERE, "hybrid_oracle.c")
BUILD_DIR = os.path.join(_HERE, "_build")
LIB_PATH = os.path.join(BUILD_DIR, "liboracle.so")

PHI_HEDGEHOG = 0
PHI_IDENTITY = 1

# -ffp-contract=off keeps a*b+c as two roundings on every host, so x86 and
# aarch64 builds of the oracle produce the same bits.
CFLAGS = ["-O2", "-std=c11", "-fPIC", "-shared", "-pthread", "-ffp-contract=off"]


class OracleError(RuntimeError):
    pass


def build_oracle(source: str = SOURCE, out: str = LIB_PATH, extra_flags=()) -> str:
    """Compile the oracle C source into a shared library and return its path."""
    os.makedirs(os.path.dirname(out), exist_ok=True)
    tmp = f"{out}.{os.getpid()}.{threading.get_ident()}.tmp"
    cmd = ["gcc", *CFLAGS, *extra_flags, source, "-o", tmp, "-lm"]
    subprocess.run(cmd, check=True, capture_output=True)
    os.replace(tmp, out)
    return out


def _dptr(a: np.ndarray):
    return a.ctypes.data_as(ctypes.POINTER(ctypes.c_double))


def _f64(a, name):
    if a is None:
        return None
    a = np.ascontiguousarray(np.asarray(a, dtype=np.float64))
    return a


def default_threads() -> int:
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:  # pragma: no cover
        return os.cpu_count() or 1


class Oracle:
    """A loaded oracle library.  ``Oracle()`` loads (building if needed) the
    default build; ``Oracle(path)`` loads another build of the same source."""

    def __init__(self, path: str | None = None):
        if path is None:
            if not os.path.exists(LIB_PATH) or os.path.getmtime(LIB_PATH) < os.path.getmtime(SOURCE):
                build_oracle()
            path = LIB_PATH
        self.path = path
        lib = ctypes.CDLL(path)
        D = ctypes.POINTER(ctypes.c_double)
        I = ctypes.c_int
        lib.oracle_feature_map.argtypes = [ctypes.c_long, I, I, I, I, D, D, D]
        lib.oracle_commit.argtypes = [I, I, I, I, I, I, D, D, D, D, D, I]
        lib.oracle_block_attn.argtypes = [I, I, I, I, I, I, I, D, D, D, D, D, D, D, D, I]
        lib.oracle_block_attn_prefix.argtypes = [I, I, I, I, I, I, I, D, D, D, D, D, D, D,
                                                 ctypes.POINTER(ctypes.c_int), I, D, I]
        lib.oracle_train_forward.argtypes = [I, I, I, I, I, I, I, D, D, D, D, D, D, I]
        lib.oracle_train_backward.argtypes = [I, I, I, I, I, I, I, D, D, D, D, D, D, D, D, I]
        for fn in (lib.oracle_feature_map, lib.oracle_commit, lib.oracle_block_attn,
                   lib.oracle_block_attn_prefix, lib.oracle_train_forward,
                   lib.oracle_train_backward):
            fn.restype = ctypes.c_int
        self.lib = lib

    @staticmethod
    def _check(rc, what):
        if rc == -2:
            raise OracleError(f"{what}: an exponent argument left [-700, 700]")
        if rc != 0:
            raise OracleError(f"{what}: bad arguments (rc={rc})")

    # -- phi ---------------------------------------------------------------
    def feature_map(self, X, W):
        """X [n_rows, n_heads_x, d], W [Hkv, d, F] -> Phi [n_rows, n_heads_x, 2F]."""
        X = _f64(X, "X")
        W = _f64(W, "W")
        n_rows, n_heads_x, d = X.shape
        Hkv, d2, F = W.shape
        assert d2 == d
        out = np.zeros((n_rows, n_heads_x, 2 * F), dtype=np.float64)
        rc = self.lib.oracle_feature_map(n_rows, n_heads_x, Hkv, d, F, _dptr(X), _dptr(W), _dptr(out))
        self._check(rc, "feature_map")
        return out

    # -- commit ------------------------------------------------------------
    def commit(self, K, V, W, S, z, phi_kind=PHI_HEDGEHOG, n_threads=None, F=None):
        """Fold the T tokens of K, V [n_req, T, Hkv, d] into S, z (in place)."""
        K = _f64(K, "K")
        V = _f64(V, "V")
        n_req, T, Hkv, d = K.shape
        assert V.shape == K.shape
        if phi_kind == PHI_HEDGEHOG:
            W = _f64(W, "W")
            F = W.shape[2]
            P2 = 2 * F
            wp = _dptr(W)
        else:
            F = d if F is None else F
            P2 = d
            wp = None
        assert S.dtype == np.float64 and S.flags.c_contiguous and S.shape == (n_req, Hkv, P2, d)
        assert z.dtype == np.float64 and z.flags.c_contiguous and z.shape == (n_req, Hkv, P2)
        rc = self.lib.oracle_commit(n_req, T, Hkv, d, F, phi_kind, _dptr(K), _dptr(V), wp,
                                    _dptr(S), _dptr(z), n_threads or default_threads())
        self._check(rc, "commit")

    def empty_state(self, n_req, Hkv, d, F=None, phi_kind=PHI_HEDGEHOG):
        P2 = 2 * F if phi_kind == PHI_HEDGEHOG else d
        return (np.zeros((n_req, Hkv, P2, d), dtype=np.float64),
                np.zeros((n_req, Hkv, P2), dtype=np.float64))

    # -- one active block ----------------------------------------------------
    def block_attn(self, Q, K, V, W, alpha, S, z, phi_kind=PHI_HEDGEHOG, n_threads=None):
        """Route 1: the cross-block branch read from the state (S, z)."""
        Q, K, V, alpha, S, z = (_f64(a, "") for a in (Q, K, V, alpha, S, z))
        n_req, B, Hq, d = Q.shape
        Hkv = K.shape[2]
        if phi_kind == PHI_HEDGEHOG:
            W = _f64(W, "W")
            F = W.shape[2]
            wp = _dptr(W)
        else:
            F, wp = d, None
        O = np.zeros_like(Q)
        rc = self.lib.oracle_block_attn(n_req, B, Hq, Hkv, d, F, phi_kind, _dptr(Q), _dptr(K),
                                        _dptr(V), wp, _dptr(alpha), _dptr(S), _dptr(z), _dptr(O),
                                        n_threads or default_threads())
        self._check(rc, "block_attn")
        return O

    def block_attn_prefix(self, Q, K, V, W, alpha, Kp, Vp, prefix_len, phi_kind=PHI_HEDGEHOG,
                          n_threads=None):
        """Route 2: the cross-block branch summed token by token over the explicit
        prefix Kp, Vp [n_req, P_max, Hkv, d] (first prefix_len[r] tokens used)."""
        Q, K, V, alpha, Kp, Vp = (_f64(a, "") for a in (Q, K, V, alpha, Kp, Vp))
        n_req, B, Hq, d = Q.shape
        Hkv = K.shape[2]
        P_max = Kp.shape[1]
        plen = np.ascontiguousarray(np.asarray(prefix_len, dtype=np.int32))
        if phi_kind == PHI_HEDGEHOG:
            W = _f64(W, "W")
            F = W.shape[2]
            wp = _dptr(W)
        else:
            F, wp = d, None
        O = np.zeros_like(Q)
        rc = self.lib.oracle_block_attn_prefix(
            n_req, B, Hq, Hkv, d, F, phi_kind, _dptr(Q), _dptr(K), _dptr(V), wp, _dptr(alpha),
            _dptr(Kp), _dptr(Vp), plen.ctypes.data_as(ctypes.POINTER(ctypes.c_int)), P_max,
            _dptr(O), n_threads or default_threads())
        self._check(rc, "block_attn_prefix")
        return O

    # -- training form (Stage 1 attention transfer) ---------------------------
    def train_forward(self, Q, K, V, W, alpha, B, n_threads=None):
        """Every block of each sequence against the state of the blocks before
        it.  Q [n_seq, L, Hq, d], K, V [n_seq, L, Hkv, d] -> O [n_seq, L, Hq, d]."""
        Q, K, V, W, alpha = (_f64(a, "") for a in (Q, K, V, W, alpha))
        n_seq, L, Hq, d = Q.shape
        Hkv, F = K.shape[2], W.shape[2]
        O = np.zeros_like(Q)
        rc = self.lib.oracle_train_forward(n_seq, L, B, Hq, Hkv, d, F, _dptr(Q), _dptr(K),
                                           _dptr(V), _dptr(W), _dptr(alpha), _dptr(O),
                                           n_threads or default_threads())
        self._check(rc, "train_forward")
        return O

    def train_backward(self, Q, K, V, W, alpha, dO, B, n_threads=None):
        """Gradient of sum(dO * O) with respect to W [Hkv, d, F] and alpha [Hq]."""
        Q, K, V, W, alpha, dO = (_f64(a, "") for a in (Q, K, V, W, alpha, dO))
        n_seq, L, Hq, d = Q.shape
        Hkv, F = K.shape[2], W.shape[2]
        dW = np.zeros_like(W)
        dalpha = np.zeros_like(alpha)
        rc = self.lib.oracle_train_backward(n_seq, L, B, Hq, Hkv, d, F, _dptr(Q), _dptr(K),
                                            _dptr(V), _dptr(W), _dptr(alpha), _dptr(dO),
                                            _dptr(dW), _dptr(dalpha),
                                            n_threads or default_threads())
        self._check(rc, "train_backward")
        return dW, dalpha


_default = None
_lock = threading.Lock()


def load() -> Oracle:
    global _default
    with _lock:
        if _default is None:
            _default = Oracle()
        return _default
