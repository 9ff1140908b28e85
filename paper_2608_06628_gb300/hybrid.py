"""Python binding of the block-hybrid attention C ABI (include/hybrid.h).

Argument marshalling only: every function here forwards to the entry point of
``libhybrid.so`` with the same name.  Tensors are passed as device pointers
(``tensor.data_ptr()``); torch is used for device memory and streams and
nothing else.  There is no fallback: if the library is missing or fails to
load, every call raises.
"""
from __future__ import annotations

import ctypes
import os

from . import build as _build

HYBRID_OK = 0
HYBRID_ERR_INVALID_ARG = 1
HYBRID_ERR_UNSUPPORTED = 2
HYBRID_ERR_CUDA = 3
HYBRID_ERR_TIMEOUT = 4
HYBRID_ERR_DEVICE = 5

HYBRID_F32 = 0
HYBRID_BF16 = 1

EXPORTED = (
    "hybrid_state_bytes", "hybrid_state_init", "hybrid_feature_map", "hybrid_block_attn",
    "hybrid_block_attn_commit", "hybrid_block_attn_commit_logical", "hybrid_commit_block", "hybrid_commit_ragged",
    "hybrid_state_unpack",
    "hybrid_state_pack", "hybrid_train_workspace_bytes", "hybrid_train_forward", "hybrid_train_backward",
    "hybrid_debug_arm_wait_timeout", "hybrid_check", "hybrid_status_str",
)


class hybrid_cfg(ctypes.Structure):
    _fields_ = [
        ("head_dim", ctypes.c_int),
        ("feat_dim", ctypes.c_int),
        ("n_q_heads", ctypes.c_int),
        ("n_kv_heads", ctypes.c_int),
        ("block_size", ctypes.c_int),
        ("io_dtype", ctypes.c_int),
    ]

    def __repr__(self):
        return (f"hybrid_cfg(d={self.head_dim}, F={self.feat_dim}, Hq={self.n_q_heads}, "
                f"Hkv={self.n_kv_heads}, B={self.block_size}, io_dtype={self.io_dtype})")


class HybridError(RuntimeError):
    def __init__(self, status: int, what: str):
        super().__init__(f"{what}: {hybrid_status_str(status)}")
        self.status = status


_lib = None


def lib(path: str | None = None):
    """Load libhybrid.so (once).  Raises if it is missing."""
    global _lib
    if _lib is not None and path is None:
        return _lib
    path = path or _build.LIB_PATH
    if not os.path.exists(path):
        raise ImportError(f"libhybrid.so not built ({path}); run __graft_entry__.build()")
    L = ctypes.CDLL(path)
    P = ctypes.c_void_p
    I = ctypes.c_int
    cfgp = ctypes.POINTER(hybrid_cfg)
    L.hybrid_state_bytes.argtypes = [cfgp]
    L.hybrid_state_bytes.restype = ctypes.c_size_t
    L.hybrid_state_init.argtypes = [cfgp, P, I, P]
    L.hybrid_feature_map.argtypes = [cfgp, P, I, I, P, P, P]
    L.hybrid_block_attn.argtypes = [cfgp, P, P, P, P, P, P, I, P, P]
    L.hybrid_block_attn_commit.argtypes = [cfgp, P, P, P, P, P, P, I, P, P]
    L.hybrid_block_attn_commit_logical.argtypes = [cfgp, P, P, P, P, P, P, P, I, P, P]
    L.hybrid_commit_block.argtypes = [cfgp, P, P, I, P, P, I, P]
    L.hybrid_commit_ragged.argtypes = [cfgp, P, P, ctypes.POINTER(ctypes.c_int), I, P, P, P]
    L.hybrid_state_unpack.argtypes = [cfgp, P, I, P, P, P]
    L.hybrid_state_pack.argtypes = [cfgp, P, P, P, I, P]
    S = ctypes.c_size_t
    L.hybrid_train_workspace_bytes.argtypes = [cfgp, I, I]
    L.hybrid_train_workspace_bytes.restype = S
    L.hybrid_train_forward.argtypes = [cfgp, P, P, P, P, P, I, I, P, P, S, P]
    L.hybrid_train_backward.argtypes = [cfgp, P, P, P, P, P, P, I, I, P, S, P, P, P]
    L.hybrid_debug_arm_wait_timeout.argtypes = [ctypes.c_ulonglong]
    L.hybrid_check.argtypes = [P]
    L.hybrid_status_str.argtypes = [I]
    L.hybrid_status_str.restype = ctypes.c_char_p
    for name in EXPORTED:
        if name not in ("hybrid_state_bytes", "hybrid_status_str", "hybrid_train_workspace_bytes"):
            getattr(L, name).restype = ctypes.c_int
    if path == _build.LIB_PATH:
        _lib = L
    return L


def make_cfg(head_dim, feat_dim, n_q_heads, n_kv_heads, block_size, io_dtype) -> hybrid_cfg:
    if not isinstance(io_dtype, int):
        import torch
        io_dtype = HYBRID_BF16 if io_dtype == torch.bfloat16 else HYBRID_F32
    return hybrid_cfg(head_dim, feat_dim, n_q_heads, n_kv_heads, block_size, io_dtype)


def _ptr(x):
    if x is None:
        return None
    if isinstance(x, int):
        return x
    return x.data_ptr()


def _stream(stream):
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def _ret(status, what, check):
    if check and status != HYBRID_OK:
        raise HybridError(status, what)
    return status


def hybrid_status_str(status: int) -> str:
    return lib().hybrid_status_str(int(status)).decode()


def hybrid_state_bytes(cfg: hybrid_cfg) -> int:
    return int(lib().hybrid_state_bytes(ctypes.byref(cfg)))


def hybrid_state_init(cfg, state_ptrs, n_req, stream=None, check=True):
    st = lib().hybrid_state_init(ctypes.byref(cfg), _ptr(state_ptrs), int(n_req), _stream(stream))
    return _ret(st, "hybrid_state_init", check)


def hybrid_feature_map(cfg, X, n_rows, n_heads_x, W, Phi, stream=None, check=True):
    st = lib().hybrid_feature_map(ctypes.byref(cfg), _ptr(X), int(n_rows), int(n_heads_x), _ptr(W),
                                  _ptr(Phi), _stream(stream))
    return _ret(st, "hybrid_feature_map", check)


def hybrid_block_attn(cfg, Q, K, V, W, alpha, state_ptrs, n_req, O, stream=None, check=True):
    st = lib().hybrid_block_attn(ctypes.byref(cfg), _ptr(Q), _ptr(K), _ptr(V), _ptr(W), _ptr(alpha),
                                 _ptr(state_ptrs), int(n_req), _ptr(O), _stream(stream))
    return _ret(st, "hybrid_block_attn", check)


def hybrid_block_attn_commit(cfg, Q, K, V, W, alpha, state_ptrs, n_req, O, stream=None, check=True):
    st = lib().hybrid_block_attn_commit(ctypes.byref(cfg), _ptr(Q), _ptr(K), _ptr(V), _ptr(W),
                                        _ptr(alpha), _ptr(state_ptrs), int(n_req), _ptr(O),
                                        _stream(stream))
    return _ret(st, "hybrid_block_attn_commit", check)


def hybrid_block_attn_commit_logical(cfg, Q, K, V, W, alpha, S_logical, z_logical, n_req, O, stream=None,
                                     check=True):
    st = lib().hybrid_block_attn_commit_logical(ctypes.byref(cfg), _ptr(Q), _ptr(K), _ptr(V), _ptr(W),
                                                _ptr(alpha), _ptr(S_logical), _ptr(z_logical), int(n_req),
                                                _ptr(O), _stream(stream))
    return _ret(st, "hybrid_block_attn_commit_logical", check)


def hybrid_commit_block(cfg, K, V, n_tok, W, state_ptrs, n_req, stream=None, check=True):
    st = lib().hybrid_commit_block(ctypes.byref(cfg), _ptr(K), _ptr(V), int(n_tok), _ptr(W),
                                   _ptr(state_ptrs), int(n_req), _stream(stream))
    return _ret(st, "hybrid_commit_block", check)


def hybrid_commit_ragged(cfg, K, V, tok_offsets, W, state_ptrs, n_req, stream=None, check=True):
    """Prompt prefill with per-request lengths: request r folds rows
    tok_offsets[r]:tok_offsets[r + 1] of the packed K, V [total, Hkv, d]."""
    offs = [int(x) for x in tok_offsets]
    if len(offs) != int(n_req) + 1:
        raise ValueError(f"tok_offsets needs n_req + 1 = {int(n_req) + 1} entries, got {len(offs)}")
    arr = (ctypes.c_int * len(offs))(*offs)
    st = lib().hybrid_commit_ragged(ctypes.byref(cfg), _ptr(K), _ptr(V), arr, int(n_req), _ptr(W),
                                    _ptr(state_ptrs), _stream(stream))
    return _ret(st, "hybrid_commit_ragged", check)


def hybrid_state_unpack(cfg, state_ptrs, n_req, S_logical, z_logical, stream=None, check=True):
    st = lib().hybrid_state_unpack(ctypes.byref(cfg), _ptr(state_ptrs), int(n_req), _ptr(S_logical),
                                   _ptr(z_logical), _stream(stream))
    return _ret(st, "hybrid_state_unpack", check)


def hybrid_state_pack(cfg, S_logical, z_logical, state_ptrs, n_req, stream=None, check=True):
    st = lib().hybrid_state_pack(ctypes.byref(cfg), _ptr(S_logical), _ptr(z_logical), _ptr(state_ptrs),
                                 int(n_req), _stream(stream))
    return _ret(st, "hybrid_state_pack", check)


def hybrid_train_workspace_bytes(cfg, n_seq, seq_len) -> int:
    return int(lib().hybrid_train_workspace_bytes(ctypes.byref(cfg), int(n_seq), int(seq_len)))


def hybrid_train_forward(cfg, Q, K, V, W, alpha, n_seq, seq_len, O, workspace, workspace_bytes, stream=None,
                         check=True):
    st = lib().hybrid_train_forward(ctypes.byref(cfg), _ptr(Q), _ptr(K), _ptr(V), _ptr(W), _ptr(alpha),
                                    int(n_seq), int(seq_len), _ptr(O), _ptr(workspace), int(workspace_bytes),
                                    _stream(stream))
    return _ret(st, "hybrid_train_forward", check)


def hybrid_train_backward(cfg, Q, K, V, W, alpha, dO, n_seq, seq_len, workspace, workspace_bytes, dW, dalpha,
                          stream=None, check=True):
    st = lib().hybrid_train_backward(ctypes.byref(cfg), _ptr(Q), _ptr(K), _ptr(V), _ptr(W), _ptr(alpha),
                                     _ptr(dO), int(n_seq), int(seq_len), _ptr(workspace),
                                     int(workspace_bytes), _ptr(dW), _ptr(dalpha), _stream(stream))
    return _ret(st, "hybrid_train_backward", check)


def hybrid_debug_arm_wait_timeout(wait_ns, check=True):
    """Test hook: the next persistent step launch gives up its waits after
    wait_ns nanoseconds and withholds one barrier arrival (see hybrid.h)."""
    st = lib().hybrid_debug_arm_wait_timeout(int(wait_ns))
    return _ret(st, "hybrid_debug_arm_wait_timeout", check)


def hybrid_check(stream=None, check=True):
    st = lib().hybrid_check(_stream(stream))
    return _ret(st, "hybrid_check", check)
