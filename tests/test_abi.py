"""The C-ABI library on the host, without a GPU: it loads, exports every entry
point include/hybrid.h declares, sizes states correctly and rejects bad
arguments before touching the device."""
import ctypes
import os
import re

import pytest

from paper_2608_06628_gb300 import build as B
from paper_2608_06628_gb300 import hybrid as H

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def L():
    B.build()
    return H.lib()


def declared_functions():
    names = []
    for hdr in sorted(os.listdir(os.path.join(ROOT, "include"))):
        if hdr.endswith(".h"):
            text = open(os.path.join(ROOT, "include", hdr)).read()
            text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
            names += re.findall(r"\b(hybrid_[a-z_]+)\s*\(", text)
    return sorted(set(names))


def test_header_declares_the_boundary():
    names = declared_functions()
    for must in ("hybrid_state_init", "hybrid_feature_map", "hybrid_block_attn",
                 "hybrid_commit_block", "hybrid_check", "hybrid_status_str", "hybrid_state_bytes"):
        assert must in names


def test_every_declared_symbol_is_exported(L):
    for name in declared_functions():
        assert hasattr(L, name), f"{name} declared in include/ but not exported"
    assert set(H.EXPORTED) <= set(declared_functions())


def cfg(d=128, F=128, Hq=16, Hkv=4, Bs=32, dt=H.HYBRID_BF16):
    return H.hybrid_cfg(d, F, Hq, Hkv, Bs, dt)


def test_state_bytes(L):
    # Hkv * (2F*d + 2F) * 4
    assert H.hybrid_state_bytes(cfg()) == 4 * (2 * 128 * 128 + 2 * 128) * 4
    assert H.hybrid_state_bytes(cfg(d=64, F=64, Hkv=2)) == 2 * (2 * 64 * 64 + 2 * 64) * 4
    assert H.hybrid_state_bytes(cfg(F=256, Hq=16, Hkv=16)) == 16 * (2 * 256 * 128 + 2 * 256) * 4
    # unsupported sizes give 0
    assert H.hybrid_state_bytes(cfg(d=96)) == 0
    assert H.hybrid_state_bytes(cfg(F=100)) == 0
    assert H.hybrid_state_bytes(cfg(Bs=0)) == 0
    assert H.hybrid_state_bytes(cfg(Hq=6, Hkv=4)) == 0


@pytest.mark.parametrize("bad,code", [
    (dict(d=96), H.HYBRID_ERR_UNSUPPORTED),
    (dict(F=48), H.HYBRID_ERR_UNSUPPORTED),
    (dict(Bs=129), H.HYBRID_ERR_UNSUPPORTED),
    (dict(dt=7), H.HYBRID_ERR_UNSUPPORTED),
    (dict(Hq=6, Hkv=4), H.HYBRID_ERR_INVALID_ARG),
    (dict(Hq=4, Hkv=8), H.HYBRID_ERR_INVALID_ARG),
])
def test_bad_cfg_rejected_on_host(L, bad, code):
    c = cfg(**bad)
    fake = 1 << 20   # never dereferenced: validation fails first
    assert L.hybrid_block_attn(ctypes.byref(c), fake, fake, fake, fake, fake, fake, 1, fake, None) == code
    assert L.hybrid_commit_block(ctypes.byref(c), fake, fake, 32, fake, fake, 1, None) == code
    assert L.hybrid_state_init(ctypes.byref(c), fake, 1, None) == code


def test_null_and_misaligned_pointers_rejected_on_host(L):
    c = cfg()
    ok = 1 << 20
    assert L.hybrid_block_attn(ctypes.byref(c), None, ok, ok, ok, ok, ok, 1, ok, None) == H.HYBRID_ERR_INVALID_ARG
    assert L.hybrid_block_attn(ctypes.byref(c), ok + 8, ok, ok, ok, ok, ok, 1, ok, None) == H.HYBRID_ERR_INVALID_ARG
    assert L.hybrid_block_attn(ctypes.byref(c), ok, ok, ok, ok, ok + 2, ok, 1, ok, None) == H.HYBRID_ERR_INVALID_ARG
    assert L.hybrid_commit_block(ctypes.byref(c), ok, None, 32, ok, ok, 1, None) == H.HYBRID_ERR_INVALID_ARG
    assert L.hybrid_commit_block(ctypes.byref(c), ok, ok, -1, ok, ok, 1, None) == H.HYBRID_ERR_INVALID_ARG
    assert L.hybrid_block_attn(ctypes.byref(c), ok, ok, ok, ok, ok, ok, -1, ok, None) == H.HYBRID_ERR_INVALID_ARG
    assert L.hybrid_feature_map(ctypes.byref(c), ok, 4, 3, ok, ok, None) == H.HYBRID_ERR_INVALID_ARG
    assert L.hybrid_block_attn(None, ok, ok, ok, ok, ok, ok, 1, ok, None) == H.HYBRID_ERR_INVALID_ARG


def test_empty_batches_are_no_ops(L):
    c = cfg()
    assert L.hybrid_block_attn(ctypes.byref(c), None, None, None, None, None, None, 0, None, None) == H.HYBRID_OK
    assert L.hybrid_commit_block(ctypes.byref(c), None, None, 32, None, None, 0, None) == H.HYBRID_OK
    assert L.hybrid_commit_block(ctypes.byref(c), None, None, 0, None, None, 5, None) == H.HYBRID_OK
    assert L.hybrid_state_init(ctypes.byref(c), None, 0, None) == H.HYBRID_OK


def test_status_strings(L):
    for s in range(6):
        assert H.hybrid_status_str(s).startswith("HYBRID_")
    assert "UNKNOWN" in H.hybrid_status_str(99)


def test_binding_names_match_abi():
    for name in H.EXPORTED:
        assert callable(getattr(H, name))
