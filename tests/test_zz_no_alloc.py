"""hybrid_block_attn_commit_logical: the fused step and commit on states kept in
the logical layout, through the library's static scratch (no allocation).

Compared with the pointer-array entry point (hybrid_block_attn_commit on the
same states packed into a pool) over two consecutive calls: outputs and
committed states must match bit for bit (same kernels, same packed bytes).
"""
import numpy as np
import pytest
import torch

from paper_2608_06628_gb300 import hybrid as H
from paper_2608_06628_gb300 import workloads as wk
from paper_2608_06628_gb300.state_pool import StatePool

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _device():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_06628_gb300 import build
    build.build()
    torch.cuda.set_device(0)


def _logical(cfg, pool, n, wl):
    S = torch.empty((n, wl.Hkv, 2 * wl.F, wl.d), dtype=torch.float32, device="cuda")
    z = torch.empty((n, wl.Hkv, 2 * wl.F), dtype=torch.float32, device="cuda")
    H.hybrid_state_unpack(cfg, pool.all_ptrs(), n, S, z)
    return S, z


def test_logical_entry_matches_pointer_path_on_two_calls():
    wl = wk.C3.with_(n_req=12)
    cfg = H.make_cfg(wl.d, wl.F, wl.Hq, wl.Hkv, wl.B, wl.io_dtype)
    W, alpha = wk.params(wl, device="cuda")
    pool = StatePool(cfg, wl.n_req, "cuda")
    ptrs = pool.all_ptrs()
    H.hybrid_state_init(cfg, ptrs, wl.n_req)
    plen = np.array([32 * (i % 5) for i in range(wl.n_req)])
    for b in range(int(plen.max()) // wl.B):
        reqs = np.nonzero(plen > b * wl.B)[0]
        K, V = wk.prefix_kv(wl, b, "cuda", n_req=len(reqs))
        H.hybrid_commit_block(cfg, K, V, wl.B, W, pool.ptr_array(reqs.tolist()), len(reqs))
    S_log, z_log = _logical(cfg, pool, wl.n_req, wl)
    H.hybrid_check()

    # set-up call (looks the scratch address up), then measure free device memory
    H.hybrid_block_attn_commit_logical(cfg, None, None, None, None, None, S_log, z_log, 0, None)
    torch.cuda.synchronize()
    free_before = torch.cuda.mem_get_info()[0]
    for call in range(2):
        Q, K, V = wk.block_qkv(wl, ("no_alloc", call), "cuda")
        O_ref, O_log = torch.empty_like(Q), torch.empty_like(Q)
        H.hybrid_block_attn_commit(cfg, Q, K, V, W, alpha, ptrs, wl.n_req, O_ref)
        H.hybrid_block_attn_commit_logical(cfg, Q, K, V, W, alpha, S_log, z_log, wl.n_req, O_log)
        H.hybrid_check()
        assert torch.equal(O_ref, O_log), f"call {call}: outputs differ"
        S_ref, z_ref = _logical(cfg, pool, wl.n_req, wl)
        H.hybrid_check()
        assert torch.equal(S_ref, S_log), f"call {call}: committed S differs"
        assert torch.equal(z_ref, z_log), f"call {call}: committed z differs"
    torch.cuda.synchronize()
    assert torch.cuda.mem_get_info()[0] == free_before


def test_logical_entry_rejects_more_than_the_scratch():
    wl = wk.C5
    cfg = H.make_cfg(wl.d, wl.F, wl.Hq, wl.Hkv, wl.B, wl.io_dtype)
    per_req = H.hybrid_state_bytes(cfg)
    n = (64 << 20) // per_req + 1   # one request more than the scratch holds
    dummy = torch.empty(16, dtype=torch.float32, device="cuda")
    st = H.hybrid_block_attn_commit_logical(cfg, dummy, dummy, dummy, dummy, dummy, dummy, dummy, n, dummy,
                                            check=False)
    assert st == H.HYBRID_ERR_UNSUPPORTED
    assert H.hybrid_check(check=False) == H.HYBRID_OK
