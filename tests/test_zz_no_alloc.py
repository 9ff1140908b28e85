"""hybrid_block_attn_commit_logical: the fused step and commit for callers that
cannot allocate device memory and keep their states in the logical layout.
The entry point works in the library's own static scratch instead.

It is compared with the pointer-array entry point (hybrid_block_attn_commit on
the same states packed into a pool) over two consecutive calls. Outputs and
committed states must match bit for bit, because the same kernels run on the
same packed bytes. That is tighter than the bf16 parity bound the other tests
use (rel-L2 <= 1e-2 against the oracle).

Every tensor is allocated, and every kernel the two entry points launch is
loaded, in one warm-up call before free device memory is sampled. The measured
calls then run on preallocated buffers, so a change of free memory can only
come from the entry point itself. The file is named so that pytest collects it
last; it also passes when run alone in a fresh process.
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


def test_logical_entry_matches_pointer_path_on_two_calls():
    wl = wk.C3.with_(n_req=12)
    n, P2 = wl.n_req, 2 * wl.F
    cfg = H.make_cfg(wl.d, wl.F, wl.Hq, wl.Hkv, wl.B, wl.io_dtype)
    W, alpha = wk.params(wl, device="cuda")
    pool = StatePool(cfg, n, "cuda")
    ptrs = pool.all_ptrs()
    H.hybrid_state_init(cfg, ptrs, n)
    plen = np.array([32 * (i % 5) for i in range(n)])
    for b in range(int(plen.max()) // wl.B):
        reqs = np.nonzero(plen > b * wl.B)[0]
        K, V = wk.prefix_kv(wl, b, "cuda", n_req=len(reqs))
        H.hybrid_commit_block(cfg, K, V, wl.B, W, pool.ptr_array(reqs.tolist()), len(reqs))

    def buf(*shape):
        return torch.empty(shape, dtype=torch.float32, device="cuda")

    # every buffer of the warm-up and the two measured calls, allocated up front
    S_log, z_log = buf(n, wl.Hkv, P2, wl.d), buf(n, wl.Hkv, P2)
    S_ref, z_ref = buf(n, wl.Hkv, P2, wl.d), buf(n, wl.Hkv, P2)
    S_got = [buf(n, wl.Hkv, P2, wl.d) for _ in range(2)]
    z_got = [buf(n, wl.Hkv, P2) for _ in range(2)]
    S_want = [buf(n, wl.Hkv, P2, wl.d) for _ in range(2)]
    z_want = [buf(n, wl.Hkv, P2) for _ in range(2)]
    inputs = [wk.block_qkv(wl, ("no_alloc", call), "cuda") for call in ("warm", 0, 1)]
    O_ref = [torch.empty_like(inputs[0][0]) for _ in range(3)]
    O_log = [torch.empty_like(inputs[0][0]) for _ in range(3)]
    H.hybrid_state_unpack(cfg, ptrs, n, S_log, z_log)
    H.hybrid_check()

    def one_call(i):
        Q, K, V = inputs[i]
        H.hybrid_block_attn_commit(cfg, Q, K, V, W, alpha, ptrs, n, O_ref[i])
        H.hybrid_block_attn_commit_logical(cfg, Q, K, V, W, alpha, S_log, z_log, n, O_log[i])
        H.hybrid_state_unpack(cfg, ptrs, n, S_ref, z_ref)
        H.hybrid_check()

    # warm-up: the set-up call (n_req = 0 looks the scratch address up), then one
    # full call of both entry points, which loads every kernel they launch
    H.hybrid_block_attn_commit_logical(cfg, None, None, None, None, None, None, None, 0, None)
    one_call(0)
    torch.cuda.synchronize()
    free_before = torch.cuda.mem_get_info()[0]
    reserved_before = torch.cuda.memory_reserved()
    for call in range(2):
        one_call(call + 1)
        S_got[call].copy_(S_log)
        z_got[call].copy_(z_log)
        S_want[call].copy_(S_ref)
        z_want[call].copy_(z_ref)
    torch.cuda.synchronize()
    assert torch.cuda.mem_get_info()[0] == free_before, "free device memory changed"
    assert torch.cuda.memory_reserved() == reserved_before, "torch reserved more memory"

    assert torch.equal(O_ref[0], O_log[0]), "warm-up call: outputs differ"
    for call in range(2):
        assert torch.equal(O_ref[call + 1], O_log[call + 1]), f"call {call}: outputs differ"
        assert torch.equal(S_want[call], S_got[call]), f"call {call}: committed S differs"
        assert torch.equal(z_want[call], z_got[call]), f"call {call}: committed z differs"
    # the second call started from the first call's committed state
    assert not torch.equal(S_got[0], S_got[1])


def test_logical_entry_rejects_more_than_the_scratch():
    wl = wk.C5
    cfg = H.make_cfg(wl.d, wl.F, wl.Hq, wl.Hkv, wl.B, wl.io_dtype)
    per_req = H.hybrid_state_bytes(cfg)
    n = ((64 << 20) - 255) // (per_req + 8) + 1   # one request more than the scratch holds
    dummy = torch.empty(16, dtype=torch.float32, device="cuda")
    st = H.hybrid_block_attn_commit_logical(cfg, dummy, dummy, dummy, dummy, dummy, dummy, dummy, n, dummy,
                                            check=False)
    assert st == H.HYBRID_ERR_UNSUPPORTED
    assert H.hybrid_check(check=False) == H.HYBRID_OK
