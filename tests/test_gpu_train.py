"""Training form (Section 3.2, Stage 1 attention transfer) on the GPU against
the fp64 oracle, through the C ABI: the output of every block of a sequence
and the gradient of sum(dO * O) with respect to W and alpha.

bf16 inputs with fp32 states and gradients: rel-L2 <= 1e-2 for O, dW and
dalpha.  The oracle sees host copies of exactly the tensors the GPU consumed.
"""
import numpy as np
import pytest
import torch

import oracle
from gpu_harness import h64, rel_l2
from paper_2608_06628_gb300 import hybrid as H
from paper_2608_06628_gb300 import workloads as wk

pytestmark = pytest.mark.gpu

TOL = 1e-2


@pytest.fixture(scope="module", autouse=True)
def _device():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_06628_gb300 import build
    build.build()
    torch.cuda.set_device(0)


def TW(name, n, L, Hq, Hkv, d, F, B, seed):
    return wk.Workload(name, torch.bfloat16, n, Hq, Hkv, d, F, B, seed, seq_len=L)


def run_gpu(wl, Q, K, V, W, alpha, dO):
    cfg = H.make_cfg(wl.d, wl.F, wl.Hq, wl.Hkv, wl.B, wl.io_dtype)
    n_seq, L = Q.shape[0], Q.shape[1]
    nbytes = H.hybrid_train_workspace_bytes(cfg, n_seq, L)
    assert nbytes > 0
    ws = torch.empty(nbytes + 1024, dtype=torch.uint8, device="cuda")
    ptr = (ws.data_ptr() + 1023) & ~1023
    O = torch.empty_like(Q)
    H.hybrid_train_forward(cfg, Q, K, V, W, alpha, n_seq, L, O, ptr, nbytes)
    dW = torch.empty(W.shape, dtype=torch.float32, device="cuda")
    dalpha = torch.empty(wl.Hq, dtype=torch.float32, device="cuda")
    H.hybrid_train_backward(cfg, Q, K, V, W, alpha, dO, n_seq, L, ptr, nbytes, dW, dalpha)
    H.hybrid_check()
    return O, dW, dalpha


def inputs(wl, n_seq=None, seq_len=None):
    Q, K, V, dO = wk.train_batch(wl, device="cuda", n_seq=n_seq, seq_len=seq_len)
    W, alpha = wk.params(wl, 0, "cuda")
    return Q, K, V, W, alpha, dO


CASES = [
    TW("gqa_d128_f128_b32", 2, 128, 8, 2, 128, 128, 32, 41),
    TW("gqa_d64_f64_b16", 3, 80, 4, 2, 64, 64, 16, 42),
    TW("mha_d128_f64_b32", 2, 96, 2, 2, 128, 64, 32, 43),
    TW("g2_d128_f128_b64", 1, 192, 4, 2, 128, 128, 64, 44),
    TW("g8_d64_f128_b16", 1, 64, 8, 1, 64, 128, 16, 45),
]


@pytest.mark.parametrize("wl", CASES, ids=[w.name for w in CASES])
def test_train_parity(wl):
    Q, K, V, W, alpha, dO = inputs(wl)
    O, dW, dalpha = run_gpu(wl, Q, K, V, W, alpha, dO)
    orc = oracle.load()
    args = (h64(Q), h64(K), h64(V), h64(W), h64(alpha))
    O_ref = orc.train_forward(*args, wl.B)
    dW_ref, da_ref = orc.train_backward(*args, h64(dO), wl.B)
    for got, want, what in ((O, O_ref, "O"), (dW, dW_ref, "dW"), (dalpha, da_ref, "dalpha")):
        g = h64(got)
        assert np.all(np.isfinite(g)), f"{wl.name} {what}: non-finite"
        r = rel_l2(g, want)
        assert r <= TOL, f"{wl.name} {what}: rel-L2 {r:.3e}"


def test_train_stress_keys_and_saturated_gate():
    """Keys x 8 (scores up to ~30, the stress setting of the decoding configs) and
    one gate saturated at alpha = +inf (w = 1, so its dalpha is 0)."""
    wl = TW("k8_sat", 2, 128, 8, 2, 128, 128, 32, 47).with_(k_scale=8.0)
    Q, K, V, W, alpha, dO = inputs(wl)
    alpha[3] = float("inf")
    O, dW, dalpha = run_gpu(wl, Q, K, V, W, alpha, dO)
    orc = oracle.load()
    args = (h64(Q), h64(K), h64(V), h64(W), h64(alpha))
    O_ref = orc.train_forward(*args, wl.B)
    dW_ref, da_ref = orc.train_backward(*args, h64(dO), wl.B)
    assert rel_l2(h64(O), O_ref) <= TOL
    assert rel_l2(h64(dW), dW_ref) <= TOL
    assert rel_l2(h64(dalpha), da_ref) <= TOL
    assert float(dalpha[3]) == 0.0


def test_train_single_block_has_no_gradient():
    """One block per sequence: no prefix anywhere, so O is the in-block softmax
    and dW is exactly zero; dalpha is zero up to rounding."""
    wl = TW("single_block", 2, 32, 4, 1, 128, 128, 32, 46)
    Q, K, V, W, alpha, dO = inputs(wl)
    O, dW, dalpha = run_gpu(wl, Q, K, V, W, alpha, dO)
    orc = oracle.load()
    O_ref = orc.train_forward(h64(Q), h64(K), h64(V), h64(W), h64(alpha), wl.B)
    assert rel_l2(h64(O), O_ref) <= TOL
    assert float(dW.abs().max()) == 0.0
    assert float(dalpha.abs().max()) < 1e-3


def test_train_constant_values_full_size():
    """V = 1 everywhere makes O = 1 for any W and alpha, so the gradients vanish,
    at the full training-batch size (8 sequences of 2048 tokens)."""
    wl = wk.T1
    Q, K, V, W, alpha, dO = inputs(wl)
    _, dW_r, da_r = run_gpu(wl, Q, K, V, W, alpha, dO)
    V1 = torch.ones_like(V)
    O1, dW1, da1 = run_gpu(wl, Q, K, V1, W, alpha, dO)
    assert float((O1.float() - 1).abs().max()) < 1e-2
    assert float(dW1.norm()) < 1e-2 * float(dW_r.norm())
    assert float(da1.norm()) < 1e-2 * float(da_r.norm())


def test_train_full_length_sequence():
    """One 2048-token sequence of the training batch's shape (64 blocks, GQA
    16:4, d = F = 128) against the oracle: O, dW and dalpha."""
    wl = wk.T1
    Q, K, V, W, alpha, dO = inputs(wl, n_seq=1)
    O, dW, dalpha = run_gpu(wl, Q, K, V, W, alpha, dO)
    orc = oracle.load()
    args = (h64(Q), h64(K), h64(V), h64(W), h64(alpha))
    O_ref = orc.train_forward(*args, wl.B)
    dW_ref, da_ref = orc.train_backward(*args, h64(dO), wl.B)
    assert rel_l2(h64(O), O_ref) <= TOL
    assert rel_l2(h64(dW), dW_ref) <= TOL
    assert rel_l2(h64(dalpha), da_ref) <= TOL


def test_train_gradient_linear_in_dO():
    """At the full training-batch size: the gradient is linear in dO."""
    wl = wk.T1
    Q, K, V, W, alpha, dO = inputs(wl)
    dO2 = wk.train_batch(wl, tag=1, device="cuda")[3]
    _, dW1, da1 = run_gpu(wl, Q, K, V, W, alpha, dO)
    _, dW2, da2 = run_gpu(wl, Q, K, V, W, alpha, dO2)
    _, dW3, da3 = run_gpu(wl, Q, K, V, W, alpha, (dO.float() + dO2.float()).to(dO.dtype))
    assert rel_l2(h64(dW3), h64(dW1) + h64(dW2)) <= TOL
    assert rel_l2(h64(da3), h64(da1) + h64(da2)) <= TOL


def test_train_calls_allocate_nothing():
    """After a first call (kernel attributes set), forward and backward allocate no
    device memory: free device memory is unchanged across further calls, and the
    results are bitwise repeatable on the same workspace."""
    wl = TW("no_alloc", 2, 128, 8, 2, 128, 128, 32, 48)
    Q, K, V, W, alpha, dO = inputs(wl)
    cfg = H.make_cfg(wl.d, wl.F, wl.Hq, wl.Hkv, wl.B, wl.io_dtype)
    n, L = Q.shape[0], Q.shape[1]
    nbytes = H.hybrid_train_workspace_bytes(cfg, n, L)
    ws = torch.empty(nbytes + 1024, dtype=torch.uint8, device="cuda")
    ptr = (ws.data_ptr() + 1023) & ~1023
    outs = []
    for call in range(3):
        O = torch.empty_like(Q)
        dW = torch.empty(W.shape, dtype=torch.float32, device="cuda")
        da = torch.empty(wl.Hq, dtype=torch.float32, device="cuda")
        torch.cuda.synchronize()
        free_before = torch.cuda.mem_get_info()[0]
        H.hybrid_train_forward(cfg, Q, K, V, W, alpha, n, L, O, ptr, nbytes)
        H.hybrid_train_backward(cfg, Q, K, V, W, alpha, dO, n, L, ptr, nbytes, dW, da)
        H.hybrid_check()
        if call > 0:
            assert torch.cuda.mem_get_info()[0] == free_before, f"call {call} allocated device memory"
        outs.append((O, dW, da))
    assert torch.equal(outs[1][0], outs[2][0])
    # dW and dalpha add their partial sums in a fixed order
    assert torch.equal(outs[1][1], outs[2][1])
    assert torch.equal(outs[1][2], outs[2][2])


def test_train_gradients_bitwise_repeatable():
    """At the full training-batch size (many CTAs per state head in the dW
    reduction, 64 blocks per sequence in the dalpha one), two backward passes on
    separate workspaces give the same dW and dalpha bits."""
    wl = wk.T1
    Q, K, V, W, alpha, dO = inputs(wl)
    _, dW1, da1 = run_gpu(wl, Q, K, V, W, alpha, dO)
    _, dW2, da2 = run_gpu(wl, Q, K, V, W, alpha, dO)
    assert torch.equal(dW1, dW2)
    assert torch.equal(da1, da2)
