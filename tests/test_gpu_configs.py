"""The five workload configurations at their full sizes, against the fp64 oracle.

The GPU runs every request of the configuration; the oracle follows a seeded
sample of requests (always including the shortest and the longest prefix),
consuming host copies of exactly the tensors the GPU saw.  Tolerances are the
ones of gpu_harness.TOL (bf16 I/O with fp32 state: rel-L2 <= 1e-2 for outputs
and committed states).
"""
import numpy as np
import pytest
import torch

from gpu_harness import Pair, assert_parity, h64
from paper_2608_06628_gb300 import hybrid as H
from paper_2608_06628_gb300 import workloads as wk

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _device():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_06628_gb300 import build
    build.build()
    torch.cuda.set_device(0)


def _sample(plen, n_extra, seed):
    """Indices of the shortest and longest prefix plus n_extra seeded others."""
    rng = np.random.default_rng(seed)
    picks = {int(np.argmin(plen)), int(np.argmax(plen))}
    rest = [i for i in range(len(plen)) if i not in picks]
    picks.update(int(i) for i in rng.choice(rest, size=min(n_extra, len(rest)), replace=False))
    return np.array(sorted(picks))


def _fused_call(pair, tag):
    """One hybrid_block_attn_commit over the whole batch (the bench's launch);
    returns the GPU output of the tracked requests and the oracle's."""
    wl = pair.wl
    Q, K, V = wk.block_qkv(wl, tag, pair.dev)
    O = torch.empty_like(Q)
    H.hybrid_block_attn_commit(pair.cfg, Q, K, V, pair.W, pair.alpha, pair.ptrs, wl.n_req, O)
    H.hybrid_check()
    t = torch.as_tensor(pair.tracked, device=pair.dev)
    want = pair.orc.block_attn(h64(Q[t]), h64(K[t]), h64(V[t]), pair.W64, pair.alpha64, pair.S, pair.z)
    pair.orc.commit(h64(K[t]), h64(V[t]), pair.W64, pair.S, pair.z)
    return h64(O[t]), want


def test_c2_full_step_plus_commit():
    """c2: 8 requests, MHA 16 heads, prefix 2048 (64 commits); one call = one
    denoising step plus the commit of its block."""
    wl = wk.C2
    pair = Pair(wl, tracked=[0, 3, 7])
    pair.build_prefixes(wk.prefix_lengths(wl))
    S, z = pair.gpu_state()
    assert_parity(S, pair.S, wl.io_dtype, "c2 prefix state S", units="state")
    got, want = _fused_call(pair, "c2_step")
    assert_parity(got, want, wl.io_dtype, "c2 output", units="out")
    S, z = pair.gpu_state()
    assert_parity(S, pair.S, wl.io_dtype, "c2 committed state S", units="state")
    assert_parity(z, pair.z, wl.io_dtype, "c2 committed state z", units="state")


def test_c3_full_bench_launch():
    """c3 (the bench workload): 64 ragged requests, GQA 16:4, in the launch
    configuration bench.py times (hybrid_block_attn_commit over the batch)."""
    wl = wk.C3
    plen = wk.prefix_lengths(wl)
    pair = Pair(wl, tracked=_sample(plen, 3, 101))
    pair.build_prefixes(plen)
    for step in range(2):
        got, want = _fused_call(pair, ("c3_step", step))
        assert_parity(got, want, wl.io_dtype, f"c3 output, step {step}", units="out")
        S, z = pair.gpu_state()
        assert_parity(S, pair.S, wl.io_dtype, f"c3 committed state S, step {step}", units="state")
        assert_parity(z, pair.z, wl.io_dtype, f"c3 committed state z, step {step}", units="state")
    # the attention-only step against the grown state as well
    Q, K, V = wk.block_qkv(wl, "c3_attn", pair.dev)
    got, want, _ = pair.step(Q, K, V)
    assert_parity(got, want, wl.io_dtype, "c3 attention-only output", units="out")


def test_c4_decode_loop_drift():
    """c4: 32 requests, 6 hybrid layers x 64 blocks x 8 denoising steps from an
    empty state.  Seven steps per block are attention-only; the eighth computes
    the step and commits its block in one call.  The oracle follows two requests
    through every layer and commit; their outputs are checked on sampled steps
    and their states after the final block (accumulated drift)."""
    wl = wk.C4
    tracked = [0, wl.n_req - 1]
    pairs = [Pair(wl, layer=L, tracked=tracked) for L in range(wl.layers)]
    t = torch.as_tensor(tracked, device="cuda")
    checked = 0
    for blk in range(wl.blocks):
        for step in range(wl.steps_per_block):
            last = step == wl.steps_per_block - 1
            sample = (blk in (0, 17, wl.blocks - 1)) and step in (0, wl.steps_per_block - 1)
            for L, pair in enumerate(pairs):
                Q, K, V = wk.block_qkv(wl, ("c4", L, blk, step), pair.dev)
                O = torch.empty_like(Q)
                fn = H.hybrid_block_attn_commit if last else H.hybrid_block_attn
                fn(pair.cfg, Q, K, V, pair.W, pair.alpha, pair.ptrs, wl.n_req, O)
                if sample:
                    H.hybrid_check()
                    want = pair.orc.block_attn(h64(Q[t]), h64(K[t]), h64(V[t]), pair.W64, pair.alpha64,
                                               pair.S, pair.z)
                    assert_parity(h64(O[t]), want, wl.io_dtype, f"c4 layer {L} block {blk} step {step}", units="out")
                    checked += 1
                if last:
                    pair.orc.commit(h64(K[t]), h64(V[t]), pair.W64, pair.S, pair.z)
    H.hybrid_check()
    assert checked == 6 * wl.layers
    for L, pair in enumerate(pairs):
        S, z = pair.gpu_state()
        assert_parity(S, pair.S, wl.io_dtype, f"c4 final state S, layer {L}", units="state")
        assert_parity(z, pair.z, wl.io_dtype, f"c4 final state z, layer {L}", units="state")


def test_c5_full_sampled():
    """c5: 256 requests, 16 heads, F = 256, B = 64, ragged prefixes 1k-32k with
    keys x8 (normaliser and softmax range).  The GPU builds every prefix; the
    oracle rebuilds 8 seeded requests (the shortest, the longest and six others),
    then checks a step and the following commit on them.  The step is also checked for every
    request, the oracle reading the GPU's prefix states (a full oracle rebuild of
    all 256 prefixes is out of reach)."""
    wl = wk.C5
    plen = wk.prefix_lengths(wl)
    pair = Pair(wl, tracked=_sample(plen, 6, 105))
    assert len(pair.tracked) == 8
    pair.build_prefixes(plen)
    S, z = pair.gpu_state()
    assert_parity(S, pair.S, wl.io_dtype, "c5 prefix state S", units="state")
    assert_parity(z, pair.z, wl.io_dtype, "c5 prefix state z", units="state")
    Q, K, V = wk.block_qkv(wl, "c5_step", pair.dev)
    got, want, O = pair.step(Q, K, V)
    assert_parity(got, want, wl.io_dtype, "c5 output", units="out")
    for r0 in range(0, wl.n_req, 32):
        reqs = np.arange(r0, min(r0 + 32, wl.n_req))
        Sg, zg = pair.gpu_state(reqs)
        t = torch.as_tensor(reqs, device=pair.dev)
        want = pair.orc.block_attn(h64(Q[t]), h64(K[t]), h64(V[t]), pair.W64, pair.alpha64, Sg, zg)
        assert_parity(h64(O[t]), want, wl.io_dtype, f"c5 output, requests {r0}..{reqs[-1]}", units="out")
    pair.commit(K, V)
    S, z = pair.gpu_state()
    assert_parity(S, pair.S, wl.io_dtype, "c5 committed state S", units="state")
    assert_parity(z, pair.z, wl.io_dtype, "c5 committed state z", units="state")
