"""CUDA path vs the fp64 oracle, element by element, through the C ABI.

Sizes span several tiles and ragged tails while the oracle still finishes in
seconds.  Tolerances (written in gpu_harness.TOL): fp32 I/O rel-L2 <= 1e-5 and
max-abs <= 1e-4; bf16 I/O with fp32 state rel-L2 <= 1e-2, for outputs and for
committed states alike.
"""
import math

import numpy as np
import pytest
import torch

from gpu_harness import Pair, assert_parity, h64, rel_l2
from paper_2608_06628_gb300 import hybrid as H
from paper_2608_06628_gb300 import workloads as wk
from paper_2608_06628_gb300.state_pool import StatePool

pytestmark = pytest.mark.gpu

BF16, F32 = torch.bfloat16, torch.float32


@pytest.fixture(scope="module", autouse=True)
def _device():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_06628_gb300 import build
    build.build()
    torch.cuda.set_device(0)


def W_(name, dt, n, Hq, Hkv, d, F, B, seed, pmin=0, pmax=0, k_scale=1.0):
    return wk.Workload(name, dt, n, Hq, Hkv, d, F, B, seed, pmin, pmax, k_scale)


# small cases: (workload, explicit ragged prefix lengths)
SMALL = [
    (wk.C1, None),
    (W_("mha_bf16", BF16, 3, 4, 4, 128, 128, 32, 11), [64, 0, 96]),
    (W_("gqa4_bf16", BF16, 5, 8, 2, 128, 128, 32, 12), [0, 32, 96, 160, 256]),
    (W_("f256_b64_k8_bf16", BF16, 3, 2, 2, 128, 256, 64, 13, k_scale=8.0), [0, 128, 384]),
    (W_("d64_f64_bf16", BF16, 4, 4, 2, 64, 64, 32, 14), [32, 64, 0, 128]),
    (W_("d64_f16_b16_f32", F32, 3, 2, 1, 64, 16, 16, 15), [16, 48, 0]),
    (W_("f32_b48_ragged_rows", F32, 2, 3, 3, 128, 32, 48, 16), [96, 48]),
    (W_("bf16_b48_f32feat", BF16, 2, 4, 4, 128, 32, 48, 17), [48, 144]),
    (W_("bf16_g8_b32_generic", BF16, 2, 8, 1, 128, 64, 32, 18), [64, 32]),
    (W_("bf16_b16_g2", BF16, 3, 4, 2, 128, 128, 16, 19), [16, 0, 80]),
    (W_("bf16_b64_g2", BF16, 2, 4, 2, 64, 128, 64, 20), [128, 64]),
    # d > F on the two-issuer readout: P'V waits for the second issuer's tiles
    (W_("bf16_d128_f64_b64", BF16, 2, 4, 2, 128, 64, 64, 27), [64, 0]),
    (W_("f32_mha_f128", F32, 2, 2, 2, 128, 128, 32, 21), [64, 32]),
    # F = 256 on the tensor cores: phi+ and phi- read out in turn; commits in one
    # pass per sign.  GQA with d = 64; 320 commit passes over 152 CTAs; G = 4, B = 16
    (W_("f256_gqa2_d64_b32", BF16, 4, 4, 2, 64, 256, 32, 22), [32, 0, 96, 160]),
    (W_("f256_many_units", BF16, 40, 8, 4, 128, 256, 32, 23), list((np.arange(40) % 4) * 32)),
    (W_("f256_g4_b16", BF16, 3, 8, 2, 128, 256, 16, 24), [16, 48, 0]),
    # G = 1, B = 64: the step spreads its 64 rows over all four TMEM lane quarters
    (W_("spread_f128_b64", BF16, 3, 4, 4, 128, 128, 64, 25), [64, 0, 128]),
    (W_("spread_d64_f64_b64", BF16, 3, 2, 2, 64, 64, 64, 26), [128, 64, 0]),
]


def _plen(wl, plen):
    return wk.prefix_lengths(wl) if plen is None else np.asarray(plen, dtype=np.int64)


@pytest.mark.parametrize("wl,plen", SMALL, ids=[w.name for w, _ in SMALL])
def test_commit_then_step_parity(wl, plen):
    pair = Pair(wl)
    plen = _plen(wl, plen)
    pair.build_prefixes(plen)
    S, z = pair.gpu_state()
    assert_parity(S, pair.S, wl.io_dtype, "prefix state S", units="state")
    assert_parity(z, pair.z, wl.io_dtype, "prefix state z", units="state")
    Q, K, V = wk.block_qkv(wl, "step", pair.dev)
    got, want, _ = pair.step(Q, K, V)
    assert_parity(got, want, wl.io_dtype, "block attention output", units="out")
    # fold the active block in (the final denoising step's K/V) and compare the state
    pair.commit(K, V)
    S, z = pair.gpu_state()
    assert_parity(S, pair.S, wl.io_dtype, "post-commit state S", units="state")
    assert_parity(z, pair.z, wl.io_dtype, "post-commit state z", units="state")
    # a second step against the grown state
    Q2, K2, V2 = wk.block_qkv(wl, "step2", pair.dev)
    got, want, _ = pair.step(Q2, K2, V2)
    assert_parity(got, want, wl.io_dtype, "second step output", units="out")


@pytest.mark.parametrize("dt", [F32, BF16])
@pytest.mark.parametrize("d,F,nh,Hkv", [(64, 16, 2, 1), (128, 128, 16, 4), (128, 256, 3, 3), (64, 64, 4, 4)])
def test_feature_map_parity(dt, d, F, nh, Hkv):
    import oracle
    g = torch.Generator(device="cuda").manual_seed(d * 1000 + F + nh)
    n_rows = 37
    X = (torch.randn((n_rows, nh, d), generator=g, device="cuda") * 1.5).to(dt)
    W = (torch.randn((Hkv, d, F), generator=g, device="cuda") / math.sqrt(d)).to(dt)
    cfg = H.make_cfg(d, F, nh, Hkv, 32, dt)
    Phi = torch.empty((n_rows, nh, 2 * F), dtype=torch.float32, device="cuda")
    H.hybrid_feature_map(cfg, X, n_rows, nh, W, Phi)
    H.hybrid_check()
    want = oracle.load().feature_map(h64(X), h64(W))
    # phi is computed and returned in float32 from exactly representable inputs
    assert_parity(h64(Phi), want, F32, "phi")


def test_state_layout_matches_header_formula():
    """pack/unpack round trip is exact, and the raw bytes follow the documented
    offset formula (f/32)*32*d + e*32 + 4*(((f%32)/4) ^ (e%8)) + f%4, z at 2F*d + f."""
    d, F, Hkv = 64, 32, 2
    cfg = H.make_cfg(d, F, 2, Hkv, 16, F32)
    pool = StatePool(cfg, 3, "cuda")
    ptrs = pool.all_ptrs()
    g = torch.Generator(device="cuda").manual_seed(5)
    S = torch.randn((3, Hkv, 2 * F, d), generator=g, device="cuda")
    z = torch.randn((3, Hkv, 2 * F), generator=g, device="cuda")
    H.hybrid_state_pack(cfg, S, z, ptrs, 3)
    S2, z2 = torch.empty_like(S), torch.empty_like(z)
    H.hybrid_state_unpack(cfg, ptrs, 3, S2, z2)
    H.hybrid_check()
    assert torch.equal(S, S2) and torch.equal(z, z2)
    raw = pool.slab.view(3, Hkv, -1).cpu().numpy()
    Sh, zh = S.cpu().numpy(), z.cpu().numpy()
    f = np.arange(2 * F)[:, None]
    e = np.arange(d)[None, :]
    off = (f // 32) * 32 * d + e * 32 + 4 * (((f % 32) // 4) ^ (e % 8)) + f % 4
    for r in range(3):
        for h in range(Hkv):
            assert np.array_equal(raw[r, h][off], Sh[r, h])
            assert np.array_equal(raw[r, h][2 * F * d + np.arange(2 * F)], zh[r, h])


def test_state_init_zeroes():
    cfg = H.make_cfg(128, 128, 16, 4, 32, BF16)
    pool = StatePool(cfg, 4, "cuda")
    pool.slab.fill_(7.0)
    H.hybrid_state_init(cfg, pool.ptr_array([0, 2]), 2)
    H.hybrid_check()
    n = pool.slot_bytes // 4
    assert torch.count_nonzero(pool.slab[:n]) == 0
    assert torch.all(pool.slab[n:2 * n] == 7.0)
    assert torch.count_nonzero(pool.slab[2 * n:3 * n]) == 0


# ---------------------------------------------------------------------------
# edge cases
# ---------------------------------------------------------------------------
EDGE_WL = [W_("edge_gqa_bf16", BF16, 3, 8, 2, 128, 128, 32, 31),
           W_("edge_gqa_k24_bf16", BF16, 3, 8, 2, 128, 128, 32, 33, k_scale=24.0),
           W_("edge_f32", F32, 2, 2, 2, 64, 64, 16, 32),
           # the one-CTA-per-unit tensor-core step: F = 256 (phi+ then phi-), and G B = 128
           W_("edge_f256_k8_bf16", BF16, 3, 2, 2, 128, 256, 64, 34, k_scale=8.0),
           W_("edge_b64_g2_bf16", BF16, 3, 4, 2, 64, 128, 64, 35)]


@pytest.mark.parametrize("wl", EDGE_WL, ids=[w.name for w in EDGE_WL])
def test_gate_limits(wl):
    pair = Pair(wl)
    pair.build_prefixes(np.full(wl.n_req, 2 * wl.B))
    Q, K, V = wk.block_qkv(wl, "gate", pair.dev)
    for a in (math.inf, -math.inf, 30.0, -30.0, 0.0):
        alpha = torch.full((wl.Hq,), a, dtype=torch.float32, device=pair.dev)
        got, want, _ = pair.step(Q, K, V, alpha)
        assert_parity(got, want, wl.io_dtype, f"alpha={a}", units="out")


@pytest.mark.parametrize("wl", EDGE_WL, ids=[w.name for w in EDGE_WL])
def test_empty_prefix_is_block_softmax(wl):
    pair = Pair(wl)
    Q, K, V = wk.block_qkv(wl, "empty", pair.dev)
    got, want, O = pair.step(Q, K, V)
    assert_parity(got, want, wl.io_dtype, "empty prefix", units="out")
    G = wl.Hq // wl.Hkv
    q = Q.float().permute(0, 2, 1, 3)
    k = K.float().repeat_interleave(G, dim=2).permute(0, 2, 1, 3)
    v = V.float().repeat_interleave(G, dim=2).permute(0, 2, 1, 3)
    ref = torch.nn.functional.scaled_dot_product_attention(q, k, v).permute(0, 2, 1, 3)
    assert rel_l2(h64(O), h64(ref)) <= (1e-5 if wl.io_dtype == F32 else 1e-2)


@pytest.mark.parametrize("wl", EDGE_WL, ids=[w.name for w in EDGE_WL])
def test_values_one_give_one(wl):
    pair = Pair(wl)
    reqs = np.arange(wl.n_req)
    for b in range(3):
        K, _ = wk.prefix_kv(wl, b, pair.dev)
        pair.commit(K, torch.ones_like(K), reqs)
    Q, K, _ = wk.block_qkv(wl, "ones", pair.dev)
    got, want, O = pair.step(Q, K, torch.ones_like(K))
    assert np.max(np.abs(h64(O) - 1.0)) <= (1e-5 if wl.io_dtype == F32 else 4e-3)


@pytest.mark.parametrize("wl", EDGE_WL, ids=[w.name for w in EDGE_WL])
def test_tied_keys(wl):
    """All keys equal: the in-block softmax is uniform (every score ties)."""
    pair = Pair(wl)
    pair.build_prefixes(np.full(wl.n_req, wl.B))
    Q, K, V = wk.block_qkv(wl, "ties", pair.dev)
    K = K[:, :1].expand_as(K).contiguous()
    got, want, _ = pair.step(Q, K, V)
    assert_parity(got, want, wl.io_dtype, "tied keys", units="out")


# Sec. 3.1's two forms of the cross-block branch: the recurrent state (S, z) built by
# the CUDA commits and read by the CUDA step, against the oracle's token-by-token sum
# over the explicit prefix (lin_num = sum_t (phi(q) . phi(k_t)) v_t, Eq. 1's quadratic
# form with the Hedgehog map), which never forms a state
EQ1_WL = [(W_("eq1_gqa_bf16", BF16, 3, 8, 2, 128, 128, 32, 53), [0, 64, 160]),
          (W_("eq1_f256_g1_bf16", BF16, 3, 2, 2, 128, 256, 64, 54), [128, 0, 192])]


@pytest.mark.parametrize("wl,plen", EQ1_WL, ids=[w.name for w, _ in EQ1_WL])
def test_state_route_matches_quadratic_prefix_form(wl, plen):
    pair = Pair(wl, tracked=[])
    plen = np.asarray(plen)
    P_max = int(plen.max())
    Kp = torch.zeros((wl.n_req, max(P_max, 1), wl.Hkv, wl.d), dtype=wl.io_dtype)
    Vp = torch.zeros_like(Kp)
    for b in range(P_max // wl.B):
        reqs = np.nonzero(plen > b * wl.B)[0]
        K, V = wk.prefix_kv(wl, b, pair.dev)
        idx = torch.as_tensor(reqs, device=pair.dev)
        pair.commit(K[idx], V[idx], reqs)
        Kp[reqs, b * wl.B:(b + 1) * wl.B] = K[idx].cpu()
        Vp[reqs, b * wl.B:(b + 1) * wl.B] = V[idx].cpu()
    Q, K, V = wk.block_qkv(wl, "eq1", pair.dev)
    O = torch.empty_like(Q)
    H.hybrid_block_attn(pair.cfg, Q, K, V, pair.W, pair.alpha, pair.ptrs, wl.n_req, O)
    H.hybrid_check()
    want = pair.orc.block_attn_prefix(h64(Q), h64(K), h64(V), pair.W64, pair.alpha64, h64(Kp), h64(Vp), plen)
    assert_parity(h64(O), want, wl.io_dtype, "state route vs prefix form", units="out")


def test_permuted_and_subset_pointer_arrays():
    """A batch may list any subset of states in any order: the output of a
    request depends only on its own state pointer."""
    wl = W_("perm_bf16", BF16, 6, 8, 2, 128, 128, 32, 41)
    pair = Pair(wl)
    pair.build_prefixes(np.array([32, 64, 96, 128, 160, 192]))
    Q, K, V = wk.block_qkv(wl, "perm", pair.dev)
    O = torch.empty_like(Q)
    H.hybrid_block_attn(pair.cfg, Q, K, V, pair.W, pair.alpha, pair.ptrs, wl.n_req, O)
    order = [4, 1, 5]
    idx = torch.as_tensor(order, device=pair.dev)
    O2 = torch.empty_like(Q[idx])
    H.hybrid_block_attn(pair.cfg, Q[idx].contiguous(), K[idx].contiguous(), V[idx].contiguous(),
                        pair.W, pair.alpha, pair.pool.ptr_array(order), len(order), O2)
    H.hybrid_check()
    assert torch.equal(O[idx], O2)


def test_deterministic():
    wl = W_("det_bf16", BF16, 4, 16, 4, 128, 128, 32, 42)
    pair = Pair(wl)
    pair.build_prefixes(np.array([64, 32, 0, 96]))
    Q, K, V = wk.block_qkv(wl, "det", pair.dev)
    O1, O2 = torch.empty_like(Q), torch.empty_like(Q)
    H.hybrid_block_attn(pair.cfg, Q, K, V, pair.W, pair.alpha, pair.ptrs, wl.n_req, O1)
    H.hybrid_block_attn(pair.cfg, Q, K, V, pair.W, pair.alpha, pair.ptrs, wl.n_req, O2)
    H.hybrid_check()
    assert torch.equal(O1, O2)
    # commits are deterministic too: two pools, same commits, identical bytes
    pair2 = Pair(wl)
    pair2.build_prefixes(np.array([64, 32, 0, 96]))
    torch.cuda.synchronize()
    assert torch.equal(pair.pool.slab, pair2.pool.slab)


def test_state_copy_out_and_back_resumes():
    """The state is the resumable object: copying a state's bytes out and back
    (e.g. to host memory) gives identical subsequent outputs."""
    wl = W_("resume_bf16", BF16, 2, 4, 4, 128, 128, 32, 43)
    pair = Pair(wl)
    pair.build_prefixes(np.array([96, 64]))
    saved = pair.pool.slab.cpu().clone()
    Q, K, V = wk.block_qkv(wl, "resume", pair.dev)
    O1 = torch.empty_like(Q)
    H.hybrid_block_attn(pair.cfg, Q, K, V, pair.W, pair.alpha, pair.ptrs, wl.n_req, O1)
    pair.pool.slab.fill_(0.0)
    pair.pool.slab.copy_(saved.to(pair.dev))
    O2 = torch.empty_like(Q)
    H.hybrid_block_attn(pair.cfg, Q, K, V, pair.W, pair.alpha, pair.ptrs, wl.n_req, O2)
    H.hybrid_check()
    assert torch.equal(O1, O2)


def _u_ranges(wl, W, Q):
    """Per state head, the largest row range max_f u - min_f u of U = Q W_g."""
    G = wl.Hq // wl.Hkv
    q = Q.float().reshape(wl.n_req, wl.B, wl.Hkv, G, wl.d)
    U = torch.einsum("nbhgd,hdf->nbhgf", q, W.float().reshape(wl.Hkv, wl.d, wl.F))
    return (U.amax(-1) - U.amin(-1)).amax(dim=(0, 1, 3)).cpu().numpy()


@pytest.mark.parametrize("scaled_heads", [(), (0, 1), (1,)], ids=["from_phi_plus", "u_again", "mixed"])
def test_f256_phi_minus_paths(scaled_heads):
    """F = 256 step: phi- is derived from phi+ while every row of a unit has a range of
    U = Q W within 64, and U is formed again otherwise (W x 20 on the listed state
    heads); "mixed" runs both kinds of unit in one launch.  Both against the oracle."""
    wl = W_("f256_phi_minus", BF16, 4, 4, 2, 128, 256, 32, 37)
    pair = Pair(wl)
    if scaled_heads:
        W = pair.W.float()
        for g in scaled_heads:
            W[g] *= 20.0
        pair.W = W.to(pair.W.dtype)
        pair.W64 = h64(pair.W)
    pair.build_prefixes(np.array([32, 0, 96, 64]))
    Q, K, V = wk.block_qkv(wl, "phim", pair.dev)
    rng = _u_ranges(wl, pair.W, Q)
    for g in range(wl.Hkv):
        assert (rng[g] > 64.0) if g in scaled_heads else (rng[g] < 32.0), (g, rng)
    got, want, _ = pair.step(Q, K, V)
    assert_parity(got, want, wl.io_dtype, f"W x 20 on heads {scaled_heads}", units="out")
    pair.commit(K, V)
    S, z = pair.gpu_state()
    assert_parity(S, pair.S, wl.io_dtype, "state after the commit", units="state")
    Q2, K2, V2 = wk.block_qkv(wl, "phim2", pair.dev)
    got, want, _ = pair.step(Q2, K2, V2)
    assert_parity(got, want, wl.io_dtype, "second step", units="out")


BADPTR_WL = [W_("badptr_bf16", BF16, 3, 4, 4, 128, 128, 32, 44),
             W_("badptr_f256", BF16, 3, 2, 2, 128, 256, 64, 45)]


@pytest.mark.parametrize("wl", BADPTR_WL, ids=[w.name for w in BADPTR_WL])
def test_bad_state_pointer_is_reported_not_faulted(wl):
    """A null or misaligned entry in d_state_ptrs is skipped on the device and
    reported by hybrid_check; the context stays usable."""
    pair = Pair(wl)
    Q, K, V = wk.block_qkv(wl, "bad", pair.dev)
    good = pair.pool.ptr_array([0, 1, 2])
    for bad_value in (0, pair.pool.slot_ptr(1) + 4):
        ptrs = good.clone()
        ptrs[1] = bad_value
        O = torch.zeros_like(Q)
        H.hybrid_block_attn(pair.cfg, Q, K, V, pair.W, pair.alpha, ptrs, 3, O)
        assert H.hybrid_check(check=False) == H.HYBRID_ERR_DEVICE
        H.hybrid_commit_block(pair.cfg, K, V, wl.B, pair.W, ptrs, 3)
        assert H.hybrid_check(check=False) == H.HYBRID_ERR_DEVICE
    # the error word was cleared and the device still works
    O = torch.empty_like(Q)
    H.hybrid_block_attn(pair.cfg, Q, K, V, pair.W, pair.alpha, good, 3, O)
    assert H.hybrid_check(check=False) == H.HYBRID_OK


# More units than SMs, so the persistent kernels take two or three units per CTA:
# request 0's units end one CTA's range and request 1's start it (bad-then-good and
# good-then-bad inside one CTA's run)
BADRUN_WL = [W_("badrun_c3_shape", BF16, 80, 8, 4, 128, 128, 32, 51),
             W_("badrun_f256_g1", BF16, 60, 3, 3, 128, 256, 64, 52)]


@pytest.mark.parametrize("wl", BADRUN_WL, ids=[w.name for w in BADRUN_WL])
def test_bad_state_pointer_inside_a_run_of_units(wl):
    """A request whose state pointer is unusable is skipped inside a CTA's run of
    units: the error is reported, its output rows are left as they were, and every
    other request's output (and, for the fused step + commit, its committed state)
    is the oracle's."""
    tracked = [0, 1, 2, 3, wl.n_req - 1]
    pair = Pair(wl, tracked=tracked)
    pair.build_prefixes(np.full(wl.n_req, 2 * wl.B))
    Q, K, V = wk.block_qkv(wl, "badrun", pair.dev)
    t = torch.as_tensor(tracked, device=pair.dev)
    want = pair.orc.block_attn(h64(Q[t]), h64(K[t]), h64(V[t]), pair.W64, pair.alpha64, pair.S, pair.z)
    for bad in (0, 1):
        keep = [i for i, r in enumerate(tracked) if r != bad]
        ptrs = pair.ptrs.clone()
        ptrs[bad] = 0
        O = torch.full_like(Q, 7.0)
        H.hybrid_block_attn(pair.cfg, Q, K, V, pair.W, pair.alpha, ptrs, wl.n_req, O)
        assert H.hybrid_check(check=False) == H.HYBRID_ERR_DEVICE
        assert torch.all(O[bad] == 7.0), "the skipped request's output was written"
        assert_parity(h64(O[t])[keep], want[keep], wl.io_dtype, f"step, request {bad} skipped", units="out")
    if wl.B != 32:
        return
    # step + commit on the same batch with request 1 skipped (the fused kernel)
    bad = 1
    keep = [i for i, r in enumerate(tracked) if r != bad]
    ptrs = pair.ptrs.clone()
    ptrs[bad] = 0
    O = torch.full_like(Q, 7.0)
    H.hybrid_block_attn_commit(pair.cfg, Q, K, V, pair.W, pair.alpha, ptrs, wl.n_req, O)
    assert H.hybrid_check(check=False) == H.HYBRID_ERR_DEVICE
    assert torch.all(O[bad] == 7.0), "the skipped request's output was written"
    assert_parity(h64(O[t])[keep], want[keep], wl.io_dtype, "step + commit, request 1 skipped", units="out")
    tk = torch.as_tensor([tracked[i] for i in keep], device=pair.dev)
    S_want, z_want = pair.S[keep].copy(), pair.z[keep].copy()
    pair.orc.commit(h64(K[tk]), h64(V[tk]), pair.W64, S_want, z_want)
    S_got, z_got = pair.gpu_state([tracked[i] for i in keep])
    assert_parity(S_got, S_want, wl.io_dtype, "state after step + commit", units="state")
    S_bad, _ = pair.gpu_state([bad])
    assert_parity(S_bad, pair.S[[tracked.index(bad)]], wl.io_dtype, "skipped request's state", units="state")


def test_bounded_wait_timeout_is_reported_not_hung():
    """A bounded device wait that runs out comes back as HYBRID_ERR_TIMEOUT from
    hybrid_check, with the context usable.  The hook arms one step launch with a
    1 ms limit and makes its math warps withhold one arrival on a barrier that no
    asynchronous copy targets; every role then leaves through the failure path.
    Two units per CTA on some CTAs (160 units on at most 152 CTAs) and one on the
    rest, so both a unit's own wait and the next unit's start meet the flag."""
    wl = W_("timeout_c3_shape", BF16, 40, 16, 4, 128, 128, 32, 50)
    pair = Pair(wl)
    pair.build_prefixes(np.full(wl.n_req, 64))
    Q, K, V = wk.block_qkv(wl, "timeout", pair.dev)
    O = torch.zeros_like(Q)
    H.hybrid_debug_arm_wait_timeout(1_000_000)
    H.hybrid_block_attn(pair.cfg, Q, K, V, pair.W, pair.alpha, pair.ptrs, wl.n_req, O)
    assert H.hybrid_check(check=False) == H.HYBRID_ERR_TIMEOUT
    # the launch consumed the setting: the next one runs normally and is correct
    got, want, _ = pair.step(Q, K, V)
    assert H.hybrid_check(check=False) == H.HYBRID_OK
    assert_parity(got, want, wl.io_dtype, "after a timed-out launch", units="out")
    # disarming leaves later launches alone
    H.hybrid_debug_arm_wait_timeout(1_000_000)
    H.hybrid_debug_arm_wait_timeout(0)
    got, want, _ = pair.step(Q, K, V)
    assert_parity(got, want, wl.io_dtype, "after disarming", units="out")


PREFILL = [
    # 6 units x 8 chunks: every unit's chunks are spread over 8 CTAs and combined
    # by the reduce-adds, on top of a prefix already in the state
    (W_("prefill_split_runs", BF16, 3, 4, 2, 128, 128, 32, 46), 1000, 64),
    # 80 units x 3 chunks on 152 CTAs: ranges cross unit boundaries; 44-token tail
    (W_("prefill_cross_units", BF16, 20, 8, 4, 128, 128, 32, 47), 300, 0),
    # d = F = 64, a one-token last chunk
    (W_("prefill_d64_f64", BF16, 4, 4, 4, 64, 64, 32, 48), 257, 32),
    # F = 256: six chunks per sign pass, a one-token tail
    (W_("prefill_f256", BF16, 3, 2, 2, 128, 256, 32, 49), 161, 64),
]


@pytest.mark.parametrize("wl,T,prefix", PREFILL, ids=[w.name for w, _, _ in PREFILL])
def test_prefill_split_across_ctas(wl, T, prefix):
    """Long prompt prefills (hybrid_commit_block with n_tok = T) against the
    oracle, the state holding an earlier prefix of `prefix` tokens."""
    pair = Pair(wl)
    if prefix:
        pair.build_prefixes(np.full(wl.n_req, prefix, dtype=np.int64))
    K, V = wk.prefix_kv(wl, 1, pair.dev, n_tok=T)
    pair.commit(K, V)
    S, z = pair.gpu_state()
    assert_parity(S, pair.S, BF16, f"prefill {T} S", units="state")
    assert_parity(z, pair.z, BF16, f"prefill {T} z", units="state")


RAGGED = [
    # token-major prefill kernel: long and empty prompts, tails of 1 and 1 + 128 tokens
    (W_("ragged_prefill", BF16, 7, 4, 2, 128, 128, 32, 61), [300, 0, 129, 1, 1000, 64, 257], 64),
    # per-unit reduction kernel: every prompt at most 64 tokens
    (W_("ragged_short", BF16, 5, 4, 4, 128, 64, 32, 62), [32, 0, 17, 64, 1], 0),
    # F = 256: one pass per sign, a prompt longer than a block
    (W_("ragged_f256", BF16, 3, 2, 2, 128, 256, 64, 63), [100, 0, 33], 64),
    # float32: the FMA kernel once per request
    (W_("ragged_f32", F32, 3, 2, 1, 64, 32, 16, 64), [20, 0, 7], 16),
]


def _ragged_commit(pair, lens, tag):
    """hybrid_commit_ragged on packed K, V; the oracle folds each tracked request's
    own tokens alone."""
    wl = pair.wl
    lens = np.asarray(lens, dtype=np.int64)
    offs = np.concatenate([[0], np.cumsum(lens)])
    K, V = wk.prefix_kv(wl, tag, pair.dev, n_req=1, n_tok=int(offs[-1]))
    Kp, Vp = K[0].contiguous(), V[0].contiguous()
    H.hybrid_commit_ragged(pair.cfg, Kp, Vp, offs.tolist(), pair.W, pair.ptrs, wl.n_req)
    H.hybrid_check()
    for i, r in enumerate(pair.tracked):
        if lens[r] == 0:
            continue
        a, b = int(offs[r]), int(offs[r + 1])
        Sx, zx = pair.S[i:i + 1].copy(), pair.z[i:i + 1].copy()
        pair.orc.commit(h64(Kp[a:b][None]), h64(Vp[a:b][None]), pair.W64, Sx, zx)
        pair.S[i:i + 1], pair.z[i:i + 1] = Sx, zx


@pytest.mark.parametrize("wl,lens,prefix", RAGGED, ids=[w.name for w, _, _ in RAGGED])
def test_ragged_prefill(wl, lens, prefix):
    """Prompts of different lengths in one hybrid_commit_ragged call, on top of a
    prefix already in the state; an empty prompt leaves its state unchanged."""
    pair = Pair(wl)
    if prefix:
        pair.build_prefixes(np.full(wl.n_req, prefix, dtype=np.int64))
    _ragged_commit(pair, lens, 71)
    S, z = pair.gpu_state()
    assert_parity(S, pair.S, wl.io_dtype, "ragged prefill S", units="state")
    assert_parity(z, pair.z, wl.io_dtype, "ragged prefill z", units="state")


def test_ragged_prefill_more_requests_than_one_launch():
    """2100 requests of 0-3 tokens: two launches of at most 2048 requests, offsets
    rebased for the second; the requests on both sides of the split are checked."""
    wl = W_("ragged_many", BF16, 2100, 2, 1, 64, 64, 32, 65)
    pair = Pair(wl, tracked=[0, 1, 3, 2046, 2047, 2048, 2049, 2099])
    lens = np.arange(wl.n_req) % 4
    _ragged_commit(pair, lens, 72)
    S, z = pair.gpu_state()
    assert_parity(S, pair.S, wl.io_dtype, "ragged S", units="state")
    assert_parity(z, pair.z, wl.io_dtype, "ragged z", units="state")


def test_prefill_commit_long_ragged():
    """Prompt prefill: commits of many tokens (T not a multiple of 32) in one call
    equal the same tokens committed in B-sized pieces."""
    wl = W_("prefill_bf16", BF16, 3, 4, 2, 128, 64, 32, 45)
    pair = Pair(wl)
    K, V = wk.prefix_kv(wl, 0, pair.dev, n_tok=161)
    pair.commit(K, V)
    S, z = pair.gpu_state()
    assert_parity(S, pair.S, BF16, "prefill S", units="state")
    assert_parity(z, pair.z, BF16, "prefill z", units="state")


# ---------------------------------------------------------------------------
# fused step + commit (hybrid_block_attn_commit)
# ---------------------------------------------------------------------------
FUSED = [
    (W_("fused_gqa4", BF16, 5, 8, 2, 128, 128, 32, 51), [0, 32, 96, 160, 256]),
    (W_("fused_mha_d64_f64", BF16, 3, 4, 4, 64, 64, 32, 52), [64, 0, 32]),
    (W_("fused_gqa4_many_units", BF16, 40, 16, 4, 128, 128, 32, 53), None),   # 160 units > 152 SMs
    (W_("fused_b16_fallback", BF16, 3, 4, 2, 128, 128, 16, 54), [16, 0, 48]),  # B != 32: step + commit
    # keys x24: scores near 60 make some warps take the exact phi+ rescale
    (W_("fused_gqa4_k24", BF16, 3, 8, 2, 128, 128, 32, 56, k_scale=24.0), [32, 0, 96]),
    # F = 64: one 32-feature chunk per part, the output takes the whole second half
    (W_("fused_d128_f64", BF16, 4, 8, 4, 128, 64, 32, 57), [0, 64, 32, 96]),
    # d = 64, F = 128: a ring longer than a unit; 192 units, two or more per CTA
    (W_("fused_d64_f128_many", BF16, 48, 16, 4, 64, 128, 32, 58), None),
    # F = 256: the step, then the commit, from one call
    (W_("fused_f256_step_then_commit", BF16, 3, 4, 2, 128, 256, 32, 59), [32, 0, 64]),
]


@pytest.mark.parametrize("wl,plen", FUSED, ids=[w.name for w, _ in FUSED])
def test_fused_step_commit_parity(wl, plen):
    pair = Pair(wl)
    plen = (np.arange(wl.n_req) % 5) * wl.B if plen is None else np.asarray(plen, dtype=np.int64)
    pair.build_prefixes(plen)
    for step in range(3):   # three consecutive committing steps
        Q, K, V = wk.block_qkv(wl, ("fused", step), pair.dev)
        O = torch.empty_like(Q)
        H.hybrid_block_attn_commit(pair.cfg, Q, K, V, pair.W, pair.alpha, pair.ptrs, wl.n_req, O)
        H.hybrid_check()
        t = torch.as_tensor(pair.tracked, device=Q.device)
        want = pair.orc.block_attn(h64(Q[t]), h64(K[t]), h64(V[t]), pair.W64, pair.alpha64,
                                   pair.S, pair.z)
        assert_parity(h64(O[t]), want, wl.io_dtype, f"fused output, step {step}", units="out")
        pair.orc.commit(h64(K[t]), h64(V[t]), pair.W64, pair.S, pair.z)
        S, z = pair.gpu_state()
        assert_parity(S, pair.S, wl.io_dtype, f"fused state S, step {step}", units="state")
        assert_parity(z, pair.z, wl.io_dtype, f"fused state z, step {step}", units="state")


def test_fused_matches_separate_calls():
    """hybrid_block_attn_commit equals hybrid_block_attn then hybrid_commit_block
    (both within the bf16 tolerance of each other)."""
    wl = W_("fused_vs_separate", BF16, 6, 16, 4, 128, 128, 32, 55)
    a, b = Pair(wl), Pair(wl)
    plen = np.array([32, 64, 0, 128, 96, 32])
    a.build_prefixes(plen)
    b.build_prefixes(plen)
    Q, K, V = wk.block_qkv(wl, "fvs", a.dev)
    O1, O2 = torch.empty_like(Q), torch.empty_like(Q)
    H.hybrid_block_attn_commit(a.cfg, Q, K, V, a.W, a.alpha, a.ptrs, wl.n_req, O1)
    H.hybrid_block_attn(b.cfg, Q, K, V, b.W, b.alpha, b.ptrs, wl.n_req, O2)
    H.hybrid_commit_block(b.cfg, K, V, wl.B, b.W, b.ptrs, wl.n_req)
    H.hybrid_check()
    assert rel_l2(h64(O1), h64(O2)) <= 1e-2
    Sa, za = a.gpu_state()
    Sb, zb = b.gpu_state()
    assert rel_l2(Sa, Sb) <= 1e-3 and rel_l2(za, zb) <= 1e-4
