"""Pins that tie the fp64 oracle to facts fixed by the paper and by mathematics,
not to the oracle itself.

Each ``pin_*`` function takes a loaded :class:`oracle.Oracle` and raises
``AssertionError`` if the oracle disagrees with:
  * hand-derived worked examples (``tests/golden/hand_derived.json``),
  * an independent library routine (torch's scaled_dot_product_attention in
    fp64, scipy's softmax),
  * closed forms and invariants of Section 3.1 / Eq. 1.

The functions are plain so that ``test_oracle_mutants.py`` can run all of them
against deliberately broken builds of the oracle in a subprocess and check
that every planted mistake trips at least one pin.

Run as a script: ``python tests/oracle_pins.py <liboracle.so>`` prints one line
per failing pin and exits 0.
"""
from __future__ import annotations

import json
import math
import os
import sys

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

from oracle import PHI_HEDGEHOG, PHI_IDENTITY, Oracle  # noqa: E402

GOLDEN = os.path.join(HERE, "golden", "hand_derived.json")


def _golden():
    with open(GOLDEN) as fh:
        return json.load(fh)


def _rng(seed):
    return np.random.default_rng(seed)


def _close(a, b, rtol=1e-12, atol=1e-12, what=""):
    a = np.asarray(a, dtype=np.float64)
    b = np.asarray(b, dtype=np.float64)
    assert a.shape == b.shape, f"{what}: shape {a.shape} vs {b.shape}"
    err = np.abs(a - b)
    tol = atol + rtol * np.abs(b)
    assert np.all(err <= tol), f"{what}: max abs err {err.max():.3e}"


def _random_problem(rng, n_req=2, B=3, Hq=2, Hkv=1, d=4, F=3, P_max=5, w_std=None,
                    prefix_len=None, k_scale=1.0):
    Q = rng.standard_normal((n_req, B, Hq, d))
    K = rng.standard_normal((n_req, B, Hkv, d)) * k_scale
    V = rng.standard_normal((n_req, B, Hkv, d))
    W = rng.standard_normal((Hkv, d, F)) * (w_std if w_std is not None else 1.0 / math.sqrt(d))
    alpha = rng.uniform(0.0, 1.0, size=Hq)
    Kp = rng.standard_normal((n_req, P_max, Hkv, d)) * k_scale
    Vp = rng.standard_normal((n_req, P_max, Hkv, d))
    if prefix_len is None:
        prefix_len = rng.integers(0, P_max + 1, size=n_req)
    return dict(Q=Q, K=K, V=V, W=W, alpha=alpha, Kp=Kp, Vp=Vp,
                prefix_len=np.asarray(prefix_len, dtype=np.int32))


def _state_from_prefix(orc, p, phi_kind=PHI_HEDGEHOG):
    """Build (S, z) with the oracle's commit, one request at a time (ragged)."""
    n_req, P_max, Hkv, d = p["Kp"].shape
    F = p["W"].shape[2]
    S, z = orc.empty_state(n_req, Hkv, d, F, phi_kind)
    for r in range(n_req):
        P = int(p["prefix_len"][r])
        Sr, zr = S[r:r + 1].copy(), z[r:r + 1].copy()
        orc.commit(p["Kp"][r:r + 1, :P], p["Vp"][r:r + 1, :P], p["W"], Sr, zr, phi_kind=phi_kind)
        S[r], z[r] = Sr[0], zr[0]
    return S, z


def _sdpa(Q, K, V):
    """Exact bidirectional softmax attention over the active block (library routine)."""
    import torch
    n_req, B, Hq, d = Q.shape
    G = Hq // K.shape[2]
    q = torch.from_numpy(Q).permute(0, 2, 1, 3)
    k = torch.from_numpy(np.repeat(K, G, axis=2)).permute(0, 2, 1, 3)
    v = torch.from_numpy(np.repeat(V, G, axis=2)).permute(0, 2, 1, 3)
    o = torch.nn.functional.scaled_dot_product_attention(q, k, v)
    return o.permute(0, 2, 1, 3).contiguous().numpy()


# ---------------------------------------------------------------------------
# hand-derived worked examples
# ---------------------------------------------------------------------------
def pin_golden_phi(orc):
    g = _golden()
    c = g["phi_w_layout"]
    X = np.array(c["x"]).reshape(1, 1, c["d"])
    W = np.array(c["W"]).reshape(1, c["d"], c["F"])
    _close(orc.feature_map(X, W)[0, 0], c["phi"], what="phi_w_layout")
    c = g["phi_sign_swap"]
    W = np.array(c["W"]).reshape(1, c["d"], c["F"])
    for x, phi in zip(c["x_list"], c["phi_list"]):
        _close(orc.feature_map(np.array(x).reshape(1, 1, c["d"]), W)[0, 0], phi, what="phi_sign_swap")


def pin_golden_commit(orc):
    c = _golden()["commit_two_tokens"]
    d, F = c["d"], c["F"]
    W = np.array(c["W"]).reshape(1, d, F)
    K = np.array(c["K"]).reshape(1, 2, 1, d)
    V = np.array(c["V"]).reshape(1, 2, 1, d)
    S, z = orc.empty_state(1, 1, d, F)
    orc.commit(K, V, W, S, z)
    _close(S[0, 0], c["S"], what="commit S")
    _close(z[0, 0], c["z"], what="commit z")
    # the same two tokens committed one at a time
    S2, z2 = orc.empty_state(1, 1, d, F)
    orc.commit(K[:, :1], V[:, :1], W, S2, z2)
    orc.commit(K[:, 1:], V[:, 1:], W, S2, z2)
    _close(S2[0, 0], c["S"], what="commit S, two calls")


def pin_golden_merge(orc):
    c = _golden()["merge_gate_d1"]
    W = np.array(c["W"]).reshape(1, 1, 1)
    Q = np.array(c["q"]).reshape(1, 2, 1, 1)
    K = np.array(c["k"]).reshape(1, 2, 1, 1)
    V = np.array(c["v"]).reshape(1, 2, 1, 1)
    Kp = np.array(c["k_prefix"]).reshape(1, 1, 1, 1)
    Vp = np.array(c["v_prefix"]).reshape(1, 1, 1, 1)
    S, z = orc.empty_state(1, 1, 1, 1)
    orc.commit(Kp, Vp, W, S, z)
    for alpha, want in zip(c["alpha_list"], c["out_list"]):
        a = np.array([alpha])
        O1 = orc.block_attn(Q, K, V, W, a, S, z)
        O2 = orc.block_attn_prefix(Q, K, V, W, a, Kp, Vp, [1])
        _close(O1.ravel(), [want, want], what=f"merge route 1 alpha={alpha}")
        _close(O2.ravel(), [want, want], what=f"merge route 2 alpha={alpha}")


def pin_golden_scale(orc):
    c = _golden()["softmax_scale_d4"]
    d, F = c["d"], c["F"]
    W = np.zeros((1, d, F))
    Q = np.array(c["q"]).reshape(1, 2, 1, d)
    K = np.array(c["k"]).reshape(1, 2, 1, d)
    V = np.array(c["v"]).reshape(1, 2, 1, d)
    S, z = orc.empty_state(1, 1, d, F)
    O = orc.block_attn(Q, K, V, W, np.array([0.3]), S, z)
    _close(O[0, :, 0], c["out"], what="softmax scale")


# ---------------------------------------------------------------------------
# independent library routines
# ---------------------------------------------------------------------------
def pin_phi_vs_scipy(orc):
    from scipy.special import softmax
    rng = _rng(11)
    for (n, H, Hkv, d, F) in [(5, 4, 2, 8, 6), (3, 2, 2, 16, 16), (4, 3, 1, 5, 7)]:
        X = rng.standard_normal((n, H, d)) * 2.0
        W = rng.standard_normal((Hkv, d, F))
        Phi = orc.feature_map(X, W)
        G = H // Hkv
        for h in range(H):
            U = X[:, h, :] @ W[h // G]
            want = np.concatenate([softmax(U, axis=1), softmax(-U, axis=1)], axis=1)
            _close(Phi[:, h, :], want, rtol=1e-13, atol=1e-15, what="phi vs scipy")


def pin_empty_prefix_is_softmax(orc):
    rng = _rng(12)
    for (n_req, B, Hq, Hkv, d, F) in [(2, 5, 4, 2, 8, 4), (1, 16, 2, 2, 16, 8), (3, 3, 3, 1, 4, 2)]:
        p = _random_problem(rng, n_req, B, Hq, Hkv, d, F, P_max=0, prefix_len=[0] * n_req)
        S, z = orc.empty_state(n_req, Hkv, d, F)
        for alpha in (p["alpha"], np.full(Hq, -3.0), np.full(Hq, math.inf)):
            O = orc.block_attn(p["Q"], p["K"], p["V"], p["W"], alpha, S, z)
            _close(O, _sdpa(p["Q"], p["K"], p["V"]), rtol=1e-11, atol=1e-12, what="empty prefix")


# ---------------------------------------------------------------------------
# closed forms and invariants
# ---------------------------------------------------------------------------
def pin_phi_invariants(orc):
    rng = _rng(13)
    X = rng.standard_normal((7, 2, 6)) * 3.0
    W = rng.standard_normal((2, 6, 5))
    Phi = orc.feature_map(X, W)
    F = 5
    assert np.all(Phi > 0), "phi must be positive"
    _close(Phi[..., :F].sum(-1), np.ones((7, 2)), what="softmax(xW) sums to 1")
    _close(Phi[..., F:].sum(-1), np.ones((7, 2)), what="softmax(-xW) sums to 1")
    Phi_neg = orc.feature_map(-X, W)
    _close(Phi_neg[..., :F], Phi[..., F:], what="phi(-x) swaps halves")
    _close(Phi_neg[..., F:], Phi[..., :F], what="phi(-x) swaps halves")
    Z = orc.feature_map(X, np.zeros_like(W))
    _close(Z, np.full_like(Z, 1.0 / F), what="W = 0 gives phi = 1/F")


def pin_w_zero_closed_form(orc):
    """W = 0: phi = 1/F everywhere, so phi(q).phi(k) = 2/F and
    out = (w sum_j a_j v_j + (2/F) sum_t v_t) / (w sum_j a_j + 2P/F)."""
    rng = _rng(14)
    n_req, B, Hq, Hkv, d, F, P_max = 3, 4, 4, 2, 8, 6, 7
    p = _random_problem(rng, n_req, B, Hq, Hkv, d, F, P_max, prefix_len=[0, 3, 7])
    p["W"] = np.zeros_like(p["W"])
    p["alpha"] = np.array([-1.0, 0.0, 0.7, 2.5])
    S, z = _state_from_prefix(orc, p)
    O = orc.block_attn(p["Q"], p["K"], p["V"], p["W"], p["alpha"], S, z)
    G = Hq // Hkv
    want = np.zeros_like(O)
    for r in range(n_req):
        P = int(p["prefix_len"][r])
        for h in range(Hq):
            g = h // G
            w = 1.0 / (1.0 + math.exp(-p["alpha"][h]))
            A = np.exp(p["Q"][r, :, h] @ p["K"][r, :, g].T / math.sqrt(d))    # [B, B]
            vsum = p["Vp"][r, :P, g].sum(0)
            want[r, :, h] = (w * (A @ p["V"][r, :, g]) + (2.0 / F) * vsum) / \
                            (w * A.sum(1, keepdims=True) + 2.0 * P / F)
    _close(O, want, rtol=1e-11, atol=1e-12, what="W=0 closed form")


def pin_identity_phi_no_gate_is_eq1(orc):
    """Identity feature map, w = 0 (alpha = -inf): out = sum_t (q.k_t) v_t / sum_t q.k_t (Eq. 1)."""
    rng = _rng(15)
    n_req, B, Hq, Hkv, d, P_max = 2, 3, 2, 1, 5, 6
    Q = rng.uniform(0.0, 1.0, (n_req, B, Hq, d))
    K = rng.uniform(0.0, 1.0, (n_req, B, Hkv, d))
    V = rng.standard_normal((n_req, B, Hkv, d))
    Kp = rng.uniform(0.0, 1.0, (n_req, P_max, Hkv, d))
    Vp = rng.standard_normal((n_req, P_max, Hkv, d))
    plen = [6, 4]
    alpha = np.full(Hq, -math.inf)
    S = np.zeros((n_req, Hkv, d, d))
    z = np.zeros((n_req, Hkv, d))
    for r in range(n_req):
        Sr, zr = S[r:r + 1].copy(), z[r:r + 1].copy()
        orc.commit(Kp[r:r + 1, :plen[r]], Vp[r:r + 1, :plen[r]], None, Sr, zr, phi_kind=PHI_IDENTITY)
        S[r], z[r] = Sr[0], zr[0]
    O1 = orc.block_attn(Q, K, V, None, alpha, S, z, phi_kind=PHI_IDENTITY)
    O2 = orc.block_attn_prefix(Q, K, V, None, alpha, Kp, Vp, plen, phi_kind=PHI_IDENTITY)
    want = np.zeros_like(O1)
    for r in range(n_req):
        for h in range(Hq):
            kern = Q[r, :, h] @ Kp[r, :plen[r], h // (Hq // Hkv)].T     # [B, P]
            want[r, :, h] = (kern @ Vp[r, :plen[r], h // (Hq // Hkv)]) / kern.sum(1, keepdims=True)
    _close(O1, want, rtol=1e-11, atol=1e-12, what="identity phi, state route")
    _close(O2, want, rtol=1e-11, atol=1e-12, what="identity phi, prefix route")


def pin_values_one_give_one(orc):
    """V = 1 in the block and the prefix: the shared normaliser gives out = 1 exactly."""
    rng = _rng(16)
    p = _random_problem(rng, 3, 5, 4, 2, 6, 4, 9, prefix_len=[0, 4, 9])
    p["V"] = np.ones_like(p["V"])
    p["Vp"] = np.ones_like(p["Vp"])
    S, z = _state_from_prefix(orc, p)
    O = orc.block_attn(p["Q"], p["K"], p["V"], p["W"], p["alpha"], S, z)
    _close(O, np.ones_like(O), rtol=1e-12, atol=1e-12, what="V = 1")


def pin_affine_in_values(orc):
    """out(c V + b 1) = c out(V) + b (attention weights do not depend on V)."""
    rng = _rng(17)
    p = _random_problem(rng, 2, 4, 2, 2, 6, 3, 8, prefix_len=[5, 8])
    S, z = _state_from_prefix(orc, p)
    O = orc.block_attn(p["Q"], p["K"], p["V"], p["W"], p["alpha"], S, z)
    c, b = -2.5, 0.75
    q = dict(p)
    q["V"] = c * p["V"] + b
    q["Vp"] = c * p["Vp"] + b
    S2, z2 = _state_from_prefix(orc, q)
    O2 = orc.block_attn(q["Q"], q["K"], q["V"], q["W"], q["alpha"], S2, z2)
    _close(O2, c * O + b, rtol=1e-11, atol=1e-11, what="affine in V")


def pin_routes_agree_exhaustive(orc):
    """State route (S, z built block by block) equals the explicit prefix sum,
    over tiny shapes: B in {1,2,3}, prefix of 0, 1 or 3 blocks, d in {4,8},
    F in {2,4}, GQA group 1 or 2, and the gate at -inf, finite and +inf."""
    rng = _rng(18)
    for B in (1, 2, 3):
        for n_blocks in (0, 1, 3):
            for d in (4, 8):
                for F in (2, 4):
                    for (Hq, Hkv) in ((1, 1), (2, 1), (4, 2)):
                        P = n_blocks * B
                        p = _random_problem(rng, 2, B, Hq, Hkv, d, F, max(P, 1), prefix_len=[P, P])
                        S, z = orc.empty_state(2, Hkv, d, F)
                        for blk in range(n_blocks):      # commit block by block
                            sl = slice(blk * B, (blk + 1) * B)
                            orc.commit(p["Kp"][:, sl], p["Vp"][:, sl], p["W"], S, z)
                        alphas = [p["alpha"], np.full(Hq, math.inf)]
                        if P > 0:
                            alphas.append(np.full(Hq, -math.inf))
                        for alpha in alphas:
                            O1 = orc.block_attn(p["Q"], p["K"], p["V"], p["W"], alpha, S, z)
                            O2 = orc.block_attn_prefix(p["Q"], p["K"], p["V"], p["W"], alpha,
                                                       p["Kp"], p["Vp"], p["prefix_len"])
                            _close(O1, O2, rtol=1e-11, atol=1e-12,
                                   what=f"routes B={B} blocks={n_blocks} d={d} F={F} Hq={Hq}")


def pin_state_is_explicit_sum(orc):
    """S = sum_t phi(k_t) v_t^T and z = sum_t phi(k_t), with phi taken from the
    feature map on its own, and commits associative across calls."""
    rng = _rng(19)
    n_req, T, Hkv, d, F = 2, 7, 3, 5, 4
    K = rng.standard_normal((n_req, T, Hkv, d))
    V = rng.standard_normal((n_req, T, Hkv, d))
    W = rng.standard_normal((Hkv, d, F)) / math.sqrt(d)
    S, z = orc.empty_state(n_req, Hkv, d, F)
    orc.commit(K, V, W, S, z)
    Phi = orc.feature_map(K.reshape(n_req * T, Hkv, d), W).reshape(n_req, T, Hkv, 2 * F)
    want_S = np.einsum("rtgf,rtge->rgfe", Phi, V)
    want_z = Phi.sum(1)
    _close(S, want_S, what="S explicit sum")
    _close(z, want_z, what="z explicit sum")
    S2, z2 = orc.empty_state(n_req, Hkv, d, F)
    for (a, b) in ((0, 3), (3, 4), (4, 7)):
        orc.commit(K[:, a:b], V[:, a:b], W, S2, z2)
    _close(S2, S, what="commit associativity")
    _close(z2, z, what="commit associativity (z)")


def pin_permutations(orc):
    """Permuting the active block permutes the outputs (no in-block mask);
    permuting the prefix leaves the output unchanged."""
    rng = _rng(20)
    p = _random_problem(rng, 2, 6, 2, 1, 4, 3, 6, prefix_len=[6, 2])
    O = orc.block_attn_prefix(p["Q"], p["K"], p["V"], p["W"], p["alpha"], p["Kp"], p["Vp"],
                              p["prefix_len"])
    perm = rng.permutation(6)
    Op = orc.block_attn_prefix(p["Q"][:, perm], p["K"][:, perm], p["V"][:, perm], p["W"],
                               p["alpha"], p["Kp"], p["Vp"], p["prefix_len"])
    _close(Op, O[:, perm], what="block permutation")
    S, z = _state_from_prefix(orc, p)
    q = dict(p)
    q["Kp"] = p["Kp"][:, ::-1].copy()
    q["Vp"] = p["Vp"][:, ::-1].copy()
    q["prefix_len"] = np.array([6, 6], dtype=np.int32)      # request 0: full prefix reversed
    S2, z2 = _state_from_prefix(orc, q)
    _close(S2[0], S[0], rtol=1e-12, atol=1e-13, what="prefix permutation (state)")
    _close(z2[0], z[0], rtol=1e-12, atol=1e-13, what="prefix permutation (z)")


def pin_gqa_grouping(orc):
    """Query heads of one group share the state and W: identical q and alpha
    within a group give identical outputs; heads of different groups read
    different states."""
    rng = _rng(21)
    n_req, B, Hq, Hkv, d, F = 2, 3, 4, 2, 6, 3
    p = _random_problem(rng, n_req, B, Hq, Hkv, d, F, 5, prefix_len=[5, 3])
    p["Q"][:, :, 1] = p["Q"][:, :, 0]
    p["Q"][:, :, 3] = p["Q"][:, :, 2]
    p["alpha"][1] = p["alpha"][0]
    p["alpha"][3] = p["alpha"][2]
    S, z = _state_from_prefix(orc, p)
    O = orc.block_attn(p["Q"], p["K"], p["V"], p["W"], p["alpha"], S, z)
    _close(O[:, :, 1], O[:, :, 0], rtol=0, atol=0, what="GQA group 0")
    _close(O[:, :, 3], O[:, :, 2], rtol=0, atol=0, what="GQA group 1")
    # head 2 uses kv head 1: equal to a single-head problem on kv head 1
    single = {k: v for k, v in p.items()}
    O1 = orc.block_attn(p["Q"][:, :, 2:3], p["K"][:, :, 1:2], p["V"][:, :, 1:2], p["W"][1:2],
                        p["alpha"][2:3], S[:, 1:2].copy(), z[:, 1:2].copy())
    _close(O[:, :, 2:3], O1, rtol=0, atol=0, what="GQA head->state mapping")
    del single


def pin_gate_limits(orc):
    """alpha -> +inf gives w = 1; alpha -> -inf gives w = 0 (linear branch only,
    i.e. phi-kernel attention over the prefix as in Eq. 1)."""
    rng = _rng(22)
    p = _random_problem(rng, 2, 4, 2, 2, 6, 3, 6, prefix_len=[6, 1])
    S, z = _state_from_prefix(orc, p)
    O_inf = orc.block_attn(p["Q"], p["K"], p["V"], p["W"], np.full(2, math.inf), S, z)
    O_big = orc.block_attn(p["Q"], p["K"], p["V"], p["W"], np.full(2, 40.0), S, z)
    _close(O_inf, O_big, rtol=1e-12, atol=1e-12, what="alpha=+inf vs 40")
    O_neg = orc.block_attn(p["Q"], p["K"], p["V"], p["W"], np.full(2, -math.inf), S, z)
    Phi_q = orc.feature_map(p["Q"].reshape(-1, 2, 6), p["W"]).reshape(2, 4, 2, 6)
    want = np.zeros_like(O_neg)
    for r in range(2):
        P = int(p["prefix_len"][r])
        Phi_k = orc.feature_map(p["Kp"][r, :P], p["W"])          # [P, Hkv, 2F]
        for h in range(2):
            kern = Phi_q[r, :, h] @ Phi_k[:, h].T                  # [B, P]
            want[r, :, h] = kern @ p["Vp"][r, :P, h] / kern.sum(1, keepdims=True)
    _close(O_neg, want, rtol=1e-11, atol=1e-12, what="alpha=-inf is pure linear attention")


def pin_large_keys(orc):
    """Keys scaled x8 (the stress case): the route comparison still holds and
    the output stays a convex combination of the values."""
    rng = _rng(23)
    p = _random_problem(rng, 2, 8, 2, 2, 16, 8, 16, prefix_len=[16, 9], k_scale=8.0)
    S, z = _state_from_prefix(orc, p)
    O1 = orc.block_attn(p["Q"], p["K"], p["V"], p["W"], p["alpha"], S, z)
    O2 = orc.block_attn_prefix(p["Q"], p["K"], p["V"], p["W"], p["alpha"], p["Kp"], p["Vp"],
                               p["prefix_len"])
    _close(O1, O2, rtol=1e-10, atol=1e-12, what="large keys routes")
    for r in range(2):
        P = int(p["prefix_len"][r])
        for h in range(2):
            vals = np.concatenate([p["V"][r, :, h], p["Vp"][r, :P, h]], 0)
            assert np.all(O1[r, :, h] <= vals.max(0) + 1e-9), "convexity (max)"
            assert np.all(O1[r, :, h] >= vals.min(0) - 1e-9), "convexity (min)"


# --------------------------------------------------------------------------
# Training form (Sec. 3.2, Stage 1): every block of a sequence against the
# state of the blocks before it, and the gradient with respect to W and alpha.
# --------------------------------------------------------------------------
def _train_problem(rng, n_seq=2, n_blk=3, B=2, Hq=4, Hkv=2, d=4, F=3):
    L = n_blk * B
    return dict(
        Q=rng.standard_normal((n_seq, L, Hq, d)),
        K=rng.standard_normal((n_seq, L, Hkv, d)),
        V=rng.standard_normal((n_seq, L, Hkv, d)),
        W=rng.standard_normal((Hkv, d, F)) / math.sqrt(d),
        alpha=rng.uniform(-1.0, 1.5, Hq),
        dO=rng.standard_normal((n_seq, L, Hq, d)),
        B=B, n_blk=n_blk)


def pin_train_forward_is_prefix_route(orc):
    """Block n of a training sequence is one block-hybrid step whose linear
    branch is summed token by token over the n*B earlier tokens (Eq. 1 route,
    which never forms a state)."""
    p = _train_problem(_rng(31), n_seq=2, n_blk=4, B=3, Hq=4, Hkv=2, d=5, F=3)
    B = p["B"]
    O = orc.train_forward(p["Q"], p["K"], p["V"], p["W"], p["alpha"], B)
    for n in range(p["n_blk"]):
        blk = slice(n * B, (n + 1) * B)
        On = orc.block_attn_prefix(p["Q"][:, blk], p["K"][:, blk], p["V"][:, blk], p["W"],
                                   p["alpha"], p["K"], p["V"], [n * B] * 2)
        _close(O[:, blk], On, rtol=1e-11, atol=1e-12, what=f"training block {n}")


def _train_loss(orc, p, W, alpha):
    O = orc.train_forward(p["Q"], p["K"], p["V"], W, alpha, p["B"], n_threads=1)
    return float(np.sum(p["dO"] * O))


def pin_train_backward_finite_differences(orc):
    """dW and dalpha are the derivatives of sum(dO * O): central differences of
    the training forward, element by element."""
    p = _train_problem(_rng(32))
    dW, dalpha = orc.train_backward(p["Q"], p["K"], p["V"], p["W"], p["alpha"], p["dO"], p["B"])
    h = 1e-6
    fd_W = np.zeros_like(p["W"])
    for idx in np.ndindex(*p["W"].shape):
        Wp, Wm = p["W"].copy(), p["W"].copy()
        Wp[idx] += h
        Wm[idx] -= h
        fd_W[idx] = (_train_loss(orc, p, Wp, p["alpha"]) - _train_loss(orc, p, Wm, p["alpha"])) / (2 * h)
    fd_a = np.zeros_like(p["alpha"])
    for i in range(p["alpha"].size):
        ap, am = p["alpha"].copy(), p["alpha"].copy()
        ap[i] += h
        am[i] -= h
        fd_a[i] = (_train_loss(orc, p, p["W"], ap) - _train_loss(orc, p, p["W"], am)) / (2 * h)
    _close(dW, fd_W, rtol=1e-6, atol=1e-7, what="dW vs central differences")
    _close(dalpha, fd_a, rtol=1e-6, atol=1e-7, what="dalpha vs central differences")
    assert np.abs(fd_W).max() > 1e-3 and np.abs(fd_a).max() > 1e-3, "degenerate problem"


def pin_train_backward_single_block(orc):
    """With one block per sequence no query has a prefix: O is the in-block
    softmax alone, independent of W and alpha, so both gradients are zero
    (dW exactly: every state and state gradient is zero; dalpha to rounding,
    as the two terms of dw cancel)."""
    p = _train_problem(_rng(33), n_blk=1, B=4)
    dW, dalpha = orc.train_backward(p["Q"], p["K"], p["V"], p["W"], p["alpha"], p["dO"], p["B"])
    assert np.all(dW == 0.0) and np.abs(dalpha).max() < 1e-12, "gradients without any prefix"


def pin_train_backward_constant_values(orc):
    """V = 1 everywhere makes every output exactly 1 for any W and alpha (the
    attention mass sums to one), so both gradients vanish."""
    p = _train_problem(_rng(34), n_blk=4)
    p["V"] = np.ones_like(p["V"])
    dW, dalpha = orc.train_backward(p["Q"], p["K"], p["V"], p["W"], p["alpha"], p["dO"], p["B"])
    assert np.abs(dW).max() < 1e-12 and np.abs(dalpha).max() < 1e-12, "gradients with V = 1"


def pin_train_backward_linear_in_dO(orc):
    """The gradient of sum(dO * O) is linear in dO."""
    p = _train_problem(_rng(35))
    rng = _rng(36)
    d1, d2 = p["dO"], rng.standard_normal(p["dO"].shape)
    args = (p["Q"], p["K"], p["V"], p["W"], p["alpha"])
    g1 = orc.train_backward(*args, d1, p["B"])
    g2 = orc.train_backward(*args, d2, p["B"])
    g3 = orc.train_backward(*args, 2.0 * d1 - 3.0 * d2, p["B"])
    for a, b, c, what in zip(g1, g2, g3, ("dW", "dalpha")):
        _close(c, 2.0 * a - 3.0 * b, rtol=1e-10, atol=1e-12, what=f"{what} linear in dO")


def pin_train_backward_saturated_gate(orc):
    """w = sigmoid(alpha) is flat at alpha = +inf: dalpha is zero there, and dW
    is the gradient of the model whose gate is exactly 1."""
    p = _train_problem(_rng(37))
    a = p["alpha"].copy()
    a[1] = np.inf
    dW, dalpha = orc.train_backward(p["Q"], p["K"], p["V"], p["W"], a, p["dO"], p["B"])
    assert dalpha[1] == 0.0 and np.all(np.isfinite(dW)), "saturated gate"


def pin_thread_count_changes_nothing(orc):
    """The oracle fans independent (request, head) units out over threads; every
    route gives the same bits on 1 thread and on 7 (more threads than units for
    some calls, fewer for others), so no unit is skipped, repeated or shares
    scratch with another."""
    p = _random_problem(_rng(41), n_req=5, B=3, Hq=4, Hkv=2, d=6, F=3, P_max=4)
    S1, z1 = orc.empty_state(5, 2, 6, 3)
    S7, z7 = orc.empty_state(5, 2, 6, 3)
    orc.commit(p["Kp"], p["Vp"], p["W"], S1, z1, n_threads=1)
    orc.commit(p["Kp"], p["Vp"], p["W"], S7, z7, n_threads=7)
    _close(S7, S1, rtol=0, atol=0, what="commit S")
    _close(z7, z1, rtol=0, atol=0, what="commit z")
    args = (p["Q"], p["K"], p["V"], p["W"], p["alpha"])
    _close(orc.block_attn(*args, S1, z1, n_threads=7), orc.block_attn(*args, S1, z1, n_threads=1),
           rtol=0, atol=0, what="state route")
    _close(orc.block_attn_prefix(*args, p["Kp"], p["Vp"], p["prefix_len"], n_threads=7),
           orc.block_attn_prefix(*args, p["Kp"], p["Vp"], p["prefix_len"], n_threads=1),
           rtol=0, atol=0, what="prefix route")
    t = _train_problem(_rng(42), n_seq=3, n_blk=3, B=2, Hq=4, Hkv=2, d=4, F=3)
    targs = (t["Q"], t["K"], t["V"], t["W"], t["alpha"])
    _close(orc.train_forward(*targs, t["B"], n_threads=7), orc.train_forward(*targs, t["B"], n_threads=1),
           rtol=0, atol=0, what="training forward")
    g7 = orc.train_backward(*targs, t["dO"], t["B"], n_threads=7)
    g1 = orc.train_backward(*targs, t["dO"], t["B"], n_threads=1)
    for a, b, what in zip(g7, g1, ("dW", "dalpha")):
        _close(a, b, rtol=0, atol=0, what=f"training {what}")


ALL_PINS = [v for k, v in sorted(globals().items()) if k.startswith("pin_")]


def run_all(orc):
    failures = []
    for pin in ALL_PINS:
        try:
            pin(orc)
        except Exception as exc:  # noqa: BLE001 -- report every kind of failure
            failures.append(f"{pin.__name__}: {type(exc).__name__}: {str(exc)[:160]}")
    return failures


if __name__ == "__main__":
    orc = Oracle(sys.argv[1]) if len(sys.argv) > 1 else Oracle()
    for line in run_all(orc):
        print("FAIL", line)
    print("DONE")
