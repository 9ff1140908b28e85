"""Runs the CUDA path and the fp64 oracle side by side on the same seeded inputs.

The oracle only ever sees host copies of the inputs the GPU consumed (never a
GPU result); GPU states are compared after unpacking to the logical layout.
"""
from __future__ import annotations

import numpy as np
import torch

import oracle
from paper_2608_06628_gb300 import hybrid as H
from paper_2608_06628_gb300 import workloads as wk
from paper_2608_06628_gb300.state_pool import StatePool

# Tolerances: fp32 I/O -> rel-L2 <= 1e-5 and max-abs <= 1e-4;
#             bf16 I/O with fp32 state -> rel-L2 <= 1e-2.
TOL = {torch.float32: dict(rel=1e-5, abs=1e-4), torch.bfloat16: dict(rel=1e-2, abs=None)}


def h64(t: torch.Tensor) -> np.ndarray:
    return t.detach().to(torch.float64).cpu().numpy()


def rel_l2(got, want):
    got = np.asarray(got, dtype=np.float64)
    want = np.asarray(want, dtype=np.float64)
    den = np.linalg.norm(want)
    return float(np.linalg.norm(got - want) / (den if den > 0 else 1.0))


# Axes that index one unit of work in each kind of compared array:
#   "out"   [n, B, Hq, d]     one (request, query head)
#   "state" [n, Hkv, 2F, d] and z [n, Hkv, 2F]: one (request, state head)
UNIT_AXES = {"out": (0, 2), "state": (0, 1)}


def unit_rel_l2(got, want, axes):
    """rel-L2 of every unit (the indices along `axes`), as an array over units."""
    got = np.asarray(got, dtype=np.float64)
    want = np.asarray(want, dtype=np.float64)
    rest = tuple(i for i in range(got.ndim) if i not in axes)
    g = np.transpose(got, axes + rest).reshape(int(np.prod([got.shape[i] for i in axes])), -1)
    w = np.transpose(want, axes + rest).reshape(g.shape)
    num = np.linalg.norm(g - w, axis=1)
    den = np.linalg.norm(w, axis=1)
    return num / np.where(den > 0, den, 1.0)


def assert_parity(got, want, dtype, what="", units=None):
    """Element-wise parity of a GPU result with the oracle's.

    The bound of the dtype applies to the whole tensor and, for bf16, also to
    every unit on its own (units = "out" or "state", see UNIT_AXES), so that an
    error confined to one (request, head) cannot hide in the batch's norm."""
    got = np.asarray(got, dtype=np.float64)
    want = np.asarray(want, dtype=np.float64)
    assert got.shape == want.shape, f"{what}: shapes {got.shape} vs {want.shape}"
    assert np.all(np.isfinite(got)), f"{what}: non-finite values"
    tol = TOL[dtype]
    r = rel_l2(got, want)
    assert r <= tol["rel"], f"{what}: rel-L2 {r:.3e} > {tol['rel']}"
    worst = None
    if units is not None and dtype == torch.bfloat16 and got.size:
        per = unit_rel_l2(got, want, UNIT_AXES[units])
        k = int(np.argmax(per))
        worst = float(per[k])
        assert worst <= tol["rel"], f"{what}: unit {k} rel-L2 {worst:.3e} > {tol['rel']}"
    if tol["abs"] is not None:
        m = float(np.max(np.abs(got - want))) if got.size else 0.0
        assert m <= tol["abs"], f"{what}: max-abs {m:.3e} > {tol['abs']}"
    print(f"parity {what}: rel-L2 {r:.2e}" + (f", worst unit {worst:.2e}" if worst is not None else ""))
    return r


class Pair:
    """GPU states for all requests of a workload plus oracle states for the
    tracked subset (all requests by default)."""

    def __init__(self, wl: wk.Workload, device="cuda", layer=0, tracked=None, orc=None):
        self.wl = wl
        self.dev = torch.device(device)
        self.cfg = H.make_cfg(wl.d, wl.F, wl.Hq, wl.Hkv, wl.B, wl.io_dtype)
        self.W, self.alpha = wk.params(wl, layer, self.dev)
        self.W64 = h64(self.W)
        self.alpha64 = h64(self.alpha)
        self.pool = StatePool(self.cfg, wl.n_req, self.dev)
        self.ptrs = self.pool.all_ptrs()
        H.hybrid_state_init(self.cfg, self.ptrs, wl.n_req)
        self.orc = orc or oracle.load()
        self.tracked = np.arange(wl.n_req) if tracked is None else np.asarray(tracked)
        self.S, self.z = self.orc.empty_state(len(self.tracked), wl.Hkv, wl.d, wl.F)

    # -- commits ---------------------------------------------------------------
    def commit(self, K, V, reqs=None):
        """Fold K, V [len(reqs), T, Hkv, d] into requests `reqs` on both sides."""
        wl = self.wl
        reqs = np.arange(wl.n_req) if reqs is None else np.asarray(reqs)
        if len(reqs) == 0:
            return
        ptrs = self.pool.ptr_array(reqs.tolist())
        H.hybrid_commit_block(self.cfg, K, V, K.shape[1], self.W, ptrs, len(reqs))
        pos = {int(r): i for i, r in enumerate(reqs)}
        sel = [i for i, r in enumerate(self.tracked) if int(r) in pos]
        if sel:
            rows = torch.as_tensor([pos[int(self.tracked[i])] for i in sel], device=K.device)
            Sx, zx = self.S[sel].copy(), self.z[sel].copy()
            self.orc.commit(h64(K[rows]), h64(V[rows]), self.W64, Sx, zx)
            self.S[sel], self.z[sel] = Sx, zx

    def build_prefixes(self, plen, layer=0):
        """Ragged prefixes: block b is committed for every request with plen > b*B."""
        wl = self.wl
        n_blocks = int(np.max(plen)) // wl.B if len(plen) else 0
        for b in range(n_blocks):
            reqs = np.nonzero(plen > b * wl.B)[0]
            K, V = wk.prefix_kv(wl, b, self.dev, layer=layer)
            idx = torch.as_tensor(reqs, device=self.dev)
            self.commit(K[idx], V[idx], reqs)

    # -- one step ----------------------------------------------------------------
    def step(self, Q, K, V, alpha=None):
        """GPU block attention for all requests; oracle output for the tracked ones."""
        alpha = self.alpha if alpha is None else alpha
        O = torch.empty_like(Q)
        H.hybrid_block_attn(self.cfg, Q, K, V, self.W, alpha, self.ptrs, self.wl.n_req, O)
        H.hybrid_check()
        t = torch.as_tensor(self.tracked, device=Q.device)
        want = self.orc.block_attn(h64(Q[t]), h64(K[t]), h64(V[t]), self.W64, h64(alpha),
                                   self.S, self.z)
        return h64(O[t]), want, O

    def gpu_state(self, reqs=None):
        wl = self.wl
        reqs = self.tracked if reqs is None else np.asarray(reqs)
        P2 = 2 * wl.F
        S = torch.empty((len(reqs), wl.Hkv, P2, wl.d), dtype=torch.float32, device=self.dev)
        z = torch.empty((len(reqs), wl.Hkv, P2), dtype=torch.float32, device=self.dev)
        H.hybrid_state_unpack(self.cfg, self.pool.ptr_array(reqs.tolist()), len(reqs), S, z)
        H.hybrid_check()
        return h64(S), h64(z)
