"""Seeded synthetic inputs shaped like the paper's decoding setting.

This module only draws random numbers: it holds none of the method's
arithmetic, and both the CUDA path and the CPU oracle consume what it makes
(the oracle through host copies of the very tensors the GPU saw).

Recipe (every configuration):
  * Q, K, V ~ N(0, 1) drawn in float32, then rounded to the I/O dtype
    (round-to-nearest-even for bfloat16); K optionally scaled (x8 stress).
  * W ~ N(0, 1/d) per state head, rounded to the I/O dtype.
  * alpha ~ U(0, 1) per query head (so w = sigmoid(alpha) in [0.5, 0.731]).
  * Prefixes are built by successive block commits of fresh K/V; ragged
    prefix lengths are multiples of the block size drawn uniformly.
Sub-streams are keyed by (base seed, purpose, layer, block, step) so any one
block can be regenerated on its own.  Large tensors are drawn on the device
with a CUDA generator (reproducible on the same GPU type); the oracle receives
host copies of exactly the tensors used.
"""
from __future__ import annotations

import dataclasses
import hashlib

import numpy as np
import torch


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    io_dtype: torch.dtype
    n_req: int
    Hq: int
    Hkv: int
    d: int
    F: int
    B: int
    seed: int
    prefix_min: int = 0       # tokens, multiple of B
    prefix_max: int = 0
    k_scale: float = 1.0
    w_var: float | None = None   # variance of W entries; default 1/d
    layers: int = 1
    steps_per_block: int = 1
    blocks: int = 0           # decode loop length (config 4)
    seq_len: int = 0          # training form: tokens per sequence (n_req sequences)
    description: str = ""

    @property
    def w_std(self) -> float:
        return float(np.sqrt(self.w_var if self.w_var is not None else 1.0 / self.d))

    def with_(self, **kw) -> "Workload":
        return dataclasses.replace(self, **kw)


# The five configurations of the decoding hot path.
C1 = Workload("c1_fp32_tiny", torch.float32, n_req=1, Hq=2, Hkv=2, d=64, F=64, B=16, seed=0,
              prefix_min=64, prefix_max=64, w_var=1.0 / 64,
              description="fp32, batch 1, 2 heads, d 64, F 64, B 16, prefix of 4 blocks")
C2 = Workload("c2_bf16_b8_mha", torch.bfloat16, n_req=8, Hq=16, Hkv=16, d=128, F=128, B=32, seed=1,
              prefix_min=2048, prefix_max=2048,
              description="bf16, batch 8, 16 heads, d 128, F 128, B 32, prefix 2048")
C3 = Workload("c3_bf16_b64_gqa_ragged", torch.bfloat16, n_req=64, Hq=16, Hkv=4, d=128, F=128, B=32,
              seed=2, prefix_min=256, prefix_max=8192,
              description="bf16, batch 64, GQA 16:4, d 128, F 128, B 32, ragged prefixes 256-8192")
C4 = Workload("c4_bf16_decode_loop", torch.bfloat16, n_req=32, Hq=16, Hkv=16, d=128, F=128, B=32,
              seed=3, layers=6, steps_per_block=8, blocks=64,
              description="bf16, batch 32, 6 layers x 8 steps x 64 blocks from empty state")
C5 = Workload("c5_bf16_b256_f256_k8", torch.bfloat16, n_req=256, Hq=16, Hkv=16, d=128, F=256, B=64,
              seed=4, prefix_min=1024, prefix_max=32768, k_scale=8.0,
              description="bf16, batch 256, 16 heads, d 128, F 256, B 64, ragged 1k-32k, K x8")
CONFIGS = {w.name: w for w in (C1, C2, C3, C4, C5)}

# Training form (Stage 1 attention transfer): batches of whole sequences with
# the layer shape of configuration 3; the paper's transfer runs over moderate
# generation lengths (2048-token sequences here).
T1 = Workload("t1_bf16_stage1_8x2048_gqa", torch.bfloat16, n_req=8, Hq=16, Hkv=4, d=128, F=128, B=32,
              seed=5, seq_len=2048,
              description="bf16, 8 sequences of 2048 tokens (64 blocks of 32), GQA 16:4, d 128, F 128")


def sub_seed(base: int, *tags) -> int:
    """Deterministic 63-bit seed for the sub-stream named by tags."""
    h = hashlib.sha256(repr((int(base),) + tuple(tags)).encode()).digest()
    return int.from_bytes(h[:8], "little") & ((1 << 63) - 1)


def _gen(device, seed):
    g = torch.Generator(device=device)
    g.manual_seed(seed)
    return g


def _randn(shape, seed, device, dtype, scale=1.0):
    x = torch.randn(shape, generator=_gen(device, seed), device=device, dtype=torch.float32)
    if scale != 1.0:
        x = x * scale
    return x.to(dtype)


def params(wl: Workload, layer: int = 0, device="cpu"):
    """W [Hkv, d, F] (io dtype) and alpha [Hq] (float32) of one hybrid layer."""
    W = _randn((wl.Hkv, wl.d, wl.F), sub_seed(wl.seed, "W", layer), "cpu", wl.io_dtype, wl.w_std)
    g = _gen("cpu", sub_seed(wl.seed, "alpha", layer))
    alpha = torch.rand((wl.Hq,), generator=g, dtype=torch.float32)
    return W.to(device), alpha.to(device)


def prefix_lengths(wl: Workload) -> np.ndarray:
    """Committed prefix length (tokens) of every request."""
    if wl.prefix_max == wl.prefix_min:
        return np.full(wl.n_req, wl.prefix_min, dtype=np.int64)
    rng = np.random.default_rng(sub_seed(wl.seed, "prefix_len"))
    lo, hi = wl.prefix_min // wl.B, wl.prefix_max // wl.B
    return rng.integers(lo, hi + 1, size=wl.n_req).astype(np.int64) * wl.B


def block_qkv(wl: Workload, tag, device="cpu", n_req=None):
    """Q [n, B, Hq, d], K, V [n, B, Hkv, d] of one active block (io dtype)."""
    n = wl.n_req if n_req is None else n_req
    Q = _randn((n, wl.B, wl.Hq, wl.d), sub_seed(wl.seed, "Q", tag), device, wl.io_dtype)
    K = _randn((n, wl.B, wl.Hkv, wl.d), sub_seed(wl.seed, "K", tag), device, wl.io_dtype, wl.k_scale)
    V = _randn((n, wl.B, wl.Hkv, wl.d), sub_seed(wl.seed, "V", tag), device, wl.io_dtype)
    return Q, K, V


def train_batch(wl: Workload, tag=0, device="cpu", n_seq=None, seq_len=None):
    """Q, dO [n, L, Hq, d] and K, V [n, L, Hkv, d] of a training batch (io dtype).
    dO stands in for the gradient of the attention-transfer loss."""
    n = wl.n_req if n_seq is None else n_seq
    L = wl.seq_len if seq_len is None else seq_len
    Q = _randn((n, L, wl.Hq, wl.d), sub_seed(wl.seed, "tQ", tag), device, wl.io_dtype)
    K = _randn((n, L, wl.Hkv, wl.d), sub_seed(wl.seed, "tK", tag), device, wl.io_dtype, wl.k_scale)
    V = _randn((n, L, wl.Hkv, wl.d), sub_seed(wl.seed, "tV", tag), device, wl.io_dtype)
    dO = _randn((n, L, wl.Hq, wl.d), sub_seed(wl.seed, "tdO", tag), device, wl.io_dtype)
    return Q, K, V, dO


def prefix_kv(wl: Workload, block: int, device="cpu", n_req=None, n_tok=None, layer: int = 0):
    """K, V [n, T, Hkv, d] of committed prefix block `block` (T = B by default)."""
    n = wl.n_req if n_req is None else n_req
    T = wl.B if n_tok is None else n_tok
    K = _randn((n, T, wl.Hkv, wl.d), sub_seed(wl.seed, "pK", layer, block), device, wl.io_dtype,
               wl.k_scale)
    V = _randn((n, T, wl.Hkv, wl.d), sub_seed(wl.seed, "pV", layer, block), device, wl.io_dtype)
    return K, V
