"""The seeded input generators shared by the CUDA path and the oracle: the recipe
they state (distributions, rounding, prefix lengths, shapes of the five decoding
configurations) and their determinism, checked on the CPU."""
import numpy as np
import torch

from paper_2608_06628_gb300 import workloads as wk


def test_configurations_have_the_stated_shapes():
    shapes = {n: (w.io_dtype, w.n_req, w.Hq, w.Hkv, w.d, w.F, w.B, w.prefix_min, w.prefix_max, w.k_scale)
              for n, w in wk.CONFIGS.items()}
    assert shapes == {
        "c1_fp32_tiny": (torch.float32, 1, 2, 2, 64, 64, 16, 64, 64, 1.0),
        "c2_bf16_b8_mha": (torch.bfloat16, 8, 16, 16, 128, 128, 32, 2048, 2048, 1.0),
        "c3_bf16_b64_gqa_ragged": (torch.bfloat16, 64, 16, 4, 128, 128, 32, 256, 8192, 1.0),
        "c4_bf16_decode_loop": (torch.bfloat16, 32, 16, 16, 128, 128, 32, 0, 0, 1.0),
        "c5_bf16_b256_f256_k8": (torch.bfloat16, 256, 16, 16, 128, 256, 64, 1024, 32768, 8.0),
    }
    c4 = wk.C4
    assert (c4.layers, c4.steps_per_block, c4.blocks) == (6, 8, 64)
    assert wk.C1.w_std == 1.0 / 8.0 and wk.C3.w_std == float(np.sqrt(1.0 / 128))


def test_draws_are_deterministic_and_keyed_by_purpose():
    wl = wk.C3.with_(n_req=3)
    a = wk.block_qkv(wl, ("t", 1))
    b = wk.block_qkv(wl, ("t", 1))
    c = wk.block_qkv(wl, ("t", 2))
    for x, y, z in zip(a, b, c):
        assert torch.equal(x, y) and not torch.equal(x, z)
    Q, K, V = a
    assert Q.shape == (3, 32, 16, 128) and K.shape == V.shape == (3, 32, 4, 128)
    # Q, K and V come from different sub-streams
    assert not torch.equal(Q[:, :, :4], K) and not torch.equal(K, V)
    # a prefix block can be regenerated on its own, per layer
    k0, v0 = wk.prefix_kv(wl, 5)
    k1, _ = wk.prefix_kv(wl, 5)
    k2, _ = wk.prefix_kv(wl, 5, layer=1)
    assert torch.equal(k0, k1) and not torch.equal(k0, k2) and not torch.equal(k0, v0)
    assert wk.sub_seed(2, "Q", 1) == wk.sub_seed(2, "Q", 1) != wk.sub_seed(2, "Q", 2)
    assert 0 <= wk.sub_seed(123, "x") < (1 << 63)


def test_distributions_and_rounding():
    wl = wk.C3
    Q, K, V = wk.block_qkv(wl, "stats", n_req=16)
    for t in (Q, K, V):
        assert t.dtype == torch.bfloat16
        x = t.double()
        assert abs(float(x.mean())) < 0.01 and abs(float(x.std()) - 1.0) < 0.01
    # the bf16 values are the round-to-nearest-even images of the fp32 draws
    g = torch.Generator().manual_seed(wk.sub_seed(wl.seed, "Q", "stats"))
    q32 = torch.randn(Q.shape, generator=g, dtype=torch.float32)
    bits = q32.view(torch.int32).to(torch.int64)
    rne = ((bits + 0x7FFF + ((bits >> 16) & 1)) >> 16) << 16
    assert torch.equal(Q.float(), rne.to(torch.int32).view(torch.float32))
    # K scaled for the stress configuration
    K5 = wk.block_qkv(wk.C5, "stats", n_req=4)[1].double()
    assert abs(float(K5.std()) - 8.0) < 0.1
    W, alpha = wk.params(wl)
    assert W.shape == (4, 128, 128) and W.dtype == torch.bfloat16
    assert abs(float(W.double().std()) * np.sqrt(128) - 1.0) < 0.02
    assert alpha.shape == (16,) and alpha.dtype == torch.float32
    assert float(alpha.min()) >= 0.0 and float(alpha.max()) < 1.0
    W1, _ = wk.params(wk.C1)
    assert W1.dtype == torch.float32 and abs(float(W1.std()) - 1.0 / 8.0) < 0.01


def test_prefix_lengths_are_block_multiples_in_range():
    for wl in (wk.C3, wk.C5):
        p = wk.prefix_lengths(wl)
        assert p.shape == (wl.n_req,) and np.all(p % wl.B == 0)
        assert p.min() >= wl.prefix_min and p.max() <= wl.prefix_max
        assert len(np.unique(p)) > wl.n_req // 4      # ragged, not a constant
        assert np.array_equal(p, wk.prefix_lengths(wl))
    assert np.all(wk.prefix_lengths(wk.C2) == 2048) and np.all(wk.prefix_lengths(wk.C4) == 0)


def test_training_batch_shapes():
    Q, K, V, dO = wk.train_batch(wk.T1, n_seq=2, seq_len=64)
    assert Q.shape == dO.shape == (2, 64, 16, 128) and K.shape == V.shape == (2, 64, 4, 128)
    assert not torch.equal(Q, dO)
    assert wk.T1.seq_len % wk.T1.B == 0
