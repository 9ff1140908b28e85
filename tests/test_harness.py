"""The parity harness itself (CPU): a bf16 error confined to one (request,
head) unit passes the batch-wide rel-L2 bound but fails the per-unit one."""
import numpy as np
import pytest
import torch

from gpu_harness import assert_parity, unit_rel_l2


def test_unit_axes_pick_request_and_head():
    rng = np.random.default_rng(0)
    want = rng.standard_normal((5, 32, 16, 128))       # [n, B, Hq, d]
    got = want.copy()
    got[3, :, 7, :5] += 0.5                            # one (request 3, head 7) unit
    per = unit_rel_l2(got, want, (0, 2))
    assert per.shape == (5 * 16,)
    assert np.argmax(per) == 3 * 16 + 7
    assert np.count_nonzero(per) == 1
    S = rng.standard_normal((4, 4, 256, 128))          # [n, Hkv, 2F, d]
    S2 = S.copy()
    S2[2, 1] *= 1.05
    per = unit_rel_l2(S2, S, (0, 1))
    assert np.argmax(per) == 2 * 4 + 1 and np.isclose(per.max(), 0.05)


def test_localised_bf16_error_is_caught_per_unit():
    rng = np.random.default_rng(1)
    want = rng.standard_normal((5, 32, 16, 128))
    got = want * (1 + 1e-3 * rng.standard_normal(want.shape))
    got[1, :, 4, :] *= 1.05                            # one (request, head) unit 5% off
    assert np.linalg.norm(got - want) / np.linalg.norm(want) < 1e-2   # hidden in the batch's norm
    with pytest.raises(AssertionError, match="unit"):
        assert_parity(got, want, torch.bfloat16, "planted", units="out")
    ok = want * (1 + 1e-3 * rng.standard_normal(want.shape))
    assert assert_parity(ok, want, torch.bfloat16, "clean", units="out") < 2e-3
