"""The bf16 rounding check of the GPU parity tests, on the CPU.

It must accept a step whose stored weights are the round-to-nearest-even of
pre-rounding values that differ from the oracle's by a small gap, and must
catch a weight that is one ulp off where no rounding boundary lies between
the two pre-rounding values, or one that is not the rounding of the GPU's own
value.
"""
import numpy as np

import oracle.malt_ref as ref
from tests.gpu_harness import bf16_rounding, bf16_ulp


def _case(seed=3, n=20000, gap_rel=1e-2):
    rng = np.random.default_rng(seed)
    W_prev = ref.round_to_bf16(rng.normal(0, 0.02, n))
    dW_ref = rng.normal(0, 4e-4, n)
    dW_gpu = dW_ref * (1 + gap_rel * rng.standard_normal(n))
    x_ref = W_prev - dW_ref
    x_gpu = W_prev - dW_gpu
    slack = 2.0 ** -21 * (np.abs(x_gpu) + np.abs(dW_gpu))
    return x_gpu, x_ref, slack, dW_ref


def test_correct_rounding_passes():
    x_gpu, x_ref, slack, dW_ref = _case()
    r = bf16_rounding(ref.round_to_bf16(x_gpu), x_gpu, x_ref, slack, dW_ref)
    assert r["own_mismatch"] == 0 and r["oracle_mismatch_off_boundary"] == 0
    # a 1 % gap with updates of a few ulps straddles some boundaries, within
    # what the 2e-2 update tolerance allows
    assert 0 < r["straddle"] <= r["straddle_allowed"]


def test_one_ulp_error_away_from_a_boundary_is_caught():
    x_gpu, x_ref, slack, dW_ref = _case()
    W = ref.round_to_bf16(x_gpu)
    r0 = bf16_rounding(W, x_gpu, x_ref, slack, dW_ref)
    lo, hi = np.minimum(x_gpu, x_ref) - slack, np.maximum(x_gpu, x_ref) + slack
    clean = np.flatnonzero(ref.round_to_bf16(lo) == ref.round_to_bf16(hi))
    k = clean[len(clean) // 2]
    W[k] += bf16_ulp(W[k])
    r = bf16_rounding(W, x_gpu, x_ref, slack, dW_ref)
    assert r["own_mismatch"] == 1 and r["oracle_mismatch_off_boundary"] == 1
    assert r["straddle"] == r0["straddle"]


def test_wrong_gpu_rounding_is_caught_even_when_it_matches_the_oracle():
    # the GPU stores rn(x_ref) where its own value rounds elsewhere: the
    # oracle agrees, but the weight is not what the kernel's arithmetic gives
    x_gpu, x_ref, slack, dW_ref = _case(gap_rel=0.5)
    W = ref.round_to_bf16(x_ref)
    r = bf16_rounding(W, x_gpu, x_ref, slack, dW_ref)
    assert r["own_mismatch"] > 0


def test_canary_margins_catch_writes_past_a_buffer():
    """The harness's caller buffers sit between canary margins; a write just
    before or just past a buffer (planted here, on the CPU) is caught, writes
    inside it are not."""
    import torch
    from tests.gpu_harness import CANARY, canaries_intact, guarded
    for dtype in (torch.float32, torch.bfloat16):
        t, buf = guarded((5, 7), dtype, "cpu")
        assert t.is_contiguous() and t.data_ptr() % 16 == 0 and canaries_intact(buf)
        t.fill_(3.0)
        assert canaries_intact(buf)
        for k in (CANARY - 1, CANARY + t.numel()):      # just before, just after
            _, b2 = guarded((5, 7), dtype, "cpu")
            b2[k] = 1.0
            assert not canaries_intact(b2), (dtype, k)
