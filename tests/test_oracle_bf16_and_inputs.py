"""Pins for the oracle's bf16 conversions and checks of the input generator.

The oracle rounds doubles to bf16 directly (one rounding); the input generator
rounds float32 with an integer bit trick. They are separate implementations,
so agreement on float32-representable values checks both.
"""
import numpy as np
import pytest

import oracle
from paper_2601_02819_gb300 import inputs


def test_bf16_round_half_even_pins():
    # 1 + 2^-8 lies halfway between 1 and 1 + 2^-7: ties go to the even value 1.
    # 1 + 3*2^-8 lies halfway between 1 + 2^-7 and 1 + 2^-6: ties go to 1 + 2^-6.
    vals = np.array([1.0, 1 + 2**-8, 1 + 3 * 2**-8, -(1 + 2**-8), 223.5, 159.5, 95.5,
                     1 + 2**-8 + 2**-30, 0.0, -0.0, 1e39, -1e39, 2.0**-140])
    bits = oracle.f64_to_bf16(vals)
    expect = [0x3F80, 0x3F80, 0x3F82, 0xBF80, 0x4360, 0x4320, 0x42BF, 0x3F81, 0x0000, 0x8000,
              0x7F80, 0xFF80, 0x0000]
    assert [int(b) for b in bits] == expect
    back = oracle.bf16_to_f64(bits[:7])
    assert list(back) == [1.0, 1.0, 1 + 2**-6, -1.0, 224.0, 160.0, 95.5]


def test_bf16_subnormal_grid():
    # Smallest bf16 subnormal is 2^-133; 1.5 * 2^-133 is a tie -> even (2 * 2^-133).
    bits = oracle.f64_to_bf16(np.array([2.0**-133, 1.5 * 2.0**-133, 2.0**-134 * 1.01]))
    assert [int(b) for b in bits] == [0x0001, 0x0002, 0x0001]


def test_bf16_matches_generator_rounding_on_float32_values():
    rng = np.random.default_rng(7)
    x = (rng.standard_normal(200_000) * np.exp(rng.uniform(-20, 20, 200_000))).astype(np.float32)
    a = oracle.f64_to_bf16(x.astype(np.float64))
    b = inputs.f32_to_bf16_bits(x)
    assert np.array_equal(a, b)
    assert np.array_equal(oracle.bf16_to_f64(b), inputs.bf16_bits_to_f32(b).astype(np.float64))


def test_generator_is_seeded_and_shaped():
    w = inputs.WORKLOADS["tiny_2k"]
    a = inputs.make_inputs(w, with_grad=True)
    b = inputs.make_inputs(w, with_grad=True)
    for k in ("Q", "K", "V", "dO", "ids", "mask"):
        assert np.array_equal(a[k], b[k]), k
    assert a["Q"].shape == (1, 2, 2048, 128) and a["Q"].dtype == np.uint16
    assert a["K"].shape == (1, 1, 2048, 128)
    assert a["mask"].shape == (1, 2048)
    dens = a["mask"].mean()
    assert 0.06 < dens < 0.10  # about 8% punctuation
    q = inputs.bf16_bits_to_f32(a["Q"])
    assert abs(q.mean()) < 0.02 and abs(q.std() - 1) < 0.02


def test_sentence_like_gaps():
    rng = np.random.default_rng(3)
    pset = inputs.punct_id_set(rng)
    ids = inputs.draw_token_ids(rng, 2, 20000, "sentence", (9, 25), pset)
    mask = np.isin(ids, pset)
    for b in range(2):
        pos = np.nonzero(mask[b])[0]
        gaps = np.diff(pos)
        assert gaps.min() >= 9 and gaps.max() <= 25
    assert 0.05 < mask.mean() < 0.07  # ~6% density, as the prefill workloads state


def test_none_placement_has_no_punctuation():
    w = inputs.custom(B=1, L=512, Hq=2, Hkv=1, punct="none")
    x = inputs.make_inputs(w)
    assert x["mask"].sum() == 0


def test_drawn_block_lists_are_valid_and_seeded():
    # The attention-only parity tests feed these lists to both sides: every
    # list must be ascending, unique, inside [0, qb], hold the first and the
    # query's own block, have min(topk, qb + 1) entries and -1 padding.
    from paper_2601_02819_gb300 import inputs
    idx, cnt = inputs.random_block_lists(np.random.default_rng(3), 2, 3, 70, 9)
    idx2, cnt2 = inputs.random_block_lists(np.random.default_rng(3), 2, 3, 70, 9)
    assert np.array_equal(idx, idx2) and np.array_equal(cnt, cnt2)
    assert idx.shape == (2, 3, 70, 9) and idx.dtype == np.int32 and cnt.dtype == np.int32
    for b in range(2):
        for g in range(3):
            for qb in range(70):
                n, row = cnt[b, g, qb], idx[b, g, qb]
                assert n == min(9, qb + 1)
                assert row[0] == 0 and row[n - 1] == qb
                assert np.all(np.diff(row[:n]) > 0) and np.all(row[n:] == -1)
    # not always the same earlier blocks
    assert len({tuple(idx[0, 0, qb, 1:8]) for qb in range(40, 70)}) > 20
