"""phsa_prefill_append: chunked prefill into the caches with the representative
keys of completed blocks computed from the same loads (block-level caching,
Section 3.2; Eq. 6-8 for the keys).

Sequences are filled chunk by chunk with ragged chunk boundaries. Afterwards
the caches must hold exactly the appended rows and flags, and every full
block's key must be within one bf16 ulp of the oracle's (oracle.block_repr over
the finished cache) and bit-identical to phsa_build_block_repr over the
finished cache.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2601_02819_gb300 import inputs, phsa
from parity import bf16_bits, to_dev_bf16, ulp_distance

pytestmark = pytest.mark.gpu

D, M = 128, 64


def _rand(rng, *s):
    return inputs.f32_to_bf16_bits(rng.standard_normal(s).astype(np.float32))


class Caches:
    def __init__(self, B, Hkv, Lc, bm=M):
        self.bm = bm
        self.K = torch.zeros((B, Hkv, Lc, D), dtype=torch.bfloat16, device="cuda")
        self.V = torch.zeros_like(self.K)
        self.mask = torch.zeros((B, Lc), dtype=torch.uint8, device="cuda")
        self.Kr = torch.zeros((B, Hkv, Lc // bm, D), dtype=torch.bfloat16, device="cuda")

    def append(self, b0, b1, kc, vc, fc, lens, lam):
        """One call over sequences [b0, b1) (a contiguous slice of the caches)."""
        phsa.phsa_prefill_append(to_dev_bf16(kc), to_dev_bf16(vc),
                                 torch.tensor(lens, dtype=torch.int32, device="cuda"),
                                 self.K[b0:b1], self.V[b0:b1], self.mask[b0:b1], self.Kr[b0:b1],
                                 lam, flag_chunk=None if fc is None else torch.from_numpy(fc).cuda(),
                                 block_size=self.bm)


def _check(c, Kfull, Vfull, flags, totals, lam):
    bm = c.bm
    Kh, Vh, mh = bf16_bits(c.K), bf16_bits(c.V), c.mask.cpu().numpy()
    for b, n in enumerate(totals):
        assert np.array_equal(Kh[b, :, :n], Kfull[b, :, :n])
        assert np.array_equal(Vh[b, :, :n], Vfull[b, :, :n])
        assert np.array_equal(mh[b, :n], flags[b, :n])
        assert not Kh[b, :, n:].any() and not Vh[b, :, n:].any()
        T = n // bm
        if T == 0:
            continue
        got = bf16_bits(c.Kr)[b:b + 1, :, :T]
        ref = oracle.block_repr(Kfull[b:b + 1, :, :n], flags[b:b + 1, :n], bm, lam)
        assert ulp_distance(got, ref[:, :, :T]).max() <= 1
        full = phsa.phsa_build_block_repr(c.K[b:b + 1, :, :T * bm].contiguous(),
                                          c.mask[b:b + 1, :T * bm].contiguous(), lam,
                                          block_size=bm)
        torch.cuda.synchronize()
        assert np.array_equal(bf16_bits(full), got)


@pytest.mark.parametrize("lam", [0.5, 0.0, 1.0])
def test_chunked_prefill_matches_oracle_and_full_build(lam):
    rng = np.random.default_rng(int(lam * 10) + 7)
    B, Hkv, Lc = 3, 2, 64 * 9
    totals = [64 * 9, 64 * 5 + 37, 130]
    plans = [[1, 63, 64, 129, 100, 150, 69], [37, 64, 64, 1, 191], [130]]
    Kfull, Vfull = _rand(rng, B, Hkv, Lc, D), _rand(rng, B, Hkv, Lc, D)
    flags = (rng.random((B, Lc)) < 0.08).astype(np.uint8)
    flags[0, :M] = 1                      # an all-punctuation block
    flags[1, M:2 * M] = 0                 # a block without punctuation
    c = Caches(B, Hkv, Lc)
    for b, plan in enumerate(plans):
        assert sum(plan) == totals[b]
        p0 = 0
        for C in plan:
            c.append(b, b + 1, np.ascontiguousarray(Kfull[b:b + 1, :, p0:p0 + C]),
                     np.ascontiguousarray(Vfull[b:b + 1, :, p0:p0 + C]),
                     np.ascontiguousarray(flags[b:b + 1, p0:p0 + C]), [p0 + C], lam)
            p0 += C
    torch.cuda.synchronize()
    assert phsa.phsa_get_device_status() == 0
    _check(c, Kfull, Vfull, flags, totals, lam)


def test_one_call_over_sequences_at_different_lengths():
    # one chunk length, three sequences whose chunks start at 13, 64 and 100
    rng = np.random.default_rng(11)
    B, Hkv, Lc, lam, C = 3, 2, 64 * 6, 0.5, 150
    starts = [13, 64, 100]
    Kfull, Vfull = _rand(rng, B, Hkv, Lc, D), _rand(rng, B, Hkv, Lc, D)
    flags = (rng.random((B, Lc)) < 0.08).astype(np.uint8)
    c = Caches(B, Hkv, Lc)
    for b, p0 in enumerate(starts):  # the prefixes, one call each
        c.append(b, b + 1, np.ascontiguousarray(Kfull[b:b + 1, :, :p0]),
                 np.ascontiguousarray(Vfull[b:b + 1, :, :p0]),
                 np.ascontiguousarray(flags[b:b + 1, :p0]), [p0], lam)
    kc = np.stack([Kfull[b, :, p0:p0 + C] for b, p0 in enumerate(starts)])
    vc = np.stack([Vfull[b, :, p0:p0 + C] for b, p0 in enumerate(starts)])
    fc = np.stack([flags[b, p0:p0 + C] for b, p0 in enumerate(starts)])
    c.append(0, B, kc, vc, fc, [p0 + C for p0 in starts], lam)
    torch.cuda.synchronize()
    assert phsa.phsa_get_device_status() == 0
    _check(c, Kfull, Vfull, flags, [p0 + C for p0 in starts], lam)


def test_chunk_without_flags_uses_the_cached_mask():
    rng = np.random.default_rng(3)
    B, Hkv, Lc, lam = 2, 1, 64 * 4, 0.3
    Kfull = _rand(rng, B, Hkv, Lc, D)
    flags = (rng.random((B, Lc)) < 0.1).astype(np.uint8)
    c = Caches(B, Hkv, Lc)
    c.mask.copy_(torch.from_numpy(flags))  # the mask already holds the flags
    for p0, C in ((0, 100), (100, 156)):
        kc = np.ascontiguousarray(Kfull[:, :, p0:p0 + C])
        c.append(0, B, kc, kc, None, [p0 + C] * B, lam)
    torch.cuda.synchronize()
    assert phsa.phsa_get_device_status() == 0
    _check(c, Kfull, Kfull, flags, [Lc] * B, lam)


def test_lengths_that_do_not_fit_are_rejected_on_the_device():
    rng = np.random.default_rng(5)
    B, Hkv, Lc, C = 3, 1, 64 * 2, 64
    kc = _rand(rng, B, Hkv, C, D)
    c = Caches(B, Hkv, Lc)
    # sequence 0 fits; 1 is shorter than the chunk; 2 runs past the capacity
    c.append(0, B, kc, kc, np.ones((B, C), np.uint8), [64, 63, Lc + 1], 0.5)
    torch.cuda.synchronize()
    assert phsa.phsa_get_device_status() == -5  # PHSA_ERR_DEVICE_INDEX
    Kh = bf16_bits(c.K)
    assert np.array_equal(Kh[0, :, :64], kc[0])
    assert not Kh[1].any() and not Kh[2].any()
    assert c.mask.cpu().numpy()[1:].sum() == 0


@pytest.mark.parametrize("bm", [16, 32])
def test_chunked_prefill_at_small_block_sizes(bm):
    # chunks shorter than a block, chunks that complete several blocks, and
    # chunk boundaries on and off the block grid
    rng = np.random.default_rng(40 + bm)
    B, Hkv, Lc, lam = 3, 2, 64 * 5, 0.5
    plans = [[1, bm - 1, bm, 3 * bm + 5, 7, 100, 64 * 5 - 5 * bm - 112],
             [bm + 3, 2 * bm - 3, 1, 150], [bm // 2, bm // 2, bm // 2]]
    totals = [sum(p) for p in plans]
    Kfull, Vfull = _rand(rng, B, Hkv, Lc, D), _rand(rng, B, Hkv, Lc, D)
    flags = (rng.random((B, Lc)) < 0.08).astype(np.uint8)
    flags[0, :bm] = 1                     # an all-punctuation block
    flags[1, bm:2 * bm] = 0               # a block without punctuation
    c = Caches(B, Hkv, Lc, bm)
    for b, plan in enumerate(plans):
        p0 = 0
        for C in plan:
            c.append(b, b + 1, np.ascontiguousarray(Kfull[b:b + 1, :, p0:p0 + C]),
                     np.ascontiguousarray(Vfull[b:b + 1, :, p0:p0 + C]),
                     np.ascontiguousarray(flags[b:b + 1, p0:p0 + C]), [p0 + C], lam)
            p0 += C
    torch.cuda.synchronize()
    assert phsa.phsa_get_device_status() == 0
    _check(c, Kfull, Vfull, flags, totals, lam)
