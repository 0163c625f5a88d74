"""Serving-side entry points on the GPU vs the oracle: the punctuation
indicator (Eq. 4-5) and the append of each sequence's new token to the caches,
then a token-by-token decode loop (append, then the fused decode step) that
must leave the representative keys equal to the oracle's over the grown caches.

The indicator is integer work: bit-exact. The append is a data move: the caches
must equal the numpy assignment of the new rows, byte for byte.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2601_02819_gb300 import inputs, phsa
from parity import (LSE_ABS, assert_close, bf16_bits, bf16_to_f64, compare_selection,
                    to_dev_bf16, ulp_distance)

pytestmark = pytest.mark.gpu

D, M = 128, 64
SCALE = D ** -0.5
I32 = np.iinfo(np.int32)


def _mask(ids, pset):
    got = phsa.phsa_punct_mask(torch.from_numpy(np.ascontiguousarray(ids)).cuda(),
                               torch.from_numpy(np.ascontiguousarray(pset, np.int32)).cuda())
    return got.cpu().numpy()


@pytest.mark.parametrize("name", ["prefill_32k", "train_8k_x4", "long_131k_p15"])
def test_punct_mask_on_workload_ids_matches_oracle(name):
    # the token ids of the workload's punctuation recipe (its full B x L)
    w = inputs.WORKLOADS[name]
    rng = np.random.default_rng(w.seed)
    pset = inputs.punct_id_set(rng)
    ids = inputs.draw_token_ids(rng, w.B, w.L, w.punct, w.punct_gap, pset)
    got = _mask(ids, pset)
    assert got.shape == ids.shape
    assert np.array_equal(got, oracle.punct_mask(ids, pset))
    assert got.sum() > 0


@pytest.mark.parametrize("n_punct,n", [(0, 1000), (1, 1), (37, 100003), (4096, 70001)])
def test_punct_mask_set_sizes_and_extreme_ids(n_punct, n):
    rng = np.random.default_rng(n_punct + n)
    pset = rng.integers(-50000, 50000, size=n_punct).astype(np.int32)
    if n_punct >= 4:  # duplicates and the int32 extremes inside the set
        pset[:4] = [I32.max, I32.min, pset[5 % n_punct], -1]
    ids = rng.integers(-50000, 50000, size=n).astype(np.int32)
    hit = rng.random(n) < 0.3
    if n_punct:
        ids[hit] = pset[rng.integers(0, n_punct, size=int(hit.sum()))]
    ids[: min(n, 3)] = [I32.max, I32.min, 0][: min(n, 3)]
    got = _mask(ids, pset)
    assert np.array_equal(got, oracle.punct_mask(ids, pset))


def test_punct_mask_int_max_outside_the_set_is_not_punctuation():
    # INT_MAX pads the sorted set on the device; it must not match unless it is in P.
    pset = np.array([3, 9, 1], np.int32)  # padded to 4 entries
    ids = np.array([I32.max, 3, 4, 9, 1, I32.max - 1], np.int32)
    assert list(_mask(ids, pset)) == [0, 1, 0, 1, 1, 0]
    assert list(_mask(ids, np.append(pset, I32.max))) == [1, 1, 0, 1, 1, 0]


def test_punct_mask_rejects_sets_above_4096():
    ids = torch.zeros(8, dtype=torch.int32, device="cuda")
    with pytest.raises(phsa.PhsaError):
        phsa.phsa_punct_mask(ids, torch.zeros(4097, dtype=torch.int32, device="cuda"))


def test_decode_append_writes_row_len_minus_one():
    B, Hkv, Lc = 6, 3, 64 * 3 + 5
    rng = np.random.default_rng(2)
    f = lambda *s: inputs.f32_to_bf16_bits(rng.standard_normal(s).astype(np.float32))
    K, V = f(B, Hkv, Lc, D), f(B, Hkv, Lc, D)
    mask = (rng.random((B, Lc)) < 0.1).astype(np.uint8)
    kn, vn = f(B, Hkv, D), f(B, Hkv, D)
    flag = np.array([1, 0, 2, 1, 1, 0], np.uint8)  # any nonzero flag is punctuation
    lens = np.array([1, Lc, 0, 64, Lc + 1, 77], np.int32)  # 0: nothing; Lc + 1: error
    Kd, Vd, md = to_dev_bf16(K), to_dev_bf16(V), torch.from_numpy(mask).cuda()
    phsa.phsa_get_device_status()
    phsa.phsa_decode_append(to_dev_bf16(kn), to_dev_bf16(vn), torch.from_numpy(lens).cuda(), Kd,
                            Vd, torch.from_numpy(flag).cuda(), md)
    assert phsa.phsa_get_device_status() == -5  # the length beyond the cache
    for b in range(B):
        if 1 <= lens[b] <= Lc:
            p = lens[b] - 1
            K[b, :, p], V[b, :, p], mask[b, p] = kn[b], vn[b], flag[b] != 0
    assert np.array_equal(bf16_bits(Kd), K)
    assert np.array_equal(bf16_bits(Vd), V)
    assert np.array_equal(md.cpu().numpy(), mask)
    # without flags the mask is left as it is
    lens2 = np.array([2, 3, 4, 5, 6, 7], np.int32)
    phsa.phsa_decode_append(to_dev_bf16(vn), to_dev_bf16(kn), torch.from_numpy(lens2).cuda(), Kd,
                            Vd)
    for b in range(B):
        K[b, :, lens2[b] - 1], V[b, :, lens2[b] - 1] = vn[b], kn[b]
    torch.cuda.synchronize()
    assert np.array_equal(bf16_bits(Kd), K) and np.array_equal(bf16_bits(Vd), V)
    assert np.array_equal(md.cpu().numpy(), mask)
    assert phsa.phsa_get_device_status() == 0


@pytest.mark.parametrize("Hq,Hkv", [(4, 2), (2, 2)])
def test_decode_loop_append_then_step_matches_oracle(Hq, Hkv):
    # Token-by-token generation: ids -> indicator on the device, append k, v and
    # the flag, then one fused decode step. After 80 steps (every sequence
    # fills at least one block) the representative keys equal the oracle's over
    # the grown caches, and the last step's selection and attention match it.
    B, Lc, topk, n_init, n_local, lam = 4, 64 * 10, 6, 1, 2, 0.5
    rng = np.random.default_rng(40 + Hq)
    f = lambda *s: inputs.f32_to_bf16_bits(rng.standard_normal(s).astype(np.float32))
    pset = inputs.punct_id_set(rng)
    K, V = np.zeros((B, Hkv, Lc, D), np.uint16), np.zeros((B, Hkv, Lc, D), np.uint16)
    mask = np.zeros((B, Lc), np.uint8)
    lens = np.array([64 * 2 + 3, 64 * 5 - 1, 64 * 7 + 40, 10], np.int32)
    for b in range(B):  # the prompts
        K[b, :, :lens[b]], V[b, :, :lens[b]] = f(Hkv, lens[b], D), f(Hkv, lens[b], D)
        ids = inputs.draw_token_ids(rng, 1, int(lens[b]), "uniform8", (9, 25), pset)
        mask[b, :lens[b]] = oracle.punct_mask(ids, pset)[0]
    Kd, Vd, md = to_dev_bf16(K), to_dev_bf16(V), torch.from_numpy(mask).cuda()
    Krd = phsa.phsa_build_block_repr(Kd, md, lam)
    for b in range(B):  # blocks not yet filled hold nothing
        Krd[b, :, lens[b] // M:] = 0
    psd = torch.from_numpy(pset).cuda()
    for step in range(80):
        lens += 1
        kn, vn, q = f(B, Hkv, D), f(B, Hkv, D), f(B, Hq, D)
        ids = inputs.draw_token_ids(rng, B, 1, "uniform8", (9, 25), pset)[:, 0]
        flag = phsa.phsa_punct_mask(torch.from_numpy(ids).cuda(), psd)
        ld = torch.from_numpy(lens).cuda()
        phsa.phsa_decode_append(to_dev_bf16(kn), to_dev_bf16(vn), ld, Kd, Vd, flag, md)
        qd = to_dev_bf16(q)
        gi, gc, O, lse = phsa.phsa_decode_step(qd, Kd, Vd, md, ld, lam, Krd, topk, n_init,
                                               n_local)
        for b in range(B):
            K[b, :, lens[b] - 1], V[b, :, lens[b] - 1] = kn[b], vn[b]
            mask[b, lens[b] - 1] = ids[b] in pset
    torch.cuda.synchronize()
    assert phsa.phsa_get_device_status() == 0
    assert np.array_equal(bf16_bits(Kd), K) and np.array_equal(md.cpu().numpy(), mask)
    Kr = oracle.block_repr(K, mask, M, lam)
    got = bf16_bits(Krd)
    for b in range(B):
        T = lens[b] // M
        assert ulp_distance(got[b, :, :T], Kr[b, :, :T]).max() <= 1
        assert np.all(got[b, :, T:] == 0)
    oi, oc, oa = oracle.decode_select(q, Kr, lens, Lc, M, topk, n_init, n_local, SCALE,
                                      want_agg=True)
    bad, _, differ, msgs = compare_selection(gi.cpu().numpy().reshape(-1, topk),
                                             gc.cpu().numpy().reshape(-1), oi.reshape(-1, topk),
                                             oc.reshape(-1), oa.reshape(len(oc.reshape(-1)), -1))
    assert bad == 0, msgs[:5]
    if differ == 0:
        Or, lr = oracle.decode_attn(q, K, V, oi, oc, lens, M, SCALE)
        assert_close("O", bf16_to_f64(O), Or)
        assert np.abs(lse.cpu().numpy() - lr).max() <= LSE_ABS
