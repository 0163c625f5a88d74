"""Decode at block sizes m = 16 and 32 on the GPU vs the oracle.

The decode attention packs 64 / m selected blocks into one 64-row ring slot and
the refresh of a just-filled block reads it from its place in the slot; the
selection scores blocks of m. Checked as at m = 64: each stage on the oracle's
inputs (selection on the oracle's representative keys, attention on the
oracle's lists), the fused step against the three calls bit for bit, the
incremental refresh against the oracle, and the paper's 32k block setting
(blocks of 16, 8 initial, 32 local and 16 Top-K blocks) at full size on
sampled units. Tolerances as in parity.py.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2601_02819_gb300 import inputs
from paper_2601_02819_gb300 import phsa
from parity import (LSE_ABS, assert_close, bf16_bits, bf16_to_f64, compare_selection,
                    to_dev_bf16, ulp_distance)

pytestmark = pytest.mark.gpu

D = 128
SCALE = D ** -0.5


def _rand(rng, *s):
    return inputs.f32_to_bf16_bits(rng.standard_normal(s).astype(np.float32))


def _case(seed, B, Hq, Hkv, Lc):
    rng = np.random.default_rng(seed)
    q, K, V = _rand(rng, B, Hq, D), _rand(rng, B, Hkv, Lc, D), _rand(rng, B, Hkv, Lc, D)
    mask = (rng.random((B, Lc)) < 0.06).astype(np.uint8)
    return q, K, V, mask


def _select_and_attend(bm, q, K, V, mask, lens, topk, n_init, n_local, agg):
    Lc = K.shape[2]
    Kr = oracle.block_repr(K, mask, bm, 0.5)
    qd, Kd, Vd = to_dev_bf16(q), to_dev_bf16(K), to_dev_bf16(V)
    ld = torch.from_numpy(lens).cuda()
    gi, gc = phsa.phsa_decode_select(qd, to_dev_bf16(Kr), ld, Lc, topk, n_init, n_local,
                                     aggregation=agg, block_size=bm)
    oi, oc, oa = oracle.decode_select(q, Kr, lens, Lc, bm, topk, n_init, n_local, SCALE,
                                      want_agg=True, aggregation=agg)
    torch.cuda.synchronize()
    bad, _, differ, msgs = compare_selection(gi.cpu().numpy().reshape(-1, topk),
                                             gc.cpu().numpy().reshape(-1),
                                             oi.reshape(-1, topk), oc.reshape(-1),
                                             oa.reshape(len(oc.reshape(-1)), -1))
    assert bad == 0, msgs[:5]
    assert differ <= 1
    O, lse = phsa.phsa_decode_attn(qd, Kd, Vd, torch.from_numpy(oi).cuda(),
                                   torch.from_numpy(oc).cuda(), ld, block_size=bm)
    Or, lr = oracle.decode_attn(q, K, V, oi, oc, lens, bm, SCALE)
    torch.cuda.synchronize()
    assert_close("O", bf16_to_f64(O), Or)
    assert np.abs(lse.cpu().numpy() - lr).max() <= LSE_ABS
    assert phsa.phsa_get_device_status() == 0


@pytest.mark.parametrize("bm", [16, 32])
@pytest.mark.parametrize("Hq,Hkv,topk,n_init,n_local,agg", [
    (4, 2, 12, 2, 4, "softmax_sum"),   # G = 2
    (2, 2, 10, 1, 2, "softmax_sum"),   # G = 1
    (4, 2, 12, 2, 4, "max_logit"),
    (2, 1, 70, 1, 1, "softmax_sum"),   # a budget of more than 32 scored blocks
])
def test_decode_selection_and_attention_match_oracle(bm, Hq, Hkv, topk, n_init, n_local, agg):
    # lengths on, just past and just before block boundaries, one of a single
    # token, and counts that leave the last ring slot part-filled
    Lc = 64 * 50 + 8
    lens = np.array([Lc, 64 * 41 + 1, 64 * 23, 64 * 9 + 17, 65, 1, bm * 7, bm * 3 + bm // 2],
                    np.int32)
    q, K, V, mask = _case(Hq * 10 + topk + bm, len(lens), Hq, Hkv, Lc)
    _select_and_attend(bm, q, K, V, mask, lens, topk, n_init, n_local, agg)


@pytest.mark.parametrize("bm", [16, 32])
@pytest.mark.parametrize("topk", [24, 60])
def test_decode_long_candidate_lists(bm, topk):
    # more than 512 candidates: the selection's top-k takes them 512 at a time
    # in registers (18 picks), or in rounds over shared memory (54 picks)
    Lc = 16 * 1400
    lens = np.array([Lc, Lc - 5, Lc // 2 + 3], np.int32)
    q, K, V, mask = _case(91 + bm + topk, 3, 4, 2, Lc)
    _select_and_attend(bm, q, K, V, mask, lens, topk, 2, 4, "softmax_sum")


@pytest.mark.parametrize("bm", [16, 32])
def test_decode_update_repr_follows_appended_tokens(bm):
    # Caches that grow one token per step: the representative key of a block
    # appears when its last token is appended, and no other row of Krepr moves.
    B, Hkv, Lc = 3, 2, 64 * 6
    rng = np.random.default_rng(7 + bm)
    K = _rand(rng, B, Hkv, Lc, D)
    mask = (rng.random((B, Lc)) < 0.1).astype(np.uint8)
    lens = np.array([bm * 5 + bm - 4, bm * 3 + bm - 1, 5], np.int32)
    Kd = to_dev_bf16(K)
    md = torch.from_numpy(mask).cuda()
    Krd = phsa.phsa_build_block_repr(Kd, md, 0.5, block_size=bm)
    for b in range(B):  # blocks not yet filled hold nothing
        Krd[b, :, lens[b] // bm:] = 0
    for step in range(2 * bm + 6):
        lens += 1
        for b in range(B):  # append: the new token's key and punctuation flag
            p = lens[b] - 1
            K[b, :, p] = _rand(rng, Hkv, D)
            mask[b, p] = rng.random() < 0.3
        Kd.copy_(to_dev_bf16(K))
        md.copy_(torch.from_numpy(mask))
        phsa.phsa_decode_update_repr(Kd, md, torch.from_numpy(lens).cuda(), 0.5, Krd,
                                     block_size=bm)
    torch.cuda.synchronize()
    got = bf16_bits(Krd)
    ref = oracle.block_repr(K, mask, bm, 0.5)
    for b in range(B):
        T = lens[b] // bm
        d = ulp_distance(got[b, :, :T], ref[b, :, :T])
        assert d.max() <= 1, (b, d.max())
        assert np.all(got[b, :, T:] == 0)
    assert phsa.phsa_get_device_status() == 0


@pytest.mark.parametrize("bm", [16, 32])
@pytest.mark.parametrize("Hq,Hkv,n_init,n_local,topk", [(4, 2, 1, 2, 10), (2, 2, 2, 3, 12)])
def test_decode_step_equals_the_three_calls(bm, Hq, Hkv, n_init, n_local, topk):
    # The fused step (selection; attention with the refresh of just-filled
    # blocks, read from their place in a ring slot of 64 / m blocks) must
    # reproduce update_repr -> select -> attn bit for bit, over appends that
    # fill blocks at different steps for different sequences.
    B, Lc = 5, 64 * 12
    rng = np.random.default_rng(11 + Hq + bm)
    K, V = _rand(rng, B, Hkv, Lc, D), _rand(rng, B, Hkv, Lc, D)
    mask = (rng.random((B, Lc)) < 0.1).astype(np.uint8)
    lens = np.array([bm * 3 - 2, bm * 5 - 1, bm * 2, 1, bm * 17 - 3], np.int32)
    Kd, Vd, md = to_dev_bf16(K), to_dev_bf16(V), torch.from_numpy(mask).cuda()
    Kr_a = phsa.phsa_build_block_repr(Kd, md, 0.5, block_size=bm)
    for b in range(B):  # blocks not yet filled hold nothing
        Kr_a[b, :, lens[b] // bm:] = 0
    Kr_b = Kr_a.clone()
    for step in range(bm + 4):
        lens += 1
        q = to_dev_bf16(_rand(rng, B, Hq, D))
        ld = torch.from_numpy(lens).cuda()
        phsa.phsa_decode_update_repr(Kd, md, ld, 0.5, Kr_a, block_size=bm)
        ia, ca = phsa.phsa_decode_select(q, Kr_a, ld, Lc, topk, n_init, n_local, block_size=bm)
        Oa, la = phsa.phsa_decode_attn(q, Kd, Vd, ia, ca, ld, block_size=bm)
        ib, cb, Ob, lb = phsa.phsa_decode_step(q, Kd, Vd, md, ld, 0.5, Kr_b, topk, n_init,
                                               n_local, block_size=bm)
        torch.cuda.synchronize()
        assert torch.equal(ia, ib) and torch.equal(ca, cb), step
        assert torch.equal(Oa.view(torch.int16), Ob.view(torch.int16)), step
        assert torch.equal(la, lb), step
        assert torch.equal(Kr_a.view(torch.int16), Kr_b.view(torch.int16)), step
    assert phsa.phsa_get_device_status() == 0


def test_decode_workload_m16_full_size_sampled():
    # 64 sequences x 32768 cached tokens, 16 q / 8 kv heads, blocks of 16 with
    # 8 initial, 32 local and 16 selected blocks (Top-K 56): the whole batch
    # runs on the GPU through the fused step; sampled units are checked.
    w = inputs.DECODE_WORKLOADS["decode_32k_b64_m16"]
    bm = w.block_size
    x = inputs.make_decode_inputs(w, "cuda")
    Krd = phsa.phsa_build_block_repr(x["K"], x["mask_dev"], w.lam, block_size=bm)
    gi, gc, O, lse = phsa.phsa_decode_step(x["q"], x["K"], x["V"], x["mask_dev"], x["lens_dev"],
                                           w.lam, Krd, w.topk, w.n_init, w.n_local,
                                           block_size=bm)
    torch.cuda.synchronize()
    assert phsa.phsa_get_device_status() == 0
    gi, gc = gi.cpu().numpy(), gc.cpu().numpy()
    rng = np.random.default_rng(5)
    units = [(0, 0), (w.B - 1, w.Hkv - 1)] + [(int(b), int(g)) for b, g in zip(
        rng.integers(0, w.B, 6), rng.integers(0, w.Hkv, 6))]
    agree = 0
    for b, g in units:
        Kbg = bf16_bits(x["K"][b:b + 1, g:g + 1])
        Vbg = bf16_bits(x["V"][b:b + 1, g:g + 1])
        qbg = bf16_bits(x["q"][b:b + 1, 2 * g:2 * g + 2])
        mb = x["mask"][b:b + 1]
        Kr = oracle.block_repr(Kbg, mb, bm, w.lam)
        assert ulp_distance(bf16_bits(Krd[b:b + 1, g:g + 1]), Kr).max() <= 1
        lb = x["lens"][b:b + 1]
        oi, oc, oa = oracle.decode_select(qbg, Kr, lb, w.L, bm, w.topk, w.n_init, w.n_local,
                                          SCALE, want_agg=True)
        bad, _, differ, msgs = compare_selection(gi[b, g][None], gc[b, g][None],
                                                 oi.reshape(1, -1), oc.reshape(-1),
                                                 oa.reshape(1, -1))
        assert bad == 0, msgs
        if differ:
            continue  # a near-tie decided the other way: attention inputs differ
        agree += 1
        Or, lr = oracle.decode_attn(qbg, Kbg, Vbg, oi, oc, lb, bm, SCALE)
        assert_close(f"O ({b},{g})", bf16_to_f64(O[b:b + 1, 2 * g:2 * g + 2]), Or)
        assert np.abs(lse[b, 2 * g:2 * g + 2].cpu().numpy() - lr[0]).max() <= LSE_ABS
    assert agree >= len(units) - 2
