"""Decode on the GPU vs the oracle: one new token per sequence.

Stage-isolated as for prefill: the attention kernel is driven by the oracle's
selection, and the selection by the oracle's representative keys, so each
stage is checked on its own. Selection: bit-exact outside the 1e-3 band on the
aggregate. Attention: max-abs 2e-2, rel-L2 1e-2, lse within 1e-3.
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

D, M = 128, 64
SCALE = D ** -0.5


def _case(seed, B, Hq, Hkv, Lc, lens):
    rng = np.random.default_rng(seed)
    f = lambda *s: inputs.f32_to_bf16_bits(rng.standard_normal(s).astype(np.float32))
    q, K, V = f(B, Hq, D), f(B, Hkv, Lc, D), f(B, Hkv, Lc, D)
    mask = (rng.random((B, Lc)) < 0.06).astype(np.uint8)
    return q, K, V, mask, np.asarray(lens, np.int32)


@pytest.mark.parametrize("Hq,Hkv,topk,n_init,n_local", [
    (4, 2, 6, 1, 1),   # G = 2
    (2, 2, 5, 2, 2),   # G = 1, wider forced set
    (2, 1, 40, 1, 1),  # G = 2, budget above the two-level top-k
])
def test_decode_selection_and_attention_match_oracle(Hq, Hkv, topk, n_init, n_local):
    Lc = 64 * 50 + 8
    lens = [Lc, 64 * 41 + 1, 64 * 23, 64 * 9 + 17, 65, 1]
    q, K, V, mask, lens = _case(Hq * 10 + topk, len(lens), Hq, Hkv, Lc, lens)
    Kr = oracle.block_repr(K, mask, M, 0.5)
    qd, Kd, Vd = to_dev_bf16(q), to_dev_bf16(K), to_dev_bf16(V)
    ld = torch.from_numpy(lens).cuda()
    gi, gc = phsa.phsa_decode_select(qd, to_dev_bf16(Kr), ld, Lc, topk, n_init, n_local)
    oi, oc, oa = oracle.decode_select(q, Kr, lens, Lc, M, topk, n_init, n_local, SCALE,
                                      want_agg=True)
    torch.cuda.synchronize()
    bad, excl, differ, msgs = compare_selection(gi.cpu().numpy().reshape(-1, topk),
                                                gc.cpu().numpy().reshape(-1),
                                                oi.reshape(-1, topk), oc.reshape(-1),
                                                oa.reshape(len(oc.reshape(-1)), -1))
    assert bad == 0, msgs[:5]
    assert differ <= 1
    O, lse = phsa.phsa_decode_attn(qd, Kd, Vd, torch.from_numpy(oi).cuda(),
                                   torch.from_numpy(oc).cuda(), ld)
    Or, lr = oracle.decode_attn(q, K, V, oi, oc, lens, M, SCALE)
    torch.cuda.synchronize()
    assert_close("O", bf16_to_f64(O), Or)
    assert np.abs(lse.cpu().numpy() - lr).max() <= LSE_ABS
    assert phsa.phsa_get_device_status() == 0


def test_decode_empty_sequences_and_bad_lengths():
    Lc = 64 * 4
    q, K, V, mask, lens = _case(3, 3, 4, 2, Lc, [0, 70, Lc + 1])
    Kr = oracle.block_repr(K, mask, M, 0.5)
    ld = torch.from_numpy(lens).cuda()
    phsa.phsa_get_device_status()
    gi, gc = phsa.phsa_decode_select(to_dev_bf16(q), to_dev_bf16(Kr), ld, Lc, 3)
    O, lse = phsa.phsa_decode_attn(to_dev_bf16(q), to_dev_bf16(K), to_dev_bf16(V), gi, gc, ld)
    assert phsa.phsa_get_device_status() == -5  # the length beyond the cache is reported
    gc, gi = gc.cpu().numpy(), gi.cpu().numpy()
    assert np.all(gc[0] == 0) and np.all(gi[0] == -1)
    assert np.all(gc[2] == 0) and np.all(gi[2] == -1)
    O, lse = bf16_to_f64(O), lse.cpu().numpy()
    assert np.all(O[0] == 0) and np.all(np.isneginf(lse[0]))
    assert np.all(O[2] == 0) and np.all(np.isneginf(lse[2]))
    oi, oc = oracle.decode_select(q[1:2], Kr[1:2], lens[1:2], Lc, M, 3, 1, 1, SCALE)
    assert np.array_equal(gi[1], oi[0]) and np.array_equal(gc[1], oc[0])


def test_decode_update_repr_follows_appended_tokens():
    # Caches that grow one token per step: the representative key of a block
    # appears when its last token is appended, and no other row of Krepr moves.
    B, Hkv, Lc = 3, 2, 64 * 6
    rng = np.random.default_rng(7)
    f = lambda *s: inputs.f32_to_bf16_bits(rng.standard_normal(s).astype(np.float32))
    K = f(B, Hkv, Lc, D)
    mask = (rng.random((B, Lc)) < 0.1).astype(np.uint8)
    lens = np.array([64 * 2 + 60, 64 * 3 + 63, 5], np.int32)
    Kd = to_dev_bf16(K)
    md = torch.from_numpy(mask).cuda()
    Krd = phsa.phsa_build_block_repr(Kd, md, 0.5)
    for b in range(B):  # blocks not yet filled hold nothing
        Krd[b, :, lens[b] // M:] = 0
    for step in range(70):
        lens += 1
        for b in range(B):  # append: the new token's key and punctuation flag
            p = lens[b] - 1
            K[b, :, p] = f(Hkv, D)
            mask[b, p] = rng.random() < 0.3
        Kd.copy_(to_dev_bf16(K))
        md.copy_(torch.from_numpy(mask))
        phsa.phsa_decode_update_repr(Kd, md, torch.from_numpy(lens).cuda(), 0.5, Krd)
    torch.cuda.synchronize()
    got = bf16_bits(Krd)
    ref = oracle.block_repr(K, mask, M, 0.5)
    for b in range(B):
        T = lens[b] // M
        d = ulp_distance(got[b, :, :T], ref[b, :, :T])
        assert d.max() <= 1, (b, d.max())
        assert np.all(got[b, :, T:] == 0)
    assert phsa.phsa_get_device_status() == 0


def test_decode_workload_full_size_sampled():
    # 64 sequences x 32768 cached tokens, 16 q / 8 kv heads, topk 14: the whole
    # batch runs on the GPU; sampled (sequence, KV head) units are checked.
    w = inputs.DECODE_WORKLOADS["decode_32k_b64"]
    x = inputs.make_decode_inputs(w, "cuda")
    Krd = phsa.phsa_build_block_repr(x["K"], x["mask_dev"], w.lam)
    phsa.phsa_decode_update_repr(x["K"], x["mask_dev"], x["lens_dev"], w.lam, Krd)
    gi, gc = phsa.phsa_decode_select(x["q"], Krd, x["lens_dev"], w.L, w.topk, w.n_init,
                                     w.n_local)
    O, lse = phsa.phsa_decode_attn(x["q"], x["K"], x["V"], gi, gc, x["lens_dev"])
    torch.cuda.synchronize()
    assert phsa.phsa_get_device_status() == 0
    gi, gc = gi.cpu().numpy(), gc.cpu().numpy()
    rng = np.random.default_rng(5)
    units = [(0, 0), (w.B - 1, w.Hkv - 1)] + [(int(b), int(g)) for b, g in zip(
        rng.integers(0, w.B, 8), rng.integers(0, w.Hkv, 8))]
    agree = 0
    for b, g in units:
        Kbg = bf16_bits(x["K"][b:b + 1, g:g + 1])
        Vbg = bf16_bits(x["V"][b:b + 1, g:g + 1])
        qbg = bf16_bits(x["q"][b:b + 1, 2 * g:2 * g + 2])
        mb = x["mask"][b:b + 1]
        Kr = oracle.block_repr(Kbg, mb, M, w.lam)
        d = ulp_distance(bf16_bits(Krd[b:b + 1, g:g + 1]), Kr)
        assert d.max() <= 1
        lb = x["lens"][b:b + 1]
        oi, oc, oa = oracle.decode_select(qbg, Kr, lb, w.L, M, w.topk, w.n_init, w.n_local,
                                          SCALE, want_agg=True)
        bad, _, differ, msgs = compare_selection(gi[b, g][None], gc[b, g][None], oi.reshape(1, -1),
                                                 oc.reshape(-1), oa.reshape(1, -1))
        assert bad == 0, msgs
        if differ:
            continue  # a near-tie decided the other way: attention inputs differ
        agree += 1
        Or, lr = oracle.decode_attn(qbg, Kbg, Vbg, oi, oc, lb, M, SCALE)
        assert_close(f"O ({b},{g})", bf16_to_f64(O[b:b + 1, 2 * g:2 * g + 2]), Or)
        assert np.abs(lse[b, 2 * g:2 * g + 2].cpu().numpy() - lr[0]).max() <= LSE_ABS
    assert agree >= len(units) - 2


@pytest.mark.parametrize("Hq,Hkv,n_init,n_local,topk", [(4, 2, 1, 1, 6), (2, 2, 2, 3, 9)])
def test_decode_step_equals_the_three_calls(Hq, Hkv, n_init, n_local, topk):
    # The fused step (selection; attention with the refresh of just-filled blocks)
    # must reproduce update_repr -> select -> attn bit for bit, over appends that
    # fill blocks at different steps for different sequences.
    B, Lc = 5, 64 * 12
    rng = np.random.default_rng(11 + Hq)
    f = lambda *s: inputs.f32_to_bf16_bits(rng.standard_normal(s).astype(np.float32))
    K, V = f(B, Hkv, Lc, D), f(B, Hkv, Lc, D)
    mask = (rng.random((B, Lc)) < 0.1).astype(np.uint8)
    lens = np.array([64 * 3 - 2, 64 * 5 - 1, 64 * 2, 1, 64 * 7 - 3], np.int32)
    Kd, Vd, md = to_dev_bf16(K), to_dev_bf16(V), torch.from_numpy(mask).cuda()
    Kr_a = phsa.phsa_build_block_repr(Kd, md, 0.5)
    for b in range(B):  # blocks not yet filled hold nothing
        Kr_a[b, :, lens[b] // M:] = 0
    Kr_b = Kr_a.clone()
    for step in range(6):
        lens += 1
        q = to_dev_bf16(f(B, Hq, D))
        ld = torch.from_numpy(lens).cuda()
        phsa.phsa_decode_update_repr(Kd, md, ld, 0.5, Kr_a)
        ia, ca = phsa.phsa_decode_select(q, Kr_a, ld, Lc, topk, n_init, n_local)
        Oa, la = phsa.phsa_decode_attn(q, Kd, Vd, ia, ca, ld)
        ib, cb, Ob, lb = phsa.phsa_decode_step(q, Kd, Vd, md, ld, 0.5, Kr_b, topk, n_init, n_local)
        torch.cuda.synchronize()
        assert torch.equal(ia, ib) and torch.equal(ca, cb), step
        assert torch.equal(Oa.view(torch.int16), Ob.view(torch.int16)), step
        assert torch.equal(la, lb), step
        assert torch.equal(Kr_a.view(torch.int16), Kr_b.view(torch.int16)), step
    assert phsa.phsa_get_device_status() == 0


@pytest.mark.parametrize("Hq,Hkv", [(4, 2), (2, 2)])
def test_decode_max_logit_rule_matches_oracle(Hq, Hkv):
    Lc = 64 * 50 + 8
    lens = [Lc, 64 * 41 + 1, 64 * 23, 64 * 9 + 17, 65, 1]
    q, K, V, mask, lens = _case(77 + Hq, len(lens), Hq, Hkv, Lc, lens)
    Kr = oracle.block_repr(K, mask, M, 0.5)
    ld = torch.from_numpy(lens).cuda()
    gi, gc = phsa.phsa_decode_select(to_dev_bf16(q), to_dev_bf16(Kr), ld, Lc, 6, 2, 2,
                                     aggregation="max_logit")
    oi, oc, oa = oracle.decode_select(q, Kr, lens, Lc, M, 6, 2, 2, SCALE, want_agg=True,
                                      aggregation="max_logit")
    torch.cuda.synchronize()
    bad, excl, differ, msgs = compare_selection(gi.cpu().numpy().reshape(-1, 6),
                                                gc.cpu().numpy().reshape(-1),
                                                oi.reshape(-1, 6), oc.reshape(-1),
                                                oa.reshape(len(oc.reshape(-1)), -1))
    assert bad == 0, msgs[:5]
    assert differ <= 1
    # the fused step takes the same rule
    Kd, Vd, md = to_dev_bf16(K), to_dev_bf16(V), torch.from_numpy(mask).cuda()
    Krd = to_dev_bf16(Kr)
    si, sc, O, lse = phsa.phsa_decode_step(to_dev_bf16(q), Kd, Vd, md, ld, 0.5, Krd, 6, 2, 2,
                                           aggregation="max_logit")
    torch.cuda.synchronize()
    assert torch.equal(si, gi) and torch.equal(sc, gc)
    assert phsa.phsa_get_device_status() == 0
