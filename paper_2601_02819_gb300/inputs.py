"""Seeded synthetic inputs for the PHSA sparse-attention hot path.

This module only *draws* inputs. It holds none of the method's arithmetic: no
block representation, no scoring, no attention. Both the CUDA path and the CPU
oracle are fed from here, so it must stay free of either.

Workloads stand in for the paper's settings (Section 4.1: Qwen3-0.6B-class
attention, 16 query heads sharing 8 KV heads, head dim 128, contexts of 4k-32k
tokens and beyond) and for its long-context evaluations (NIAH, LongBench),
whose data is not used. Values are N(0,1) draws rounded to bf16; token ids are
drawn from a 32768-id vocabulary in which 64 ids play the role of the
punctuation set P of Eq. 4-5, and the punctuation indicator I(x in P) of Eq. 7
is returned as a uint8 mask.

bf16 tensors are carried as numpy ``uint16`` bit patterns (round-to-nearest-
even from float32), which both sides decode exactly.
"""
from __future__ import annotations

import dataclasses
import numpy as np

VOCAB = 32768
N_PUNCT_IDS = 64


@dataclasses.dataclass(frozen=True)
class Workload:
    """Shape and selection budget of one synthetic workload.

    ``topk`` is the total number of KV blocks each (query block, KV head)
    attends, forced blocks included; ``n_init``/``n_local`` are the forced
    initial and local blocks (Algorithm 1 inputs n_init and w, in blocks).
    """
    name: str
    B: int
    L: int
    Hq: int
    Hkv: int
    D: int = 128
    block_size: int = 64
    topk: int = 8
    n_init: int = 1
    n_local: int = 1
    lam: float = 0.5
    punct: str = "uniform8"      # "uniform8" | "sentence" | "none"
    punct_gap: tuple = (9, 25)   # sentence-like gap range (tokens) between punctuation
    per_head_scale: bool = False
    seed: int = 1234

    @property
    def G(self) -> int:
        return self.Hq // self.Hkv

    @property
    def T(self) -> int:
        return self.L // self.block_size

    @property
    def NQB(self) -> int:
        return -(-self.L // self.block_size)

    @property
    def sm_scale(self) -> float:
        return 1.0 / float(np.sqrt(self.D))


# The named workloads. Sizes follow the paper's model class (Qwen3-0.6B: 16 q
# heads / 8 kv heads / d=128) and context lengths (4k-32k, plus 131k).
WORKLOADS = {
    "tiny_2k": Workload("tiny_2k", B=1, L=2048, Hq=2, Hkv=1, topk=8,
                        punct="uniform8", seed=1234 + 1),
    "prefill_32k": Workload("prefill_32k", B=1, L=32768, Hq=16, Hkv=8, topk=14,
                            punct="sentence", punct_gap=(9, 25),
                            per_head_scale=True, seed=1234 + 2),
    # The paper's 32k setting as printed: blocks of 16 tokens, 128 initial and
    # 512 local tokens (8 and 32 blocks) and 16 Top-K blocks; the same tensors
    # as prefill_32k (same seed).
    "prefill_32k_m16": Workload("prefill_32k_m16", B=1, L=32768, Hq=16, Hkv=8, block_size=16,
                                topk=56, n_init=8, n_local=32, punct="sentence",
                                punct_gap=(9, 25), per_head_scale=True, seed=1234 + 2),
    "train_8k_x4": Workload("train_8k_x4", B=4, L=8192, Hq=16, Hkv=8, topk=8,
                            punct="sentence", punct_gap=(9, 25), seed=1234 + 3),
    "long_131k_p0": Workload("long_131k_p0", B=1, L=131072, Hq=16, Hkv=8, topk=32,
                             punct="none", seed=1234 + 5),
    "long_131k_p3": Workload("long_131k_p3", B=1, L=131072, Hq=16, Hkv=8, topk=32,
                             punct="sentence", punct_gap=(17, 50), seed=1234 + 5),
    "long_131k_p15": Workload("long_131k_p15", B=1, L=131072, Hq=16, Hkv=8, topk=32,
                              punct="sentence", punct_gap=(4, 10), seed=1234 + 5),
}


# Decode: B sequences, each with a cache of L tokens whose last token (position
# L - 1) is the new one, the query of that step.
DECODE_WORKLOADS = {
    "decode_32k_b64": Workload("decode_32k_b64", B=64, L=32768, Hq=16, Hkv=8, topk=14,
                               punct="sentence", punct_gap=(9, 25), seed=1234 + 4),
    # the paper's 32k block setting (blocks of 16; 8 initial, 32 local and 16
    # Top-K blocks) on the same caches
    "decode_32k_b64_m16": Workload("decode_32k_b64_m16", B=64, L=32768, Hq=16, Hkv=8,
                                   block_size=16, topk=56, n_init=8, n_local=32,
                                   punct="sentence", punct_gap=(9, 25), seed=1234 + 4),
}


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round float32 values to bf16 (nearest, ties to even); return uint16 bits."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    rounded = u + np.uint32(0x7FFF) + ((u >> np.uint32(16)) & np.uint32(1))
    return (rounded >> np.uint32(16)).astype(np.uint16)


def bf16_bits_to_f32(h: np.ndarray) -> np.ndarray:
    """Exact decode of bf16 bit patterns to float32."""
    return (np.asarray(h, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


def punct_id_set(rng: np.random.Generator) -> np.ndarray:
    """The stand-in punctuation set P: 64 distinct ids of the vocabulary."""
    return np.sort(rng.choice(VOCAB, size=N_PUNCT_IDS, replace=False)).astype(np.int32)


def draw_token_ids(rng: np.random.Generator, B: int, L: int, punct: str,
                   gap: tuple, pset: np.ndarray) -> np.ndarray:
    """Token ids [B, L] int32 with the requested punctuation placement.

    ``uniform8``: each token is punctuation with probability 0.08.
    ``sentence``: punctuation every g tokens, g uniform on [gap[0], gap[1]].
    ``none``: no punctuation at all.
    """
    is_p = np.zeros((B, L), dtype=bool)
    if punct == "uniform8":
        is_p = rng.random((B, L)) < 0.08
    elif punct == "sentence":
        lo, hi = gap
        for b in range(B):
            n_gaps = L // lo + 2
            gaps = rng.integers(lo, hi + 1, size=n_gaps)
            pos = np.cumsum(gaps) - 1
            pos = pos[pos < L]
            is_p[b, pos] = True
    elif punct != "none":
        raise ValueError(f"unknown punctuation placement {punct!r}")
    others = np.setdiff1d(np.arange(VOCAB, dtype=np.int32), pset)
    ids = others[rng.integers(0, others.size, size=(B, L))]
    ids[is_p] = pset[rng.integers(0, pset.size, size=int(is_p.sum()))]
    return ids.astype(np.int32)


def _normal_bf16(rng: np.random.Generator, shape, head_axis: int | None,
                 per_head_scale: bool) -> np.ndarray:
    x = rng.standard_normal(size=shape, dtype=np.float32)
    if per_head_scale:
        s = rng.uniform(0.5, 2.0, size=shape[head_axis]).astype(np.float32)
        bshape = [1] * len(shape)
        bshape[head_axis] = shape[head_axis]
        x *= s.reshape(bshape)
    return f32_to_bf16_bits(x)


def make_inputs(w: Workload, with_grad: bool = False, seed: int | None = None) -> dict:
    """Draw one batch for workload ``w``.

    Returns a dict of numpy arrays: Q [B,Hq,L,D], K/V [B,Hkv,L,D] (uint16 bf16
    bits), ids [B,L] int32, punct_ids [64] int32, mask [B,L] uint8 (1 where the
    token id is in the punctuation set), and dO [B,Hq,L,D] when ``with_grad``.
    """
    rng = np.random.default_rng(w.seed if seed is None else seed)
    pset = punct_id_set(rng)
    ids = draw_token_ids(rng, w.B, w.L, w.punct, w.punct_gap, pset)
    mask = np.isin(ids, pset).astype(np.uint8)
    out = {
        "Q": _normal_bf16(rng, (w.B, w.Hq, w.L, w.D), 1, w.per_head_scale),
        "K": _normal_bf16(rng, (w.B, w.Hkv, w.L, w.D), 1, w.per_head_scale),
        "V": _normal_bf16(rng, (w.B, w.Hkv, w.L, w.D), 1, w.per_head_scale),
        "ids": ids,
        "punct_ids": pset,
        "mask": mask,
    }
    if with_grad:
        out["dO"] = f32_to_bf16_bits(rng.standard_normal(size=(w.B, w.Hq, w.L, w.D),
                                                          dtype=np.float32))
    return out


def make_decode_inputs(w: Workload, device, seed: int | None = None) -> dict:
    """Draw one decode batch for workload ``w`` directly on a torch ``device``.

    The caches are too large to draw on the host (4.3 GB each at 64 x 32k), so
    the N(0,1) values come from torch's seeded generator on that device, in
    float32, rounded to bf16 (nearest, ties to even). Returns q [B,Hq,D], K, V
    [B,Hkv,L,D] bf16 tensors on the device; mask [B,L] as numpy uint8 and as a
    device tensor (mask_dev); lens [B] int32 (numpy and lens_dev), all equal to L.
    """
    import torch

    s = w.seed if seed is None else seed
    rng = np.random.default_rng(s)
    pset = punct_id_set(rng)
    ids = draw_token_ids(rng, w.B, w.L, w.punct, w.punct_gap, pset)
    mask = np.isin(ids, pset).astype(np.uint8)
    gen = torch.Generator(device=device)
    gen.manual_seed(s)

    def normal(shape):
        out = torch.empty(shape, dtype=torch.bfloat16, device=device)
        for b in range(shape[0]):  # one sequence at a time keeps the fp32 draw small
            out[b] = torch.randn(shape[1:], generator=gen, device=device,
                                 dtype=torch.float32).to(torch.bfloat16)
        return out

    K = normal((w.B, w.Hkv, w.L, w.D))
    V = normal((w.B, w.Hkv, w.L, w.D))
    q = normal((w.B, w.Hq, w.D))
    lens = np.full((w.B,), w.L, dtype=np.int32)
    return {"q": q, "K": K, "V": V, "mask": mask, "ids": ids, "punct_ids": pset,
            "mask_dev": torch.from_numpy(mask).to(device), "lens": lens,
            "lens_dev": torch.from_numpy(lens).to(device)}


def random_block_lists(rng: np.random.Generator, B: int, Hkv: int, NQB: int,
                       topk: int) -> tuple[np.ndarray, np.ndarray]:
    """Random valid block lists for the attention stage alone: per (b, g, qb)
    the first block, the query's own block and random earlier blocks,
    min(topk, qb + 1) in all, ascending and -1 padded. Drawn, not selected:
    feeding the same lists to both sides isolates the attention kernels.
    Returns (block_idx [B, Hkv, NQB, topk] int32, block_cnt [B, Hkv, NQB] int32)."""
    idx = np.full((B, Hkv, NQB, topk), -1, np.int32)
    cnt = np.zeros((B, Hkv, NQB), np.int32)
    for b in range(B):
        for g in range(Hkv):
            for qb in range(NQB):
                n = min(topk, qb + 1)
                s = {0, qb}
                if n > len(s):
                    s |= set((rng.choice(qb - 1, size=n - len(s), replace=False) + 1).tolist())
                s = sorted(s)
                idx[b, g, qb, :len(s)] = s
                cnt[b, g, qb] = len(s)
    return idx, cnt


def custom(name: str = "custom", **kw) -> Workload:
    """A workload with explicit sizes (used by tests for ragged/edge shapes)."""
    return Workload(name=name, **kw)
