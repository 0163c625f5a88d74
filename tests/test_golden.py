"""Pins taken from numbers the paper prints (fixtures under tests/golden/)."""
import json
import os

import numpy as np

import oracle
from paper_2601_02819_gb300.inputs import f32_to_bf16_bits

GOLD = os.path.join(os.path.dirname(__file__), "golden")


def load(name):
    with open(os.path.join(GOLD, name)) as f:
        return json.load(f)


def test_worked_example_punctuation_mask():
    g = load("worked_example_punct.json")
    mask = oracle.punct_mask(np.array(g["ids"]), g["punct_ids"])
    assert mask.tolist() == g["expected_mask"]


def test_budget_convention_reproduces_the_reported_sparsity():
    g = load("sparsity_32k.json")
    active = g["init_tokens"] + g["local_tokens"] + g["paper_topk"] * g["paper_block_size"]
    assert round(100 * (1 - active / g["L"]), 1) == g["reported_sparsity_percent"]
    # The same active-token count expressed in 64-token blocks, forced blocks included.
    assert g["this_library_topk_blocks_incl_forced"] * g["this_library_block_size"] == active


def test_oracle_budget_gives_that_many_active_tokens_per_query():
    g = load("sparsity_32k.json")
    m, topk = g["this_library_block_size"], g["this_library_topk_blocks_incl_forced"]
    rng = np.random.default_rng(20)
    L = 64 * 40
    Q = f32_to_bf16_bits(rng.standard_normal((1, 2, L, 128)).astype(np.float32))
    Kr = f32_to_bf16_bits(rng.standard_normal((1, 1, L // m, 128)).astype(np.float32))
    idx, cnt = oracle.select_blocks(Q, Kr, L, m, topk, 1, 1, 128 ** -0.5)
    assert np.all(cnt[0, 0, topk - 1:] == topk)
    assert np.all(cnt[0, 0, :topk] == np.arange(1, topk + 1))
    # tokens a query in a full later block attends (its own block contributes up to m)
    assert topk * m == g["init_tokens"] + g["local_tokens"] + g["paper_topk"] * g["paper_block_size"]
