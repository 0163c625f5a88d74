"""Stage (a) on the GPU vs the oracle: representative keys within 1 bf16 ulp."""
import numpy as np
import pytest
import torch

import oracle
from paper_2601_02819_gb300 import inputs
from paper_2601_02819_gb300 import phsa
from parity import bf16_bits, to_dev_bf16, ulp_distance

pytestmark = pytest.mark.gpu


def run(K, mask, lam):
    Kd = to_dev_bf16(K)
    md = torch.from_numpy(np.ascontiguousarray(mask)).cuda()
    out = phsa.phsa_build_block_repr(Kd, md, lam)
    torch.cuda.synchronize()
    return bf16_bits(out)


@pytest.mark.parametrize("name", ["tiny_2k", "prefill_32k", "long_131k_p0", "long_131k_p15"])
def test_repr_matches_oracle(name):
    w = inputs.WORKLOADS[name]
    x = inputs.make_inputs(w)
    got = run(x["K"], x["mask"], w.lam)
    ref = oracle.block_repr(x["K"], x["mask"], w.block_size, w.lam)
    d = ulp_distance(got, ref)
    assert d.max() <= 1, f"max ulp distance {d.max()}"
    assert (d > 0).mean() < 0.01  # rounding-boundary cases only


@pytest.mark.parametrize("lam", [0.0, 0.5, 1.0])
@pytest.mark.parametrize("density", ["none", "all", "sparse"])
def test_repr_lambda_and_density_edges(lam, density):
    rng = np.random.default_rng(5)
    B, Hkv, L = 2, 3, 64 * 9 + 37  # ragged tail: 9 full blocks
    K = inputs.f32_to_bf16_bits(rng.standard_normal((B, Hkv, L, 128)).astype(np.float32))
    if density == "none":
        mask = np.zeros((B, L), np.uint8)
    elif density == "all":
        mask = np.ones((B, L), np.uint8)
    else:
        mask = (rng.random((B, L)) < 0.05).astype(np.uint8)
    got = run(K, mask, lam)
    ref = oracle.block_repr(K, mask, 64, lam)
    assert got.shape == (B, Hkv, 9, 128)
    assert ulp_distance(got, ref).max() <= 1


def test_repr_constant_block_is_exact():
    K = inputs.f32_to_bf16_bits(np.full((1, 2, 256, 128), -0.6875, np.float32))
    mask = np.zeros((1, 256), np.uint8)
    mask[0, 3::17] = 1
    got = run(K, mask, 0.3)
    assert np.all(got == K[0, 0, 0, 0])
