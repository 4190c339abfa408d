"""Pins for the oracle's random numbers and bf16 rounding.

* Philox4x32-10 against the published known-answer vectors
  (tests/golden/philox4x32_10_kat.txt).
* The uniform map u = ((x >> 9) + 0.5) 2^-23 is exact in fp32 and strictly
  inside (0, 1); the Gumbel transform is -log(-log u).
* bf16 rounding against torch's own float32 -> bfloat16 conversion (a library
  routine), including halfway cases (ties to even).
"""
import os

import numpy as np
import pytest

import oracle as O

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "philox4x32_10_kat.txt")


def _kat():
    rows = []
    for line in open(GOLDEN):
        if line.startswith("#") or not line.strip():
            continue
        v = [int(t, 16) for t in line.split()]
        rows.append((v[0:4], v[4:6], v[6:10]))
    return rows


@pytest.mark.parametrize("ctr,key,expect", _kat())
def test_philox_known_answers(ctr, key, expect):
    assert O.philox(ctr, key).tolist() == expect


def test_uniform_layout_and_range():
    seed = 0x1234_5678_9ABC_DEF0
    for index in (0, 1, 2, 3, 4, 77, 151935):
        for pos in (0, 5):
            out = O.philox([index >> 2, pos, 1, 9], [seed & 0xFFFFFFFF, seed >> 32])
            x = int(out[index & 3])
            u = O.uniform(seed, index, pos, 1, 9)
            assert u == ((x >> 9) + 0.5) / 2 ** 23
            assert 0.0 < u < 1.0
            assert np.float32(u) == u  # exactly representable in fp32
            assert O.gumbel(seed, index, pos, 1, 9) == pytest.approx(-np.log(-np.log(u)), rel=1e-15)


def test_uniform_is_uniform():
    # 4000 draws: Kolmogorov-Smirnov against U(0,1) (fixed seed, deterministic)
    from scipy import stats
    u = np.array([O.uniform(99, i, 3, 0, 1) for i in range(4000)])
    assert stats.kstest(u, "uniform").pvalue > 1e-3


def test_round_bf16_matches_torch():
    torch = pytest.importorskip("torch")
    rng = np.random.Generator(np.random.PCG64(7))
    xs = np.concatenate([
        rng.standard_normal(2000) * 10.0 ** rng.integers(-8, 8, 2000),
        # exact halfway points between adjacent bf16 values: ties to even
        (np.arange(1, 200, dtype=np.float64) * 2 + 1) * 2.0 ** -8,
        -(np.arange(1, 200, dtype=np.float64) * 2 + 1) * 2.0 ** -8,
        [1e-39, -3e-40, 2.5e-41, 3.0e38],
    ]).astype(np.float32)
    ref = torch.from_numpy(xs).to(torch.bfloat16).to(torch.float64).numpy()
    got = np.array([O.round_bf16(float(x)) for x in xs])
    np.testing.assert_array_equal(got, ref)
