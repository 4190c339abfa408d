"""Pins for the oracle's base-logit readout s = W_lm h (Sec. 4.1, Fig. 2a:
the target-sized LM head that produces the drafter's base logits s_k) and
Algorithm 1's Y^(0) = argmax_v s_k,v.

* The fp64 sums equal numpy's float64 matmul of the stored operands.
* The stored s is that sum rounded once to bf16 (the separately pinned
  rounding helper) or to fp32.
* Y^(0) is numpy's first-index argmax of the stored row (exact ties go to
  the smallest id), including rows built with exact ties.
* A planted closed form: W_lm with one-hot rows reads single coordinates of h.
"""
import numpy as np
import pytest

import oracle as O
from paper_2608_02438_gb300 import workloads as W


@pytest.mark.parametrize("dtype,V,H,N", [("bf16", 97, 40, 5), ("f32", 64, 33, 3), ("bf16", 1000, 256, 16)])
def test_lm_head_matches_numpy(dtype, V, H, N):
    rng = np.random.Generator(np.random.PCG64(V + H))
    Wl = W.to_storage((rng.standard_normal((V, H)) * 0.05).astype(np.float32), dtype)
    h = W.to_storage(rng.standard_normal((N, H)).astype(np.float32), dtype)
    od = O.BF16 if dtype == "bf16" else O.F32
    s_exact, s_store, am = O.lm_head(Wl, h, od)
    want = W.to_f32(h, dtype).astype(np.float64) @ W.to_f32(Wl, dtype).astype(np.float64).T
    np.testing.assert_allclose(s_exact, want, rtol=1e-12, atol=1e-12)
    if dtype == "bf16":
        rounded = np.array([[O.round_bf16(x) for x in row] for row in s_exact], np.float32)
        np.testing.assert_array_equal(W.to_f32(s_store, dtype), rounded)
    else:
        np.testing.assert_array_equal(s_store, s_exact.astype(np.float32))
    np.testing.assert_array_equal(am, np.argmax(W.to_f32(s_store, dtype), axis=1))


def test_lm_head_ties_and_one_hot_rows():
    V, H = 12, 6
    Wl = np.zeros((V, H), np.float32)
    for v in range(V):
        Wl[v, v % H] = 1.0                      # row v reads coordinate v mod H
    h = np.array([[0.5, 3.0, -1.0, 3.0, 0.0, 2.0]], np.float32)
    s_exact, s_store, am = O.lm_head(Wl, h, O.F32)
    np.testing.assert_array_equal(s_exact[0], [h[0, v % H] for v in range(V)])
    assert am[0] == 1                           # 3.0 at ids 1, 3, 7, 9: the smallest wins
