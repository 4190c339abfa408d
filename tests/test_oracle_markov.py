"""Pins for the sequential decode and the Markov-head comparison head.

* The Markov head (the comparison head of Sec. 2 and Table 3, whose
  correction for token k is indexed by the id of token k-1) is read as the
  refiner with its hidden-state slots, mixer and Trans MLP set to zero
  (workloads.markov_head_weights).  Its logits then have the closed form
  l_k = s_k + W_r bf16(W_in[:, 2r:3r] W_e[x_{k-1}]) (numpy matmul; the bf16
  rounding of the W_r operand by the separately pinned rounding helper), and
  its sequential decode is the step-by-step argmax (or the fixed-noise draw)
  of those logits, checked here against a numpy decode loop.
* The sequential decode Y* of Theorem 1 with the full refiner is pinned by
  the Theorem 1 tests (test_oracle_jacobi.py); here additionally: position k
  of Y* is the selection of the refiner's logits at k given y*_<k (numpy
  argmax over oracle.forward, which is pinned stage by stage).
"""
import numpy as np
import pytest

import oracle as O
from paper_2608_02438_gb300 import workloads as W


def _weights(V=29, r=8, H=6, B=5, seed=3, dtype="bf16"):
    rng = np.random.Generator(np.random.PCG64(seed))
    w = {"W_e": rng.standard_normal((V, r)), "W_h": rng.standard_normal((r, H)),
         "W_g": rng.standard_normal((r, H)), "W_in": rng.standard_normal((r, 3 * r)) * 0.5,
         "L": np.tril(rng.standard_normal((r, B, B)), -1), "W1": rng.standard_normal((2 * r, r)),
         "W2": rng.standard_normal((r, 2 * r)), "W_r": rng.standard_normal((V, r))}
    w = {k: W.to_storage(v.astype(np.float32), dtype) for k, v in w.items()}
    h = W.to_storage(rng.standard_normal((B, H)).astype(np.float32), dtype)
    s = W.to_storage(rng.standard_normal((B, V)).astype(np.float32), dtype)
    return w, h, s, int(rng.integers(0, V))


def _f(a, dtype="bf16"):
    return W.to_f32(a, dtype).astype(np.float64)


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_markov_head_logits_closed_form(dtype):
    V, r, H, B = 29, 8, 6, 5
    w, h, s, anchor = _weights(V, r, H, B, dtype=dtype)
    mw = W.markov_head_weights(w)
    od = O.BF16 if dtype == "bf16" else O.F32
    m = O.Model(mw, H, V, r, B, od, O.SILU)
    x = np.array([anchor, 3, 17, 0, 28], np.int32)
    ell, z, c = O.forward(m, h, s, x)
    Ein = _f(w["W_in"], dtype)[:, 2 * r:]
    for k in range(B):
        ck = Ein @ _f(w["W_e"], dtype)[x[k]]
        zop = np.array([O.round_bf16(v) for v in ck]) if dtype == "bf16" else ck
        np.testing.assert_allclose(c[k], ck, rtol=1e-12, atol=1e-12)
        np.testing.assert_allclose(z[k], ck, rtol=1e-12, atol=1e-12)
        np.testing.assert_allclose(ell[k], _f(s, dtype)[k] + _f(w["W_r"], dtype) @ zop, rtol=1e-12, atol=1e-12)


@pytest.mark.parametrize("T", [0.0, 1.0])
def test_markov_head_sequential_decode_is_stepwise_selection(T):
    V, r, H, B = 29, 8, 6, 5
    w, h, s, anchor = _weights(V, r, H, B, seed=8)
    mw = W.markov_head_weights(w)
    m = O.Model(mw, H, V, r, B, O.BF16, O.SILU)
    ystar, _ = O.sequential(m, h, s, anchor, T, seed=4, offset=2)
    Ein = _f(w["W_in"])[:, 2 * r:]
    prev = anchor
    for k in range(B):
        ck = Ein @ _f(w["W_e"])[prev]
        ell = _f(s)[k] + _f(w["W_r"]) @ np.array([O.round_bf16(v) for v in ck])
        if T == 0:
            want = int(np.argmax(ell.astype(np.float32)))
        else:
            want = O.select(ell, T, seed=4, offset=2, k=k)[0]    # the draw itself is pinned in test_oracle_margins
        assert ystar[k] == want
        prev = want


@pytest.mark.parametrize("T", [0.0, 1.0])
def test_sequential_decode_position_k_selects_from_its_prefix(T):
    V, r, H, B = 29, 8, 6, 5
    w, h, s, anchor = _weights(V, r, H, B, seed=11)
    m = O.Model(w, H, V, r, B, O.BF16, O.SILU)
    ystar, _ = O.sequential(m, h, s, anchor, T, seed=7, offset=1)
    for k in range(B):
        # any continuation after position k: position k's logits do not depend on it (Prop. 1)
        x = np.concatenate([[anchor], ystar[:-1]]).astype(np.int32)
        x[k + 1:] = (x[k + 1:] + 5) % V
        ell, _, _ = O.forward(m, h, s, x)
        want = int(np.argmax(ell[k].astype(np.float32))) if T == 0 else O.select(ell[k], T, seed=7, offset=1, k=k)[0]
        assert ystar[k] == want
