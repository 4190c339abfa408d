"""Pins for the oracle's acceptance rules (Sec. 3.1; Sec. 4.3 identity).

* Greedy: the definition's special cases (draft equal to the target argmax
  gives n = B plus the bonus argmax of row B+1; a first-position mismatch
  gives n = 0 and the target's argmax; a mismatch at position m gives n = m).
* Lossless: with W_r = 0 the refined draft distribution is q_k = softmax(s_k/T)
  in closed form.  Over seeds, (a) the emitted first token follows the target
  p_1 (chi-square), and (b) the empirical acceptance rate at the first
  position equals sum_v min(p, q) = 1 - TV(p, q) within a binomial 99.99%
  interval, as the paper states for speculative sampling.
* When everything is accepted the bonus token follows p_{B+1}.
"""
import numpy as np
import pytest
from scipy import special, stats

import oracle as O
from paper_2608_02438_gb300 import workloads as W


def _model(V=6, B=3, r=4, H=5, seed=0, zero_readout=False):
    rng = np.random.Generator(np.random.PCG64(seed))
    w = {
        "W_e": rng.standard_normal((V, r)), "W_h": rng.standard_normal((r, H)) * 0.5,
        "W_g": rng.standard_normal((r, H)) * 0.5, "W_in": rng.standard_normal((r, 3 * r)) * 0.5,
        "L": np.tril(rng.standard_normal((r, B, B)), -1), "W1": rng.standard_normal((2 * r, r)) * 0.5,
        "W2": rng.standard_normal((r, 2 * r)) * 0.5, "W_r": rng.standard_normal((V, r)),
    }
    if zero_readout:
        w["W_r"] = np.zeros((V, r))
    ws = {k: v.astype(np.float32) for k, v in w.items()}
    h = rng.standard_normal((B, H)).astype(np.float32)
    s = (rng.standard_normal((B, V)) * 1.2).astype(np.float32)
    return O.Model(ws, H, V, r, B, O.F32, O.SILU), h, s, int(rng.integers(0, V))


def test_greedy_special_cases():
    m, h, s, anchor = _model(V=11, B=4, seed=1)
    rng = np.random.Generator(np.random.PCG64(2))
    tgt = rng.standard_normal((m.B + 1, m.V)).astype(np.float32)
    targ = np.argmax(tgt, axis=1).astype(np.int32)
    dummy = np.zeros(m.B)
    z = np.zeros((m.B, m.r))
    n, out, _ = O.accept(m, tgt, s, targ[: m.B], dummy, dummy, z, 0.0, 0, 0)
    assert n == m.B and out.tolist() == targ.tolist()
    y = targ[: m.B].copy()
    y[0] = (y[0] + 1) % m.V
    n, out, _ = O.accept(m, tgt, s, y, dummy, dummy, z, 0.0, 0, 0)
    assert n == 0 and out[0] == targ[0] and (out[1:] == -1).all()
    y = targ[: m.B].copy()
    y[2] = (y[2] + 3) % m.V
    n, out, _ = O.accept(m, tgt, s, y, dummy, dummy, z, 0.0, 0, 0)
    assert n == 2 and out[:3].tolist() == targ[:3].tolist() and (out[3:] == -1).all()


def test_greedy_ties_take_smallest_id():
    m, h, s, anchor = _model(V=8, B=2, seed=3)
    tgt = np.zeros((3, 8), np.float32)
    tgt[0, [2, 5]] = 1.0
    y = np.array([5, 0], np.int32)
    n, out, _ = O.accept(m, tgt, s, y, np.zeros(2), np.zeros(2), np.zeros((2, m.r)), 0.0, 0, 0)
    assert n == 0 and out[0] == 2


@pytest.mark.parametrize("T", [1.0, 0.8])
def test_lossless_first_token_follows_target_and_rate_is_one_minus_tv(T):
    m, h, s, anchor = _model(V=6, B=3, seed=5, zero_readout=True)
    rng = np.random.Generator(np.random.PCG64(6))
    tgt = (rng.standard_normal((m.B + 1, m.V)) * 1.3).astype(np.float32)
    n = 30000
    seeds = np.arange(n, dtype=np.uint64) * 7 + 1
    acc, out = O.refine_accept_seeds(m, h, s, tgt, anchor, None, T, seeds, 9, m.B + 1)
    p1 = special.softmax(tgt[0].astype(np.float64) / T)
    q1 = special.softmax(s[0].astype(np.float64) / T)
    counts = np.bincount(out[:, 0], minlength=m.V)
    assert stats.chisquare(counts, p1 * n).pvalue > 1e-4
    rate = float(np.minimum(p1, q1).sum())
    assert rate == pytest.approx(1.0 - 0.5 * np.abs(p1 - q1).sum(), abs=1e-12)
    emp = float((acc >= 1).mean())
    half = 3.9 * np.sqrt(rate * (1 - rate) / n)
    assert abs(emp - rate) < half
    # second emitted token, given the first was accepted, follows p_2
    sel = acc >= 1
    counts2 = np.bincount(out[sel, 1], minlength=m.V)
    p2 = special.softmax(tgt[1].astype(np.float64) / T)
    assert stats.chisquare(counts2, p2 * sel.sum()).pvalue > 1e-4


def test_lossless_bonus_follows_last_row():
    # target == refined draft distribution at every position: all accepted
    m, h, s, anchor = _model(V=5, B=2, seed=8, zero_readout=True)
    rng = np.random.Generator(np.random.PCG64(9))
    tgt = np.concatenate([s, (rng.standard_normal((1, m.V)) * 1.1).astype(np.float32)], axis=0)
    n = 20000
    acc, out = O.refine_accept_seeds(m, h, s, tgt, anchor, None, 1.0, np.arange(n, dtype=np.uint64) + 3, 0,
                                     m.B + 1)
    full = acc == m.B
    assert full.mean() > 0.999
    counts = np.bincount(out[full, m.B], minlength=m.V)
    assert stats.chisquare(counts, special.softmax(tgt[m.B].astype(np.float64)) * full.sum()).pvalue > 1e-4
