"""Pins for the oracle's decision margins, which decide the near-ties that the
GPU parity rule may excuse (a wrong margin would excuse real mismatches).

* T = 0: the margin is the gap between the largest and the second-largest
  logit (Algorithm 1's argmax), checked on hand-built rows with a known gap,
  on exact ties (gap 0) and against numpy's sort on random rows.
* T > 0: the fixed-noise hierarchical Gumbel-max takes two argmax decisions,
  the group (score lse_g(l / T) + Gumbel) and the member inside the drawn
  group (l_v / T + Gumbel); the margin is the smaller of their top-2 gaps.
  It is recomputed here in numpy from the Philox words (pinned by the
  published known-answer vectors), not from the oracle's Gumbel helper.
* Jacobi: margins[j][k] is the margin of the decision pass j + 1 took at
  position k, recomputed from the refiner's logits of Y^(j); min_margin is
  their minimum.
* Acceptance: the per-decision gaps are the target row's top-2 gap (T = 0)
  and |u q - p| / p of the accept test (T > 0, Sec. 3.1), recomputed with
  scipy's softmax.
"""
import numpy as np
import pytest
from scipy import special

import oracle as O
from paper_2608_02438_gb300 import workloads as W


def _gumbel(seed, index, position, stream, offset):
    x = int(O.philox([index >> 2, position, stream, offset], [seed & 0xFFFFFFFF, seed >> 32])[index & 3])
    u = ((x >> 9) + 0.5) / 2 ** 23
    return -np.log(-np.log(u))


def _top2_gap(v):
    s = np.sort(np.asarray(v, np.float64))[::-1]
    return s[0] - s[1]


def test_greedy_margin_known_gap():
    row = np.zeros(50)
    row[7] = 1.0
    row[31] = 0.75
    row[3] = 0.5
    y, _, _, mg = O.select(row, 0.0)
    assert y == 7 and mg == 0.25
    row[31] = 1.0                                   # exact tie: smallest id, margin 0
    y, _, _, mg = O.select(row, 0.0)
    assert y == 7 and mg == 0.0


def test_greedy_margin_random_rows():
    rng = np.random.Generator(np.random.PCG64(4))
    for _ in range(40):
        row = rng.standard_normal(int(rng.integers(2, 300)))
        _, _, _, mg = O.select(row, 0.0)
        assert mg == pytest.approx(_top2_gap(row), abs=0, rel=1e-15)


@pytest.mark.parametrize("V,T,seed,k", [(96, 1.0, 3, 0), (70, 0.7, 11, 4), (200, 1.3, 5, 9), (33, 1.0, 2, 1)])
def test_sampling_margin_is_the_smaller_gap_of_both_draws(V, T, seed, k):
    rng = np.random.Generator(np.random.PCG64(V + seed))
    ell = rng.standard_normal(V) * 2.0
    offset = 6
    y, _, _, mg = O.select(ell, T, seed=seed, offset=offset, k=k)
    x = ell / T
    G = O.GROUP
    ng = (V + G - 1) // G
    score = np.array([special.logsumexp(x[g * G:(g + 1) * G]) + _gumbel(seed, g, k, O.STREAM_GROUP, offset)
                      for g in range(ng)])
    g = int(np.argmax(score))
    lo, hi = g * G, min(V, g * G + G)
    member = np.array([x[v] + _gumbel(seed, v, k, O.STREAM_ELEM, offset) for v in range(lo, hi)])
    assert y == lo + int(np.argmax(member))
    gm = _top2_gap(score) if ng > 1 else np.inf
    mm = _top2_gap(member) if hi - lo > 1 else np.inf
    assert mg == pytest.approx(min(gm, mm), rel=1e-9, abs=1e-12)


def test_sampling_margin_single_group_of_one():
    # one group with one member: no competing choice at either level
    _, _, _, mg = O.select(np.array([0.3]), 1.0, seed=1, offset=0, k=0)
    assert mg == np.inf


def _model(V=23, B=6, H=7, r=5, seed=8):
    rng = np.random.Generator(np.random.PCG64(seed))
    w = {"W_e": rng.standard_normal((V, r)) * 2, "W_h": rng.standard_normal((r, H)) * 0.5,
         "W_g": rng.standard_normal((r, H)) * 0.5, "W_in": rng.standard_normal((r, 3 * r)) * 0.7,
         "L": np.tril(rng.standard_normal((r, B, B)), -1), "W1": rng.standard_normal((2 * r, r)) * 0.7,
         "W2": rng.standard_normal((r, 2 * r)) * 0.7, "W_r": rng.standard_normal((V, r)) * 1.5}
    ws = {k: v.astype(np.float32) for k, v in w.items()}
    h = rng.standard_normal((B, H)).astype(np.float32)
    s = rng.standard_normal((B, V)).astype(np.float32)
    return O.Model(ws, H, V, r, B, O.F32, O.SILU), h, s, int(rng.integers(0, V))


@pytest.mark.parametrize("T", [0.0, 1.0])
def test_jacobi_margins_per_pass_and_position(T):
    m, h, s, anchor = _model()
    res = O.jacobi(m, h, s, anchor, None, T, 3, 4, K_max=m.B, trajectory=True)
    traj, margins = res["trajectory"], res["margins"]
    assert res["iters"] >= 2 and margins.shape == (res["iters"], m.B)
    G = O.GROUP
    for j in range(res["iters"]):
        x = np.concatenate([[anchor], traj[j, :-1]]).astype(np.int32)
        ell, _, _ = O.forward(m, h, s, x)
        for k in range(m.B):
            if T == 0:
                want = _top2_gap(ell[k])
            else:
                xs = ell[k] / T
                score = np.array([special.logsumexp(xs[g * G:(g + 1) * G])
                                  + _gumbel(3, g, k, O.STREAM_GROUP, 4) for g in range((m.V + G - 1) // G)])
                g = int(np.argmax(score))
                lo, hi = g * G, min(m.V, g * G + G)
                member = [xs[v] + _gumbel(3, v, k, O.STREAM_ELEM, 4) for v in range(lo, hi)]
                want = _top2_gap(member)   # V < 32: one group, so only the member decision competes
            assert margins[j, k] == pytest.approx(want, rel=1e-9, abs=1e-12)
    assert res["min_margin"] == margins.min()


def test_accept_gaps_greedy():
    m, h, s, anchor = _model(V=19, B=4, seed=2)
    rng = np.random.Generator(np.random.PCG64(3))
    tgt = rng.standard_normal((m.B + 1, m.V)).astype(np.float32)
    targ = np.argmax(tgt, axis=1).astype(np.int32)
    y = targ[: m.B].copy()
    y[2] = (y[2] + 1) % m.V                         # accept 0 and 1, reject at 2
    z = np.zeros((m.B, m.r))
    n, out, mg, gaps = O.accept(m, tgt, s, y, np.zeros(m.B), np.zeros(m.B), z, 0.0, 0, 0, with_gaps=True)
    assert n == 2
    for k in range(3):
        assert gaps[k] == pytest.approx(_top2_gap(tgt[k]), rel=1e-15)
    assert np.isinf(gaps[3])
    assert gaps[m.B + 1] == gaps[2]                 # the token emitted is row 2's argmax
    assert mg == min(gaps[:3])


def test_accept_gaps_lossless():
    m, h, s, anchor = _model(V=19, B=4, seed=5)
    rng = np.random.Generator(np.random.PCG64(6))
    tgt = (rng.standard_normal((m.B + 1, m.V)) * 1.5).astype(np.float32)
    T, seed, offset = 1.0, 9, 2
    res = O.jacobi(m, h, s, anchor, None, T, seed, offset, K_max=m.B)
    n, out, mg, gaps = O.accept(m, tgt, s, res["tokens"], res["lse"], res["sel"], res["z_final"], T, seed, offset,
                                with_gaps=True)
    for k in range(min(n + 1, m.B)):
        p = special.softmax(tgt[k].astype(np.float64) / T)[res["tokens"][k]]
        q = np.exp(res["sel"][k] - res["lse"][k])
        x = int(O.philox([0, k, O.STREAM_ACCEPT, offset], [seed, 0])[0])
        u = ((x >> 9) + 0.5) / 2 ** 23
        assert gaps[k] == pytest.approx(abs(u * q - p) / p, rel=1e-9)
    for k in range(n + 1, m.B):
        assert np.isinf(gaps[k])
    assert np.isfinite(gaps[m.B + 1]) and gaps[m.B + 1] > 0
    assert mg == pytest.approx(min(gaps[: min(n + 1, m.B)].min(), gaps[m.B + 1]))
