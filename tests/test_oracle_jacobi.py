"""Pins for the oracle's selection and Jacobi refinement (Sec. 4.2).

* T = 0 selection is numpy's first-index argmax of the fp32-rounded logits.
* T > 0 selection (fixed-noise hierarchical Gumbel-max) draws exactly from
  softmax(l / T): chi-square over seeds against the closed-form softmax,
  with partial last groups; lse matches scipy's logsumexp.
* Theorem 1: from any seed Jacobi reaches the sequential decode Y*, position
  k is pinned after k passes (Eq. monotone), K_max = B always yields Y*.
* Uniqueness: brute force over all V^B blocks of tiny problems finds exactly
  one fixed point, and it is Y*; Jacobi from every one of the V^B seeds
  reaches it within B passes.
* T > 0 refinement: the distribution of the final block over seeds matches
  the autoregressive factorisation of Prop. 1, prod_k p^r_k(x_k | x_<k),
  enumerated over all blocks (chi-square).
"""
import itertools

import numpy as np
import pytest
from scipy import special, stats

import oracle as O
from paper_2608_02438_gb300 import workloads as W


def _strong_model(H=6, V=5, r=4, B=3, seed=0, dtype=O.F32, act=O.SILU, scale=1.0):
    rng = np.random.Generator(np.random.PCG64(seed))
    w = {
        "W_e": rng.standard_normal((V, r)) * 2.0 * scale, "W_h": rng.standard_normal((r, H)) * 0.5,
        "W_g": rng.standard_normal((r, H)) * 0.5, "W_in": rng.standard_normal((r, 3 * r)) * 0.7,
        "L": np.tril(rng.standard_normal((r, B, B)), -1), "W1": rng.standard_normal((2 * r, r)) * 0.7,
        "W2": rng.standard_normal((r, 2 * r)) * 0.7, "W_r": rng.standard_normal((V, r)) * 1.5 * scale,
    }
    wd = "bf16" if dtype == O.BF16 else "f32"
    ws = {k: W.to_storage(v.astype(np.float32), wd) for k, v in w.items()}
    h = W.to_storage(rng.standard_normal((B, H)).astype(np.float32), wd)
    s = W.to_storage(rng.standard_normal((B, V)).astype(np.float32), wd)
    anchor = int(rng.integers(0, V))
    return O.Model(ws, H, V, r, B, dtype, act), h, s, anchor


# ----------------------------------------------------------------- select

def test_select_greedy_is_first_argmax():
    rng = np.random.Generator(np.random.PCG64(1))
    for trial in range(50):
        v = rng.integers(0, 6, 97).astype(np.float64) * 0.25   # many exact ties
        v += rng.standard_normal(97) * (1e-9 if trial % 2 else 0.0)
        y, _, sel, _ = O.select(v, 0.0)
        assert y == int(np.argmax(v.astype(np.float32)))
        assert sel == v[y]


@pytest.mark.parametrize("V,T", [(70, 0.7), (32, 1.0), (5, 2.0), (129, 1.0)])
def test_select_sampling_is_softmax(V, T):
    rng = np.random.Generator(np.random.PCG64(V))
    ell = rng.standard_normal(V) * 1.5
    ell[rng.integers(0, V)] += 2.0
    n = 20000
    counts = np.zeros(V)
    for seed in range(n):
        y, lse, sel, _ = O.select(ell, T, seed=seed, offset=3, k=2)
        counts[y] += 1
    p = special.softmax(ell / T)
    # pool cells with small expectation to keep the chi-square valid
    order = np.argsort(p)
    exp_c, obs_c, acc_e, acc_o = [], [], 0.0, 0.0
    for i in order:
        acc_e += n * p[i]
        acc_o += counts[i]
        if acc_e >= 20:
            exp_c.append(acc_e); obs_c.append(acc_o); acc_e = acc_o = 0.0
    if acc_e > 0:
        exp_c[-1] += acc_e; obs_c[-1] += acc_o
    assert stats.chisquare(obs_c, exp_c).pvalue > 1e-4
    assert lse == pytest.approx(special.logsumexp(ell / T), rel=1e-13)
    assert sel == pytest.approx(ell[y] / T, rel=1e-15)


def test_select_noise_is_fixed_across_calls():
    rng = np.random.Generator(np.random.PCG64(9))
    ell = rng.standard_normal(200)
    a = O.select(ell, 1.0, seed=5, offset=1, k=3)
    b = O.select(ell, 1.0, seed=5, offset=1, k=3)
    assert a == b
    # other (offset, position) keys draw other noise
    assert len({O.select(ell, 1.0, seed=5, offset=o, k=3)[0] for o in range(40)}) > 5
    assert len({O.select(ell, 1.0, seed=5, offset=1, k=k)[0] for k in range(40)}) > 5


@pytest.mark.parametrize("T", [0.0, 1.0])
def test_each_pass_reads_the_previous_iterate(T):
    # Eq. (jacobi-update): Y^(j+1)_k = Select(R(Y^(j)))_k, all positions at once
    m, h, s, anchor = _strong_model(H=9, V=23, r=6, B=7, seed=8)
    res = O.jacobi(m, h, s, anchor, None, T, 3, 4, K_max=7, trajectory=True)
    traj = res["trajectory"]
    assert res["iters"] >= 3
    for j in range(res["iters"]):
        x = np.concatenate([[anchor], traj[j, :-1]]).astype(np.int32)
        ell, _, _ = O.forward(m, h, s, x)
        nxt = [O.select(ell[k], T, seed=3, offset=4, k=k)[0] for k in range(m.B)]
        np.testing.assert_array_equal(traj[j + 1], nxt)


# ----------------------------------------------------------------- Theorem 1

@pytest.mark.parametrize("seed", range(12))
@pytest.mark.parametrize("T", [0.0, 1.0])
def test_theorem1_fixed_point_is_sequential(seed, T):
    m, h, s, anchor = _strong_model(H=9, V=23, r=6, B=7, seed=seed)
    rng = np.random.Generator(np.random.PCG64(100 + seed))
    ystar, _ = O.sequential(m, h, s, anchor, T, seed=seed, offset=2)
    for trial in range(3):
        draft = rng.integers(0, m.V, m.B).astype(np.int32) if trial else None
        res = O.jacobi(m, h, s, anchor, draft, T, seed, 2, K_max=m.B + 1, trajectory=True)
        assert res["converged"] == 1
        assert res["iters"] <= m.B + 1
        np.testing.assert_array_equal(res["tokens"], ystar)
        traj = res["trajectory"]
        for j in range(1, traj.shape[0]):             # Eq. (monotone): y_k^(j) = y*_k for k <= j
            np.testing.assert_array_equal(traj[j, :j], ystar[:j])
        capped = O.jacobi(m, h, s, anchor, draft, T, seed, 2, K_max=m.B)
        np.testing.assert_array_equal(capped["tokens"], ystar)


def test_consistent_draft_converges_in_one_pass():
    m, h, s, anchor = _strong_model(H=9, V=23, r=6, B=7, seed=3)
    ystar, _ = O.sequential(m, h, s, anchor, 0.0)
    res = O.jacobi(m, h, s, anchor, ystar, 0.0, 0, 0, K_max=7)
    assert res["iters"] == 1 and res["converged"] == 1


def test_zero_readout_keeps_argmax_draft():
    m, h, s, anchor = _strong_model(H=9, V=23, r=6, B=7, seed=4)
    w = dict(m.w)
    w["W_r"] = np.zeros_like(w["W_r"])
    m0 = O.Model(w, m.H, m.V, m.r, m.B, m.dtype, m.act)
    res = O.jacobi(m0, h, s, anchor, None, 0.0, 0, 0, K_max=7)
    np.testing.assert_array_equal(res["tokens"], np.argmax(W.to_f32(s, "f32"), axis=1))
    assert res["iters"] == 1 and res["converged"] == 1


def test_fixed_k_runs_all_passes():
    m, h, s, anchor = _strong_model(H=9, V=23, r=6, B=7, seed=6)
    res = O.jacobi(m, h, s, anchor, None, 0.0, 0, 0, K_max=5, fixed_K=True)
    assert res["iters"] == 5


# ----------------------------------------------------------------- uniqueness

@pytest.mark.parametrize("V,B,T,seed", [(4, 3, 0.0, 0), (5, 3, 0.0, 1), (8, 3, 0.0, 2), (4, 4, 0.0, 3),
                                        (5, 3, 1.0, 4), (4, 4, 0.7, 5)])
def test_brute_force_unique_fixed_point(V, B, T, seed):
    m, h, s, anchor = _strong_model(H=5, V=V, r=4, B=B, seed=seed)
    ystar, _ = O.sequential(m, h, s, anchor, T, seed=seed, offset=0)
    fixed = []
    for blk in itertools.product(range(V), repeat=B):
        x = np.array((anchor,) + blk[:-1], np.int32)
        ell, _, _ = O.forward(m, h, s, x)
        sel = [O.select(ell[k], T, seed=seed, offset=0, k=k)[0] for k in range(B)]
        if list(blk) == sel:
            fixed.append(blk)
        res = O.jacobi(m, h, s, anchor, np.array(blk, np.int32), T, seed, 0, K_max=B + 1)
        assert res["converged"] == 1 and res["iters"] <= B + 1
        np.testing.assert_array_equal(res["tokens"], ystar)
    assert fixed == [tuple(int(t) for t in ystar)]


# ----------------------------------------------------------------- T > 0 law

def test_sampling_fixed_point_follows_prop1_factorisation():
    V, B, T = 4, 3, 1.0
    m, h, s, anchor = _strong_model(H=5, V=V, r=4, B=B, seed=21, scale=0.4)
    probs = {}
    for blk in itertools.product(range(V), repeat=B):
        x = np.array((anchor,) + blk[:-1], np.int32)
        ell, _, _ = O.forward(m, h, s, x)
        p = 1.0
        for k in range(B):
            p *= special.softmax(ell[k] / T)[blk[k]]
        probs[blk] = p
    n = 30000
    tok, iters = O.jacobi_seeds(m, h, s, anchor, None, T, np.arange(n, dtype=np.uint64) + 77, 5, B + 1)
    assert (iters <= B + 1).all()
    keys = list(probs)
    idx = {k: i for i, k in enumerate(keys)}
    counts = np.zeros(len(keys))
    for row in tok:
        counts[idx[tuple(int(t) for t in row)]] += 1
    expect = np.array([probs[k] for k in keys]) * n
    assert abs(expect.sum() - n) < 1e-6 * n
    keep = expect >= 5
    obs = np.append(counts[keep], counts[~keep].sum())
    exp = np.append(expect[keep], expect[~keep].sum())
    assert stats.chisquare(obs, exp).pvalue > 1e-4
