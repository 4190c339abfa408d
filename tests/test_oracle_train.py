"""Pins for the oracle's training objective and its gradient (Sec. 4.3).

* Every weight's analytic gradient matches central finite differences of
  L_total on randomly chosen elements (fp32 storage, so the forward has no
  rounding), for each reading of sigma.
* L(p^b), the drafter-anchor term, equals its closed form from scipy's
  log-softmax (it involves no refiner weight: its gradient is zero).
* With a_l1 = 0 the readout gradient is the textbook softmax cross-entropy
  gradient sum_k w_k (p_k - onehot(x*_k)) z_k^T (numpy, from the oracle's
  pinned forward at the teacher-forced inputs).
* The L1 term's value is |p - q|_1 of the two softmaxes (scipy), and
  |p - q|_1 = 2 (1 - sum min(p, q)) (the acceptance identity the paper
  cites).
"""
import numpy as np
import pytest
from scipy import special

import oracle as O


def _setup(V=11, B=4, r=5, H=6, seed=0, act=O.SILU):
    rng = np.random.Generator(np.random.PCG64(seed))
    w = {"W_e": rng.standard_normal((V, r)), "W_h": rng.standard_normal((r, H)) * 0.5,
         "W_g": rng.standard_normal((r, H)) * 0.5, "W_in": rng.standard_normal((r, 3 * r)) * 0.5,
         "L": np.tril(rng.standard_normal((r, B, B)), -1) * 0.5, "W1": rng.standard_normal((2 * r, r)) * 0.5,
         "W2": rng.standard_normal((r, 2 * r)) * 0.5, "W_r": rng.standard_normal((V, r))}
    w = {k: v.astype(np.float32) for k, v in w.items()}
    h = rng.standard_normal((B, H)).astype(np.float32)
    s = (rng.standard_normal((B, V)) * 1.5).astype(np.float32)
    tgt = (rng.standard_normal((B, V)) * 1.5).astype(np.float32)
    ystar = rng.integers(0, V, B).astype(np.int32)
    anchor = int(rng.integers(0, V))
    return w, h, s, tgt, ystar, anchor, (V, B, r, H, act)


def _total(w, dims, h, s, tgt, ystar, anchor, **kw):
    V, B, r, H, act = dims
    m = O.Model(w, H, V, r, B, O.F32, act)
    loss, _ = O.train_step(m, h, s, tgt, ystar, anchor, grads=False, **kw)
    return loss[3]


@pytest.mark.parametrize("act", [O.SILU, O.GELU, O.RELU])
def test_gradient_matches_finite_differences(act):
    w, h, s, tgt, ystar, anchor, dims = _setup(seed=3 + act, act=act)
    V, B, r, H, _ = dims
    kw = dict(a_ce=0.7, a_l1=1.3, gamma=3.0, lam=0.4, beta=0.6)
    m = O.Model(w, H, V, r, B, O.F32, act)
    loss, g = O.train_step(m, h, s, tgt, ystar, anchor, **kw)
    rng = np.random.Generator(np.random.PCG64(100 + act))
    for name in O.GRAD_NAMES:
        flat = w[name].reshape(-1)
        idx = rng.choice(flat.size, min(12, flat.size), replace=False)
        if name == "L":   # only the strictly lower part of L is read
            tri = np.nonzero(np.tril(np.ones((B, B)), -1)[None].repeat(r, 0).reshape(-1))[0]
            idx = rng.choice(tri, min(12, tri.size), replace=False)
        for i in idx:
            wp = {k: v.copy() for k, v in w.items()}
            wm = {k: v.copy() for k, v in w.items()}
            x0 = float(flat[i])
            step = np.float32(1e-3) * np.float32(max(1.0, abs(x0)))
            wp[name].reshape(-1)[i] = np.float32(x0 + step)
            wm[name].reshape(-1)[i] = np.float32(x0 - step)
            dx = float(wp[name].reshape(-1)[i]) - float(wm[name].reshape(-1)[i])
            num = (_total(wp, dims, h, s, tgt, ystar, anchor, **kw) - _total(wm, dims, h, s, tgt, ystar, anchor, **kw)) / dx
            ana = g[name].reshape(-1)[i]
            assert ana == pytest.approx(num, rel=3e-4, abs=3e-5), (name, i, ana, num)


def test_anchor_term_and_l1_closed_forms():
    w, h, s, tgt, ystar, anchor, dims = _setup(seed=8)
    V, B, r, H, act = dims
    m = O.Model(w, H, V, r, B, O.F32, act)
    a_ce, a_l1, gam = 0.8, 1.7, 2.5
    loss, _ = O.train_step(m, h, s, tgt, ystar, anchor, a_ce=a_ce, a_l1=a_l1, gamma=gam, grads=False)
    want = 0.0
    for k in range(B):
        p = special.softmax(s[k].astype(np.float64))
        q = special.softmax(tgt[k].astype(np.float64))
        l1 = np.abs(p - q).sum()
        assert l1 == pytest.approx(2.0 * (1.0 - np.minimum(p, q).sum()), rel=1e-12)
        want += np.exp(-k / gam) * (a_ce * -special.log_softmax(s[k].astype(np.float64))[ystar[k]] + a_l1 * l1)
    assert loss[1] == pytest.approx(want, rel=1e-12)


def test_cross_entropy_readout_gradient_is_softmax_minus_onehot():
    w, h, s, tgt, ystar, anchor, dims = _setup(seed=12)
    V, B, r, H, act = dims
    m = O.Model(w, H, V, r, B, O.F32, act)
    gam = 3.5
    # beta = 0: only the teacher-forced forward contributes
    loss, g = O.train_step(m, h, s, tgt, ystar, anchor, a_ce=1.0, a_l1=0.0, gamma=gam, lam=0.0, beta=0.0)
    x = np.concatenate([[anchor], ystar[:-1]]).astype(np.int32)
    ell, z, _ = O.forward(m, h, s, x)
    want = np.zeros((V, r))
    ce = 0.0
    for k in range(B):
        p = special.softmax(ell[k])
        oh = np.zeros(V)
        oh[ystar[k]] = 1.0
        want += np.exp(-k / gam) * np.outer(p - oh, z[k])
        ce += np.exp(-k / gam) * -np.log(p[ystar[k]])
    np.testing.assert_allclose(g["W_r"], want, rtol=1e-10, atol=1e-12)
    assert loss[0] == pytest.approx(ce, rel=1e-12) and loss[3] == pytest.approx(ce, rel=1e-12)


def test_refiner_losses_from_the_pinned_forward():
    """L(p^r) (teacher-forced inputs x*_{k-1}) and L(p^r-hat) (inputs the
    drafter's first-argmax of s_{k-1}) from oracle.forward and scipy, CE and
    L1 terms both, and L_total's weighting; bf16 storage included (the loss
    path then sees the forward's bf16 operand roundings, which oracle.forward
    shares)."""
    for dt in (O.F32, O.BF16):
        w, h, s, tgt, ystar, anchor, dims = _setup(seed=21 + dt)
        V, B, r, H, act = dims
        if dt == O.BF16:
            from paper_2608_02438_gb300 import workloads as W
            w = {k: W.to_storage(v, "bf16") for k, v in w.items()}
            h, s, tgt = (W.to_storage(a, "bf16") for a in (h, s, tgt))
            f = lambda a: W.to_f32(a, "bf16").astype(np.float64)
        else:
            f = lambda a: a.astype(np.float64)
        m = O.Model(w, H, V, r, B, dt, act)
        a_ce, a_l1, gam, lam, beta = 0.9, 1.1, 2.0, 0.25, 0.45
        loss, _ = O.train_step(m, h, s, tgt, ystar, anchor, a_ce=a_ce, a_l1=a_l1, gamma=gam, lam=lam, beta=beta,
                               grads=False)
        xr = np.concatenate([[anchor], ystar[:-1]]).astype(np.int32)
        xc = np.concatenate([[anchor], np.argmax(f(s), axis=1)[:-1]]).astype(np.int32)
        want = []
        for x in (xr, xc):
            ell = O.forward(m, h, s, x)[0]
            tot = 0.0
            for k in range(B):
                p = special.softmax(ell[k])
                q = special.softmax(f(tgt)[k])
                tot += np.exp(-k / gam) * (a_ce * -np.log(p[ystar[k]]) + a_l1 * np.abs(p - q).sum())
            want.append(tot)
        assert loss[0] == pytest.approx(want[0], rel=1e-11)
        assert loss[2] == pytest.approx(want[1], rel=1e-11)
        assert loss[3] == pytest.approx(loss[0] + lam * loss[1] + beta * loss[2], rel=1e-14)
