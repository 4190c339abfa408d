"""Pins for the oracle's refiner map R_theta + Correct (Sec. 4.1).

Each stage is pinned by a special case that reduces it to a library routine
or a closed form, so that a dropped term, a wrong index or a transposed
operand in the oracle fails one of these:

* Fuse slots: W_in = [I|0|0], [0|I|0], [0|0|I] isolate W_h h_k, W_g g and
  W_e[x_{k-1}] (numpy matmul / mean / row lookup).
* Mix with a Toeplitz L equals a causal depthwise conv1d of kernel size B
  (the paper's remark after Prop. 1; torch.nn.functional.conv1d).
* The fold identity c_k = sum_{j<=k} M_{k,j} a~_j with
  M_{k,j} = diag(delta_jk + L_{k,j}) W_in (Sec. 4.1, "Low overhead").
* Trans closed forms: ReLU with W_1 = [I; -I], W_2 = [I, I] gives c + |c|;
  SiLU / GELU with identity blocks give c + silu(c) / c + gelu(c)
  (torch.nn.functional).
* Read + Correct: l = s + W_r z (numpy matmul).
* bf16 operand points: c before W_1, u before W_2 and z before W_r are
  rounded (torch bfloat16 casts), the residual uses the unrounded c.
* Prop. 1 (token part): l_k is bit-identical under any change of x_j, j >= k.
"""
import numpy as np
import pytest

import oracle as O
from paper_2608_02438_gb300 import workloads as W

torch = pytest.importorskip("torch")


def _model(H, V, r, B, dtype=O.F32, act=O.SILU, seed=0, **over):
    rng = np.random.Generator(np.random.PCG64(seed))
    w = {
        "W_e": rng.standard_normal((V, r)), "W_h": rng.standard_normal((r, H)) * 0.3,
        "W_g": rng.standard_normal((r, H)) * 0.3, "W_in": rng.standard_normal((r, 3 * r)) * 0.3,
        "L": np.tril(rng.standard_normal((r, B, B)), -1) * 0.5, "W1": rng.standard_normal((2 * r, r)) * 0.3,
        "W2": rng.standard_normal((r, 2 * r)) * 0.3, "W_r": rng.standard_normal((V, r)) * 0.3,
    }
    w.update(over)
    wd = "bf16" if dtype == O.BF16 else "f32"
    ws = {k: W.to_storage(np.asarray(v, np.float32), wd) for k, v in w.items()}
    return O.Model(ws, H, V, r, B, dtype, act), ws


def _io(H, V, B, dtype=O.F32, seed=1):
    rng = np.random.Generator(np.random.PCG64(seed))
    wd = "bf16" if dtype == O.BF16 else "f32"
    h = W.to_storage(rng.standard_normal((B, H)).astype(np.float32), wd)
    s = W.to_storage(rng.standard_normal((B, V)).astype(np.float32), wd)
    x = rng.integers(0, V, B).astype(np.int32)
    return h, s, x


def _f(a, dtype=O.F32):
    return W.to_f32(a, "bf16" if dtype == O.BF16 else "f32").astype(np.float64)


H, V, r, B = 10, 37, 6, 5


def _eye_in(slot):
    w = np.zeros((r, 3 * r))
    w[:, slot * r:(slot + 1) * r] = np.eye(r)
    return w


def test_fuse_slots():
    h, s, x = _io(H, V, B)
    zero_L = np.zeros((r, B, B))
    for slot in range(3):
        m, ws = _model(H, V, r, B, W_in=_eye_in(slot), L=zero_L)
        _, _, c = O.forward(m, h, s, x)
        hh = _f(h)
        if slot == 0:
            want = hh @ _f(ws["W_h"]).T
        elif slot == 1:
            want = np.broadcast_to(_f(ws["W_g"]) @ hh.mean(axis=0), (B, r))
        else:
            want = _f(ws["W_e"])[x]
        np.testing.assert_allclose(c, want, rtol=1e-12, atol=1e-12)


def test_mix_toeplitz_is_causal_depthwise_conv1d():
    rng = np.random.Generator(np.random.PCG64(3))
    taps = rng.standard_normal((r, B))          # taps[d, o] multiplies a_{k-o}; taps[:, 0] = 1
    taps[:, 0] = 1.0
    taps = taps.astype(np.float32).astype(np.float64)   # the stored (fp32) values
    L = np.zeros((r, B, B))
    for k in range(B):
        for j in range(k):
            L[:, k, j] = taps[:, k - j]
    m, ws = _model(H, V, r, B, W_in=_eye_in(2), L=L)
    h, s, x = _io(H, V, B)
    _, _, c = O.forward(m, h, s, x)
    a = torch.from_numpy(_f(ws["W_e"])[x].T.copy())[None]          # [1, r, B]
    kernel = torch.from_numpy(np.ascontiguousarray(taps[:, ::-1]))[:, None, :]  # [r, 1, B]
    want = torch.nn.functional.conv1d(torch.nn.functional.pad(a, (B - 1, 0)), kernel, groups=r)
    np.testing.assert_allclose(c, want[0].numpy().T, rtol=1e-12, atol=1e-12)


def test_fold_identity():
    m, ws = _model(H, V, r, B, seed=4)
    h, s, x = _io(H, V, B, seed=5)
    _, _, c = O.forward(m, h, s, x)
    hh = _f(h)
    g = hh.mean(axis=0)
    Win, L = _f(ws["W_in"]), _f(ws["L"])
    at = [np.concatenate([_f(ws["W_h"]) @ hh[j], _f(ws["W_g"]) @ g, _f(ws["W_e"])[x[j]]]) for j in range(B)]
    for k in range(B):
        ck = np.zeros(r)
        for j in range(k + 1):
            diag = np.full(r, 1.0 if j == k else 0.0) + (L[:, k, j] if j < k else 0.0)
            Mkj = diag[:, None] * Win
            ck += Mkj @ at[j]
        np.testing.assert_allclose(c[k], ck, rtol=1e-11, atol=1e-11)


@pytest.mark.parametrize("act", [O.RELU, O.SILU, O.GELU])
def test_trans_closed_forms(act):
    zero_L = np.zeros((r, B, B))
    if act == O.RELU:
        W1 = np.vstack([np.eye(r), -np.eye(r)])
        W2 = np.hstack([np.eye(r), np.eye(r)])
    else:
        W1 = np.vstack([np.eye(r), np.zeros((r, r))])
        W2 = np.hstack([np.eye(r), np.zeros((r, r))])
    m, ws = _model(H, V, r, B, act=act, W_in=_eye_in(2), L=zero_L, W1=W1, W2=W2)
    h, s, x = _io(H, V, B)
    _, z, c = O.forward(m, h, s, x)
    ct = torch.from_numpy(c)
    if act == O.RELU:
        want = ct + ct.abs()
    elif act == O.SILU:
        want = ct + torch.nn.functional.silu(ct)
    else:
        want = ct + torch.nn.functional.gelu(ct)
    np.testing.assert_allclose(z, want.numpy(), rtol=1e-12, atol=1e-12)


def test_read_correct_is_matmul():
    m, ws = _model(H, V, r, B, seed=8)
    h, s, x = _io(H, V, B, seed=9)
    ell, z, _ = O.forward(m, h, s, x)
    np.testing.assert_allclose(ell, _f(s) + z @ _f(ws["W_r"]).T, rtol=1e-12, atol=1e-12)


def test_bf16_operand_rounding_points():
    # c = a + 0.37 a_{k-1} is not bf16-representable, so rounding c before W_1
    # is visible; the residual must use the unrounded c.
    L = np.zeros((r, B, B))
    for k in range(1, B):
        L[:, k, k - 1] = 0.37
    W1 = np.vstack([0.3 * np.eye(r), np.zeros((r, r))])
    W2 = np.hstack([np.eye(r), np.zeros((r, r))])
    Wr = np.zeros((V, r))
    Wr[:r] = 0.5 * np.eye(r)
    m, ws = _model(H, V, r, B, dtype=O.BF16, act=O.RELU, W_in=_eye_in(2), L=L, W1=W1, W2=W2, W_r=Wr)
    h, s, x = _io(H, V, B, dtype=O.BF16)
    ell, z, c = O.forward(m, h, s, x)
    bf = lambda t: t.to(torch.bfloat16).to(torch.float64)
    e = torch.from_numpy(_f(ws["W_e"], O.BF16)[x])
    l37 = float(_f(ws["L"], O.BF16)[0, 1, 0])          # 0.37 as stored in bf16
    c_want = e.clone()
    c_want[1:] += l37 * e[:-1]                        # exact-arithmetic Mix
    w1 = float(bf(torch.tensor(0.3)))                   # W_1 is stored in bf16
    u = bf(torch.relu(w1 * bf(c_want)))               # rounded c feeds W_1, rounded u feeds W_2
    z_want = c_want + u                                 # residual on the unrounded c
    np.testing.assert_allclose(c, c_want.numpy(), rtol=1e-14, atol=1e-14)
    np.testing.assert_allclose(z, z_want.numpy(), rtol=1e-14, atol=1e-14)
    want_ell = _f(s, O.BF16).copy()
    want_ell[:, :r] += 0.5 * bf(z_want).numpy()        # rounded z feeds W_r
    np.testing.assert_array_equal(ell, want_ell)


def test_causal_in_tokens_prop1():
    m, ws = _model(H, V, r, B, seed=11)
    h, s, x = _io(H, V, B, seed=12)
    base, _, _ = O.forward(m, h, s, x)
    rng = np.random.Generator(np.random.PCG64(13))
    for k in range(B):
        for trial in range(3):
            x2 = x.copy()
            x2[k + 1:] = rng.integers(0, V, B - k - 1)   # position k reads x_0..x_k only
            ell2, _, _ = O.forward(m, h, s, x2)
            np.testing.assert_array_equal(ell2[k], base[k])
        x3 = x.copy()
        x3[k] = (x[k] + 1) % V                            # ... and does read x_k
        ell3, _, _ = O.forward(m, h, s, x3)
        assert not np.array_equal(ell3[k], base[k])
