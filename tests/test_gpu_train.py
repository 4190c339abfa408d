"""GPU parity of the refiner training step (Sec. 4.3) through the C ABI
(xpress_train_step) against the oracle (oracle.train_step, summed over the
blocks), and of the tensor-core product it is built on (xpress_debug_gemm).

Tolerances, from the arithmetic:
* The product hook multiplies bf16 operands exactly and accumulates in fp32,
  so |C - AB^T| <= K 2^-24 sum_k |a_k b_k| elementwise (any summation order).
* Loss: the GPU's forward equals the oracle's up to fp32 accumulation and the
  hi + lo representation of u_h and u_g (relative 2^-17) before W_in; where
  that moves c across a bf16 rounding boundary, z moves by one bf16 ulp
  (2^-8 relative) and every logit by at most 2^-8 |W_r z|, below 1e-3 of the
  loss for these inputs; the L1 sums are fp32 over V ids (relative V 2^-24).
  Bound used: |dL| <= 2e-3 |L| + 2e-3.
* Gradients: every backward product takes bf16 operands (dL/dl, dL/dz, dL/dt,
  dL/da, the Fuse operand; relative rounding 2^-9 each, unbiased), and the
  longest chain (dL/dl -> dz -> dt -> dc -> da -> u_h -> W_h) holds six such
  roundings, so the relative Frobenius error of every gradient is at most
  about 6 x 2 x 2^-9 = 2.3e-2; bound used 2^-5 = 3.1e-2.  The sign of p - q is
  taken in fp32 on both sides of a near-tie; a flip there moves dL/dl_v by
  2 a_l1 p_v, inside the same bound; with ReLU, sigma'(t) takes the other
  branch where a one-ulp move of c carries t across 0, which stays a small
  fraction of the elements (measured 2.6e-2 relative on dW_1 with paper-scale
  weights before u_h and u_g were passed as hi + lo pairs, when such moves
  were common).
Cases: a vocabulary that is not a multiple of the 64- and 128-id tiles (2080),
one ragged row tile (48 positions) and two (80), the three readings of sigma,
paper-scale and strong-coupling weights, the drafter argmax given or computed,
accumulation into the gradient buffers, and the Qwen3-8B shape (V = 151936,
H = 4096) at 2 blocks.
"""
import numpy as np
import pytest

import oracle as O
from paper_2608_02438_gb300 import workloads as W

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

LOSS_RTOL, LOSS_ATOL = 2e-3, 2e-3
GRAD_REL = 2.0 ** -5


@pytest.fixture(scope="module")
def X():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_02438_gb300 import binding, build
    build.build()
    binding.load()
    return binding


def _bf16_dev(X, a):
    return X.to_device(a, X.XPRESS_BF16)


@pytest.mark.parametrize("a_mn,b_mn", [(0, 0), (0, 1), (1, 0), (1, 1)])
@pytest.mark.parametrize("accumulate", [0, 1])
def test_product_layouts(X, a_mn, b_mn, accumulate):
    M, N, K = 200, 192, 136
    rng = np.random.Generator(np.random.PCG64(10 * a_mn + 20 * b_mn + accumulate))
    A = W.to_storage(rng.standard_normal((M, K), dtype=np.float32), "bf16")
    B = W.to_storage(rng.standard_normal((N, K), dtype=np.float32), "bf16")
    A64, B64 = W.to_f32(A, "bf16").astype(np.float64), W.to_f32(B, "bf16").astype(np.float64)
    dA = _bf16_dev(X, np.ascontiguousarray(A.T) if a_mn else A)
    dB = _bf16_dev(X, np.ascontiguousarray(B.T) if b_mn else B)
    C0 = rng.standard_normal((M, N)).astype(np.float32) if accumulate else np.zeros((M, N), np.float32)
    dC = torch.from_numpy(C0.copy()).cuda()
    X.xpress_debug_gemm(dA.data_ptr(), a_mn, dB.data_ptr(), b_mn, M, N, K, dC.data_ptr(), accumulate,
                        torch.cuda.current_stream().cuda_stream)
    torch.cuda.synchronize()
    want = C0.astype(np.float64) + A64 @ B64.T
    bound = K * 2.0 ** -24 * (np.abs(A64) @ np.abs(B64).T) + 4 * 2.0 ** -24 * np.abs(want) + 1e-30
    err = np.abs(dC.cpu().numpy().astype(np.float64) - want)
    assert (err <= bound).all(), f"max excess {(err - bound).max():.3g}"


def _run(X, cfg, w, inp, act, xhat=None, grads=None, kw=None):
    kw = kw or {}
    ref = X.Refiner({k: _bf16_dev(X, v) for k, v in w.items()}, cfg.H, cfg.V, cfg.r, cfg.B, X.XPRESS_BF16, act)
    d = {k: _bf16_dev(X, inp[k]) for k in ("h", "s", "target")}
    ys = torch.from_numpy(inp["ystar"]).cuda()
    an = torch.from_numpy(inp["anchor"]).cuda()
    xh = None if xhat is None else torch.from_numpy(xhat).cuda()
    loss, g = ref.train_step(d["h"], d["s"], d["target"], ys, an, xhat=xh, grads=grads, **kw)
    torch.cuda.synchronize()
    assert ref.device_status("train", inp["h"].shape[0]) == X.XPRESS_OK
    out = loss.cpu().numpy(), {k: v.cpu().numpy().astype(np.float64) for k, v in g.items()}
    return out, ref, g


def _oracle(cfg, w, inp, act, kw):
    m = O.Model(w, cfg.H, cfg.V, cfg.r, cfg.B, O.BF16, act)
    b = inp["h"].shape[0]
    losses, tot = [], None
    for i in range(b):
        loss, g = O.train_step(m, inp["h"][i], inp["s"][i], inp["target"][i], inp["ystar"][i], int(inp["anchor"][i]),
                               **kw)
        losses.append(loss)
        tot = g if tot is None else {k: tot[k] + g[k] for k in tot}
    return np.array(losses), tot


def _compare(loss_g, grads_g, loss_o, grads_o, label=""):
    np.testing.assert_allclose(loss_g, loss_o, rtol=LOSS_RTOL, atol=LOSS_ATOL)
    report = [f"loss max rel {np.max(np.abs(loss_g - loss_o) / np.abs(loss_o)):.2e}"]
    for name, go in grads_o.items():
        gg = grads_g[name]
        if name == "L":                    # only the strictly lower triangle is a gradient
            mask = np.tril(np.ones(go.shape[1:]), -1)[None].astype(bool).repeat(go.shape[0], 0)
            assert np.all(gg[~mask] == 0.0), "gL outside the strictly lower triangle"
            gg, go = gg[mask], go[mask]
        rel = np.linalg.norm(gg - go) / max(np.linalg.norm(go), 1e-30)
        report.append(f"d{name} {rel:.2e}")
        assert rel <= GRAD_REL, f"d{name}: relative Frobenius error {rel:.3g} > {GRAD_REL:.3g}"
    print(f"\n[train parity {label}] " + ", ".join(report))


KW = dict(a_ce=1.0, a_l1=1.0, gamma=4.0, lam=0.6, beta=0.3)


@pytest.mark.parametrize("b,coupling,act", [(3, "paper", O.SILU), (5, "strong", O.SILU), (3, "strong", O.GELU),
                                            (5, "paper", O.RELU)])
def test_train_step_matches_oracle(X, b, coupling, act):
    cfg = W.Config("train_tiny", b=b, B=16, H=256, V=2080, r=256, dtype=W.BF16, K_max=16, logits="gauss4_spike",
                   seed=4100 + b)
    w = W.make_weights(cfg.H, cfg.V, cfg.r, cfg.B, cfg.dtype, 4200 + b, coupling)
    inp = W.make_train_inputs(cfg)
    kw = dict(a_ce=0.9, a_l1=1.2, gamma=3.0, lam=0.6, beta=0.3)
    (loss_g, grads_g), ref, _ = _run(X, cfg, w, inp, act, kw=kw)
    ref.close()
    loss_o, grads_o = _oracle(cfg, w, inp, act, kw)
    _compare(loss_g, grads_g, loss_o, grads_o, f"b={b} {coupling} act={act}")


def test_train_step_xhat_and_accumulation(X):
    cfg = W.Config("train_acc", b=3, B=16, H=256, V=2080, r=256, dtype=W.BF16, K_max=16, logits="gauss4_spike",
                   seed=4300)
    w = W.make_weights(cfg.H, cfg.V, cfg.r, cfg.B, cfg.dtype, 4301, "strong")
    inp = W.make_train_inputs(cfg)
    (loss1, g1), ref, gt = _run(X, cfg, w, inp, O.SILU, kw=KW)
    # the drafter's argmax given explicitly: the same step
    xhat = np.argmax(W.to_f32(inp["s"], "bf16"), axis=-1).astype(np.int32)
    (loss2, g2), ref2, _ = _run(X, cfg, w, inp, O.SILU, xhat=xhat, kw=KW)
    np.testing.assert_array_equal(loss1, loss2)
    for k in g1:
        np.testing.assert_allclose(g2[k], g1[k], rtol=1e-5, atol=1e-7 * np.abs(g1[k]).max())
    # a second step into the same buffers adds the same gradient again
    d = {k: _bf16_dev(X, inp[k]) for k in ("h", "s", "target")}
    ref.train_step(d["h"], d["s"], d["target"], torch.from_numpy(inp["ystar"]).cuda(),
                   torch.from_numpy(inp["anchor"]).cuda(), grads=gt, **KW)
    torch.cuda.synchronize()
    for k, v in gt.items():
        np.testing.assert_allclose(v.cpu().numpy(), 2.0 * g1[k], rtol=1e-5, atol=1e-6 * np.abs(g1[k]).max())
    ref.close()
    ref2.close()


def test_train_step_qwen3_shape(X):
    cfg = W.TRAIN_CONFIGS["qwen3_8b_train"]
    w = W.config_weights("qwen3_8b_greedy")
    inp = W.make_train_inputs(cfg, b=2)
    (loss_g, grads_g), ref, _ = _run(X, cfg, w, inp, O.SILU, kw=KW)
    ref.close()
    loss_o, grads_o = _oracle(cfg, w, inp, O.SILU, KW)
    _compare(loss_g, grads_g, loss_o, grads_o, "qwen3_8b_train b=2")


def test_train_step_rejects(X):
    cfg = W.tiny_config("trej", b=1, B=8, H=128, V=1024, r=256, dtype=W.F32, seed=4400)
    w = W.make_weights(cfg.H, cfg.V, cfg.r, cfg.B, cfg.dtype, 4401, "paper")
    ref = X.Refiner({k: X.to_device(v, X.XPRESS_F32) for k, v in w.items()}, cfg.H, cfg.V, cfg.r, cfg.B,
                    X.XPRESS_F32)
    z = torch.zeros(8, dtype=torch.int32, device="cuda")
    f = torch.zeros((1, 8, 1024), dtype=torch.float32, device="cuda")
    with pytest.raises(X.XpressError) as err:
        ref.train_step(torch.zeros((1, 8, 128), device="cuda"), f, f, z, z[:1])
    assert err.value.code == X.XPRESS_ERR_UNSUPPORTED
    ref.close()
