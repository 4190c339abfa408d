"""GPU parity of the sequential decode (Theorem 1) and of the Markov-head
comparison head, through the C ABI (mode = XPRESS_MODE_SEQUENTIAL).

The sequential decode evaluates one position per pass, B dependent passes:
its tokens must equal the oracle's Y* exactly (oracle.sequential), every
block reports B passes and completion, pass j writes position j of the
trajectory with y*_j, and the float outputs of each position (z, l_y, lse)
equal those of the oracle's converged Jacobi run, whose last pass evaluates
every position with the same prefix (Theorem 1).  Cases: the persistent
kernel (at most 32 tokens, blocks of 16 and of 32 positions) and the
multi-kernel graph (more tokens), T = 0 and T > 0, the full refiner with
strong coupling and the Markov-head reading (workloads.markov_head_weights:
only the previous token's folded embedding feeds the correction), and the
Qwen3-8B shape at batch 1.
"""
import numpy as np
import pytest

import oracle as O
from paper_2608_02438_gb300 import workloads as W

from _parity import Z_TOL, LOGIT_TOL, device_inputs, oracle_model

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def X():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_02438_gb300 import binding, build
    build.build()
    binding.load()
    return binding


def _check_sequential(X, cfg, w, inp, markov=False):
    if markov:
        w = W.markov_head_weights(w)
    dt = X.XPRESS_BF16 if cfg.dtype == W.BF16 else X.XPRESS_F32
    ref = X.Refiner({k: X.to_device(v, dt) for k, v in w.items()}, cfg.H, cfg.V, cfg.r, cfg.B, dt)
    d = device_inputs(dt, inp)
    b = inp["h"].shape[0]
    out = ref.refine_block(d["h"], d["s"], d["draft"], d["anchor"], d["temperature"], d["seed"], inp["offset"],
                           cfg.B, want_traj=True, mode=X.XPRESS_MODE_SEQUENTIAL)
    torch.cuda.synchronize()
    assert ref.device_status("refine", b) == X.XPRESS_OK
    g = {k: (v.cpu().numpy() if v is not None else None) for k, v in out.items()}
    m = oracle_model(cfg, w)
    for i in range(b):
        T = float(inp["temperature"][i])
        ystar, margins = O.sequential(m, inp["h"][i], inp["s"][i], int(inp["anchor"][i]), T, int(inp["seed"][i]),
                                      inp["offset"])
        if not np.array_equal(g["tokens"][i], ystar):
            k = int(np.nonzero(g["tokens"][i] != ystar)[0][0])
            raise AssertionError(f"block {i}: gpu {g['tokens'][i].tolist()} | Y* {ystar.tolist()}; first difference "
                                 f"at position {k}, oracle margin {margins[k]:.3g}")
        assert int(g["iters"][i]) == cfg.B and int(g["converged"][i]) == 1
        np.testing.assert_array_equal(np.diagonal(g["trajectory"][i])[: cfg.B], ystar)
        jac = O.jacobi(m, inp["h"][i], inp["s"][i], int(inp["anchor"][i]), None, T, int(inp["seed"][i]),
                       inp["offset"], cfg.B)
        np.testing.assert_array_equal(jac["tokens"], ystar)               # Theorem 1
        zt, lt = Z_TOL[cfg.dtype], LOGIT_TOL[cfg.dtype]
        np.testing.assert_allclose(g["z_final"][i], jac["z_final"], atol=zt, rtol=zt, err_msg=f"z block {i}")
        np.testing.assert_allclose(g["logit_sel"][i], jac["sel"], atol=lt * (1.0 / T if T > 0 else 1.0),
                                   err_msg=f"logit_sel block {i}")
        if T > 0:
            np.testing.assert_allclose(g["lse"][i], jac["lse"], atol=lt / T, err_msg=f"lse block {i}")
    ref.close()
    return g


# (b, B): the persistent kernel for b * B <= 32 (blocks of at most 16 form all
# of c in every Trans CTA; 32-position blocks exchange it), the graph otherwise
@pytest.mark.parametrize("b,B,temps", [(1, 16, (0.0,)), (2, 16, (1.0, 0.0)), (1, 32, (0.0,)), (3, 8, (1.0,)),
                                       (6, 16, (0.0, 1.0)), (4, 32, (1.0, 0.0))])
@pytest.mark.parametrize("markov", [False, True])
def test_sequential_decode_matches_oracle(X, b, B, temps, markov):
    cfg = W.tiny_config("seq", b=b, B=B, H=128, V=2080, r=256, dtype=W.BF16, temps=temps, seed=3000 + b * B)
    w = W.make_weights(cfg.H, cfg.V, cfg.r, cfg.B, cfg.dtype, 3100 + b * B, "strong")
    inp = W.make_inputs(cfg)
    _check_sequential(X, cfg, w, inp, markov)


def test_sequential_decode_fp32(X):
    cfg = W.tiny_config("seq32", b=2, B=16, H=256, V=1024, r=256, dtype=W.F32, temps=(0.0, 1.0), seed=3300)
    w = W.make_weights(cfg.H, cfg.V, cfg.r, cfg.B, cfg.dtype, 3301, "strong")
    _check_sequential(X, cfg, w, W.make_inputs(cfg))


@pytest.mark.parametrize("markov", [False, True])
def test_sequential_decode_qwen3_shape(X, markov):
    cfg, w, inp = W.make_workload("qwen3_8b_greedy")
    _check_sequential(X, cfg, w, inp, markov)


def test_sequential_mode_needs_k_max_of_at_least_b(X):
    cfg = W.tiny_config("seqk", b=1, B=8, H=128, V=2080, r=256, dtype=W.BF16, seed=3400)
    w = W.make_weights(cfg.H, cfg.V, cfg.r, cfg.B, cfg.dtype, 3401, "strong")
    inp = W.make_inputs(cfg)
    ref = X.Refiner({k: X.to_device(v, X.XPRESS_BF16) for k, v in w.items()}, cfg.H, cfg.V, cfg.r, cfg.B,
                    X.XPRESS_BF16)
    d = device_inputs(X.XPRESS_BF16, inp)
    with pytest.raises(X.XpressError) as err:
        ref.refine_block(d["h"], d["s"], d["draft"], d["anchor"], d["temperature"], d["seed"], inp["offset"],
                         cfg.B - 1, mode=X.XPRESS_MODE_SEQUENTIAL)
    assert err.value.code == X.XPRESS_ERR_INVALID_ARG
    ref.close()
