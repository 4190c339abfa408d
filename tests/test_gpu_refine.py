"""GPU parity of xpress_refine_block / xpress_accept against the CPU oracle.

Every case runs the CUDA path through the C ABI and the oracle on the same
seeded inputs; tokens, pass counts, convergence flags and accept lengths must
match exactly (documented near-ties excused, see tests/_parity.py), float
outputs within the stated tolerances.

Cases: the fp32 tiny configuration (CUDA-core Read) with the paper's init and
with strong coupling; bf16 strong-coupling shapes that exercise the tcgen05
Read with a ragged vocabulary tile (V = 2080 = 8.125 tiles of 256), the
replicated small-token layout (<= 32 tokens) and several 128-token tiles;
and the full Qwen3-8B-shape configurations at batch 1 (greedy and T = 1).
"""
import numpy as np
import pytest

import oracle as O
from paper_2608_02438_gb300 import workloads as W

from _parity import (compare_accept, compare_blocks, device_inputs, golden_oracle, load_golden, oracle_model,
                     run_oracle)

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


def _refiner(X, cfg, weights):
    dt = X.XPRESS_BF16 if cfg.dtype == W.BF16 else X.XPRESS_F32
    dev = {k: X.to_device(v, dt) for k, v in weights.items()}
    return X.Refiner(dev, cfg.H, cfg.V, cfg.r, cfg.B, dt), dt


def _run(X, cfg, weights, inp, K_max=None, fixed_K=False, want_logits=False, seqs=None):
    ref, dt = _refiner(X, cfg, weights)
    d = device_inputs(dt, inp, seqs)
    out = ref.refine_block(d["h"], d["s"], d["draft"], d["anchor"], d["temperature"], d["seed"], inp["offset"],
                           K_max or cfg.K_max, fixed_K=fixed_K, want_logits=want_logits, want_traj=True)
    torch.cuda.synchronize()
    assert ref.device_status("refine", d["h"].shape[0]) == X.XPRESS_OK
    host = {k: (v.cpu().numpy() if v is not None else None) for k, v in out.items()}
    return ref, d, host


def _oracle_all(cfg, weights, inp, seqs, K_max=None, fixed_K=False):
    m = oracle_model(cfg, weights)
    return m, {i: run_oracle(m, inp, i, K_max or cfg.K_max, fixed_K) for i in seqs}


def _check(X, cfg, weights, inp, K_max=None, fixed_K=False, logits=True):
    seqs = list(range(inp["h"].shape[0]))
    ref, d, g = _run(X, cfg, weights, inp, K_max, fixed_K, want_logits=logits)
    m, orc = _oracle_all(cfg, weights, inp, seqs, K_max, fixed_K)
    compare_blocks(g, orc, seqs, cfg.dtype, check_logits=g["refined_logits"] if logits else None, m=m, inp=inp)
    return ref, d, g, m, orc


def test_tiny_fp32_paper_init(X):
    cfg, w, inp = W.make_workload("tiny_fp32")
    _check(X, cfg, w, inp)


@pytest.mark.parametrize("temps", [(0.0,), (1.0,), (0.0, 0.7)])
def test_tiny_fp32_strong_coupling(X, temps):
    cfg = W.tiny_config("fp32s", b=4, B=16, H=256, V=1024, r=256, dtype=W.F32, temps=temps, seed=77)
    w = W.make_weights(cfg.H, cfg.V, cfg.r, cfg.B, cfg.dtype, 78, "strong")
    inp = W.make_inputs(cfg)
    _, _, g, _, orc = _check(X, cfg, w, inp)
    assert max(o["iters"] for o in orc.values()) >= 3      # multi-pass trajectories were exercised


# b * B <= 32 runs the persistent kernel: blocks of at most 16 form c in every
# Trans CTA ((1, 16), (3, 8), (2, 16)), larger blocks exchange it ((1, 32),
# (1, 24)); the others run the multi-kernel graph.
@pytest.mark.parametrize("b,B,temps", [(1, 16, (0.0,)), (3, 8, (1.0,)), (2, 16, (0.0, 1.0)), (1, 32, (0.0,)),
                                       (1, 24, (1.0,)), (5, 8, (0.0, 1.0)), (20, 8, (1.0, 0.0)),
                                       (9, 32, (0.0, 0.8))])
def test_bf16_tensor_core_path(X, b, B, temps):
    cfg = W.tiny_config("bf16s", b=b, B=B, H=128, V=2080, r=256, dtype=W.BF16, temps=temps, seed=1000 + b)
    w = W.make_weights(cfg.H, cfg.V, cfg.r, cfg.B, cfg.dtype, 2000 + b, "strong")
    inp = W.make_inputs(cfg)
    _, _, g, _, orc = _check(X, cfg, w, inp)
    assert max(o["iters"] for o in orc.values()) >= 2


# A vocabulary that is not a multiple of 32 (or of 128): the last Read range
# ends in a partial 32-row quarter whose box reaches past V (zero-filled), and
# the graph path's last 256-row tile is ragged.
@pytest.mark.parametrize("b,B,temps", [(1, 16, (0.0,)), (2, 16, (1.0, 0.0)), (4, 16, (0.0, 1.0))])
def test_bf16_ragged_vocabulary(X, b, B, temps):
    cfg = W.tiny_config("bf16v", b=b, B=B, H=128, V=2088, r=256, dtype=W.BF16, temps=temps, seed=1500 + b)
    w = W.make_weights(cfg.H, cfg.V, cfg.r, cfg.B, cfg.dtype, 2500 + b, "strong")
    inp = W.make_inputs(cfg)
    _check(X, cfg, w, inp)


# Read ranges of several 128-row blocks (V = 40008 over 144 Read CTAs: 256 or
# 288 rows each, i.e. 2 full blocks and possibly a partial third, the last
# range ending in a partial quarter),
# so that the W_r ring of the persistent kernel wraps within a pass and runs
# ahead across passes (16 of them) at a size the oracle finishes in seconds.
@pytest.mark.parametrize("b,temps", [(1, (0.0,)), (2, (1.0, 0.0))])
def test_bf16_multi_block_read_ranges(X, b, temps):
    cfg = W.tiny_config("bf16r", b=b, B=16, H=128, V=40008, r=256, dtype=W.BF16, temps=temps, seed=1700 + b)
    w = W.make_weights(cfg.H, cfg.V, cfg.r, cfg.B, cfg.dtype, 2700 + b, "strong")
    inp = W.make_inputs(cfg)
    _, _, _, _, orc = _check(X, cfg, w, inp)
    assert max(o["iters"] for o in orc.values()) >= 2


def test_bf16_fixed_k_and_cap(X):
    cfg = W.tiny_config("bf16k", b=6, B=16, H=128, V=2080, r=256, dtype=W.BF16, temps=(0.0, 1.0), seed=31)
    w = W.make_weights(cfg.H, cfg.V, cfg.r, cfg.B, cfg.dtype, 32, "strong")
    inp = W.make_inputs(cfg)
    _check(X, cfg, w, inp, K_max=5, fixed_K=True, logits=False)
    _check(X, cfg, w, inp, K_max=2, fixed_K=False, logits=False)


def test_no_draft_seeds_with_argmax(X):
    cfg = W.tiny_config("bf16n", b=3, B=8, H=128, V=2080, r=256, dtype=W.BF16, seed=41)
    w = W.make_weights(cfg.H, cfg.V, cfg.r, cfg.B, cfg.dtype, 42, "strong")
    inp = W.make_inputs(cfg)
    ref, dt = _refiner(X, cfg, w)
    d = device_inputs(dt, inp)
    out = ref.refine_block(d["h"], d["s"], None, d["anchor"], d["temperature"], d["seed"], inp["offset"], cfg.K_max)
    torch.cuda.synchronize()
    m = oracle_model(cfg, w)
    for i in range(cfg.b):
        o = O.jacobi(m, inp["h"][i], inp["s"][i], int(inp["anchor"][i]), None, 0.0, int(inp["seed"][i]),
                     inp["offset"], cfg.K_max)
        assert out["tokens"][i].cpu().numpy().tolist() == o["tokens"].tolist()
        assert int(out["iters"][i]) == o["iters"]


def test_repeat_calls_are_deterministic(X):
    cfg = W.tiny_config("bf16d", b=5, B=8, H=128, V=2080, r=256, dtype=W.BF16, temps=(1.0, 0.0), seed=51)
    w = W.make_weights(cfg.H, cfg.V, cfg.r, cfg.B, cfg.dtype, 52, "strong")
    inp = W.make_inputs(cfg)
    ref, dt = _refiner(X, cfg, w)
    d = device_inputs(dt, inp)
    outs = []
    for _ in range(3):
        o = ref.refine_block(d["h"], d["s"], d["draft"], d["anchor"], d["temperature"], d["seed"], inp["offset"],
                             cfg.K_max)
        torch.cuda.synchronize()
        outs.append({k: v.cpu().numpy().copy() for k, v in o.items() if v is not None})
    for o in outs[1:]:
        for k in ("tokens", "iters", "converged", "lse", "logit_sel", "z_final"):
            np.testing.assert_array_equal(o[k], outs[0][k], err_msg=k)


@pytest.mark.parametrize("name", ["qwen3_8b_greedy", "qwen3_8b_t1"])
def test_qwen3_shape_batch1(X, name):
    cfg, w, inp = W.make_workload(name)
    _check(X, cfg, w, inp)


# ----------------------------------------------------------------- accept

def _accept_check(X, cfg, w, inp):
    ref, d, g, m, orc = _check(X, cfg, w, inp, logits=False)
    b = inp["h"].shape[0]
    out_dev = ref.refine_block(d["h"], d["s"], d["draft"], d["anchor"], d["temperature"], d["seed"], inp["offset"],
                               cfg.K_max)
    acc = ref.accept(d["target"], d["s"], out_dev["tokens"], out_dev["lse"], out_dev["logit_sel"],
                     out_dev["z_final"], d["temperature"], d["seed"], inp["offset"])
    torch.cuda.synchronize()
    assert ref.device_status("accept", b) == X.XPRESS_OK
    alen = acc["accept_len"].cpu().numpy()
    otok = acc["out_tokens"].cpu().numpy()
    expect = {}
    for i in range(b):
        o = orc[i]
        n, out, _, gaps = O.accept(m, inp["target"][i], inp["s"][i], o["tokens"], o["lse"], o["sel"], o["z_final"],
                                   float(inp["temperature"][i]), int(inp["seed"][i]), inp["offset"], with_gaps=True)
        expect[i] = (n, out, gaps)
    compare_accept(alen, otok, expect, list(range(b)), inp["temperature"])
    return alen


@pytest.mark.parametrize("temps", [(0.0,), (1.0,), (0.0, 1.0)])
def test_accept_tiny(X, temps):
    cfg = W.tiny_config("acc", b=12, B=8, H=128, V=2080, r=256, dtype=W.BF16, temps=temps, seed=61,
                        logits="gauss4_spike", draft="sample")
    w = W.make_weights(cfg.H, cfg.V, cfg.r, cfg.B, cfg.dtype, 62, "strong")
    inp = W.make_inputs(cfg)
    _accept_check(X, cfg, w, inp)


# Batches of at most 8 blocks take the decisions inside the draw kernel (no
# separate decision launch): greedy and sampling blocks mixed, and a batch of
# one of each kind.
@pytest.mark.parametrize("b,temps", [(8, (0.0, 1.0)), (1, (1.0,)), (1, (0.0,))])
def test_accept_small_batches(X, b, temps):
    cfg = W.tiny_config("accs", b=b, B=16, H=128, V=2080, r=256, dtype=W.BF16, temps=temps, seed=63 + b,
                        logits="gauss4_spike", draft="sample")
    w = W.make_weights(cfg.H, cfg.V, cfg.r, cfg.B, cfg.dtype, 64 + b, "strong")
    inp = W.make_inputs(cfg)
    _accept_check(X, cfg, w, inp)


# A hidden size that is not a multiple of 64: the persistent kernel reads h
# and the folded projection by 64-wide K tiles, so these calls take the
# multi-kernel path; results must not change.
def test_hidden_size_not_a_multiple_of_64(X):
    cfg = W.tiny_config("h136", b=1, B=16, H=136, V=2080, r=256, dtype=W.BF16, temps=(0.0,), seed=1900)
    w = W.make_weights(cfg.H, cfg.V, cfg.r, cfg.B, cfg.dtype, 1901, "strong")
    inp = W.make_inputs(cfg)
    _check(X, cfg, w, inp)


@pytest.mark.parametrize("name", ["qwen3_8b_greedy", "qwen3_8b_t1"])
def test_accept_qwen3_shape(X, name):
    cfg, w, inp = W.make_workload(name)
    _accept_check(X, cfg, w, inp)


# ------------------------------------------------- full-size batched configs

# Every block of the batch-32 and batch-64 workloads against the oracle's
# stored outputs (tests/golden/make_goldens.py writes them with the oracle
# alone; the file's input digest must match the inputs drawn here).  Blocks
# flagged consistent carry the oracle's fixed point Y* as their draft and
# must converge in one pass.
@pytest.mark.parametrize("name", ["serving_b32", "long_b64"])
def test_batched_full_size_all_blocks(X, name):
    cfg, w, inp = W.make_workload(name)
    gold = load_golden(name, w, inp)
    ref, d, g = _run(X, cfg, w, inp)
    b = inp["h"].shape[0]
    orc = {i: golden_oracle(gold, i) for i in range(b)}
    compare_blocks(g, orc, list(range(b)), cfg.dtype, inp=inp)
    if cfg.consistent_frac > 0:
        cons = inp["consistent"]
        assert cons.any()
        assert (g["iters"][cons] == 1).all() and (g["converged"][cons] == 1).all()
        np.testing.assert_array_equal(g["tokens"][cons], inp["draft"][cons])
    # acceptance on the same blocks, from the GPU's refinement outputs
    out_dev = ref.refine_block(d["h"], d["s"], d["draft"], d["anchor"], d["temperature"], d["seed"], inp["offset"],
                               cfg.K_max)
    acc = ref.accept(d["target"], d["s"], out_dev["tokens"], out_dev["lse"], out_dev["logit_sel"],
                     out_dev["z_final"], d["temperature"], d["seed"], inp["offset"])
    torch.cuda.synchronize()
    assert ref.device_status("accept", b) == X.XPRESS_OK
    expect = {i: (int(gold["accept_len"][i]), gold["out_tokens"][i], gold["accept_gaps"][i].astype(np.float64))
              for i in range(b)}
    compare_accept(acc["accept_len"].cpu().numpy(), acc["out_tokens"].cpu().numpy(), expect, list(range(b)),
                   inp["temperature"])
