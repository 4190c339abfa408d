"""The persistent small-batch kernel's control area across calls.

Bf16 calls of at most 32 evaluated tokens run as one persistent kernel whose
CTAs hand work to one another through counters in the caller's workspace:
two control blocks alternate from call to call (a parity word says which),
each call clearing the block the next one uses, and a refiner clears a
workspace's area the first time it meets it.  These tests interleave calls
of different batch sizes on two workspaces of one refiner, and run many calls
back to back, and require every call to give exactly the first call's outputs
(which are themselves checked against the oracle).
"""
import numpy as np
import pytest

from paper_2608_02438_gb300 import workloads as W

from _parity import compare_blocks, device_inputs, oracle_model, run_oracle

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


def _setup(X, b, seed):
    cfg = W.tiny_config("persist", b=b, B=16, H=128, V=2080, r=256, dtype=W.BF16, temps=(0.0, 1.0), seed=seed)
    w = W.make_weights(cfg.H, cfg.V, cfg.r, cfg.B, cfg.dtype, 4000, "strong")
    inp = W.make_inputs(cfg)
    return cfg, w, inp


def _call(X, ref, cfg, inp, ws):
    d = device_inputs(X.XPRESS_BF16, inp)
    b = d["h"].shape[0]
    out = ref.alloc_outputs(b, traj_K=cfg.K_max)
    blk_in = X.XpressBlockIn(b, d["h"].data_ptr(), d["s"].data_ptr(), d["draft"].data_ptr(), d["anchor"].data_ptr(),
                             d["temperature"].data_ptr(), d["seed"].data_ptr(), inp["offset"], cfg.K_max, 0)
    blk_out = X.XpressBlockOut(*[None if out.get(n) is None else out[n].data_ptr() for n in
                                 ("tokens", "iters", "converged", "lse", "logit_sel", "z_final", "refined_logits",
                                  "trajectory")])
    X.xpress_refine_block(ref.handle, blk_in, blk_out, ws.data_ptr(), ws.numel(), ref.stream.cuda_stream)
    torch.cuda.synchronize()
    assert X.xpress_get_device_status(ws.data_ptr(), ref.stream.cuda_stream) == X.XPRESS_OK
    return {k: out[k].cpu().numpy().copy() for k in ("tokens", "iters", "converged", "lse", "logit_sel", "z_final",
                                                     "trajectory")}


def test_interleaved_workspaces_and_batch_sizes(X):
    cfg1, w, inp1 = _setup(X, 1, 4100)
    cfg2, _, inp2 = _setup(X, 2, 4200)
    ref = X.Refiner({k: X.to_device(v, X.XPRESS_BF16) for k, v in w.items()}, cfg1.H, cfg1.V, cfg1.r, cfg1.B,
                    X.XPRESS_BF16)
    size = max(X.xpress_refine_workspace_size(ref.handle, 1), X.xpress_refine_workspace_size(ref.handle, 2))
    ws_a = torch.empty(size, dtype=torch.uint8, device="cuda")
    ws_b = torch.empty(size, dtype=torch.uint8, device="cuda")
    ws_a.fill_(0xA5)                                  # garbage the first call must not trust
    ws_b.fill_(0x5A)
    first = {1: _call(X, ref, cfg1, inp1, ws_a), 2: _call(X, ref, cfg2, inp2, ws_b)}
    # the first calls against the oracle
    for cfg, inp, got in ((cfg1, inp1, first[1]), (cfg2, inp2, first[2])):
        m = oracle_model(cfg, w)
        seqs = list(range(cfg.b))
        orc = {i: run_oracle(m, inp, i, cfg.K_max) for i in seqs}
        compare_blocks(got, orc, seqs, cfg.dtype)
    order = [(1, ws_b), (2, ws_a), (1, ws_a), (1, ws_a), (2, ws_b), (2, ws_a), (1, ws_b), (2, ws_b), (1, ws_a)]
    for k, (b, ws) in enumerate(order):
        cfg, inp = (cfg1, inp1) if b == 1 else (cfg2, inp2)
        got = _call(X, ref, cfg, inp, ws)
        for name in ("tokens", "iters", "converged"):
            np.testing.assert_array_equal(got[name], first[b][name], err_msg=f"call {k} (b={b}): {name}")
    ref.close()


def test_many_calls_on_one_workspace(X):
    cfg, w, inp = _setup(X, 2, 4300)
    ref = X.Refiner({k: X.to_device(v, X.XPRESS_BF16) for k, v in w.items()}, cfg.H, cfg.V, cfg.r, cfg.B,
                    X.XPRESS_BF16)
    ws = torch.empty(X.xpress_refine_workspace_size(ref.handle, 2), dtype=torch.uint8, device="cuda")
    first = _call(X, ref, cfg, inp, ws)
    for k in range(12):
        got = _call(X, ref, cfg, inp, ws)
        for name in ("tokens", "iters", "converged"):
            np.testing.assert_array_equal(got[name], first[name], err_msg=f"call {k}: {name}")
    ref.close()
