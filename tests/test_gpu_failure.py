"""Failure detection of the persistent small-batch kernel, without a GPU fault.

Every wait of the persistent kernel for another CTA's progress is bounded
(2 s by default).  xpress_set_wait_limit(refiner, 0) makes each such wait give
up unless its counter has already been reached at its first poll, so the
first wait that must actually wait (a Trans CTA for the Read CTAs'
precompute, at the latest the end of the first pass) runs out.  The test
checks that the call then returns (the stream synchronises), that the status
word reads XPRESS_ERR_TIMEOUT, and that the next calls on the same workspace,
with the default limit back, are clean and match the CPU oracle exactly.

The batch-32 graph path with at most 32 tokens (k_read_tcv, used when the
persistent kernel cannot be launched, or with XPRESS_SMALL=0) is covered by
re-running the small-batch parity cases in a child process with
XPRESS_SMALL=0.
"""
import os
import subprocess
import sys

import numpy as np
import pytest

from paper_2608_02438_gb300 import workloads as W

from _parity import compare_blocks, device_inputs, oracle_model, run_oracle

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def X():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_02438_gb300 import binding, build
    build.build()
    binding.load()
    return binding


def test_wait_that_runs_out_reports_timeout_and_leaves_the_workspace_usable(X):
    cfg = W.tiny_config("timeout", b=2, B=16, H=1024, V=2080, r=256, dtype=W.BF16, temps=(0.0, 1.0), seed=91)
    w = W.make_weights(cfg.H, cfg.V, cfg.r, cfg.B, cfg.dtype, 92, "strong")
    inp = W.make_inputs(cfg)
    ref = X.Refiner({k: X.to_device(v, X.XPRESS_BF16) for k, v in w.items()}, cfg.H, cfg.V, cfg.r, cfg.B,
                    X.XPRESS_BF16)
    d = device_inputs(X.XPRESS_BF16, inp)
    m = oracle_model(cfg, w)
    orc = {i: run_oracle(m, inp, i, cfg.K_max) for i in range(cfg.b)}

    def call():
        out = ref.refine_block(d["h"], d["s"], d["draft"], d["anchor"], d["temperature"], d["seed"], inp["offset"],
                               cfg.K_max, want_traj=True)
        torch.cuda.synchronize()                       # returns: every CTA has left
        return out

    for rnd in range(2):
        X.xpress_set_wait_limit(ref.handle, 0)
        call()
        assert ref.device_status("refine", cfg.b) == X.XPRESS_ERR_TIMEOUT, f"round {rnd}"
        X.xpress_set_wait_limit(ref.handle, 2_000_000_000)
        for _ in range(2):
            out = call()
            assert ref.device_status("refine", cfg.b) == X.XPRESS_OK
            g = {k: (v.cpu().numpy() if v is not None else None) for k, v in out.items()}
            compare_blocks(g, orc, list(range(cfg.b)), cfg.dtype, inp=inp)
    ref.close()


def test_small_batch_graph_path_parity_in_child_process():
    env = dict(os.environ, XPRESS_SMALL="0")
    cmd = [sys.executable, "-m", "pytest", "-x", "-q", "-m", "gpu", "-p", "no:cacheprovider",
           os.path.join(ROOT, "tests", "test_gpu_refine.py"), "-k", "tensor_core_path or ragged_vocabulary or no_draft"]
    r = subprocess.run(cmd, cwd=ROOT, env=env, capture_output=True, text=True, timeout=900)
    assert r.returncode == 0, r.stdout[-4000:] + r.stderr[-2000:]
    assert " passed" in r.stdout
