"""The stored oracle outputs of the batched full-size workloads
(tests/golden/make_goldens.py) are self-consistent, without re-running the
oracle: Algorithm 1's outputs agree with the stored trajectory (the final
tokens are the last iterate; a converged block's last pass changed nothing),
blocks given the oracle's fixed point as their draft converge in one pass,
pass counts stay within K_max, margins are recorded for every executed pass,
and the stored acceptance follows the greedy rule where T = 0 and emits
exactly accept_len + 1 tokens everywhere."""
import os

import numpy as np
import pytest

from paper_2608_02438_gb300 import workloads as W

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


@pytest.mark.parametrize("name", ["serving_b32", "long_b64"])
def test_golden_is_self_consistent(name):
    g = np.load(os.path.join(GOLDEN, f"{name}.npz"))
    cfg = W.CONFIGS[name]
    b, B, K = cfg.b, cfg.B, cfg.K_max
    assert g["tokens"].shape == (b, B) and g["z_final"].shape == (b, B, cfg.r)
    assert len(str(g["digest"])) == 16
    temps = np.array([cfg.temps[i % len(cfg.temps)] for i in range(b)])
    for i in range(b):
        it = int(g["iters"][i])
        assert 1 <= it <= K
        traj = g["trajectory"][i]
        assert (traj[: it + 1] >= 0).all() and (traj[it + 1:] == -1).all()
        np.testing.assert_array_equal(traj[0], g["draft"][i])
        np.testing.assert_array_equal(traj[it], g["tokens"][i])
        assert int(g["converged"][i]) == int(np.array_equal(traj[it], traj[it - 1]))
        assert np.isfinite(g["margins"][i, :it]).all() and np.isnan(g["margins"][i, it:]).all()
        n = int(g["accept_len"][i])
        out = g["out_tokens"][i]
        assert 0 <= n <= B and (out[: n + 1] >= 0).all() and (out[n + 1:] == -1).all()
        np.testing.assert_array_equal(out[:n], g["tokens"][i, :n])
        if temps[i] <= 0:
            # the greedy rule stops at the first refined token that differs from the target's
            assert n == B or out[n] != g["tokens"][i, n]
    cons = g["consistent"]
    if cfg.consistent_frac > 0:
        assert cons.sum() == round(cfg.consistent_frac * b)
        assert (g["iters"][cons] == 1).all() and (g["converged"][cons] == 1).all()
        np.testing.assert_array_equal(g["tokens"][cons], g["draft"][cons])
