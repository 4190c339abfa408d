"""Writes the oracle's expected outputs for every block of the two batched
full-size workloads (batch 32 x block 16 at T = 1 with 25% consistent drafts;
batch 64 x block 32 with T alternating 0 / 1), so that the GPU parity tests
can compare all blocks without running the slow CPU oracle on the GPU host.

Only the oracle (``oracle/``) and the seeded input draws
(``paper_2608_02438_gb300.workloads``) are used; nothing here comes from the
CUDA path.  Each file records a digest of the inputs it was computed from;
the tests recompute it and refuse a file whose inputs differ.

For the batch-32 workload the blocks flagged ``consistent`` get the oracle's
fixed point Y* (Theorem 1: Jacobi with K_max = B from the sampled draft) as
their draft, so that they converge in one pass; those drafts are stored too
(``draft``) and are what the tests and the benchmark feed both sides.

Usage: python tests/golden/make_goldens.py [serving_b32] [long_b64]
"""
from __future__ import annotations

import multiprocessing as mp
import os
import sys
import time

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(os.path.dirname(HERE))
sys.path.insert(0, ROOT)
sys.path.insert(0, os.path.dirname(HERE))

import oracle as O  # noqa: E402
from _parity import input_digest  # noqa: E402
from paper_2608_02438_gb300 import workloads as W  # noqa: E402

NAMES = ("serving_b32", "long_b64")
_G = {}


def path_of(name: str) -> str:
    return os.path.join(HERE, f"{name}.npz")


def _model():
    cfg, w = _G["cfg"], _G["w"]
    return O.Model(w, cfg.H, cfg.V, cfg.r, cfg.B, O.BF16 if cfg.dtype == W.BF16 else O.F32)


def _ystar(i):
    cfg, inp = _G["cfg"], _G["inp"]
    o = O.jacobi(_model(), inp["h"][i], inp["s"][i], int(inp["anchor"][i]), inp["draft"][i],
                 float(inp["temperature"][i]), int(inp["seed"][i]), inp["offset"], cfg.B)
    return i, o["tokens"]


def _block(i):
    cfg, inp = _G["cfg"], _G["inp"]
    m = _model()
    T, seed = float(inp["temperature"][i]), int(inp["seed"][i])
    o = O.jacobi(m, inp["h"][i], inp["s"][i], int(inp["anchor"][i]), inp["draft"][i], T, seed, inp["offset"],
                 cfg.K_max, trajectory=True)
    n, out, _, gaps = O.accept(m, inp["target"][i], inp["s"][i], o["tokens"], o["lse"], o["sel"], o["z_final"], T,
                               seed, inp["offset"], with_gaps=True)
    return i, o, n, out, gaps


def make(name: str, procs: int) -> str:
    t0 = time.time()
    cfg, w, inp = W.make_workload(name)
    digest = input_digest(w, inp)
    _G.update(cfg=cfg, w=w, inp=inp)
    ctx = mp.get_context("fork")           # CPU only: no GPU context exists in this process
    b, B, K = inp["h"].shape[0], cfg.B, cfg.K_max
    draft = inp["draft"].copy()
    if cfg.consistent_frac > 0:
        idx = [int(i) for i in np.nonzero(inp["consistent"])[0]]
        with ctx.Pool(procs) as pool:
            for i, y in pool.imap_unordered(_ystar, idx):
                draft[i] = y
        inp["draft"] = draft
    res = dict(digest=np.array(digest), draft=draft, consistent=inp["consistent"],
               tokens=np.zeros((b, B), np.int32), iters=np.zeros(b, np.int32), converged=np.zeros(b, np.int32),
               lse=np.zeros((b, B), np.float32), sel=np.zeros((b, B), np.float32),
               z_final=np.zeros((b, B, cfg.r), np.float32),
               trajectory=np.full((b, K + 1, B), -1, np.int32), margins=np.full((b, K, B), np.nan, np.float32),
               accept_len=np.zeros(b, np.int32), out_tokens=np.zeros((b, B + 1), np.int32),
               accept_gaps=np.zeros((b, B + 2), np.float32))
    with ctx.Pool(procs) as pool:
        for i, o, n, out, gaps in pool.imap_unordered(_block, range(b)):
            it = o["iters"]
            res["tokens"][i], res["iters"][i], res["converged"][i] = o["tokens"], it, o["converged"]
            res["lse"][i], res["sel"][i], res["z_final"][i] = o["lse"], o["sel"], o["z_final"]
            res["trajectory"][i, : it + 1] = o["trajectory"]
            res["margins"][i, :it] = o["margins"]
            res["accept_len"][i], res["out_tokens"][i], res["accept_gaps"][i] = n, out, gaps
    path = path_of(name)
    np.savez_compressed(path, **res)
    print(f"{name}: {b} blocks, digest {digest}, {time.time() - t0:.0f} s -> {path}", flush=True)
    return path


if __name__ == "__main__":
    names = [a for a in sys.argv[1:] if a in NAMES] or list(NAMES)
    for nm in names:
        make(nm, os.cpu_count() or 4)
