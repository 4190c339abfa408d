#!/usr/bin/env python
"""Throughput of the xPress refinement pass on GB300 (refined draft blocks/s).

One step = one refinement call (Algorithm 1 to convergence, device-side loop)
plus acceptance against the target logits, over one batch of synthetic blocks
already resident in HBM.  Default workload: the Qwen3-8B shape at batch 1,
block 16, greedy (``qwen3_8b_greedy``).  L2 is flushed (a 512 MB write)
between timed steps; steps are timed with CUDA events on the launching stream.

Also reported on the same JSON line:
  e2e           the same metric with host (pinned) inputs copied in and the
                results copied out inside the timed region;
  roofline      the dominant kernel launched alone (cold L2) against the
                measured HBM copy bandwidth: for bf16 calls of at most 32
                tokens the persistent kernel that runs the whole refinement,
                otherwise the Read + Correct + selection kernel;
  cpu_baseline  the CPU oracle on whole blocks of the same workload, on one
                core and on every core (one spawned process per core);
  fixed_K_us    the refinement with exactly K = 1, 4, 6, 8 passes (Table 3's
                shape), and accepted tokens/s = sum over blocks of
                (accepted + 1) per step;
  clocks        nvidia-smi samples taken during the timed steps.

``--impl reference`` times the CPU oracle instead (the reference arm).
Multi-GPU: one process per GPU (torchrun); blocks are independent, so every
rank runs its own batch (weak scaling) and the job time is the max over ranks.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "refined draft blocks/s (Qwen3-8B shape, block 16)"
CSRC = "paper_2608_02438_gb300/csrc/"
# sources of the kernel the roofline reports, and the ncu summary taken on them
SMALL_SOURCES = [CSRC + f for f in ("refine_small.cu", "tcv_common.cuh", "mlp_common.cuh", "reduce_common.cuh",
                                    "common.cuh")]
SMALL_SUMMARY = "profiles/k_refine_small_qwen3_8b_greedy.txt"
READ_SOURCES = [CSRC + "read_tc.cu", CSRC + "common.cuh"]
READ_SUMMARIES = {"long_b64": "profiles/k_read_tc_long_b64.txt"}
LM_SOURCES = [CSRC + "lm_head.cu", CSRC + "common.cuh"]
TRAIN_SOURCES = [CSRC + f for f in ("train_read.cu", "train_common.cuh", "kernels.h", "common.cuh")]
TRAIN_SUMMARIES = {"dz": "profiles/k_train_tok_dz_qwen3_8b_train.txt", "dW_r": "profiles/k_train_voc_qwen3_8b_train.txt"}
LM_SUMMARIES = {16: "profiles/k_lm_head32_qwen3_8b_n16.txt"}


def dist_env():
    return int(os.environ.get("RANK", 0)), int(os.environ.get("WORLD_SIZE", 1)), int(os.environ.get("LOCAL_RANK", 0))


def source_hash(paths):
    """Hash of the kernel sources' code: // comments and blank lines are left
    out, so that a comment edit does not orphan a profile taken on the code."""
    h = hashlib.sha256()
    for p in paths:
        with open(os.path.join(ROOT, p), encoding="utf-8") as f:
            for line in f:
                code = line.split("//", 1)[0].rstrip()
                if code:
                    h.update(code.encode() + b"\n")
    return h.hexdigest()[:16]


def profiled_traffic(summary: str, bytes_hash: str):
    """dram bytes per launch from the committed ncu summary, if it was taken
    on the current kernel sources."""
    path = os.path.join(ROOT, summary) if summary else ""
    if not path or not os.path.isfile(path):
        return None
    kv = {}
    for line in open(path):
        if ":" in line and not line.startswith("#"):
            k, v = line.split(":", 1)
            kv[k.strip()] = v.strip()
    if kv.get("source_hash") != bytes_hash or "dram_bytes_per_launch" not in kv:
        return None
    try:
        return float(kv["dram_bytes_per_launch"])
    except ValueError:
        return None


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        d = json.load(open(path))
        return float(d["hbm_gbs"]), float(d["bf16_tflops"]), "measured"
    return 6800.0, 1900.0, "fallback"


class ClockSampler:
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.out = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "50"], stdout=self.out,
                                         stderr=subprocess.DEVNULL)
        except (OSError, ValueError):
            self.proc = None
        time.sleep(0.3)
        return self

    def __exit__(self, *a):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self):
        self.out.flush()
        self.out.seek(0)
        sms, mx, reasons = [], 0.0, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in self.out.read().splitlines():
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 8:
                continue
            try:
                sms.append(float(parts[0]))
                mx = max(mx, float(parts[1]))
            except ValueError:
                continue
            for n, v in zip(names, parts[4:8]):
                if v.lower() in ("active", "0x1", "1"):
                    reasons.add(n)
        if not sms:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
        return {"sm_mhz": float(np.median(sms)), "sm_max_mhz": mx, "reasons": sorted(reasons), "samples": len(sms)}


GOLDEN_DRAFTS = {"serving_b32": "tests/golden/serving_b32.npz"}


def workload(name: str, seed_offset: int = 0):
    """The named workload; for serving_b32 the blocks flagged consistent get
    the oracle's fixed point Y* as their draft (stored by
    tests/golden/make_goldens.py with the oracle alone), so that they converge
    in one pass as the configuration intends."""
    from paper_2608_02438_gb300 import workloads as W
    cfg, w, inp = W.make_workload(name, seed_offset=seed_offset)
    path = GOLDEN_DRAFTS.get(name)
    if path and seed_offset == 0:
        g = np.load(os.path.join(ROOT, path))
        draft = g["draft"]
        keep = ~inp["consistent"]
        if draft.shape != inp["draft"].shape or not np.array_equal(draft[keep], inp["draft"][keep]):
            raise RuntimeError(f"{path} does not match the {name} inputs drawn here")
        inp["draft"] = draft.copy()
    return cfg, w, inp


_POOL_DATA = {}


def _oracle_blocks(args):
    """Worker: whole blocks (Algorithm 1 + acceptance) with the oracle on
    arrays memory-mapped from `folder`; returns (blocks done, seconds)."""
    folder, meta, blocks = args
    import oracle as O
    if folder not in _POOL_DATA:
        a = {k: np.load(os.path.join(folder, k + ".npy"), mmap_mode="r") for k in meta["arrays"]}
        w = {k: np.ascontiguousarray(a[k]) for k in ("W_e", "W_h", "W_g", "W_in", "L", "W1", "W2", "W_r")}
        m = O.Model(w, meta["H"], meta["V"], meta["r"], meta["B"], O.BF16 if meta["bf16"] else O.F32)
        _POOL_DATA[folder] = (m, a)
    m, a = _POOL_DATA[folder]
    t0 = time.perf_counter()
    for i in blocks:
        res = O.jacobi(m, np.ascontiguousarray(a["h"][i]), np.ascontiguousarray(a["s"][i]), int(a["anchor"][i]),
                       np.ascontiguousarray(a["draft"][i]), float(a["temperature"][i]), int(a["seed"][i]),
                       meta["offset"], meta["K_max"])
        O.accept(m, np.ascontiguousarray(a["target"][i]), np.ascontiguousarray(a["s"][i]), res["tokens"], res["lse"],
                 res["sel"], res["z_final"], float(a["temperature"][i]), int(a["seed"][i]), meta["offset"])
    return len(blocks), time.perf_counter() - t0


def cpu_baseline(name: str, budget_s: float = 30.0, inputs=None):
    """The CPU oracle as it stands (plain C, fp64), timed on whole blocks of
    the same workload: on one core, then on every core (one process per core,
    started with spawn, each refining and accepting its own blocks).  Returns
    a dict with blocks/s for both, the cores used and a description."""
    import multiprocessing as mp
    import oracle as O
    O.build()
    cfg, w, inp = inputs if inputs is not None else workload(name)
    b = inp["h"].shape[0]
    cores = max(1, len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else (os.cpu_count() or 1))
    with tempfile.TemporaryDirectory() as folder:
        arrays = dict(w)
        arrays.update({k: inp[k] for k in ("h", "s", "target", "draft", "anchor", "temperature", "seed")})
        for k, v in arrays.items():
            np.save(os.path.join(folder, k + ".npy"), np.ascontiguousarray(v))
        meta = dict(arrays=list(arrays), H=cfg.H, V=cfg.V, r=cfg.r, B=cfg.B, bf16=cfg.dtype == "bf16",
                    offset=inp["offset"], K_max=cfg.K_max)
        ctx = mp.get_context("spawn")          # the parent holds a CUDA context: never fork it
        with ctx.Pool(cores) as pool:
            # one block per worker first (start-up and page-in), then the timed rounds
            pool.map(_oracle_blocks, [(folder, meta, [k % b]) for k in range(cores)])
            n1, t1 = pool.apply(_oracle_blocks, ((folder, meta, [0]),))
            one = 1.0 / t1
            per_worker = max(1, int(budget_s / 2 * one))      # about budget_s / 2 of wall time
            t0 = time.perf_counter()
            done = pool.map(_oracle_blocks, [(folder, meta, [(k * per_worker + j) % b for j in range(per_worker)])
                                             for k in range(cores)])
            wall = time.perf_counter() - t0
    total = sum(d[0] for d in done)
    return {"one_core": one, "all_cores": total / wall, "cores": cores, "blocks": total, "wall_s": wall,
            "sample": (f"{cfg.name}: whole blocks (Algorithm 1 to convergence + acceptance), fp64 oracle; "
                       f"1 core: 1 block in {t1:.2f} s; {cores} cores: {total} blocks ({per_worker} per process) "
                       f"in {wall:.1f} s")}


def run_reference(args):
    rank, world, _ = dist_env()
    if rank != 0:
        return 0
    t0 = time.perf_counter()
    cfg, w, inp = workload(args.config)
    cb = cpu_baseline(args.config, budget_s=min(60.0, 10.0 * max(1, args.steps)), inputs=(cfg, w, inp))
    val = cb["all_cores"]
    line = {"impl": "reference", "metric": METRIC, "value": val, "unit": "blocks/s", "n_gpus": args.gpus,
            "steps": cb["blocks"], "steps_requested": args.steps, "warmup": 1,
            "ms_per_step": 1000.0 / val, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "f64", "data": "synthetic",
            "config": {"workload": cfg.name, "batch": inp["h"].shape[0], "block": cfg.B, "hidden": cfg.H,
                       "vocab": cfg.V, "rank": cfg.r, "K_max": cfg.K_max},
            "cpu_baseline": {"value": val, "unit": "blocks/s", "cores": cb["cores"], "kind": "oracle",
                             "one_core": cb["one_core"], "sample": cb["sample"]},
            "e2e": {"value": val, "unit": "blocks/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
            "wall_s": time.perf_counter() - t0}
    print(json.dumps(line), flush=True)
    return 0


def lm_head_line(us, nbytes, flops, hbm, tc_peak, tokens):
    """The base-logit LM head against its roofline: the weight stream (HBM)
    for few tokens, the bf16 tensor pipe once the arithmetic intensity nears
    the ridge point."""
    gbs = nbytes / (us * 1e-6) / 1e9
    tfs = flops / (us * 1e-6) / 1e12
    tensor = flops / nbytes >= 0.75 * tc_peak * 1e3 / hbm
    return {"kernel": "k_lm_head32" if tokens <= 32 else "k_lm_head256", "us_per_call": us, "tokens": tokens,
            "bytes_per_call": nbytes, "flops_per_call": flops, "achieved_gbs": gbs, "achieved_tflops": tfs,
            "bound": "tensor" if tensor else "hbm", "peak": tc_peak if tensor else hbm,
            "frac": tfs / tc_peak if tensor else gbs / hbm,
            "note": "s = W_lm h (bf16 out) + Y^(0) = argmax s, L2 flushed; peaks of measured"}


def train_inputs_device(torch, cfg, dev, seed):
    """The training workload drawn on the device with the recipe of
    workloads.make_train_inputs (h ~ N(0, 1); s = W_lm h for a tied-size LM
    head W_lm ~ N(0, 0.02^2), drawn through the Cholesky factor of each
    block's B x B covariance; target = s + N(0, 1); y* drawn from
    softmax(target) by the Gumbel-max trick; anchor uniform), in seconds
    instead of the half minute the host draw of 2 x 78 M logits takes."""
    g = torch.Generator(device=dev)
    g.manual_seed(seed)
    b, B, H, V = cfg.b, cfg.B, cfg.H, cfg.V
    h = torch.randn((b, B, H), generator=g, device=dev).to(torch.bfloat16)
    h64 = h.double().cpu().numpy()              # the B x B factors on the host (numpy)
    cov = 0.02 ** 2 * (h64 @ h64.transpose(0, 2, 1)) + 1e-12 * np.eye(B)
    chol = torch.from_numpy(np.linalg.cholesky(cov).astype(np.float32)).to(dev)
    s = torch.empty((b, B, V), dtype=torch.bfloat16, device=dev)
    tgt = torch.empty_like(s)
    ystar = torch.empty((b, B), dtype=torch.int32, device=dev)
    for i in range(b):
        si = chol[i] @ torch.randn((B, V), generator=g, device=dev)
        ti = si + torch.randn((B, V), generator=g, device=dev)
        s[i] = si.to(torch.bfloat16)
        tgt[i] = ti.to(torch.bfloat16)
        u = torch.rand((B, V), generator=g, device=dev, dtype=torch.float64) * (1 - 2e-12) + 1e-12
        ystar[i] = torch.argmax(tgt[i].float() - torch.log(-torch.log(u)).float(), dim=-1).int()
    anchor = torch.randint(0, V, (b,), generator=g, device=dev, dtype=torch.int32)
    return dict(h=h, s=s, target=tgt, ystar=ystar, anchor=anchor)


def train_pass_line(name, kernel, us, flops, nbytes, hbm, tc_peak):
    """One vocabulary pass of the training step against its roofline: the
    bf16 tensor pipe when its arithmetic intensity is at or above the ridge
    point of the measured peaks, else HBM."""
    tfs = flops / (us * 1e-6) / 1e12
    gbs = nbytes / (us * 1e-6) / 1e9
    tensor = flops / nbytes >= tc_peak * 1e3 / hbm
    return {"pass": name, "kernel": kernel, "us": us, "flops": flops, "bytes": nbytes, "achieved_tflops": tfs,
            "achieved_gbs": gbs, "tensor_frac": tfs / tc_peak, "hbm_frac": gbs / hbm,
            "bound": "tensor" if tensor else "hbm", "frac": tfs / tc_peak if tensor else gbs / hbm}


def train_measure(torch, X, W, ref, dev, timed_us, hbm, tc_peak, d=None, cfg=None):
    """The refiner training step (Sec. 4.3) on the training workload: the whole
    step and each vocabulary pass alone, CUDA events, L2 flushed before each
    call."""
    cfg = cfg or W.TRAIN_CONFIGS["qwen3_8b_train"]
    d = d or train_inputs_device(torch, cfg, dev, cfg.seed)
    b, B, V, r = cfg.b, cfg.B, cfg.V, cfg.r
    grads = ref.alloc_grads()
    loss = torch.empty((b, 4), dtype=torch.float32, device=dev)

    def call(which=None):
        ref.train_step(d["h"], d["s"], d["target"], d["ystar"], d["anchor"], grads=grads, loss=loss,
                       profile_pass=which)

    call()
    torch.cuda.synchronize()
    if ref.device_status("train", b) != X.XPRESS_OK or not bool(torch.isfinite(loss).all()):
        raise RuntimeError("training step: device status error or non-finite loss")
    step_us = timed_us(call)
    P = b * B
    NR = (P + 63) // 64 * 128
    rows = 2 * P
    wr, st = V * r * 2, P * V * 2
    splits = max(1, min((ref.torch.cuda.get_device_properties(dev).multi_processor_count + NR // 256) // (NR // 128),
                        (V + 63) // 64))
    f1 = 2.0 * V * r * rows
    passes = [("lse", "k_train_tok", f1, wr + st + NR * r * 2),
              ("tv", "k_train_tok", f1, wr + 2 * st + NR * r * 2),
              ("dz", "k_train_tok", 2 * f1, wr + 2 * st + NR * r * 2 + splits * NR * r * 4),
              ("dW_r", "k_train_voc", 2 * f1, wr + 2 * st + NR * r * 2 + 2 * V * r * 4)]
    lines = [train_pass_line(n, k, timed_us(lambda i=i: call(i)), f, nb, hbm, tc_peak)
             for i, (n, k, f, nb) in enumerate(passes)]
    thash = source_hash(TRAIN_SOURCES)
    for ln in lines:
        # DRAM bytes of the pass from its committed ncu summary (same sources)
        ln["traffic"] = profiled_traffic(TRAIN_SUMMARIES.get(ln["pass"], ""), thash) if cfg.name == "qwen3_8b_train" \
            else None
        ln["dram_gbs"] = ln["traffic"] / (ln["us"] * 1e-6) / 1e9 if ln["traffic"] else None
    launches = 14 + 10 + 4              # 14 products, 10 other kernels, 4 vocabulary passes (and 3 memsets)
    return {"workload": cfg.name, "blocks": b, "block": B, "positions": P, "refiner_rows": rows, "hidden": cfg.H,
            "vocab": V, "us_per_step": step_us, "positions_per_s": P / (step_us * 1e-6),
            "launches_per_step": launches, "passes": lines,
            "dominant": max(lines, key=lambda x: x["us"])["pass"],
            "loss_total_mean": float(loss[:, 3].mean().item()),
            "data": "synthetic, drawn on the device with the workload recipe",
            "note": "L2 flushed before each call; peaks of measured; gradients added into fp32 buffers"}


def run_xpress(args):
    import torch
    from paper_2608_02438_gb300 import binding as X
    from paper_2608_02438_gb300 import build as BLD
    from paper_2608_02438_gb300 import workloads as W

    rank, world, local = dist_env()
    if world > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl")
    dev = torch.device("cuda", local if world > 1 else 0)
    torch.cuda.set_device(dev)
    BLD.build()
    cfg, w, inp = workload(args.config, seed_offset=rank)
    dt = X.XPRESS_BF16 if cfg.dtype == W.BF16 else X.XPRESS_F32
    ref = X.Refiner({k: X.to_device(v, dt) for k, v in w.items()}, cfg.H, cfg.V, cfg.r, cfg.B, dt)
    stream = ref.stream
    b = inp["h"].shape[0]
    host = {"h": inp["h"], "s": inp["s"], "target": inp["target"], "draft": inp["draft"], "anchor": inp["anchor"],
            "temperature": inp["temperature"], "seed": inp["seed"].view(np.int64)}
    d = {k: (X.to_device(v, dt) if k in ("h", "s", "target") else torch.from_numpy(np.ascontiguousarray(v)).cuda())
         for k, v in host.items()}
    out = ref.alloc_outputs(b)
    acc = dict(accept_len=torch.empty(b, dtype=torch.int32, device=dev),
               out_tokens=torch.empty((b, cfg.B + 1), dtype=torch.int32, device=dev))
    flush = torch.empty(512 * 2 ** 20, dtype=torch.uint8, device=dev)

    def step():
        ref.refine_block(d["h"], d["s"], d["draft"], d["anchor"], d["temperature"], d["seed"], inp["offset"],
                         cfg.K_max, out=out)
        ref.accept(d["target"], d["s"], out["tokens"], out["lse"], out["logit_sel"], out["z_final"],
                   d["temperature"], d["seed"], inp["offset"], out=acc)

    with torch.cuda.stream(stream):
        for _ in range(max(3, args.warmup)):
            step()
        torch.cuda.synchronize()
        if ref.device_status("refine", b) != X.XPRESS_OK or ref.device_status("accept", b) != X.XPRESS_OK:
            raise RuntimeError("device status error")
        passes = ref.pass_count(b)
        ctl = ref.control_words(b)
        evaluated = ctl[4]                       # tokens evaluated over all passes
        # bf16 calls of at most 32 tokens run as one persistent kernel (unless
        # XPRESS_SMALL=0); others: init + precompute (two split-K GEMMs) +
        # Fuse/Mix, then per pass Trans + Read + reduce.  Then the two
        # acceptance kernels.
        persistent = (dt == X.XPRESS_BF16 and b * cfg.B <= 32 and os.environ.get("XPRESS_SMALL", "1") != "0")
        small = b * cfg.B <= 32
        acc_launches = 2 if b <= 8 else 3         # rows, (decide,) draw: small batches decide in the draw kernel
        if persistent:
            per_step_launches = 1 + acc_launches
        else:
            # per pass: Trans (k_mix_mlp, or k_mix_c + two k_trans_tc for bf16
            # above 32 tokens), Read, reduce (fused into the Read at <= 32 tokens)
            per_pass = 2 if small else (5 if dt == X.XPRESS_BF16 else 3)
            per_step_launches = 1 + (1 if small else 2) + 1 + passes * per_pass + acc_launches
        starts = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
        ends = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
        if world > 1:
            torch.distributed.barrier()
        torch.cuda.synchronize()
        with ClockSampler(dev.index) as clk:
            for i in range(args.steps):
                flush.zero_()
                starts[i].record(stream)
                step()
                ends[i].record(stream)
            torch.cuda.synchronize()
        ms = float(sum(s.elapsed_time(e) for s, e in zip(starts, ends)))
        if world > 1:
            tt = torch.tensor([ms], device=dev, dtype=torch.float64)
            torch.distributed.all_reduce(tt, op=torch.distributed.ReduceOp.MAX)
            ms = float(tt.item())
        value = world * b * args.steps / (ms / 1000.0)
        # accepted tokens: each block emits its accepted draft tokens plus the
        # target's correction or bonus token (Sec. 3.1), per step of refinement
        # + acceptance; every step refines the same blocks
        emitted = int((acc["accept_len"].to(torch.int64) + 1).sum().item())
        accepted_tps = world * emitted * args.steps / (ms / 1000.0)

        # e2e: pinned host inputs in, results out, inside the timed region.  A
        # step's inputs sit in one pinned staging buffer and its results in one
        # device buffer (the tensors are views), so each direction is one copy.
        def packed(arrays, device):
            offs, total = {}, 0
            for k, a in arrays.items():
                offs[k] = total
                total += (a.nbytes + 255) // 256 * 256
            buf = torch.empty(total, dtype=torch.uint8, device=device)
            return buf, offs

        host_in = {k: np.ascontiguousarray(v) for k, v in host.items()}   # storage format (bf16 as bits)
        hbuf, offs = packed(host_in, "cpu")
        hbuf = hbuf.pin_memory()
        dbuf = torch.empty_like(hbuf, device=dev)
        dt_of = {"h": torch.bfloat16 if dt == X.XPRESS_BF16 else torch.float32}
        dt_of["s"] = dt_of["target"] = dt_of["h"]
        de = {}
        for k, a in host_in.items():
            raw = torch.from_numpy(a.reshape(-1).view(np.uint8))
            hbuf[offs[k]:offs[k] + raw.numel()].copy_(raw)
            tdt = dt_of[k] if k in dt_of else {np.dtype(np.int32): torch.int32, np.dtype(np.float32): torch.float32,
                                                np.dtype(np.int64): torch.int64}[a.dtype]
            de[k] = dbuf[offs[k]:offs[k] + raw.numel()].view(tdt).view(a.shape)
        res = torch.empty(b * cfg.B + b + b * (cfg.B + 1), dtype=torch.int32, device=dev)
        res_host = torch.empty_like(res, device="cpu").pin_memory()
        out_e = dict(out)
        out_e["tokens"] = res[:b * cfg.B].view(b, cfg.B)
        acc_e = dict(accept_len=res[b * cfg.B:b * cfg.B + b],
                     out_tokens=res[b * cfg.B + b:].view(b, cfg.B + 1))
        h2d = int(hbuf.numel())
        d2h = int(res.numel() * 4)
        n_e2e = max(10, min(args.steps, 300))
        e_s = [torch.cuda.Event(enable_timing=True) for _ in range(n_e2e)]
        e_e = [torch.cuda.Event(enable_timing=True) for _ in range(n_e2e)]
        for i in range(n_e2e):
            flush.zero_()
            e_s[i].record(stream)
            dbuf.copy_(hbuf, non_blocking=True)
            ref.refine_block(de["h"], de["s"], de["draft"], de["anchor"], de["temperature"], de["seed"],
                             inp["offset"], cfg.K_max, out=out_e)
            ref.accept(de["target"], de["s"], out_e["tokens"], out_e["lse"], out_e["logit_sel"], out_e["z_final"],
                       de["temperature"], de["seed"], inp["offset"], out=acc_e)
            res_host.copy_(res, non_blocking=True)
            e_e[i].record(stream)
        torch.cuda.synchronize()
        if not np.array_equal(res_host[:b * cfg.B].numpy().reshape(b, cfg.B), out["tokens"].cpu().numpy()):
            raise RuntimeError("e2e tokens differ from the device-resident run")
        ms_e2e = float(sum(s.elapsed_time(e) for s, e in zip(e_s, e_e)))
        if world > 1:
            tt = torch.tensor([ms_e2e], device=dev, dtype=torch.float64)
            torch.distributed.all_reduce(tt, op=torch.distributed.ReduceOp.MAX)
            ms_e2e = float(tt.item())
        e2e_value = world * b * n_e2e / (ms_e2e / 1000.0)

        # roofline of the dominant kernel, launched alone with L2 flushed
        # before it (and, for context, with the previous launch's data in L2)
        step()
        torch.cuda.synchronize()
        ws_ptr, _ = ref.workspace("refine", b)
        n_tok = b * cfg.B
        reps = 50
        r_s = [torch.cuda.Event(enable_timing=True) for _ in range(reps)]
        r_e = [torch.cuda.Event(enable_timing=True) for _ in range(reps)]

        def dominant():
            if persistent:       # the whole refinement is this one launch
                ref.refine_block(d["h"], d["s"], d["draft"], d["anchor"], d["temperature"], d["seed"],
                                 inp["offset"], cfg.K_max, out=out)
            else:                # Read + Correct + selection over all b * B positions
                X.xpress_profile_read(ref.handle, ws_ptr, b, stream.cuda_stream)

        for cold in (True, False):
            for i in range(reps):
                if not persistent:
                    X.xpress_profile_read_prepare(ref.handle, ws_ptr, b, n_tok, stream.cuda_stream)
                if cold:
                    flush.zero_()
                r_s[i].record(stream)
                dominant()
                r_e[i].record(stream)
            torch.cuda.synchronize()
            times = [s.elapsed_time(e) for s, e in zip(r_s, r_e)]
            if cold:
                read_ms = float(np.mean(times))
            else:
                read_warm_ms = float(np.median(times[2:]))
        # Table 3's shape: the refinement with exactly K passes on every block
        # (no early exit), the sequential decode (B dependent passes) and the
        # Markov-head comparison head decoded the same way; L2 flushed before
        # each call
        def timed_us(call, reps=12):
            fs = [torch.cuda.Event(enable_timing=True) for _ in range(reps)]
            fe = [torch.cuda.Event(enable_timing=True) for _ in range(reps)]
            for i in range(reps):
                flush.zero_()
                fs[i].record(stream)
                call()
                fe[i].record(stream)
            torch.cuda.synchronize()
            return 1000.0 * float(np.mean([s.elapsed_time(e) for s, e in zip(fs[2:], fe[2:])]))

        fixed_us = {K: timed_us(lambda: ref.refine_block(d["h"], d["s"], d["draft"], d["anchor"], d["temperature"],
                                                         d["seed"], inp["offset"], K, fixed_K=True, out=out))
                    for K in (1, 4, 6, 8)}
        seq_K = max(cfg.K_max, cfg.B)
        seq_us = timed_us(lambda: ref.refine_block(d["h"], d["s"], d["draft"], d["anchor"], d["temperature"],
                                                   d["seed"], inp["offset"], seq_K, out=out,
                                                   mode=X.XPRESS_MODE_SEQUENTIAL))
        if ref.device_status("refine", b) != X.XPRESS_OK:
            raise RuntimeError("device status error (fixed-K / sequential calls)")
        mref = X.Refiner({k: X.to_device(v, dt) for k, v in W.markov_head_weights(w).items()}, cfg.H, cfg.V, cfg.r,
                         cfg.B, dt, stream=stream)
        markov_us = timed_us(lambda: mref.refine_block(d["h"], d["s"], d["draft"], d["anchor"], d["temperature"],
                                                       d["seed"], inp["offset"], seq_K, out=out,
                                                       mode=X.XPRESS_MODE_SEQUENTIAL))
        if mref.device_status("refine", b) != X.XPRESS_OK:
            raise RuntimeError("device status error (Markov head)")
        mref.close()

        lm_us, lm_bytes, train = None, None, None
        if dt == X.XPRESS_BF16:
            # the base logits s = W_lm h of the same hidden states (Fig. 2a), with
            # Y^(0) = argmax s: a tied-size LM head W_lm ~ N(0, 0.02^2) [V, H],
            # drawn on the device with a seeded generator
            gen = torch.Generator(device=dev)
            gen.manual_seed(20260101)
            W_lm = (torch.randn((cfg.V, cfg.H), generator=gen, device=dev, dtype=torch.float32) * 0.02).to(
                torch.bfloat16)
            h_flat = d["h"].reshape(b * cfg.B, cfg.H)
            s_lm = torch.empty((b * cfg.B, cfg.V), dtype=W_lm.dtype, device=dev)
            y0_lm = torch.empty(b * cfg.B, dtype=torch.int32, device=dev)
            lm_ws = torch.empty(X.xpress_lm_head_workspace_size(cfg.V, b * cfg.B) + 256, dtype=torch.uint8, device=dev)
            lm_ptr = (lm_ws.data_ptr() + 255) & ~255

            def lm_call():
                X.xpress_lm_head(W_lm.data_ptr(), cfg.V, cfg.H, h_flat.data_ptr(), b * cfg.B, s_lm.data_ptr(),
                                 y0_lm.data_ptr(), lm_ptr, lm_ws.numel() - (lm_ptr - lm_ws.data_ptr()), stream.cuda_stream)

            lm_call()
            lm_us = timed_us(lm_call, reps=20)
            lm_bytes = cfg.V * cfg.H * 2 + b * cfg.B * cfg.H * 2 + b * cfg.B * cfg.V * 2
            del W_lm, s_lm
            if cfg.H == 4096 and cfg.V == 151936 and cfg.B == 16:
                hbm0, tc0, _ = peaks()
                train = train_measure(torch, X, W, ref, dev, timed_us, hbm0, tc0)
    esz = 2 if dt == X.XPRESS_BF16 else 4
    sms = ref.torch.cuda.get_device_properties(dev).multi_processor_count
    if persistent:
        # algorithmic bytes of one call: the folded projection [2r, H] fp32 and
        # h once; per pass W_r; per evaluated token its s row, its E' row, its
        # z operand and a 32-byte partial per vocabulary range (written, read)
        read_kernel = "k_refine_small"
        S = min(sms - 8, (cfg.V + 127) // 128)
        read_bytes = (2 * cfg.r * cfg.H * 4 + n_tok * cfg.H * esz + passes * cfg.V * cfg.r * esz
                      + evaluated * (cfg.V * esz + cfg.r * 4 + cfg.r * esz + 2 * S * 32))
        summary, srcs = SMALL_SUMMARY, SMALL_SOURCES
    else:
        read_kernel = "k_read_tcv" if small else "k_read_tc"
        rows = 128 if small else 256
        S = min(sms, (cfg.V + rows - 1) // rows)
        read_bytes = cfg.V * cfg.r * esz + n_tok * cfg.V * esz + n_tok * cfg.r * esz + S * n_tok * 32
        summary, srcs = READ_SUMMARIES.get(cfg.name, ""), READ_SOURCES
    hbm, tc_peak, src = peaks()
    achieved = read_bytes / (read_ms / 1000.0) / 1e9
    # large token counts: the LM-head product 2 V r N; the roofline is the
    # tensor pipe (bf16 dense, measured) when its arithmetic intensity is near
    # the ridge (batch 64 x block 32: 224 of 284 flop/byte), else HBM
    read_flops = 2.0 * cfg.V * cfg.r * n_tok
    tensor_bound = (not persistent) and (not small) and read_flops / read_bytes >= 0.75 * tc_peak * 1e3 / hbm
    achieved_tf = read_flops / (read_ms / 1000.0) / 1e12
    rhash = source_hash(srcs)
    traffic = profiled_traffic(summary, rhash)

    dram_gbs = traffic / (read_ms / 1000.0) / 1e9 if traffic else None
    if rank == 0:
        cb = cpu_baseline(args.config, inputs=(cfg, w, inp))
        line = {
            "metric": METRIC, "value": value, "unit": "blocks/s", "n_gpus": world, "steps": args.steps,
            "warmup": max(3, args.warmup), "ms_per_step": ms / args.steps, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16" if dt == X.XPRESS_BF16 else "f32",
            "data": "synthetic",
            "config": {"workload": cfg.name, "batch_per_gpu": b, "block": cfg.B, "hidden": cfg.H, "vocab": cfg.V,
                       "rank": cfg.r, "K_max": cfg.K_max, "temperature": float(inp["temperature"][0]),
                       "l2": "flushed between steps (512 MB write)"},
            "tokens_per_s": value * cfg.B,
            "accepted_tokens_per_s": accepted_tps,
            "emitted_tokens_per_step": emitted,
            "passes_per_step": passes,
            "fixed_K_us_per_call": {str(k): v for k, v in fixed_us.items()},
            "fixed_K_us_per_pass": (fixed_us[8] - fixed_us[1]) / 7.0,
            "sequential_decode_us_per_call": seq_us,
            "markov_head_us_per_call": markov_us,
            "lm_head": None if lm_us is None else dict(
                lm_head_line(lm_us, lm_bytes, 2.0 * cfg.V * cfg.H * b * cfg.B, hbm, tc_peak, b * cfg.B),
                traffic=profiled_traffic(LM_SUMMARIES.get(b * cfg.B, ""), source_hash(LM_SOURCES))),
            "train_step": train,
            "e2e": {"value": e2e_value, "unit": "blocks/s", "h2d_bytes_per_step": int(h2d),
                    "d2h_bytes_per_step": int(d2h), "steps": n_e2e},
            "gpu_launches": per_step_launches * args.steps,
            "roofline": {"bound": "tensor" if tensor_bound else "hbm",
                         "achieved": achieved_tf if tensor_bound else achieved,
                         "peak": tc_peak if tensor_bound else hbm, "unit": "TFLOP/s" if tensor_bound else "GB/s",
                         "frac": (achieved_tf / tc_peak) if tensor_bound else achieved / hbm,
                         "algorithmic_gbs": achieved, "algorithmic_hbm_frac": achieved / hbm,
                         "traffic": traffic, "dram_gbs": dram_gbs,
                         "dram_frac": dram_gbs / hbm if dram_gbs else None, "peak_source": src,
                         "kernel": read_kernel, "bytes_per_launch": read_bytes, "launch_ms": read_ms,
                         "launch_ms_l2_warm": read_warm_ms,
                         "tokens_per_launch": n_tok, "passes_per_launch": passes if persistent else 1,
                         "tokens_evaluated_per_launch": evaluated if persistent else n_tok,
                         "source_hash": rhash},
            "cpu_baseline": {"value": cb["all_cores"], "unit": "blocks/s", "cores": cb["cores"], "kind": "oracle",
                             "one_core": cb["one_core"], "sample": cb["sample"]},
            "clocks": clk.summary(),
        }
        print(json.dumps(line), flush=True)
    if world > 1:
        torch.distributed.destroy_process_group()
    return 0


def run_train(args):
    """--config qwen3_8b_train: the refiner training step (Sec. 4.3) alone,
    K timed steps after W warm-up steps, L2 flushed between steps, one JSON
    line (training positions/s); the launch list and kernel captures of the
    training kernels are taken on this command."""
    import torch
    from paper_2608_02438_gb300 import binding as X
    from paper_2608_02438_gb300 import build as BLD
    from paper_2608_02438_gb300 import workloads as W

    rank, world, local = dist_env()
    if world > 1:
        print(json.dumps({"impl": "xpress", "unavailable": "the training line runs on one GPU"}))
        return 0
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    BLD.build()
    cfg = W.TRAIN_CONFIGS[args.config]
    w = W.make_weights(cfg.H, cfg.V, cfg.r, cfg.B, cfg.dtype, cfg.seed, "paper")
    ref = X.Refiner({k: X.to_device(v, X.XPRESS_BF16) for k, v in w.items()}, cfg.H, cfg.V, cfg.r, cfg.B,
                    X.XPRESS_BF16)
    stream = ref.stream
    flush = torch.empty(512 * 2 ** 20, dtype=torch.uint8, device=dev)
    hbm, tc_peak, src = peaks()

    def timed_us(call, reps=12):
        fs = [torch.cuda.Event(enable_timing=True) for _ in range(reps)]
        fe = [torch.cuda.Event(enable_timing=True) for _ in range(reps)]
        for i in range(reps):
            flush.zero_()
            fs[i].record(stream)
            call()
            fe[i].record(stream)
        torch.cuda.synchronize()
        return 1000.0 * float(np.mean([s.elapsed_time(e) for s, e in zip(fs[2:], fe[2:])]))

    with torch.cuda.stream(stream):
        d = train_inputs_device(torch, cfg, dev, cfg.seed)
        grads = ref.alloc_grads()
        loss = torch.empty((cfg.b, 4), dtype=torch.float32, device=dev)

        def step():
            ref.train_step(d["h"], d["s"], d["target"], d["ystar"], d["anchor"], grads=grads, loss=loss)

        for _ in range(max(3, args.warmup)):
            step()
        torch.cuda.synchronize()
        if ref.device_status("train", cfg.b) != X.XPRESS_OK:
            raise RuntimeError("device status error")
        st = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
        en = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
        with ClockSampler(dev.index) as clk:
            for i in range(args.steps):
                flush.zero_()
                st[i].record(stream)
                step()
                en[i].record(stream)
            torch.cuda.synchronize()
        ms = float(sum(s.elapsed_time(e) for s, e in zip(st, en)))
        tr = train_measure(torch, X, W, ref, dev, timed_us, hbm, tc_peak, d=d, cfg=cfg)
    P = cfg.b * cfg.B
    dom = max(tr["passes"], key=lambda x: x["us"])
    line = {"metric": "refiner training positions/s (Qwen3-8B shape, block 16)", "value": P * args.steps / (ms / 1e3),
            "unit": "positions/s", "n_gpus": 1, "steps": args.steps, "warmup": max(3, args.warmup),
            "ms_per_step": ms / args.steps, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "bf16", "data": "synthetic",
            "config": {"workload": cfg.name, "blocks": cfg.b, "block": cfg.B, "hidden": cfg.H, "vocab": cfg.V,
                       "rank": cfg.r, "l2": "flushed between steps (512 MB write)"},
            "gpu_launches": tr["launches_per_step"] * args.steps,
            "roofline": {"bound": dom["bound"], "kernel": dom["kernel"], "pass": dom["pass"],
                         "achieved": dom["achieved_tflops"] if dom["bound"] == "tensor" else dom["achieved_gbs"],
                         "peak": tc_peak if dom["bound"] == "tensor" else hbm,
                         "unit": "TFLOP/s" if dom["bound"] == "tensor" else "GB/s", "frac": dom["frac"],
                         "traffic": dom.get("traffic"), "dram_gbs": dom.get("dram_gbs"),
                         "dram_frac": dom["dram_gbs"] / hbm if dom.get("dram_gbs") else None, "peak_source": src,
                         "source_hash": source_hash(TRAIN_SOURCES)},
            "train_step": tr, "clocks": clk.summary()}
    print(json.dumps(line), flush=True)
    ref.close()
    return 0


def main():
    ap = argparse.ArgumentParser(description=__doc__.splitlines()[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", default="xpress", choices=["xpress", "reference"])
    ap.add_argument("--config", default="qwen3_8b_greedy")
    args = ap.parse_args()
    if args.impl == "reference":
        return run_reference(args)
    from paper_2608_02438_gb300 import workloads as W
    if args.config in W.TRAIN_CONFIGS:
        return run_train(args)
    return run_xpress(args)


if __name__ == "__main__":
    sys.exit(main())
