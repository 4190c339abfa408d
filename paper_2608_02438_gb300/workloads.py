"""Seeded synthetic workloads for the refinement pass.

This module only draws inputs: refiner weights, drafter hidden states h, base
logits s, target logits, draft tokens, anchors, temperatures and per-sequence
RNG seeds.  It holds none of the method's arithmetic; both the CUDA path and
the CPU oracle consume exactly the bytes it produces.

Storage convention: fp32 workloads hold ``float32`` arrays; bf16 workloads
hold ``uint16`` arrays with the bf16 bit patterns (values drawn in fp32 and
rounded to nearest-even).

Shapes follow the paper's Qwen3-8B / dFlash setting (Sec. 5.1): block 16
(32 for the long-block case), hidden 4096, vocabulary 151936, refiner rank
r = 256 (Sec. 4.1).  The paper's evaluation data (GSM8K ... MT-Bench) and its
trained weights are not available, so these seeded draws stand in for them:

* weights ~ N(0, 0.02^2) (the stated init scale), L strictly lower-triangular;
* h ~ N(0, 1);
* base logits s = W_lm h for a random tied-size LM head W_lm ~ N(0, 0.02^2):
  for fixed h each vocabulary column s[:, v] is an independent
  N(0, 0.02^2 h h^T) vector, which is drawn directly (Cholesky of the B x B
  covariance) instead of materialising the 622M-entry W_lm;
* "strong coupling" test weights (W_e ~ N(0,1), L ~ N(0, 0.3^2),
  W_r ~ N(0, 0.3^2)) make the token-dependent term large so that Jacobi runs
  several iterations; they are parity-test inputs, not measured workloads.
"""
from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np

F32, BF16 = "f32", "bf16"


@dataclass(frozen=True)
class Config:
    name: str
    b: int
    B: int
    H: int
    V: int
    r: int
    dtype: str
    K_max: int
    temps: tuple = (0.0,)            # cycled over sequences
    logits: str = "lm_head"          # lm_head | gauss4_spike | zipf
    draft: str = "argmax"            # argmax | sample
    consistent_frac: float = 0.0     # fraction of sequences whose draft is set to Y*
    seed: int = 20260000
    notes: str = field(default="", compare=False)


CONFIGS = {
    "tiny_fp32": Config("tiny_fp32", b=1, B=16, H=256, V=1024, r=256, dtype=F32, K_max=16,
                        seed=20260000, notes="batch 1, block 16, hidden 256, vocab 1024, fp32, T=0"),
    "qwen3_8b_greedy": Config("qwen3_8b_greedy", b=1, B=16, H=4096, V=151936, r=256, dtype=BF16,
                              K_max=16, seed=20260001,
                              notes="batch 1, block 16, Qwen3-8B shape, bf16, T=0"),
    "qwen3_8b_t1": Config("qwen3_8b_t1", b=1, B=16, H=4096, V=151936, r=256, dtype=BF16, K_max=16,
                          temps=(1.0,), logits="gauss4_spike", draft="sample", seed=20260002,
                          notes="batch 1, block 16, Qwen3-8B shape, bf16, T=1 lossless"),
    "serving_b32": Config("serving_b32", b=32, B=16, H=4096, V=151936, r=256, dtype=BF16, K_max=16,
                          temps=(1.0,), logits="gauss4_spike", draft="sample", consistent_frac=0.25,
                          seed=20260003, notes="batch 32, block 16, bf16, T=1, 25% consistent drafts"),
    "long_b64": Config("long_b64", b=64, B=32, H=4096, V=151936, r=256, dtype=BF16, K_max=32,
                       temps=(0.0, 1.0), logits="zipf", draft="argmax", seed=20260004,
                       notes="batch 64, block 32, bf16, T alternating 0/1, Zipf(1.1) prior"),
}


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round float32 to bf16 (nearest, ties to even); returns uint16 bits."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    sixteen = np.uint32(16)
    t = np.right_shift(u, sixteen)
    np.bitwise_and(t, np.uint32(1), out=t)
    np.add(t, np.uint32(0x7FFF), out=t)
    np.add(t, u, out=t)
    np.right_shift(t, sixteen, out=t)
    return t.astype(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    return np.left_shift(np.ascontiguousarray(b, dtype=np.uint16).astype(np.uint32), np.uint32(16)).view(np.float32)


def to_storage(x: np.ndarray, dtype: str) -> np.ndarray:
    return f32_to_bf16_bits(x) if dtype == BF16 else np.ascontiguousarray(x, dtype=np.float32)


def to_f32(x: np.ndarray, dtype: str) -> np.ndarray:
    return bf16_bits_to_f32(x) if dtype == BF16 else np.asarray(x, dtype=np.float32)


def _normal(rng, shape, std):
    return rng.standard_normal(size=shape, dtype=np.float32) * np.float32(std)


def make_weights(H: int, V: int, r: int, B: int, dtype: str, seed: int, coupling: str = "paper") -> dict:
    """Refiner weights with the paper's shapes (Sec. 4.1)."""
    rng = np.random.Generator(np.random.PCG64(seed))
    strong = coupling == "strong"
    w = {
        "W_e": _normal(rng, (V, r), 1.0 if strong else 0.02),
        "W_h": _normal(rng, (r, H), 0.02),
        "W_g": _normal(rng, (r, H), 0.02),
        "W_in": _normal(rng, (r, 3 * r), 0.02),
        "L": _normal(rng, (r, B, B), 0.3 if strong else 0.02),
        "W1": _normal(rng, (2 * r, r), 0.02),
        "W2": _normal(rng, (r, 2 * r), 0.02),
        "W_r": _normal(rng, (V, r), 0.3 if strong else 0.02),
    }
    w["L"] *= np.tril(np.ones((B, B), np.float32), k=-1)[None]
    return {k: to_storage(v, dtype) for k, v in w.items()}


def _lm_head_logits(rng, h32: np.ndarray, V: int) -> np.ndarray:
    """Draw s = W_lm h for W_lm ~ N(0, 0.02^2) [V, H] without building W_lm."""
    h64 = h32.astype(np.float64)
    cov = 0.02 ** 2 * (h64 @ h64.T)
    chol = np.linalg.cholesky(cov + 1e-12 * np.eye(cov.shape[0]))
    zs = rng.standard_normal(size=(V, h32.shape[0]), dtype=np.float32)
    return (zs @ chol.T.astype(np.float32)).T.astype(np.float32)


def _gumbel_sample(rng, logits: np.ndarray) -> np.ndarray:
    """Drafter-side sampling of Y^(0) from softmax(s) (the drafter, not the refiner)."""
    u = rng.random(size=logits.shape) * (1.0 - 2e-12) + 1e-12      # float64, strictly inside (0, 1)
    g = (-np.log(-np.log(u))).astype(np.float32)
    return np.argmax(logits + g, axis=-1).astype(np.int32)


def make_inputs(cfg: Config, b: int | None = None, seed_offset: int = 0) -> dict:
    """Per-block inputs for ``b`` sequences (default cfg.b).

    Returns a dict with h [b,B,H], s [b,B,V], target [b,B+1,V] (storage
    dtype), draft [b,B] int32, anchor [b] int32, temperature [b] float32,
    seed [b] uint64, offset (int), consistent [b] bool (sequences whose draft a
    test replaces by the oracle's Y*; the draft here is then a placeholder).
    """
    b = cfg.b if b is None else b
    rng = np.random.Generator(np.random.PCG64(cfg.seed + 7919 * seed_offset + 1))
    B, H, V = cfg.B, cfg.H, cfg.V
    h = _normal(rng, (b, B, H), 1.0)
    h_st = to_storage(h, cfg.dtype)
    h32 = to_f32(h_st, cfg.dtype)
    s = np.empty((b, B, V), np.float32)
    tgt = np.empty((b, B + 1, V), np.float32)
    if cfg.logits == "lm_head":
        for i in range(b):
            s[i] = _lm_head_logits(rng, h32[i], V)
        tgt[:] = _normal(rng, (b, B + 1, V), 4.0)
    elif cfg.logits == "gauss4_spike":
        s[:] = _normal(rng, (b, B, V), 4.0)
        tgt[:] = _normal(rng, (b, B + 1, V), 4.0)
        spike_tok = int(rng.integers(0, V))
        spike_pos = rng.random(size=(b, B)) < 0.2
        for i, k in zip(*np.nonzero(spike_pos)):
            s[i, k, spike_tok] += 8.0
            tgt[i, k, spike_tok] += 8.0
    elif cfg.logits == "zipf":
        prior = -1.1 * np.log(np.arange(1, V + 1, dtype=np.float64))
        prior -= np.log(np.exp(prior).sum())
        s[:] = _normal(rng, (b, B, V), 2.0) + prior.astype(np.float32)
        tgt[:, :B] = s + _normal(rng, (b, B, V), 1.0)
        tgt[:, B] = _normal(rng, (b, V), 2.0) + prior.astype(np.float32)
    else:
        raise ValueError(cfg.logits)
    s_st = to_storage(s, cfg.dtype)
    tgt_st = to_storage(tgt, cfg.dtype)
    s32 = to_f32(s_st, cfg.dtype)
    temps = np.array([cfg.temps[i % len(cfg.temps)] for i in range(b)], np.float32)
    if cfg.draft == "argmax":
        draft = np.argmax(s32, axis=-1).astype(np.int32)
    else:
        draft = _gumbel_sample(rng, s32)
        greedy = temps == 0
        draft[greedy] = np.argmax(s32[greedy], axis=-1)
    anchor = rng.integers(0, V, size=b).astype(np.int32)
    seeds = (np.uint64(cfg.seed) * np.uint64(1000003) + np.arange(b, dtype=np.uint64)
             + np.uint64(seed_offset) * np.uint64(65537))
    consistent = np.zeros(b, bool)
    if cfg.consistent_frac > 0:
        nc = int(round(cfg.consistent_frac * b))
        consistent[rng.permutation(b)[:nc]] = True
    return dict(h=h_st, s=s_st, target=tgt_st, draft=draft, anchor=anchor, temperature=temps,
                seed=seeds.astype(np.uint64), offset=int(7 + seed_offset), consistent=consistent)


# The training workload of Sec. 4.3 (a batch of blocks with target logits and
# ground-truth tokens); the paper gives no batch size, 32 blocks of 16 is the
# serving batch of the refinement benchmark.
TRAIN_CONFIGS = {
    "qwen3_8b_train": Config("qwen3_8b_train", b=32, B=16, H=4096, V=151936, r=256, dtype=BF16, K_max=16,
                             seed=20260005, notes="training batch 32 x block 16, Qwen3-8B shape, bf16"),
}


def make_train_inputs(cfg: Config, b: int | None = None, seed_offset: int = 0) -> dict:
    """Inputs of one training step for ``b`` blocks (default cfg.b): h [b,B,H]
    and s [b,B,V] as in make_inputs (cfg.logits recipe), target logits of the
    same positions [b,B,V] = s + N(0, 1) (a target that mostly agrees with the
    drafter), ground-truth tokens y* [b,B] drawn from softmax(target) (the
    target model's own samples), anchor [b]."""
    b = cfg.b if b is None else b
    rng = np.random.Generator(np.random.PCG64(cfg.seed + 7919 * seed_offset + 3))
    B, H, V = cfg.B, cfg.H, cfg.V
    h = _normal(rng, (b, B, H), 1.0)
    h_st = to_storage(h, cfg.dtype)
    h32 = to_f32(h_st, cfg.dtype)
    s = np.empty((b, B, V), np.float32)
    if cfg.logits == "lm_head":
        for i in range(b):
            s[i] = _lm_head_logits(rng, h32[i], V)
    else:
        s[:] = _normal(rng, (b, B, V), 4.0)
    tgt = s + _normal(rng, (b, B, V), 1.0)
    s_st = to_storage(s, cfg.dtype)
    tgt_st = to_storage(tgt, cfg.dtype)
    ystar = _gumbel_sample(rng, to_f32(tgt_st, cfg.dtype))
    anchor = rng.integers(0, V, size=b).astype(np.int32)
    return dict(h=h_st, s=s_st, target=tgt_st, ystar=ystar, anchor=anchor)


def markov_head_weights(weights: dict) -> dict:
    """The Markov-head comparison head (Sec. 2, Sec. 5 Table 3) in the
    refiner's notation: the correction for position k depends only on the id
    of token k-1, through the folded token slot -- the same W_e, W_in and W_r,
    with the hidden-state slots (W_h, W_g), the mixer L and the Trans MLP
    (W_1, W_2) switched off (zero).  Then z_k = c_k = W_in[:, 2r:3r] W_e[x_{k-1}]
    and l_k = s_k + W_r z_k, a rank-r bias table indexed by the previous
    token, decoded one position after another."""
    out = dict(weights)
    for k in ("W_h", "W_g", "L", "W1", "W2"):
        out[k] = np.zeros_like(weights[k])
    return out


_WEIGHT_CACHE: dict = {}


def config_weights(name: str, coupling: str = "paper") -> dict:
    """Weights of a named configuration (cached per process; treat as read-only)."""
    key = (name, coupling)
    if key not in _WEIGHT_CACHE:
        cfg = CONFIGS[name]
        _WEIGHT_CACHE[key] = make_weights(cfg.H, cfg.V, cfg.r, cfg.B, cfg.dtype,
                                          cfg.seed + (101 if coupling == "strong" else 0), coupling)
    return _WEIGHT_CACHE[key]


def make_workload(name: str, b: int | None = None, coupling: str = "paper", seed_offset: int = 0):
    cfg = CONFIGS[name]
    return cfg, config_weights(name, coupling), make_inputs(cfg, b, seed_offset)


def tiny_config(name="tiny", b=2, B=5, H=12, V=40, r=8, dtype=F32, K_max=None, temps=(0.0,),
                logits="lm_head", draft="argmax", seed=1234) -> Config:
    """Small shapes for CPU pins and quick GPU parity cases."""
    return Config(name, b=b, B=B, H=H, V=V, r=r, dtype=dtype, K_max=K_max or B, temps=temps,
                  logits=logits, draft=draft, seed=seed)
