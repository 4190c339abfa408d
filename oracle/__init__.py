"""Reference CPU oracle for the xPress refinement pass (arXiv 2608.02438).

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` may import this
package.  The product path never imports it, and it shares no code with the
CUDA library: the arithmetic lives in ``xpress_oracle.c`` (plain C, fp64), this
module only marshals numpy arrays through ctypes.

What each entry point follows (see the C file for the details):

* :func:`forward`     -- the refiner map R_theta composed with Correct
  (Sec. 4.1, Eq. fuse / mix / mlp / read / correct).
* :func:`select`      -- per-position re-selection: argmax at T = 0
  (Algorithm 1); fixed-noise hierarchical Gumbel-max at T > 0 (a reading: the
  paper defines only the argmax update).
* :func:`jacobi`      -- Algorithm 1 (Sec. 4.2).
* :func:`sequential`  -- the sequential decode Y* of Theorem 1.
* :func:`accept`      -- greedy / lossless acceptance (Sec. 3.1, Sec. 4.3).
* :func:`lm_head`     -- the base logits s = W_lm h and Algorithm 1's
  Y^(0) = argmax s (Sec. 4.1, Fig. 2a).
* :func:`train_step`  -- the training objective of Sec. 4.3 and its gradient
  with respect to every refiner weight.
* :func:`philox`, :func:`uniform`, :func:`gumbel` -- Philox4x32-10
  (Salmon et al., SC'11) and the counter layout shared by both sides.

Parity pins: every function above is pinned by ``tests/test_oracle_*.py``
against closed forms, library routines, brute force or invariants that do not
call back into this module's arithmetic.
"""
from __future__ import annotations

import ctypes as C
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "xpress_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD, "libxpress_oracle.so")
_lock = threading.Lock()
_lib = None

F32, BF16 = 0, 1
SILU, GELU, RELU = 0, 1, 2
STREAM_GROUP, STREAM_ELEM, STREAM_ACCEPT, STREAM_RESID = 0, 1, 2, 3
GROUP = 32


def build(force: bool = False) -> str:
    """Compile the oracle with the host C compiler (no GPU needed)."""
    os.makedirs(_BUILD, exist_ok=True)
    if force or not os.path.exists(_LIB_PATH) or os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC):
        tmp = _LIB_PATH + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-o", tmp, _SRC, "-lm"])
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


class _Model(C.Structure):
    _fields_ = [("H", C.c_int), ("V", C.c_int), ("r", C.c_int), ("B", C.c_int),
                ("dtype", C.c_int), ("act", C.c_int)] + [
        (n, C.c_void_p) for n in ("W_e", "W_h", "W_g", "W_in", "L", "W1", "W2", "W_r")]


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = C.CDLL(build())
            P, I, D, U64, U32 = C.c_void_p, C.c_int, C.c_double, C.c_uint64, C.c_uint32
            MP = C.POINTER(_Model)
            lib.xo_round_bf16.argtypes = [D]
            lib.xo_round_bf16.restype = D
            lib.xo_philox4x32_10.argtypes = [P, P, P]
            lib.xo_uniform.argtypes = [U64, U32, U32, U32, U32]
            lib.xo_uniform.restype = D
            lib.xo_gumbel.argtypes = [U64, U32, U32, U32, U32]
            lib.xo_gumbel.restype = D
            lib.xo_forward.argtypes = [MP, P, P, P, P, P, P]
            lib.xo_select.argtypes = [P, I, D, U64, U32, I, P, P, P, P]
            lib.xo_jacobi.argtypes = [MP, P, P, C.c_int32, P, D, U64, U32, I, I, P, P, P, P, P, P, P, P, P]
            lib.xo_sequential.argtypes = [MP, P, P, C.c_int32, D, U64, U32, P, P]
            lib.xo_accept.argtypes = [MP, P, P, P, P, P, P, D, U64, U32, P, P, P, P]
            lib.xo_jacobi_seeds.argtypes = [MP, P, P, C.c_int32, P, D, P, I, U32, I, P, P]
            lib.xo_refine_accept_seeds.argtypes = [MP, P, P, P, C.c_int32, P, D, P, I, U32, I, P, P]
            lib.xo_lm_head.argtypes = [P, P, I, I, I, I, P, P, P]
            lib.xo_train_step.argtypes = [MP, P, P, P, P, C.c_int32, D, D, D, D, D, P] + [P] * 8
            for f in ("xo_forward", "xo_select", "xo_jacobi", "xo_sequential", "xo_accept",
                      "xo_jacobi_seeds", "xo_refine_accept_seeds", "xo_lm_head", "xo_train_step"):
                getattr(lib, f).restype = I
            _lib = lib
    return _lib


def _ptr(a):
    return None if a is None else a.ctypes.data_as(C.c_void_p)


def _storage(a, dtype):
    """Arrays are float32 (fp32 contract) or uint16 bf16 bit patterns."""
    want = np.float32 if dtype == F32 else np.uint16
    a = np.ascontiguousarray(a)
    if a.dtype != want:
        raise TypeError(f"expected {want.__name__} storage, got {a.dtype}")
    return a


class Model:
    """Refiner weights (Sec. 4.1) with the shapes the paper gives:
    W_e [V, r] (row x = W_e[x]), W_h, W_g [r, H], W_in [r, 3r],
    L [r, B, B] (strictly lower part used), W1 [2r, r], W2 [r, 2r], W_r [V, r].
    """

    NAMES = ("W_e", "W_h", "W_g", "W_in", "L", "W1", "W2", "W_r")

    def __init__(self, weights: dict, H: int, V: int, r: int, B: int, dtype: int, act: int = SILU):
        self.H, self.V, self.r, self.B, self.dtype, self.act = H, V, r, B, dtype, act
        shapes = {"W_e": (V, r), "W_h": (r, H), "W_g": (r, H), "W_in": (r, 3 * r),
                  "L": (r, B, B), "W1": (2 * r, r), "W2": (r, 2 * r), "W_r": (V, r)}
        self.w = {}
        for n in self.NAMES:
            a = _storage(weights[n], dtype)
            if a.shape != shapes[n]:
                raise ValueError(f"{n}: shape {a.shape} != {shapes[n]}")
            self.w[n] = a
        self.c = _Model(H, V, r, B, dtype, act, *[_ptr(self.w[n]) for n in self.NAMES])

    def _a(self, x, shape):
        a = _storage(x, self.dtype)
        if a.shape != shape:
            raise ValueError(f"shape {a.shape} != {shape}")
        return a


def round_bf16(x: float) -> float:
    return _load().xo_round_bf16(float(x))


def philox(ctr, key):
    lib = _load()
    c = np.ascontiguousarray(ctr, dtype=np.uint32)
    k = np.ascontiguousarray(key, dtype=np.uint32)
    out = np.zeros(4, dtype=np.uint32)
    lib.xo_philox4x32_10(_ptr(c), _ptr(k), _ptr(out))
    return out


def uniform(seed, index, position, stream, offset):
    return _load().xo_uniform(seed, index, position, stream, offset)


def gumbel(seed, index, position, stream, offset):
    return _load().xo_gumbel(seed, index, position, stream, offset)


def forward(m: Model, h, s, x):
    """R_theta + Correct for all B positions; x = (x_0 = anchor, x_1..x_{B-1}).
    Returns (ell [B, V], z [B, r], c [B, r]) in float64."""
    h = m._a(h, (m.B, m.H))
    s = m._a(s, (m.B, m.V))
    x = np.ascontiguousarray(x, dtype=np.int32)
    assert x.shape == (m.B,)
    ell = np.empty((m.B, m.V))
    z = np.empty((m.B, m.r))
    c = np.empty((m.B, m.r))
    if _load().xo_forward(C.byref(m.c), _ptr(h), _ptr(s), _ptr(x), _ptr(ell), _ptr(z), _ptr(c)):
        raise ValueError("token id out of range")
    return ell, z, c


def select(ell_row, T, seed=0, offset=0, k=0):
    """Returns (y, lse, sel, margin)."""
    e = np.ascontiguousarray(ell_row, dtype=np.float64)
    y = np.zeros(1, np.int32)
    out = np.zeros(3)
    lib = _load()
    lib.xo_select(_ptr(e), e.size, float(T), seed, offset, k, _ptr(y), _ptr(out[0:]),
                  out[1:].ctypes.data_as(C.c_void_p), out[2:].ctypes.data_as(C.c_void_p))
    return int(y[0]), out[0], out[1], out[2]


def jacobi(m: Model, h, s, anchor, draft, T, seed, offset, K_max, fixed_K=False, trajectory=False):
    """Algorithm 1.  Returns a dict with tokens, iters, converged, lse, sel,
    z_final (unrounded z of the last pass), min_margin, and when asked the
    trajectory Y^(0..iters) and the per-pass decision margins."""
    h = m._a(h, (m.B, m.H))
    s = m._a(s, (m.B, m.V))
    d = None if draft is None else np.ascontiguousarray(draft, dtype=np.int32)
    tok = np.zeros(m.B, np.int32)
    it = np.zeros(1, np.int32)
    cv = np.zeros(1, np.int32)
    lse = np.zeros(m.B)
    sel = np.zeros(m.B)
    z = np.zeros((m.B, m.r))
    mm = np.zeros(1)
    traj = np.full((K_max + 1, m.B), -1, np.int32) if trajectory else None
    margins = np.full((K_max, m.B), np.nan) if trajectory else None
    rc = _load().xo_jacobi(C.byref(m.c), _ptr(h), _ptr(s), int(anchor), _ptr(d), float(T), int(seed),
                           int(offset), int(K_max), int(bool(fixed_K)), _ptr(tok), _ptr(it), _ptr(cv),
                           _ptr(lse), _ptr(sel), _ptr(z), _ptr(mm), _ptr(traj), _ptr(margins))
    if rc:
        raise ValueError("invalid arguments")
    out = dict(tokens=tok, iters=int(it[0]), converged=int(cv[0]), lse=lse, sel=sel, z_final=z,
               min_margin=float(mm[0]))
    if trajectory:
        out["trajectory"] = traj[: out["iters"] + 1]
        out["margins"] = margins[: out["iters"]]
    return out


def sequential(m: Model, h, s, anchor, T=0.0, seed=0, offset=0):
    """Sequential decode Y* (Theorem 1).  Returns (ystar, margins)."""
    h = m._a(h, (m.B, m.H))
    s = m._a(s, (m.B, m.V))
    y = np.zeros(m.B, np.int32)
    mg = np.zeros(m.B)
    if _load().xo_sequential(C.byref(m.c), _ptr(h), _ptr(s), int(anchor), float(T), int(seed), int(offset),
                             _ptr(y), _ptr(mg)):
        raise ValueError("invalid arguments")
    return y, mg


def accept(m: Model, target, s, tokens, lse, sel, z_final, T, seed, offset, with_gaps=False):
    """Acceptance (Sec. 3.1).  Returns (accept_len, out_tokens [B+1], margin),
    plus, with ``with_gaps``, the per-decision margins gaps [B+2]: gaps[k]
    (k < B) of the decision at position k (T = 0: top-2 gap of target row k;
    T > 0: |u q - p| / p of the accept test), gaps[B+1] of the final token's
    draw (top-2 margin); +inf where nothing was decided."""
    tgt = m._a(target, (m.B + 1, m.V))
    s = m._a(s, (m.B, m.V))
    y = np.ascontiguousarray(tokens, dtype=np.int32)
    lse = np.ascontiguousarray(lse, dtype=np.float64)
    sel = np.ascontiguousarray(sel, dtype=np.float64)
    z = np.ascontiguousarray(z_final, dtype=np.float64)
    n = np.zeros(1, np.int32)
    out = np.zeros(m.B + 1, np.int32)
    mg = np.zeros(1)
    gaps = np.zeros(m.B + 2)
    if _load().xo_accept(C.byref(m.c), _ptr(tgt), _ptr(s), _ptr(y), _ptr(lse), _ptr(sel), _ptr(z),
                         float(T), int(seed), int(offset), _ptr(n), _ptr(out), _ptr(mg), _ptr(gaps)):
        raise ValueError("invalid arguments")
    if with_gaps:
        return int(n[0]), out, float(mg[0]), gaps
    return int(n[0]), out, float(mg[0])


def lm_head(W_lm, h, dtype):
    """Base logits s = W_lm h (Sec. 4.1, Fig. 2a) for W_lm [V, H] and h [N, H]
    in the storage dtype (F32 or BF16).  Returns (s_exact [N, V] float64,
    s_store [N, V] in the storage dtype, argmax [N] of the stored rows)."""
    W_lm = _storage(W_lm, dtype)
    h = _storage(h, dtype)
    V, H = W_lm.shape
    N = h.shape[0]
    assert h.shape == (N, H)
    s_exact = np.empty((N, V))
    s_store = np.empty((N, V), np.float32 if dtype == F32 else np.uint16)
    am = np.empty(N, np.int32)
    if _load().xo_lm_head(_ptr(W_lm), _ptr(h), V, H, N, dtype, _ptr(s_exact), _ptr(s_store), _ptr(am)):
        raise ValueError("invalid arguments")
    return s_exact, s_store, am


GRAD_NAMES = ("W_e", "W_h", "W_g", "W_in", "L", "W1", "W2", "W_r")


def train_step(m: Model, h, s, target, ystar, anchor, a_ce=1.0, a_l1=1.0, gamma=4.0, lam=0.6, beta=0.3,
               grads=True):
    """Sec. 4.3 on one block (T = 1): losses (L(p^r), L(p^b), L(p^r-hat),
    L_total) and, with grads, dL_total/dtheta for every refiner weight (dict
    of float64 arrays shaped like the weights).  lam weighs the drafter-anchor
    term and beta the consistency term, as in the total-loss equation; the
    defaults are the experimental section's values by role (consistency 0.3,
    anchor 0.6 at the start of its annealing)."""
    h = m._a(h, (m.B, m.H))
    s = m._a(s, (m.B, m.V))
    tgt = m._a(target, (m.B, m.V))
    y = np.ascontiguousarray(ystar, dtype=np.int32)
    loss = np.zeros(4)
    g = {n: np.zeros(m.w[n].shape) for n in GRAD_NAMES} if grads else None
    ptrs = [_ptr(g[n]) if grads else None for n in GRAD_NAMES]
    if _load().xo_train_step(C.byref(m.c), _ptr(h), _ptr(s), _ptr(tgt), _ptr(y), int(anchor), float(a_ce),
                             float(a_l1), float(gamma), float(lam), float(beta), _ptr(loss), *ptrs):
        raise ValueError("invalid arguments")
    return loss, g


def jacobi_seeds(m: Model, h, s, anchor, draft, T, seeds, offset, K_max):
    h = m._a(h, (m.B, m.H))
    s = m._a(s, (m.B, m.V))
    d = None if draft is None else np.ascontiguousarray(draft, dtype=np.int32)
    seeds = np.ascontiguousarray(seeds, dtype=np.uint64)
    tok = np.zeros((seeds.size, m.B), np.int32)
    it = np.zeros(seeds.size, np.int32)
    if _load().xo_jacobi_seeds(C.byref(m.c), _ptr(h), _ptr(s), int(anchor), _ptr(d), float(T), _ptr(seeds),
                               seeds.size, int(offset), int(K_max), _ptr(tok), _ptr(it)):
        raise ValueError("invalid arguments")
    return tok, it


def refine_accept_seeds(m: Model, h, s, target, anchor, draft, T, seeds, offset, K_max):
    h = m._a(h, (m.B, m.H))
    s = m._a(s, (m.B, m.V))
    tgt = m._a(target, (m.B + 1, m.V))
    d = None if draft is None else np.ascontiguousarray(draft, dtype=np.int32)
    seeds = np.ascontiguousarray(seeds, dtype=np.uint64)
    n = np.zeros(seeds.size, np.int32)
    out = np.zeros((seeds.size, m.B + 1), np.int32)
    if _load().xo_refine_accept_seeds(C.byref(m.c), _ptr(h), _ptr(s), _ptr(tgt), int(anchor), _ptr(d),
                                      float(T), _ptr(seeds), seeds.size, int(offset), int(K_max), _ptr(n),
                                      _ptr(out)):
        raise ValueError("invalid arguments")
    return n, out
