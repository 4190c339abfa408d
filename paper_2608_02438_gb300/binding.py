"""Thin ctypes binding of libxpress.so (include/xpress.h).

The functions keep the C names (``xpress_refiner_create``, ``xpress_refine_block``,
``xpress_accept`` ...) and only marshal arguments; every step of the pass runs
in the library's CUDA kernels.  PyTorch is used for device memory and streams.
Importing this module does not need a GPU; it raises if the library is missing.

:class:`Refiner` wraps the calls for torch tensors: weights and inputs are
device tensors (bf16 storage as ``torch.bfloat16``, fp32 as ``torch.float32``,
token ids ``torch.int32``, seeds ``torch.int64`` holding the uint64 bits).
"""
from __future__ import annotations

import ctypes as C
import os
import re

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)
LIB_PATH = os.path.join(HERE, "_build", "libxpress.so")
HEADER = os.path.join(ROOT, "include", "xpress.h")

XPRESS_F32, XPRESS_BF16 = 0, 1
XPRESS_ACT_SILU, XPRESS_ACT_GELU, XPRESS_ACT_RELU = 0, 1, 2
XPRESS_MODE_JACOBI, XPRESS_MODE_SEQUENTIAL = 0, 1
XPRESS_OK = 0
XPRESS_ERR_INVALID_ARG, XPRESS_ERR_UNSUPPORTED, XPRESS_ERR_CUDA = -1, -2, -3
XPRESS_ERR_WORKSPACE, XPRESS_ERR_TIMEOUT, XPRESS_ERR_DEVICE_CHECK = -4, -5, -6


class XpressWeights(C.Structure):
    _fields_ = [("H", C.c_int), ("V", C.c_int), ("r", C.c_int), ("B", C.c_int), ("dtype", C.c_int),
                ("act", C.c_int)] + [(n, C.c_void_p) for n in ("W_e", "W_h", "W_g", "W_in", "L", "W1", "W2", "W_r")]


class XpressBlockIn(C.Structure):
    _fields_ = [("b", C.c_int), ("h", C.c_void_p), ("s", C.c_void_p), ("draft", C.c_void_p),
                ("anchor", C.c_void_p), ("temperature", C.c_void_p), ("seed", C.c_void_p),
                ("offset", C.c_uint32), ("K_max", C.c_int), ("fixed_K", C.c_int), ("mode", C.c_int)]


class XpressBlockOut(C.Structure):
    _fields_ = [(n, C.c_void_p) for n in ("tokens", "iters", "converged", "lse", "logit_sel", "z_final",
                                          "refined_logits", "trajectory")]


class XpressAcceptIn(C.Structure):
    _fields_ = [("b", C.c_int)] + [(n, C.c_void_p) for n in ("target", "s", "tokens", "lse", "logit_sel",
                                                             "z_final", "temperature", "seed")] + [
        ("offset", C.c_uint32)]


class XpressTrainIn(C.Structure):
    _fields_ = [("b", C.c_int), ("B", C.c_int)] + [(n, C.c_void_p) for n in ("h", "s", "target", "ystar", "anchor",
                                                                              "xhat")] + [
        (n, C.c_float) for n in ("a_ce", "a_l1", "gamma", "lambda_", "beta")]


class XpressTrainOut(C.Structure):
    _fields_ = [(n, C.c_void_p) for n in ("loss", "gW_e", "gW_h", "gW_g", "gW_in", "gL", "gW1", "gW2", "gW_r")]


_lib = None


def declared_symbols() -> list[str]:
    """Every function name include/xpress.h declares."""
    text = open(HEADER).read()
    return sorted(set(re.findall(r"^(?:int|size_t|const char \*)\s*\*?\s*(xpress_\w+)\s*\(", text, re.M)))


def load(path: str = LIB_PATH):
    """Loads libxpress.so; raises if it has not been built (no fallback)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise RuntimeError(f"{path} is missing: run paper_2608_02438_gb300.build.build() first")
    lib = C.CDLL(path)
    P, I, S = C.c_void_p, C.c_int, C.c_size_t
    lib.xpress_version.restype = I
    lib.xpress_status_string.argtypes = [I]
    lib.xpress_status_string.restype = C.c_char_p
    lib.xpress_refiner_create.argtypes = [C.POINTER(XpressWeights), P, C.POINTER(P)]
    lib.xpress_refiner_create.restype = I
    lib.xpress_refiner_destroy.argtypes = [P]
    lib.xpress_refiner_destroy.restype = I
    lib.xpress_refine_workspace_size.argtypes = [P, I]
    lib.xpress_refine_workspace_size.restype = S
    lib.xpress_refine_block.argtypes = [P, C.POINTER(XpressBlockIn), C.POINTER(XpressBlockOut), P, S, P]
    lib.xpress_refine_block.restype = I
    lib.xpress_accept_workspace_size.argtypes = [P, I]
    lib.xpress_accept_workspace_size.restype = S
    lib.xpress_accept.argtypes = [P, C.POINTER(XpressAcceptIn), P, P, P, S, P]
    lib.xpress_accept.restype = I
    lib.xpress_get_device_status.argtypes = [P, P, C.POINTER(C.c_int32)]
    lib.xpress_get_device_status.restype = I
    lib.xpress_get_pass_count.argtypes = [P, P, C.POINTER(C.c_int32)]
    lib.xpress_get_pass_count.restype = I
    lib.xpress_accept_noalloc.argtypes = [P, C.POINTER(XpressAcceptIn), P, P, P]
    lib.xpress_accept_noalloc.restype = I
    lib.xpress_lm_head_workspace_size.argtypes = [I, I]
    lib.xpress_lm_head_workspace_size.restype = S
    lib.xpress_lm_head.argtypes = [P, I, I, P, I, P, P, P, S, P]
    lib.xpress_lm_head.restype = I
    lib.xpress_set_wait_limit.argtypes = [P, C.c_uint64]
    lib.xpress_set_wait_limit.restype = I
    lib.xpress_train_workspace_size.argtypes = [P, I, I]
    lib.xpress_train_workspace_size.restype = S
    lib.xpress_train_step.argtypes = [P, C.POINTER(XpressTrainIn), C.POINTER(XpressTrainOut), P, S, P]
    lib.xpress_train_step.restype = I
    lib.xpress_profile_train.argtypes = [P, C.POINTER(XpressTrainIn), C.POINTER(XpressTrainOut), P, S, I, P]
    lib.xpress_profile_train.restype = I
    lib.xpress_debug_gemm.argtypes = [P, I, P, I, I, I, I, P, I, P]
    lib.xpress_debug_gemm.restype = I
    lib.xpress_profile_read_prepare.argtypes = [P, P, I, I, P]
    lib.xpress_profile_read_prepare.restype = I
    lib.xpress_profile_read.argtypes = [P, P, I, P]
    lib.xpress_profile_read.restype = I
    _lib = lib
    return lib


class XpressError(RuntimeError):
    def __init__(self, where, code):
        msg = load().xpress_status_string(code).decode()
        super().__init__(f"{where}: {msg} ({code})")
        self.code = code


def _check(where, code):
    if code != XPRESS_OK:
        raise XpressError(where, code)


def _p(t):
    return None if t is None else C.c_void_p(t.data_ptr())


# ------------------------------------------------------------ raw C names

def xpress_refiner_create(weights: XpressWeights, stream: int) -> C.c_void_p:
    h = C.c_void_p()
    _check("xpress_refiner_create", load().xpress_refiner_create(C.byref(weights), C.c_void_p(stream), C.byref(h)))
    return h


def xpress_refiner_destroy(handle) -> None:
    _check("xpress_refiner_destroy", load().xpress_refiner_destroy(handle))


def xpress_refine_workspace_size(handle, b: int) -> int:
    return load().xpress_refine_workspace_size(handle, b)


def xpress_refine_block(handle, blk_in: XpressBlockIn, blk_out: XpressBlockOut, ws_ptr: int, ws_bytes: int,
                        stream: int) -> None:
    _check("xpress_refine_block", load().xpress_refine_block(handle, C.byref(blk_in), C.byref(blk_out),
                                                              C.c_void_p(ws_ptr), ws_bytes, C.c_void_p(stream)))


def xpress_accept_workspace_size(handle, b: int) -> int:
    return load().xpress_accept_workspace_size(handle, b)


def xpress_accept(handle, acc_in: XpressAcceptIn, accept_len_ptr: int, out_tokens_ptr: int, ws_ptr: int,
                  ws_bytes: int, stream: int) -> None:
    _check("xpress_accept", load().xpress_accept(handle, C.byref(acc_in), C.c_void_p(accept_len_ptr),
                                                 C.c_void_p(out_tokens_ptr), C.c_void_p(ws_ptr), ws_bytes,
                                                 C.c_void_p(stream)))


def xpress_accept_noalloc(handle, acc_in: XpressAcceptIn, accept_len_ptr: int, out_tokens_ptr: int,
                          stream: int) -> None:
    _check("xpress_accept_noalloc", load().xpress_accept_noalloc(handle, C.byref(acc_in), C.c_void_p(accept_len_ptr),
                                                                 C.c_void_p(out_tokens_ptr), C.c_void_p(stream)))


def xpress_get_device_status(ws_ptr: int, stream: int) -> int:
    v = C.c_int32()
    _check("xpress_get_device_status", load().xpress_get_device_status(C.c_void_p(ws_ptr), C.c_void_p(stream),
                                                                        C.byref(v)))
    return v.value


def xpress_get_pass_count(ws_ptr: int, stream: int) -> int:
    v = C.c_int32()
    _check("xpress_get_pass_count", load().xpress_get_pass_count(C.c_void_p(ws_ptr), C.c_void_p(stream), C.byref(v)))
    return v.value


def xpress_lm_head_workspace_size(V: int, N: int) -> int:
    return load().xpress_lm_head_workspace_size(V, N)


def xpress_lm_head(W_lm_ptr: int, V: int, H: int, h_ptr: int, N: int, s_ptr, argmax_ptr, ws_ptr: int, ws_bytes: int,
                   stream: int) -> None:
    _check("xpress_lm_head", load().xpress_lm_head(C.c_void_p(W_lm_ptr), V, H, C.c_void_p(h_ptr), N,
                                                   C.c_void_p(s_ptr) if s_ptr else None,
                                                   C.c_void_p(argmax_ptr) if argmax_ptr else None,
                                                   C.c_void_p(ws_ptr), ws_bytes, C.c_void_p(stream)))


def lm_head(W_lm, h, s_out=None, argmax_out=None, stream=None) -> int:
    """Base logits s = W_lm h (bf16 device tensors W_lm [V, H], h [N, H];
    s_out [N, V] bf16 and / or argmax_out [N] int32 device tensors) on
    `stream` (default: torch's current stream).  Returns XPRESS_OK."""
    import torch
    V, H = W_lm.shape
    N = h.shape[0]
    st = stream if stream is not None else torch.cuda.current_stream()
    size = xpress_lm_head_workspace_size(V, N)
    ws = torch.empty(size + 256, dtype=torch.uint8, device=W_lm.device)
    ptr = (ws.data_ptr() + 255) & ~255
    xpress_lm_head(W_lm.data_ptr(), V, H, h.data_ptr(), N, None if s_out is None else s_out.data_ptr(),
                   None if argmax_out is None else argmax_out.data_ptr(), ptr, size, st.cuda_stream)
    lm_head.workspace = ws                       # kept alive until the next call (the launch is asynchronous)
    return XPRESS_OK


def xpress_train_workspace_size(handle, b: int, B: int) -> int:
    return load().xpress_train_workspace_size(handle, b, B)


def xpress_train_step(handle, tin: XpressTrainIn, tout: XpressTrainOut, ws_ptr: int, ws_bytes: int,
                      stream: int) -> None:
    _check("xpress_train_step", load().xpress_train_step(handle, C.byref(tin), C.byref(tout), C.c_void_p(ws_ptr),
                                                         ws_bytes, C.c_void_p(stream)))


def xpress_profile_train(handle, tin: XpressTrainIn, tout: XpressTrainOut, ws_ptr: int, ws_bytes: int, which: int,
                         stream: int) -> None:
    _check("xpress_profile_train", load().xpress_profile_train(handle, C.byref(tin), C.byref(tout),
                                                               C.c_void_p(ws_ptr), ws_bytes, which,
                                                               C.c_void_p(stream)))


def xpress_debug_gemm(A_ptr: int, a_mn: int, B_ptr: int, b_mn: int, M: int, N: int, K: int, C_ptr: int,
                      accumulate: int, stream: int) -> None:
    _check("xpress_debug_gemm", load().xpress_debug_gemm(C.c_void_p(A_ptr), a_mn, C.c_void_p(B_ptr), b_mn, M, N, K,
                                                         C.c_void_p(C_ptr), accumulate, C.c_void_p(stream)))


def xpress_set_wait_limit(handle, limit_ns: int) -> None:
    _check("xpress_set_wait_limit", load().xpress_set_wait_limit(handle, limit_ns))


def xpress_profile_read_prepare(handle, ws_ptr: int, b: int, n_tokens: int, stream: int) -> None:
    _check("xpress_profile_read_prepare", load().xpress_profile_read_prepare(handle, C.c_void_p(ws_ptr), b, n_tokens,
                                                                              C.c_void_p(stream)))


def xpress_profile_read(handle, ws_ptr: int, b: int, stream: int) -> None:
    _check("xpress_profile_read", load().xpress_profile_read(handle, C.c_void_p(ws_ptr), b, C.c_void_p(stream)))


# ------------------------------------------------------------ torch helper

class Refiner:
    """A refiner built from device weight tensors (names as in Sec. 4.1)."""

    NAMES = ("W_e", "W_h", "W_g", "W_in", "L", "W1", "W2", "W_r")

    def __init__(self, weights: dict, H: int, V: int, r: int, B: int, dtype: int, act: int = XPRESS_ACT_SILU,
                 stream=None):
        import torch
        self.torch = torch
        self.H, self.V, self.r, self.B, self.dtype, self.act = H, V, r, B, dtype, act
        self.weights = {n: weights[n].contiguous() for n in self.NAMES}
        w = XpressWeights(H, V, r, B, dtype, act, *[self.weights[n].data_ptr() for n in self.NAMES])
        self.stream = stream if stream is not None else torch.cuda.current_stream()
        self.handle = xpress_refiner_create(w, self.stream.cuda_stream)
        self._ws = {}

    def close(self):
        if self.handle:
            xpress_refiner_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def workspace(self, kind: str, b: int):
        key = (kind, b)
        if key not in self._ws:
            if kind == "train":
                size = xpress_train_workspace_size(self.handle, b, self.B)
            else:
                size = (xpress_refine_workspace_size if kind == "refine" else xpress_accept_workspace_size)(
                    self.handle, b)
            self._ws[key] = self.torch.empty(size + 256, dtype=self.torch.uint8, device="cuda")
        buf = self._ws[key]
        ptr = (buf.data_ptr() + 255) & ~255
        return ptr, buf.numel() - (ptr - buf.data_ptr())

    def alloc_outputs(self, b: int, want_logits: bool = False, traj_K: int = 0) -> dict:
        """Output tensors; traj_K > 0 adds the debug trajectory [b, traj_K, B]
        (traj_K must equal the call's K_max), filled with -1."""
        t = self.torch
        return dict(tokens=t.empty((b, self.B), dtype=t.int32, device="cuda"),
                    iters=t.empty(b, dtype=t.int32, device="cuda"),
                    converged=t.empty(b, dtype=t.int32, device="cuda"),
                    lse=t.empty((b, self.B), dtype=t.float32, device="cuda"),
                    logit_sel=t.empty((b, self.B), dtype=t.float32, device="cuda"),
                    z_final=t.empty((b, self.B, self.r), dtype=t.float32, device="cuda"),
                    refined_logits=t.empty((b, self.B, self.V), dtype=t.float32, device="cuda") if want_logits
                    else None,
                    trajectory=t.full((b, traj_K, self.B), -1, dtype=t.int32, device="cuda") if traj_K > 0
                    else None)

    def refine_block(self, h, s, draft, anchor, temperature, seed, offset: int, K_max: int, fixed_K: bool = False,
                     out: dict | None = None, want_logits: bool = False, want_traj: bool = False,
                     mode: int = XPRESS_MODE_JACOBI) -> dict:
        b = h.shape[0]
        out = out if out is not None else self.alloc_outputs(b, want_logits, K_max if want_traj else 0)
        if out.get("trajectory") is not None and tuple(out["trajectory"].shape) != (b, K_max, self.B):
            raise ValueError("trajectory must be [b, K_max, B]")
        blk_in = XpressBlockIn(b, h.data_ptr(), s.data_ptr(), None if draft is None else draft.data_ptr(),
                               anchor.data_ptr(), temperature.data_ptr(), seed.data_ptr(), offset, K_max,
                               int(bool(fixed_K)), int(mode))
        blk_out = XpressBlockOut(*[None if out.get(n) is None else out[n].data_ptr() for n in
                                   ("tokens", "iters", "converged", "lse", "logit_sel", "z_final",
                                    "refined_logits", "trajectory")])
        ws, wsb = self.workspace("refine", b)
        xpress_refine_block(self.handle, blk_in, blk_out, ws, wsb, self.stream.cuda_stream)
        return out

    def accept(self, target, s, tokens, lse, logit_sel, z_final, temperature, seed, offset: int, out=None):
        t = self.torch
        b = target.shape[0]
        if out is None:
            out = dict(accept_len=t.empty(b, dtype=t.int32, device="cuda"),
                       out_tokens=t.empty((b, self.B + 1), dtype=t.int32, device="cuda"))
        acc_in = XpressAcceptIn(b, target.data_ptr(), None if s is None else s.data_ptr(), tokens.data_ptr(),
                                None if lse is None else lse.data_ptr(),
                                None if logit_sel is None else logit_sel.data_ptr(),
                                None if z_final is None else z_final.data_ptr(), temperature.data_ptr(),
                                seed.data_ptr(), offset)
        ws, wsb = self.workspace("accept", b)
        xpress_accept(self.handle, acc_in, out["accept_len"].data_ptr(), out["out_tokens"].data_ptr(), ws, wsb,
                      self.stream.cuda_stream)
        return out

    GRAD_NAMES = ("W_e", "W_h", "W_g", "W_in", "L", "W1", "W2", "W_r")

    def alloc_grads(self) -> dict:
        """Zeroed fp32 gradient buffers shaped like the weights."""
        t = self.torch
        return {n: t.zeros(self.weights[n].shape, dtype=t.float32, device="cuda") for n in self.GRAD_NAMES}

    def train_step(self, h, s, target, ystar, anchor, xhat=None, a_ce=1.0, a_l1=1.0, gamma=4.0, lam=0.6, beta=0.3,
                   grads: dict | None = None, loss=None, profile_pass: int | None = None) -> tuple:
        """One training step (Sec. 4.3) on b blocks: returns (loss [b, 4],
        grads); the gradients are added into `grads` (allocated zeroed when
        None).  profile_pass (benchmarks): launch only that vocabulary pass of
        a step already run with the same arguments."""
        t = self.torch
        b = h.shape[0]
        grads = grads if grads is not None else self.alloc_grads()
        loss = loss if loss is not None else t.empty((b, 4), dtype=t.float32, device="cuda")
        tin = XpressTrainIn(b, self.B, h.data_ptr(), s.data_ptr(), target.data_ptr(), ystar.data_ptr(),
                            anchor.data_ptr(), None if xhat is None else xhat.data_ptr(), a_ce, a_l1, gamma, lam, beta)
        tout = XpressTrainOut(loss.data_ptr(), *[grads[n].data_ptr() for n in self.GRAD_NAMES])
        ws, wsb = self.workspace("train", b)
        if profile_pass is None:
            xpress_train_step(self.handle, tin, tout, ws, wsb, self.stream.cuda_stream)
        else:
            xpress_profile_train(self.handle, tin, tout, ws, wsb, profile_pass, self.stream.cuda_stream)
        return loss, grads

    def device_status(self, kind: str = "refine", b: int = 1) -> int:
        ws, _ = self.workspace(kind, b)
        return xpress_get_device_status(ws, self.stream.cuda_stream)

    def control_words(self, b: int):
        """The refine workspace's control words (passes run, tokens evaluated
        over all passes, ...), read after a synchronize; for measurement."""
        self.torch.cuda.synchronize()
        ws, _ = self.workspace("refine", b)
        buf = self._ws[("refine", b)]
        off = ws - buf.data_ptr() + 64
        return buf[off:off + 32].view(self.torch.int32).cpu().tolist()

    def pass_count(self, b: int) -> int:
        ws, _ = self.workspace("refine", b)
        return xpress_get_pass_count(ws, self.stream.cuda_stream)


def to_device(arr, dtype: int, device="cuda"):
    """numpy storage array (float32, or uint16 bf16 bits) -> torch device tensor."""
    import numpy as np
    import torch
    if dtype == XPRESS_BF16:
        a = np.ascontiguousarray(arr, dtype=np.uint16).view(np.int16)
        return torch.from_numpy(a).to(device).view(torch.bfloat16)
    return torch.from_numpy(np.ascontiguousarray(arr, dtype=np.float32)).to(device)
