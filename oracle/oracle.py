"""Python face of the float64 CPU oracle (``moe_oracle.c``).

TEST INFRASTRUCTURE ONLY: the test-suite, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` may import this module; the product path
(the CUDA library and its binding) never does, and this module imports
nothing from the product package.

Every function takes and returns numpy arrays.  bf16 tensors travel as their
uint16 bit patterns, FP8/FP4 codes as uint8, scales as float32 (FP8) or
uint8 E4M3 codes (NVFP4), exactly as they are stored on the device.

What the oracle computes is one decode step of the MoE FFN layer of the
paper's served models (Section 4 "Setup": Qwen3-Coder-480B FP8,
Qwen3-235B-A22B NVFP4; decode is weight-read bound, Section 2.1).  The
numeric readings are listed in the header of ``moe_oracle.c``.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

FMT_FP8 = 1
FMT_NVFP4 = 2

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "moe_oracle.c")
_OUT_DIR = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_OUT_DIR, "liboracle.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile ``moe_oracle.c`` with the host C compiler (OpenMP on)."""
    with _lock:
        if (not force and os.path.exists(_LIB_PATH)
                and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
            return _LIB_PATH
        os.makedirs(_OUT_DIR, exist_ok=True)
        tmp = _LIB_PATH + f".tmp{os.getpid()}"
        cmd = ["gcc", "-O2", "-fopenmp", "-shared", "-fPIC", "-o", tmp, _SRC, "-lm"]
        subprocess.run(cmd, check=True)
        os.replace(tmp, _LIB_PATH)
        return _LIB_PATH


def _load():
    global _lib
    if _lib is None:
        path = build()
        lib = ctypes.CDLL(path)
        P = ctypes.c_void_p
        I = ctypes.c_int
        lib.oracle_e4m3.restype = ctypes.c_double
        lib.oracle_e4m3.argtypes = [ctypes.c_uint8]
        lib.oracle_e2m1.restype = ctypes.c_double
        lib.oracle_e2m1.argtypes = [ctypes.c_uint8]
        lib.oracle_bf16.restype = ctypes.c_double
        lib.oracle_bf16.argtypes = [ctypes.c_uint16]
        lib.oracle_dequant.argtypes = [I, I, I, P, P, P, I, P]
        lib.oracle_router_logits.argtypes = [P, P, P, I, I, I, P]
        lib.oracle_topk.argtypes = [P, I, I, I, I, P, P]
        lib.oracle_permute.argtypes = [P, I, I, I, P, P, P, P, P]
        lib.oracle_moe_tokens.argtypes = [I, I, I, I, P, P, P, P, P, P, P, P, P, P, P, P, I, I,
                                          P, P, I, P]
        lib.oracle_expert_vec.argtypes = [I, I, I, P, P, P, P, P, P, P, P, P, I, P, P]
        lib.oracle_rmsnorm_bf16.argtypes = [P, I, I, ctypes.c_double, P]
        lib.oracle_to_bf16.argtypes = [P, ctypes.c_size_t, P]
        _lib = lib
    return _lib


def _p(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _c(a, dtype):
    return np.ascontiguousarray(a, dtype=dtype)


# ------------------------------------------------------------------ codecs
def e4m3(code: int) -> float:
    """OCP OFP8 E4M3 value of one code (0x7F/0xFF are NaN)."""
    return _load().oracle_e4m3(int(code) & 0xFF)


def e2m1(nibble: int) -> float:
    """OCP E2M1 value of one 4-bit code."""
    return _load().oracle_e2m1(int(nibble) & 0xF)


def bf16_value(bits: int) -> float:
    return _load().oracle_bf16(int(bits) & 0xFFFF)


def to_bf16_bits(v: np.ndarray) -> np.ndarray:
    """Round float64 values to bf16 (nearest, ties to even); returns uint16 bits."""
    v = _c(v, np.float64)
    out = np.empty(v.shape, np.uint16)
    _load().oracle_to_bf16(_p(v), v.size, _p(out))
    return out


# ------------------------------------------------------------------ weights
class ExpertWeights:
    """The three expert matrices of one layer in their stored (quantised) form.

    fp8:   w_* uint8 [E, N, K];   s_* float32 [E, N/128, K/128];  ts_* None
    nvfp4: w_* uint8 [E, N, K/2]; s_* uint8   [E, N, K/16];       ts_* float32 [E]
    gate/up have (N, K) = (I, H); down has (N, K) = (H, I).
    """

    def __init__(self, fmt, E, H, I, w_gate, w_up, w_down, s_gate, s_up, s_down,
                 ts_gate=None, ts_up=None, ts_down=None):
        self.fmt, self.E, self.H, self.I = fmt, E, H, I
        self.w_gate, self.w_up, self.w_down = (_c(w_gate, np.uint8), _c(w_up, np.uint8),
                                               _c(w_down, np.uint8))
        sdt = np.float32 if fmt == FMT_FP8 else np.uint8
        self.s_gate, self.s_up, self.s_down = _c(s_gate, sdt), _c(s_up, sdt), _c(s_down, sdt)
        if fmt == FMT_NVFP4:
            self.ts_gate, self.ts_up, self.ts_down = (_c(ts_gate, np.float32),
                                                      _c(ts_up, np.float32),
                                                      _c(ts_down, np.float32))
        else:
            self.ts_gate = self.ts_up = self.ts_down = None

    def dequant(self, which: str, e: int) -> np.ndarray:
        """One expert matrix as float64 [N, K]."""
        N, K = (self.I, self.H) if which in ("gate", "up") else (self.H, self.I)
        w, s, ts = (getattr(self, "w_" + which), getattr(self, "s_" + which),
                    getattr(self, "ts_" + which))
        out = np.empty((N, K), np.float64)
        _load().oracle_dequant(self.fmt, N, K, _p(w), _p(s), _p(ts), int(e), _p(out))
        return out


# ------------------------------------------------------------------ router
def router_logits(x_bits, router_w, router_bias=None) -> np.ndarray:
    """float64 logits [T, E] of bf16 x [T, H] against fp32 router rows [E, H]."""
    x_bits = _c(x_bits, np.uint16)
    router_w = _c(router_w, np.float32)
    T, H = x_bits.shape
    E = router_w.shape[0]
    b = None if router_bias is None else _c(router_bias, np.float32)
    out = np.empty((T, E), np.float64)
    _load().oracle_router_logits(_p(x_bits), _p(router_w), _p(b), T, H, E, _p(out))
    return out


def topk(logits, k: int, renorm: bool = True):
    """Top-k ids (value desc, index asc) and gate weights of float64 logits [T, E]."""
    logits = _c(logits, np.float64)
    T, E = logits.shape
    ids = np.empty((T, k), np.int32)
    gates = np.empty((T, k), np.float64)
    _load().oracle_topk(_p(logits), T, E, int(k), int(bool(renorm)), _p(ids), _p(gates))
    return ids, gates


def permute(ids, E: int):
    """counts[E], offsets[E+1], sorted[T*k], inv[T*k], active[E+1] of ids [T, k]."""
    ids = _c(ids, np.int32)
    T, k = ids.shape
    counts = np.empty(E, np.int32)
    offsets = np.empty(E + 1, np.int32)
    sorted_ = np.empty(T * k, np.int32)
    inv = np.empty(T * k, np.int32)
    active = np.zeros(E + 1, np.int32)
    _load().oracle_permute(_p(ids), T, k, E, _p(counts), _p(offsets), _p(sorted_), _p(inv),
                           _p(active))
    return counts, offsets, sorted_, inv, active


# ------------------------------------------------------------------ layer
def moe_tokens(w: ExpertWeights, x_bits, ids, gates, tokens=None, residual_bits=None):
    """float64 layer output [len(tokens), H] for the listed tokens, given the routing."""
    x_bits = _c(x_bits, np.uint16)
    ids = _c(ids, np.int32)
    gates = _c(gates, np.float64)
    T, H = x_bits.shape
    k = ids.shape[1]
    if tokens is None:
        tokens = np.arange(T, dtype=np.int32)
    tokens = _c(tokens, np.int32)
    res = None if residual_bits is None else _c(residual_bits, np.uint16)
    out = np.zeros((tokens.size, H), np.float64)
    _load().oracle_moe_tokens(w.fmt, w.E, w.H, w.I, _p(w.w_gate), _p(w.w_up), _p(w.w_down),
                              _p(w.s_gate), _p(w.s_up), _p(w.s_down), _p(w.ts_gate),
                              _p(w.ts_up), _p(w.ts_down), _p(x_bits), _p(ids), _p(gates), T, k,
                              _p(res), _p(tokens), tokens.size, _p(out))
    return out


def expert_vec(w: ExpertWeights, e: int, x) -> np.ndarray:
    """y[H] = W_d,e (silu(W_g,e x) * (W_u,e x)) for a float64 vector x[H]."""
    x = _c(x, np.float64)
    y = np.empty(w.H, np.float64)
    _load().oracle_expert_vec(w.fmt, w.H, w.I, _p(w.w_gate), _p(w.w_up), _p(w.w_down),
                              _p(w.s_gate), _p(w.s_up), _p(w.s_down), _p(w.ts_gate),
                              _p(w.ts_up), _p(w.ts_down), int(e), _p(x), _p(y))
    return y


def rmsnorm_bf16(x_bits, eps: float = 1e-6) -> np.ndarray:
    """bf16( x / sqrt(mean(x^2) + eps) ) per row; uint16 bits in and out."""
    x_bits = _c(x_bits, np.uint16)
    T, H = x_bits.shape
    out = np.empty_like(x_bits)
    _load().oracle_rmsnorm_bf16(_p(x_bits), T, H, float(eps), _p(out))
    return out


def layer(w: ExpertWeights, x_bits, router_w, k: int, router_bias=None, renorm=True,
          tokens=None, residual_bits=None):
    """The whole layer from the oracle's own routing: (out[n_tok, H], ids, gates, logits)."""
    logits = router_logits(x_bits, router_w, router_bias)
    ids, gates = topk(logits, k, renorm)
    out = moe_tokens(w, x_bits, ids, gates, tokens, residual_bits)
    return out, ids, gates, logits
