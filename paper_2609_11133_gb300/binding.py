"""ctypes binding of libmoe.so (the C ABI in include/moe.h).

Argument marshalling only: every function here calls the C function of the
same name and raises ``MoeError`` on a non-zero status.  The layer's steps
take torch tensors that already live on the GPU and pass their device
pointers and the current CUDA stream; the host-only calls (workspace sizes,
the kernel count of a layer call, the expert kernels' stage split) take host
values.  No computation happens in Python, and there is no fallback: if the
library cannot be loaded, calling this module's functions raises.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional

import torch

from . import build as _build

MOE_FMT_FP8_B128 = 1
MOE_FMT_NVFP4 = 2
MOE_FLAG_NO_RENORM = 0x1
MOE_FLAG_PRENORM_RMS = 0x2
MOE_FLAG_DETERMINISTIC = 0x4
_FLAG_TEST_STALL = 0x100  # test hook of moe_decode_layer (see moe.h)

_STATUS = {
    0: "MOE_OK", -1: "MOE_ERR_INVALID_ARG", -2: "MOE_ERR_UNSUPPORTED_SHAPE",
    -3: "MOE_ERR_WORKSPACE_TOO_SMALL", -4: "MOE_ERR_CUDA", -5: "MOE_ERR_DEVICE_TIMEOUT",
    -6: "MOE_ERR_BAD_EXPERT_ID", -7: "MOE_ERR_UNSUPPORTED_DEVICE",
}


class MoeError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__(f"{where}: {_STATUS.get(status, status)}")


class ExpertWeightsC(ctypes.Structure):
    _fields_ = [("fmt", ctypes.c_int), ("E", ctypes.c_int), ("H", ctypes.c_int),
                ("I", ctypes.c_int), ("w_gate", ctypes.c_void_p), ("w_up", ctypes.c_void_p),
                ("w_down", ctypes.c_void_p), ("s_gate", ctypes.c_void_p),
                ("s_up", ctypes.c_void_p), ("s_down", ctypes.c_void_p),
                ("ts_gate", ctypes.c_void_p), ("ts_up", ctypes.c_void_p),
                ("ts_down", ctypes.c_void_p)]


_lib = None
_P = ctypes.c_void_p
_I = ctypes.c_int
_SZ = ctypes.c_size_t

# name -> argtypes (restype int unless noted)
_SIGS = {
    "moe_version": [],
    "moe_workspace_size": [ctypes.POINTER(ExpertWeightsC), _I, _I, ctypes.POINTER(_SZ)],
    "moe_workspace_size_flags": [ctypes.POINTER(ExpertWeightsC), _I, _I, _I,
                                 ctypes.POINTER(_SZ)],
    "moe_route_workspace_size": [_I, _I, ctypes.POINTER(_SZ)],
    "moe_layer_kernel_count": [ctypes.POINTER(ExpertWeightsC), _I, _I, ctypes.POINTER(_I)],
    "moe_cost_split_stage": [_P, _I, _I, _I, _I, _I, _I, ctypes.c_longlong, ctypes.c_longlong,
                             ctypes.POINTER(_I)],
    "moe_stage_order": [_P, _I, _I, _I, _I, _I, _I, _I, _P, _P, _P],
    "moe_workspace_init": [_P, _SZ, _P],
    "moe_read_status": [_P, _SZ, ctypes.POINTER(_I), _P],
    "moe_route_topk": [_P, _P, _P, _I, _I, _I, _I, _I, _P, _P, _P, _P, _SZ, _P],
    "moe_permute": [_P, _I, _I, _I, _P, _P, _P, _P, _P, _P],
    "moe_expert_ffn": [_P, ctypes.POINTER(ExpertWeightsC), _P, _P, _P, _I, _I, _P, _P, _SZ, _P],
    "moe_combine": [_P, _P, _P, _I, _I, _I, _P, _P, _P],
    "moe_decode_layer": [_P, _P, _P, ctypes.POINTER(ExpertWeightsC), _I, _I, _I, _P, _P, _P,
                         _SZ, _P],
    "moe_decode_layer_noalloc": [_P, _P, _P, ctypes.POINTER(ExpertWeightsC), _I, _I, _I, _P, _P,
                                 _P],
    "moe_noalloc_read_status": [ctypes.POINTER(_I), _P],
    "moe_decode_layer_ex": [_P, _P, _P, ctypes.POINTER(ExpertWeightsC), _I, _I, _I, _P, _P, _P,
                            _SZ, _P, _P, _P, ctypes.POINTER(_P), _P],
}


def lib_path() -> str:
    return _build.LIB_PATH


def load(build_if_missing: bool = True):
    """Load libmoe.so (building it first if it is missing or stale)."""
    global _lib
    if _lib is None:
        path = _build.build() if build_if_missing else _build.LIB_PATH
        if not os.path.exists(path):
            raise RuntimeError(f"libmoe.so not found at {path}")
        lib = ctypes.CDLL(path)
        for name, args in _SIGS.items():
            fn = getattr(lib, name)
            fn.argtypes = args
            fn.restype = ctypes.c_int
        lib.moe_status_string.argtypes = [ctypes.c_int]
        lib.moe_status_string.restype = ctypes.c_char_p
        _lib = lib
    return _lib


def _check(rc: int, where: str):
    if rc != 0:
        raise MoeError(rc, where)


def _ptr(t: Optional[torch.Tensor]):
    if t is None:
        return None
    if not t.is_cuda:
        raise ValueError("tensor must be on the GPU")
    if not t.is_contiguous():
        raise ValueError("tensor must be contiguous")
    return ctypes.c_void_p(t.data_ptr())


def _stream(stream=None):
    s = torch.cuda.current_stream() if stream is None else stream
    return ctypes.c_void_p(s.cuda_stream)


def weights_struct(w) -> ExpertWeightsC:
    """C view of a layer's expert weights (any object with the synth.LayerWeights fields)."""
    return ExpertWeightsC(w.fmt, w.E, w.H, w.I, _ptr(w.w_gate), _ptr(w.w_up), _ptr(w.w_down),
                          _ptr(w.s_gate), _ptr(w.s_up), _ptr(w.s_down),
                          _ptr(getattr(w, "ts_gate", None)), _ptr(getattr(w, "ts_up", None)),
                          _ptr(getattr(w, "ts_down", None)))


def status_string(rc: int) -> str:
    return load().moe_status_string(rc).decode()


def moe_version() -> int:
    return load().moe_version()


def moe_workspace_size(w, T: int, k: int, flags: int = 0) -> int:
    """Workspace bytes of a moe_decode_layer call with these flags (flags = 0:
    moe_workspace_size, which also covers moe_expert_ffn)."""
    n = _SZ(0)
    ws = weights_struct(w)
    if flags:
        _check(load().moe_workspace_size_flags(ctypes.byref(ws), T, k, flags, ctypes.byref(n)),
               "moe_workspace_size_flags")
    else:
        _check(load().moe_workspace_size(ctypes.byref(ws), T, k, ctypes.byref(n)),
               "moe_workspace_size")
    return n.value


def moe_layer_kernel_count(w, T: int, k: int) -> int:
    n = _I(0)
    ws = weights_struct(w)
    _check(load().moe_layer_kernel_count(ctypes.byref(ws), T, k, ctypes.byref(n)),
           "moe_layer_kernel_count")
    return n.value


def moe_route_workspace_size(T: int, E: int) -> int:
    n = _SZ(0)
    _check(load().moe_route_workspace_size(T, E, ctypes.byref(n)), "moe_route_workspace_size")
    return n.value


def moe_cost_split_stage(counts, NT: int, rtiles: int, KB: int, a: int, b: int, num: int,
                         den: int) -> int:
    """The expert kernels' stage split for num / den of the total cost, run on the host
    (counts: tokens per expert, any int sequence)."""
    arr = (ctypes.c_int32 * len(counts))(*[int(c) for c in counts])
    out = _I(0)
    _check(load().moe_cost_split_stage(arr, len(counts), NT, rtiles, KB, a, b, num, den,
                                       ctypes.byref(out)), "moe_cost_split_stage")
    return out.value


def moe_stage_order(counts, NT: int, rtiles: int, KB: int, slab: int, s_begin: int, n: int):
    """Stages s_begin .. s_begin + n - 1 in the FP8 tensor-core kernel's order, run on the
    host: (item, K-block, run_end) lists."""
    arr = (ctypes.c_int32 * len(counts))(*[int(c) for c in counts])
    item, kb, end = ((ctypes.c_int32 * max(n, 1))() for _ in range(3))
    _check(load().moe_stage_order(arr, len(counts), NT, rtiles, KB, slab, s_begin, n, item, kb,
                                  end), "moe_stage_order")
    return list(item[:n]), list(kb[:n]), list(end[:n])


def alloc_workspace(nbytes: int, device=None) -> torch.Tensor:
    """A zeroed uint8 workspace tensor (256-byte aligned by the caching allocator)."""
    return torch.zeros(max(nbytes, 256), dtype=torch.uint8, device=device or "cuda")


def moe_workspace_init(ws: torch.Tensor, stream=None):
    _check(load().moe_workspace_init(_ptr(ws), ws.numel(), _stream(stream)), "moe_workspace_init")


def moe_read_status(ws: torch.Tensor, stream=None) -> int:
    st = _I(0)
    _check(load().moe_read_status(_ptr(ws), ws.numel(), ctypes.byref(st), _stream(stream)),
           "moe_read_status")
    return st.value


def moe_route_topk(x, router_w, router_bias, k: int, topk_ids, topk_w, ws, logits_out=None,
                   renorm: bool = True, stream=None):
    T, H = x.shape
    E = router_w.shape[0]
    _check(load().moe_route_topk(_ptr(x), _ptr(router_w), _ptr(router_bias), T, H, E, k,
                                 int(bool(renorm)), _ptr(topk_ids), _ptr(topk_w),
                                 _ptr(logits_out), _ptr(ws), ws.numel(), _stream(stream)),
           "moe_route_topk")


def moe_permute(topk_ids, E: int, counts, offsets, sorted_assign, inv_perm, active, stream=None):
    T, k = topk_ids.shape
    _check(load().moe_permute(_ptr(topk_ids), T, k, E, _ptr(counts), _ptr(offsets),
                              _ptr(sorted_assign), _ptr(inv_perm), _ptr(active), _stream(stream)),
           "moe_permute")


def moe_expert_ffn(x, w, offsets, sorted_assign, active, k: int, y_perm, ws, stream=None):
    T = x.shape[0]
    c = weights_struct(w)
    _check(load().moe_expert_ffn(_ptr(x), ctypes.byref(c), _ptr(offsets), _ptr(sorted_assign),
                                 _ptr(active), T, k, _ptr(y_perm), _ptr(ws), ws.numel(),
                                 _stream(stream)), "moe_expert_ffn")


def moe_combine(y_perm, topk_w, inv_perm, out, residual=None, stream=None):
    T, k = topk_w.shape
    H = out.shape[1]
    _check(load().moe_combine(_ptr(y_perm), _ptr(topk_w), _ptr(inv_perm), T, k, H,
                              _ptr(residual), _ptr(out), _stream(stream)), "moe_combine")


def moe_decode_layer(x, router_w, router_bias, w, k: int, out, ws, flags: int = 0,
                     residual=None, stream=None):
    T = x.shape[0]
    c = weights_struct(w)
    _check(load().moe_decode_layer(_ptr(x), _ptr(router_w), _ptr(router_bias), ctypes.byref(c),
                                   T, k, flags, _ptr(residual), _ptr(out), _ptr(ws), ws.numel(),
                                   _stream(stream)), "moe_decode_layer")


def moe_decode_layer_ex(x, router_w, router_bias, w, k: int, out, ws, flags: int = 0,
                        residual=None, logits_out=None, topk_ids_out=None, topk_w_out=None,
                        events=None, stream=None):
    """events: None or 4 torch.cuda.Event(enable_timing=True) recorded around the kernels."""
    T = x.shape[0]
    c = weights_struct(w)
    ev = None
    if events is not None:
        for e in events:  # torch creates the CUDA event lazily on first record
            if e.cuda_event == 0:
                e.record()
        ev = (ctypes.c_void_p * 4)(*[ctypes.c_void_p(e.cuda_event) for e in events])
    _check(load().moe_decode_layer_ex(_ptr(x), _ptr(router_w), _ptr(router_bias),
                                      ctypes.byref(c), T, k, flags, _ptr(residual), _ptr(out),
                                      _ptr(ws), ws.numel(), _ptr(logits_out), _ptr(topk_ids_out),
                                      _ptr(topk_w_out), ev, _stream(stream)),
           "moe_decode_layer_ex")


def moe_decode_layer_noalloc(x, router_w, router_bias, w, k: int, out, flags: int = 0,
                             residual=None, stream=None):
    """The fused layer on the library's own 16 MiB scratch array (no workspace
    argument, no allocation); for callers that may not allocate device memory."""
    T = x.shape[0]
    c = weights_struct(w)
    _check(load().moe_decode_layer_noalloc(_ptr(x), _ptr(router_w), _ptr(router_bias),
                                           ctypes.byref(c), T, k, flags, _ptr(residual),
                                           _ptr(out), _stream(stream)),
           "moe_decode_layer_noalloc")


def moe_noalloc_read_status(stream=None) -> int:
    """Read and clear the device status word of moe_decode_layer_noalloc's array."""
    st = _I(0)
    _check(load().moe_noalloc_read_status(ctypes.byref(st), _stream(stream)),
           "moe_noalloc_read_status")
    return st.value
