"""Thin ctypes binding of libonexn.so (include/onexn.h), same call names.

Argument marshalling only: numpy arrays for the host calls, torch device
tensors (pointers and the current CUDA stream) for ``onexn_conv_fwd``.  All
arithmetic happens in the library.  Importing this module loads the shared
library and fails loudly if it has not been built; there is no fallback.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

ONEXN_OK, ONEXN_EINVAL, ONEXN_EUNSUPPORTED, ONEXN_ENOMEM = 0, 1, 2, 3
ONEXN_ECUDA, ONEXN_EDEVICE, ONEXN_ETIMEOUT = 4, 5, 6
ONEXN_F32, ONEXN_BF16 = 0, 1
ONEXN_GRAN_TAP, ONEXN_GRAN_KERNEL = 0, 1
ONEXN_RELU = 0x1
ONEXN_RELU6 = 0x2
ONEXN_DECODED = 0x10
ONEXN_REUSE_DECODE = 0x20
ONEXN_ACCUMULATE = 0x40
ONEXN_CHECK_INPUT = 0x80
ONEXN_ALGO_SHIFT = 8
ONEXN_ALGO_MASK = 0xF << ONEXN_ALGO_SHIFT
ONEXN_ALGO_AUTO = 0 << ONEXN_ALGO_SHIFT
ONEXN_ALGO_FMA = 1 << ONEXN_ALGO_SHIFT
ONEXN_ALGO_MMA = 2 << ONEXN_ALGO_SHIFT
ONEXN_ALGO_TC = 3 << ONEXN_ALGO_SHIFT
ALGO_NAMES = {ONEXN_ALGO_FMA: "fma", ONEXN_ALGO_MMA: "mma", ONEXN_ALGO_TC: "tc"}
ALGO_BY_NAME = {v: k for k, v in ALGO_NAMES.items()}
ALGO_BY_NAME["auto"] = ONEXN_ALGO_AUTO

_STATUS = {0: "OK", 1: "EINVAL", 2: "EUNSUPPORTED", 3: "ENOMEM", 4: "ECUDA", 5: "EDEVICE",
           6: "ETIMEOUT"}

_SO = os.path.join(os.path.dirname(os.path.abspath(__file__)), "_lib", "libonexn.so")

# Every function the header declares, with its ctypes signature.
_P = ctypes.c_void_p
_I32, _I64, _DBL, _U32 = ctypes.c_int, ctypes.c_int64, ctypes.c_double, ctypes.c_uint


class ConvDesc(ctypes.Structure):
    """Mirror of onexn_conv_desc."""
    _fields_ = [(n, ctypes.c_int) for n in (
        "B", "H", "W", "C_in", "C_out", "KH", "KW",
        "stride_h", "stride_w", "pad_h", "pad_w", "dil_h", "dil_w")]


SIGNATURES = {
    "onexn_last_error": ([], ctypes.c_char_p),
    "onexn_version": ([], _I32),
    "onexn_keep_count": ([_I64, _DBL, _P], _I32),
    "onexn_prune": ([_P, _I32, _I32, _I32, _I32, _I32, _DBL, _I32, _P, _P], _I32),
    "onexn_rearrange": ([_P, _I32, _I32, _I32, _I32, _P, _I32, _I32, _I32, _P], _I32),
    "onexn_pack": ([_P, _P, _I32, _I32, _I32, _I32, _I32, _I32, _P, _P, _P, _I64, _P], _I32),
    "onexn_packed_validate": ([_P, _P, _I32, _I64, _I32], _I32),
    "onexn_conv_out_shape": ([ctypes.POINTER(ConvDesc), _P, _P], _I32),
    "onexn_conv_fwd": ([ctypes.POINTER(ConvDesc), _P, _P, _P, _I32, _I64, _P, _P, _P, _I32,
                        _U32, _P, ctypes.c_size_t, _P], _I32),
    "onexn_conv_workspace_size": ([ctypes.POINTER(ConvDesc), _I32, _I64, _I32, _U32, _P], _I32),
    "onexn_conv_algo": ([ctypes.POINTER(ConvDesc), _I32, _I64, _I32, _U32, ctypes.c_size_t, _P],
                        _I32),
    "onexn_conv_tc_form": ([ctypes.POINTER(ConvDesc), _I32, _I64, _I32, _P], _I32),
    "onexn_conv_halo_geometry": ([ctypes.POINTER(ConvDesc), _I32, _I64, _P, _P, _P], _I32),
    "onexn_device_status": ([_I32, _P], _I32),
    "onexn_selftest_timeout": ([_P], _I32),
    "onexn_probe_ffma": ([_I32, _I32, _P, _P], _I32),
    "onexn_probe_mma_issue": ([_I32, _I32, _I32, _I32, _P], _I32),
    "onexn_conv_fwd_noalloc": ([ctypes.POINTER(ConvDesc), _P, _P, _P, _I32, _I64, _P, _P, _P, _I32,
                                _U32, _P], _I32),
    "onexn_conv_fwd_host": ([ctypes.POINTER(ConvDesc), _P, _P, _P, _I32, _I64, _P, _P, _P, _I32,
                             _U32, _P, ctypes.c_size_t, _P], _I32),
    "onexn_conv_host_workspace_size": ([ctypes.POINTER(ConvDesc), _I32, _I64, _I32, _U32, _P], _I32),
    "onexn_conv_fwd_ex": ([ctypes.POINTER(ConvDesc), _P, _P, _P, _I32, _I64, _P, _P, _P, _P, _I32,
                           _U32, _P, ctypes.c_size_t, _P], _I32),
    "onexn_dwconv_fwd": ([ctypes.POINTER(ConvDesc), _P, _P, _P, _P, _I32, _U32, _P], _I32),
    "onexn_dwproj_fwd": ([ctypes.POINTER(ConvDesc), _P, _P, _P, _P, _P, _I32, _I64, _I32, _P, _P, _P, _P, _I32,
                          _U32, _P, ctypes.c_size_t, _P], _I32),
    "onexn_prune_device_workspace_size": ([_I32, _I32, _I32, _I32, _I32, _I32, _P], _I32),
    "onexn_prune_device": ([_P, _I32, _I32, _I32, _I32, _I32, _DBL, _I32, _P, _P, _P, ctypes.c_size_t, _P],
                           _I32),
    "onexn_pack_device_workspace_size": ([_I32, _I32, _P], _I32),
    "onexn_conv_bwd_data_workspace_size": ([ctypes.POINTER(ConvDesc), _I32, _I64, _I32, _P], _I32),
    "onexn_conv_bwd_data": ([ctypes.POINTER(ConvDesc), _P, _P, _P, _I32, _I64, _P, _P, _I32, _U32, _P,
                             ctypes.c_size_t, _P], _I32),
    "onexn_conv_bwd_weight_workspace_size": ([ctypes.POINTER(ConvDesc), _I32, _I32, _P], _I32),
    "onexn_conv_bwd_weight": ([ctypes.POINTER(ConvDesc), _P, _P, _I32, _I64, _P, _P, _P, _P, _I32, _P,
                               ctypes.c_size_t, _P], _I32),
    "onexn_pack_device": ([_P, _P, _I32, _I32, _I32, _I32, _I32, _I32, _P, _P, _P, _I64, _P, ctypes.c_size_t,
                           _P], _I32),
}


class OnexnError(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__(f"{_STATUS.get(status, status)}: {msg}")
        self.status = status


def _load():
    if not os.path.exists(_SO):
        raise ImportError(f"libonexn.so is not built ({_SO}); run __graft_entry__.build()")
    lib = ctypes.CDLL(_SO)
    for name, (args, res) in SIGNATURES.items():
        fn = getattr(lib, name)
        fn.argtypes = args
        fn.restype = res
    return lib


lib = _load()
LIB_PATH = _SO


def _check(status: int):
    if status != ONEXN_OK:
        raise OnexnError(status, lib.onexn_last_error().decode())


def _np_ptr(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _f32(a):
    return np.ascontiguousarray(a, dtype=np.float32)


def onexn_version() -> int:
    return lib.onexn_version()


def onexn_keep_count(total_blocks: int, rate: float) -> int:
    out = ctypes.c_int64(0)
    _check(lib.onexn_keep_count(int(total_blocks), float(rate), ctypes.byref(out)))
    return out.value


def onexn_prune(W, N: int, rate: float, gran: int = ONEXN_GRAN_TAP):
    """Host W [C_out, C_in, KH, KW] fp32 -> (mask uint8 [G, KH*KW*C_in], kept)."""
    W = _f32(W)
    C_out, C_in, KH, KW = W.shape
    G = C_out // N if N > 0 else 0
    mask = np.empty((max(G, 1), KH * KW * C_in), np.uint8)
    kept = ctypes.c_int64(0)
    _check(lib.onexn_prune(_np_ptr(W), C_out, C_in, KH, KW, int(N), float(rate), int(gran),
                           _np_ptr(mask), ctypes.byref(kept)))
    return mask, kept.value


def onexn_rearrange(W_l, W_next=None):
    """Returns (W_l', W_next' or None, perm); inputs are copied, not modified."""
    W_l = np.array(W_l, dtype=np.float32, order="C", copy=True)
    C_out, C_in, KH, KW = W_l.shape
    perm = np.empty(C_out, np.int32)
    if W_next is not None:
        W_next = np.array(W_next, dtype=np.float32, order="C", copy=True)
        Cn, Cin_n, KHn, KWn = W_next.shape
        if Cin_n != C_out:
            raise OnexnError(ONEXN_EINVAL, "next layer's C_in differs from C_out")
    else:
        Cn = KHn = KWn = 0
    _check(lib.onexn_rearrange(_np_ptr(W_l), C_out, C_in, KH, KW, _np_ptr(W_next), Cn, KHn, KWn,
                               _np_ptr(perm)))
    return W_l, W_next, perm


def onexn_pack(W, mask, N: int, wdtype: int = ONEXN_F32):
    """BSR encoding -> (P int32 [G+1], I int32 [t], D [t, N] float32 or uint16 bf16 bits)."""
    W = _f32(W)
    mask = np.ascontiguousarray(mask, dtype=np.uint8)
    C_out, C_in, KH, KW = W.shape
    G = C_out // N
    t_cap = int(mask.sum())
    P = np.empty(G + 1, np.int32)
    I = np.empty(max(t_cap, 1), np.int32)
    D = np.empty((max(t_cap, 1), N), np.float32 if wdtype == ONEXN_F32 else np.uint16)
    t = ctypes.c_int64(0)
    _check(lib.onexn_pack(_np_ptr(W), _np_ptr(mask), C_out, C_in, KH, KW, int(N), int(wdtype),
                          _np_ptr(P), _np_ptr(I), _np_ptr(D), t_cap, ctypes.byref(t)))
    return P, I[:t.value].copy(), D[:t.value].copy()


def onexn_packed_validate(P, I, G: int, t: int, K: int) -> None:
    P = np.ascontiguousarray(P, np.int32)
    I = np.ascontiguousarray(I, np.int32)
    _check(lib.onexn_packed_validate(_np_ptr(P), _np_ptr(I) if I.size else None, int(G), int(t),
                                     int(K)))


def make_desc(B, H, W, C_in, C_out, KH=1, KW=1, stride=(1, 1), pad=(0, 0), dil=(1, 1)):
    s = stride if isinstance(stride, (tuple, list)) else (stride, stride)
    p = pad if isinstance(pad, (tuple, list)) else (pad, pad)
    d = dil if isinstance(dil, (tuple, list)) else (dil, dil)
    return ConvDesc(B, H, W, C_in, C_out, KH, KW, s[0], s[1], p[0], p[1], d[0], d[1])


def onexn_conv_out_shape(desc: ConvDesc):
    ho, wo = ctypes.c_int(0), ctypes.c_int(0)
    _check(lib.onexn_conv_out_shape(ctypes.byref(desc), ctypes.byref(ho), ctypes.byref(wo)))
    return ho.value, wo.value


def onexn_conv_algo(desc: ConvDesc, N: int, t: int, dtype: int, flags: int = 0,
                    workspace_bytes: int = 0) -> int:
    out = ctypes.c_uint(0)
    _check(lib.onexn_conv_algo(ctypes.byref(desc), int(N), int(t), int(dtype), int(flags),
                               int(workspace_bytes), ctypes.byref(out)))
    return out.value


ONEXN_GEMM_IM2COL = 0
ONEXN_GEMM_IM2COL_WIDE = 1
ONEXN_GEMM_HALO_RESIDENT = 2
ONEXN_GEMM_HALO_STREAMED = 3
GEMM_FORMS = {ONEXN_GEMM_IM2COL: "im2col", ONEXN_GEMM_IM2COL_WIDE: "im2col_wide",
              ONEXN_GEMM_HALO_RESIDENT: "halo_resident", ONEXN_GEMM_HALO_STREAMED: "halo_streamed"}


def onexn_conv_tc_form(desc: ConvDesc, N: int, t: int, dtype: int) -> str:
    out = ctypes.c_int(0)
    _check(lib.onexn_conv_tc_form(ctypes.byref(desc), int(N), int(t), int(dtype), ctypes.byref(out)))
    return GEMM_FORMS[out.value]


def onexn_conv_halo_geometry(desc: ConvDesc, N: int, t: int) -> dict:
    geom = (ctypes.c_int * 8)()
    taps = (ctypes.c_uint32 * 49)()
    phases = (ctypes.c_uint32 * 4)()
    _check(lib.onexn_conv_halo_geometry(ctypes.byref(desc), int(N), int(t), geom, taps, phases))
    n_ph, n_taps = geom[5], geom[6]
    return {"Wp": geom[0], "Hp": geom[1], "lower_w": geom[2], "lower_h": geom[3], "halo_pix": geom[4],
            "bn": geom[7],
            "taps": [(taps[i] >> 16, taps[i] & 0xFFFF) for i in range(n_taps)],
            "phases": [(phases[i] & 0xFF, (phases[i] >> 8) & 0xFF, (phases[i] >> 16) & 0xFF, phases[i] >> 24)
                       for i in range(n_ph)]}


def onexn_conv_workspace_size(desc: ConvDesc, N: int, t: int, dtype: int, flags: int = 0) -> int:
    out = ctypes.c_size_t(0)
    _check(lib.onexn_conv_workspace_size(ctypes.byref(desc), int(N), int(t), int(dtype),
                                         int(flags), ctypes.byref(out)))
    return out.value


def onexn_conv_fwd(desc: ConvDesc, P, I, D, N: int, t: int, x, y, bias, dtype: int,
                   flags: int = 0, workspace=None, stream=None) -> None:
    """Launch the convolution.  P, I, D, x, y, bias, workspace are torch CUDA
    tensors (bias and workspace may be None); stream is a torch.cuda.Stream
    or None (the current stream)."""
    import torch
    if stream is None:
        stream = torch.cuda.current_stream(x.device)
    ptr = (lambda tns: None if tns is None else ctypes.c_void_p(tns.data_ptr()))
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    _check(lib.onexn_conv_fwd(ctypes.byref(desc), ptr(P), ptr(I), ptr(D), int(N), int(t), ptr(x),
                              ptr(y), ptr(bias), int(dtype), int(flags), ptr(workspace),
                              int(ws_bytes), ctypes.c_void_p(stream.cuda_stream)))


def onexn_conv_fwd_ex(desc: ConvDesc, P, I, D, N: int, t: int, x, y, bias, residual, dtype: int,
                      flags: int = 0, workspace=None, stream=None) -> None:
    """onexn_conv_fwd with a residual: y = act(conv(x) + bias + residual)."""
    import torch
    if stream is None:
        stream = torch.cuda.current_stream(x.device)
    ptr = (lambda tns: None if tns is None else ctypes.c_void_p(tns.data_ptr()))
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    _check(lib.onexn_conv_fwd_ex(ctypes.byref(desc), ptr(P), ptr(I), ptr(D), int(N), int(t), ptr(x),
                                 ptr(y), ptr(bias), ptr(residual), int(dtype), int(flags), ptr(workspace),
                                 int(ws_bytes), ctypes.c_void_p(stream.cuda_stream)))


def onexn_dwconv_fwd(desc: ConvDesc, W, bias, x, y, dtype: int, flags: int = 0, stream=None) -> None:
    """The dense depthwise convolution (W: CUDA fp32 [C, KH, KW])."""
    import torch
    if stream is None:
        stream = torch.cuda.current_stream(x.device)
    ptr = (lambda tns: None if tns is None else ctypes.c_void_p(tns.data_ptr()))
    _check(lib.onexn_dwconv_fwd(ctypes.byref(desc), ptr(W), ptr(bias), ptr(x), ptr(y), int(dtype), int(flags),
                                ctypes.c_void_p(stream.cuda_stream)))


def onexn_conv_fwd_noalloc(desc: ConvDesc, P, I, D, N: int, t: int, x, y, bias, dtype: int,
                           flags: int = 0, stream=None) -> None:
    """The tensor-core convolution with the library's fixed 8 MiB scratch:
    no workspace argument and no allocation, for callers that cannot
    allocate device memory.  Calls that overlap on the GPU share the scratch
    and race; see include/onexn.h."""
    import torch
    if stream is None:
        stream = torch.cuda.current_stream(x.device)
    ptr = (lambda tns: None if tns is None else ctypes.c_void_p(tns.data_ptr()))
    _check(lib.onexn_conv_fwd_noalloc(ctypes.byref(desc), ptr(P), ptr(I), ptr(D), int(N), int(t),
                                      ptr(x), ptr(y), ptr(bias), int(dtype), int(flags),
                                      ctypes.c_void_p(stream.cuda_stream)))


def onexn_conv_host_workspace_size(desc: ConvDesc, N: int, t: int, dtype: int, flags: int = 0) -> int:
    out = ctypes.c_size_t(0)
    _check(lib.onexn_conv_host_workspace_size(ctypes.byref(desc), int(N), int(t), int(dtype),
                                              int(flags), ctypes.byref(out)))
    return out.value


def onexn_conv_fwd_host(desc: ConvDesc, P, I, D, N: int, t: int, x_host, y_host, bias, dtype: int,
                        flags: int = 0, workspace=None, stream=None) -> None:
    """The convolution on host-memory activations: x_host and y_host are CPU
    tensors (pinned for overlapped copies), P, I, D, bias and workspace CUDA
    tensors; stream a torch.cuda.Stream or None (the current stream).  The
    call is asynchronous: synchronise the stream before reading y_host."""
    import torch
    if stream is None:
        stream = torch.cuda.current_stream(workspace.device)
    ptr = (lambda tns: None if tns is None else ctypes.c_void_p(tns.data_ptr()))
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    _check(lib.onexn_conv_fwd_host(ctypes.byref(desc), ptr(P), ptr(I), ptr(D), int(N), int(t),
                                   ptr(x_host), ptr(y_host), ptr(bias), int(dtype), int(flags),
                                   ptr(workspace), int(ws_bytes), ctypes.c_void_p(stream.cuda_stream)))


def onexn_device_status(clear: bool = True) -> int:
    """ONEXN_OK, ONEXN_EDEVICE (checked mode found malformed P / I) or
    ONEXN_ETIMEOUT (a bounded in-kernel wait ran out)."""
    st = ctypes.c_int(0)
    _check(lib.onexn_device_status(int(bool(clear)), ctypes.byref(st)))
    return st.value


def onexn_selftest_timeout(stream=None) -> None:
    """Launch the bounded-wait self-test kernel (about one second on the
    GPU); afterwards onexn_device_status() reports ONEXN_ETIMEOUT."""
    import torch
    st = torch.cuda.current_stream() if stream is None else stream
    _check(lib.onexn_selftest_timeout(ctypes.c_void_p(st.cuda_stream)))


def onexn_probe_ffma(blocks: int, iters: int, sink, stream=None) -> None:
    """Launch the FFMA-chain measurement kernel (16 * iters flops per thread,
    256 threads per block); sink a CUDA float tensor of >= blocks elements."""
    import torch
    st = torch.cuda.current_stream() if stream is None else stream
    _check(lib.onexn_probe_ffma(int(blocks), int(iters), ctypes.c_void_p(sink.data_ptr()),
                                ctypes.c_void_p(st.cuda_stream)))


def onexn_probe_mma_issue(N: int, issuers: int, a_tmem: bool, iters: int, stream=None) -> None:
    """Launch the tcgen05.mma issue-rate measurement kernel (one CTA per SM,
    4 * iters MMAs of M=128 x N x K=16 per issuing warp)."""
    import torch
    st = torch.cuda.current_stream() if stream is None else stream
    _check(lib.onexn_probe_mma_issue(int(N), int(issuers), int(bool(a_tmem)), int(iters),
                                     ctypes.c_void_p(st.cuda_stream)))


def _cuda_stream(t, stream):
    import torch
    return torch.cuda.current_stream(t.device) if stream is None else stream


def onexn_prune_device(W, N: int, rate: float, gran: int = ONEXN_GRAN_TAP, mask=None, workspace=None,
                       stream=None):
    """Device W (CUDA fp32 [C_out, C_in, KH, KW]) -> (mask CUDA uint8 [G, K], kept),
    the same mask as onexn_prune.  mask / workspace are allocated if None."""
    import torch
    C_out, C_in, KH, KW = W.shape
    if N < 1 or C_out % N:
        raise OnexnError(ONEXN_EINVAL, f"N={N} must divide C_out={C_out}")
    G, K = C_out // N, KH * KW * C_in
    n = ctypes.c_size_t(0)
    _check(lib.onexn_prune_device_workspace_size(C_out, C_in, KH, KW, int(N), int(gran), ctypes.byref(n)))
    if mask is None:
        mask = torch.empty((G, K), dtype=torch.uint8, device=W.device)
    if workspace is None:
        workspace = torch.empty(max(n.value, 256), dtype=torch.uint8, device=W.device)
    kept = ctypes.c_int64(0)
    s = _cuda_stream(W, stream)
    _check(lib.onexn_prune_device(ctypes.c_void_p(W.data_ptr()), C_out, C_in, KH, KW, int(N), float(rate),
                                  int(gran), ctypes.c_void_p(mask.data_ptr()), ctypes.byref(kept),
                                  ctypes.c_void_p(workspace.data_ptr()), workspace.numel(),
                                  ctypes.c_void_p(s.cuda_stream)))
    return mask, kept.value


def onexn_pack_device(W, mask, N: int, t: int, wdtype: int = ONEXN_F32, stream=None):
    """Device BSR encoding -> (P CUDA int32 [G+1], I CUDA int32 [t], D CUDA
    [t, N] float32 or bfloat16), the same as onexn_pack; t = the mask's
    count (I and D are sized from it)."""
    import torch
    C_out, C_in, KH, KW = W.shape
    if N < 1 or C_out % N:
        raise OnexnError(ONEXN_EINVAL, f"N={N} must divide C_out={C_out}")
    G = C_out // N
    n = ctypes.c_size_t(0)
    _check(lib.onexn_pack_device_workspace_size(C_out, int(N), ctypes.byref(n)))
    ws = torch.empty(max(n.value, 256), dtype=torch.uint8, device=W.device)
    P = torch.empty(G + 1, dtype=torch.int32, device=W.device)
    I = torch.empty(max(t, 1), dtype=torch.int32, device=W.device)
    D = torch.empty((max(t, 1), N), dtype=torch.float32 if wdtype == ONEXN_F32 else torch.bfloat16,
                    device=W.device)
    s = _cuda_stream(W, stream)
    ptr = (lambda x: ctypes.c_void_p(x.data_ptr()))
    _check(lib.onexn_pack_device(ptr(W), ptr(mask), C_out, C_in, KH, KW, int(N), int(wdtype), ptr(P), ptr(I),
                                 ptr(D), int(t), ptr(ws), ws.numel(), ctypes.c_void_p(s.cuda_stream)))
    return P, I[:t], D[:t]


def onexn_conv_bwd_data_workspace_size(desc: ConvDesc, N: int, t: int, dtype: int) -> int:
    out = ctypes.c_size_t(0)
    _check(lib.onexn_conv_bwd_data_workspace_size(ctypes.byref(desc), int(N), int(t), int(dtype),
                                                  ctypes.byref(out)))
    return out.value


def onexn_conv_bwd_data(desc: ConvDesc, P, I, D, N: int, t: int, dy, dx, dtype: int, flags: int = 0,
                        workspace=None, stream=None) -> None:
    """Input gradient of the pruned convolution (CUDA tensors; dy is the
    gradient of the pre-activation output)."""
    s = _cuda_stream(dy, stream)
    ptr = (lambda x: None if x is None else ctypes.c_void_p(x.data_ptr()))
    _check(lib.onexn_conv_bwd_data(ctypes.byref(desc), ptr(P), ptr(I), ptr(D), int(N), int(t), ptr(dy), ptr(dx),
                                   int(dtype), int(flags), ptr(workspace),
                                   0 if workspace is None else workspace.numel(), ctypes.c_void_p(s.cuda_stream)))


def onexn_conv_bwd_weight_workspace_size(desc: ConvDesc, N: int, dtype: int) -> int:
    out = ctypes.c_size_t(0)
    _check(lib.onexn_conv_bwd_weight_workspace_size(ctypes.byref(desc), int(N), int(dtype), ctypes.byref(out)))
    return out.value


def onexn_conv_bwd_weight(desc: ConvDesc, P, I, N: int, t: int, x, dy, dD, db, dtype: int, workspace=None,
                          stream=None) -> None:
    """Kept-weight gradient in BSR order (dD CUDA fp32 [t, N]) and optionally
    the bias gradient (db CUDA fp32 [C_out])."""
    s = _cuda_stream(dy, stream)
    ptr = (lambda x_: None if x_ is None else ctypes.c_void_p(x_.data_ptr()))
    _check(lib.onexn_conv_bwd_weight(ctypes.byref(desc), ptr(P), ptr(I), int(N), int(t), ptr(x), ptr(dy), ptr(dD),
                                     ptr(db), int(dtype), ptr(workspace),
                                     0 if workspace is None else workspace.numel(), ctypes.c_void_p(s.cuda_stream)))
