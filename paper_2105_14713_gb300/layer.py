"""1xN-pruned convolution layers (and MobileNet-V2's inverted-residual block)
on the onexn C ABI.

``PrunedConv2d`` runs the offline steps once on the host -- block scoring
and selection (``onexn_prune``), BSR encoding (``onexn_pack``), the index
check (``onexn_packed_validate``) -- copies (P, I, D) and the bias to the
GPU, and then calls ``onexn_conv_fwd`` per forward pass.  Filter
rearrangement (``onexn_rearrange``) is applied by the caller across a pair
of layers before pruning, as in the paper's workflow (Sec. 3.3).
"""
from __future__ import annotations

import ctypes

import numpy as np
import torch

from . import onexn as _c


def act_flags(relu) -> int:
    """False / True / "relu6" -> 0 / ONEXN_RELU / ONEXN_RELU6."""
    if relu == "relu6":
        return _c.ONEXN_RELU6
    return _c.ONEXN_RELU if relu else 0


class PrunedConv2d:
    def __init__(self, weight, N: int, rate: float, *, bias=None, stride=1, padding=0,
                 dilation=1, dtype: str = "f32", gran: int = _c.ONEXN_GRAN_TAP,
                 device="cuda", mask=None, reuse_decoded: bool = True):
        W = np.ascontiguousarray(np.asarray(weight, np.float32))
        self.reuse_decoded = bool(reuse_decoded)
        self.C_out, self.C_in, self.KH, self.KW = W.shape
        self.N = int(N)
        self.rate = float(rate)
        self.dtype = dtype
        self.cdtype = _c.ONEXN_F32 if dtype == "f32" else _c.ONEXN_BF16
        self.stride = stride if isinstance(stride, (tuple, list)) else (stride, stride)
        self.padding = padding if isinstance(padding, (tuple, list)) else (padding, padding)
        self.dilation = dilation if isinstance(dilation, (tuple, list)) else (dilation, dilation)
        if mask is None:
            mask, self.kept = _c.onexn_prune(W, self.N, self.rate, gran)
        else:
            self.kept = None
        self.mask = mask
        P, I, D = _c.onexn_pack(W, mask, self.N, self.cdtype)
        self.t = len(I)
        _c.onexn_packed_validate(P, I, self.C_out // self.N, self.t, self.KH * self.KW * self.C_in)
        self.P_host, self.I_host, self.D_host = P, I, D
        dev = torch.device(device)
        self.device = dev
        self.P = torch.from_numpy(P).to(dev)
        self.I = torch.from_numpy(np.ascontiguousarray(I) if self.t else np.zeros(1, np.int32)).to(dev)
        if self.cdtype == _c.ONEXN_F32:
            Dt = torch.from_numpy(D if self.t else np.zeros((1, self.N), np.float32))
        else:
            Dt = torch.from_numpy((D if self.t else np.zeros((1, self.N), np.uint16)).view(np.int16))
            Dt = Dt.view(torch.bfloat16)
        self.D = Dt.to(dev).contiguous()
        self.bias = None if bias is None else torch.as_tensor(
            np.asarray(bias, np.float32)).to(dev).contiguous()
        self._ws = {}            # per input shape: device workspace (bytes as uint8)
        self._args = {}          # per buffers / layout / flags / stream: marshalled C arguments
        self._descs = []
        # workspaces whose decoded weights a completed-in-order tc call has
        # written: later calls on them pass ONEXN_DECODED and skip the decode
        # (until D changes: an optimizer step bumps its version counter)
        self._decoded = set()
        self._d_version = self.D._version

    @property
    def torch_dtype(self):
        return torch.float32 if self.cdtype == _c.ONEXN_F32 else torch.bfloat16

    def desc(self, B: int, H: int, W: int) -> _c.ConvDesc:
        return _c.make_desc(B, H, W, self.C_in, self.C_out, self.KH, self.KW, self.stride,
                            self.padding, self.dilation)

    def out_shape(self, x_shape):
        B, H, W, _ = x_shape
        Ho, Wo = _c.onexn_conv_out_shape(self.desc(B, H, W))
        return (B, Ho, Wo, self.C_out)

    def workspace(self, x_shape, flags: int = 0):
        """Device workspace for this input shape (allocated once, reused)."""
        B, H, W, _ = x_shape
        key = (B, H, W, flags & 0xF00)
        if key not in self._ws:
            n = _c.onexn_conv_workspace_size(self.desc(B, H, W), self.N, self.t, self.cdtype, flags)
            self._ws[key] = torch.empty(max(n, 256), dtype=torch.uint8, device=self.device) if n else None
        return self._ws[key]

    def _reuse_flag(self) -> int:
        return _c.ONEXN_REUSE_DECODE if self.reuse_decoded else 0

    def algo(self, x_shape, flags: int = 0) -> str:
        """The family forward runs for this input shape (and forced flags)."""
        B, H, W, _ = x_shape
        ws = self.workspace(x_shape, flags)
        a = _c.onexn_conv_algo(self.desc(B, H, W), self.N, self.t, self.cdtype, flags | self._reuse_flag(),
                               0 if ws is None else ws.numel())
        return _c.ALGO_NAMES[a]

    def tc_form(self, x_shape) -> str:
        """The form the tensor-core family's GEMM takes for this input shape:
        "im2col", "im2col_wide", "halo_resident" or "halo_streamed"."""
        B, H, W, _ = x_shape
        return _c.onexn_conv_tc_form(self.desc(B, H, W), self.N, self.t, self.cdtype)

    def forward(self, x: torch.Tensor, y: torch.Tensor = None, relu=False,
                algo: int = _c.ONEXN_ALGO_AUTO, stream=None, residual: torch.Tensor = None) -> torch.Tensor:
        """x: NHWC CUDA tensor of this layer's dtype.  Returns y (NHWC):
        y = act(conv(x) + bias + residual), act = none, ReLU (relu=True) or
        ReLU6 (relu="relu6"); residual is optional (shape of y; may be y).

        The checked and marshalled C arguments are cached per (x, y,
        residual, stream, flags) buffers and layout, so a layer called again
        on the same buffers costs one C call."""
        if y is None:
            y = torch.empty(self.out_shape(x.shape), dtype=x.dtype, device=x.device)
        s = torch.cuda.current_stream(x.device) if stream is None else stream
        if self.D._version != self._d_version:          # weights updated in place: decode again
            self._decoded.clear()
            self._args.clear()
            self._d_version = self.D._version
        flags = act_flags(relu) | algo | self._reuse_flag()
        key = (x.data_ptr(), y.data_ptr(), x.shape, x.stride(), x.dtype, y.shape, y.stride(), y.dtype,
               None if residual is None else (residual.data_ptr(), residual.shape, residual.stride(),
                                              residual.dtype),
               flags, s.cuda_stream)
        args = self._args.get(key)
        if args is None:
            if len(self._args) >= 64:
                self._args.clear()
                self._descs.clear()
            args = self._marshal(x, y, flags, s, residual)
            self._args[key] = args
        st = _c.lib.onexn_conv_fwd_ex(*args[0])
        if st != _c.ONEXN_OK:
            raise _c.OnexnError(st, _c.lib.onexn_last_error().decode(errors="replace"))
        if args[1] is not None and args[1] not in self._decoded:
            # this call decoded the weights into the workspace: later calls
            # (ordered after it on the caller's streams, as calls sharing a
            # workspace must be) run the GEMM alone
            self._decoded.add(args[1])
            self._args.pop(key, None)
        return y

    def _marshal(self, x, y, flags, s, residual=None):
        if x.dtype != self.torch_dtype or not x.is_cuda or not x.is_contiguous():
            raise ValueError(f"x must be a contiguous CUDA {self.torch_dtype} NHWC tensor")
        B, H, W, C = x.shape
        if C != self.C_in:
            raise ValueError(f"x has {C} channels, layer expects {self.C_in}")
        if tuple(y.shape) != tuple(self.out_shape(x.shape)) or y.dtype != x.dtype or not y.is_contiguous() \
                or y.device != x.device:
            raise ValueError(f"y must be a contiguous {x.dtype} tensor of shape {self.out_shape(x.shape)}")
        if residual is not None and (tuple(residual.shape) != tuple(y.shape) or residual.dtype != y.dtype
                                     or not residual.is_contiguous() or residual.device != y.device):
            raise ValueError("residual must be a contiguous tensor like y")
        desc = self.desc(B, H, W)
        ws = self.workspace(x.shape, flags & _c.ONEXN_ALGO_MASK)
        ptr = (lambda t: None if t is None else ctypes.c_void_p(t.data_ptr()))
        ws_bytes = 0 if ws is None else ws.numel()
        # the tc family decodes the weights into the workspace; once that has
        # happened on this workspace, skip it (ONEXN_DECODED)
        ws_key = None
        if ws is not None and self.reuse_decoded:
            al = _c.onexn_conv_algo(desc, self.N, self.t, self.cdtype, flags, ws_bytes)
            if al == _c.ONEXN_ALGO_TC:
                ws_key = ws.data_ptr()
                if ws_key in self._decoded:
                    flags |= _c.ONEXN_DECODED
                    ws_key = None
        self._descs.append(desc)                 # kept alive for the cached byref
        return ((ctypes.byref(desc), ptr(self.P), ptr(self.I), ptr(self.D), self.N, self.t, ptr(x), ptr(y),
                 ptr(self.bias), ptr(residual), self.cdtype, flags, ptr(ws), ws_bytes,
                 ctypes.c_void_p(s.cuda_stream)), ws_key)

    __call__ = forward

    def host_workspace(self, x_shape, flags: int = 0):
        """Device workspace of forward_host for this input shape (allocated
        once, reused)."""
        B, H, W, _ = x_shape
        key = ("host", B, H, W, flags & 0xF00)
        if key not in self._ws:
            n = _c.onexn_conv_host_workspace_size(self.desc(B, H, W), self.N, self.t, self.cdtype, flags)
            self._ws[key] = torch.empty(max(n, 256), dtype=torch.uint8, device=self.device)
        return self._ws[key]

    def forward_dwproj(self, h: torch.Tensor, dw_w_tap: torch.Tensor, dw_b, dw_stride: int,
                       y: torch.Tensor = None, relu=False, residual: torch.Tensor = None, stream=None):
        """This 1x1 layer applied to relu6(depthwise3x3(h)) with the depthwise
        computed inside the GEMM (onexn_dwproj_fwd; fp32): h NHWC
        [B, H, W, C_in]; dw_w_tap CUDA fp32 [9, C_in] (tap-major); dw_b CUDA
        fp32 [C_in] or None; pad 1, stride dw_stride."""
        B, H, W, C = h.shape
        if C != self.C_in or self.KH != 1 or self.KW != 1:
            raise ValueError("forward_dwproj needs a 1x1 layer whose C_in is h's channel count")
        dw_desc = _c.make_desc(B, H, W, C, C, 3, 3, dw_stride, 1, 1)
        Ho, Wo = _c.onexn_conv_out_shape(dw_desc)
        shape = (B, Ho, Wo, self.C_out)
        if y is None:
            y = torch.empty(shape, dtype=h.dtype, device=h.device)
        s = torch.cuda.current_stream(h.device) if stream is None else stream
        if self.D._version != self._d_version:
            self._decoded.clear()
            self._args.clear()
            self._d_version = self.D._version
        flags = act_flags(relu) | _c.ONEXN_ALGO_TC | self._reuse_flag()
        key = ("dwproj", h.data_ptr(), y.data_ptr(), h.shape, dw_w_tap.data_ptr(),
               None if dw_b is None else dw_b.data_ptr(), dw_stride,
               None if residual is None else residual.data_ptr(), flags, s.cuda_stream)
        args = self._args.get(key)
        if args is None:
            if h.dtype != torch.float32 or not h.is_contiguous() or tuple(y.shape) != shape:
                raise ValueError("forward_dwproj: h must be contiguous fp32 and y of shape %s" % (shape,))
            ws = self.workspace((B, Ho, Wo, C), _c.ONEXN_ALGO_TC)
            ws_key = None
            f = flags
            if self.reuse_decoded:
                ws_key = ws.data_ptr()
                if ws_key in self._decoded:
                    f |= _c.ONEXN_DECODED
                    ws_key = None
            dd = _c.ConvDesc(*[getattr(dw_desc, n) for n, _ in _c.ConvDesc._fields_])
            self._descs.append(dd)
            ptr = (lambda t: None if t is None else ctypes.c_void_p(t.data_ptr()))
            args = ((ctypes.byref(dd), ptr(dw_w_tap), ptr(dw_b), ptr(self.P), ptr(self.I), ptr(self.D), self.N,
                     self.t, self.C_out, ptr(h), ptr(y), ptr(self.bias), ptr(residual), self.cdtype, f, ptr(ws),
                     ws.numel(), ctypes.c_void_p(s.cuda_stream)), ws_key)
            self._args[key] = args
        st = _c.lib.onexn_dwproj_fwd(*args[0])
        if st != _c.ONEXN_OK:
            raise _c.OnexnError(st, _c.lib.onexn_last_error().decode(errors="replace"))
        if args[1] is not None and args[1] not in self._decoded:
            self._decoded.add(args[1])
            self._args.pop(key, None)
        return y

    # ---------------------------------------------- fine-tuning (mask fixed)

    def backward(self, x: torch.Tensor, dy: torch.Tensor, dx: torch.Tensor = None, *, need_dx: bool = True,
                 need_dw: bool = True, need_db: bool = True, accumulate: bool = False, stream=None):
        """Gradients with the mask held fixed (onexn_conv_bwd_data /
        onexn_conv_bwd_weight): dy is the gradient of the pre-activation
        output (NHWC like forward's y).  Returns (dx, dD, db): dx like x
        (added to a given dx with accumulate=True), dD fp32 [t, N] in D's
        order (only the kept blocks), db fp32 [C_out]; None where not asked."""
        if dy.dtype != self.torch_dtype or not dy.is_cuda or not dy.is_contiguous():
            raise ValueError(f"dy must be a contiguous CUDA {self.torch_dtype} NHWC tensor")
        if x.dtype != self.torch_dtype or not x.is_contiguous():
            raise ValueError(f"x must be a contiguous CUDA {self.torch_dtype} NHWC tensor")
        B, H, W, _ = x.shape
        if tuple(dy.shape) != tuple(self.out_shape(x.shape)):
            raise ValueError(f"dy must have shape {self.out_shape(x.shape)}")
        desc = self.desc(B, H, W)
        s = torch.cuda.current_stream(x.device) if stream is None else stream
        dD = db = None
        if need_dx:
            if dx is None:
                dx = (torch.zeros_like(x) if accumulate else torch.empty_like(x))
            key = ("bwd_data", B, H, W)
            if key not in self._ws:
                n = _c.onexn_conv_bwd_data_workspace_size(desc, self.N, self.t, self.cdtype)
                self._ws[key] = torch.empty(max(n, 256), dtype=torch.uint8, device=self.device)
            _c.onexn_conv_bwd_data(desc, self.P, self.I, self.D, self.N, self.t, dy, dx, self.cdtype,
                                   _c.ONEXN_ACCUMULATE if accumulate else 0, self._ws[key], s)
        else:
            dx = None
        if need_dw or need_db:
            key = ("bwd_weight", B, H, W)
            if key not in self._ws:
                n = _c.onexn_conv_bwd_weight_workspace_size(desc, self.N, self.cdtype)
                self._ws[key] = torch.empty(max(n, 256), dtype=torch.uint8, device=self.device)
            dD = torch.empty((max(self.t, 1), self.N), dtype=torch.float32, device=x.device)[:self.t]
            db = torch.empty(self.C_out, dtype=torch.float32, device=x.device) if need_db else None
            _c.onexn_conv_bwd_weight(desc, self.P, self.I, self.N, self.t, x, dy, dD if self.t else None, db,
                                     self.cdtype, self._ws[key], s)
            if not need_dw:
                dD = None
        return dx, dD, db

    def parameters(self):
        """The trainable tensors of the pruned layer: D (the kept blocks, Sec.
        3.4) and the bias, with requires_grad set; the mask (P, I) is fixed."""
        self.D.requires_grad_(True)
        out = [self.D]
        if self.bias is not None:
            self.bias.requires_grad_(True)
            out.append(self.bias)
        return out

    def train_forward(self, x: torch.Tensor) -> torch.Tensor:
        """Forward as a differentiable op of (x, D, bias) for fine-tuning:
        the backward runs onexn_conv_bwd_data / onexn_conv_bwd_weight.  The
        output is the linear (pre-activation) convolution; apply the
        activation with torch (its backward is elementwise)."""
        return _PrunedConvFn.apply(x, self.D, self.bias, self)

    def forward_host(self, x_host: torch.Tensor, y_host: torch.Tensor = None, relu: bool = False,
                     algo: int = _c.ONEXN_ALGO_AUTO, stream=None, sync: bool = True) -> torch.Tensor:
        """End to end from host memory (onexn_conv_fwd_host): the input is
        copied in and the output copied out chunk by chunk, overlapped with
        the convolution.  x_host: contiguous CPU NHWC tensor of this layer's
        dtype (pinned for overlapped copies).  y_host: optional CPU output
        (allocated pinned if None).  With sync=False the call returns after
        enqueueing: synchronise `stream` before reading y_host."""
        if x_host.dtype != self.torch_dtype or x_host.is_cuda or not x_host.is_contiguous():
            raise ValueError(f"x_host must be a contiguous CPU {self.torch_dtype} NHWC tensor")
        B, H, W, C = x_host.shape
        if C != self.C_in:
            raise ValueError(f"x_host has {C} channels, layer expects {self.C_in}")
        shape = self.out_shape(x_host.shape)
        if y_host is None:
            y_host = torch.empty(shape, dtype=x_host.dtype, pin_memory=True)
        elif tuple(y_host.shape) != tuple(shape) or y_host.dtype != x_host.dtype or y_host.is_cuda \
                or not y_host.is_contiguous():
            raise ValueError(f"y_host must be a contiguous CPU {x_host.dtype} tensor of shape {shape}")
        if stream is None:
            stream = torch.cuda.current_stream(self.device)
        flags = act_flags(relu) | algo
        _c.onexn_conv_fwd_host(self.desc(B, H, W), self.P, self.I, self.D, self.N, self.t, x_host,
                               y_host, self.bias, self.cdtype, flags,
                               self.host_workspace(x_host.shape, algo), stream)
        if sync:
            stream.synchronize()
        return y_host


class _PrunedConvFn(torch.autograd.Function):
    @staticmethod
    def forward(ctx, x, D, bias, layer):
        ctx.layer = layer
        ctx.save_for_backward(x)
        with torch.no_grad():
            return layer.forward(x.contiguous())

    @staticmethod
    def backward(ctx, gy):
        (x,) = ctx.saved_tensors
        layer = ctx.layer
        need_dx, need_dw, need_db = ctx.needs_input_grad[0], ctx.needs_input_grad[1], ctx.needs_input_grad[2]
        dx, dD, db = layer.backward(x.contiguous(), gy.contiguous(), need_dx=need_dx, need_dw=need_dw,
                                    need_db=need_db)
        if dD is not None:
            dD = dD.to(layer.D.dtype)
        return dx, dD, db, None


class DepthwiseConv2d:
    """The dense depthwise convolution between the pruned 1x1 convolutions of
    a MobileNet-V2 block (onexn_dwconv_fwd).  weight: [C, 1, KH, KW] or
    [C, KH, KW] fp32 (not pruned)."""

    def __init__(self, weight, *, bias=None, stride=1, padding=1, dilation=1, dtype: str = "f32",
                 device="cuda"):
        Wd = np.ascontiguousarray(np.asarray(weight, np.float32))
        if Wd.ndim == 4:
            Wd = Wd[:, 0]
        self.C, self.KH, self.KW = Wd.shape
        self.dtype = dtype
        self.cdtype = _c.ONEXN_F32 if dtype == "f32" else _c.ONEXN_BF16
        self.stride = stride if isinstance(stride, (tuple, list)) else (stride, stride)
        self.padding = padding if isinstance(padding, (tuple, list)) else (padding, padding)
        self.dilation = dilation if isinstance(dilation, (tuple, list)) else (dilation, dilation)
        self.device = torch.device(device)
        self.W = torch.from_numpy(Wd).to(self.device).contiguous()
        self.bias = None if bias is None else torch.as_tensor(np.asarray(bias, np.float32)).to(self.device)
        self._args = {}
        self._descs = []

    def desc(self, B: int, H: int, W: int) -> _c.ConvDesc:
        return _c.make_desc(B, H, W, self.C, self.C, self.KH, self.KW, self.stride, self.padding,
                            self.dilation)

    def out_shape(self, x_shape):
        B, H, W, _ = x_shape
        Ho, Wo = _c.onexn_conv_out_shape(self.desc(B, H, W))
        return (B, Ho, Wo, self.C)

    def forward(self, x: torch.Tensor, y: torch.Tensor = None, relu=False, stream=None) -> torch.Tensor:
        if y is None:
            y = torch.empty(self.out_shape(x.shape), dtype=x.dtype, device=x.device)
        s = torch.cuda.current_stream(x.device) if stream is None else stream
        flags = act_flags(relu)
        key = (x.data_ptr(), y.data_ptr(), x.shape, x.dtype, y.shape, flags, s.cuda_stream)
        args = self._args.get(key)
        if args is None:
            if not (x.is_cuda and x.is_contiguous() and y.is_contiguous() and x.shape[3] == self.C
                    and tuple(y.shape) == tuple(self.out_shape(x.shape)) and y.dtype == x.dtype):
                raise ValueError("x / y do not match the depthwise layer")
            if len(self._args) >= 64:
                self._args.clear()
                self._descs.clear()
            B, H, W, _ = x.shape
            desc = self.desc(B, H, W)
            self._descs.append(desc)
            ptr = (lambda t: None if t is None else ctypes.c_void_p(t.data_ptr()))
            args = (ctypes.byref(desc), ptr(self.W), ptr(self.bias), ptr(x), ptr(y), self.cdtype, flags,
                    ctypes.c_void_p(s.cuda_stream))
            self._args[key] = args
        st = _c.lib.onexn_dwconv_fwd(*args)
        if st != _c.ONEXN_OK:
            raise _c.OnexnError(st, _c.lib.onexn_last_error().decode(errors="replace"))
        return y

    __call__ = forward


class InvertedResidual:
    """MobileNet-V2's inverted-residual block on the onexn kernels:
    expand 1x1 (1xN-pruned, ReLU6; absent for expansion 1) -> depthwise 3x3
    (dense, ReLU6, stride s) -> project 1x1 (1xN-pruned, linear), plus the
    block input when s == 1 and C_in == C_out (fused into the project's
    epilogue).  The filters of the expand layer may be rearranged (Sec. 3.3)
    before pruning, with the permutation carried through the depthwise
    channels into the project layer's inputs (reading C10).  Intermediate
    buffers are allocated per input shape on the first call and reused, so
    later calls allocate nothing (and can be captured into a CUDA graph)."""

    def __init__(self, w_expand, b_expand, w_dw, b_dw, w_project, b_project, *, stride: int, N: int,
                 rate: float, dtype: str = "f32", rearrange: bool = True, device="cuda", fuse_dw=False):
        w_dw = np.asarray(w_dw, np.float32)
        w_dw = w_dw[:, 0] if w_dw.ndim == 4 else w_dw
        b_dw = None if b_dw is None else np.asarray(b_dw, np.float32)
        w_project = np.asarray(w_project, np.float32)
        self.expand = None
        if w_expand is not None:
            w_expand = np.asarray(w_expand, np.float32)
            b_expand = None if b_expand is None else np.asarray(b_expand, np.float32)
            if rearrange:
                w_expand, w_project, perm = _c.onexn_rearrange(w_expand, w_project)
                b_expand = None if b_expand is None else b_expand[perm]
                w_dw = w_dw[perm]
                b_dw = None if b_dw is None else b_dw[perm]
            self.expand = PrunedConv2d(w_expand, N, rate, bias=b_expand, dtype=dtype, device=device)
        # the weights as run (after the rearrangement), for checks
        self.w_expand, self.b_expand, self.w_dw, self.b_dw = w_expand, b_expand, w_dw, b_dw
        self.w_project = w_project
        self.b_project = None if b_project is None else np.asarray(b_project, np.float32)
        self.dw = DepthwiseConv2d(w_dw, bias=b_dw, stride=stride, padding=1, dtype=dtype, device=device)
        self.project = PrunedConv2d(w_project, N, rate, bias=b_project, dtype=dtype, device=device)
        c_in = self.expand.C_in if self.expand is not None else w_dw.shape[0]
        self.residual = stride == 1 and w_project.shape[0] == c_in
        self.dtype = dtype
        self.stride = stride
        self._bufs = {}
        # the depthwise fused into the projection's GEMM (onexn_dwproj_fwd,
        # fp32): True = always, "auto" = for at most FUSE_PIXELS output
        # pixels, False (default) = never.  Measured on GB300 the fused form
        # is slower (MobileNet-V2's 17 blocks at batch 1: 1.43 ms against
        # 0.325 ms): the GEMM's four A-producing warps wait an L2 latency per
        # tap, where the separate depthwise kernel keeps nine loads in flight
        # per thread at full occupancy.
        self.fuse_dw = fuse_dw
        C = w_dw.shape[0]
        self.dw_w_tap = torch.from_numpy(np.ascontiguousarray(w_dw.reshape(C, 9).T)).to(device)
        self.dw_b_dev = None if b_dw is None else torch.from_numpy(np.ascontiguousarray(b_dw)).to(device)

    def buffers(self, x_shape, dtype, device):
        key = tuple(x_shape)
        if key not in self._bufs:
            h = self.expand.out_shape(x_shape) if self.expand is not None else tuple(x_shape)
            d = self.dw.out_shape(h)
            o = self.project.out_shape(d)
            self._bufs[key] = (torch.empty(h, dtype=dtype, device=device) if self.expand is not None else None,
                               torch.empty(d, dtype=dtype, device=device),
                               torch.empty(o, dtype=dtype, device=device))
        return self._bufs[key]

    FUSE_PIXELS = 4096

    def fused(self, x_shape) -> bool:
        if self.dtype != "f32" or self.fuse_dw is False:
            return False
        if self.fuse_dw is True:
            return True
        B, H, W, _ = x_shape
        Ho, Wo = (H - 1) // self.stride + 1, (W - 1) // self.stride + 1
        return B * Ho * Wo <= self.FUSE_PIXELS

    def forward(self, x: torch.Tensor, stream=None) -> torch.Tensor:
        h, d, o = self.buffers(x.shape, x.dtype, x.device)
        if self.expand is not None:
            self.expand(x, h, relu="relu6", stream=stream)
        else:
            h = x
        res = x if self.residual else None
        if self.fused(x.shape):
            self.project.forward_dwproj(h, self.dw_w_tap, self.dw_b_dev, self.stride, o, residual=res,
                                        stream=stream)
        else:
            self.dw(h, d, relu="relu6", stream=stream)
            self.project(d, o, stream=stream, residual=res)
        return o

    __call__ = forward
