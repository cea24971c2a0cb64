"""CPU oracle for 1xN pruning and the 1xN-pruned convolution (fp64).

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and
the CPU-baseline / reference legs of ``bench.py`` may import this package.
The product library (``paper_2105_14713_gb300``) never imports it, and the
two share no code: the arithmetic lives in ``oracle.c`` next to this file,
written from the paper (Sec. 3.1-3.4, Eq. 1-7), and this module only
marshals numpy arrays into it.

Functions (each follows the passage named in its docstring):

* ``keep_count``   -- Eq. 1 constraint, kept-block count (reading C3)
* ``block_scores`` -- Eq. 4 block l1 norms
* ``prune``        -- top-(1-p) mask of the solution stated after Eq. 5
* ``rearrange``    -- Sec. 3.3 filter rearrangement
* ``pack``/``unpack`` -- Sec. 3.4 BSR encoding (D, I, P) and its inverse
* ``conv_masked``  -- Eq. 6 masked direct convolution (+bias, ReLU)
* ``conv_bsr``     -- Eq. 7 block-wise decode from (P, I, D)
* ``round_bf16``   -- RNE rounding of fp32 to bfloat16 values
* ``dwconv``       -- dense depthwise convolution of MobileNet-V2's block
* ``conv_backward_data`` / ``conv_backward_weight`` / ``bsr_gather`` --
  gradients of Eq. 6 with the mask held fixed (fine-tuning, Sec. 3.2/4.1)
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

GRAN_TAP = 0
GRAN_KERNEL = 1

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_SO = os.path.join(_BUILD, "liboracle.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile oracle.c with gcc into oracle/_build/liboracle.so."""
    os.makedirs(_BUILD, exist_ok=True)
    if (not force and os.path.exists(_SO)
            and os.path.getmtime(_SO) >= os.path.getmtime(_SRC)):
        return _SO
    tmp = _SO + f".{os.getpid()}.tmp"
    cmd = ["gcc", "-O2", "-fopenmp", "-ffp-contract=off", "-std=c11",
           "-Wall", "-shared", "-fPIC", _SRC, "-o", tmp, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _SO)
    return _SO


class _Geom(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int) for n in (
        "B", "H", "W", "C_in", "C_out", "KH", "KW",
        "sh", "sw", "ph", "pw", "dh", "dw", "relu")]


def _load():
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        lib = ctypes.CDLL(build())
        P = ctypes.c_void_p
        i32, i64, dbl = ctypes.c_int, ctypes.c_int64, ctypes.c_double
        lib.oracle_keep_count.argtypes = [i64, dbl]
        lib.oracle_keep_count.restype = i64
        lib.oracle_block_scores.argtypes = [P, i32, i32, i32, i32, i32, i32, P]
        lib.oracle_prune.argtypes = [P, i32, i32, i32, i32, i32, dbl, i32, P, P]
        lib.oracle_prune.restype = i32
        lib.oracle_rearrange.argtypes = [P, i32, i32, i32, i32, P, i32, i32, i32, P]
        lib.oracle_rearrange.restype = i32
        lib.oracle_round_bf16.argtypes = [P, P, i64]
        lib.oracle_pack.argtypes = [P, P, i32, i32, i32, i32, i32, i32, P, P, P, i64]
        lib.oracle_pack.restype = i64
        lib.oracle_unpack.argtypes = [P, P, P, i32, i32, i32, i32, i32, P]
        lib.oracle_conv_masked.argtypes = [P, P, P, P, ctypes.POINTER(_Geom), i32,
                                           P, i64, P, P]
        lib.oracle_conv_bsr.argtypes = [P, P, P, P, i32, P, ctypes.POINTER(_Geom),
                                        i32, P, i64, P]
        lib.oracle_dwconv.argtypes = [P, P, P, ctypes.POINTER(_Geom), P]
        lib.oracle_conv_backward_data.argtypes = [P, P, P, ctypes.POINTER(_Geom), i32, P, P]
        lib.oracle_conv_backward_weight.argtypes = [P, P, P, ctypes.POINTER(_Geom), i32, P, P]
        lib.oracle_num_threads.restype = i32
        _lib = lib
        return lib


def _ptr(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _c(a, dtype):
    return None if a is None else np.ascontiguousarray(a, dtype=dtype)


def num_threads() -> int:
    return int(_load().oracle_num_threads())


def keep_count(total_blocks: int, rate: float) -> int:
    """Kept blocks for rate p over `total_blocks` blocks (Eq. 1; reading C3)."""
    return int(_load().oracle_keep_count(int(total_blocks), float(rate)))


def block_scores(W, N: int, gran: int = GRAN_TAP) -> np.ndarray:
    """Block l1 norms of Eq. 4: [G, KH*KW*C_in] (tap) or [G, C_in] (kernel)."""
    W = _c(W, np.float32)
    C_out, C_in, KH, KW = W.shape
    nb = KH * KW * C_in if gran == GRAN_TAP else C_in
    out = np.empty((C_out // N, nb), np.float64)
    _load().oracle_block_scores(_ptr(W), C_out, C_in, KH, KW, N, gran, _ptr(out))
    return out


def prune(W, N: int, rate: float, gran: int = GRAN_TAP):
    """1xN mask (solution after Eq. 5).  Returns (mask [G, KH*KW*C_in] uint8, kept)."""
    W = _c(W, np.float32)
    C_out, C_in, KH, KW = W.shape
    mask = np.empty((C_out // N, KH * KW * C_in), np.uint8)
    kept = ctypes.c_int64(0)
    rc = _load().oracle_prune(_ptr(W), C_out, C_in, KH, KW, N, float(rate), gran,
                              _ptr(mask), ctypes.byref(kept))
    if rc != 0:
        raise ValueError("oracle_prune: invalid arguments")
    return mask, int(kept.value)


def rearrange(W_l, W_next=None):
    """Sec. 3.3: returns (W_l', W_next' or None, perm int32[C_out])."""
    W_l = np.array(W_l, dtype=np.float32, copy=True, order="C")
    C_out, C_in, KH, KW = W_l.shape
    perm = np.empty(C_out, np.int32)
    if W_next is not None:
        W_next = np.array(W_next, dtype=np.float32, copy=True, order="C")
        Cn, Cin_n, KHn, KWn = W_next.shape
        assert Cin_n == C_out
    else:
        Cn = KHn = KWn = 0
    _load().oracle_rearrange(_ptr(W_l), C_out, C_in, KH, KW, _ptr(W_next), Cn, KHn,
                             KWn, _ptr(perm))
    return W_l, W_next, perm


def round_bf16(a) -> np.ndarray:
    """fp32 -> nearest-even bfloat16 value, returned as fp32."""
    a = _c(a, np.float32)
    out = np.empty_like(a)
    _load().oracle_round_bf16(_ptr(a), _ptr(out), a.size)
    return out


def pack(W, mask, N: int, dtype: str = "f32"):
    """Sec. 3.4 BSR encoding.  Returns (P int32[G+1], I int32[t], D [t, N]).

    D is float32 for dtype 'f32' and uint16 bfloat16 bits for 'bf16'."""
    W = _c(W, np.float32)
    mask = _c(mask, np.uint8)
    C_out, C_in, KH, KW = W.shape
    G = C_out // N
    t_cap = int(mask.sum())
    P = np.empty(G + 1, np.int32)
    I = np.empty(max(t_cap, 1), np.int32)
    D = np.empty((max(t_cap, 1), N), np.float32 if dtype == "f32" else np.uint16)
    t = _load().oracle_pack(_ptr(W), _ptr(mask), C_out, C_in, KH, KW, N,
                            0 if dtype == "f32" else 1, _ptr(P), _ptr(I), _ptr(D), t_cap)
    assert t == t_cap
    return P, I[:t].copy(), D[:t].copy()


def unpack(P, I, D, shape, N: int) -> np.ndarray:
    """Inverse of `pack` for fp32 D: the dense masked OIHW weights."""
    C_out, C_in, KH, KW = shape
    W = np.empty(shape, np.float32)
    P, I, D = _c(P, np.int32), _c(I, np.int32), _c(D, np.float32)
    _load().oracle_unpack(_ptr(P), _ptr(I), _ptr(D), C_out, C_in, KH, KW, N, _ptr(W))
    return W


def out_hw(H, W, KH, KW, stride=(1, 1), pad=(0, 0), dil=(1, 1)):
    Ho = (H + 2 * pad[0] - dil[0] * (KH - 1) - 1) // stride[0] + 1
    Wo = (W + 2 * pad[1] - dil[1] * (KW - 1) - 1) // stride[1] + 1
    return Ho, Wo


def _act_code(relu):
    """False / True / "relu6" (or 0 / 1 / 2): none, ReLU, ReLU6."""
    if relu == "relu6" or (not isinstance(relu, bool) and relu == 2):
        return 2
    return int(bool(relu))


def _geom(x_shape, C_out, KH, KW, stride, pad, dil, relu):
    B, H, W, C_in = x_shape
    return _Geom(B, H, W, C_in, C_out, KH, KW, stride[0], stride[1], pad[0], pad[1],
                 dil[0], dil[1], _act_code(relu))


def activation(y, relu):
    """The activation applied after bias (and residual): none, ReLU, ReLU6."""
    code = _act_code(relu)
    if code >= 1:
        y = np.maximum(y, 0.0)
    if code == 2:
        y = np.minimum(y, 6.0)
    return y


def conv_masked(x, W, mask=None, bias=None, N: int = 1, stride=(1, 1), pad=(0, 0),
                dil=(1, 1), relu=False, pixels=None, want_abs=False, residual=None):
    """Eq. 6: y = (W (+) T) * x (+bias, activation), NHWC, fp64 accumulation.

    relu: False / True / "relu6".  residual (optional, the output's shape or
    [len(pixels), C_out]): y = act(conv + bias + residual), the residual add
    of MobileNet-V2's inverted-residual block, applied here in numpy.

    x: [B, H, W, C_in] float32 (already rounded if the path is bf16);
    W: [C_out, C_in, KH, KW] float32; mask: [C_out/N, KH*KW*C_in] or None.
    pixels: optional int64 list of flattened output pixels (b*Ho*Wo+oh*Wo+ow);
    then y is [len(pixels), C_out], else [B, Ho, Wo, C_out].
    want_abs also returns sum |w x| + |b| per output (reading C12)."""
    if residual is not None:
        out = conv_masked(x, W, mask, bias, N, stride, pad, dil, False, pixels, want_abs)
        y, a = out if want_abs else (out, None)
        y = activation(y + np.asarray(residual, np.float64).reshape(y.shape), relu)
        if a is not None:
            a = a + np.abs(np.asarray(residual, np.float64)).reshape(a.shape)
        return (y, a) if want_abs else y
    x, W = _c(x, np.float32), _c(W, np.float32)
    C_out, C_in, KH, KW = W.shape
    B, H, Wd, Cx = x.shape
    assert Cx == C_in
    g = _geom(x.shape, C_out, KH, KW, stride, pad, dil, relu)
    Ho, Wo = out_hw(H, Wd, KH, KW, stride, pad, dil)
    mask = _c(mask, np.uint8)
    bias = _c(bias, np.float32)
    pix = _c(pixels, np.int64)
    n = len(pix) if pix is not None else B * Ho * Wo
    y = np.empty((n, C_out), np.float64)
    a = np.empty((n, C_out), np.float64) if want_abs else None
    _load().oracle_conv_masked(_ptr(x), _ptr(W), _ptr(mask), _ptr(bias), ctypes.byref(g),
                               N, _ptr(pix), n, _ptr(y), _ptr(a))
    if pix is None:
        y = y.reshape(B, Ho, Wo, C_out)
        a = a.reshape(B, Ho, Wo, C_out) if a is not None else None
    return (y, a) if want_abs else y


def dwconv(x, W, bias=None, stride=(1, 1), pad=(0, 0), dil=(1, 1), relu=False):
    """Dense depthwise convolution: y[b,oh,ow,c] = act(bias[c] + sum_{kh,kw}
    W[c,kh,kw] * x[b, oh*s-p+kh*d, ow*s-p+kw*d, c]), NHWC, fp64.
    x: [B, H, W, C] float32; W: [C, KH, KW] float32."""
    x, W = _c(x, np.float32), _c(W, np.float32)
    C, KH, KW = W.shape
    B, H, Wd, Cx = x.shape
    assert Cx == C
    g = _geom(x.shape, C, KH, KW, stride, pad, dil, relu)
    Ho, Wo = out_hw(H, Wd, KH, KW, stride, pad, dil)
    bias = _c(bias, np.float32)
    y = np.empty((B, Ho, Wo, C), np.float64)
    _load().oracle_dwconv(_ptr(x), _ptr(W), _ptr(bias), ctypes.byref(g), _ptr(y))
    return y


def conv_bsr(x, P, I, D, C_out, KH, KW, N, bias=None, stride=(1, 1), pad=(0, 0),
             dil=(1, 1), relu=False, pixels=None):
    """Eq. 7: block-wise decode of the BSR weights.  D fp32 or uint16 (bf16 bits)."""
    x = _c(x, np.float32)
    B, H, Wd, C_in = x.shape
    P, I = _c(P, np.int32), _c(I, np.int32)
    D = np.ascontiguousarray(D)
    dt = 1 if D.dtype == np.uint16 else 0
    if dt == 0:
        D = D.astype(np.float32, copy=False)
    g = _geom(x.shape, C_out, KH, KW, stride, pad, dil, relu)
    Ho, Wo = out_hw(H, Wd, KH, KW, stride, pad, dil)
    bias = _c(bias, np.float32)
    pix = _c(pixels, np.int64)
    n = len(pix) if pix is not None else B * Ho * Wo
    y = np.empty((n, C_out), np.float64)
    _load().oracle_conv_bsr(_ptr(x), _ptr(P), _ptr(I), _ptr(D), dt, _ptr(bias),
                            ctypes.byref(g), N, _ptr(pix), n, _ptr(y))
    return y.reshape(B, Ho, Wo, C_out) if pix is None else y


def conv_backward_data(dy, W, mask, N: int, in_hw, stride=(1, 1), pad=(0, 0), dil=(1, 1),
                       want_abs=False):
    """Gradient of Eq. 6's pre-activation output with respect to the input,
    the mask held fixed: dx[b,ih,iw,c] = sum over (o, kh, kw, oh, ow) with
    oh*s - p + kh*d = ih (and likewise for w) of mask * W[o,c,kh,kw] *
    dy[b,oh,ow,o].  dy: [B, Ho, Wo, C_out] float32 (the values the GPU
    sees); W: [C_out, C_in, KH, KW]; in_hw = (H, W) of the input.
    Returns dx [B, H, W, C_in] fp64 (and sum of |terms| if want_abs)."""
    dy, W = _c(dy, np.float32), _c(W, np.float32)
    C_out, C_in, KH, KW = W.shape
    B, Ho, Wo, Cy = dy.shape
    H, Wd = in_hw
    assert Cy == C_out and out_hw(H, Wd, KH, KW, stride, pad, dil) == (Ho, Wo)
    g = _geom((B, H, Wd, C_in), C_out, KH, KW, stride, pad, dil, False)
    mask = _c(mask, np.uint8)
    dx = np.empty((B, H, Wd, C_in), np.float64)
    a = np.empty_like(dx) if want_abs else None
    _load().oracle_conv_backward_data(_ptr(dy), _ptr(W), _ptr(mask), ctypes.byref(g), N, _ptr(dx), _ptr(a))
    return (dx, a) if want_abs else dx


def conv_backward_weight(x, dy, kernel, mask, N: int, stride=(1, 1), pad=(0, 0), dil=(1, 1),
                         want_abs=False):
    """Gradient of Eq. 6's pre-activation output with respect to the kept
    weights, the mask held fixed: dW[o,c,kh,kw] = mask * sum_{b,oh,ow}
    dy[b,oh,ow,o] * x[b, oh*s - p + kh*d, ow*s - p + kw*d, c] (zero where
    pruned).  x: [B, H, W, C_in], dy: [B, Ho, Wo, C_out] float32; kernel =
    (KH, KW).  Returns dW [C_out, C_in, KH, KW] fp64 (and sum |terms|)."""
    x, dy = _c(x, np.float32), _c(dy, np.float32)
    KH, KW = kernel
    B, H, Wd, C_in = x.shape
    C_out = dy.shape[3]
    assert dy.shape[:3] == (B,) + out_hw(H, Wd, KH, KW, stride, pad, dil)
    g = _geom(x.shape, C_out, KH, KW, stride, pad, dil, False)
    mask = _c(mask, np.uint8)
    dW = np.empty((C_out, C_in, KH, KW), np.float64)
    a = np.empty_like(dW) if want_abs else None
    _load().oracle_conv_backward_weight(_ptr(x), _ptr(dy), _ptr(mask), ctypes.byref(g), N, _ptr(dW), _ptr(a))
    return (dW, a) if want_abs else dW


def bsr_gather(dW, P, I, N: int):
    """The kept blocks of a dense [C_out, C_in, KH, KW] array in BSR order
    (Sec. 3.4): out[z, n] = dW[g*N + n, c, kh, kw] for P[g] <= z < P[g+1]
    and I[z] = (kh*KW + kw)*C_in + c.  Returns [t, N] (dW's dtype)."""
    dW = np.asarray(dW)
    C_out, C_in, KH, KW = dW.shape
    P, I = np.asarray(P, np.int64), np.asarray(I, np.int64)
    out = np.zeros((len(I), N), dW.dtype)
    for g in range(C_out // N):
        for z in range(P[g], P[g + 1]):
            tap, c = divmod(int(I[z]), C_in)
            kh, kw = divmod(tap, KW)
            out[z] = dW[g * N:(g + 1) * N, c, kh, kw]
    return out
