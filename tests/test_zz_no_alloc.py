"""The allocation-free entry point, onexn_conv_fwd_noalloc.

Some callers cannot allocate device memory (for example code running while
a stream is captured into a CUDA graph, or a plug-in that only receives
pointers from a framework that owns the memory).  For them the library keeps
the tensor-core family's scratch in a fixed 8 MiB device array instead of a
caller workspace.  These tests call it through the C ABI and check that two
calls in a row, on different layers, give the same output as the regular
onexn_conv_fwd with a workspace.  The file name sorts last so that a run that
stops at the first failure has already run every other test."""
import ctypes

import numpy as np
import pytest
import torch

from paper_2105_14713_gb300 import onexn as ox
from paper_2105_14713_gb300 import workloads as wl
from paper_2105_14713_gb300.layer import PrunedConv2d

pytestmark = pytest.mark.gpu


def _layer_and_input(layer):
    conv = PrunedConv2d(wl.weights(layer).numpy(), layer.N, layer.rate, bias=wl.bias(layer).numpy(),
                        stride=layer.stride, padding=layer.pad, dilation=layer.dil, dtype="bf16")
    x = wl.activations(layer).to(torch.bfloat16).cuda()
    return conv, x


def _noalloc(conv, x, relu):
    y = torch.empty(conv.out_shape(x.shape), dtype=torch.bfloat16, device="cuda")
    B, H, W, _ = x.shape
    d = conv.desc(B, H, W)
    st = ox.lib.onexn_conv_fwd_noalloc(
        ctypes.byref(d), ctypes.c_void_p(conv.P.data_ptr()), ctypes.c_void_p(conv.I.data_ptr()),
        ctypes.c_void_p(conv.D.data_ptr()), conv.N, conv.t, ctypes.c_void_p(x.data_ptr()),
        ctypes.c_void_p(y.data_ptr()), ctypes.c_void_p(conv.bias.data_ptr()), ox.ONEXN_BF16,
        ox.ONEXN_RELU if relu else 0, ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
    assert st == ox.ONEXN_OK, ox.lib.onexn_last_error()
    return y


def test_noalloc_matches_workspace_entry_two_calls_in_a_row():
    layers = [
        wl.ConvLayer("na_3x3", 4, 14, 14, 128, 128, 3, 3, 1, 1, 1, N=8, rate=0.5, dtype="bf16", seed=1),
        wl.ConvLayer("na_1x1_s2", 3, 15, 15, 64, 256, 1, 1, 2, 0, 1, N=16, rate=0.7, dtype="bf16", seed=2),
    ]
    outs = []
    for i, layer in enumerate(layers):
        conv, x = _layer_and_input(layer)
        y_na = _noalloc(conv, x, relu=(i == 0))
        y_ws = conv(x, relu=(i == 0), algo=ox.ONEXN_ALGO_TC)
        torch.cuda.synchronize()
        a, b = y_na.float().cpu().numpy(), y_ws.float().cpu().numpy()
        scale = np.abs(b).max() + 1e-30
        assert np.max(np.abs(a - b)) <= 4e-3 * scale, layer.name
        outs.append(a)
    assert ox.onexn_device_status() == ox.ONEXN_OK


def test_noalloc_rejects_layers_beyond_the_scratch():
    # 1024 x 3*3*512 bf16 = 9 MiB of decoded weights > the 8 MiB scratch
    d = ox.make_desc(1, 4, 4, 512, 1024, 3, 3, 1, 1, 1)
    one = torch.zeros(16, dtype=torch.int32, device="cuda")
    st = ox.lib.onexn_conv_fwd_noalloc(ctypes.byref(d), ctypes.c_void_p(one.data_ptr()),
                                       ctypes.c_void_p(one.data_ptr()),
                                       ctypes.c_void_p(one.data_ptr()), 8, 1,
                                       ctypes.c_void_p(one.data_ptr()), ctypes.c_void_p(one.data_ptr() + 32),
                                       None, ox.ONEXN_BF16, 0, None)
    assert st == ox.ONEXN_EINVAL
    assert b"scratch" in ox.lib.onexn_last_error()
    # fp32 needs twice as many 4-byte values: 36 MiB here
    st = ox.lib.onexn_conv_fwd_noalloc(ctypes.byref(d), None, None, None, 8, 1, None, None, None,
                                       ox.ONEXN_F32, 0, None)
    assert st == ox.ONEXN_EINVAL
    assert b"scratch" in ox.lib.onexn_last_error()
