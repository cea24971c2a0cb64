"""The allocation-free entry point, onexn_conv_fwd_noalloc.

Some callers cannot allocate device memory: code running while a stream is
captured into a CUDA graph (an allocation there breaks the capture), hosts
that forbid allocation after start-up so that latency stays predictable, or
a plug-in that only receives pointers from a framework that owns the memory.
For them the library keeps the tensor-core family's scratch in a fixed 8 MiB
device array instead of a caller workspace.  These tests call it through the
C ABI on five layers in a row (the last three run the GEMM on halo tiles:
a stride-1 3x3 layer with its weights resident in shared memory, one with
them streamed, and a stride-2 3x3 layer over its four input phases) and
then on the first layer again (so it runs over what the others left in the
shared array), and check each output
against the fp64 oracle and bit for bit against the regular onexn_conv_fwd
with a workspace (the same kernels on the same decoded weights and the same
tile plan).  The file name sorts last so that a run that stops at the first
failure has already run every other test."""
import ctypes

import numpy as np
import pytest
import torch

from paper_2105_14713_gb300 import onexn as ox
from paper_2105_14713_gb300 import workloads as wl
from paper_2105_14713_gb300.layer import PrunedConv2d
from tests.gpu_util import norm_err, oracle_ref, tol

pytestmark = pytest.mark.gpu


def _layer_and_input(layer):
    W, b = wl.weights(layer).numpy(), wl.bias(layer).numpy()
    conv = PrunedConv2d(W, layer.N, layer.rate, bias=b, stride=layer.stride, padding=layer.pad,
                        dilation=layer.dil, dtype="bf16")
    x_cpu = wl.activations(layer)
    return conv, x_cpu, x_cpu.to(torch.bfloat16).cuda(), W, b


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


LAYERS = [
    wl.ConvLayer("na_3x3", 16, 7, 7, 128, 128, 3, 3, 1, 1, 1, N=8, rate=0.5, dtype="bf16", seed=1),
    wl.ConvLayer("na_1x1_s2", 3, 15, 15, 64, 256, 1, 1, 2, 0, 1, N=16, rate=0.7, dtype="bf16", seed=2),
    wl.ConvLayer("na_3x3_halo", 2, 28, 28, 64, 64, 3, 3, 1, 1, 1, N=16, rate=0.7, dtype="bf16", seed=3),
    wl.ConvLayer("na_3x3_streamed", 2, 28, 28, 256, 128, 3, 3, 1, 1, 1, N=16, rate=0.7, dtype="bf16", seed=4),
    wl.ConvLayer("na_3x3_s2_phases", 1, 56, 56, 64, 128, 3, 3, 2, 1, 1, N=16, rate=0.5, dtype="bf16", seed=5),
]
FORMS = ["im2col", "im2col", "halo_resident", "halo_streamed", "halo_streamed"]


def test_noalloc_five_layers_then_the_first_again():
    runs = [(0, True), (1, False), (2, True), (3, True), (4, False), (0, True)]
    for i, relu in runs:
        layer = LAYERS[i]
        conv, x_cpu, x, W, b = _layer_and_input(layer)
        assert conv.tc_form(x.shape) == FORMS[i], layer.name
        y_na = _noalloc(conv, x, relu)
        y_ws = conv(x, relu=relu, algo=ox.ONEXN_ALGO_TC)
        torch.cuda.synchronize()
        assert torch.equal(y_na, y_ws), layer.name
        y_ref, absacc = oracle_ref(layer, W, x_cpu, b, relu=relu)
        y = y_na.float().cpu().numpy().reshape(-1, layer.C_out).astype(np.float64)
        assert norm_err(y, y_ref, absacc) <= tol(layer), layer.name
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
