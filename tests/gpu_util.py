"""Helpers for the GPU parity tests: run one layer through the C ABI and the
oracle on the same seeded inputs, and measure the normalised error

    err = |y - y_ref| / (sum_kept |w x| + |b| + 1e-30)          (reading C12)

against the fp64 oracle.  Tolerances: fp32 1e-5, bf16 1e-2."""
from __future__ import annotations

import numpy as np
import torch

import oracle
from paper_2105_14713_gb300 import onexn as ox
from paper_2105_14713_gb300 import workloads as wl
from paper_2105_14713_gb300.layer import PrunedConv2d

TOL = {"f32": 1e-5, "bf16": 1e-2}


def to_device_input(x_cpu: torch.Tensor, dtype: str) -> torch.Tensor:
    t = x_cpu if dtype == "f32" else x_cpu.to(torch.bfloat16)
    return t.contiguous().cuda()


def oracle_input(x_cpu: torch.Tensor, dtype: str) -> np.ndarray:
    """The values the GPU sees, as fp32 (bf16-rounded for the bf16 path)."""
    x = x_cpu.numpy()
    return x if dtype == "f32" else oracle.round_bf16(x)


TOL_BF16_ROUNDED = 4e-3     # bf16 output rounding (2^-8 relative, 8 significant bits) + fp32 accumulation


def oracle_ref(layer, W, x_cpu, b, *, relu=False, pixels=None, gran=ox.ONEXN_GRAN_TAP,
               master=False):
    """fp64 oracle output and sum |w x| + |b| on the values the GPU sees
    (bf16-rounded for the bf16 path), or on the fp32 master values."""
    rounded = layer.dtype == "bf16" and not master
    xo = oracle.round_bf16(x_cpu.numpy()) if rounded else x_cpu.numpy()
    Wo = oracle.round_bf16(W) if rounded else W
    mask_o, _ = oracle.prune(W, layer.N, layer.rate, gran)
    y_ref, absacc = oracle.conv_masked(xo, Wo, mask_o, b, layer.N, (layer.stride,) * 2,
                                       (layer.pad,) * 2, (layer.dil,) * 2, relu=relu,
                                       pixels=pixels, want_abs=True)
    return y_ref.reshape(-1, layer.C_out), absacc.reshape(-1, layer.C_out)


def run_layer(layer: wl.ConvLayer, *, relu=False, with_bias=True, algo=ox.ONEXN_ALGO_AUTO,
              pixels=None, gran=ox.ONEXN_GRAN_TAP, W=None, x_cpu=None, master=False):
    """Returns (y_gpu [n, C_out] fp64, y_ref, absacc, conv) on all or sampled pixels."""
    if W is None:
        W = wl.weights(layer).numpy()
    if x_cpu is None:
        x_cpu = wl.activations(layer)
    b = wl.bias(layer).numpy() if with_bias else None
    conv = PrunedConv2d(W, layer.N, layer.rate, bias=b, stride=layer.stride, padding=layer.pad,
                        dilation=layer.dil, dtype=layer.dtype, gran=gran)
    y = conv(to_device_input(x_cpu, layer.dtype), relu=relu, algo=algo)
    torch.cuda.synchronize()
    y = y.float().cpu().numpy().reshape(-1, layer.C_out).astype(np.float64)
    if pixels is not None:
        y = y[np.asarray(pixels)]
    y_ref, absacc = oracle_ref(layer, W, x_cpu, b, relu=relu, pixels=pixels, gran=gran,
                               master=master)
    return y, y_ref, absacc, conv


def tol(layer, master=False) -> float:
    if layer.dtype == "f32":
        return TOL["f32"]
    return TOL["bf16"] if master else TOL_BF16_ROUNDED


def norm_err(y, y_ref, absacc) -> float:
    if y.size == 0:
        return 0.0
    return float(np.max(np.abs(y - y_ref) / (absacc + 1e-30)))
