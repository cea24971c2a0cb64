"""GPU parity of the sparse tensor-core family (ONEXN_ALGO_MMA, bf16) against
the fp64 oracle: Eq. 7 with only the kept blocks multiplied.

Cases cover block widths 16..128, rates 0..1 (empty groups, all-pruned
layers), channel counts that leave a partial 64-channel chunk or an empty
half-chunk, ragged pixel tiles, partial group tiles, every TMA path (tiled
1x1, im2col with stride, padding and dilation) and the fused residual with
ReLU6.  Tolerance 4e-3 (bf16 output rounding) on bf16-rounded inputs,
normalised by sum |w x| + |b|."""
import numpy as np
import pytest
import torch

import oracle
from paper_2105_14713_gb300 import onexn as ox
from paper_2105_14713_gb300 import workloads as wl
from paper_2105_14713_gb300.layer import PrunedConv2d
from tests.gpu_util import norm_err, run_layer, tol

pytestmark = pytest.mark.gpu

L = wl.ConvLayer
MMA = ox.ONEXN_ALGO_MMA


def _run(layer, **kw):
    y, yr, a, conv = run_layer(layer, algo=MMA, **kw)
    B, H, W = layer.B, layer.H, layer.W
    assert conv.algo((B, H, W, layer.C_in), MMA) == "mma"
    return norm_err(y, yr, a)


@pytest.mark.parametrize("rate", [0.0, 0.3, 0.7, 0.9, 1.0])
@pytest.mark.parametrize("N", [16, 32])
def test_rates(N, rate):
    # 72 input channels: a second, partial chunk whose upper half-chunk is
    # empty; 160 outputs: a partial last group tile; 390 pixels: a ragged
    # last pixel tile
    layer = L("mma_rates", 2, 15, 13, 72, 160, 3, 3, 1, 1, 1, N=N, rate=rate, dtype="bf16", seed=N + int(10 * rate))
    assert _run(layer, relu=True) <= tol(layer)


@pytest.mark.parametrize("N", [64, 128])
def test_wide_blocks(N):
    layer = L("mma_wide", 2, 12, 12, 64, 256, 3, 3, 1, 1, 1, N=N, rate=0.5, dtype="bf16", seed=N)
    assert _run(layer) <= tol(layer)


GEOMS = [
    # name, B, H, W, C_in, C_out, KH, KW, stride, pad, dil
    ("1x1_tiled", 3, 13, 11, 64, 64, 1, 1, 1, 0, 1),
    ("1x1_c200", 2, 9, 9, 200, 48, 1, 1, 1, 0, 1),
    ("1x1_s2", 2, 15, 15, 40, 32, 1, 1, 2, 0, 1),
    ("3x3_s2", 3, 15, 13, 32, 64, 3, 3, 2, 1, 1),
    ("3x3_d2", 2, 16, 16, 48, 32, 3, 3, 1, 2, 2),
    ("1x3", 2, 9, 20, 16, 32, 1, 3, 1, 1, 1),
    ("5x5_p0_c8", 1, 20, 20, 8, 32, 5, 5, 1, 0, 1),
]


@pytest.mark.parametrize("geom", GEOMS, ids=[g[0] for g in GEOMS])
def test_geometries(geom):
    name, B, H, W, Ci, Co, KH, KW, s, p, d = geom
    layer = L(name, B, H, W, Ci, Co, KH, KW, s, p, d, N=16, rate=0.6, dtype="bf16", seed=Ci)
    assert _run(layer, relu=True) <= tol(layer)


def test_resnet50_stage3_3x3_shape():
    """A ResNet-50 stage-3 3x3 layer (256 -> 256, 14x14) at the stack's
    block width and rate (N = 16, 70%), batch 8: 36 chunks per tile."""
    layer = L("r50_s3_3x3", 8, 14, 14, 256, 256, 3, 3, 1, 1, 1, N=16, rate=0.7, dtype="bf16", seed=11)
    assert _run(layer, relu=True) <= tol(layer)


@pytest.mark.parametrize("aliased", [False, True])
def test_residual_and_relu6(aliased):
    layer = L("mma_res", 3, 14, 14, 64, 64, 1, 1, 1, 0, 1, N=16, rate=0.5, dtype="bf16", seed=5)
    W, b = wl.weights(layer).numpy(), wl.bias(layer).numpy()
    conv = PrunedConv2d(W, 16, 0.5, bias=b, dtype="bf16")
    xd = wl.activations(layer).to(torch.bfloat16).cuda()
    rng = np.random.default_rng(3)
    r = torch.from_numpy((3 * rng.standard_normal((3, 14, 14, 64))).astype(np.float32)).to(torch.bfloat16).cuda()
    r_host = r.float().cpu().numpy()
    y = r.clone() if aliased else torch.empty_like(r)
    conv(xd, y, relu="relu6", algo=MMA, residual=y if aliased else r)
    mask, _ = oracle.prune(W, 16, 0.5)
    ref, absacc = oracle.conv_masked(xd.float().cpu().numpy(), oracle.round_bf16(W), mask, b, 16, relu="relu6",
                                     residual=r_host, want_abs=True)
    err = np.max(np.abs(y.float().cpu().numpy().astype(np.float64) - ref) / (absacc + np.abs(r_host) + 1e-30))
    assert err <= 4e-3
    assert (ref == 6).any() and (ref == 0).any()


def test_unsupported_cases_are_refused():
    desc = ox.make_desc(1, 8, 8, 64, 64, 3, 3, 1, 1)
    for N, dt in ((8, ox.ONEXN_BF16), (16, ox.ONEXN_F32), (4, ox.ONEXN_BF16)):
        with pytest.raises(ox.OnexnError) as ei:
            ox.onexn_conv_algo(desc, N, 1, dt, MMA, 1 << 40)
        assert ei.value.status == ox.ONEXN_EUNSUPPORTED


def test_repeated_calls_are_identical():
    """The plan table is rebuilt every call and the kernel has no state: two
    calls give the same bits."""
    layer = L("mma_rep", 2, 14, 14, 128, 128, 3, 3, 1, 1, 1, N=16, rate=0.7, dtype="bf16", seed=2)
    W = wl.weights(layer).numpy()
    conv = PrunedConv2d(W, 16, 0.7, bias=wl.bias(layer).numpy(), padding=1, dtype="bf16")
    x = wl.activations(layer).to(torch.bfloat16).cuda()
    y1 = conv(x, algo=MMA).clone()
    y2 = conv(x, algo=MMA)
    torch.cuda.synchronize()
    assert torch.equal(y1, y2)
    assert ox.onexn_device_status(clear=True) == ox.ONEXN_OK
