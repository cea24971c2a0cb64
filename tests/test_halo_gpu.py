"""GPU parity of the halo-tile forms of the bf16 tensor-core GEMM against
the fp64 oracle (Eq. 6 / Eq. 7).

Stride-1 spatial bf16 layers whose padding wastes at most 15% of the M rows
run on halo tiles: one im2col load of the tile's input rows per 64-channel
chunk, each tap's A operand a row-shifted view of it.
 * Resident weights: tiles of whole output rows in the padded row width;
   the column tile's decoded weights stay in shared memory, so it needs
   them to fit next to two halo slots, and a column tile at least as wide
   as the im2col GEMM's.  Cases: one and two MMA warps, one and two column
   tiles, a half-empty channel chunk, one to four output rows per tile,
   padding 0 / 1 / 2, dilation 2, 1x3 and 3x1 kernels.
 * Streamed weights: tiles of 256 consecutive positions of the padded
   output space (two M = 128 halves, across rows and images), the weights
   streamed one kernel row of taps (3x3) or one tap per stage.  Cases: 64-
   and 128-column tiles, two and four column tiles, a partial channel chunk
   and a partial column tile, 1 to 8 chunks, padding 0 / 1 / 2, dilation 2,
   5x5, 3x1 and 1x3 kernels, and a last tile past the last image.
 * Strided layers on the streamed form, split into the phases of their
   input (one strided load per chunk and phase, each tap a shift within
   its phase): stride 2 with 3x3 (four phases of 4, 2, 2 and 1 taps), 5x5
   (25 taps), padding 0 and 1, an odd input size, dilation 2 (one phase),
   a partial channel chunk and a partial column tile.
A layer of each form with the residual + ReLU6 epilogue, and every case's
form checked.  The 28-wide 5x5 and the 7x7 3x3 cases would waste 23% of a
halo tile and run the im2col form, checked here all the same.  Tolerance: 4e-3 = 2^-8 output
rounding on bf16-rounded inputs, normalised by sum |w x| + |b|."""
import numpy as np
import pytest
import torch

import oracle
from paper_2105_14713_gb300 import onexn as ox
from paper_2105_14713_gb300 import workloads as wl
from paper_2105_14713_gb300.layer import PrunedConv2d
from tests.gpu_util import TOL_BF16_ROUNDED, norm_err, run_layer

pytestmark = pytest.mark.gpu

L = wl.ConvLayer

HALO_GEOMS = [
    # name, B, H, W, C_in, C_out, KH, KW, pad, dil, N, form
    ("r50_s1_like", 2, 28, 28, 64, 64, 3, 3, 1, 1, 16, "halo_resident"),     # two MMA warps, four rows per tile
    ("r50_s2_like", 2, 28, 28, 128, 128, 3, 3, 1, 1, 16, "halo_resident"),   # two column tiles of 64, two chunks
    ("w56_co128", 1, 56, 56, 64, 128, 3, 3, 1, 1, 16, "halo_resident"),      # two rows per tile, two column tiles
    ("w112_c32", 1, 112, 112, 32, 32, 3, 3, 1, 1, 8, "halo_resident"),       # one row per tile, half-empty chunk
    ("5x5_p2", 1, 28, 28, 32, 64, 5, 5, 2, 1, 16, "im2col"),                 # 32x32 padded: 23% dropped
    ("7x7_im2col", 4, 7, 7, 64, 64, 3, 3, 1, 1, 16, "im2col"),               # 8x8 padded: 23% dropped
    ("3x3_d2", 2, 28, 28, 64, 64, 3, 3, 2, 2, 16, "halo_resident"),
    ("3x3_p0", 2, 30, 30, 64, 64, 3, 3, 0, 1, 16, "halo_resident"),
    ("3x1_p1", 2, 28, 28, 64, 64, 3, 1, 1, 1, 16, "halo_resident"),
    ("1x3_p1", 2, 26, 28, 64, 64, 1, 3, 1, 1, 16, "halo_resident"),
    ("w40_c72_co96", 1, 40, 40, 72, 96, 3, 3, 1, 1, 8, "halo_streamed"),     # partial chunk and column tile
    ("st_c256_co256", 2, 28, 28, 256, 256, 3, 3, 1, 1, 16, "halo_streamed"),  # two column tiles, 4 chunks
    ("st_c256_co512", 1, 28, 28, 256, 512, 3, 3, 1, 1, 16, "halo_streamed"),  # four column tiles
    ("st_co64_c512", 2, 28, 28, 512, 64, 3, 3, 1, 1, 16, "halo_streamed"),    # 64 columns, four accumulators, 8 chunks
    ("st_d2", 1, 56, 56, 128, 128, 3, 3, 2, 2, 16, "halo_streamed"),          # dilation 2, two B stages
    ("st_5x5", 1, 56, 56, 128, 128, 5, 5, 2, 1, 16, "halo_streamed"),         # one tap per stage
    ("st_3x1", 2, 28, 28, 512, 128, 3, 1, 1, 1, 16, "halo_streamed"),
    ("st_1x3", 2, 26, 28, 512, 128, 1, 3, 1, 1, 16, "halo_streamed"),
    ("st_p0", 2, 30, 30, 256, 128, 3, 3, 0, 1, 16, "halo_streamed"),
    ("st_w120", 1, 120, 120, 128, 128, 3, 3, 1, 1, 16, "halo_streamed"),    # 122-wide rows: 502-position loads
    ("st_b1", 1, 28, 28, 256, 128, 3, 3, 1, 1, 16, "halo_streamed"),        # 4 tiles on 152 SMs
]


@pytest.mark.parametrize("geom", HALO_GEOMS, ids=[g[0] for g in HALO_GEOMS])
@pytest.mark.parametrize("rate", [0.0, 0.7])
def test_halo_layers_match_oracle(geom, rate):
    name, B, H, W, Ci, Co, KH, KW, p, d, N, form = geom
    layer = L(name, B, H, W, Ci, Co, KH, KW, 1, p, d, N=N, rate=rate, dtype="bf16", seed=Ci + Co)
    y, yr, a, conv = run_layer(layer, relu=True, algo=ox.ONEXN_ALGO_TC)
    assert conv.algo((B, H, W, Ci), ox.ONEXN_ALGO_TC) == "tc"
    assert conv.tc_form((B, H, W, Ci)) == form
    assert norm_err(y, yr, a) <= TOL_BF16_ROUNDED
    # the same layer again with its decoded weights resident is bitwise the same
    x = wl.activations(layer).to(torch.bfloat16).cuda()
    y1 = conv(x, relu=True, algo=ox.ONEXN_ALGO_TC)
    y2 = conv(x, relu=True, algo=ox.ONEXN_ALGO_TC)
    torch.cuda.synchronize()
    assert torch.equal(y1, y2)


STRIDED_GEOMS = [
    # name, B, H, W, C_in, C_out, KH, KW, stride, pad, dil, N
    ("s2_3x3_c128", 2, 56, 56, 128, 128, 3, 3, 2, 1, 1, 16),    # ResNet-50 stage-2 b1 shape: 29x29 phase space
    ("s2_3x3_c256", 2, 28, 28, 256, 256, 3, 3, 2, 1, 1, 16),    # stage-3 b1 shape: 15x15, two column tiles
    ("s2_3x3_odd", 2, 29, 29, 64, 128, 3, 3, 2, 1, 1, 8),       # odd input: 15x15 output, 16x16 phase space
    ("s2_5x5", 1, 56, 56, 128, 128, 5, 5, 2, 2, 1, 16),         # 25 taps in four phases
    ("s2_3x3_p0", 2, 57, 57, 128, 128, 3, 3, 2, 0, 1, 16),
    ("s2_3x3_d2", 1, 56, 56, 128, 128, 3, 3, 2, 2, 2, 16),      # every tap in one phase
    ("s2_c72_co96", 1, 56, 56, 72, 96, 3, 3, 2, 1, 1, 8),       # partial chunk and column tile
    ("s2_co64", 2, 56, 56, 128, 64, 3, 3, 2, 1, 1, 16),         # 64-column tiles
    ("s2_w120", 1, 120, 120, 128, 128, 3, 3, 2, 1, 1, 16),      # 61-wide phase rows
]


@pytest.mark.parametrize("geom", STRIDED_GEOMS, ids=[g[0] for g in STRIDED_GEOMS])
@pytest.mark.parametrize("rate", [0.0, 0.7])
def test_halo_strided_layers_match_oracle(geom, rate):
    name, B, H, W, Ci, Co, KH, KW, s, p, d, N = geom
    layer = L(name, B, H, W, Ci, Co, KH, KW, s, p, d, N=N, rate=rate, dtype="bf16", seed=Ci + Co + s)
    y, yr, a, conv = run_layer(layer, relu=True, algo=ox.ONEXN_ALGO_TC)
    assert conv.tc_form((B, H, W, Ci)) == "halo_streamed"
    assert norm_err(y, yr, a) <= TOL_BF16_ROUNDED
    x = wl.activations(layer).to(torch.bfloat16).cuda()
    y1 = conv(x, relu=True, algo=ox.ONEXN_ALGO_TC)
    y2 = conv(x, relu=True, algo=ox.ONEXN_ALGO_TC)
    torch.cuda.synchronize()
    assert torch.equal(y1, y2)


@pytest.mark.parametrize("C_in,H,s,form", [(64, 28, 1, "halo_resident"), (256, 28, 1, "halo_streamed"),
                                           (128, 56, 2, "halo_streamed")])
def test_halo_residual_relu6(C_in, H, s, form):
    layer = L("halo_res", 2, H, H, C_in, 64, 3, 3, s, 1, 1, N=16, rate=0.5, dtype="bf16", seed=11)
    W, b = wl.weights(layer).numpy(), wl.bias(layer).numpy()
    conv = PrunedConv2d(W, 16, 0.5, bias=b, stride=s, padding=1, dtype="bf16")
    assert conv.tc_form((2, H, H, C_in)) == form
    x = wl.activations(layer).to(torch.bfloat16).cuda()
    rng = np.random.default_rng(7)
    r = torch.from_numpy((3 * rng.standard_normal((2, 28, 28, 64))).astype(np.float32)).to(torch.bfloat16).cuda()
    y = conv(x, relu="relu6", algo=ox.ONEXN_ALGO_TC, residual=r)
    torch.cuda.synchronize()
    mask, _ = oracle.prune(W, 16, 0.5, ox.ONEXN_GRAN_TAP)
    ref, absacc = oracle.conv_masked(x.float().cpu().numpy(), oracle.round_bf16(W), mask, b, 16, (s, s), (1, 1),
                                     relu="relu6", residual=r.float().cpu().numpy(), want_abs=True)
    e = norm_err(y.float().cpu().numpy().reshape(-1, 64).astype(np.float64), ref.reshape(-1, 64),
                 absacc.reshape(-1, 64))
    assert e <= TOL_BF16_ROUNDED
    assert (ref == 6).any() and (ref == 0).any()     # both clamps exercised


@pytest.mark.parametrize("C_in,form", [(64, "halo_resident"), (512, "halo_streamed")])
def test_halo_empty_batch_and_output_untouched_outside(C_in, form):
    """A batch of zero images launches nothing; y's bytes past the layer's
    output are never written (the stores stay inside y)."""
    layer = L("halo_guard", 1, 28, 28, C_in, 64, 3, 3, 1, 1, 1, N=16, rate=0.5, dtype="bf16", seed=2)
    W = wl.weights(layer).numpy()
    conv = PrunedConv2d(W, 16, 0.5, padding=1, dtype="bf16")
    assert conv.tc_form((1, 28, 28, C_in)) == form
    x0 = torch.empty((0, 28, 28, C_in), dtype=torch.bfloat16, device="cuda")
    assert conv(x0, algo=ox.ONEXN_ALGO_TC).shape == (0, 28, 28, 64)
    x = wl.activations(layer).to(torch.bfloat16).cuda()
    big = torch.full((2 * 28 * 28 * 64,), 7.0, dtype=torch.bfloat16, device="cuda")
    big[: 28 * 28 * 64] = float("nan")
    y = big[: 28 * 28 * 64].view(1, 28, 28, 64)
    conv(x, y, algo=ox.ONEXN_ALGO_TC)
    torch.cuda.synchronize()
    assert torch.all(big[28 * 28 * 64:] == 7.0)
    assert not torch.any(torch.isnan(y))           # every output written


@pytest.mark.parametrize("B,H,C_in,C_out,s,form", [
    (32, 28, 128, 128, 1, "halo_streamed"), (64, 28, 64, 256, 1, "im2col"), (256, 28, 128, 128, 1, "halo_streamed"),
    (256, 56, 128, 128, 2, "halo_streamed"), (256, 28, 256, 256, 2, "im2col")],
    ids=["bn128", "bn256", "r50_s2_3x3", "r50_s2_b1_3x3_s2", "r50_s3_b1_3x3_s2"])
def test_halo_streamed_sampled(B, H, C_in, C_out, s, form):
    """Enough pixel tiles that the im2col GEMM takes 128- or 256-column
    tiles, wider than the resident-weights form allows: at 128 columns the
    layer runs the streamed-weights form (ResNet-50's stage-2 3x3 layers and
    the stride-2 one at batch 256 among them), at 256 it keeps the im2col
    form (the halo would be loaded once per 128-column tile); checked on
    3000 seeded output pixels over every image, plus every pixel of the last
    image."""
    layer = L("halo_wide", B, H, H, C_in, C_out, 3, 3, s, 1, 1, N=16, rate=0.5, dtype="bf16", seed=B + s)
    ho = (H - 1) // s + 1
    rng = np.random.default_rng(B)
    last = np.arange(layer.pixels - ho * ho, layer.pixels)
    pix = np.unique(np.concatenate([rng.choice(layer.pixels, 3000, replace=False), last]))
    y, yr, a, conv = run_layer(layer, relu=True, algo=ox.ONEXN_ALGO_TC, pixels=pix)
    assert conv.tc_form((B, H, H, C_in)) == form
    assert norm_err(y, yr, a) <= TOL_BF16_ROUNDED
    x = wl.activations(layer).to(torch.bfloat16).cuda()
    y1 = conv(x, relu=True, algo=ox.ONEXN_ALGO_TC)
    y2 = conv(x, relu=True, algo=ox.ONEXN_ALGO_TC)
    torch.cuda.synchronize()
    assert torch.equal(y1, y2)
