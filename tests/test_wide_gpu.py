"""GPU parity of the im2col GEMM on 256-row tiles against the fp64 oracle
(Eq. 6 / Eq. 7).

bf16 layers for which the 128-row plan takes 128-column tiles (more than 76
pixel tiles, so at least ~10k output pixels) run the tensor-core GEMM on
tiles of 256 output pixels (two 128-row halves with their own accumulators
and A tiles sharing every B tile) when their K loop has 32 or more
64-channel chunks, or, for stride-1 spatial layers, 16 or more chunks and
two full rounds of 256-row tiles, unless a halo form takes them: the
spatial cases here have 7x7 outputs, whose padding would waste 23% of a
halo tile (as on ResNet-50's stage 4).  The cases (3x3 over 256 channels:
36 chunks) cover a last tile whose second half is partly or wholly past the
output, fewer output channels than the column tile, a ragged round split
across CTAs (stream-K), a stride-2 layer and a 1x1 layer over 2048
channels, and the residual + ReLU6 epilogue; a strided 18-chunk and a 1x1
16-chunk layer of the same size check the boundary of the choice (128-row
tiles).  Every case checks the form it runs.
Checked on 2000 seeded output pixels spread over every image, plus every
pixel of the last tile.  Tolerance: 4e-3 = 2^-8 output rounding on
bf16-rounded inputs, normalised by sum |w x| + |b|."""
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

WIDE_GEOMS = [
    # name, B, H, W, C_in, C_out, KH, KW, stride, pad, N, form
    ("3x3_c256", 256, 7, 7, 256, 128, 3, 3, 1, 1, 16, "im2col_wide"),         # 12544 pixels = 49 tiles of 256
    ("3x3_half_partly", 208, 7, 7, 256, 128, 3, 3, 1, 1, 16, "im2col_wide"),  # last tile: second half 80 of 128 rows
    ("3x3_half_empty", 200, 7, 7, 256, 128, 3, 3, 1, 1, 16, "im2col_wide"),   # last tile: second half wholly past y
    ("3x3_cout96", 256, 7, 7, 256, 96, 3, 3, 1, 1, 8, "im2col_wide"),         # 96 of 128 columns
    ("3x3_cout512_rounds", 200, 7, 7, 256, 512, 3, 3, 1, 1, 16, "im2col_wide"),  # 156 tiles: a ragged second round
    ("3x3_s2_c256", 256, 14, 14, 256, 128, 3, 3, 2, 1, 16, "im2col_wide"),    # strided traversal of each half, 36 chunks
    ("1x1_k2048", 64, 14, 14, 2048, 128, 1, 1, 1, 0, 16, "im2col_wide"),      # plain-matrix A, 32 chunks
    ("3x3_s2_128rows", 256, 14, 14, 128, 128, 3, 3, 2, 1, 16, "im2col"),      # strided, 18 chunks: 128-row tiles
    ("1x1_k1024_128rows", 64, 14, 14, 1024, 128, 1, 1, 1, 0, 8, "im2col"),    # 1x1: 128-row tiles
]


def _pixels(layer, seed):
    """2000 seeded pixels plus the whole last 256-row tile."""
    rng = np.random.default_rng(seed)
    last = np.arange((layer.pixels - 1) // 256 * 256, layer.pixels)
    return np.unique(np.concatenate([rng.choice(layer.pixels, 2000, replace=False), last]))


@pytest.mark.parametrize("geom", WIDE_GEOMS, ids=[g[0] for g in WIDE_GEOMS])
@pytest.mark.parametrize("rate", [0.0, 0.7])
def test_wide_tiles_match_oracle(geom, rate):
    name, B, H, W, Ci, Co, KH, KW, s, p, N, form = geom
    layer = L(name, B, H, W, Ci, Co, KH, KW, s, p, 1, N=N, rate=rate, dtype="bf16", seed=Ci + Co + B)
    pix = _pixels(layer, B)
    y, yr, a, conv = run_layer(layer, relu=True, algo=ox.ONEXN_ALGO_TC, pixels=pix)
    assert conv.algo((B, H, W, Ci), ox.ONEXN_ALGO_TC) == "tc"
    assert conv.tc_form((B, H, W, Ci)) == form
    assert norm_err(y, yr, a) <= TOL_BF16_ROUNDED
    # again with the decoded weights resident: bitwise the same
    x = wl.activations(layer).to(torch.bfloat16).cuda()
    y1 = conv(x, relu=True, algo=ox.ONEXN_ALGO_TC)
    y2 = conv(x, relu=True, algo=ox.ONEXN_ALGO_TC)
    torch.cuda.synchronize()
    assert torch.equal(y1, y2)


def test_wide_tiles_residual_relu6():
    layer = L("wide_res", 256, 7, 7, 256, 128, 3, 3, 1, 1, 1, N=16, rate=0.5, dtype="bf16", seed=13)
    W, b = wl.weights(layer).numpy(), wl.bias(layer).numpy()
    conv = PrunedConv2d(W, 16, 0.5, bias=b, padding=1, dtype="bf16")
    assert conv.tc_form((256, 7, 7, 256)) == "im2col_wide"
    x = wl.activations(layer).to(torch.bfloat16).cuda()
    rng = np.random.default_rng(9)
    r = torch.from_numpy((3 * rng.standard_normal((256, 7, 7, 128))).astype(np.float32)).to(torch.bfloat16).cuda()
    y = conv(x, relu="relu6", algo=ox.ONEXN_ALGO_TC, residual=r)
    torch.cuda.synchronize()
    pix = _pixels(layer, 9)
    mask, _ = oracle.prune(W, 16, 0.5, ox.ONEXN_GRAN_TAP)
    r_pix = r.float().cpu().numpy().reshape(-1, 128)[pix]
    ref, absacc = oracle.conv_masked(x.float().cpu().numpy(), oracle.round_bf16(W), mask, b, 16, (1, 1), (1, 1),
                                     relu="relu6", pixels=pix, residual=r_pix, want_abs=True)
    got = y.float().cpu().numpy().reshape(-1, 128)[pix].astype(np.float64)
    assert norm_err(got, ref, absacc) <= TOL_BF16_ROUNDED
    assert (ref == 6).any() and (ref == 0).any()


RESIDENT_GEOMS = [
    # name, B, H, W, C_in, C_out, dtype: 1x1 layers whose K loop fits in the stage ring
    ("bf16_k128_cout512", 64, 28, 28, 128, 512, "bf16"),    # 2 chunks, 2 column tiles of 256 on 152 CTAs
    ("bf16_k256_cout1024", 128, 14, 14, 256, 1024, "bf16"),  # 4 chunks, 4 column tiles
    ("bf16_k256_cout768", 128, 14, 14, 256, 768, "bf16"),   # 3 column tiles: 152 CTAs do not divide, B streamed
    ("f32_k96_cout512", 32, 28, 28, 96, 512, "f32"),        # 3 chunks of 32 channels, hi and lo B parts
]


@pytest.mark.parametrize("geom", RESIDENT_GEOMS, ids=[g[0] for g in RESIDENT_GEOMS])
def test_resident_weights_multi_chunk(geom):
    """1x1 layers with a short K loop: each CTA keeps its column tile's B
    chunks in the stage ring (loaded by its first tile) when every tile it
    takes has the same column tile; checked on sampled pixels of every
    image, and bitwise equal on a second call with the weights resident."""
    name, B, H, W, Ci, Co, dt = geom
    layer = L(name, B, H, W, Ci, Co, 1, 1, 1, 0, 1, N=16, rate=0.7, dtype=dt, seed=Co)
    pix = _pixels(layer, Co)
    y, yr, a, conv = run_layer(layer, relu=True, algo=ox.ONEXN_ALGO_TC, pixels=pix)
    tol = TOL_BF16_ROUNDED if dt == "bf16" else 1e-5
    assert norm_err(y, yr, a) <= tol
    x = wl.activations(layer)
    x = (x if dt == "f32" else x.to(torch.bfloat16)).cuda()
    y1 = conv(x, relu=True, algo=ox.ONEXN_ALGO_TC)
    y2 = conv(x, relu=True, algo=ox.ONEXN_ALGO_TC)
    torch.cuda.synchronize()
    assert torch.equal(y1, y2)
