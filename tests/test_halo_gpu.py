"""GPU parity of the halo-tile form of the bf16 tensor-core GEMM against the
fp64 oracle (Eq. 6 / Eq. 7).

The tensor-core family runs a stride-1 spatial bf16 layer on halo tiles when
its output rows fill at least 85% of the 128-row M tile (output widths such
as 28, 30, 56 and 112), a column tile's decoded weights fit in shared
memory next to two halo slots, and that tile is at least as wide as the
im2col GEMM's: whole output rows per tile in the padded row
width, one im2col load of the tile's input rows per 64-channel chunk, and
each tap's A operand a row-shifted view of it.  The cases cover one and two
MMA warps, one and two column tiles (each CTA keeping its own tile's
weights), a half-empty channel chunk, one and two and four output rows per
tile, padding 0 / 1 / 2, dilation 2, 1x3 and 3x1 kernels, and the residual +
ReLU6 epilogue; the 40-wide 72-channel and the 5x5 cases do not fit and run
the im2col form, checked here all the same.  Tolerance: 4e-3 = 2^-8 output
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
    # name, B, H, W, C_in, C_out, KH, KW, pad, dil, N
    ("r50_s1_like", 2, 28, 28, 64, 64, 3, 3, 1, 1, 16),       # two MMA warps, four rows per tile
    ("r50_s2_like", 2, 28, 28, 128, 128, 3, 3, 1, 1, 16),     # two column tiles of 64 (few tiles), two chunks
    ("w40_c72_co96", 1, 40, 40, 72, 96, 3, 3, 1, 1, 8),       # im2col form (weights do not fit)
    ("w56_co128", 1, 56, 56, 64, 128, 3, 3, 1, 1, 16),        # two rows per tile, two column tiles
    ("w112_c32", 1, 112, 112, 32, 32, 3, 3, 1, 1, 8),         # one row per tile, half-empty chunk
    ("5x5_p2", 1, 28, 28, 32, 64, 5, 5, 2, 1, 16),           # im2col form (weights do not fit)
    ("3x3_d2", 2, 28, 28, 64, 64, 3, 3, 2, 2, 16),
    ("3x3_p0", 2, 30, 30, 64, 64, 3, 3, 0, 1, 16),
    ("3x1_p1", 2, 28, 28, 64, 64, 3, 1, 1, 1, 16),
    ("1x3_p1", 2, 26, 28, 64, 64, 1, 3, 1, 1, 16),
]


@pytest.mark.parametrize("geom", HALO_GEOMS, ids=[g[0] for g in HALO_GEOMS])
@pytest.mark.parametrize("rate", [0.0, 0.7])
def test_halo_layers_match_oracle(geom, rate):
    name, B, H, W, Ci, Co, KH, KW, p, d, N = geom
    layer = L(name, B, H, W, Ci, Co, KH, KW, 1, p, d, N=N, rate=rate, dtype="bf16", seed=Ci + Co)
    y, yr, a, conv = run_layer(layer, relu=True, algo=ox.ONEXN_ALGO_TC)
    assert conv.algo((B, H, W, Ci), ox.ONEXN_ALGO_TC) == "tc"
    assert norm_err(y, yr, a) <= TOL_BF16_ROUNDED
    # the same layer again with its decoded weights resident is bitwise the same
    x = wl.activations(layer).to(torch.bfloat16).cuda()
    y1 = conv(x, relu=True, algo=ox.ONEXN_ALGO_TC)
    y2 = conv(x, relu=True, algo=ox.ONEXN_ALGO_TC)
    torch.cuda.synchronize()
    assert torch.equal(y1, y2)


def test_halo_residual_relu6():
    layer = L("halo_res", 2, 28, 28, 64, 64, 3, 3, 1, 1, 1, N=16, rate=0.5, dtype="bf16", seed=11)
    W, b = wl.weights(layer).numpy(), wl.bias(layer).numpy()
    conv = PrunedConv2d(W, 16, 0.5, bias=b, padding=1, dtype="bf16")
    x = wl.activations(layer).to(torch.bfloat16).cuda()
    rng = np.random.default_rng(7)
    r = torch.from_numpy((3 * rng.standard_normal((2, 28, 28, 64))).astype(np.float32)).to(torch.bfloat16).cuda()
    y = conv(x, relu="relu6", algo=ox.ONEXN_ALGO_TC, residual=r)
    torch.cuda.synchronize()
    mask, _ = oracle.prune(W, 16, 0.5, ox.ONEXN_GRAN_TAP)
    ref, absacc = oracle.conv_masked(x.float().cpu().numpy(), oracle.round_bf16(W), mask, b, 16, (1, 1), (1, 1),
                                     relu="relu6", residual=r.float().cpu().numpy(), want_abs=True)
    e = norm_err(y.float().cpu().numpy().reshape(-1, 64).astype(np.float64), ref.reshape(-1, 64),
                 absacc.reshape(-1, 64))
    assert e <= TOL_BF16_ROUNDED
    assert (ref == 6).any() and (ref == 0).any()     # both clamps exercised


def test_halo_empty_batch_and_output_untouched_outside():
    """A batch of zero images launches nothing; y's bytes past the layer's
    output are never written (the per-row stores stay inside y)."""
    layer = L("halo_guard", 1, 28, 28, 64, 64, 3, 3, 1, 1, 1, N=16, rate=0.5, dtype="bf16", seed=2)
    W = wl.weights(layer).numpy()
    conv = PrunedConv2d(W, 16, 0.5, padding=1, dtype="bf16")
    x0 = torch.empty((0, 28, 28, 64), dtype=torch.bfloat16, device="cuda")
    assert conv(x0, algo=ox.ONEXN_ALGO_TC).shape == (0, 28, 28, 64)
    x = wl.activations(layer).to(torch.bfloat16).cuda()
    big = torch.full((2 * 28 * 28 * 64,), 7.0, dtype=torch.bfloat16, device="cuda")
    y = big[: 28 * 28 * 64].view(1, 28, 28, 64)
    conv(x, y, algo=ox.ONEXN_ALGO_TC)
    torch.cuda.synchronize()
    assert torch.all(big[28 * 28 * 64:] == 7.0)


@pytest.mark.parametrize("B,C_in,C_out", [(32, 128, 128), (64, 64, 256)], ids=["bn128", "bn256"])
def test_halo_wide_column_tiles_sampled(B, C_in, C_out):
    """Enough pixel tiles that the im2col GEMM takes 128- and 256-column
    tiles, wider than the halo form's weights allow, so the layer keeps the
    im2col form; checked on 3000 seeded output pixels over every image."""
    layer = L("halo_wide", B, 28, 28, C_in, C_out, 3, 3, 1, 1, 1, N=16, rate=0.5, dtype="bf16", seed=B)
    pix = np.sort(np.random.default_rng(B).choice(layer.pixels, 3000, replace=False))
    y, yr, a, _ = run_layer(layer, relu=True, algo=ox.ONEXN_ALGO_TC, pixels=pix)
    assert norm_err(y, yr, a) <= TOL_BF16_ROUNDED
