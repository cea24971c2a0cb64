"""GPU parity of onexn_conv_fwd against the fp64 oracle (Eq. 6 / Eq. 7).

Small cases span several 128-pixel tiles, several column tiles and a ragged
tail; every geometry feature (stride, padding, dilation, non-square
kernels, partial channel chunks) and every block width class is covered, for
each kernel family that can run the case.  Tolerances: fp32 1e-5 and bf16
1e-2 (fp32 master inputs) / 4e-3 = 2^-8 output rounding (bf16-rounded inputs), normalised by
sum |w x| + |b|."""
import numpy as np
import pytest
import torch

from paper_2105_14713_gb300 import onexn as ox
from paper_2105_14713_gb300 import workloads as wl
from tests.gpu_util import norm_err, oracle_ref, run_layer, to_device_input, tol

pytestmark = pytest.mark.gpu

L = wl.ConvLayer

GEOMS = [
    # name, B, H, W, C_in, C_out, KH, KW, stride, pad, dil
    ("1x1", 3, 13, 11, 64, 64, 1, 1, 1, 0, 1),
    ("1x1_c24", 2, 17, 9, 24, 48, 1, 1, 1, 0, 1),
    ("1x1_s2", 2, 15, 15, 40, 32, 1, 1, 2, 0, 1),
    ("3x3_p1", 2, 14, 14, 64, 64, 3, 3, 1, 1, 1),
    ("3x3_s2", 3, 15, 13, 32, 64, 3, 3, 2, 1, 1),
    ("3x3_d2", 2, 16, 16, 48, 32, 3, 3, 1, 2, 2),
    ("1x3", 2, 9, 20, 16, 32, 1, 3, 1, 1, 1),
    ("5x5_p0", 1, 20, 20, 8, 32, 5, 5, 1, 0, 1),
]

ALGOS = ox.ALGO_BY_NAME


def _algos_for(dtype, N, C_in=64, C_out=64):
    """Every family that can run this case (FMA always; the tensor-core
    families if they accept it), plus AUTO."""
    out = ["auto", "fma"]
    probe = ox.make_desc(1, 8, 8, C_in, C_out, 1, 1)
    dt = ox.ONEXN_BF16 if dtype == "bf16" else ox.ONEXN_F32
    for name in ("mma", "tc"):
        try:
            ox.onexn_conv_algo(probe, N, 1, dt, ALGOS[name], 1 << 40)
            out.append(name)
        except ox.OnexnError:
            pass
    return out


@pytest.mark.parametrize("geom", GEOMS, ids=[g[0] for g in GEOMS])
@pytest.mark.parametrize("N", [1, 2, 4, 8, 16, 32])
@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_geometry_and_block_width(geom, N, dtype):
    name, B, H, W, Ci, Co, KH, KW, s, p, d = geom
    if Co % N:
        pytest.skip("N must divide C_out")
    layer = L(name, B, H, W, Ci, Co, KH, KW, s, p, d, N=N, rate=0.5, dtype=dtype, seed=N)
    for algo in _algos_for(dtype, N, Ci, Co):
        y, yr, a, conv = run_layer(layer, relu=(N % 2 == 0), algo=ALGOS[algo])
        e = norm_err(y, yr, a)
        assert e <= tol(layer), f"{algo}: err {e:.3e}"


@pytest.mark.parametrize("rate", [0.0, 0.3, 0.7, 0.9, 1.0])
@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_rates(rate, dtype):
    layer = L("rates", 2, 12, 12, 64, 128, 3, 3, 1, 1, 1, N=8, rate=rate, dtype=dtype, seed=3)
    for algo in _algos_for(dtype, 8, 64, 128):
        y, yr, a, _ = run_layer(layer, relu=True, algo=ALGOS[algo])
        assert norm_err(y, yr, a) <= tol(layer), algo


@pytest.mark.parametrize("N", [3, 5, 6, 12, 24, 64, 128])
def test_odd_and_wide_blocks(N):
    Co = 120 if N in (3, 5, 6, 12, 24) else N * 2
    layer = L("oddN", 2, 10, 10, 32, Co, 3, 3, 1, 1, 1, N=N, rate=0.4, dtype="f32", seed=N)
    y, yr, a, _ = run_layer(layer, algo=ox.ONEXN_ALGO_FMA)
    assert norm_err(y, yr, a) <= 1e-5


def test_odd_output_channels_scalar_stores():
    layer = L("co6", 2, 9, 9, 16, 6, 1, 1, N=2, rate=0.5, dtype="f32", seed=1)
    y, yr, a, _ = run_layer(layer)
    assert norm_err(y, yr, a) <= 1e-5


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_dense_path_rate0_N_equals_cout(dtype):
    layer = L("dense", 2, 14, 14, 64, 128, 3, 3, 1, 1, 1, N=128, rate=0.0, dtype=dtype, seed=5)
    for algo in _algos_for(dtype, 128, 64, 128):
        y, yr, a, conv = run_layer(layer, algo=ALGOS[algo])
        assert conv.t == 576
        assert norm_err(y, yr, a) <= tol(layer), algo


@pytest.mark.parametrize("C_out,N", [(64, 8), (128, 16), (256, 8), (384, 32), (520, 8), (48, 8)])
def test_tc_column_tiles(C_out, N):
    """The tcgen05 family over every column-tile width (64/128/256) and a
    ragged last column tile."""
    layer = L("tc_cols", 3, 11, 13, 72, C_out, 3, 3, 1, 1, 1, N=N, rate=0.5, dtype="bf16", seed=C_out)
    y, yr, a, conv = run_layer(layer, relu=True, algo=ox.ONEXN_ALGO_TC)
    assert conv.algo((3, 11, 13, 72), ox.ONEXN_ALGO_TC) == "tc"
    assert norm_err(y, yr, a) <= tol(layer)


def test_auto_picks_tc_with_workspace_and_ffma_for_bias_only():
    layer = L("auto", 4, 32, 32, 64, 64, 1, 1, N=8, rate=0.5, dtype="bf16")
    from paper_2105_14713_gb300.layer import PrunedConv2d
    for dt in ("bf16", "f32"):
        conv = PrunedConv2d(wl.weights(layer).numpy(), 8, 0.5, dtype=dt)
        assert conv.algo((4, 32, 32, 64)) == "tc"
        empty = PrunedConv2d(wl.weights(layer).numpy(), 8, 1.0, dtype=dt)
        assert empty.t == 0 and empty.algo((4, 32, 32, 64)) == "fma"


def test_device_status_clean_after_runs():
    assert ox.onexn_device_status(clear=True) == ox.ONEXN_OK


def test_bf16_against_fp32_master_inputs():
    layer = L("master", 2, 14, 14, 64, 64, 3, 3, 1, 1, 1, N=8, rate=0.5, dtype="bf16", seed=6)
    y, yr, a, _ = run_layer(layer, relu=True, master=True)
    assert norm_err(y, yr, a) <= 1e-2


def test_kernel_granularity_mode():
    """The paper's own block (N whole KH x KW kernels of one channel)."""
    layer = L("gran", 2, 12, 12, 32, 64, 3, 3, 1, 1, 1, N=4, rate=0.5, dtype="f32", seed=7)
    y, yr, a, conv = run_layer(layer, gran=ox.ONEXN_GRAN_KERNEL)
    assert conv.t == conv.kept * 9
    assert norm_err(y, yr, a) <= 1e-5


def test_empty_batch_and_no_bias():
    layer = L("empty", 0, 8, 8, 16, 16, 3, 3, 1, 1, 1, N=4, rate=0.5, dtype="f32")
    W = wl.weights(layer).numpy()
    from paper_2105_14713_gb300.layer import PrunedConv2d
    conv = PrunedConv2d(W, 4, 0.5, padding=1)
    x = torch.zeros((0, 8, 8, 16), device="cuda")
    y = conv(x)
    assert tuple(y.shape) == (0, 8, 8, 16)
    layer2 = layer.with_(B=1)
    y, yr, a, _ = run_layer(layer2, with_bias=False)
    assert norm_err(y, yr, a) <= 1e-5


def test_streams_and_repeat_calls_are_deterministic():
    layer = L("det", 4, 16, 16, 64, 64, 3, 3, 1, 1, 1, N=8, rate=0.5, dtype="f32", seed=8)
    from paper_2105_14713_gb300.layer import PrunedConv2d
    conv = PrunedConv2d(wl.weights(layer).numpy(), 8, 0.5, padding=1, bias=wl.bias(layer).numpy())
    x = wl.activations(layer).cuda()
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        y1 = conv(x)
        y2 = conv(x)
    s.synchronize()
    assert torch.equal(y1, y2)


# tile counts around whole rounds of 152 CTAs: one tile past two rounds (a
# one-tile stream-K round after whole tiles), exactly two rounds (no split),
# and a bf16 3x3 with 36 chunks per tile and a ragged last round
SK_CASES = [
    L("sk153", 1, 139, 140, 512, 64, 1, 1, 1, 0, 1, N=8, rate=0.5, dtype="f32", seed=41),     # 153 tiles
    L("sk304", 1, 152, 256, 512, 64, 1, 1, 1, 0, 1, N=8, rate=0.5, dtype="f32", seed=42),     # 304 tiles
    L("sk_b", 2, 60, 60, 256, 128, 3, 3, 1, 1, 1, N=8, rate=0.5, dtype="bf16", seed=43),      # 57 tiles
    L("sk_b2", 10, 46, 46, 256, 128, 3, 3, 1, 1, 1, N=16, rate=0.7, dtype="bf16", seed=44),   # 166 tiles
]


@pytest.mark.parametrize("layer", SK_CASES, ids=[c.name for c in SK_CASES])
def test_stream_k_around_whole_rounds(layer):
    """Sampled parity (the first, last and random pixels of every tile
    region) where the last round of tiles is split across CTAs."""
    P = layer.pixels
    must = [0, P - 1] + [min(P - 1, 128 * k + r) for k in range(0, -(-P // 128), 16) for r in (0, 127)]
    pix = wl.sample_pixels(P, 1500, layer.seed, must=must)
    y, yr, a, conv = run_layer(layer, pixels=pix, algo=ox.ONEXN_ALGO_TC)
    assert norm_err(y, yr, a) <= tol(layer)


def test_decoded_weights_reused_across_calls():
    """After one tc call a layer passes ONEXN_DECODED and runs the GEMM
    alone; results stay bitwise equal, including the stream-K split tiles
    (8 pixel tiles < 152 SMs), whose flags the finisher resets for the next
    launch."""
    from paper_2105_14713_gb300.layer import PrunedConv2d
    for dt, seed in (("f32", 31), ("bf16", 32)):
        layer = L("decoded", 4, 16, 16, 64, 64, 3, 3, 1, 1, 1, N=8, rate=0.5, dtype=dt, seed=seed)
        W, b = wl.weights(layer).numpy(), wl.bias(layer).numpy()
        conv = PrunedConv2d(W, 8, 0.5, padding=1, bias=b, dtype=dt)
        fresh = PrunedConv2d(W, 8, 0.5, padding=1, bias=b, dtype=dt, reuse_decoded=False)
        x = to_device_input(wl.activations(layer), dt)
        assert conv.algo(x.shape) == "tc"
        ys = [conv(x).clone() for _ in range(3)]
        assert len(conv._decoded) == 1
        flags = [args[0][11] for args in conv._args.values()]
        assert flags and all(f & ox.ONEXN_DECODED for f in flags)
        y_ref = fresh(x)
        assert not fresh._decoded
        for y in ys:
            assert torch.equal(y, y_ref)
        yr, a = oracle_ref(layer, W, wl.activations(layer), b)
        yo = y_ref.float().cpu().numpy().reshape(-1, 64).astype(np.float64)
        assert norm_err(yo, yr, a) <= tol(layer)


# ------------------------------------------------ host-memory entry point

HOST_CASES = [
    # layer, forced algo
    (L("h3x3", 13, 14, 14, 64, 64, 3, 3, 1, 1, 1, N=8, rate=0.5, dtype="f32", seed=21), "auto"),
    (L("h3x3b", 13, 14, 14, 64, 64, 3, 3, 1, 1, 1, N=8, rate=0.5, dtype="bf16", seed=22), "auto"),
    (L("h1x1s2", 9, 15, 15, 32, 48, 1, 1, 2, 0, 1, N=4, rate=0.7, dtype="f32", seed=23), "fma"),
    (L("h1x1", 11, 28, 28, 96, 64, 1, 1, 1, 0, 1, N=16, rate=0.5, dtype="bf16", seed=24), "tc"),
    # 160 images of 200704 bytes: 4 chunks, so the first slot is reused
    (L("hbig", 160, 28, 28, 64, 64, 3, 3, 1, 1, 1, N=8, rate=0.5, dtype="f32", seed=25), "tc"),
    (L("hbigb", 330, 28, 28, 64, 64, 3, 3, 1, 1, 1, N=8, rate=0.5, dtype="bf16", seed=26), "auto"),
]


def _device_out_min_workspace(conv, x, flags):
    """onexn_conv_fwd with only the minimum workspace (the decoded weights
    for the tensor-core family: its GEMM then takes whole tiles only)."""
    B, H, W, _ = x.shape
    K = conv.KH * conv.KW * conv.C_in
    wmin = conv.C_out * K * (8 if conv.cdtype == ox.ONEXN_F32 else 2)
    wmin = -(-wmin // 256) * 256
    ws = torch.empty(wmin, dtype=torch.uint8, device="cuda")
    y = torch.empty(conv.out_shape(x.shape), dtype=x.dtype, device="cuda")
    ox.onexn_conv_fwd(conv.desc(B, H, W), conv.P, conv.I, conv.D, conv.N, conv.t, x, y, conv.bias,
                      conv.cdtype, flags, ws)
    return y


@pytest.mark.parametrize("case", HOST_CASES, ids=[c[0].name for c in HOST_CASES])
def test_host_entry_matches_device_entry(case):
    """onexn_conv_fwd_host (chunks of images copied in and out on internal
    streams) gives bit for bit the device entry's output when that runs whole
    tiles too (minimum workspace): every output pixel is computed by the same
    kernel in the same order, only grouped differently.  Against the device
    entry with its full workspace (split tiles summed from partial parts) the
    outputs agree to fp32 rounding."""
    layer, algo = case
    from paper_2105_14713_gb300.layer import PrunedConv2d
    conv = PrunedConv2d(wl.weights(layer).numpy(), layer.N, layer.rate, bias=wl.bias(layer).numpy(),
                        stride=layer.stride, padding=layer.pad, dilation=layer.dil, dtype=layer.dtype)
    x = wl.activations(layer)
    x = x if layer.dtype == "f32" else x.to(torch.bfloat16)
    flags = ox.ONEXN_RELU | ALGOS[algo]
    y_min = _device_out_min_workspace(conv, x.cuda(), flags).cpu()
    y_full = conv(x.cuda(), relu=True, algo=ALGOS[algo]).cpu()
    iv = torch.int16 if layer.dtype == "bf16" else torch.int32
    for pinned in (True, False):
        xh = x.pin_memory() if pinned else x.clone()
        y_host = conv.forward_host(xh, relu=True, algo=ALGOS[algo])
        assert torch.equal(y_host.view(iv), y_min.view(iv)), pinned
    # the fp32 parity tolerance on the output scale; bf16: a rounding flip
    scale = y_min.float().abs().max().item() + 1e-30
    tol_rel = 2.0 ** -7 if layer.dtype == "bf16" else 1e-5
    assert (y_full.float() - y_min.float()).abs().max().item() <= tol_rel * scale


def test_host_entry_overlapping_calls_on_two_streams():
    """Two layers enqueued back to back on different streams (the second's
    copies overlap the first's compute) both give the device entry's output
    (whole-tile form, as the host entry runs)."""
    from paper_2105_14713_gb300.layer import PrunedConv2d
    layers = [L("ov_a", 24, 28, 28, 64, 128, 3, 3, 1, 1, 1, N=8, rate=0.5, dtype="f32", seed=31),
              L("ov_b", 24, 28, 28, 64, 64, 3, 3, 1, 1, 1, N=4, rate=0.3, dtype="bf16", seed=32)]
    convs, xs, refs = [], [], []
    for layer in layers:
        conv = PrunedConv2d(wl.weights(layer).numpy(), layer.N, layer.rate, padding=1, dtype=layer.dtype)
        x = wl.activations(layer)
        x = (x if layer.dtype == "f32" else x.to(torch.bfloat16)).pin_memory()
        convs.append(conv)
        xs.append(x)
        refs.append(_device_out_min_workspace(conv, x.cuda(), 0).cpu())
    streams = [torch.cuda.Stream() for _ in layers]
    for _ in range(3):
        outs = [c.forward_host(x, stream=s, sync=False) for c, x, s in zip(convs, xs, streams)]
        torch.cuda.synchronize()
        for o, r in zip(outs, refs):
            assert torch.equal(o.float(), r.float())


def test_host_entry_empty_batch():
    from paper_2105_14713_gb300.layer import PrunedConv2d
    layer = L("hempty", 0, 8, 8, 16, 16, 3, 3, 1, 1, 1, N=4, rate=0.5, dtype="f32")
    conv = PrunedConv2d(wl.weights(layer).numpy(), 4, 0.5, padding=1)
    y = conv.forward_host(torch.zeros(0, 8, 8, 16).pin_memory())
    assert tuple(y.shape) == (0, 8, 8, 16)


# ------------------------------------------- fully connected layers as 1x1

@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("B", [1, 7, 256])
def test_fully_connected_layer_as_1x1_conv(dtype, B):
    """A fully connected layer (here MobileNet-V2's 1280 -> 1000 classifier)
    is a 1x1 convolution on a 1x1 image: x [B, 1, 1, 1280] -> y [B, 1, 1,
    1000].  Few pixel tiles, so the tensor-core GEMM splits the K loop of
    each output tile across CTAs (stream-K)."""
    layer = L("fc", B, 1, 1, 1280, 1000, 1, 1, 1, 0, 1, N=4, rate=0.5, dtype=dtype, seed=B)
    for algo in _algos_for(dtype, 4, 1280, 1000):
        y, yr, a, conv = run_layer(layer, relu=False, algo=ALGOS[algo])
        assert norm_err(y, yr, a) <= tol(layer), (algo, B)
