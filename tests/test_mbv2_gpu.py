"""GPU parity of MobileNet-V2's inverted-residual block on the onexn kernels
(the batch-1 latency workload): the dense depthwise convolution, ReLU6, the
residual add fused into the pruned convolution's epilogue, and whole blocks
checked stage by stage against the fp64 oracle (each stage fed the GPU's
own input to that stage), plus CUDA-graph capture of a block.

Tolerances as elsewhere: fp32 1e-5, bf16 4e-3 (2^-8 output rounding),
normalised by sum |w x| + |b| (+ |residual|)."""
import numpy as np
import pytest
import torch

import oracle
from paper_2105_14713_gb300 import onexn as ox
from paper_2105_14713_gb300 import workloads as wl
from paper_2105_14713_gb300.layer import DepthwiseConv2d, InvertedResidual, PrunedConv2d

pytestmark = pytest.mark.gpu

TOL = {"f32": 1e-5, "bf16": 4e-3}


def _dev(x, dtype):
    return (x if dtype == "f32" else x.to(torch.bfloat16)).cuda()


def _host32(t):
    return t.float().cpu().numpy()


def _w(W, dtype):
    """Conv weights as the GPU holds them (bf16-rounded on the bf16 path)."""
    return W if dtype == "f32" else oracle.round_bf16(W)


def _mask(conv, W, N, rate):
    """The oracle's block mask (Sec. 3.2), checked equal to the layer's."""
    m, _ = oracle.prune(W, N, rate)
    np.testing.assert_array_equal(m, conv.mask)
    return m


def _err(y, ref, absacc):
    return float(np.max(np.abs(y.astype(np.float64) - ref) / (absacc + 1e-30)))


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("stride,relu", [(1, "relu6"), (2, "relu6"), (1, False), (2, True)])
def test_depthwise_conv(dtype, stride, relu):
    rng = np.random.default_rng(stride * 10 + (relu == "relu6"))
    C = 48
    x = torch.from_numpy((2 * rng.standard_normal((3, 15, 13, C))).astype(np.float32))
    W = rng.standard_normal((C, 3, 3)).astype(np.float32)
    b = rng.standard_normal(C).astype(np.float32)
    dw = DepthwiseConv2d(W, bias=b, stride=stride, padding=1, dtype=dtype)
    xd = _dev(x, dtype)
    y = _host32(dw(xd, relu=relu))
    xs = _host32(xd)
    ref = oracle.dwconv(xs, W, b, stride=(stride, stride), pad=(1, 1), relu=relu)
    absacc = oracle.dwconv(np.abs(xs), np.abs(W), np.abs(b), stride=(stride, stride), pad=(1, 1))
    assert _err(y, ref, absacc) <= TOL[dtype]


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("k,stride,pad,dil", [(5, 1, 4, 2), (1, 2, 0, 1), (5, 2, 2, 1)])
def test_depthwise_conv_other_kernel_sizes(dtype, k, stride, pad, dil):
    """The tap-by-tap form (any KH x KW), beside the unrolled 3x3 one."""
    rng = np.random.default_rng(k * 100 + stride * 10 + dil)
    C = 24 if dtype == "f32" else 32
    x = torch.from_numpy(rng.standard_normal((2, 11, 9, C)).astype(np.float32))
    W = rng.standard_normal((C, k, k)).astype(np.float32)
    b = rng.standard_normal(C).astype(np.float32)
    dw = DepthwiseConv2d(W, bias=b, stride=stride, padding=pad, dilation=dil, dtype=dtype)
    xd = _dev(x, dtype)
    y = _host32(dw(xd, relu=True))
    xs = _host32(xd)
    g = dict(stride=(stride, stride), pad=(pad, pad), dil=(dil, dil))
    ref = oracle.dwconv(xs, W, b, relu=True, **g)
    absacc = oracle.dwconv(np.abs(xs), np.abs(W), np.abs(b), **g)
    assert y.shape == ref.shape
    assert _err(y, ref, absacc) <= TOL[dtype]


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("algo", ["fma", "tc"])
@pytest.mark.parametrize("aliased", [False, True])
def test_conv_with_residual_and_relu6(dtype, algo, aliased):
    layer = wl.ConvLayer("res", 3, 14, 14, 64, 64, 1, 1, 1, 0, 1, N=4, rate=0.5, dtype=dtype, seed=5)
    W, b = wl.weights(layer).numpy(), wl.bias(layer).numpy()
    conv = PrunedConv2d(W, 4, 0.5, bias=b, dtype=dtype)
    xd = _dev(wl.activations(layer), dtype)
    rng = np.random.default_rng(3)
    r = _dev(torch.from_numpy((3 * rng.standard_normal((3, 14, 14, 64))).astype(np.float32)), dtype)
    r_host = _host32(r)
    y = r.clone() if aliased else torch.empty_like(r)
    conv(xd, y, relu="relu6", algo=ox.ALGO_BY_NAME[algo], residual=y if aliased else r)
    ref, absacc = oracle.conv_masked(_host32(xd), _w(W, dtype), _mask(conv, W, 4, 0.5), b, 4, relu="relu6",
                                     residual=r_host,
                                     want_abs=True)
    assert _err(_host32(y), ref, absacc) <= TOL[dtype]
    assert (ref == 6).any() and (ref == 0).any()     # both clamps exercised


def _block(blk, fuse_dw="auto"):
    we, be, wd, bd, wp, bp = wl.block_weights(blk)
    return InvertedResidual(we, be, wd, bd, wp, bp, stride=blk.stride, N=blk.N, rate=blk.rate, dtype=blk.dtype,
                            fuse_dw=fuse_dw)


BLOCKS = [  # name, hw, c_in, hidden, c_out, stride  (MobileNet-V2 shapes at a smaller image)
    ("t1_no_expand", 20, 32, 32, 16, 1),
    ("expand_residual", 14, 24, 144, 24, 1),
    ("expand_stride2", 14, 24, 144, 32, 2),
    ("wide_residual", 7, 160, 960, 160, 1),
]


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("spec", BLOCKS, ids=[b[0] for b in BLOCKS])
def test_inverted_residual_block_stage_by_stage(dtype, spec):
    name, hw, c_in, hidden, c_out, stride = spec
    blk = wl.MBv2Block(name, 2, hw, c_in, hidden, c_out, stride, N=4, rate=0.5, dtype=dtype, seed=len(name))
    block = _block(blk, fuse_dw=False)          # the depthwise output is read back below
    x = _dev(wl.block_input(blk), dtype)
    out = block(x)
    torch.cuda.synchronize()
    h, d, _ = block.buffers(x.shape, x.dtype, x.device)
    xs = _host32(x)
    if block.expand is not None:
        ref, a = oracle.conv_masked(xs, _w(block.w_expand, dtype), _mask(block.expand, block.w_expand, 4, 0.5),
                                    block.b_expand, 4, relu="relu6",
                                    want_abs=True)
        assert _err(_host32(h), ref, a) <= TOL[dtype], "expand"
        hs = _host32(h)
    else:
        hs = xs
    ref = oracle.dwconv(hs, block.w_dw, block.b_dw, stride=(stride, stride), pad=(1, 1), relu="relu6")
    a = oracle.dwconv(np.abs(hs), np.abs(block.w_dw), np.abs(block.b_dw), stride=(stride, stride), pad=(1, 1))
    assert _err(_host32(d), ref, a) <= TOL[dtype], "depthwise"
    ref, a = oracle.conv_masked(_host32(d), _w(block.w_project, dtype),
                                _mask(block.project, block.w_project, 4, 0.5), block.b_project, 4,
                                residual=xs if block.residual else None, want_abs=True)
    assert block.residual == (stride == 1 and c_in == c_out)
    assert _err(_host32(out), ref, a) <= TOL[dtype], "project"


FUSED = BLOCKS + [("wide_s2_ragged", 11, 40, 240, 48, 2),      # 240 = 7.5 chunks of 32 channels
                  ("one_image_row", 1, 24, 72, 24, 1)]


@pytest.mark.parametrize("spec", FUSED, ids=[b[0] for b in FUSED])
def test_depthwise_fused_into_the_projection(spec):
    """onexn_dwproj_fwd (fp32): the projection's GEMM computes relu6(dw(h))
    itself; against the oracle's depthwise then projection (+ residual) on
    the GPU's own expand output, and against the unfused kernels."""
    name, hw, c_in, hidden, c_out, stride = spec
    blk = wl.MBv2Block(name, 2, hw, c_in, hidden, c_out, stride, N=4, rate=0.5, dtype="f32", seed=len(name) + 1)
    fused, plain = _block(blk, fuse_dw=True), _block(blk, fuse_dw=False)
    x = wl.block_input(blk).cuda()
    out = fused(x).clone()
    ref_gpu = plain(x).clone()
    torch.cuda.synchronize()
    h = plain.buffers(x.shape, x.dtype, x.device)[0]
    hs = _host32(h) if fused.expand is not None else _host32(x)
    d = oracle.dwconv(hs, fused.w_dw, fused.b_dw, stride=(stride, stride), pad=(1, 1), relu="relu6")
    xs = _host32(x)
    ref, a = oracle.conv_masked(d.astype(np.float32), fused.w_project,
                                _mask(fused.project, fused.w_project, 4, 0.5), fused.b_project, 4,
                                residual=xs if fused.residual else None, want_abs=True)
    assert _err(_host32(out), ref, a) <= 1e-5
    assert _err(_host32(out), _host32(ref_gpu).astype(np.float64), a) <= 1e-5
    # a second call runs on the resident decoded weights
    out2 = fused(x)
    torch.cuda.synchronize()
    assert torch.equal(out2, out)


def test_dwproj_rejects_bf16_and_bad_depthwise_geometry():
    from paper_2105_14713_gb300.layer import PrunedConv2d
    blk = wl.MBv2Block("rej", 1, 8, 32, 64, 32, 1, N=4, rate=0.5, dtype="bf16", seed=1)
    b16 = _block(blk)
    assert not b16.fused((1, 8, 8, 32))
    W = np.random.default_rng(0).standard_normal((32, 64, 1, 1)).astype(np.float32)
    conv = PrunedConv2d(W, 4, 0.5)
    h = torch.zeros((1, 8, 8, 64), device="cuda")
    wt = torch.zeros((9, 64), device="cuda")
    with pytest.raises(ox.OnexnError):
        conv.forward_dwproj(h, wt, None, 3)        # stride 3
    with pytest.raises((ValueError, ox.OnexnError)):
        conv.forward_dwproj(h.to(torch.bfloat16), wt, None, 1)


def test_block_end_to_end_fp32_and_cuda_graph_replay():
    blk = wl.MBv2Block("e2e", 1, 28, 32, 192, 32, 1, N=4, rate=0.5, dtype="f32", seed=3)
    block = _block(blk)
    x = wl.block_input(blk).cuda()
    y_eager = block(x).clone()
    torch.cuda.synchronize()
    # each stage against the oracle fed the GPU's own input to that stage, at
    # the fp32 tolerance (an fp64 chain from x alone would add each stage's
    # rounding, propagated through the later stages, to the comparison)
    h, d, _ = block.buffers(x.shape, x.dtype, x.device)
    xs = x.cpu().numpy()
    ref, a = oracle.conv_masked(xs, block.w_expand, _mask(block.expand, block.w_expand, 4, 0.5), block.b_expand, 4,
                                relu="relu6", want_abs=True)
    assert _err(_host32(h), ref, a) <= 1e-5, "expand"
    hs = _host32(h)
    ref = oracle.dwconv(hs, block.w_dw, block.b_dw, pad=(1, 1), relu="relu6")
    if block.fused(x.shape):
        # the projection computed the depthwise itself (fp32): its input is
        # the oracle's depthwise of the GPU's expand output
        ds = ref.astype(np.float32)
    else:
        a = oracle.dwconv(np.abs(hs), np.abs(block.w_dw), np.abs(block.b_dw), pad=(1, 1))
        assert _err(_host32(d), ref, a) <= 1e-5, "depthwise"
        ds = _host32(d)
    ref, a = oracle.conv_masked(ds, block.w_project, _mask(block.project, block.w_project, 4, 0.5),
                                block.b_project, 4, residual=xs, want_abs=True)
    assert _err(y_eager.cpu().numpy(), ref, a) <= 1e-5, "project + residual"
    # the same block captured into a CUDA graph (no allocation after the first call)
    s = torch.cuda.Stream()
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        y_graph = block(x, stream=s)
    for _ in range(3):
        g.replay()
    torch.cuda.synchronize()
    assert torch.equal(y_graph, y_eager)
