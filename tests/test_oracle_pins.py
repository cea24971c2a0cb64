"""Pins of the CPU oracle against things other than itself (no GPU).

Each test checks the oracle against what the paper and the mathematics fix:
a hand-worked example (tests/golden), exact rational arithmetic, a library
routine the special case reduces to (numpy sort, torch conv2d in fp64,
torch's bfloat16 conversion), invariants (rearrangement, BSR round trip)
or brute force on tiny inputs.
"""
import json
import os
from fractions import Fraction

import numpy as np
import pytest
import torch
import torch.nn.functional as F

import oracle

GOLD = os.path.join(os.path.dirname(__file__), "golden")


def _int_weights(shape, seed, lo=-3, hi=4):
    """Small-integer weights: every l1 sum is exact in fp64, and ties are common."""
    rng = np.random.default_rng(seed)
    return rng.integers(lo, hi, size=shape).astype(np.float32)


def _torch_conv_nhwc(x, W, stride, pad, dil, bias=None):
    xt = torch.from_numpy(np.ascontiguousarray(x, np.float64)).permute(0, 3, 1, 2)
    wt = torch.from_numpy(np.ascontiguousarray(W, np.float64))
    bt = None if bias is None else torch.from_numpy(np.asarray(bias, np.float64))
    y = F.conv2d(xt, wt, bt, stride=stride, padding=pad, dilation=dil)
    return y.permute(0, 2, 3, 1).numpy()


def _expand_mask(mask, C_out, C_in, KH, KW, N):
    """[G, KH*KW*C_in] tap-major mask -> OIHW 0/1 array."""
    G = C_out // N
    m = mask.reshape(G, KH, KW, C_in).transpose(0, 3, 1, 2)        # G, C, KH, KW
    return np.repeat(m, N, axis=0).astype(np.float32)


# --------------------------------------------------------------------------
# Hand-worked example (Sec. 3.2-3.4)
# --------------------------------------------------------------------------

def test_worked_example_golden():
    g = json.load(open(os.path.join(GOLD, "worked_example_1x1.json")))
    W = np.asarray(g["W_oc"], np.float32)[:, :, None, None]
    N = g["N"]
    np.testing.assert_array_equal(oracle.block_scores(W, N), np.asarray(g["block_scores_gk"]))
    mask, kept = oracle.prune(W, N, 0.5)
    assert kept == g["rate_0.5"]["kept"]
    np.testing.assert_array_equal(mask, np.asarray(g["rate_0.5"]["mask_gk"]))
    P, I, D = oracle.pack(W, mask, N)
    np.testing.assert_array_equal(P, g["rate_0.5"]["P"])
    np.testing.assert_array_equal(I, g["rate_0.5"]["I"])
    np.testing.assert_array_equal(D, np.asarray(g["rate_0.5"]["D"], np.float32))
    m3, k3 = oracle.prune(W, N, 0.333333)
    assert k3 == g["rate_0.333333"]["kept"]
    np.testing.assert_array_equal(m3, np.asarray(g["rate_0.333333"]["mask_gk"]))

    cv = g["conv"]
    x = np.asarray(cv["x_nhwc"], np.float32)
    b = np.asarray(cv["bias"], np.float32)
    np.testing.assert_array_equal(oracle.conv_masked(x, W, mask, None, N),
                                  cv["y_rate_0.5_no_bias"])
    np.testing.assert_array_equal(oracle.conv_masked(x, W, mask, b, N), cv["y_rate_0.5_bias"])
    np.testing.assert_array_equal(oracle.conv_masked(x, W, mask, b, N, relu=True),
                                  cv["y_rate_0.5_bias_relu"])
    np.testing.assert_array_equal(oracle.conv_bsr(x, P, I, D, 4, 1, 1, N, bias=b, relu=True),
                                  cv["y_rate_0.5_bias_relu"])
    _, _, perm = oracle.rearrange(W)
    np.testing.assert_array_equal(perm, g["rearrange"]["perm"])


# --------------------------------------------------------------------------
# Keep count (Eq. 1 constraint; reading C3) -- exact rational arithmetic
# --------------------------------------------------------------------------

@pytest.mark.parametrize("total", [1, 2, 5, 7, 16, 512, 9216, 147456, 2359296, 4718592])
@pytest.mark.parametrize("rate", [0.0, 0.1, 0.25, 0.3, 1 / 3, 0.5, 0.7, 0.9, 0.999999, 1.0])
def test_keep_count_exact(total, rate):
    r = Fraction(round(rate * 10**6), 10**6)
    want = int((total * (1 - r) + Fraction(1, 2)) // 1)      # round half up
    assert oracle.keep_count(total, rate) == want


def test_keep_count_half_rounds_up():
    assert oracle.keep_count(5, 0.5) == 3
    assert oracle.keep_count(3, 0.5) == 2
    assert oracle.keep_count(1, 0.5) == 1


# --------------------------------------------------------------------------
# Block scores and the mask (Eq. 4, solution after Eq. 5)
# --------------------------------------------------------------------------

def _numpy_scores(W, N, gran):
    C_out, C_in, KH, KW = W.shape
    a = np.abs(W.astype(np.float64)).reshape(C_out // N, N, C_in, KH, KW)
    if gran == oracle.GRAN_TAP:
        s = a.sum(axis=1)                                     # G, C, KH, KW
        return s.transpose(0, 2, 3, 1).reshape(C_out // N, -1)  # tap-major
    return a.sum(axis=(1, 3, 4))                               # G, C


def _numpy_topk_mask(scores, keep):
    G, nb = scores.shape
    flat = scores.reshape(-1)
    idx = np.arange(flat.size)
    order = np.lexsort((idx, -flat))        # score desc, then block index asc
    m = np.zeros(flat.size, np.uint8)
    m[order[:keep]] = 1
    return m.reshape(G, nb)


@pytest.mark.parametrize("shape,N", [((8, 6, 3, 3), 4), ((8, 6, 3, 3), 2), ((16, 5, 1, 3), 8),
                                     ((12, 7, 2, 2), 3), ((64, 64, 1, 1), 4)])
@pytest.mark.parametrize("gran", [oracle.GRAN_TAP, oracle.GRAN_KERNEL])
@pytest.mark.parametrize("rate", [0.0, 0.3, 0.5, 0.9, 1.0])
def test_prune_matches_exact_topk(shape, N, gran, rate):
    W = _int_weights(shape, seed=sum(shape) + N)
    C_out, C_in, KH, KW = shape
    sc = oracle.block_scores(W, N, gran)
    np.testing.assert_array_equal(sc, _numpy_scores(W, N, gran))   # exact: integer sums
    mask, kept = oracle.prune(W, N, rate, gran)
    assert kept == oracle.keep_count(sc.size, rate)
    want = _numpy_topk_mask(sc, kept)
    if gran == oracle.GRAN_KERNEL:
        want = np.tile(want[:, None, :], (1, KH * KW, 1)).reshape(C_out // N, -1)
    np.testing.assert_array_equal(mask, want)
    assert int(mask.sum()) == kept * (KH * KW if gran == oracle.GRAN_KERNEL else 1)


def test_prune_threshold_property_random():
    """The kept set maximises the summed l1 under the count: every kept block
    scores at least as much as every pruned block (Eq. 5 objective)."""
    rng = np.random.default_rng(3)
    W = rng.standard_normal((32, 16, 3, 3)).astype(np.float32)
    sc = oracle.block_scores(W, 4)
    mask, kept = oracle.prune(W, 4, 0.6)
    assert sc[mask == 1].min() >= sc[mask == 0].max()
    assert kept == (mask == 1).sum()
    np.testing.assert_allclose(sc, _numpy_scores(W, 4, oracle.GRAN_TAP), rtol=1e-14)


def test_n1_pointwise_is_weight_pruning():
    """N=1 with h=w=1 reduces 1xN pruning to weight pruning (Eq. 2)."""
    rng = np.random.default_rng(5)
    W = rng.standard_normal((24, 40, 1, 1)).astype(np.float32)
    for rate in (0.2, 0.5, 0.75):
        mask, kept = oracle.prune(W, 1, rate)
        a = np.abs(W[:, :, 0, 0]).astype(np.float64).reshape(-1)   # [o][c] = block (g=o, k=c)
        order = np.lexsort((np.arange(a.size), -a))
        want = np.zeros(a.size, np.uint8)
        want[order[:kept]] = 1
        np.testing.assert_array_equal(mask.reshape(-1), want)


def test_n_equals_cout_kernel_mode_is_input_channel_pruning():
    """N = n: one col-group holds every filter, so a block is a whole input
    channel and the mask prunes input channels by their total l1 (reading C9)."""
    W = _int_weights((16, 10, 3, 3), seed=11)
    mask, kept = oracle.prune(W, 16, 0.4, oracle.GRAN_KERNEL)
    ch = np.abs(W.astype(np.float64)).sum(axis=(0, 2, 3))
    order = np.lexsort((np.arange(10), -ch))
    keep_c = np.zeros(10, np.uint8)
    keep_c[order[:kept]] = 1
    np.testing.assert_array_equal(mask.reshape(1, 9, 10), np.broadcast_to(keep_c, (1, 9, 10)))


def test_prune_rejects_bad_args():
    W = np.ones((6, 2, 1, 1), np.float32)
    with pytest.raises(ValueError):
        oracle.prune(W, 4, 0.5)
    with pytest.raises(ValueError):
        oracle.prune(W, 3, 1.5)


# --------------------------------------------------------------------------
# Filter rearrangement (Sec. 3.3)
# --------------------------------------------------------------------------

def test_rearrange_order_and_permutation():
    W = _int_weights((12, 5, 3, 3), seed=21)
    Wn = _int_weights((7, 12, 1, 1), seed=22)
    W2, Wn2, perm = oracle.rearrange(W, Wn)
    l1 = np.abs(W.astype(np.float64)).sum(axis=(1, 2, 3))
    want = np.lexsort((np.arange(12), -l1))     # decreasing, stable
    np.testing.assert_array_equal(perm, want)
    np.testing.assert_array_equal(W2, W[perm])
    np.testing.assert_array_equal(Wn2, Wn[:, perm])
    assert np.all(np.diff(np.abs(W2.astype(np.float64)).sum(axis=(1, 2, 3))) <= 0)


@pytest.mark.parametrize("k2", [1, 3])
def test_rearrange_preserves_two_layer_composition(k2):
    """conv -> bias -> ReLU -> conv is unchanged when layer l's outputs and
    layer l+1's inputs are permuted together (Sec. 3.3)."""
    rng = np.random.default_rng(31 + k2)
    W1 = rng.standard_normal((16, 8, 3, 3)).astype(np.float32)
    b1 = rng.standard_normal(16).astype(np.float32)
    W2 = rng.standard_normal((10, 16, k2, k2)).astype(np.float32)
    x = rng.standard_normal((2, 9, 9, 8)).astype(np.float32)
    p = k2 // 2
    ref = _torch_conv_nhwc(np.maximum(_torch_conv_nhwc(x, W1, 1, 1, 1, b1), 0), W2, 1, p, 1)
    W1r, W2r, perm = oracle.rearrange(W1, W2)
    got = _torch_conv_nhwc(np.maximum(_torch_conv_nhwc(x, W1r, 1, 1, 1, b1[perm]), 0),
                           W2r, 1, p, 1)
    np.testing.assert_allclose(got, ref, rtol=1e-12, atol=1e-12)


def test_rearrange_without_next_layer():
    rng = np.random.default_rng(41)
    W = rng.standard_normal((9, 4, 1, 1)).astype(np.float32)
    W2, none, perm = oracle.rearrange(W)
    assert none is None
    np.testing.assert_array_equal(np.sort(perm), np.arange(9))
    np.testing.assert_array_equal(W2, W[perm])


# --------------------------------------------------------------------------
# BSR encoding (Sec. 3.4)
# --------------------------------------------------------------------------

@pytest.mark.parametrize("shape,N,rate", [((8, 6, 3, 3), 4, 0.5), ((8, 6, 3, 3), 2, 0.7),
                                          ((32, 16, 1, 1), 8, 0.0), ((32, 16, 1, 1), 8, 1.0),
                                          ((20, 12, 1, 3), 5, 0.45)])
def test_pack_structure_and_roundtrip(shape, N, rate):
    rng = np.random.default_rng(sum(shape))
    W = rng.standard_normal(shape).astype(np.float32)
    C_out, C_in, KH, KW = shape
    G, K = C_out // N, KH * KW * C_in
    mask, kept = oracle.prune(W, N, rate)
    P, I, D = oracle.pack(W, mask, N)
    t = int(mask.sum())
    assert P[0] == 0 and P[G] == t and len(I) == t and D.shape == (t, N)
    assert np.all(np.diff(P) >= 0)
    for g in range(G):
        seg = I[P[g]:P[g + 1]]
        assert np.all(np.diff(seg) > 0) and (len(seg) == 0 or (seg[0] >= 0 and seg[-1] < K))
        np.testing.assert_array_equal(seg, np.nonzero(mask[g])[0])
    Wm = W * _expand_mask(mask, C_out, C_in, KH, KW, N)
    np.testing.assert_array_equal(oracle.unpack(P, I, D, shape, N), Wm)


def test_pack_bf16_matches_torch_rounding():
    rng = np.random.default_rng(7)
    W = (rng.standard_normal((16, 8, 3, 3)) * 3).astype(np.float32)
    mask, _ = oracle.prune(W, 4, 0.5)
    _, _, D32 = oracle.pack(W, mask, 4, "f32")
    _, _, D16 = oracle.pack(W, mask, 4, "bf16")
    want = torch.from_numpy(D32).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    np.testing.assert_array_equal(D16, want)


def test_round_bf16_matches_torch_including_ties():
    rng = np.random.default_rng(8)
    a = rng.standard_normal(4096).astype(np.float32) * 10
    bits = a.view(np.uint32)
    bits[:512] = (bits[:512] & 0xFFFF0000) | 0x8000            # exact halfway cases
    bits[512:600] = (bits[512:600] & 0xFFFE0000) | 0x18000     # odd lsb + halfway
    want = torch.from_numpy(a).to(torch.bfloat16).float().numpy()
    np.testing.assert_array_equal(oracle.round_bf16(a), want)


# --------------------------------------------------------------------------
# Convolution (Eq. 6, Eq. 7)
# --------------------------------------------------------------------------

CONV_CASES = [
    # (B, H, W, C_in, C_out, KH, KW, stride, pad, dil)
    (1, 5, 5, 6, 8, 3, 3, 1, 1, 1),        # the 8x6x3x3 filter shape of Fig. 1
    (2, 9, 7, 6, 8, 3, 3, 2, 1, 1),
    (2, 9, 9, 4, 8, 3, 3, 1, 2, 2),
    (1, 6, 8, 5, 12, 1, 3, 1, 0, 1),
    (1, 8, 6, 3, 4, 3, 1, 2, 0, 1),
    (3, 4, 4, 16, 16, 1, 1, 1, 0, 1),
    (1, 7, 7, 2, 4, 7, 7, 2, 3, 1),
    (2, 10, 10, 3, 6, 3, 3, 3, 0, 2),
]


@pytest.mark.parametrize("case", CONV_CASES)
def test_conv_dense_equals_torch_conv2d(case):
    B, H, Wd, Ci, Co, KH, KW, s, p, d = case
    rng = np.random.default_rng(sum(case))
    x = rng.standard_normal((B, H, Wd, Ci)).astype(np.float32)
    W = rng.standard_normal((Co, Ci, KH, KW)).astype(np.float32)
    b = rng.standard_normal(Co).astype(np.float32)
    y, a = oracle.conv_masked(x, W, None, b, 1, (s, s), (p, p), (d, d), want_abs=True)
    ref = _torch_conv_nhwc(x, W, s, p, d, b)
    assert y.shape == ref.shape
    assert np.all(np.abs(y - ref) <= 1e-13 * a)


@pytest.mark.parametrize("case", CONV_CASES)
@pytest.mark.parametrize("rate", [0.3, 0.8])
def test_conv_masked_and_bsr_equal_torch_on_masked_weights(case, rate):
    B, H, Wd, Ci, Co, KH, KW, s, p, d = case
    N = 4 if Co % 4 == 0 else 2
    rng = np.random.default_rng(sum(case) + 100)
    x = np.maximum(rng.standard_normal((B, H, Wd, Ci)), 0).astype(np.float32)
    W = rng.standard_normal((Co, Ci, KH, KW)).astype(np.float32)
    b = rng.standard_normal(Co).astype(np.float32)
    mask, _ = oracle.prune(W, N, rate)
    y, a = oracle.conv_masked(x, W, mask, b, N, (s, s), (p, p), (d, d), want_abs=True)
    ref = _torch_conv_nhwc(x, W * _expand_mask(mask, Co, Ci, KH, KW, N), s, p, d, b)
    assert np.all(np.abs(y - ref) <= 1e-13 * a)
    P, I, D = oracle.pack(W, mask, N)
    yb = oracle.conv_bsr(x, P, I, D, Co, KH, KW, N, b, (s, s), (p, p), (d, d))
    np.testing.assert_array_equal(yb, y)          # same terms, same order
    yr = oracle.conv_masked(x, W, mask, b, N, (s, s), (p, p), (d, d), relu=True)
    np.testing.assert_array_equal(yr, np.maximum(y, 0))


@pytest.mark.parametrize("s,p,d", [((2, 1), (1, 0), (1, 2)), ((1, 3), (0, 2), (2, 1))])
def test_conv_asymmetric_geometry(s, p, d):
    """Different stride/pad/dilation along H and W pin each to its own axis."""
    rng = np.random.default_rng(16 + s[0])
    x = np.maximum(rng.standard_normal((2, 11, 10, 6)), 0).astype(np.float32)
    W = rng.standard_normal((8, 6, 3, 2)).astype(np.float32)
    b = rng.standard_normal(8).astype(np.float32)
    mask, _ = oracle.prune(W, 4, 0.4)
    y, a = oracle.conv_masked(x, W, mask, b, 4, s, p, d, want_abs=True)
    xt = torch.from_numpy(x.astype(np.float64)).permute(0, 3, 1, 2)
    wt = torch.from_numpy((W * _expand_mask(mask, 8, 6, 3, 2, 4)).astype(np.float64))
    ref = F.conv2d(xt, wt, torch.from_numpy(b.astype(np.float64)), stride=s, padding=p,
                   dilation=d).permute(0, 2, 3, 1).numpy()
    assert y.shape == ref.shape
    assert np.all(np.abs(y - ref) <= 1e-13 * a)
    P, I, D = oracle.pack(W, mask, 4)
    np.testing.assert_array_equal(oracle.conv_bsr(x, P, I, D, 8, 3, 2, 4, b, s, p, d), y)


def test_conv_bsr_bf16_equals_masked_on_rounded_weights():
    rng = np.random.default_rng(12)
    x = np.maximum(rng.standard_normal((2, 6, 6, 8)), 0).astype(np.float32)
    W = rng.standard_normal((16, 8, 3, 3)).astype(np.float32)
    mask, _ = oracle.prune(W, 8, 0.5)
    P, I, D16 = oracle.pack(W, mask, 8, "bf16")
    yb = oracle.conv_bsr(x, P, I, D16, 16, 3, 3, 8, None, (1, 1), (1, 1))
    ym = oracle.conv_masked(x, oracle.round_bf16(W), mask, None, 8, (1, 1), (1, 1))
    np.testing.assert_array_equal(yb, ym)


def test_conv_brute_force_python_loops():
    """Plain Python loops on the Fig. 1 filter shape (8x6x3x3, N=4)."""
    rng = np.random.default_rng(13)
    B, H, Wd, Ci, Co, K = 1, 4, 5, 6, 8, 3
    x = rng.standard_normal((B, H, Wd, Ci)).astype(np.float32)
    W = rng.standard_normal((Co, Ci, K, K)).astype(np.float32)
    b = rng.standard_normal(Co).astype(np.float32)
    mask, _ = oracle.prune(W, 4, 0.5)
    s, p, d = 2, 1, 1
    Ho, Wo = oracle.out_hw(H, Wd, K, K, (s, s), (p, p), (d, d))
    y = oracle.conv_masked(x, W, mask, b, 4, (s, s), (p, p), (d, d))
    for oh in range(Ho):
        for ow in range(Wo):
            for o in range(Co):
                acc = float(b[o])
                for kh in range(K):
                    for kw in range(K):
                        ih, iw = oh * s - p + kh * d, ow * s - p + kw * d
                        if not (0 <= ih < H and 0 <= iw < Wd):
                            continue
                        for c in range(Ci):
                            if mask[o // 4, (kh * K + kw) * Ci + c]:
                                acc += float(W[o, c, kh, kw]) * float(x[0, ih, iw, c])
                assert abs(acc - y[0, oh, ow, o]) <= 1e-12 * (1 + abs(acc))


def test_conv_rate_one_is_bias():
    """All blocks pruned (C13): the output is the bias (after ReLU)."""
    rng = np.random.default_rng(14)
    x = rng.standard_normal((1, 5, 5, 4)).astype(np.float32)
    W = rng.standard_normal((8, 4, 3, 3)).astype(np.float32)
    b = rng.standard_normal(8).astype(np.float32)
    mask, kept = oracle.prune(W, 4, 1.0)
    assert kept == 0
    P, I, D = oracle.pack(W, mask, 4)
    assert len(I) == 0 and np.all(P == 0)
    y = oracle.conv_bsr(x, P, I, D, 8, 3, 3, 4, b, (1, 1), (1, 1), relu=True)
    np.testing.assert_array_equal(y, np.broadcast_to(np.maximum(b, 0), y.shape))


def test_conv_sampled_pixels_match_full():
    rng = np.random.default_rng(15)
    x = rng.standard_normal((3, 7, 6, 8)).astype(np.float32)
    W = rng.standard_normal((8, 8, 3, 3)).astype(np.float32)
    mask, _ = oracle.prune(W, 2, 0.5)
    full = oracle.conv_masked(x, W, mask, None, 2, (2, 2), (1, 1))
    pix = np.array([0, 5, 11, 17, 30, 35], np.int64)
    part = oracle.conv_masked(x, W, mask, None, 2, (2, 2), (1, 1), pixels=pix)
    np.testing.assert_array_equal(part, full.reshape(-1, 8)[pix])
    P, I, D = oracle.pack(W, mask, 2)
    partb = oracle.conv_bsr(x, P, I, D, 8, 3, 3, 2, None, (2, 2), (1, 1), pixels=pix)
    np.testing.assert_array_equal(partb, part)


# ------------------------------------------------ MobileNet-V2 block pieces

@pytest.mark.parametrize("s,p,d", [(1, 1, 1), (2, 1, 1), (1, 2, 2), (2, 0, 1)])
def test_dwconv_equals_dense_conv_on_block_diagonal_weights(s, p, d):
    """A depthwise convolution is the dense convolution whose weight is zero
    off the channel diagonal: the oracle's two routines agree bitwise (the
    extra terms add exact zeros), and both match torch's grouped conv2d."""
    rng = np.random.default_rng(s * 7 + p * 3 + d)
    C = 6
    x = rng.standard_normal((2, 9, 8, C)).astype(np.float32)
    Wd = rng.standard_normal((C, 3, 3)).astype(np.float32)
    b = rng.standard_normal(C).astype(np.float32)
    Wfull = np.zeros((C, C, 3, 3), np.float32)
    for c in range(C):
        Wfull[c, c] = Wd[c]
    y_dw = oracle.dwconv(x, Wd, b, stride=(s, s), pad=(p, p), dil=(d, d))
    y_full = oracle.conv_masked(x, Wfull, None, b, 1, stride=(s, s), pad=(p, p), dil=(d, d))
    assert np.array_equal(y_dw, y_full)
    xt = torch.from_numpy(x.astype(np.float64)).permute(0, 3, 1, 2)
    yt = F.conv2d(xt, torch.from_numpy(Wd.astype(np.float64))[:, None], torch.from_numpy(b.astype(np.float64)),
                  stride=s, padding=p, dilation=d, groups=C).permute(0, 2, 3, 1).numpy()
    assert np.max(np.abs(y_dw - yt)) <= 1e-12 * (np.abs(yt).max() + 1)


def test_relu6_is_the_clamp_of_the_linear_output():
    rng = np.random.default_rng(11)
    x = (3 * rng.standard_normal((1, 6, 6, 8))).astype(np.float32)
    W = rng.standard_normal((8, 8, 3, 3)).astype(np.float32)
    lin = oracle.conv_masked(x, W, None, None, 1, pad=(1, 1))
    r6 = oracle.conv_masked(x, W, None, None, 1, pad=(1, 1), relu="relu6")
    assert np.array_equal(r6, np.clip(lin, 0.0, 6.0))
    assert (lin > 6).any() and (lin < 0).any()            # both clamps exercised
    Wd = rng.standard_normal((8, 3, 3)).astype(np.float32)
    assert np.array_equal(oracle.dwconv(x, Wd, pad=(1, 1), relu="relu6"),
                          np.clip(oracle.dwconv(x, Wd, pad=(1, 1)), 0.0, 6.0))


def test_residual_is_added_before_the_activation():
    rng = np.random.default_rng(12)
    x = rng.standard_normal((2, 5, 5, 4)).astype(np.float32)
    W = rng.standard_normal((4, 4, 1, 1)).astype(np.float32)
    r = rng.standard_normal((2, 5, 5, 4))
    lin = oracle.conv_masked(x, W, None, None, 1)
    assert np.array_equal(oracle.conv_masked(x, W, None, None, 1, residual=r), lin + r)
    assert np.array_equal(oracle.conv_masked(x, W, None, None, 1, residual=r, relu=True),
                          np.maximum(lin + r, 0.0))


# --------------------------------------------------------------------------
# Fine-tuning with the mask held fixed: gradients of Eq. 6
# --------------------------------------------------------------------------

def _bwd_case(case, rate, N=2, seed=0):
    B, H, Wd, Ci, Co, KH, KW, s, p, d = case
    rng = np.random.default_rng(sum(case) + seed)
    x = rng.standard_normal((B, H, Wd, Ci)).astype(np.float32)
    W = rng.standard_normal((Co, Ci, KH, KW)).astype(np.float32)
    mask, _ = oracle.prune(W, N, rate)
    Ho, Wo = oracle.out_hw(H, Wd, KH, KW, (s, s), (p, p), (d, d))
    dy = rng.standard_normal((B, Ho, Wo, Co)).astype(np.float32)
    return x, W, mask, dy, (s, s), (p, p), (d, d), rng


def _mask_oihw(mask, N, shape):
    """The [G][K] tap-major block mask expanded to W's [C_out, C_in, KH, KW]."""
    Co, Ci, KH, KW = shape
    m = np.repeat(mask, N, axis=0).reshape(Co, KH, KW, Ci)
    return m.transpose(0, 3, 1, 2).astype(bool)


@pytest.mark.parametrize("case", CONV_CASES)
@pytest.mark.parametrize("rate", [0.0, 0.5])
def test_backward_data_is_the_adjoint_of_the_forward(case, rate):
    """<conv(x), dy> = <x, dx> for the masked convolution: a dropped kernel
    flip, a transposed W, a stride/dilation slip or an ignored mask breaks
    it (the forward is the independent Eq. 6 loop)."""
    x, W, mask, dy, s, p, d, _ = _bwd_case(case, rate)
    y = oracle.conv_masked(x, W, mask, None, 2, s, p, d)
    dx = oracle.conv_backward_data(dy, W, mask, 2, x.shape[1:3], s, p, d)
    lhs, rhs = float(np.sum(y * dy)), float(np.sum(x.astype(np.float64) * dx))
    scale = float(np.sum(np.abs(y) * np.abs(dy))) + 1.0
    assert abs(lhs - rhs) <= 1e-12 * scale


@pytest.mark.parametrize("case", CONV_CASES)
def test_backward_weight_is_the_bilinear_partner(case):
    """<conv(x; W' (+) T), dy> = <W' (+) T, dW> for any W', and dW is zero
    on every pruned weight."""
    x, W, mask, dy, s, p, d, rng = _bwd_case(case, 0.5)
    dW = oracle.conv_backward_weight(x, dy, W.shape[2:], mask, 2, s, p, d)
    keep = _mask_oihw(mask, 2, W.shape)
    assert np.all(dW[~keep] == 0.0)
    W2 = rng.standard_normal(W.shape).astype(np.float32)
    y2 = oracle.conv_masked(x, W2, mask, None, 2, s, p, d)
    lhs = float(np.sum(y2 * dy))
    rhs = float(np.sum(np.where(keep, W2.astype(np.float64), 0.0) * dW))
    scale = float(np.sum(np.abs(y2) * np.abs(dy))) + 1.0
    assert abs(lhs - rhs) <= 1e-12 * scale


@pytest.mark.parametrize("case", CONV_CASES)
def test_backward_matches_torch_grad_routines(case):
    """Against torch.nn.grad.conv2d_input / conv2d_weight (fp64, NCHW) on the
    masked weights, then the mask applied to the weight gradient."""
    x, W, mask, dy, s, p, d, _ = _bwd_case(case, 0.5, seed=1)
    keep = _mask_oihw(mask, 2, W.shape)
    Wm = torch.from_numpy(np.where(keep, W, 0.0).astype(np.float64))
    xt = torch.from_numpy(x.astype(np.float64)).permute(0, 3, 1, 2)
    dyt = torch.from_numpy(dy.astype(np.float64)).permute(0, 3, 1, 2)
    dx_t = torch.nn.grad.conv2d_input(xt.shape, Wm, dyt, stride=s, padding=p, dilation=d)
    dW_t = torch.nn.grad.conv2d_weight(xt, Wm.shape, dyt, stride=s, padding=p, dilation=d)
    dx, ax = oracle.conv_backward_data(dy, W, mask, 2, x.shape[1:3], s, p, d, want_abs=True)
    dW, aw = oracle.conv_backward_weight(x, dy, W.shape[2:], mask, 2, s, p, d, want_abs=True)
    assert np.all(np.abs(dx - dx_t.permute(0, 2, 3, 1).numpy()) <= 1e-13 * (ax + 1e-300))
    assert np.all(np.abs(dW - np.where(keep, dW_t.numpy(), 0.0)) <= 1e-13 * (aw + 1e-300))


def test_backward_brute_force_scatter_loops():
    """The scatter form of both gradients in plain Python loops (every
    output position sends w * dy to the input it read, and x * dy to the
    weight it used) equals the oracle's gather form."""
    case = (2, 5, 4, 3, 4, 3, 2, 2, 1, 1)
    x, W, mask, dy, s, p, d, _ = _bwd_case(case, 0.5)
    B, H, Wd, Ci, Co, KH, KW = case[:7]
    Ho, Wo = dy.shape[1:3]
    keep = _mask_oihw(mask, 2, W.shape)
    dx = np.zeros((B, H, Wd, Ci))
    dW = np.zeros((Co, Ci, KH, KW))
    for b in range(B):
        for oh in range(Ho):
            for ow in range(Wo):
                for o in range(Co):
                    for c in range(Ci):
                        for kh in range(KH):
                            for kw in range(KW):
                                ih, iw = oh * s[0] - p[0] + kh * d[0], ow * s[1] - p[1] + kw * d[1]
                                if not keep[o, c, kh, kw] or not (0 <= ih < H and 0 <= iw < Wd):
                                    continue
                                dx[b, ih, iw, c] += float(W[o, c, kh, kw]) * float(dy[b, oh, ow, o])
                                dW[o, c, kh, kw] += float(x[b, ih, iw, c]) * float(dy[b, oh, ow, o])
    np.testing.assert_allclose(oracle.conv_backward_data(dy, W, mask, 2, (H, Wd), s, p, d), dx,
                               rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(oracle.conv_backward_weight(x, dy, (KH, KW), mask, 2, s, p, d), dW,
                               rtol=1e-12, atol=1e-12)


@pytest.mark.parametrize("shape,N", [((8, 6, 3, 3), 2), ((16, 8, 1, 1), 4), ((12, 5, 3, 1), 3)])
def test_bsr_gather_inverts_unpack(shape, N):
    """The weight gradient in BSR order (Sec. 3.4): unpacking the gathered
    kept blocks gives back the masked gradient, bit for bit."""
    rng = np.random.default_rng(shape[0] + N)
    W = rng.standard_normal(shape).astype(np.float32)
    mask, _ = oracle.prune(W, N, 0.5)
    P, I, D = oracle.pack(W, mask, N)
    g = rng.standard_normal(shape).astype(np.float32)
    keep = _mask_oihw(mask, N, shape)
    dD = oracle.bsr_gather(np.where(keep, g, 0.0).astype(np.float32), P, I, N)
    assert dD.shape == D.shape
    np.testing.assert_array_equal(oracle.unpack(P, I, dD, shape, N), np.where(keep, g, 0.0))
    # and on the weights themselves it is the pack's D
    np.testing.assert_array_equal(oracle.bsr_gather(W, P, I, N), D)
