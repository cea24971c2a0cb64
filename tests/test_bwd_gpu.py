"""GPU parity of the fine-tuning passes (mask held fixed) against the
oracle's gradients of Eq. 6: the input gradient (tensor-core path for
stride-1 layers, direct kernel for strided ones), the kept-weight gradient
in BSR order and the bias gradient, in fp32 and bf16, on ragged sizes that
span several tiles and pixel slices; plus the autograd wrapper.

Tolerances (normalised by the sum of |terms|, reading C12): fp32 1e-5
(three tf32 products per term, fp32 accumulation); bf16 input gradient
4e-3 (bf16 output rounding, 2^-8); bf16 weight gradient 1e-5 (exact bf16
products, fp32 accumulation and an fp32 result)."""
import numpy as np
import pytest
import torch

import oracle
from paper_2105_14713_gb300 import onexn as ox
from paper_2105_14713_gb300 import workloads as wl
from paper_2105_14713_gb300.layer import PrunedConv2d

pytestmark = pytest.mark.gpu

L = wl.ConvLayer

CASES = [
    # name, B, H, W, C_in, C_out, KH, KW, stride, pad, dil, N
    ("3x3_s1", 3, 13, 11, 32, 64, 3, 3, 1, 1, 1, 8),
    ("1x1", 2, 15, 9, 48, 96, 1, 1, 1, 0, 1, 4),
    ("3x3_p0", 2, 12, 10, 16, 32, 3, 3, 1, 0, 1, 4),
    ("3x3_d2", 2, 14, 12, 24, 40, 3, 3, 1, 2, 2, 8),
    ("1x3", 2, 9, 17, 32, 48, 1, 3, 1, 0, 1, 16),
    ("3x3_s2", 3, 15, 13, 32, 64, 3, 3, 2, 1, 1, 8),       # dy dilated by the stride, tensor cores
    ("1x1_s2", 2, 14, 14, 64, 128, 1, 1, 2, 0, 1, 4),      # dilated, ragged last row/column of x
    ("3x3_s2_d2", 2, 15, 15, 16, 32, 3, 3, 2, 2, 2, 4),    # dilated dy, dilated kernel
    ("3x3_s3", 2, 16, 14, 16, 32, 3, 3, 3, 1, 1, 4),       # stride 3
    ("1x1_p1", 2, 9, 9, 32, 64, 1, 1, 1, 1, 1, 8),         # padding beyond d(K-1): direct kernel
    ("3x3_s2_p3", 2, 13, 11, 32, 64, 3, 3, 2, 3, 1, 8),    # direct kernel, strided
]


def _setup(case, dtype, seed=0):
    name, B, H, W, Ci, Co, KH, KW, s, p, d, N = case
    layer = L(name, B, H, W, Ci, Co, KH, KW, s, p, d, N=N, rate=0.5, dtype=dtype, seed=seed + 3)
    Wt = wl.weights(layer).numpy()
    conv = PrunedConv2d(Wt, N, 0.5, bias=wl.bias(layer).numpy(), stride=s, padding=p, dilation=d, dtype=dtype)
    tdt = torch.float32 if dtype == "f32" else torch.bfloat16
    x = wl.activations(layer).to(tdt).cuda()
    Ho, Wo = layer.Ho, layer.Wo
    g = torch.Generator().manual_seed(seed + 11)
    dy = torch.randn((B, Ho, Wo, Co), generator=g).to(tdt).cuda()
    mask, _ = oracle.prune(Wt, N, 0.5)
    W_seen = Wt if dtype == "f32" else oracle.round_bf16(Wt)
    return layer, conv, x, dy, mask, W_seen, (s, s), (p, p), (d, d)


def _np(t):
    return t.float().cpu().numpy()


def _err(y, ref, a):
    return float(np.max(np.abs(y.astype(np.float64) - ref) / (a + 1e-30))) if y.size else 0.0


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("case", CASES, ids=[c[0] for c in CASES])
def test_input_gradient(case, dtype):
    layer, conv, x, dy, mask, W, s, p, d = _setup(case, dtype)
    dx, _, _ = conv.backward(x, dy, need_dw=False, need_db=False)
    torch.cuda.synchronize()
    ref, a = oracle.conv_backward_data(_np(dy), W, mask, layer.N, (layer.H, layer.W), s, p, d, want_abs=True)
    assert dx.shape == x.shape
    assert _err(_np(dx), ref, a) <= (1e-5 if dtype == "f32" else 4e-3)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("case", CASES, ids=[c[0] for c in CASES])
def test_kept_weight_and_bias_gradient(case, dtype):
    layer, conv, x, dy, mask, W, s, p, d = _setup(case, dtype, seed=1)
    _, dD, db = conv.backward(x, dy, need_dx=False)
    torch.cuda.synchronize()
    dW, a = oracle.conv_backward_weight(_np(x), _np(dy), (layer.KH, layer.KW), mask, layer.N, s, p, d,
                                        want_abs=True)
    P, I = conv.P_host, conv.I_host
    ref, ra = oracle.bsr_gather(dW, P, I, layer.N), oracle.bsr_gather(a, P, I, layer.N)
    assert dD.shape == (conv.t, layer.N) and dD.dtype == torch.float32
    assert _err(dD.cpu().numpy(), ref, ra) <= 1e-5
    dyn = _np(dy).astype(np.float64).reshape(-1, layer.C_out)
    assert np.all(np.abs(db.cpu().numpy() - dyn.sum(0)) <= 1e-5 * np.abs(dyn).sum(0) + 1e-30)


def test_accumulate_adds_into_dx():
    for case in (CASES[0], CASES[5], CASES[-1]):        # stride 1, dilated and direct paths
        layer, conv, x, dy, mask, W, s, p, d = _setup(case, "f32", seed=2)
        base = torch.randn(x.shape, generator=torch.Generator().manual_seed(4)).cuda()
        dx = base.clone()
        conv.backward(x, dy, dx, need_dw=False, need_db=False, accumulate=True)
        torch.cuda.synchronize()
        ref, a = oracle.conv_backward_data(_np(dy), W, mask, layer.N, (layer.H, layer.W), s, p, d, want_abs=True)
        ref = ref + _np(base)
        assert _err(_np(dx), ref, a + np.abs(_np(base))) <= 1e-5


def test_resnet50_3x3_sized_gradients_sampled():
    """8 x 28 x 28 x 128 -> 128 3x3, N=8: 50 GEMM tiles of the input
    gradient, the weight-gradient GEMM in pixel slices across every SM."""
    case = ("r50", 8, 28, 28, 128, 128, 3, 3, 1, 1, 1, 8)
    for dtype in ("f32", "bf16"):
        layer, conv, x, dy, mask, W, s, p, d = _setup(case, dtype, seed=5)
        dx, dD, db = conv.backward(x, dy)
        torch.cuda.synchronize()
        ref, a = oracle.conv_backward_data(_np(dy), W, mask, 8, (28, 28), s, p, d, want_abs=True)
        assert _err(_np(dx), ref, a) <= (1e-5 if dtype == "f32" else 4e-3)
        dW, aw = oracle.conv_backward_weight(_np(x), _np(dy), (3, 3), mask, 8, s, p, d, want_abs=True)
        assert _err(dD.cpu().numpy(), oracle.bsr_gather(dW, conv.P_host, conv.I_host, 8),
                    oracle.bsr_gather(aw, conv.P_host, conv.I_host, 8)) <= 1e-5


def test_empty_batch_gives_zero_weight_gradient():
    case = ("empty", 0, 8, 8, 16, 32, 3, 3, 1, 1, 1, 4)
    layer = L("empty", 1, 8, 8, 16, 32, 3, 3, 1, 1, 1, N=4, rate=0.5)
    conv = PrunedConv2d(wl.weights(layer).numpy(), 4, 0.5, padding=1)
    x = torch.zeros((0, 8, 8, 16), device="cuda")
    dy = torch.zeros((0, 8, 8, 32), device="cuda")
    dx, dD, db = conv.backward(x, dy)
    torch.cuda.synchronize()
    assert dx.shape == x.shape
    assert torch.count_nonzero(dD).item() == 0 and torch.count_nonzero(db).item() == 0


def test_autograd_matches_dense_masked_torch_and_fine_tuning_lowers_the_loss():
    """train_forward as a differentiable op: its gradients equal torch's
    autograd of the dense masked conv (fp64, CPU), and a few SGD steps on D
    (only the kept blocks) lower a regression loss while the mask stays."""
    case = ("ft", 2, 10, 10, 32, 64, 3, 3, 1, 1, 1, 8)
    layer, conv, x, dy, mask, W, s, p, d = _setup(case, "f32", seed=7)
    D, bias = conv.parameters()
    xg = x.clone().requires_grad_(True)
    y = conv.train_forward(xg)
    (y * dy).sum().backward()
    keep = np.repeat(mask, 8, axis=0).reshape(64, 3, 3, 32).transpose(0, 3, 1, 2).astype(bool)
    Wm = torch.from_numpy(np.where(keep, W, 0.0)).double().requires_grad_(True)
    xt = x.cpu().double().permute(0, 3, 1, 2).requires_grad_(True)
    bt = bias.detach().cpu().double().requires_grad_(True)
    yt = torch.nn.functional.conv2d(xt, Wm, bt, padding=1)
    (yt * dy.cpu().double().permute(0, 3, 1, 2)).sum().backward()
    gx = xt.grad.permute(0, 2, 3, 1).numpy()
    assert np.max(np.abs(xg.grad.cpu().numpy() - gx)) <= 1e-4 * np.max(np.abs(gx))
    gW = oracle.bsr_gather(Wm.grad.numpy(), conv.P_host, conv.I_host, 8)
    assert np.max(np.abs(D.grad.cpu().numpy() - gW)) <= 1e-4 * np.max(np.abs(gW))
    assert np.max(np.abs(bias.grad.cpu().numpy() - bt.grad.numpy())) <= 1e-4 * np.max(np.abs(bt.grad.numpy()))
    # fine-tune D toward a target made by other kept weights
    target = torch.randn(y.shape, generator=torch.Generator().manual_seed(9)).cuda()
    opt = torch.optim.SGD([D, bias], lr=1e-3)
    losses = []
    for _ in range(5):
        opt.zero_grad()
        loss = ((conv.train_forward(x) - target) ** 2).mean()
        loss.backward()
        opt.step()
        losses.append(loss.item())
    assert losses[-1] < losses[0]
    assert torch.equal(conv.P.cpu(), torch.from_numpy(conv.P_host))     # the mask never moves
