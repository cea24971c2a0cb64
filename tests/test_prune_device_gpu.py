"""Device-side prune and pack (onexn_prune_device / onexn_pack_device)
against the oracle, bit for bit: the masks (both granularities, integer
weights with many tied norms, rates 0 and 1), the kept count, and the BSR
P, I, D (fp32 copy and bf16 round-to-nearest-even)."""
import numpy as np
import pytest
import torch

import oracle
from paper_2105_14713_gb300 import onexn as ox

pytestmark = pytest.mark.gpu

SHAPES = [
    # (C_out, C_in, KH, KW, N, integer weights)
    ((16, 8, 3, 3), 4, True),
    ((64, 32, 3, 3), 8, False),
    ((48, 24, 1, 1), 2, True),
    ((96, 40, 1, 3), 3, False),
    ((512, 512, 3, 3), 8, False),      # 294912 blocks: many CTAs and rank chunks
    ((256, 64, 1, 1), 16, True),
]


def _weights(shape, integer, seed):
    rng = np.random.default_rng(seed)
    if integer:
        return rng.integers(-3, 4, size=shape).astype(np.float32)
    return (rng.standard_normal(shape) * 0.05).astype(np.float32)


@pytest.mark.parametrize("spec", SHAPES, ids=[str(s[0]) for s in SHAPES])
@pytest.mark.parametrize("gran", [ox.ONEXN_GRAN_TAP, ox.ONEXN_GRAN_KERNEL])
@pytest.mark.parametrize("rate", [0.0, 0.3, 0.5, 0.9, 1.0])
def test_prune_device_matches_oracle(spec, gran, rate):
    shape, N, integer = spec
    if gran == ox.ONEXN_GRAN_KERNEL and shape[2] * shape[3] == 1 and rate in (0.3, 0.9):
        pytest.skip("same as the tap mode for 1x1")
    W = _weights(shape, integer, sum(shape) + N)
    mask_d, kept = ox.onexn_prune_device(torch.from_numpy(W).cuda(), N, rate, gran)
    mask_o, kept_o = oracle.prune(W, N, rate, gran)
    assert kept == kept_o
    np.testing.assert_array_equal(mask_d.cpu().numpy(), mask_o)


@pytest.mark.parametrize("spec", SHAPES, ids=[str(s[0]) for s in SHAPES])
@pytest.mark.parametrize("wdtype", [ox.ONEXN_F32, ox.ONEXN_BF16])
def test_pack_device_matches_oracle(spec, wdtype):
    shape, N, integer = spec
    W = _weights(shape, integer, sum(shape) + 7)
    mask_o, _ = oracle.prune(W, N, 0.5)
    Wd = torch.from_numpy(W).cuda()
    t = int(mask_o.sum())
    P, I, D = ox.onexn_pack_device(Wd, torch.from_numpy(mask_o).cuda(), N, t, wdtype)
    Po, Io, Do = oracle.pack(W, mask_o, N, "f32" if wdtype == ox.ONEXN_F32 else "bf16")
    np.testing.assert_array_equal(P.cpu().numpy(), Po)
    np.testing.assert_array_equal(I.cpu().numpy(), Io)
    if wdtype == ox.ONEXN_F32:
        np.testing.assert_array_equal(D.cpu().numpy(), Do)
    else:
        np.testing.assert_array_equal(D.cpu().view(torch.int16).numpy().view(np.uint16), Do)


def test_prune_then_pack_on_device_feeds_the_convolution():
    """Device prune -> device pack -> the convolution, against the oracle conv."""
    from paper_2105_14713_gb300.layer import PrunedConv2d
    W = _weights((64, 32, 3, 3), False, 5)
    Wd = torch.from_numpy(W).cuda()
    mask, kept = ox.onexn_prune_device(Wd, 4, 0.5)
    P, I, D = ox.onexn_pack_device(Wd, mask, 4, kept)
    conv = PrunedConv2d(W, 4, 0.5, padding=1)
    assert torch.equal(P.cpu(), conv.P.cpu()) and torch.equal(I.cpu(), conv.I.cpu())
    assert torch.equal(D.cpu(), conv.D.cpu())
    x = torch.relu(torch.randn(2, 9, 9, 32, generator=torch.Generator().manual_seed(1)))
    y = conv(x.cuda())
    ref, a = oracle.conv_masked(x.numpy(), W, mask.cpu().numpy(), None, 4, (1, 1), (1, 1), want_abs=True)
    assert float(np.max(np.abs(y.cpu().numpy() - ref) / (a + 1e-30))) <= 1e-5


def test_pack_device_empty_mask_and_short_capacity():
    W = _weights((16, 8, 1, 1), False, 3)
    Wd = torch.from_numpy(W).cuda()
    zero = torch.zeros((4, 8), dtype=torch.uint8, device="cuda")
    P, I, D = ox.onexn_pack_device(Wd, zero, 4, 0)
    assert P.cpu().tolist() == [0] * 5
    # a capacity short of the count: P still counts every block, nothing past t_cap is written
    full = torch.ones((4, 8), dtype=torch.uint8, device="cuda")
    P, I, D = ox.onexn_pack_device(Wd, full, 4, 5)
    assert P.cpu().tolist() == [0, 8, 16, 24, 32]
    assert I.cpu().tolist() == [0, 1, 2, 3, 4]
