"""Checked mode (ONEXN_CHECK_INPUT): a validation kernel checks the device
BSR lists of Sec. 3.4 before the convolution and reports malformed ones as
ONEXN_EDEVICE through onexn_device_status.  The corrupted lists used here
stay inside the arrays (an index past K, a repeated index, a last P entry
short of t); every kernel family clamps what it reads from P and I, so
nothing is read out of bounds and the output is merely meaningless."""
import numpy as np
import pytest
import torch

from paper_2105_14713_gb300 import onexn as ox
from paper_2105_14713_gb300 import workloads as wl
from paper_2105_14713_gb300.layer import PrunedConv2d
from tests.gpu_util import norm_err, oracle_ref, tol

pytestmark = pytest.mark.gpu

ALGOS = ["fma", "tc", "mma"]


def _conv():
    layer = wl.ConvLayer("chk", 2, 10, 10, 64, 64, 3, 3, 1, 1, 1, N=16, rate=0.5, dtype="bf16", seed=4)
    W, b = wl.weights(layer).numpy(), wl.bias(layer).numpy()
    conv = PrunedConv2d(W, 16, 0.5, bias=b, padding=1, dtype="bf16")
    return layer, conv, W, b


@pytest.mark.parametrize("algo", ALGOS)
def test_valid_lists_pass_the_check(algo):
    assert ox.onexn_device_status(clear=True) in (ox.ONEXN_OK, ox.ONEXN_EDEVICE, ox.ONEXN_ETIMEOUT)
    layer, conv, W, b = _conv()
    x_cpu = wl.activations(layer)
    y = conv(x_cpu.to(torch.bfloat16).cuda(), algo=ox.ALGO_BY_NAME[algo] | ox.ONEXN_CHECK_INPUT)
    assert ox.onexn_device_status(clear=True) == ox.ONEXN_OK
    y_ref, absacc = oracle_ref(layer, W, x_cpu, b)
    assert norm_err(y.float().cpu().numpy().reshape(-1, 64).astype(np.float64), y_ref, absacc) <= tol(layer)


@pytest.mark.parametrize("kind", ["index_past_K", "repeated_index", "last_P_short"])
@pytest.mark.parametrize("algo", ALGOS)
def test_malformed_lists_are_reported(kind, algo):
    layer, conv, _, _ = _conv()
    K = 9 * 64
    I = conv.I.clone()
    P = conv.P.clone()
    if kind == "index_past_K":
        I[conv.t // 2] = K + 7
    elif kind == "repeated_index":
        I[1] = I[0]                       # group 0 keeps more than one block at rate 0.5
    else:
        P[-1] = conv.t - 1
    conv.I.copy_(I)
    conv.P.copy_(P)
    x = wl.activations(layer).to(torch.bfloat16).cuda()
    conv(x, algo=ox.ALGO_BY_NAME[algo] | ox.ONEXN_CHECK_INPUT)
    assert ox.onexn_device_status(clear=True) == ox.ONEXN_EDEVICE
    # the report clears, and the context stays usable
    _, good, _, _ = _conv()
    good(x, algo=ox.ALGO_BY_NAME[algo] | ox.ONEXN_CHECK_INPUT)
    assert ox.onexn_device_status(clear=True) == ox.ONEXN_OK
