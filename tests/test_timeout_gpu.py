"""The timeout path of the library's bounded in-kernel waits, without a GPU
fault: onexn_selftest_timeout runs a kernel whose bounded mbarrier wait has
nothing to wait for, so it runs out (about one second) and sets the status
word.  The test checks that onexn_device_status reports ONEXN_ETIMEOUT, that
the report clears, and that the context stays usable (a convolution after it
matches the oracle)."""
import pytest
import torch

from paper_2105_14713_gb300 import onexn as ox
from paper_2105_14713_gb300 import workloads as wl
from tests.gpu_util import norm_err, run_layer, tol

pytestmark = pytest.mark.gpu


def test_bounded_wait_runs_out_and_is_reported():
    assert ox.onexn_device_status(clear=True) == ox.ONEXN_OK
    ox.onexn_selftest_timeout()
    torch.cuda.synchronize()
    assert ox.onexn_device_status(clear=False) == ox.ONEXN_ETIMEOUT
    assert ox.onexn_device_status(clear=True) == ox.ONEXN_ETIMEOUT
    assert ox.onexn_device_status(clear=True) == ox.ONEXN_OK
    # the context is still usable
    layer = wl.ConvLayer("after_timeout", 2, 14, 14, 64, 64, 3, 3, 1, 1, 1, N=8, rate=0.5, dtype="f32", seed=5)
    y, y_ref, absacc, _ = run_layer(layer, algo=ox.ALGO_BY_NAME["tc"])
    assert norm_err(y, y_ref, absacc) <= tol(layer)
    assert ox.onexn_device_status(clear=True) == ox.ONEXN_OK
