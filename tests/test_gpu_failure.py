"""Failure detection on the GPU without a fault: a wait that can only run out.

With the test hook on, one consumer warp of every gate+up CTA waits on a
barrier nothing arrives at. The bounded wait gives up, the status word records
a timeout that ts_ffn_get_error reports, the kernels wind down (the other waits
that depended on that warp give up too), and the context stays usable: the
next forward with the hook off gives the same bits as before.
"""
import time

import pytest
import torch

from paper_2406_05955_gb300 import workload as wl

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def ts():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    import paper_2406_05955_gb300 as ts

    ts.lib()
    return ts


def test_bounded_wait_reports_timeout_and_context_survives(ts):
    from paper_2406_05955_gb300 import binding

    dev = torch.device("cuda")
    L = wl.ffn_layer(1024, 3584, activation=0.10, dtype=torch.bfloat16, seed=4242, device=dev)
    f = ts.Ffn(L.w_gate, L.w_up, L.w_down, max_batch=1)
    x = wl.tokens(1, 1024, seed=4243).to(dev)
    y_ref = f.forward(x).clone()
    assert f.get_error() == binding.TS_OK

    f.set_test_stall(True)
    t0 = time.time()
    f.forward(x)
    err = f.get_error()
    waited = time.time() - t0
    f.set_test_stall(False)
    assert err == binding.TS_ERR_TIMEOUT, binding.status_str(err)
    assert 0.5 < waited < 30.0, f"timed-out forward took {waited:.1f} s"

    y = f.forward(x)
    assert f.get_error() == binding.TS_OK
    assert torch.equal(y, y_ref), "the forward after a timeout differs"
    torch.cuda.synchronize()
