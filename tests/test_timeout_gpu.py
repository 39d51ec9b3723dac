"""The bounded waits of the batch-1 decode kernel: with the test switch
BISCO_TEST_WITHHOLD_COPIES the kernel requests none of its data, so every
wait runs out after its limit (one second) with no copy in flight; the
launch must report BISCO_ERR_TIMEOUT through bisco_get_device_error and
leave the context usable -- the next call is correct."""
import numpy as np
import pytest

import oracle
from paper_2607_08643_gb300 import synth

from _helpers import assert_parity, gemv_tight, to_dev

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def env():
    import torch
    import __graft_entry__
    __graft_entry__.build()
    from paper_2607_08643_gb300 import bisco
    dev = torch.device("cuda:0")
    torch.cuda.set_device(dev)
    return bisco, dev


@pytest.mark.parametrize("N,K,S,p", [
    (600, 4096, 2, 41),       # one span
    (400, 12288, 2, 123),     # three spans: the barriers between spans are still passed
])
def test_expired_wait_reports_timeout_and_the_next_call_is_correct(env, monkeypatch, N, K, S, p):
    import torch
    bisco, dev = env
    Lref = oracle.encode(synth.layer_weights(N, K, seed=301), S=S, p=p)
    L = bisco.Layer.from_numpy(Lref, dev)
    X = synth.activations(1, K, seed=302)
    x = to_dev(X, dev)
    assert bisco.bisco_get_device_error() == bisco.OK
    monkeypatch.setenv("BISCO_TEST_WITHHOLD_COPIES", "1")
    bisco.bisco_gemv(L, x)
    torch.cuda.synchronize()
    assert bisco.bisco_get_device_error() == bisco.ERR_TIMEOUT
    assert bisco.bisco_get_device_error() == bisco.OK          # read and cleared
    monkeypatch.delenv("BISCO_TEST_WITHHOLD_COPIES")
    y = bisco.bisco_gemv(L, x)
    torch.cuda.synchronize()
    assert bisco.bisco_get_device_error() == bisco.OK
    assert_parity(y.cpu().numpy(), oracle.gemv(Lref, X), gemv_tight(1))
