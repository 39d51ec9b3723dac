"""bisco_encode_noalloc: the encoder entry point that allocates nothing.

Some callers of this library cannot allocate device memory: a host
application whose own allocator has already reserved the GPU's memory and
forbids other cudaMalloc calls, or code that must not trigger the device-wide
synchronisation that cudaMalloc/cudaFree can cause.  For them the encoder
takes its scratch space from a fixed array inside the library instead of a
caller-provided workspace.  Here the entry point is called through the C ABI
twice in a row (the array keeps whatever the previous call left in it), and
each time its output bytes must equal those of bisco_encode, whose parity
with the fp64 oracle is checked elsewhere.  Encoded bytes are exact integer
data, so the comparison is bit-exact.

This file is named so that pytest collects it last.
"""
import ctypes

import numpy as np
import pytest

from paper_2607_08643_gb300 import synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def env():
    import torch
    import __graft_entry__
    __graft_entry__.build()
    from paper_2607_08643_gb300 import bisco
    dev = torch.device("cuda:0")
    torch.cuda.set_device(dev)
    return bisco, bisco.load(), dev


def _bytes(L):
    d = L.to_numpy()
    return {k: d[k] for k in ("codes", "norms", "q8", "scale", "idx")}


def test_noalloc_encode_equals_workspace_encode_on_two_calls(env):
    import torch
    bisco, lib, dev = env
    stream = torch.cuda.current_stream()
    cases = [(256, 4096, 2, 41, 1), (96, 1536, 3, 31, 2)]     # two calls in a row
    for N, K, S, p, seed in cases:
        W = torch.from_numpy(synth.layer_weights(N, K, seed=seed).view(np.int16)).to(dev)
        ref = bisco.bisco_encode(W, S, p)                     # existing entry point
        L = bisco.Layer(N, K, S, p, dev)
        st = lib.bisco_encode_noalloc(ctypes.c_void_p(W.data_ptr()), None, ctypes.byref(L.c),
                                      ctypes.c_void_p(stream.cuda_stream))
        assert st == bisco.OK
        torch.cuda.synchronize()
        assert bisco.bisco_get_device_error() == bisco.OK
        got, want = _bytes(L), _bytes(ref)
        for k in want:
            assert np.array_equal(got[k], want[k]), k


def test_noalloc_encode_rejects_k_beyond_its_array(env):
    bisco, lib, _ = env
    L = bisco.bisco_layer(4, 32776, 8, 1, 0, 0, 0x10000, 0x20000, 0, 0, 0)
    assert lib.bisco_encode_noalloc(ctypes.c_void_p(0x30000), None, ctypes.byref(L), None) \
        == bisco.ERR_UNSUPPORTED
