"""bisco_lora_apply (the low-rank compensation of Sec. III-F) against the
fp64 oracle's lora_apply.

The kernels sum in fp32, and every product they form (bf16 x bf16 in the
down projection, bf16 x fp32 inside an fma in the up projection) is exact.
The down projection adds K terms per rank row, the up projection rank terms
per output, and one fused multiply-add puts scale * sum into y.  So each
output is within (K + rank + 2) * 2^-24 (first order) of
    |y0| + |scale| * sum_r |Bm[n][r]| * sum_k |A[r][k] x[b][k]|,
the bound checked element by element here.  It is far inside the 2e-3
parity bar of the coded layers, which the end-to-end case uses."""
import numpy as np
import pytest

import oracle
from paper_2607_08643_gb300 import synth

from _helpers import TOL, max_rel_rows, to_dev

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


def _bound(A, Bm, X, Y0, scale):
    fa = synth.bf16_bits_to_f32(A).astype(np.float64)
    fb = synth.bf16_bits_to_f32(Bm).astype(np.float64)
    fx = synth.bf16_bits_to_f32(X).astype(np.float64)
    tabs = np.abs(fx) @ np.abs(fa).T                      # [B][rank]
    mag = np.abs(Y0) + abs(scale) * tabs @ np.abs(fb).T   # [B][N]
    rank, K = A.shape
    return (K + rank + 2) * 2.0 ** -24 * mag * 1.01


def _run(env, A, Bm, X, Y0, scale):
    import torch
    bisco, dev = env
    y = torch.from_numpy(np.ascontiguousarray(Y0, np.float32)).to(dev)
    bisco.bisco_lora_apply(to_dev(A, dev), to_dev(Bm, dev), to_dev(X, dev), y, scale)
    torch.cuda.synchronize()
    assert bisco.bisco_get_device_error() == 0
    return y.cpu().numpy().astype(np.float64)


CASES = [
    # N, K, rank, batch, scale
    (4096, 4096, 16, 1, 1.0),      # q_proj / o_proj, decode
    (4096, 4096, 16, 16, 0.5),     # decode batch 16
    (1024, 4096, 8, 1, 2.0),       # k_proj / v_proj, smallest rank
    (1000, 136, 24, 9, -1.5),      # ragged N, K tail below one warp pass, ragged batch block
    (300, 4096, 256, 3, 0.125),    # largest rank
    (4096, 4096, 16, 2048, 1.0),   # prefill-sized batch
]


@pytest.mark.parametrize("N,K,rank,B,scale", CASES)
def test_lora_matches_oracle(env, N, K, rank, B, scale):
    A, Bm = synth.lora_adapter(N, K, rank, seed=N + K + rank)
    X = synth.activations(B, K, seed=B + 7)
    # start from float32-representable outputs, as a layer writes them
    Y0 = synth.bf16_bits_to_f32(synth.activations(B, N, seed=B + 8)).astype(np.float64)
    ref = oracle.lora_apply(A, Bm, X, Y0, scale)
    got = _run(env, A, Bm, X, Y0, scale)
    bad = np.abs(got - ref) > _bound(A, Bm, X, Y0, scale)
    if bad.any():
        b, n = np.argwhere(bad)[0]
        pytest.fail("y[%d][%d] = %r, oracle %r (%d outputs outside the bound)"
                    % (b, n, got[b, n], ref[b, n], int(bad.sum())))


def test_lora_scale_zero_and_repeat(env):
    """scale 0 leaves y bit for bit; the result does not depend on the call."""
    N, K, rank, B = 512, 1024, 32, 5
    A, Bm = synth.lora_adapter(N, K, rank, seed=3)
    X = synth.activations(B, K, seed=4)
    Y0 = synth.bf16_bits_to_f32(synth.activations(B, N, seed=5)).astype(np.float64)
    assert np.array_equal(_run(env, A, Bm, X, Y0, 0.0), Y0.astype(np.float32))
    assert np.array_equal(_run(env, A, Bm, X, Y0, 0.75), _run(env, A, Bm, X, Y0, 0.75))


@pytest.mark.parametrize("B", [1, 4])
def test_lora_after_gemv_end_to_end(env, B):
    """A coded layer's output plus its compensation, as a caller chains them
    on one stream, against the oracle's layer output plus the oracle's
    compensation (the parity bar of the coded layer)."""
    import torch
    bisco, dev = env
    N, K, S, p, rank = 1024, 1024, 2, 11, 16
    Lref = oracle.encode(synth.layer_weights(N, K, seed=1), S=S, p=p)
    A, Bm = synth.lora_adapter(N, K, rank, seed=2)
    X = synth.activations(B, K, seed=3)
    ref = oracle.lora_apply(A, Bm, X, oracle.gemv(Lref, X), 1.0)
    L = bisco.Layer.from_numpy(Lref, dev)
    xd = to_dev(X, dev)
    y = bisco.bisco_gemv(L, xd)
    bisco.bisco_lora_apply(to_dev(A, dev), to_dev(Bm, dev), xd, y, 1.0)
    torch.cuda.synchronize()
    assert bisco.bisco_get_device_error() == 0
    assert max_rel_rows(y.cpu().numpy(), ref) <= TOL


@pytest.mark.parametrize("N,K,rank,B,scale", CASES)
def test_lora_split_down_matches_oracle(env, N, K, rank, B, scale, monkeypatch):
    """BISCO_LORA_SPLIT=1 (each rank row's K over the 8 warps of a CTA, added
    in warp order): the same bound, and deterministic."""
    monkeypatch.setenv("BISCO_LORA_SPLIT", "1")
    A, Bm = synth.lora_adapter(N, K, rank, seed=N + K + rank)
    X = synth.activations(B, K, seed=B + 7)
    Y0 = synth.bf16_bits_to_f32(synth.activations(B, N, seed=B + 8)).astype(np.float64)
    ref = oracle.lora_apply(A, Bm, X, Y0, scale)
    got = _run(env, A, Bm, X, Y0, scale)
    assert np.all(np.abs(got - ref) <= _bound(A, Bm, X, Y0, scale))
    assert np.array_equal(got, _run(env, A, Bm, X, Y0, scale))
