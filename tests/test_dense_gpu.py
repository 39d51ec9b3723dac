"""bisco_decode_dense (the materialise-then-multiply path) against the fp64
oracle's dense decode (Eq. 12 with the Eq. 10 overwrite).

fp32 output: the stage sum is exact in fp32 and rounded once after the
1/sqrt(8) scale, so each element is within 2^-22 relative of the oracle's
value (protected columns exactly).  bf16 / fp16 outputs round that fp32
value once more, within one unit in the last place of the oracle's value.
Where the stage terms cancel exactly the GPU value is 0 and the oracle's
(which scales each term by 1/sqrt(8) in fp64 before the sum) is fp64
rounding noise, so both bounds carry an absolute floor of 2^-40 times the
largest weight."""
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


def _dense(env, Lref, dtype):
    import torch
    bisco, dev = env
    L = bisco.Layer.from_numpy(Lref, dev)
    out = bisco.bisco_decode_dense(L, dtype)
    torch.cuda.synchronize()
    assert bisco.bisco_get_device_error() == 0
    return out.float().cpu().numpy().astype(np.float64)


CASES = [
    (200, 1536, 3, 20, "t4"),      # three stages, ragged N
    (100, 1000, 2, 10, "normal"),  # K % 128 != 0
    (64, 512, 1, 0, "normal"),     # one stage, no protection
    (32, 256, 2, 256, "normal"),   # every column protected
    (1024, 4096, 2, 41, "normal"),  # k_proj / v_proj
]


@pytest.mark.parametrize("N,K,S,p,dist", CASES)
def test_decode_dense_f32_matches_oracle(env, N, K, S, p, dist):
    Lref = oracle.encode(synth.layer_weights(N, K, seed=N + K + S, dist=dist), S=S, p=p)
    ref = oracle.decode_rows(Lref)
    got = _dense(env, Lref, "f32")
    floor = 2.0 ** -40 * np.abs(ref).max()
    bad = np.abs(got - ref) > 2.0 ** -22 * np.abs(ref) + floor
    if bad.any():
        i, j = np.argwhere(bad)[0]
        raise AssertionError("%d elements off; first at (%d, %d): got %r ref %r (protected: %s)"
                             % (bad.sum(), i, j, got[i, j], ref[i, j], j in set(Lref["idx"].tolist())))
    if p > 0:
        cols = Lref["idx"]
        assert np.array_equal(got[:, cols], ref[:, cols])   # scale * q8, exact


@pytest.mark.parametrize("dtype,mant", [("bf16", 8), ("f16", 11)])
@pytest.mark.parametrize("N,K,S,p,dist", CASES[:3])
def test_decode_dense_half_types(env, dtype, mant, N, K, S, p, dist):
    Lref = oracle.encode(synth.layer_weights(N, K, seed=3 * N + K, dist=dist), S=S, p=p)
    ref = oracle.decode_rows(Lref)
    got = _dense(env, Lref, dtype)
    # one unit in the last place of the reference (mant significant bits)
    ulp = np.exp2(np.floor(np.log2(np.maximum(np.abs(ref), 1e-30))) - (mant - 1))
    if dtype == "f16":
        ulp = np.maximum(ulp, 2.0 ** -24)   # fp16 subnormals are 2^-24 apart
    floor = 2.0 ** -40 * np.abs(ref).max()
    bad = np.abs(got - ref) > ulp + floor
    assert not bad.any(), (bad.sum(), got[bad][:4], ref[bad][:4])


def test_dense_then_matmul_meets_the_bar(env):
    """The materialised weight times x matches the oracle's GEMV."""
    import torch
    bisco, dev = env
    N, K, S, p = 512, 2048, 2, 21
    Lref = oracle.encode(synth.layer_weights(N, K, seed=7), S=S, p=p)
    X = synth.activations(3, K, seed=8)
    L = bisco.Layer.from_numpy(Lref, dev)
    W = bisco.bisco_decode_dense(L, "f32")
    x = to_dev(X, dev).view(torch.bfloat16).float()
    y = (x @ W.t()).cpu().numpy()
    assert max_rel_rows(y, oracle.gemv(Lref, X)) <= TOL


@pytest.mark.parametrize("N,K,S,p,dist", CASES)
def test_sequential_stage_decode_matches_oracle(env, N, K, S, p, dist):
    """bisco_decode_dense_stage stage after stage (the sequential residual
    decode): each stage term is rounded once to fp32 and added in stage
    order, S - 1 more fp32 roundings than the packed decode -- within
    S * 2^-23 relative of the oracle, protected columns exact."""
    import torch
    bisco, dev = env
    Lref = oracle.encode(synth.layer_weights(N, K, seed=N + K + S, dist=dist), S=S, p=p)
    ref = oracle.decode_rows(Lref)
    L = bisco.Layer.from_numpy(Lref, dev)
    got = bisco.bisco_decode_dense_sequential(L)
    torch.cuda.synchronize()
    assert bisco.bisco_get_device_error() == 0
    got = got.cpu().numpy().astype(np.float64)
    floor = 2.0 ** -40 * np.abs(ref).max()
    # each term |n16/sqrt(8)| is at most the chunk's largest |What| bound: use
    # the sum of term magnitudes, S * max term, as the scale of the rounding
    terms = np.zeros_like(ref)
    for s in range(S):
        n = Lref["norms"][s].view(np.float16).astype(np.float64)       # [N][K/8]
        terms += np.repeat(n, 8, axis=1) / np.sqrt(8.0)
    bad = np.abs(got - ref) > S * 2.0 ** -23 * terms + floor
    assert not bad.any(), (bad.sum(), got[bad][:4], ref[bad][:4])
    if p > 0:
        assert np.array_equal(got[:, Lref["idx"]], ref[:, Lref["idx"]])


def test_sequential_and_packed_decode_agree(env):
    import torch
    bisco, dev = env
    Lref = oracle.encode(synth.layer_weights(300, 1024, seed=77, dist="t4"), S=3, p=11)
    L = bisco.Layer.from_numpy(Lref, dev)
    seq = bisco.bisco_decode_dense_sequential(L)
    packed = bisco.bisco_decode_dense(L, "f32")
    torch.cuda.synchronize()
    d = (seq - packed).abs().max().item()
    assert d <= 4 * 2.0 ** -23 * packed.abs().max().item()


def test_stage_decode_rejects_a_stage_out_of_range(env):
    import torch
    bisco, dev = env
    Lref = oracle.encode(synth.layer_weights(16, 64, seed=5), S=2, p=1)
    L = bisco.Layer.from_numpy(Lref, dev)
    out = torch.empty((16, 64), dtype=torch.float32, device=dev)
    lib = bisco.load()
    import ctypes
    for st in (-1, 2):
        assert lib.bisco_decode_dense_stage(ctypes.byref(L.c), st, ctypes.c_void_p(out.data_ptr()), 0,
                                            None) == bisco.ERR_INVALID_ARG
