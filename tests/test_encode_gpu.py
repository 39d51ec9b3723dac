"""GPU encoder (bisco_encode) against the fp64 oracle: identical bytes."""
import numpy as np
import pytest

import oracle
from paper_2607_08643_gb300 import synth

from _helpers import to_dev

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


def gpu_encode(env, W, S, p, g=None):
    import torch
    bisco, dev = env
    gt = None if g is None else torch.from_numpy(np.ascontiguousarray(g, np.float32)).to(dev)
    L = bisco.bisco_encode(to_dev(W, dev), S, p, g=gt)
    torch.cuda.synchronize()
    return L, bisco.bisco_get_device_error()


def assert_same(got, ref):
    for k in ("codes", "norms", "q8", "scale", "idx"):
        assert got[k].shape == ref[k].shape, k
        if not np.array_equal(got[k], ref[k]):
            bad = np.argwhere(got[k] != ref[k])
            raise AssertionError("%s differs at %d places, first %s" % (k, len(bad), bad[:3].tolist()))


@pytest.mark.parametrize("N,K,S,p,dist,seed", [
    (1024, 1024, 2, 11, "normal", 0),     # single layer 1024 x 1024, 1 % protected
    (100, 1536, 3, 31, "t4", 5),          # ragged row count, S = 3
    (37, 136, 1, 0, "normal", 7),         # K % 128 != 0, no protection
    (64, 256, 3, 256, "normal", 8),       # every column protected
    (16, 8, 2, 1, "normal", 9),           # one chunk per row
    (3, 4104, 2, 50, "t4", 10),           # long rows, few of them
])
def test_encode_bit_exact(env, N, K, S, p, dist, seed):
    W = synth.layer_weights(N, K, seed=seed, dist=dist)
    L, err = gpu_encode(env, W, S, p)
    assert err == 0
    assert_same(L.to_numpy(), oracle.encode(W, S=S, p=p))


@pytest.mark.parametrize("name,S,rho", [("q_proj", 2, 1), ("k_proj", 2, 1),
                                        ("gate_proj", 3, 2), ("down_proj", 3, 2)])
def test_encode_bit_exact_full_size(env, name, S, rho):
    N, K = synth.QWEN3_8B_SHAPES[name]
    p = synth.protected_count(K, rho)
    W = synth.layer_weights(N, K, seed=11, dist="t4" if S == 3 else "normal")
    L, err = gpu_encode(env, W, S, p)
    assert err == 0
    assert_same(L.to_numpy(), oracle.encode(W, S=S, p=p))


def test_encode_with_calibration_statistic(env):
    W = synth.layer_weights(96, 512, seed=3)
    g = np.random.default_rng(4).uniform(0.1, 3.0, 512).astype(np.float32)
    L, err = gpu_encode(env, W, 2, 9, g=g)
    assert err == 0
    assert_same(L.to_numpy(), oracle.encode(W, S=2, p=9, g=g))


def test_encode_adversarial_chunks(env):
    """Zeros, -0.0, +-c*1, one-hot, equal-magnitude ties, bf16 subnormals,
    large finite values whose norms still fit fp16, tied column scores."""
    rows = []
    z = np.zeros(64, np.uint16)
    rows.append(z.copy())
    rows.append(np.full(64, 0x8000, np.uint16))                        # -0.0
    rows.append(np.where(np.arange(64) % 3, 0x3E80, 0xBE80).astype(np.uint16))  # +-0.25
    oh = z.copy(); oh[5] = 0x3F80; oh[63] = 0xBF80; rows.append(oh)    # one-hot +-1
    rows.append(np.arange(1, 65, dtype=np.uint16))                     # bf16 subnormals
    big = np.full(64, 0x4500, np.uint16)                               # 2048
    big[:8] = 0x4580                                                   # 4096: norm 11585 fits fp16
    rows.append(big)
    rows.append((np.arange(64) % 2 * 0x8000 | 0x3C00).astype(np.uint16))  # +-1 alternating
    W = np.stack(rows)
    for S, p in [(1, 0), (2, 4), (3, 9)]:
        L, err = gpu_encode(env, W, S, p)
        assert err == 0
        assert_same(L.to_numpy(), oracle.encode(W, S=S, p=p))


def test_encode_range_errors_latch_and_clear(env):
    bisco, _ = env
    big = np.full((2, 16), 0x7F7F, np.uint16)              # largest finite bf16
    L, err = gpu_encode(env, big, 1, 0)
    assert err == bisco.ERR_RANGE
    assert bisco.bisco_get_device_error() == 0               # cleared by the read
    inf = np.zeros((2, 16), np.uint16)
    inf[1, 3] = 0x7F80
    L, err = gpu_encode(env, inf, 2, 1)
    assert err == bisco.ERR_RANGE
    ok = synth.layer_weights(8, 64, seed=1)
    L, err = gpu_encode(env, ok, 2, 1)
    assert err == 0
