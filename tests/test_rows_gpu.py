"""Output-row protection and the coupled MLP set on the GPU (Sec. III-E
Eq. 9, Eq. 10 on rows) against the fp64 oracle: the encoder's bytes
bit for bit, the coupled selection exactly, and the row-protected
GEMV / GEMM / dense decode within the 2e-3 parity bar."""
import numpy as np
import pytest

import oracle
from paper_2607_08643_gb300 import synth

from _helpers import assert_parity, gemm_tight, gemv_tight, to_dev

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


def _outlier_rows(N, K, seed, dist="normal"):
    """Weights with 4 output rows scaled x20 (the rows Eq. 9 should pick)."""
    W = synth.layer_weights(N, K, seed=seed, dist=dist)
    f = synth.bf16_bits_to_f32(W).astype(np.float64)
    rng = np.random.default_rng(seed + 1)
    rows = rng.choice(N, size=min(4, N), replace=False)
    f[rows] *= 20.0
    return synth.f32_to_bf16_bits(f.astype(np.float32))


def assert_same(got, ref):
    for k in ("codes", "norms", "q8", "scale", "idx"):
        assert got[k].shape == ref[k].shape, (k, got[k].shape, ref[k].shape)
        if not np.array_equal(got[k], ref[k]):
            bad = np.argwhere(got[k] != ref[k])
            raise AssertionError("%s differs at %d places, first %s" % (k, len(bad), bad[:3].tolist()))


def gpu_encode_rows(env, W, S, p, g=None):
    import torch
    bisco, dev = env
    gt = None if g is None else torch.from_numpy(np.ascontiguousarray(g, np.float32)).to(dev)
    L = bisco.bisco_encode(to_dev(W, dev), S, p, g=gt, axis=1)
    torch.cuda.synchronize()
    return L, bisco.bisco_get_device_error()


@pytest.mark.parametrize("N,K,S,p,dist,seed", [
    (300, 1024, 2, 3, "normal", 1),       # 1 % of the rows, several tiles
    (64, 136, 2, 3, "normal", 2),         # K % 128 != 0
    (100, 1536, 3, 31, "t4", 3),          # S = 3, ragged row count
    (16, 64, 1, 16, "normal", 4),         # every row protected
    (37, 64, 2, 0, "normal", 5),          # no protection
    (2049, 8, 2, 21, "normal", 6),        # one chunk per row, rows > compaction threads
])
def test_encode_rows_bit_exact(env, N, K, S, p, dist, seed):
    W = _outlier_rows(N, K, seed, dist)
    L, err = gpu_encode_rows(env, W, S, p)
    assert err == 0
    assert_same(L.to_numpy(), oracle.encode_rows(W, S, p))


def test_encode_rows_with_weights_g(env):
    N, K, S, p = 256, 512, 2, 7
    W = _outlier_rows(N, K, 11)
    g = np.random.default_rng(12).uniform(0.5, 2.0, N).astype(np.float32)
    L, err = gpu_encode_rows(env, W, S, p, g=g)
    assert err == 0
    assert_same(L.to_numpy(), oracle.encode_rows(W, S, p, g=g))


def test_encode_rows_full_size_gate_proj(env):
    N, K = synth.QWEN3_8B_SHAPES["gate_proj"]
    p = synth.protected_count(N, 1)
    W = synth.layer_weights(N, K, seed=21, dist="t4")
    L, err = gpu_encode_rows(env, W, 2, p)
    assert err == 0
    assert_same(L.to_numpy(), oracle.encode_rows(W, 2, p))


@pytest.mark.parametrize("F,H,p,weighted", [(192, 64, 6, False), (3000, 40, 30, True),
                                            (64, 16, 64, False), (50, 24, 0, False)])
def test_select_coupled_matches_oracle(env, F, H, p, weighted):
    import torch
    bisco, dev = env
    Wg = synth.layer_weights(F, H, seed=31)
    Wu = synth.layer_weights(F, H, seed=32)
    Wd = synth.layer_weights(H, F, seed=33)
    gs = [None, None, None]
    if weighted:
        rng = np.random.default_rng(34)
        gs = [rng.uniform(0.5, 2.0, F).astype(np.float32) for _ in range(3)]
    gd = [None if g is None else torch.from_numpy(g).to(dev) for g in gs]
    idx = bisco.bisco_select_coupled(to_dev(Wg, dev), to_dev(Wu, dev), to_dev(Wd, dev), p,
                                     gg=gd[0], gu=gd[1], gd=gd[2])
    torch.cuda.synchronize()
    assert bisco.bisco_get_device_error() == 0
    ref = oracle.select_coupled(Wg, Wu, Wd, p, gg=gs[0], gu=gs[1], gd=gs[2])[0]
    assert np.array_equal(idx.cpu().numpy(), np.asarray(ref, np.int32))


def test_coupled_mlp_encode_matches_oracle(env):
    """gate/up rows and down columns on the one coupled set."""
    import torch
    bisco, dev = env
    F, H, S, p = 384, 128, 2, 8
    Wg = synth.layer_weights(F, H, seed=41)
    Wu = synth.layer_weights(F, H, seed=42)
    Wd = synth.layer_weights(H, F, seed=43)
    idx = bisco.bisco_select_coupled(to_dev(Wg, dev), to_dev(Wu, dev), to_dev(Wd, dev), p)
    Lg = bisco.bisco_encode_with_set(to_dev(Wg, dev), S, idx, axis=1)
    Lu = bisco.bisco_encode_with_set(to_dev(Wu, dev), S, idx, axis=1)
    Ld = bisco.bisco_encode_with_set(to_dev(Wd, dev), S, idx, axis=0)
    torch.cuda.synchronize()
    assert bisco.bisco_get_device_error() == 0
    rg, ru, rd = oracle.encode_coupled(Wg, Wu, Wd, S, p)
    assert_same(Lg.to_numpy(), rg)
    assert_same(Lu.to_numpy(), ru)
    assert_same(Ld.to_numpy(), rd)


def test_encode_with_set_rejects_bad_sets_on_the_device(env):
    """Out-of-order and out-of-range indices latch INVALID_ARG; an
    out-of-range one is stored as 0, so nothing reads outside the weight."""
    import torch
    bisco, dev = env
    N, K = 64, 128
    W = to_dev(synth.layer_weights(N, K, seed=51), dev)
    for axis, bad in ((1, [5, 3]), (1, [2, N + 7]), (0, [9, 9]), (0, [-1, 4])):
        idx = torch.tensor(bad, dtype=torch.int32, device=dev)
        L = bisco.bisco_encode_with_set(W, 2, idx, axis=axis)
        torch.cuda.synchronize()
        assert bisco.bisco_get_device_error() == bisco.ERR_INVALID_ARG
        stored = L.idx[:2].cpu().numpy()
        n = N if axis == 1 else K
        assert np.all((stored >= 0) & (stored < n))


def _row_layer(env, N, K, S, p, seed):
    bisco, dev = env
    W = _outlier_rows(N, K, seed)
    ref = oracle.encode_rows(W, S, p)
    return bisco.Layer.from_numpy(ref, dev), ref


@pytest.mark.parametrize("N,K,S,p,B", [
    (1024, 1024, 2, 11, 1), (1024, 1024, 2, 11, 16), (300, 4096, 2, 3, 4),
    (64, 136, 2, 3, 2), (48, 256, 3, 48, 1), (4096, 512, 2, 0, 8),
    # batch 1, K a multiple of 4096: the row-split kernel takes the rows
    (1000, 4096, 2, 10, 1), (300, 8192, 3, 30, 1), (48, 4096, 2, 48, 1),
])
def test_gemv_rows_matches_oracle(env, N, K, S, p, B):
    import torch
    bisco, dev = env
    L, ref = _row_layer(env, N, K, S, p, seed=60 + N % 7)
    x = synth.activations(B, K, seed=61)
    y = bisco.bisco_gemv(L, to_dev(x, dev))
    torch.cuda.synchronize()
    assert bisco.bisco_get_device_error() == 0
    yr = oracle.matmul(oracle.decode_rows(ref), x)
    assert_parity(y.cpu().numpy(), yr, gemv_tight(B))
    if p:
        # the protected rows alone: int8 x bf16 summed in fp32
        got = y.cpu().numpy()[:, ref["idx"]].astype(np.float64)
        want = yr[:, ref["idx"]]
        bound = K * 2.0 ** -23 * (np.abs(oracle.decode_rows(ref)[ref["idx"]]) @
                                  np.abs(synth.bf16_bits_to_f32(x).astype(np.float64)).T).T
        assert np.all(np.abs(got - want) <= bound + 1e-30)


@pytest.mark.parametrize("K", [1024, 4096])
def test_gemv_multi_mixes_row_and_column_layers(env, K):
    import torch
    bisco, dev = env
    S = 2
    Lr, rr = _row_layer(env, 512, K, S, 6, seed=71)
    Wc = synth.layer_weights(256, K, seed=72)
    rc = oracle.encode(Wc, S=S, p=11)
    Lc = bisco.Layer.from_numpy(rc, dev)
    for B in (1, 8, 16):
        x = synth.activations(B, K, seed=73 + B)
        ys = bisco.bisco_gemv_multi([Lr, Lc, Lr], to_dev(x, dev))
        torch.cuda.synchronize()
        assert bisco.bisco_get_device_error() == 0
        for y, ref in zip(ys, (rr, rc, rr)):
            assert_parity(y.cpu().numpy(), oracle.matmul(oracle.decode_rows(ref), x), gemv_tight(B))


@pytest.mark.parametrize("N,K,M", [(512, 1024, 300), (256, 512, 40), (384, 136, 130)])
def test_gemm_rows_matches_oracle(env, N, K, M):
    import torch
    bisco, dev = env
    L, ref = _row_layer(env, N, K, 2, 5, seed=80 + M)
    X = synth.activations(M, K, seed=81)
    Y = bisco.bisco_gemm(L, to_dev(X, dev))
    torch.cuda.synchronize()
    assert bisco.bisco_get_device_error() == 0
    assert_parity(Y.cpu().numpy(), oracle.matmul(oracle.decode_rows(ref), X), gemm_tight(M, K))


@pytest.mark.parametrize("dtype", ["f32", "bf16", "f16"])
def test_decode_dense_rows(env, dtype):
    import torch
    bisco, dev = env
    L, ref = _row_layer(env, 200, 256, 2, 4, seed=90)
    out = bisco.bisco_decode_dense(L, dtype)
    torch.cuda.synchronize()
    assert bisco.bisco_get_device_error() == 0
    got = out.float().cpu().numpy().astype(np.float64)
    want = oracle.decode_rows(ref)
    idx = ref["idx"]
    sc = ref["scale"].view(np.float16).astype(np.float32)[:, None]
    prot = (sc * ref["q8"][:, :256].astype(np.float32))          # exact in fp32
    if dtype == "f32":
        assert np.array_equal(got[idx], prot.astype(np.float64))
    else:
        tdt = torch.bfloat16 if dtype == "bf16" else torch.float16
        once = torch.from_numpy(prot).to(tdt).float().numpy().astype(np.float64)
        assert np.array_equal(got[idx], once)                   # one rounding of the exact value
    keep = np.setdiff1d(np.arange(200), idx)
    rel = np.abs(got[keep] - want[keep]).max() / np.abs(want[keep]).max()
    assert rel <= (2.0 ** -22 if dtype == "f32" else 2.0 ** -7)


def test_full_size_gate_proj_rows_sampled(env):
    """gate_proj 12288 x 4096 with 1 % of its rows protected, batch 1 and
    16, checked on sampled rows (all protected rows among them)."""
    import torch
    bisco, dev = env
    N, K = synth.QWEN3_8B_SHAPES["gate_proj"]
    p = synth.protected_count(N, 1)
    W = synth.layer_weights(N, K, seed=95, dist="t4")
    ref = oracle.encode_rows(W, 2, p)
    L = bisco.Layer.from_numpy(ref, dev)
    rows = np.unique(np.concatenate([ref["idx"], np.arange(0, N, 997)]))
    for B in (1, 16):
        x = synth.activations(B, K, seed=96 + B)
        y = bisco.bisco_gemv(L, to_dev(x, dev))
        torch.cuda.synchronize()
        assert bisco.bisco_get_device_error() == 0
        want = np.stack([oracle.matmul(oracle.decode_rows(ref, row0=int(r), nrows=1), x)[:, 0]
                         for r in rows], axis=1)
        assert_parity(y.cpu().numpy()[:, rows], want, gemv_tight(B))
