"""Protected payloads in FP8 E4M3, FP8 E5M2 and BF16 on the GPU (the
protected-format ablation, variants of Eq. 10) against the fp64 oracle:
the encoder's bytes bit for bit, and GEMV / GEMM / dense decode with the
protected columns replaced by scale * value(q) -- or the protected rows
overwritten (Eq. 9's row axis) -- within the 2e-3 bar."""
import numpy as np
import pytest

import oracle
from paper_2607_08643_gb300 import synth

from _helpers import assert_parity, gemm_tight, gemv_tight, sample_rows, to_dev

pytestmark = pytest.mark.gpu

FORMATS = [oracle.FMT_E4M3, oracle.FMT_E5M2, oracle.FMT_BF16]


@pytest.fixture(scope="module")
def env():
    import torch
    import __graft_entry__
    __graft_entry__.build()
    from paper_2607_08643_gb300 import bisco
    dev = torch.device("cuda:0")
    torch.cuda.set_device(dev)
    return bisco, dev


def oracle_layer(W, S, p, fmt):
    """The oracle's layer with a protected payload in format fmt: stages and
    protected set of Eq. 8 / Eq. 3 / Eq. 5-7, payload of the format."""
    L = oracle.encode(W, S=S, p=p)
    q, scale = oracle.quantize_protected_fmt(W, L["idx"], fmt)
    return dict(L, q8=q, scale=scale, fmt=fmt)


def oracle_dense(L):
    base = dict(L, p=0, q8=np.zeros((L["N"], 0), np.int8), scale=np.zeros(0, np.uint16),
                idx=np.zeros(0, np.int32))
    What = oracle.decode_rows(base)
    if L["p"]:
        What[:, L["idx"]] = oracle.protected_values_fmt(L["q8"], L["scale"], L["fmt"])
    return What


@pytest.mark.parametrize("fmt", FORMATS)
@pytest.mark.parametrize("N,K,S,p,dist,seed", [
    (1024, 1024, 2, 11, "normal", 0), (100, 1536, 3, 31, "t4", 5), (37, 136, 1, 3, "normal", 7),
])
def test_encode_formats_bit_exact(env, fmt, N, K, S, p, dist, seed):
    import torch
    bisco, dev = env
    W = synth.layer_weights(N, K, seed=seed, dist=dist)
    L = bisco.bisco_encode(to_dev(W, dev), S, p, fmt=fmt)
    torch.cuda.synchronize()
    assert bisco.bisco_get_device_error() == 0
    got, ref = L.to_numpy(), oracle_layer(W, S, p, fmt)
    for k in ("codes", "norms", "q8", "scale", "idx"):
        assert got[k].dtype == ref[k].dtype and got[k].shape == ref[k].shape, k
        assert np.array_equal(got[k], ref[k]), k


@pytest.mark.parametrize("fmt", FORMATS)
@pytest.mark.parametrize("N,K,B", [(1024, 1024, 1), (1024, 1024, 16), (300, 4096, 4), (64, 136, 2)])
def test_gemv_formats_match_oracle(env, fmt, N, K, B):
    import torch
    bisco, dev = env
    p = synth.protected_count(K, 1)
    ref = oracle_layer(synth.layer_weights(N, K, seed=N + B), 2, p, fmt)
    L = bisco.Layer.from_numpy(ref, dev)
    x = synth.activations(B, K, seed=B)
    y = bisco.bisco_gemv(L, to_dev(x, dev))
    torch.cuda.synchronize()
    assert bisco.bisco_get_device_error() == 0
    assert_parity(y.cpu().numpy(), oracle.matmul(oracle_dense(ref), x), gemv_tight(B))


@pytest.mark.parametrize("fmt", FORMATS)
@pytest.mark.parametrize("N,K", [(1000, 4096), (300, 8192)])
def test_gemv_batch1_kernel_formats_match_oracle(env, fmt, N, K):
    """Batch 1 with K a multiple of 4096: the row-split kernel takes the
    payload format itself (value(q) * scale * x in its protected term, one
    launch), against the oracle at the table decode's bound; the same bits
    on a second call."""
    import torch
    bisco, dev = env
    p = synth.protected_count(K, 2)
    ref = oracle_layer(synth.layer_weights(N, K, seed=N + 3), 2, p, fmt)
    L = bisco.Layer.from_numpy(ref, dev)
    x = synth.activations(1, K, seed=7)
    y = bisco.bisco_gemv(L, to_dev(x, dev))
    y2 = bisco.bisco_gemv(L, to_dev(x, dev))
    torch.cuda.synchronize()
    assert bisco.bisco_get_device_error() == 0
    assert_parity(y.cpu().numpy(), oracle.matmul(oracle_dense(ref), x), gemv_tight(1))
    assert torch.equal(y, y2)


def test_gemv_multi_batch1_mixed_formats(env):
    """q/k/v-like group at batch 1 with INT8, E4M3 and bf16 payloads in one
    launch of the row-split kernel."""
    import torch
    bisco, dev = env
    K = 4096
    refs = [oracle_layer(synth.layer_weights(N, K, seed=70 + i), 2, 41, fmt)
            for i, (N, fmt) in enumerate([(1500, oracle.FMT_INT8), (512, oracle.FMT_E4M3),
                                           (700, oracle.FMT_BF16)])]
    Ls = [bisco.Layer.from_numpy(r, dev) for r in refs]
    x = synth.activations(1, K, seed=71)
    ys = bisco.bisco_gemv_multi(Ls, to_dev(x, dev))
    torch.cuda.synchronize()
    assert bisco.bisco_get_device_error() == 0
    for y, r in zip(ys, refs):
        assert_parity(y.cpu().numpy(), oracle.matmul(oracle_dense(r), x), gemv_tight(1))


@pytest.mark.parametrize("fmt", FORMATS)
def test_gemm_and_multi_formats_match_oracle(env, fmt):
    import torch
    bisco, dev = env
    K = 1024
    ref = oracle_layer(synth.layer_weights(512, K, seed=3), 2, 11, fmt)
    ref8 = oracle.encode(synth.layer_weights(256, K, seed=4), S=2, p=11)
    L, L8 = bisco.Layer.from_numpy(ref, dev), bisco.Layer.from_numpy(ref8, dev)
    X = synth.activations(300, K, seed=5)
    Y = bisco.bisco_gemm(L, to_dev(X, dev))
    x = synth.activations(8, K, seed=6)
    ys = bisco.bisco_gemv_multi([L, L8], to_dev(x, dev))
    torch.cuda.synchronize()
    assert bisco.bisco_get_device_error() == 0
    assert_parity(Y.cpu().numpy(), oracle.matmul(oracle_dense(ref), X), gemm_tight(300, K))
    assert_parity(ys[0].cpu().numpy(), oracle.matmul(oracle_dense(ref), x), gemv_tight(8))
    assert_parity(ys[1].cpu().numpy(), oracle.matmul(oracle.decode_rows(ref8), x), gemv_tight(8))


@pytest.mark.parametrize("fmt", FORMATS)
def test_decode_dense_formats(env, fmt):
    import torch
    bisco, dev = env
    ref = oracle_layer(synth.layer_weights(200, 512, seed=9), 3, 9, fmt)
    L = bisco.Layer.from_numpy(ref, dev)
    out = bisco.bisco_decode_dense(L, "f32")
    torch.cuda.synchronize()
    assert bisco.bisco_get_device_error() == 0
    got = out.cpu().numpy().astype(np.float64)
    want = oracle_dense(ref)
    idx = ref["idx"]
    assert np.array_equal(got[:, idx], want[:, idx])        # scale * value(q): exact in fp32
    keep = np.setdiff1d(np.arange(512), idx)
    assert np.abs(got[:, keep] - want[:, keep]).max() <= 2.0 ** -22 * np.abs(want[:, keep]).max()


def test_full_size_q_proj_e4m3_sampled(env):
    import torch
    bisco, dev = env
    N, K = synth.QWEN3_8B_SHAPES["q_proj"]
    p = synth.protected_count(K, 1)
    W = synth.layer_weights(N, K, seed=41)
    ref = oracle_layer(W, 2, p, oracle.FMT_E4M3)
    L = bisco.Layer.from_numpy(ref, dev)
    rows = sample_rows(N)
    for B in (1, 16):
        x = synth.activations(B, K, seed=42 + B)
        y = bisco.bisco_gemv(L, to_dev(x, dev))
        torch.cuda.synchronize()
        assert bisco.bisco_get_device_error() == 0
        want = np.stack([oracle.matmul(oracle_dense(dict(ref, codes=ref["codes"][:, r:r + 1],
                                                         norms=ref["norms"][:, r:r + 1],
                                                         q8=ref["q8"][r:r + 1], N=1)), x)[:, 0]
                         for r in rows], axis=1)
        assert_parity(y.cpu().numpy()[:, rows], want, gemv_tight(B))


def oracle_rows_layer(W, S, p, fmt, idx=None):
    L = oracle.encode_rows(W, S, p, idx=idx)
    q, scale = oracle.quantize_protected_rows_fmt(W, L["idx"], fmt)
    return dict(L, q8=q, scale=scale, fmt=fmt)


def oracle_rows_dense(L):
    """Stages of the row-masked weight, protected rows = scale * value(q)."""
    N, K, p = L["N"], L["K"], L["p"]
    base = dict(L, p=0, axis=0, q8=np.zeros((N, 0), np.int8), scale=np.zeros(0, np.uint16),
                idx=np.zeros(0, np.int32))
    What = oracle.decode_rows(base)
    if p:
        qc = np.zeros((K, oracle.pad16(p)), L["q8"].dtype)        # rows as protected columns
        qc[:, :p] = L["q8"][:, :K].T
        What[L["idx"]] = oracle.protected_values_fmt(qc, L["scale"], L["fmt"]).T
    return What


@pytest.mark.parametrize("fmt", FORMATS)
def test_encode_rows_formats_bit_exact(env, fmt):
    import torch
    bisco, dev = env
    for (N, K, S, p, seed) in ((300, 1024, 2, 3, 1), (64, 136, 3, 5, 2)):
        W = synth.layer_weights(N, K, seed=seed)
        Wd = to_dev(W, dev)
        L = bisco.bisco_encode(Wd, S, p, axis=1, fmt=fmt)
        idx = torch.tensor([1, 7, N - 1], dtype=torch.int32, device=dev)
        Lg = bisco.bisco_encode_with_set(Wd, S, idx, axis=1, fmt=fmt)
        torch.cuda.synchronize()
        assert bisco.bisco_get_device_error() == 0
        for got, ref in ((L.to_numpy(), oracle_rows_layer(W, S, p, fmt)),
                         (Lg.to_numpy(), oracle_rows_layer(W, S, 3, fmt, idx=[1, 7, N - 1]))):
            for k in ("codes", "norms", "q8", "scale", "idx"):
                assert got[k].dtype == ref[k].dtype and np.array_equal(got[k], ref[k]), k


@pytest.mark.parametrize("fmt", FORMATS)
@pytest.mark.parametrize("K", [1024, 4096])
def test_gemv_gemm_rows_formats_match_oracle(env, fmt, K):
    """Protected rows in each payload format; at K = 4096 batch 1 goes to the
    row-split kernel (the rows' payload dot products after its decode)."""
    import torch
    bisco, dev = env
    N = 512
    ref = oracle_rows_layer(synth.layer_weights(N, K, seed=61), 2, 6, fmt)
    L = bisco.Layer.from_numpy(ref, dev)
    What = oracle_rows_dense(ref)
    for M in (1, 16, 300):
        X = synth.activations(M, K, seed=62 + M)
        Y = bisco.bisco_gemv(L, to_dev(X, dev)) if M <= 16 else bisco.bisco_gemm(L, to_dev(X, dev))
        torch.cuda.synchronize()
        assert bisco.bisco_get_device_error() == 0
        assert_parity(Y.cpu().numpy(), oracle.matmul(What, X),
                      gemv_tight(M) if M <= 16 else gemm_tight(M, K))
    out = bisco.bisco_decode_dense(L, "f32")
    torch.cuda.synchronize()
    got = out.cpu().numpy().astype(np.float64)
    assert np.array_equal(got[ref["idx"]], What[ref["idx"]])     # scale * value(q): exact in fp32
