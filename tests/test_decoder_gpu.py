"""The learned decoder step in table form on the GPU (Eq. 1 decoded per
Eq. 12) against the fp64 oracle: bisco_gemv_table within the 2e-3 bar and
bisco_decode_dense_table within its rounding bound, for linear and
sign-symmetric perceptron decoders with random weights."""
import math

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


def mlp_tables(S, seed, hdim=16, residual=True):
    rng = np.random.default_rng(seed)
    out = []
    for _ in range(S):
        W1 = rng.normal(0, 1.0, (hdim, 8))
        W2 = rng.normal(0, 1.0 / math.sqrt(hdim), (8, hdim))
        Wr = rng.normal(0, 0.5 / math.sqrt(hdim), (hdim, hdim)) if residual else None
        out.append(oracle.table_to_fp16(oracle.decoder_table_mlp(W1, W2, Wr)))
    return np.stack(out)


def linear_tables(S, seed):
    rng = np.random.default_rng(seed)
    return np.stack([oracle.table_to_fp16(oracle.decoder_table_linear(rng.normal(0, 1, (8, 8))))
                     for _ in range(S)])


@pytest.mark.parametrize("N,K,S,p,B,kind", [
    (1024, 1024, 2, 11, 1, "mlp"), (1024, 1024, 2, 11, 16, "linear"),
    (300, 4096, 3, 41, 4, "mlp"), (64, 136, 2, 3, 2, "linear"), (96, 512, 1, 0, 8, "mlp"),
])
def test_gemv_table_matches_oracle(env, N, K, S, p, B, kind):
    import torch
    bisco, dev = env
    W = synth.layer_weights(N, K, seed=N + K)
    ref = oracle.encode(W, S=S, p=p)
    L = bisco.Layer.from_numpy(ref, dev)
    tabs = mlp_tables(S, seed=K) if kind == "mlp" else linear_tables(S, seed=K)
    x = synth.activations(B, K, seed=5)
    y = bisco.bisco_gemv_table(L, to_dev(tabs, dev), to_dev(x, dev))
    torch.cuda.synchronize()
    assert bisco.bisco_get_device_error() == 0
    want = oracle.matmul(oracle.decode_rows_table(ref, tabs), x)
    assert max_rel_rows(y.cpu().numpy(), want) <= TOL


@pytest.mark.parametrize("N,K,S,p,kind", [
    (1000, 4096, 2, 41, "mlp"), (4096, 4096, 2, 41, "linear"), (300, 8192, 3, 82, "linear"),
    (150, 4096, 1, 0, "mlp"),
])
def test_gemv_table_batch1_kernel(env, N, K, S, p, kind, monkeypatch):
    """Batch 1 with K a multiple of 4096: the row-split kernel in table mode
    (the span's activations and the S tables in shared memory; fp16 x fp16
    products, exact, summed in fp32).  Against the oracle far inside the
    bar (fp32 sums over K terms), against the one-warp-per-row kernel
    (BISCO_GEMV_MODE forces it), and the same bits on a second call."""
    import torch
    bisco, dev = env
    ref = oracle.encode(synth.layer_weights(N, K, seed=N + 17), S=S, p=p)
    L = bisco.Layer.from_numpy(ref, dev)
    tabs = mlp_tables(S, seed=K + 1) if kind == "mlp" else linear_tables(S, seed=K + 1)
    x = synth.activations(1, K, seed=6)
    td, xd = to_dev(tabs, dev), to_dev(x, dev)
    y = bisco.bisco_gemv_table(L, td, xd)
    y2 = bisco.bisco_gemv_table(L, td, xd)
    monkeypatch.setenv("BISCO_GEMV_MODE", "stream")
    y_rows = bisco.bisco_gemv_table(L, td, xd)
    torch.cuda.synchronize()
    assert bisco.bisco_get_device_error() == 0
    want = oracle.matmul(oracle.decode_rows_table(ref, tabs), x)
    assert max_rel_rows(y.cpu().numpy(), want) <= 2e-5
    assert max_rel_rows(y.cpu().numpy(), y_rows.cpu().numpy()) <= 2e-5
    assert torch.equal(y, y2)


def test_identity_table_is_the_norm_rescale_decoder(env):
    """The binary16 table of +-1/sqrt(8) gives bisco_gemv's result up to the
    table's rounding (|fp16(1/sqrt 8) - 1/sqrt 8| relative, about 1.6e-4)."""
    import torch
    bisco, dev = env
    N, K, S, p = 512, 2048, 2, 21
    ref = oracle.encode(synth.layer_weights(N, K, seed=7), S=S, p=p)
    L = bisco.Layer.from_numpy(ref, dev)
    ident = np.array([[oracle.double_to_fp16((-1.0 if (v >> k) & 1 else 1.0) / math.sqrt(8.0))
                       for k in range(8)] for v in range(256)], np.uint16)
    tabs = np.stack([ident] * S)
    x = synth.activations(3, K, seed=8)
    y_tab = bisco.bisco_gemv_table(L, to_dev(tabs, dev), to_dev(x, dev))
    y = bisco.bisco_gemv(L, to_dev(x, dev))
    torch.cuda.synchronize()
    assert bisco.bisco_get_device_error() == 0
    assert max_rel_rows(y_tab.cpu().numpy(), y.cpu().numpy()) <= 1e-3
    assert max_rel_rows(y_tab.cpu().numpy(), oracle.matmul(oracle.decode_rows_table(ref, tabs), x)) <= TOL


@pytest.mark.parametrize("dtype", ["f32", "bf16", "f16"])
def test_decode_dense_table_matches_oracle(env, dtype):
    import torch
    bisco, dev = env
    N, K, S, p = 200, 512, 3, 9
    ref = oracle.encode(synth.layer_weights(N, K, seed=9, dist="t4"), S=S, p=p)
    L = bisco.Layer.from_numpy(ref, dev)
    tabs = mlp_tables(S, seed=10)
    out = bisco.bisco_decode_dense_table(L, to_dev(tabs, dev), dtype)
    torch.cuda.synchronize()
    assert bisco.bisco_get_device_error() == 0
    got = out.float().cpu().numpy().astype(np.float64)
    want = oracle.decode_rows_table(ref, tabs)
    absmag = oracle.decode_rows_table(ref, tabs & 0x7FFF)      # sum_s n_s |T_s|, norms >= 0
    bsq = np.ones(K, bool)
    bsq[ref["idx"]] = False
    # fp16 x fp16 products are exact in fp32; S - 1 fp32 additions
    bound = (S - 1) * 2.0 ** -24 * absmag[:, bsq]
    if dtype == "bf16":
        bound = bound + 2.0 ** -8 * np.abs(want[:, bsq]) + 2.0 ** -133
    elif dtype == "f16":
        bound = bound + 2.0 ** -11 * np.abs(want[:, bsq]) + 2.0 ** -25
    assert np.all(np.abs(got[:, bsq] - want[:, bsq]) <= bound)
    sc = ref["scale"].view(np.float16).astype(np.float32)[None, :]
    prot = sc * ref["q8"][:, :p].astype(np.float32)                  # exact in fp32
    tdt = {"f32": torch.float32, "bf16": torch.bfloat16, "f16": torch.float16}[dtype]
    once = torch.from_numpy(prot).to(tdt).float().numpy().astype(np.float64)
    assert np.array_equal(got[:, ref["idx"]], once)


def test_gemv_table_row_protected_layer(env):
    import torch
    bisco, dev = env
    N, K, S, p = 384, 1024, 2, 4
    W = synth.layer_weights(N, K, seed=11)
    ref = oracle.encode_rows(W, S, p)
    L = bisco.Layer.from_numpy(ref, dev)
    tabs = mlp_tables(S, seed=12)
    x = synth.activations(2, K, seed=13)
    y = bisco.bisco_gemv_table(L, to_dev(tabs, dev), to_dev(x, dev))
    torch.cuda.synchronize()
    assert bisco.bisco_get_device_error() == 0
    stages = dict(ref, p=0, axis=0, q8=np.zeros((N, 0), np.int8),
                  scale=np.zeros(0, np.uint16), idx=np.zeros(0, np.int32))
    What = oracle.decode_rows_table(stages, tabs)
    What[ref["idx"]] = oracle.decode_rows(ref)[ref["idx"]]           # scale * q8 rows
    assert max_rel_rows(y.cpu().numpy(), oracle.matmul(What, x)) <= TOL
