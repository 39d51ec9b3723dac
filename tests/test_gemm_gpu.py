"""bisco_gemm (prefill) against the fp64 oracle, and against bisco_gemv."""
import numpy as np
import pytest

import oracle
from paper_2607_08643_gb300 import synth

from _helpers import assert_parity, gemm_tight, max_rel_rows, rows_per_tile, sample_rows, to_dev

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


def run_gemm(env, Lref, X):
    import torch
    bisco, dev = env
    L = bisco.Layer.from_numpy(Lref, dev)
    Y = bisco.bisco_gemm(L, to_dev(X, dev))
    torch.cuda.synchronize()
    assert bisco.bisco_get_device_error() == 0
    return Y.cpu().numpy(), L


@pytest.mark.parametrize("N,K,S,p,M", [
    (1024, 1024, 2, 11, 2048),      # single layer 1024 x 1024, 2048 tokens (tensor cores)
    (1024, 1024, 2, 11, 37),        # 37 tokens: tensor cores, one 128-token tile
    (512, 1024, 2, 11, 16),         # 16 tokens: decode kernels
    (384, 2048, 3, 41, 17),         # 17 tokens: tensor cores
    (1024, 4096, 2, 41, 64),        # 64 tokens: tensor cores, stream-K
    (200, 1536, 3, 20, 130),        # ragged N and M, three stages
    (128, 512, 1, 0, 100),          # S = 1, no protected columns
    (384, 2048, 2, 130, 300),       # three 64-column protected blocks, two token tiles
    (96, 512, 2, 512, 80),          # every column protected
    (256, 12288, 2, 123, 260),      # K = 12288 (down_proj width)
    (64, 1000, 2, 10, 90),          # K % 128 != 0: decode kernels
    (128, 512, 1, 0, 1),            # one token
])
def test_gemm_matches_oracle(env, N, K, S, p, M):
    W = synth.layer_weights(N, K, seed=N ^ K)
    X = synth.activations(M, K, seed=M)
    Lref = oracle.encode(W, S=S, p=p)
    Y, _ = run_gemm(env, Lref, X)
    assert_parity(Y, oracle.gemv(Lref, X), gemm_tight(M, K))


@pytest.mark.parametrize("name", ["q_proj", "k_proj", "gate_proj", "up_proj", "down_proj"])
def test_gemm_full_size_sampled(env, name):
    """Every Qwen3-8B shape at 2048 tokens.  gate/up (12288 x 4096: 768
    tiles of 128 features x 256 tokens) make each persistent CTA walk five or
    six tiles; the sample takes two features of every 128-feature tile and
    five tokens of every 256-token tile, so every tile is checked."""
    N, K = synth.QWEN3_8B_SHAPES[name]
    S, p = 2, synth.protected_count(K, 1)
    W = synth.layer_weights(N, K, seed=23 + N % 7)
    X = synth.activations(2048, K, seed=24)
    Lref = oracle.encode(W, S=S, p=p)
    Y, _ = run_gemm(env, Lref, X)
    rows = rows_per_tile(N, 128, per=2, seed=N)
    toks = rows_per_tile(2048, 256, per=5, seed=1)
    ref = oracle.apply_rows(Lref, rows, X[toks])
    assert_parity(Y[toks][:, rows], ref, gemm_tight(2048, K), name)


@pytest.mark.parametrize("N,K,S,p,M", [
    (4096, 256, 2, 3, 4096),        # 512 tiles: every CTA runs three or four
    (2048, 512, 3, 6, 8192),        # 512 tiles, three stages
    (1152, 384, 1, 0, 8000),        # ragged last token tile, S = 1, no protection
])
def test_gemm_many_tiles_per_cta(env, N, K, S, p, M):
    """Far more tiles than SMs at small K: accumulator reuse, the TMEM
    phases and the rings carried from tile to tile, checked on every
    output feature against 320 tokens spread over all token tiles."""
    W = synth.layer_weights(N, K, seed=N + K + M)
    X = synth.activations(M, K, seed=M + 1)
    Lref = oracle.encode(W, S=S, p=p)
    Y, _ = run_gemm(env, Lref, X)
    toks = rows_per_tile(M, 256, per=10, seed=M)
    ref = oracle.gemv(Lref, X[toks])
    assert_parity(Y[toks], ref, gemm_tight(M, K), f"{N}x{K} M={M}")


def test_gemm_equals_gemv(env):
    import torch
    bisco, dev = env
    N, K, S, p = 512, 2048, 2, 21
    W = synth.layer_weights(N, K, seed=31)
    X = synth.activations(16, K, seed=32)
    Lref = oracle.encode(W, S=S, p=p)
    Y, L = run_gemm(env, Lref, X)
    y = bisco.bisco_gemv(L, to_dev(X, dev)).cpu().numpy()
    assert max_rel_rows(Y, y) <= 1e-4


@pytest.mark.parametrize("N,K,S,p,M", [
    (128, 4096, 2, 41, 200),        # one tile of 33 k-steps, split over 4 CTAs
    (256, 4096, 3, 41, 100),        # M <= 128: 128-token tiles, 2 tiles over 8 CTAs
    (1024, 4096, 2, 41, 2048),      # k_proj: 64 tiles over every SM, 2-3 pieces a tile
])
def test_gemm_split_tiles(env, N, K, S, p, M):
    """Tiles split between CTAs by the stream-K schedule, the partial sums
    added by the warp that brings a tile's last piece: the outputs against
    the oracle (every token up to 200, 5 tokens of every 256 beyond), and a
    second call equal bit for bit (the pieces are summed in CTA order)."""
    W = synth.layer_weights(N, K, seed=N + 7 * K)
    X = synth.activations(M, K, seed=M + 3)
    Lref = oracle.encode(W, S=S, p=p)
    Y, _ = run_gemm(env, Lref, X)
    Y2, _ = run_gemm(env, Lref, X)
    assert np.array_equal(Y, Y2)
    toks = np.arange(M) if M <= 200 else rows_per_tile(M, 256, per=5, seed=M)
    ref = oracle.gemv(Lref, X[toks])
    assert_parity(Y[toks], ref, gemm_tight(M, K), f"{N}x{K} M={M}")
