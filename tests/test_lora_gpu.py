"""bisco_lora_apply (the low-rank compensation of Sec. III-F) against the
fp64 oracle's lora_apply, and the compensation fused into the batch-1 GEMV
(bisco_gemv_lora, bisco_gemv_multi_lora) at the end of the file.

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

from _helpers import TOL, assert_parity, gemv_tight, max_rel_rows, to_dev

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


# ------------------------------------------ compensation fused into the GEMV
# bisco_gemv_lora / bisco_gemv_multi_lora: the batch-1 row-split kernel adds
# scale * Bm (A x) to each row it writes (t = A x formed in every CTA, in
# units of 8 ranks x 256 columns summed in a fixed order).  Against the
# oracle's layer output plus the oracle's compensation at the table decode's
# bound; against bisco_gemv + bisco_lora_apply (the same decode, the
# compensation's sums in another order) far inside it; the same bits on a
# second call.

def _fused(env, Lrefs, loras, X):
    import torch
    bisco, dev = env
    Ls = [bisco.Layer.from_numpy(L, dev) for L in Lrefs]
    dl = [None if r is None else (to_dev(r[0], dev), to_dev(r[1], dev), r[2]) for r in loras]
    xd = to_dev(X, dev)
    if len(Ls) == 1:
        ys = [bisco.bisco_gemv_lora(Ls[0], dl[0], xd)]
    else:
        ys = bisco.bisco_gemv_multi_lora(Ls, dl, xd)
    torch.cuda.synchronize()
    assert bisco.bisco_get_device_error() == 0
    return [y.cpu().numpy() for y in ys], Ls, dl, xd


@pytest.mark.parametrize("shapes", [
    [(4096, 41, 16, 0.5)],                                   # o_proj
    [(4096, 41, 16, 1.0), (1024, 41, 8, -2.0), (1024, 41, 0, 0.0)],   # q/k/v, v without one
    [(150, 5, 64, 0.25)],                                    # one row per CTA, largest rank
    [(12288, 41, 16, 1.0), (12288, 41, 32, 0.5)],            # gate/up: two CTAs per SM
])
def test_gemv_lora_fused_matches_oracle(env, shapes):
    import torch
    bisco, dev = env
    K, S = 4096, 2
    Lrefs, loras = [], []
    for i, (N, p, rank, scale) in enumerate(shapes):
        Lrefs.append(oracle.encode(synth.layer_weights(N, K, seed=600 + i), S=S, p=p))
        loras.append(None if rank == 0 else synth.lora_adapter(N, K, rank, seed=610 + i) + (scale,))
    X = synth.activations(1, K, seed=620)
    ys, Ls, dl, xd = _fused(env, Lrefs, loras, X)
    for y, L, r, Ld, rd in zip(ys, Lrefs, loras, Ls, dl):
        y0 = oracle.gemv(L, X)
        ref = y0 if r is None else oracle.lora_apply(r[0], r[1], X, y0, r[2])
        assert_parity(y, ref, gemv_tight(1))
        # the unfused chain: the same decode, then the two-kernel compensation
        yc = bisco.bisco_gemv(Ld, xd)
        if rd is not None:
            bisco.bisco_lora_apply(rd[0], rd[1], xd, yc, rd[2])
        torch.cuda.synchronize()
        assert max_rel_rows(y, yc.cpu().numpy()) <= 2e-6
    again, _, _, _ = _fused(env, Lrefs, loras, X)
    for y, y2 in zip(ys, again):
        assert np.array_equal(y, y2)


def test_gemv_lora_unsupported_shapes(env):
    """K other than 4096 is not taken by the fused kernel: UNSUPPORTED, and
    the two-kernel chain is the way to run it."""
    import torch
    bisco, dev = env
    Lref = oracle.encode(synth.layer_weights(256, 8192, seed=630), S=2, p=11)
    A, Bm = synth.lora_adapter(256, 8192, 16, seed=631)
    L = bisco.Layer.from_numpy(Lref, dev)
    x = to_dev(synth.activations(1, 8192, seed=632), dev)
    with pytest.raises(bisco.BiscoError) as e:
        bisco.bisco_gemv_lora(L, (to_dev(A, dev), to_dev(Bm, dev), 1.0), x)
    assert e.value.code == bisco.ERR_UNSUPPORTED
