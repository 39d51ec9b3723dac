"""Property tests of the fp64 oracle over generated small layers (no GPU;
hypothesis searches for edge cases: ties, zero and signed-zero chunks,
every column protected, single chunks).

Weights are dyadic (k/8 with |k| <= 64, both zero signs), so every sum of
squares is exact in binary64 and a numpy computation written from the
paper's definitions can be compared bit for bit:
  Eq. 8   the protected set is the top-p columns by L2 norm, ties to the
          lower index, stored ascending;
  Eq. 10  scale = fp16(max|W_:,j| / 127), q = clamp(rint(W / scale)), and
          the protected columns decode to scale * q exactly;
  Eq. 3   each stage's bits are the signs of its target (+0 and -0 code
          positive) and its norm the fp16 of the target chunk's L2 norm;
  Eq. 5-7 the next target is the previous one minus the decoded stage, with
          the protected positions held at zero;
  Eq. 9   the coupled score is the gate row, up row and down column norms
          added in that order, and protected rows take Eq. 10 per row.
"""
import math

import numpy as np
import pytest

import oracle

hyp = pytest.importorskip("hypothesis")
st = pytest.importorskip("hypothesis.strategies")

INV_SQRT8 = 1.0 / math.sqrt(8.0)


def _bf16(vals):
    a = np.asarray(vals, np.float32)
    return (a.view(np.uint32) >> 16).astype(np.uint16)


@st.composite
def layers(draw):
    N = draw(st.integers(1, 5))
    C = draw(st.integers(1, 4))
    K = 8 * C
    S = draw(st.integers(1, 3))
    p = draw(st.integers(0, K))
    ks = draw(st.lists(st.integers(-64, 64), min_size=N * K, max_size=N * K))
    neg0 = draw(st.lists(st.booleans(), min_size=N * K, max_size=N * K))
    vals = [(-0.0 if (z and k == 0) else k / 8.0) for k, z in zip(ks, neg0)]
    return np.array(vals, np.float64).reshape(N, K), S, p


@hyp.settings(max_examples=300, deadline=None)
@hyp.given(layers())
def test_encoder_follows_the_definitions(layer):
    Wd, S, p = layer
    N, K = Wd.shape
    W = _bf16(Wd)
    L = oracle.encode(W, S=S, p=p)
    # Eq. 8: top-p columns by norm (exact sums), ties to the lower index
    norms = np.sqrt((Wd * Wd).sum(axis=0))
    order = sorted(range(K), key=lambda j: (-norms[j], j))
    idx = np.array(sorted(order[:p]), np.int32)
    assert np.array_equal(L["idx"], idx)
    # Eq. 10 on the protected columns, and their exact decode
    What = oracle.decode_rows(L)
    for t, j in enumerate(idx):
        m = np.abs(Wd[:, j]).max()
        s16 = np.float16(m / 127.0)
        assert L["scale"][t] == s16.view(np.uint16)
        s = float(s16)
        q = np.clip(np.rint(Wd[:, j] / s), -127, 127) if s != 0.0 else np.zeros(N)
        assert np.array_equal(L["q8"][:, t].astype(np.float64), q)
        assert np.array_equal(What[:, j], s * q)
    # Eq. 3 and Eq. 5-7, stage by stage
    prot = np.zeros(K, bool)
    prot[idx] = True
    r = np.where(prot[None, :], 0.0, Wd)
    C = K // 8
    for s in range(S):
        chunks = r.reshape(N, C, 8)
        bits = np.unpackbits(L["codes"][s].reshape(N, C, 1), axis=2, bitorder="little")
        assert np.array_equal(bits.astype(bool), chunks < 0)          # +0 and -0 code positive
        sq = np.zeros((N, C))
        for k in range(8):                                            # the oracle's order
            sq = sq + chunks[:, :, k] * chunks[:, :, k]
        n16 = np.sqrt(sq).astype(np.float16)
        assert np.array_equal(L["norms"][s], n16.view(np.uint16))
        t = n16.astype(np.float64)[:, :, None] * INV_SQRT8
        rhat = np.where(bits.astype(bool), -t, t).reshape(N, K)
        r = np.where(prot[None, :], 0.0, r - rhat)
    # decode outside the protected set is the sum of the stages
    full = np.zeros((N, K))
    for s in range(S):
        bits = np.unpackbits(L["codes"][s].reshape(N, C, 1), axis=2, bitorder="little")
        t = L["norms"][s].view(np.float16).astype(np.float64)[:, :, None] * INV_SQRT8
        full = full + np.where(bits.astype(bool), -t, t).reshape(N, K)
    assert np.array_equal(What[:, ~prot], full[:, ~prot])


@hyp.settings(max_examples=200, deadline=None)
@hyp.given(layers(), st.integers(1, 3))
def test_product_is_linear_and_row_separable(layer, B):
    Wd, S, p = layer
    N, K = Wd.shape
    L = oracle.encode(_bf16(Wd), S=S, p=p)
    What = oracle.decode_rows(L)
    rng = np.random.default_rng(B)
    x = _bf16(rng.integers(-16, 17, (B, K)) / 4.0)
    y = oracle.matmul(What, x)
    xd = (x.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    assert np.allclose(y, xd @ What.T, rtol=1e-12, atol=1e-12)
    for r in range(N):                                        # any row block alone
        assert np.array_equal(oracle.decode_rows(L, row0=r, nrows=1)[0], What[r])


@hyp.settings(max_examples=200, deadline=None)
@hyp.given(layers())
def test_row_encoder_follows_the_definitions(layer):
    """Eq. 10 on rows: the top-p rows by norm (ties to the lower index), one
    scale per row, and the stages of the row-masked weight."""
    Wd, S, p = layer
    N, K = Wd.shape
    p = min(p, N)
    W = _bf16(Wd)
    L = oracle.encode_rows(W, S, p)
    norms = np.sqrt((Wd * Wd).sum(axis=1))
    idx = np.array(sorted(sorted(range(N), key=lambda i: (-norms[i], i))[:p]), np.int32)
    assert np.array_equal(L["idx"], idx)
    for t, i in enumerate(idx):
        s16 = np.float16(np.abs(Wd[i]).max() / 127.0)
        assert L["scale"][t] == s16.view(np.uint16)
        s = float(s16)
        q = np.clip(np.rint(Wd[i] / s), -127, 127) if s != 0.0 else np.zeros(K)
        assert np.array_equal(L["q8"][t, :K].astype(np.float64), q)
    Wm = W.copy()
    Wm[idx] = 0
    ref = oracle.encode(Wm, S=S, p=0)
    assert np.array_equal(L["codes"], ref["codes"]) and np.array_equal(L["norms"], ref["norms"])


@st.composite
def mlps(draw):
    F = draw(st.integers(1, 12))
    H = draw(st.integers(1, 6))
    p = draw(st.integers(0, F))

    def mat(r, c):
        ks = draw(st.lists(st.integers(-16, 16), min_size=r * c, max_size=r * c))
        return np.array(ks, np.float64).reshape(r, c) / 4.0
    return mat(F, H), mat(F, H), mat(H, F), p


@hyp.settings(max_examples=200, deadline=None)
@hyp.given(mlps())
def test_coupled_selection_follows_eq9(mlp):
    """Eq. 9: gate row norm + up row norm + down column norm, added in that
    order; the top p channels, ties to the lower index, ascending."""
    G, U, D, p = mlp
    F = G.shape[0]
    idx, scores = oracle.select_coupled(_bf16(G), _bf16(U), _bf16(D), p)
    want = (np.sqrt((G * G).sum(axis=1)) + np.sqrt((U * U).sum(axis=1))) + np.sqrt((D * D).sum(axis=0))
    assert np.array_equal(np.asarray(scores), want)
    top = sorted(sorted(range(F), key=lambda j: (-want[j], j))[:p])
    assert list(idx) == top
