"""Pins for the fp64 CPU oracle (no GPU).

Each test checks the oracle against something other than itself: a brute
force over all candidates, a closed form, a value the paper prints, an
invariant the paper states, or a library routine that reduces to the same
operation in a special case.  A plausible slip in the oracle -- a dropped
stage, a wrong sign or bit order, a transposed index, double rounding --
fails at least one of them.
"""
import itertools
import json
import math
import os

import numpy as np
import pytest
import torch

import oracle
from paper_2607_08643_gb300 import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")
INV_SQRT8 = 1.0 / math.sqrt(8.0)


def bf16(vals):
    """Exact bf16 bit patterns for values that bf16 represents exactly."""
    a = np.asarray(vals, dtype=np.float32)
    b = (a.view(np.uint32) >> 16).astype(np.uint16)
    assert np.array_equal(synth.bf16_bits_to_f32(b), a), "value not exact in bf16"
    return b


def f64(bits):
    return synth.bf16_bits_to_f32(bits).astype(np.float64)


# ---------------------------------------------------------------- numbers

def test_fp16_rounding_brute_force_all_binades():
    """Every finite binary16 value round-trips; every midpoint between two
    neighbours goes to the even one; one ulp of binary64 either side of a
    midpoint goes to the nearer neighbour; overflow and underflow edges."""
    vals = np.arange(0, 0x7C00, dtype=np.uint16).view(np.float16).astype(np.float64)
    for i in range(0, 0x7C00 - 1):
        lo, hi = vals[i], vals[i + 1]
        assert oracle.double_to_fp16(lo) == i
        assert oracle.double_to_fp16(-lo) == (i | 0x8000)
        mid = (lo + hi) / 2.0                       # exact in binary64
        even = i if i % 2 == 0 else i + 1
        assert oracle.double_to_fp16(mid) == even, hex(i)
        assert oracle.double_to_fp16(np.nextafter(mid, 0.0)) == i
        assert oracle.double_to_fp16(np.nextafter(mid, np.inf)) == i + 1
    assert oracle.double_to_fp16(65504.0) == 0x7BFF
    assert oracle.double_to_fp16(np.nextafter(65520.0, 0.0)) == 0x7BFF
    assert oracle.double_to_fp16(65520.0) == 0x7C00          # tie -> even -> inf
    assert oracle.double_to_fp16(1e300) == 0x7C00
    assert oracle.double_to_fp16(2.0 ** -25) == 0x0000        # tie -> even (0)
    assert oracle.double_to_fp16(np.nextafter(2.0 ** -25, 1.0)) == 0x0001
    assert oracle.double_to_fp16(-0.0) == 0x8000
    assert oracle.double_to_fp16(0.0) == 0x0000


def test_fp16_rounding_matches_numpy_cast():
    rng = np.random.default_rng(5)
    x = np.concatenate([rng.standard_normal(4000) * 10.0 ** rng.integers(-9, 6, 4000),
                        rng.uniform(-65530, 65530, 500)])
    with np.errstate(over="ignore"):
        want = x.astype(np.float16).view(np.uint16)
    got = np.array([oracle.double_to_fp16(v) for v in x], np.uint16)
    assert np.array_equal(got, want)


def test_fp16_and_bf16_widening_all_patterns():
    h = np.arange(65536, dtype=np.uint32).astype(np.uint16)
    ref16 = h.view(np.float16).astype(np.float64)
    with np.errstate(invalid="ignore"):
        ref_bf = synth.bf16_bits_to_f32(h).astype(np.float64)
    for v in range(0, 65536, 7):
        a, b = oracle.fp16_to_double(v), oracle.bf16_to_double(v)
        if np.isnan(ref16[v]):
            assert math.isnan(a)
        else:
            assert a == ref16[v] and math.copysign(1, a) == math.copysign(1, ref16[v])
        if np.isnan(ref_bf[v]):
            assert math.isnan(b)
        else:
            assert b == ref_bf[v]


# ------------------------------------------------------- Eq. 3 sign code

def test_sign_code_is_nearest_unit_sphere_code_brute_force():
    """Eq. 3: q = sign(u)/sqrt(b) is the nearest point of {+-1/sqrt(b)}^b to
    u = x/||x||; brute force over all 2^8 candidates on random chunks."""
    rng = np.random.default_rng(11)
    cands = np.array(list(itertools.product([1.0, -1.0], repeat=8)))   # 256 x 8
    cand_bits = np.array([sum(1 << k for k in range(8) if c[k] < 0) for c in cands])
    for _ in range(300):
        x = synth.f32_to_bf16_bits(np.float32(rng.standard_normal(8) * 0.05))
        L = oracle.encode(x.reshape(1, 8), S=1, p=0)
        xv = f64(x)
        u = xv / np.linalg.norm(xv)
        d = ((u[None, :] - cands / math.sqrt(8)) ** 2).sum(1)
        assert L["codes"][0, 0, 0] == cand_bits[np.argmin(d)]
        # and the rescaled code n*q is the nearest sign vector at that radius
        n = np.linalg.norm(xv)
        d2 = ((xv[None, :] - n * cands / math.sqrt(8)) ** 2).sum(1)
        assert L["codes"][0, 0, 0] == cand_bits[np.argmin(d2)]


def test_bit_order_and_zero_sign():
    """bit k of the chunk byte is element k, 1 = negative; +0, -0 -> 0."""
    for k in range(8):
        v = np.full(8, 0.25, np.float32)
        v[k] = -0.25
        L = oracle.encode(bf16(v).reshape(1, 8), S=1, p=0)
        assert L["codes"][0, 0, 0] == (1 << k)
    z = np.array([0.0, -0.0, 0.0, -0.0, 0.0, 0.0, -0.0, 0.0], np.float32)
    L = oracle.encode(bf16(z).reshape(1, 8), S=2, p=0)
    assert np.all(L["codes"] == 0) and np.all(L["norms"] == 0)
    # chunks land in byte c of the row in input-column order
    v = np.full(32, 0.5, np.float32)
    v[8 * 2 + 3] = -0.5
    L = oracle.encode(bf16(v).reshape(1, 32), S=1, p=0)
    assert list(L["codes"][0, 0]) == [0, 0, 1 << 3, 0]


def test_unit_code_norm_and_rescale():
    """All codes have the same l2 norm (Eq. 3), so the stage-1 reconstruction
    of a chunk has norm exactly n16."""
    rng = np.random.default_rng(3)
    W = synth.f32_to_bf16_bits(np.float32(rng.standard_normal((4, 64)) * 0.02))
    L = oracle.encode(W, S=1, p=0)
    What = oracle.decode_rows(L)
    for i in range(4):
        for c in range(8):
            n16 = oracle.fp16_to_double(L["norms"][0, i, c])
            got = np.linalg.norm(What[i, 8 * c:8 * c + 8])
            assert abs(got - n16) <= 4e-16 * max(n16, 1e-300)


def test_scaled_sign_chunk_reproduced():
    """A chunk c*s, s in {+-1}^8, is reproduced up to the fp16 rounding of its
    norm: |xhat - x| = |n16 - n|/sqrt(8) per element, and n16 is within half
    an fp16 ulp of n = c*sqrt(8)."""
    rng = np.random.default_rng(4)
    for c in [2.0 ** -5, 0.375, 3.0, 2.0 ** -10]:
        s = rng.choice([-1.0, 1.0], 8)
        x = bf16(np.float32(c * s))
        L = oracle.encode(x.reshape(1, 8), S=1, p=0)
        n = c * math.sqrt(8.0)
        n16 = oracle.fp16_to_double(L["norms"][0, 0, 0])
        ulp = 2.0 ** (math.floor(math.log2(n)) - 10)
        assert abs(n16 - n) <= ulp / 2
        xhat = oracle.decode_rows(L)[0]
        assert np.all(np.sign(xhat) == s)
        assert np.max(np.abs(xhat - c * s)) <= abs(n16 - n) / math.sqrt(8.0) + 1e-17


def test_one_hot_chunk_per_chunk_counterexample_closed_form():
    """A one-hot chunk e_0 gets the all-positive code with n16 = 1; its stage
    residual has energy exactly 2 - 2/sqrt(8) > 1 (residual stages do not
    decrease the error of every chunk, only in aggregate)."""
    x = np.zeros(8, np.float32)
    x[0] = 1.0
    L = oracle.encode(bf16(x).reshape(1, 8), S=1, p=0)
    assert L["codes"][0, 0, 0] == 0 and L["norms"][0, 0, 0] == 0x3C00
    r = 1.0 * np.eye(8)[0] - oracle.decode_rows(L)[0]
    assert abs((r ** 2).sum() - (2.0 - 2.0 / math.sqrt(8.0))) < 1e-15


# ------------------------------------------------------- Eq. 5-7 residuals

@pytest.mark.parametrize("dist,lo1,hi1,lo2,hi2", [("normal", 0.32, 0.38, 0.07, 0.11),
                                                  ("t4", 0.46, 0.55, 0.09, 0.13)])
def test_residual_energy_decreases_with_stages(dist, lo1, hi1, lo2, hi2):
    """Sec. III-D: each added stage codes the residual left by the previous
    ones, so the aggregate error energy on the BSQ-coded (unprotected)
    entries falls strictly with S."""
    W = synth.layer_weights(128, 1024, seed=7, dist=dist)
    p = synth.protected_count(1024, 1)
    Wd = f64(W)
    E = []
    for S in (1, 2, 3):
        L = oracle.encode(W, S=S, p=p)
        mask = np.ones(1024, bool)
        mask[L["idx"]] = False
        E.append(((Wd - oracle.decode_rows(L))[:, mask] ** 2).sum())
    E0 = (Wd[:, mask] ** 2).sum()
    assert E0 > E[0] > E[1] > E[2] > 0
    assert lo1 < E[0] / E0 < hi1
    assert lo2 < E[1] / E0 < hi2


def test_second_stage_codes_the_first_stage_residual():
    """Eq. 5-7: stage 2 stores sign(r1) and fp16(||r1||) of the residual
    r1 = x - rhat1, rebuilt here from the S=1 decode with numpy."""
    W = synth.layer_weights(64, 256, seed=9)
    p = 3
    L1 = oracle.encode(W, S=1, p=p)
    L2 = oracle.encode(W, S=2, p=p)
    assert np.array_equal(L1["codes"][0], L2["codes"][0])
    assert np.array_equal(L1["norms"][0], L2["norms"][0])
    Wt = f64(W)
    Wt[:, L1["idx"]] = 0.0
    R = Wt - oracle.decode_rows(dict(L1, p=0))
    R[:, L1["idx"]] = 0.0
    R = R.reshape(64, 32, 8)
    bits = ((R < 0) * (1 << np.arange(8))).sum(-1)
    assert np.array_equal(bits, L2["codes"][1])
    n16 = np.linalg.norm(R, axis=-1).astype(np.float16).view(np.uint16).astype(np.int32)
    assert np.max(np.abs(n16 - L2["norms"][1].astype(np.int32))) <= 1


def test_protected_entries_masked_in_every_stage():
    """Coding the complement by masking: stage 1 of W with protected set P
    equals stage 1 of W with those columns zeroed, and the residual at a
    protected entry is zero before every stage (so its sign bit is 0)."""
    W = synth.layer_weights(32, 128, seed=2)
    L = oracle.encode(W, S=3, p=5)
    Wz = W.copy()
    Wz[:, L["idx"]] = 0
    Lz = oracle.encode(Wz, S=1, p=0)
    assert np.array_equal(L["codes"][0], Lz["codes"][0])
    assert np.array_equal(L["norms"][0], Lz["norms"][0])
    bits = np.unpackbits(L["codes"][..., None], axis=-1, bitorder="little").reshape(3, 32, 128)
    assert np.all(bits[:, :, L["idx"]] == 0)
    assert bits[1:].sum() > 0


# ------------------------------------------------------- Eq. 8 and Eq. 10

def test_selection_matches_full_sort_and_catches_outliers():
    W = synth.layer_weights(128, 1024, seed=0)
    p = synth.protected_count(1024, 1)
    idx, scores = oracle.select_protected(W, p)
    col = np.linalg.norm(f64(W), axis=0)                       # numpy's own sum
    assert np.allclose(scores, col, rtol=1e-12, atol=0)
    order = np.lexsort((np.arange(1024), -col))
    assert np.array_equal(idx, np.sort(order[:p]))
    assert set(synth.outlier_columns(1024, seed=0, N=128)) <= set(idx.tolist())


def test_selection_ties_and_calibration_weights():
    W = bf16(np.full((4, 64), 0.5, np.float32))
    idx, _ = oracle.select_protected(W, 5)
    assert list(idx) == [0, 1, 2, 3, 4]                 # ties -> lower index
    g = np.ones(64, np.float32)
    g[[60, 61, 62]] = 2.0
    idx, _ = oracle.select_protected(W, 3, g=g)
    assert list(idx) == [60, 61, 62]                    # S_j = g_j ||W_:,j||
    Wo = synth.layer_weights(16, 64, seed=1)
    out = synth.outlier_columns(64, seed=1, N=16)
    g = np.ones(64, np.float32)
    g[out] = 0.0
    idx, _ = oracle.select_protected(Wo, 4, g=g)
    assert not set(idx.tolist()) & set(out.tolist())


def test_q8_per_channel_quantiser_closed_form():
    W = synth.layer_weights(200, 256, seed=12)
    p = 6
    L = oracle.encode(W, S=1, p=p)
    Wd = f64(W)
    for t, j in enumerate(L["idx"]):
        col = Wd[:, j]
        m = np.abs(col).max()
        s16 = np.float16(m / 127.0)                    # numpy's own rounding
        assert L["scale"][t] == s16.view(np.uint16)
        s = float(s16)
        q = L["q8"][:, t].astype(np.float64)
        assert np.all(np.abs(q) <= 127)
        assert np.array_equal(q, np.clip(np.rint(col / s), -127, 127))
        inside = np.abs(col / s) <= 127
        assert np.all(np.abs(col - s * q)[inside] <= s / 2 * (1 + 1e-15))
        assert np.abs(q[np.argmax(np.abs(col))]) >= 126
    assert np.all(L["q8"][:, p:] == 0)                 # padding is zero


def test_protected_columns_decode_to_scale_times_q8_exactly():
    W = synth.layer_weights(64, 512, seed=13)
    L = oracle.encode(W, S=2, p=9)
    What = oracle.decode_rows(L)
    for t, j in enumerate(L["idx"]):
        s = oracle.fp16_to_double(L["scale"][t])
        assert np.array_equal(What[:, j], s * L["q8"][:, t].astype(np.float64))


def test_all_zero_layer():
    W = np.zeros((8, 64), np.uint16)
    L = oracle.encode(W, S=3, p=4)
    assert np.all(L["codes"] == 0) and np.all(L["norms"] == 0)
    assert np.all(L["q8"] == 0) and np.all(L["scale"] == 0)
    assert np.all(oracle.decode_rows(L) == 0)


def test_range_and_argument_errors():
    big = np.full((1, 8), 0x7F7F, np.uint16)          # largest finite bf16
    with pytest.raises(oracle.OracleError) as e:
        oracle.encode(big, S=1, p=0)
    assert e.value.code == oracle.ERR_RANGE
    inf = np.full((1, 8), 0x7F80, np.uint16)
    with pytest.raises(oracle.OracleError) as e:
        oracle.encode(inf, S=1, p=0)
    assert e.value.code == oracle.ERR_RANGE
    with pytest.raises(oracle.OracleError) as e:
        oracle.encode(np.zeros((2, 12), np.uint16), S=1, p=0)
    assert e.value.code == oracle.ERR_INVALID_ARG
    with pytest.raises(oracle.OracleError):
        oracle.encode(np.zeros((2, 16), np.uint16), S=4, p=0)


# ------------------------------------------------------ Eq. 12 decode/apply

def test_decode_matches_independent_unpacking():
    """Eq. 12: What = sum_s Assemble(D_s(B_s)), rebuilt with numpy's bit
    unpacking (little bit order) and the Eq. 10 scatter."""
    W = synth.layer_weights(48, 256, seed=21, dist="t4")
    L = oracle.encode(W, S=3, p=7)
    bits = np.unpackbits(L["codes"][..., None], axis=-1, bitorder="little")   # S,N,C,8
    sgn = 1.0 - 2.0 * bits
    t = L["norms"].view(np.float16).astype(np.float64) * INV_SQRT8
    ref = np.zeros((48, 256))
    for s in range(3):
        ref = ref + (sgn[s] * t[s][..., None]).reshape(48, 256)
    ref[:, L["idx"]] = L["scale"].view(np.float16).astype(np.float64)[None, :] * \
        L["q8"][:, :7].astype(np.float64)
    assert np.array_equal(oracle.decode_rows(L), ref)


def test_matmul_one_hot_linearity_and_numpy():
    W = synth.layer_weights(40, 128, seed=31)
    L = oracle.encode(W, S=2, p=2)
    What = oracle.decode_rows(L)
    for j in (0, 7, 64, 127):
        e = np.zeros((1, 128), np.float32)
        e[0, j] = 1.0
        assert np.array_equal(oracle.matmul(What, bf16(e))[0], What[:, j])
    rng = np.random.default_rng(0)
    a = np.float32(rng.integers(-4, 5, (1, 128)))
    b = np.float32(rng.integers(-4, 5, (1, 128)))
    ya, yb, yab = (oracle.matmul(What, bf16(v))[0] for v in (a, b, a + b))
    assert np.allclose(ya + yb, yab, rtol=0, atol=1e-13)
    X = synth.activations(3, 128, seed=1)
    Y = oracle.matmul(What, X)
    assert np.allclose(Y, f64(X) @ What.T, rtol=1e-13, atol=1e-13)
    rows = np.array([39, 0, 17], np.int32)
    assert np.array_equal(oracle.apply_rows(L, rows, X), Y[:, rows])


def test_single_stage_no_protection_is_scaled_sign_matrix_product():
    """S = 1, p = 0: y = (1/sqrt 8) sum_c n_c <s_c, x_c>, the chunk-factored
    form, equals the dense product."""
    W = synth.layer_weights(16, 64, seed=41)
    L = oracle.encode(W, S=1, p=0)
    X = synth.activations(2, 64, seed=2)
    s = 1.0 - 2.0 * np.unpackbits(L["codes"][0][..., None], axis=-1, bitorder="little")
    n = L["norms"][0].view(np.float16).astype(np.float64)
    xc = f64(X).reshape(2, 8, 8)
    y = np.einsum("nc,nck,bck->bn", n, s, xc) / math.sqrt(8.0)
    assert np.allclose(oracle.gemv(L, X), y, rtol=1e-12, atol=1e-14)


def test_encode_is_deterministic():
    W = synth.layer_weights(64, 128, seed=8)
    a, b = oracle.encode(W, S=2, p=3), oracle.encode(W, S=2, p=3)
    for k in ("codes", "norms", "q8", "scale", "idx"):
        assert np.array_equal(a[k], b[k])


# ------------------------------------------------- storage accounting, Eq. 2

def test_paper_bit_accounting_golden():
    """Values the paper prints (tests/golden/paper_arithmetic.json)."""
    with open(os.path.join(GOLDEN, "paper_arithmetic.json")) as f:
        g = json.load(f)
    # Eq. 2: one stage stores b bits per d weights; with b = d the code-only
    # rate is 1 bit per weight per stage -- the oracle's code buffer size.
    for case in g["nominal_rate"]:
        b, d = case["b"], case["d"]
        assert b / d == case["bpw_stage"]
    N, K, S = 4096, 4096, 2
    codes_bytes = oracle.encoded_sizes(N, K, S, 0)[0]
    assert codes_bytes * 8 / (S * N * K) == 1.0
    # Sec. III-D: a q_proj of Qwen3-8B split into d = 32 chunks has 2^19 chunks
    cs = g["qproj_chunks"]
    assert cs["rows"] * cs["cols"] // cs["d"] == 2 ** cs["log2_chunks"]
    assert abs(cs["median_occupied"] / 2.0 ** cs["b"] - cs["used_fraction"]) < 0.005e-14
    # the same counting at d = 8 is the oracle's chunk count per stage
    assert oracle.encoded_sizes(4096, 4096, 1, 0)[0] == 2 ** 21


def test_encoded_sizes_closed_form():
    for (N, K), S, rho in [((1024, 1024), 2, 1), ((4096, 4096), 2, 1), ((1024, 4096), 2, 1),
                           ((12288, 4096), 3, 2), ((4096, 12288), 3, 2)]:
        p = synth.protected_count(K, rho)
        sz = oracle.encoded_sizes(N, K, S, p)
        C = K // 8
        assert sz == [S * N * C, 2 * S * N * C, N * ((p + 15) // 16 * 16), 2 * p, 4 * p]
    assert synth.protected_count(1024, 1) == 11
    # algorithmic compressed bytes (unpadded q8), 1024 x 1024, S = 2, 1 %
    p = 11
    assert 2 * 1024 * 128 * 3 + 1024 * p + 6 * p == 797762


# ------------------------------------------------- low-rank compensation

def test_lora_exact_rational_brute_force():
    """lora_apply against the exact rational value of y0 + s * Bm (A x) on a
    tiny case: the fp64 result lies within the rounding bound of a sum of
    K + rank + 2 terms."""
    from fractions import Fraction
    rank, N, K, B = 3, 5, 16, 2
    A, Bm = synth.lora_adapter(N, K, rank, seed=11, sigma_a=0.25, sigma_b=0.5)
    X = synth.activations(B, K, seed=12)
    Y0 = synth.bf16_bits_to_f32(synth.activations(B, N, seed=13)).astype(np.float64)
    scale = 0.75
    got = oracle.lora_apply(A, Bm, X, Y0, scale)
    fa, fb, fx = f64(A), f64(Bm), f64(X)
    u = 2.0 ** -53
    for b in range(B):
        t = [sum(Fraction(fa[r, k]) * Fraction(fx[b, k]) for k in range(K)) for r in range(rank)]
        tabs = [sum(abs(fa[r, k] * fx[b, k]) for k in range(K)) for r in range(rank)]
        for n in range(N):
            exact = Fraction(Y0[b, n]) + Fraction(scale) * sum(Fraction(fb[n, r]) * t[r]
                                                               for r in range(rank))
            mag = abs(Y0[b, n]) + scale * sum(abs(fb[n, r]) * tabs[r] for r in range(rank))
            assert abs(got[b, n] - float(exact)) <= 2 * (K + rank + 2) * u * mag + 1e-300


def test_lora_rank1_one_hot_closed_form():
    """A rank-1 adapter on a one-hot activation adds s * Bm[n][0] * A[0][k]
    to every output: one product, exact in fp64."""
    N, K = 7, 24
    A, Bm = synth.lora_adapter(N, K, 1, seed=21)
    for k in (0, 5, K - 1):
        x = np.zeros((1, K), np.uint16)
        x[0, k] = bf16([1.0])[0]
        y0 = np.arange(N, dtype=np.float64)[None, :] * 0.5
        got = oracle.lora_apply(A, Bm, x, y0, 0.5)
        want = y0[0] + 0.5 * f64(Bm)[:, 0] * f64(A)[0, k]
        assert np.array_equal(got[0], want)


def test_lora_against_product_matrix_and_invariants():
    """The adapter's down projection first (oracle) against the product
    matrix Bm A formed first (numpy, another association); doubling x
    doubles the correction exactly; scale 0 returns y0 bit for bit; a
    transposed Bm or a missing scale would fail."""
    rank, N, K, B = 16, 48, 256, 3
    A, Bm = synth.lora_adapter(N, K, rank, seed=31)
    X = synth.activations(B, K, seed=32)
    Y0 = synth.bf16_bits_to_f32(synth.activations(B, N, seed=33)).astype(np.float64)
    got = oracle.lora_apply(A, Bm, X, Y0, 2.0)
    want = Y0 + 2.0 * f64(X) @ (f64(Bm) @ f64(A)).T
    assert np.max(np.abs(got - want)) <= 1e-12 * np.max(np.abs(want - Y0))
    X2 = f32_bits_times_two(X)
    zero = np.zeros_like(Y0)
    assert np.array_equal(oracle.lora_apply(A, Bm, X2, zero, 1.0),
                          2.0 * oracle.lora_apply(A, Bm, X, zero, 1.0))
    assert np.array_equal(oracle.lora_apply(A, Bm, X, Y0, 0.0), Y0)


def f32_bits_times_two(bits):
    """bf16 bits of 2 * x (exponent + 1; the test values are normal and far
    from overflow)."""
    v = synth.bf16_bits_to_f32(bits)
    assert np.all(np.abs(v[v != 0]) > 1e-30) and np.all(np.abs(v) < 1e30)
    out = bf16(2.0 * v)
    return out


# ------------------------------------- output-row and coupled MLP protection

def _outlier_rows(N, K, seed):
    """bf16 bits [N][K] with 8 outlier rows (the generator's outlier columns of
    the transposed shape)."""
    return np.ascontiguousarray(synth.layer_weights(K, N, seed=seed).T)


def test_row_selection_matches_full_sort_and_catches_outliers():
    N, K, p = 96, 64, 10
    W = _outlier_rows(N, K, seed=41)
    idx, scores = oracle.select_rows(W, p)
    norms = np.sqrt((f64(W) ** 2).sum(axis=1))
    assert np.allclose(scores, norms, rtol=1e-14, atol=0)
    order = sorted(range(N), key=lambda i: (-norms[i], i))
    assert list(idx) == sorted(order[:p])
    outliers = np.argsort(-np.abs(f64(W)).max(axis=1))[:8]
    assert set(outliers.tolist()) <= set(idx.tolist())
    # ties go to the lower row; g weights the rows
    Wt = np.zeros((6, 8), np.uint16)
    Wt[[1, 3, 4]] = bf16([0.5] * 8)
    assert list(oracle.select_rows(Wt, 2)[0]) == [1, 3]
    g = np.array([1, 1, 1, 0.5, 1, 1], np.float32)
    assert list(oracle.select_rows(Wt, 2, g=g)[0]) == [1, 4]


def test_coupled_score_is_the_sum_of_three_slice_norms():
    """Eq. 9: gate row norm + up row norm + down column norm, TopK."""
    F, H, p = 80, 48, 7
    Wg = synth.layer_weights(F, H, seed=51)
    Wu = synth.layer_weights(F, H, seed=52)
    Wd = synth.layer_weights(H, F, seed=53)
    idx, scores = oracle.select_coupled(Wg, Wu, Wd, p)
    want = (np.sqrt((f64(Wg) ** 2).sum(1)) + np.sqrt((f64(Wu) ** 2).sum(1))
            + np.sqrt((f64(Wd) ** 2).sum(0)))
    assert np.allclose(scores, want, rtol=1e-14, atol=0)
    assert list(idx) == sorted(sorted(range(F), key=lambda j: (-want[j], j))[:p])
    # zero weight on gate and up leaves down's column selection (Eq. 8)
    z = np.zeros(F, np.float32)
    assert list(oracle.select_coupled(Wg, Wu, Wd, p, gg=z, gu=z)[0]) == \
        list(oracle.select_protected(Wd, p)[0])
    # zero weight on up and down leaves gate's row selection
    assert list(oracle.select_coupled(Wg, Wu, Wd, p, gu=z, gd=z)[0]) == \
        list(oracle.select_rows(Wg, p)[0])


def test_row_protection_encode_and_decode():
    """Eq. 10 on rows: one scale per protected row (closed form with numpy's
    fp16 rounding and rint), the BSQ stages of the row-masked matrix, and a
    decode that returns scale * q8 on the protected rows exactly."""
    N, K, S, p = 72, 136, 2, 6
    W = _outlier_rows(N, K, seed=61)
    L = oracle.encode_rows(W, S, p)
    idx = L["idx"]
    assert list(idx) == list(oracle.select_rows(W, p)[0])
    fw = f64(W)
    s = (np.abs(fw[idx]).max(axis=1) / 127.0).astype(np.float16)
    assert np.array_equal(L["scale"], s.view(np.uint16))
    sd = s.astype(np.float64)[:, None]
    q = np.clip(np.rint(fw[idx] / sd), -127, 127)
    assert np.array_equal(L["q8"][:, :K], q.astype(np.int8))
    assert not L["q8"][:, K:].any()
    assert np.all(np.abs(fw[idx] - sd * q) <= sd / 2 + 1e-300)
    # stages: the row-masked matrix through the column encoder with p = 0
    Wm = W.copy()
    Wm[idx] = 0
    ref = oracle.encode(Wm, S=S, p=0)
    assert np.array_equal(L["codes"], ref["codes"]) and np.array_equal(L["norms"], ref["norms"])
    assert not L["norms"][:, idx].any()
    What = oracle.decode_rows(L)
    assert np.array_equal(What[idx], sd * L["q8"][:, :K].astype(np.float64))
    keep = np.setdiff1d(np.arange(N), idx)
    assert np.array_equal(What[keep], oracle.decode_rows(ref)[keep])
    assert np.array_equal(oracle.decode_rows(L, row0=5, nrows=20), What[5:25])


def test_coupled_encode_shares_one_set():
    F, H, S, p = 64, 32, 2, 4
    Wg = synth.layer_weights(F, H, seed=71)
    Wu = synth.layer_weights(F, H, seed=72)
    Wd = synth.layer_weights(H, F, seed=73)
    Lg, Lu, Ld = oracle.encode_coupled(Wg, Wu, Wd, S, p)
    idx = oracle.select_coupled(Wg, Wu, Wd, p)[0]
    for L in (Lg, Lu, Ld):
        assert list(L["idx"]) == list(idx)
    assert Lg["axis"] == 1 and Lu["axis"] == 1 and Ld.get("axis", 0) == 0
    # down keeps the coupled set as columns: scale * q8 there, within half a
    # quantisation step of the weight
    sd = Ld["scale"].view(np.float16).astype(np.float64)[None, :]
    cols = oracle.decode_rows(Ld)[:, idx]
    assert np.array_equal(cols, sd * Ld["q8"][:, :p])
    assert np.all(np.abs(f64(Wd)[:, idx] - cols) <= sd / 2 + 1e-300)


# ------------------------------------------- FP8 / BF16 protected payloads



_FP8 = {oracle.FMT_E4M3: (torch.float8_e4m3fn, 3, 7, 448.0),
        oracle.FMT_E5M2: (torch.float8_e5m2, 2, 15, 57344.0)}


def _fp8_value_closed_form(v, mb, bias, e4m3):
    """Value of an FP8 bit pattern from the format's definition (sign,
    exponent field, mantissa field), written out independently of the
    oracle's decoder."""
    s = -1.0 if v & 0x80 else 1.0
    e = (v >> mb) & ((1 << (7 - mb)) - 1)
    m = v & ((1 << mb) - 1)
    emax = (1 << (7 - mb)) - 1
    if e4m3 and e == emax and m == (1 << mb) - 1:
        return math.nan
    if not e4m3 and e == emax:
        return math.nan if m else s * math.inf
    if e == 0:
        return s * m * 2.0 ** (1 - bias - mb)
    return s * (1 + m / 2.0 ** mb) * 2.0 ** (e - bias)


@pytest.mark.parametrize("fmt", [oracle.FMT_E4M3, oracle.FMT_E5M2])
def test_fp8_widening_all_patterns(fmt):
    """All 256 codes against torch's FP8 dtype and the format's closed form."""
    dt, mb, bias, _ = _FP8[fmt]
    mine = np.array([oracle.fp8_to_double(v, fmt) for v in range(256)])
    ref = torch.arange(256, dtype=torch.uint8).view(dt).to(torch.float64).numpy()
    assert np.array_equal(mine, ref, equal_nan=True)
    cf = np.array([_fp8_value_closed_form(v, mb, bias, fmt == oracle.FMT_E4M3) for v in range(256)])
    assert np.array_equal(mine, cf, equal_nan=True)


@pytest.mark.parametrize("fmt", [oracle.FMT_E4M3, oracle.FMT_E5M2])
def test_fp8_rounding_brute_force_nearest_ties_to_even(fmt):
    """Within range the code is the nearest finite code (brute force over all
    of them), ties to the even mantissa; exact midpoints between neighbours
    are included, and so are subnormals and both zeros."""
    dt, mb, bias, maxf = _FP8[fmt]
    codes = [v for v in range(256) if math.isfinite(oracle.fp8_to_double(v, fmt))]
    vals = np.array([oracle.fp8_to_double(v, fmt) for v in codes])
    pos = sorted({x for x in vals if x >= 0})
    rng = np.random.default_rng(5)
    xs = list(rng.uniform(-maxf, maxf, 400)) + list(rng.normal(0, 1, 400)) + \
        list(rng.normal(0, 2.0 ** (1 - bias), 200))
    xs += [(a + b) / 2 for a, b in zip(pos, pos[1:])]          # every midpoint
    xs += [-(a + b) / 2 for a, b in zip(pos, pos[1:])]
    xs += [0.0, -0.0, maxf, -maxf]
    for x in xs:
        got = oracle.double_to_fp8(x, fmt)
        d = np.abs(vals - x)
        best = np.flatnonzero(d == d.min())
        cand = [codes[i] for i in best]
        if x == 0.0:
            want = 0x80 if math.copysign(1.0, x) < 0 else 0x00
        elif len(cand) == 1:
            want = cand[0]
        else:                                  # a tie: the even mantissa
            cand = [c for c in cand if (c & 0x80) == (0x80 if x < 0 else 0)]
            even = [c for c in cand if c % 2 == 0]
            assert len(even) == 1
            want = even[0]
        assert got == want, (x, got, want)
        ref = int(torch.tensor([x], dtype=torch.float64).to(dt).view(torch.uint8)[0])
        assert got == ref, (x, got, ref)


@pytest.mark.parametrize("fmt", [oracle.FMT_E4M3, oracle.FMT_E5M2])
def test_fp8_saturates_above_the_largest_finite(fmt):
    """Reading for the protected payload: a value that rounds past the
    largest finite code takes that code, with its sign; NaN stays NaN."""
    _, _, _, maxf = _FP8[fmt]
    top = oracle.double_to_fp8(maxf, fmt)
    for x in (maxf * 1.5, maxf * 1e6, math.inf):
        assert oracle.double_to_fp8(x, fmt) == top
        assert oracle.double_to_fp8(-x, fmt) == top | 0x80
    assert math.isnan(oracle.fp8_to_double(oracle.double_to_fp8(math.nan, fmt), fmt))


@pytest.mark.parametrize("fmt", [oracle.FMT_E4M3, oracle.FMT_E5M2])
def test_fp8_protected_quantiser_closed_form(fmt):
    """Eq. 10 with an FP8 payload: scale = fp16(max|W_:,j| / largest FP8),
    q = fp8(W / scale) with torch's FP8 cast as the rounding reference,
    and a decoded value within half an FP8 step of the weight."""
    dt, mb, bias, maxf = _FP8[fmt]
    W = synth.layer_weights(96, 256, seed=81)
    idx = oracle.select_protected(W, 7)[0]
    q, scale = oracle.quantize_protected_fmt(W, idx, fmt)
    assert q.shape == (96, 16) and q.dtype == np.uint8
    assert not q[:, 7:].any()
    Wd = f64(W)
    got = oracle.protected_values_fmt(q, scale, fmt)
    for t, j in enumerate(idx):
        col = Wd[:, j]
        s16 = np.float16(np.abs(col).max() / maxf)
        assert scale[t] == s16.view(np.uint16)
        s = float(s16)
        r = col / s
        assert np.all(np.abs(r) <= maxf * (1 + 2.0 ** -10))
        rc = np.clip(r, -maxf, maxf)
        ref = torch.from_numpy(rc).to(dt).view(torch.uint8).numpy()
        assert np.array_equal(q[:, t], ref)
        # decoded = s * value(q); the error is at most half an FP8 ulp of
        # |W/s| (relative 2^-(mb+1) for normals, absolute half the
        # subnormal step below), plus the saturation margin at the top
        ulp_half = np.maximum(np.abs(rc) * 2.0 ** -(mb + 1), 2.0 ** (-bias - mb))
        assert np.all(np.abs(got[:, t] - s * rc) <= s * ulp_half)
        assert np.all(np.abs(r - rc) <= maxf * 2.0 ** -10)


def test_bf16_protected_payload_is_the_weight():
    W = synth.layer_weights(40, 128, seed=82)
    idx = oracle.select_protected(W, 5)[0]
    q, scale = oracle.quantize_protected_fmt(W, idx, oracle.FMT_BF16)
    assert q.dtype == np.uint16 and np.all(scale == 0x3C00)
    assert np.array_equal(q[:, :5], W[:, idx]) and not q[:, 5:].any()
    assert np.array_equal(oracle.protected_values_fmt(q, scale, oracle.FMT_BF16), f64(W)[:, idx])


def test_int8_format_matches_the_int8_quantiser():
    """FMT_INT8 through the format-generic entry is Eq. 10's INT8 quantiser."""
    W = synth.layer_weights(48, 256, seed=83)
    L = oracle.encode(W, S=1, p=6)
    q, scale = oracle.quantize_protected_fmt(W, L["idx"], oracle.FMT_INT8)
    assert np.array_equal(q, L["q8"]) and np.array_equal(scale, L["scale"])
    dec = oracle.protected_values_fmt(q, scale, oracle.FMT_INT8)
    assert np.array_equal(dec, oracle.decode_rows(L)[:, L["idx"]])


# ------------------------------------------------ learned decoder step (Eq. 1)

def _signs(v):
    """The +-1 sign vector of code byte v (bit k set <=> element k negative),
    by numpy's own bit unpacking."""
    b = np.unpackbits(np.array([v], np.uint8), bitorder="little")
    return 1.0 - 2.0 * b.astype(np.float64)


def test_linear_decoder_table_identity_permutation_and_scaling():
    T = oracle.decoder_table_linear(np.eye(8))
    for v in range(256):
        assert np.array_equal(T[v], _signs(v) * INV_SQRT8)
    perm = [3, 0, 7, 1, 6, 2, 5, 4]                   # not an involution
    P = np.zeros((8, 8))
    P[np.arange(8), perm] = 1.0                       # output k reads code position perm[k]
    T = oracle.decoder_table_linear(P)
    for v in range(256):
        assert np.array_equal(T[v], _signs(v)[perm] * INV_SQRT8)
    d = np.array([1, 2, 4, 8, 0.5, 0.25, -1, -2.0])
    T = oracle.decoder_table_linear(np.diag(d))
    for v in range(256):
        assert np.array_equal(T[v], d * (_signs(v) * INV_SQRT8))


def _dyadic_linear_table(seed):
    """A linear decoder whose fp16 table is exact: A = sqrt(8) * B with B of
    small dyadic entries, so T = A q rounds to B * signs exactly."""
    rng = np.random.default_rng(seed)
    B = rng.integers(-8, 9, size=(8, 8)) / 8.0
    T16 = oracle.table_to_fp16(oracle.decoder_table_linear(math.sqrt(8.0) * B))
    vals = T16.view(np.float16).astype(np.float64)
    for v in range(256):
        assert np.array_equal(vals[v], B @ _signs(v))
    return B, T16


def test_linear_decoder_equals_transformed_activations():
    """With D(q) = A q, y = sum_c n * (A q_c) . x_c = sum_c n * q_c . (A^T x_c):
    decoding with the table and multiplying gives the same output as the
    identity-decoder sign codes against per-chunk transformed activations."""
    N, K, S, p = 24, 96, 2, 3
    W = synth.layer_weights(N, K, seed=91)
    L = oracle.encode(W, S=S, p=p)
    tabs, Bs = [], []
    for s in range(S):
        B, T16 = _dyadic_linear_table(92 + s)
        tabs.append(T16)
        Bs.append(B)
    What = oracle.decode_rows_table(L, np.stack(tabs))
    x = synth.activations(2, K, seed=93)
    y = oracle.matmul(What, x)
    xd = f64(x)
    prot = np.zeros(K, bool)
    prot[L["idx"]] = True
    xm = np.where(prot, 0.0, xd)                       # BSQ part sees masked x
    C = K // 8
    bits = np.unpackbits(L["codes"].reshape(S, N, C, 1), axis=3, bitorder="little")
    sg = 1.0 - 2.0 * bits.astype(np.float64)           # [S][N][C][8]
    n = L["norms"].view(np.float16).astype(np.float64)  # [S][N][C]
    ref = np.zeros((2, N))
    for s in range(S):
        xt = np.einsum("kj,bck->bcj", Bs[s], xm.reshape(2, C, 8))   # B^T x per chunk
        ref += np.einsum("nc,ncj,bcj->bn", n[s], sg[s], xt)
    sc = L["scale"].view(np.float16).astype(np.float64)
    ref += xd[:, L["idx"]] @ (sc[None, :] * L["q8"][:, :p].astype(np.float64)).T
    assert np.allclose(y, ref, rtol=1e-12, atol=1e-12 * np.abs(ref).max())


def test_table_decode_with_exact_identity_table():
    """A table of +-1/2 (exact in binary16) is the norm-rescale decoder with
    1/sqrt(8) replaced by 1/2: the BSQ columns are numpy's sum of
    n * sign / 2 exactly, and the protected columns are scale * q8."""
    N, K, S = 16, 64, 3
    W = synth.layer_weights(N, K, seed=94)
    L = oracle.encode(W, S=S, p=2)
    half = np.array([[oracle.double_to_fp16(0.5 * sv) for sv in _signs(v)] for v in range(256)],
                    np.uint16)
    What = oracle.decode_rows_table(L, np.stack([half] * S))
    C = K // 8
    bits = np.unpackbits(L["codes"].reshape(S, N, C, 1), axis=3, bitorder="little")
    n = L["norms"].view(np.float16).astype(np.float64)[..., None]
    ref = ((1.0 - 2.0 * bits) * n * 0.5).sum(axis=0).reshape(N, K)
    base = oracle.decode_rows(L)
    ref[:, L["idx"]] = base[:, L["idx"]]
    assert np.array_equal(What, ref)


def test_table_decode_one_hot_table_picks_its_code():
    """A table that is 1 at one (code byte, element) and 0 elsewhere, on one
    stage only, returns that stage's norm exactly where that stage's chunk
    carries that code, and 0 everywhere else outside the protected set."""
    N, K, S = 12, 64, 2
    W = synth.layer_weights(N, K, seed=95)
    L = oracle.encode(W, S=S, p=0)
    C = K // 8
    for s0 in range(S):
        v0 = int(L["codes"].reshape(S, N, C)[s0, 3, 5])
        k0 = 6
        tabs = np.zeros((S, 256, 8), np.uint16)
        tabs[s0, v0, k0] = 0x3C00                     # 1.0
        What = oracle.decode_rows_table(L, tabs)
        want = np.zeros((N, K))
        cs = L["codes"].reshape(S, N, C)[s0]
        ns = L["norms"].reshape(S, N, C)[s0].view(np.float16).astype(np.float64)
        for i in range(N):
            for c in range(C):
                if cs[i, c] == v0:
                    want[i, 8 * c + k0] = ns[i, c]
        assert np.array_equal(What, want)
        assert What[3, 8 * 5 + k0] != 0 or ns[3, 5] == 0


def test_mlp_decoder_odd_residual_and_limits():
    rng = np.random.default_rng(96)
    hdim = 16
    W1 = rng.normal(size=(hdim, 8))
    W2 = rng.normal(size=(8, hdim))
    Wr = rng.normal(size=(hdim, hdim)) / 4
    for wr in (None, Wr):
        T = oracle.decoder_table_mlp(W1, W2, wr)
        assert np.array_equal(T[255 - np.arange(256)], -T)      # D(-q) = -D(q)
    # a zero residual block adds tanh(0) = 0
    assert np.array_equal(oracle.decoder_table_mlp(W1, W2, np.zeros((hdim, hdim))),
                          oracle.decoder_table_mlp(W1, W2))
    # one hidden unit: T[v] = W2[:, 0] * tanh(W1[0] . q(v))
    T = oracle.decoder_table_mlp(W1[:1], W2[:, :1])
    for v in (0, 1, 77, 200, 255):
        h = math.tanh(float(np.dot(W1[0], _signs(v) * INV_SQRT8)))
        assert np.allclose(T[v], W2[:, 0] * h, rtol=1e-14, atol=1e-15)
    # small inputs: tanh(e z) = e z (1 - (e z)^2/3 + ...), so the table tends to
    # the linear decoder e W2 W1 q; with the residual block, e (W2 (I + Wr) W1) q
    eps = 1e-5
    lin = oracle.decoder_table_linear(W2 @ W1)
    T = oracle.decoder_table_mlp(eps * W1, W2)
    assert np.allclose(T / eps, lin, rtol=0, atol=1e-8 * np.abs(lin).max())
    lin_r = oracle.decoder_table_linear(W2 @ (np.eye(hdim) + Wr) @ W1)
    T = oracle.decoder_table_mlp(eps * W1, W2, Wr)
    assert np.allclose(T / eps, lin_r, rtol=0, atol=1e-8 * np.abs(lin_r).max())
    with pytest.raises(oracle.OracleError):
        oracle.decoder_table_mlp(np.zeros((0, 8)), np.zeros((8, 0)))


def test_encode_with_given_columns_reduces_to_eq8_encode():
    """Given the very set Eq. 8 selects, the given-set encoder is the
    ordinary encoder byte for byte; a different set moves the masking."""
    W = synth.layer_weights(48, 136, seed=101, dist="t4")
    for S, p in ((1, 3), (2, 5), (3, 17)):
        ref = oracle.encode(W, S=S, p=p)
        got = oracle.encode_given(W, S, ref["idx"])
        for k in ("codes", "norms", "q8", "scale", "idx"):
            assert np.array_equal(got[k], ref[k]), (S, p, k)
    other = np.array([0, 7, 8, 135], np.int32)
    L = oracle.encode_given(W, 2, other)
    What = oracle.decode_rows(L)
    sc = L["scale"].view(np.float16).astype(np.float64)
    assert np.array_equal(What[:, other], sc[None, :] * L["q8"][:, :4].astype(np.float64))
    Wm = f64(W)
    Wm[:, other] = 0.0
    # the stage-1 norms are those of the chunks with the given columns zeroed
    n1 = np.sqrt((Wm.reshape(48, 17, 8) ** 2).sum(axis=2)).astype(np.float16)
    assert np.array_equal(L["norms"][0], n1.view(np.uint16))
    with pytest.raises(oracle.OracleError):
        oracle.encode_given(W, 2, np.array([5, 3], np.int32))        # not ascending
    with pytest.raises(oracle.OracleError):
        oracle.encode_given(W, 2, np.array([136], np.int32))         # out of range


@pytest.mark.parametrize("fmt", [oracle.FMT_INT8, oracle.FMT_E4M3, oracle.FMT_E5M2, oracle.FMT_BF16])
def test_row_quantiser_in_every_format(fmt):
    """Eq. 10 on rows in any payload format: INT8 equals the row encoder's
    own quantiser (or_quantize_protected_rows) byte for byte; every format
    keeps one scale per row with the format's closed form, and the decoded
    rows are within half a step of the weights."""
    N, K = 40, 136
    W = synth.layer_weights(N, K, seed=111)
    idx = np.array([3, 17, 39], np.int32)
    q, scale = oracle.quantize_protected_rows_fmt(W, idx, fmt)
    assert q.shape == (3, oracle.pad16(K)) and not q[:, K:].any()
    if fmt == oracle.FMT_INT8:
        L = oracle.encode_rows(W, 2, 3, idx=idx)
        assert np.array_equal(q, L["q8"]) and np.array_equal(scale, L["scale"])
    fw = f64(W)[idx]
    F = {oracle.FMT_INT8: 127.0, oracle.FMT_E4M3: 448.0, oracle.FMT_E5M2: 57344.0}
    if fmt == oracle.FMT_BF16:
        assert np.all(scale == 0x3C00) and np.array_equal(q[:, :K], W[idx])
    else:
        s16 = (np.abs(fw).max(axis=1) / F[fmt]).astype(np.float16)
        assert np.array_equal(scale, s16.view(np.uint16))
    qc = np.zeros((K, oracle.pad16(3)), q.dtype)                       # as protected columns
    qc[:, :3] = q[:, :K].T
    vals = oracle.protected_values_fmt(qc, scale, fmt).T                  # [p][K]
    sd = scale.view(np.float16).astype(np.float64)[:, None]
    rel = {oracle.FMT_INT8: None, oracle.FMT_E4M3: 2.0 ** -4, oracle.FMT_E5M2: 2.0 ** -3,
           oracle.FMT_BF16: 0.0}[fmt]
    if rel is None:
        assert np.all(np.abs(vals - fw) <= sd / 2 * (1 + 1e-12))
    else:
        assert np.all(np.abs(vals - fw) <= rel * np.abs(fw) + sd * 2.0 ** -9)
