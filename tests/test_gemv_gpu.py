"""bisco_gemv (decode, B <= 16) against the fp64 oracle.

Parity bar: per activation row, max|y - y_ref| / max|y_ref| <= 2e-3.  The
oracle encodes its own layer and the GPU runs on a copy of those bytes, so
no oracle input comes from the CUDA path."""
import os

import numpy as np
import pytest

import oracle
from paper_2607_08643_gb300 import synth

from _helpers import TIGHT_MMA, TOL, assert_parity, gemv_tight, max_rel_rows, sample_rows, to_dev

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


def run_gemv(env, Lref, X, plan=None, extra_env=None):
    """bisco_gemv on a device copy of the oracle's layer; `plan` forces the
    clustered kernel with tiling "WM,CK,NSLOT,WQ", `extra_env` sets other
    tuning variables for the call."""
    import torch
    bisco, dev = env
    L = bisco.Layer.from_numpy(Lref, dev)
    env_vars = dict(extra_env or {})
    if plan:
        env_vars.update(BISCO_GEMV_PLAN=plan, BISCO_GEMV_MODE="cluster")
    old = {k: os.environ.get(k) for k in env_vars}
    os.environ.update(env_vars)
    try:
        y = bisco.bisco_gemv(L, to_dev(X, dev))
    finally:
        for k, v in old.items():
            if v is None:
                del os.environ[k]
            else:
                os.environ[k] = v
    torch.cuda.synchronize()
    assert bisco.bisco_get_device_error() == 0
    return y.cpu().numpy()


@pytest.mark.parametrize("N,K,S,p,B,dist", [
    (1024, 1024, 2, 11, 1, "normal"),     # single layer 1024 x 1024, batch 1
    (1024, 1024, 2, 11, 16, "normal"),
    (100, 1536, 3, 20, 3, "t4"),          # ragged N, three stages
    (256, 4096, 2, 41, 9, "normal"),      # B = 9: two MMA n-tiles
    (64, 1000, 2, 10, 4, "normal"),       # K % 128 != 0
    (48, 512, 1, 0, 1, "normal"),         # S = 1, no protection
    (32, 640, 2, 640, 2, "normal"),       # every column protected
    (16, 128, 3, 2, 16, "t4"),            # one slab, ragged slab
    (200, 2176, 2, 23, 8, "t4"),          # K not a multiple of the 512 slab
])
def test_gemv_matches_oracle(env, N, K, S, p, B, dist):
    W = synth.layer_weights(N, K, seed=N + K, dist=dist)
    X = synth.activations(B, K, seed=B)
    Lref = oracle.encode(W, S=S, p=p)
    y = run_gemv(env, Lref, X)
    assert_parity(y, oracle.gemv(Lref, X), gemv_tight(B))


@pytest.mark.parametrize("plan", ["1,1,0,4", "2,2,0,4", "4,4,3,4", "2,1,2,2", "4,3,2,2",
                                  "4,8,2,1", "8,1,0,1", "1,2,0,2", "2,5,3,2", "4,1,8,1"])
@pytest.mark.parametrize("B", [1, 5, 16])
def test_gemv_every_tiling(env, plan, B):
    """Every tile height and slot width of the clustered kernel, cluster
    split-K factors (including ranks left with no columns) and ring depths
    give the same answer."""
    N, K, S, p = 208, 4096, 2, 41
    W = synth.layer_weights(N, K, seed=2)
    X = synth.activations(B, K, seed=3)
    Lref = oracle.encode(W, S=S, p=p)
    y = run_gemv(env, Lref, X, plan=plan)
    assert_parity(y, oracle.gemv(Lref, X), TIGHT_MMA)       # the clustered kernel decodes by MMA


@pytest.mark.parametrize("N,K,S,p,B,nslot", [
    (100, 1536, 3, 20, 3, 2),      # one tile per CTA, ragged rows, K not a slot multiple
    (208, 4096, 2, 41, 1, 3),      # odd ring depth
    (64, 640, 1, 0, 8, 2),         # no protection, B = 8
    (2500, 1024, 2, 11, 1, 2),     # several tiles per CTA, ring wraps across tiles
    (2500, 1024, 2, 11, 5, 7),
    (2500, 2176, 3, 23, 2, 4),     # a slot straddles the end of K
    (5000, 512, 2, 300, 1, 5),     # three q8 boxes per tile, many tiles per CTA
    (2500, 1024, 2, 11, 16, 3),    # batch 16: two MMA n-tiles
    (2500, 2176, 3, 23, 12, 2),    # batch 12, K not a slot multiple
    (300, 4096, 2, 41, 9, 3),      # batch 9: second n-tile one row wide
])
def test_gemv_streaming_path(env, N, K, S, p, B, nslot):
    """The persistent streaming kernel (reducer warp, int8 slab double
    buffer, ring carried across tiles) at forced ring depths."""
    W = synth.layer_weights(N, K, seed=N + p)
    X = synth.activations(B, K, seed=B + 1)
    Lref = oracle.encode(W, S=S, p=p)
    y = run_gemv(env, Lref, X, extra_env={"BISCO_GEMV_MODE": "stream",
                                         "BISCO_GEMV_NSLOT": str(nslot)})
    assert_parity(y, oracle.gemv(Lref, X), gemv_tight(B))


@pytest.mark.parametrize("name,S,rho,B", [("q_proj", 2, 1, 1), ("q_proj", 2, 1, 16),
                                          ("k_proj", 2, 1, 1), ("o_proj", 2, 1, 4),
                                          ("gate_proj", 3, 2, 1), ("down_proj", 3, 2, 1),
                                          ("down_proj", 2, 1, 16)])
def test_gemv_full_size_sampled_rows(env, name, S, rho, B):
    N, K = synth.QWEN3_8B_SHAPES[name]
    p = synth.protected_count(K, rho)
    W = synth.layer_weights(N, K, seed=17, dist="t4" if S == 3 else "normal")
    X = synth.activations(B, K, seed=18)
    Lref = oracle.encode(W, S=S, p=p)
    y = run_gemv(env, Lref, X)
    rows = sample_rows(N)
    assert_parity(y[:, rows], oracle.apply_rows(Lref, rows, X), gemv_tight(B))


def test_gemv_one_hot_columns_and_linearity(env):
    """One-hot activations return columns of What (the protected ones exactly
    scale * q8); the map is linear in x."""
    N, K, S, p = 64, 512, 2, 6
    W = synth.layer_weights(N, K, seed=5)
    Lref = oracle.encode(W, S=S, p=p)
    cols = [0, 7, 255, 511, int(Lref["idx"][0]), int(Lref["idx"][-1])]
    X = np.zeros((len(cols), K), np.uint16)
    for b, j in enumerate(cols):
        X[b, j] = 0x3F80                                   # 1.0
    y = run_gemv(env, Lref, X)
    What = oracle.decode_rows(Lref)
    for b, j in enumerate(cols):
        assert np.allclose(y[b], What[:, j], rtol=0, atol=1e-6 * np.abs(What[:, j]).max())
    X2 = synth.activations(2, K, seed=6)
    y2 = run_gemv(env, Lref, X2)
    ref = oracle.gemv(Lref, X2)
    assert_parity(y2, ref, TIGHT_MMA)


def test_gemv_zero_and_tiny_activations(env):
    N, K, S, p = 32, 256, 2, 3
    W = synth.layer_weights(N, K, seed=8)
    Lref = oracle.encode(W, S=S, p=p)
    y = run_gemv(env, Lref, np.zeros((2, K), np.uint16))
    assert np.all(y == 0)


def _multi(env, Lrefs, X, extra_env=None):
    import torch
    bisco, dev = env
    Ls = [bisco.Layer.from_numpy(L, dev) for L in Lrefs]
    old = {k: os.environ.get(k) for k in (extra_env or {})}
    os.environ.update(extra_env or {})
    try:
        ys = bisco.bisco_gemv_multi(Ls, to_dev(X, dev))
    finally:
        for k, v in old.items():
            if v is None:
                del os.environ[k]
            else:
                os.environ[k] = v
    torch.cuda.synchronize()
    assert bisco.bisco_get_device_error() == 0
    return [y.cpu().numpy() for y in ys]


@pytest.mark.parametrize("B", [1, 3, 8, 12])
@pytest.mark.parametrize("nslot", [None, 3])
def test_gemv_multi_matches_oracle(env, B, nslot):
    """Grouped launch over layers sharing x with different N and protected
    sets (one layer unprotected); B = 12 takes the per-layer path."""
    K, S = 2048, 2
    shapes = [(300, 21), (64, 0), (1000, 33)]
    Lrefs = [oracle.encode(synth.layer_weights(N, K, seed=40 + i), S=S, p=p)
             for i, (N, p) in enumerate(shapes)]
    X = synth.activations(B, K, seed=41)
    ys = _multi(env, Lrefs, X, {"BISCO_GEMV_NSLOT": str(nslot)} if nslot else None)
    for y, L in zip(ys, Lrefs):
        assert_parity(y, oracle.gemv(L, X), gemv_tight(B))


def test_gemv_multi_qkv_full_size(env):
    """q/k/v of one Qwen3-8B attention layer in one launch, batch 1."""
    K, S = 4096, 2
    p = synth.protected_count(K, 1)
    names = ("q_proj", "k_proj", "v_proj")
    Lrefs = [oracle.encode(synth.layer_weights(synth.QWEN3_8B_SHAPES[n][0], K, seed=60 + i),
                           S=S, p=p) for i, n in enumerate(names)]
    X = synth.activations(1, K, seed=61)
    ys = _multi(env, Lrefs, X)
    for y, L, n in zip(ys, Lrefs, names):
        rows = sample_rows(L["N"], n=24)
        assert_parity(y[:, rows], oracle.apply_rows(L, rows, X), gemv_tight(1), n)


def test_gemv_multi_single_layer_matches_gemv(env):
    import torch
    bisco, dev = env
    K, S = 1024, 3
    Lref = oracle.encode(synth.layer_weights(2500, K, seed=70, dist="t4"), S=S, p=11)
    X = synth.activations(2, K, seed=71)
    (ym,) = _multi(env, [Lref], X)
    y = run_gemv(env, Lref, X)
    assert max_rel_rows(ym, y) <= 1e-5
    assert_parity(ym, oracle.gemv(Lref, X), TIGHT_MMA)


# ---------------------------------------------------------------- batch 1
# Batch 1 decodes through nibble tables of x: a launch of one layer builds
# them with its protected columns masked, a grouped launch shares unmasked
# tables and removes each layer's protected BSQ terms afterwards.  Both are
# checked where the layout has edges: protected columns on chunk and ring-slot
# boundaries (2048-column slots), whole protected chunks, K not a slot multiple.

def _boosted(N, K, cols, seed, S_dist="normal"):
    """Weights whose protected set (Eq. 8 top-p) is exactly `cols`."""
    W = synth.layer_weights(N, K, seed=seed, dist=S_dist, n_outliers=0)
    w = synth.bf16_bits_to_f32(W).astype(np.float64)
    w[:, cols] *= 50.0
    return synth.f32_to_bf16_bits(w.astype(np.float32))


BOUNDARY_COLS = [0, 7, 8, 15, 2040, 2041, 2042, 2043, 2044, 2045, 2046, 2047, 2048, 2055, 4095]


@pytest.mark.parametrize("K,S", [(4096, 2), (4096, 3), (2176, 2)])
def test_gemv_table_decode_protected_on_boundaries(env, K, S):
    cols = [c for c in BOUNDARY_COLS if c < K]
    Lref = oracle.encode(_boosted(2500, K, cols, seed=80 + K), S=S, p=len(cols))
    assert sorted(Lref["idx"].tolist()) == cols
    X = synth.activations(1, K, seed=81)
    y = run_gemv(env, Lref, X)
    assert_parity(y, oracle.gemv(Lref, X), gemv_tight(1))


def test_gemv_table_decode_grouped_correction_on_boundaries(env):
    """Grouped launch: shared unmasked tables, per-layer correction of the
    protected BSQ terms, with protected sets that differ between layers."""
    K, S = 4096, 2
    sets = [BOUNDARY_COLS, [1, 2047, 2049, 3000], []]
    Lrefs = []
    for i, cols in enumerate(sets):
        W = _boosted(400 + 300 * i, K, cols, seed=90 + i) if cols else \
            synth.layer_weights(400 + 300 * i, K, seed=90 + i)
        Lrefs.append(oracle.encode(W, S=S, p=len(cols)))
    X = synth.activations(1, K, seed=93)
    ys = _multi(env, Lrefs, X)
    for y, L in zip(ys, Lrefs):
        assert_parity(y, oracle.gemv(L, X), gemv_tight(1))


def test_gemv_multi_fully_protected_layer(env):
    """A layer with every column protected (its tables are all correction)
    next to an unprotected one, batch 1."""
    K, S = 512, 2
    Lrefs = [oracle.encode(synth.layer_weights(300, K, seed=95), S=S, p=K),
             oracle.encode(synth.layer_weights(200, K, seed=96), S=S, p=0)]
    X = synth.activations(1, K, seed=97)
    ys = _multi(env, Lrefs, X)
    for y, L in zip(ys, Lrefs):
        assert_parity(y, oracle.gemv(L, X), gemv_tight(1))


@pytest.mark.parametrize("N,K,S,p", [(2500, 4096, 2, 41), (2500, 2176, 3, 23), (300, 1024, 1, 11)])
def test_gemv_batch1_both_decodes(env, N, K, S, p):
    """Batch 1 through the table decode and through the MMA decode
    (BISCO_GEMV_LUT=0) on the streaming kernel: both meet the bar."""
    W = synth.layer_weights(N, K, seed=N + K + S)
    X = synth.activations(1, K, seed=98)
    Lref = oracle.encode(W, S=S, p=p)
    ref = oracle.gemv(Lref, X)
    for lut in ("1", "0"):
        y = run_gemv(env, Lref, X, extra_env={"BISCO_GEMV_MODE": "stream", "BISCO_GEMV_LUT": lut})
        assert_parity(y, ref, gemv_tight(1, tables=lut == "1"), lut)


def test_gemv_batch1_zero_activations(env):
    N, K, S, p = 2500, 2048, 2, 21
    Lref = oracle.encode(synth.layer_weights(N, K, seed=99), S=S, p=p)
    y = run_gemv(env, Lref, np.zeros((1, K), np.uint16))
    assert np.all(y == 0)


# ------------------------------------------------- batch 1, row-split kernel
# K a multiple of 4096 at batch 1 goes to the row-split kernel: each layer
# of a launch gets whole CTAs, each CTA a run of rows that it walks span by
# span (4096 columns, one table at a time), each warp a run of the CTA's
# items through its own ring of bulk copies.  The cases cover rows fewer
# than SMs, ragged row runs, S = 1..3, K = 4096 / 8192 / 12288, layers
# without protection, int8 rows too large to stage in shared memory, and
# groups of several layers.

@pytest.mark.parametrize("N,K,S,p", [
    (16, 4096, 1, 0),          # 16 rows: 16 one-row CTAs
    (150, 4096, 2, 41),        # one row per CTA, two left idle
    (153, 4096, 3, 41),        # 152 CTAs, one with two rows
    (1000, 4096, 2, 0),        # no protection
    (2500, 4096, 3, 82),       # ragged row runs, S = 3
    (500, 8192, 2, 82),        # two 4096-column spans per stage
    (300, 12288, 2, 123),      # three spans (down_proj width)
    (4000, 4096, 2, 2000),     # int8 rows read from global memory at the end
])
def test_gemv_b1_matches_oracle(env, N, K, S, p):
    W = synth.layer_weights(N, K, seed=N + K + S + p, dist="t4" if S == 3 else "normal")
    X = synth.activations(1, K, seed=N + 5)
    Lref = oracle.encode(W, S=S, p=p)
    y = run_gemv(env, Lref, X)
    assert_parity(y, oracle.gemv(Lref, X), gemv_tight(1))
    # the same bits on a second call (no atomics, a fixed summation order)
    assert np.array_equal(y, run_gemv(env, Lref, X))


@pytest.mark.parametrize("K,shapes", [
    (4096, [(300, 21), (64, 0), (1000, 33)]),                 # layers of unequal row counts
    (4096, [(4096, 41), (1024, 41), (1024, 41)]),             # q/k/v of one attention layer
    (4096, [(3000, 41), (2000, 0), (1500, 41), (4000, 10)]),  # four layers
    (4096, [(200, 5), (7, 3), (150, 0)]),                     # a 7-row layer between larger ones
    (12288, [(700, 123), (90, 0), (333, 60)]),                # three spans, three layers
    (4096, [(12288, 41), (12288, 41)]),                       # gate/up: two CTAs per SM (the step's dominant call)
])
def test_gemv_b1_groups_match_oracle(env, K, shapes):
    S = 2
    Lrefs = [oracle.encode(synth.layer_weights(N, K, seed=200 + i), S=S, p=p)
             for i, (N, p) in enumerate(shapes)]
    X = synth.activations(1, K, seed=201)
    ys = _multi(env, Lrefs, X)
    for y, L in zip(ys, Lrefs):
        rows = sample_rows(L["N"], n=64) if L["N"] > 2000 else np.arange(L["N"], dtype=np.int32)
        assert_parity(y[:, rows], oracle.apply_rows(L, rows, X), gemv_tight(1))


def test_gemv_b1_equals_streaming_kernel(env):
    """The row-split kernel and the streaming kernel's table decode (same
    tables, other summation order) agree far inside the table bound."""
    N, K, S, p = 2500, 4096, 2, 41
    Lref = oracle.encode(synth.layer_weights(N, K, seed=211), S=S, p=p)
    X = synth.activations(1, K, seed=212)
    y1 = run_gemv(env, Lref, X)
    y0 = run_gemv(env, Lref, X, extra_env={"BISCO_GEMV_B1": "0"})
    assert max_rel_rows(y1, y0) <= 2e-5
