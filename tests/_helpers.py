"""Shared test helpers (no method arithmetic)."""
import numpy as np

# Parity bar for floating-point outputs: per activation row b,
#   max_i |y_gpu[b,i] - y_ref[b,i]| / max_i |y_ref[b,i]| <= 2e-3
# against the fp64 oracle.
TOL = 2e-3

# Tighter bounds, one per decode arithmetic, beside the bar above.  One
# mis-signed element of a stage, a dropped chunk-stage or a wrong protected
# term moves a row's error by about 2e-3 of max|y| on these layers, which is
# at the bar; each bound below sits well under that and a few times above
# what its path's rounding gives.
#
# MMA decode (batch >= 2, and batch 1 with the tables switched off): every
# product n16 * (+-1) * x is exact in the fp16 x fp16 -> fp32 MMA (x is bf16
# used as fp16, exact for these magnitudes), protected terms are q8 (exact
# fp16 integers) times scale * x split into fp16 hi + lo (2^-22 relative),
# and only the fp32 sums round: a random walk of K / 16 MMA k-steps of
# 2^-24 relative roundings, a few 1e-6 of max|y|.
TIGHT_MMA = 2e-5
# Batch-1 table decode: each signed half-sum of four activations is one
# fp16 rounding (2^-11 relative, sigma 2^-11 / sqrt(3)) before it meets the
# exact fp16 norm; summed over K / 8 * S chunk-stages that is a random walk
# of the same growth as y itself, about 1-3e-4 of max|y| (the CPU emulation
# in test_numerics_model.py measures 1.1-1.9e-4 at full q_proj and down_proj
# size).
TIGHT_TABLE = 5e-4
# Prefill GEMM on the tensor cores: the S decoded stages of a weight are
# added in fp16 before the MMA, S - 1 roundings of 2^-11 relative each per
# weight (exact for S = 1); the same random walk gives about
# 2^-11 * sqrt((S - 1) / 3) = 2.8e-4 (S = 2) and 4e-4 (S = 3).
TIGHT_GEMM = 8e-4


def gemv_tight(B, tables=True):
    """The bound of bisco_gemv at batch B (tables: the batch-1 table decode
    may run)."""
    return TIGHT_TABLE if (B == 1 and tables) else TIGHT_MMA


def gemm_tight(M, K):
    """The bound of bisco_gemm: the tensor-core path for M > 16 and
    K % 128 == 0, otherwise the decode kernels of bisco_gemv."""
    return TIGHT_GEMM if (M > 16 and K % 128 == 0) else gemv_tight(M)


def max_rel_rows(y, ref):
    y = np.atleast_2d(np.asarray(y, np.float64))
    ref = np.atleast_2d(np.asarray(ref, np.float64))
    assert y.shape == ref.shape, (y.shape, ref.shape)
    errs = [np.abs(y[b] - ref[b]).max() / max(np.abs(ref[b]).max(), 1e-30)
            for b in range(ref.shape[0])]
    return float(max(errs)) if errs else 0.0


def assert_parity(y, ref, tight, what=""):
    """The 2e-3 bar and the path's own tighter bound."""
    err = max_rel_rows(y, ref)
    assert err <= TOL, f"{what} max-rel {err:.3e} above the 2e-3 bar"
    assert err <= tight, f"{what} max-rel {err:.3e} above the path bound {tight:.1e}"
    return err


def to_dev(a, dev):
    import torch
    a = np.ascontiguousarray(a)
    if a.dtype == np.uint16:
        a = a.view(np.int16)
    return torch.from_numpy(a).to(dev)


def sample_rows(N, n=48, seed=0):
    rng = np.random.default_rng(seed)
    rows = set([0, N - 1, N // 2]) | set(rng.choice(N, size=min(n, N), replace=False).tolist())
    return np.array(sorted(rows), np.int32)


def rows_per_tile(N, tile, per=2, seed=0):
    """`per` rows from every `tile`-row block of N (first and last rows
    included), so a sampled check reaches every tile of a kernel."""
    rng = np.random.default_rng(seed)
    rows = {0, N - 1}
    for t0 in range(0, N, tile):
        n = min(tile, N - t0)
        rows |= set((t0 + rng.choice(n, size=min(per, n), replace=False)).tolist())
    return np.array(sorted(rows), np.int32)
