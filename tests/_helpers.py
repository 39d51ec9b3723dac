"""Shared test helpers (no method arithmetic)."""
import numpy as np

# Parity bar for floating-point outputs: per activation row b,
#   max_i |y_gpu[b,i] - y_ref[b,i]| / max_i |y_ref[b,i]| <= 2e-3
# against the fp64 oracle.
TOL = 2e-3


def max_rel_rows(y, ref):
    y = np.atleast_2d(np.asarray(y, np.float64))
    ref = np.atleast_2d(np.asarray(ref, np.float64))
    assert y.shape == ref.shape, (y.shape, ref.shape)
    errs = [np.abs(y[b] - ref[b]).max() / max(np.abs(ref[b]).max(), 1e-30)
            for b in range(ref.shape[0])]
    return float(max(errs)) if errs else 0.0


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
