"""fp64 CPU oracle for the BiSCo-LLM hot path -- TEST INFRASTRUCTURE ONLY.

Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import this package.  The product library never loads it and
shares no code with it.  The arithmetic lives in ``bisco_oracle.c`` (plain C,
binary64, ``-ffp-contract=off``); this module compiles it with gcc and
marshals numpy arrays through ctypes.

Functions and the paper passages they follow:

* :func:`encode`            Sec. III-E Eq. 8 (protected columns), Eq. 10 (Q8),
                            Sec. III-C Eq. 3 and Sec. III-D Eq. 5-7 (stages)
* :func:`select_protected`  Eq. 8
* :func:`decode_rows`       Sec. III-G Eq. 12 with the Eq. 10 scatter
* :func:`matmul`            y = What x (plain definition)
* :func:`select_rows`, :func:`select_coupled`, :func:`encode_rows`,
  :func:`encode_given`, :func:`encode_coupled`
                            output-row protection and the coupled MLP
                            channel score (Sec. III-E Eq. 9) with Eq. 10 on
                            rows (the CUDA library's protect_axis = 1 and
                            bisco_select_coupled are checked against these)
* :func:`double_to_fp8`, :func:`fp8_to_double`, :func:`quantize_protected_fmt`,
  :func:`quantize_protected_rows_fmt`, :func:`protected_values_fmt`
                            FP8 E4M3 / E5M2 and BF16 protected payloads (the
                            paper's protected-format ablation) as variants of
                            Eq. 10, on protected columns or rows
* :func:`decoder_table_linear`, :func:`decoder_table_mlp`, :func:`decode_rows_table`
                            the decoder step of Eq. 1 as a table over the 256
                            code bytes (linear, or odd tanh perceptron with an
                            optional residual block), decoded per Eq. 12 (the
                            CUDA library's bisco_gemv_table and
                            bisco_decode_dense_table are checked against these)
* :func:`lora_apply`        y0 + scale * Bm (A x), the optional low-rank
                            compensation of Sec. III-F (plain definition)
* :func:`apply_rows`        decode + matmul on a list of rows
* :func:`double_to_fp16`, :func:`fp16_to_double`, :func:`bf16_to_double`
                            the number formats the storage uses

Parity status: every function is pinned by ``tests/test_oracle_pins.py``
except whole-model quality, which needs trained codecs and real checkpoints
(parity unpinned, out of scope).
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "bisco_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_LIB = os.path.join(_BUILD, "libbisco_oracle.so")
_lock = threading.Lock()
_lib = None
# Tests that plant a mistake in a copy of bisco_oracle.c point this at the
# copy's build, to check that the pins catch it.
_LIB_OVERRIDE = os.environ.get("BISCO_ORACLE_LIB")

OK, ERR_INVALID_ARG, ERR_RANGE = 0, 1, 3
FMT_INT8, FMT_E4M3, FMT_E5M2, FMT_BF16 = 0, 1, 2, 3

CFLAGS = ["-O2", "-std=c11", "-ffp-contract=off", "-fno-fast-math", "-fPIC", "-shared"]


def build(force: bool = False) -> str:
    """Compile bisco_oracle.c into _build/libbisco_oracle.so (gcc, fp64)."""
    os.makedirs(_BUILD, exist_ok=True)
    if (not force and os.path.exists(_LIB)
            and os.path.getmtime(_LIB) >= os.path.getmtime(_SRC)):
        return _LIB
    tmp = _LIB + ".%d.tmp" % os.getpid()
    subprocess.check_call(["gcc", *CFLAGS, "-o", tmp, _SRC, "-lm"])
    os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        lib = ctypes.CDLL(_LIB_OVERRIDE or build())
        P = ctypes.c_void_p
        i32, i64 = ctypes.c_int32, ctypes.c_int64
        lib.or_bf16_to_double.restype = ctypes.c_double
        lib.or_bf16_to_double.argtypes = [ctypes.c_uint16]
        lib.or_fp16_to_double.restype = ctypes.c_double
        lib.or_fp16_to_double.argtypes = [ctypes.c_uint16]
        lib.or_double_to_fp16.restype = ctypes.c_uint16
        lib.or_double_to_fp16.argtypes = [ctypes.c_double]
        lib.or_pad16.restype = i32
        lib.or_pad16.argtypes = [i32]
        lib.or_encoded_sizes.restype = ctypes.c_int
        lib.or_encoded_sizes.argtypes = [i32, i32, i32, i32, P]
        lib.or_select_protected.restype = ctypes.c_int
        lib.or_select_protected.argtypes = [P, P, i32, i32, i32, P, P]
        lib.or_quantize_protected.restype = ctypes.c_int
        lib.or_quantize_protected.argtypes = [P, i32, i32, P, i32, P, P]
        lib.or_encode_stages.restype = ctypes.c_int
        lib.or_encode_stages.argtypes = [P, i32, i32, i32, P, i32, P, P]
        lib.or_encode.restype = ctypes.c_int
        lib.or_encode.argtypes = [P, P, i32, i32, i32, i32, P, P, P, P, P]
        lib.or_decode_rows.restype = None
        lib.or_decode_rows.argtypes = [P, P, P, P, P, i32, i32, i32, i32, i32, i32, P]
        lib.or_matmul.restype = None
        lib.or_matmul.argtypes = [P, i32, i32, P, i32, P]
        lib.or_apply_rows.restype = ctypes.c_int
        lib.or_apply_rows.argtypes = [P, P, P, P, P, i32, i32, i32, i32, P, i32, P, i32, P]
        lib.or_select_rows.restype = ctypes.c_int
        lib.or_select_rows.argtypes = [P, P, i32, i32, i32, P, P]
        lib.or_select_coupled.restype = ctypes.c_int
        lib.or_select_coupled.argtypes = [P, P, P, P, P, P, i32, i32, i32, P, P]
        lib.or_quantize_protected_rows.restype = ctypes.c_int
        lib.or_quantize_protected_rows.argtypes = [P, i32, i32, P, i32, P, P]
        lib.or_encode_rows.restype = ctypes.c_int
        lib.or_encode_rows.argtypes = [P, P, i32, i32, i32, i32, P, P, P, P, P, P]
        lib.or_decode_rows_axis1.restype = None
        lib.or_decode_rows_axis1.argtypes = [P, P, P, P, P, i32, i32, i32, i32, i32, i32, P]
        lib.or_double_to_fp8.restype = ctypes.c_uint8
        lib.or_double_to_fp8.argtypes = [ctypes.c_double, ctypes.c_int]
        lib.or_fp8_to_double.restype = ctypes.c_double
        lib.or_fp8_to_double.argtypes = [ctypes.c_uint8, ctypes.c_int]
        lib.or_quantize_protected_fmt.restype = ctypes.c_int
        lib.or_quantize_protected_fmt.argtypes = [P, i32, i32, P, i32, ctypes.c_int, P, P]
        lib.or_protected_value_fmt.restype = ctypes.c_double
        lib.or_protected_value_fmt.argtypes = [P, P, i32, ctypes.c_int, i32, i32]
        lib.or_decoder_table_linear.restype = None
        lib.or_decoder_table_linear.argtypes = [P, P]
        lib.or_decoder_table_mlp.restype = ctypes.c_int
        lib.or_decoder_table_mlp.argtypes = [P, i32, P, P, P]
        lib.or_decode_rows_table.restype = None
        lib.or_decode_rows_table.argtypes = [P, P, P, P, P, P, i32, i32, i32, i32, i32, i32, P]
        lib.or_lora_apply.restype = ctypes.c_int
        lib.or_lora_apply.argtypes = [P, P, i32, i32, i32, ctypes.c_double, P, i32, P, P]
        del i64
        _lib = lib
        return lib


def _ptr(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _c(a, dtype):
    return np.ascontiguousarray(a, dtype=dtype)


class OracleError(RuntimeError):
    def __init__(self, code):
        super().__init__("oracle status %d" % code)
        self.code = code


# ------------------------------------------------------------------ numbers

def bf16_to_double(b: int) -> float:
    return _load().or_bf16_to_double(int(b))


def fp16_to_double(h: int) -> float:
    return _load().or_fp16_to_double(int(h))


def double_to_fp16(x: float) -> int:
    return int(_load().or_double_to_fp16(float(x)))


def pad16(p: int) -> int:
    return (p + 15) // 16 * 16


def encoded_sizes(N, K, S, p):
    out = np.zeros(5, np.int64)
    rc = _load().or_encoded_sizes(N, K, S, p, _ptr(out))
    if rc:
        raise OracleError(rc)
    return [int(v) for v in out]


# ------------------------------------------------------------------ encode

def select_protected(W_bits, p, g=None):
    """Eq. 8: returns (idx ascending int32[p], scores float64[K])."""
    W_bits = _c(W_bits, np.uint16)
    N, K = W_bits.shape
    idx = np.zeros(max(p, 1), np.int32)
    scores = np.zeros(K, np.float64)
    gg = None if g is None else _c(g, np.float32)
    rc = _load().or_select_protected(_ptr(W_bits), _ptr(gg), N, K, p, _ptr(idx), _ptr(scores))
    if rc:
        raise OracleError(rc)
    return idx[:p].copy(), scores


def encode(W_bits, S, p, g=None):
    """Whole encoder.  W_bits: uint16[N][K] bf16 bit patterns.

    Returns a dict with codes uint8[S][N][K/8], norms uint16[S][N][K/8],
    q8 int8[N][pad16(p)], scale uint16[p], idx int32[p]."""
    W_bits = _c(W_bits, np.uint16)
    N, K = W_bits.shape
    C = K // 8 if K % 8 == 0 else 1
    codes = np.zeros((S, N, C), np.uint8)
    norms = np.zeros((S, N, C), np.uint16)
    q8 = np.zeros((N, max(pad16(p), 16)), np.int8)
    scale = np.zeros(max(p, 1), np.uint16)
    idx = np.zeros(max(p, 1), np.int32)
    gg = None if g is None else _c(g, np.float32)
    rc = _load().or_encode(_ptr(W_bits), _ptr(gg), N, K, S, p, _ptr(codes), _ptr(norms),
                           _ptr(q8), _ptr(scale), _ptr(idx))
    if rc:
        raise OracleError(rc)
    return dict(N=N, K=K, S=S, p=p, codes=codes, norms=norms,
                q8=q8[:, :pad16(p)].copy(), scale=scale[:p].copy(), idx=idx[:p].copy())


def select_rows(W_bits, p, g=None):
    """Output-row selection: returns (idx ascending int32[p], scores float64[N])."""
    W_bits = _c(W_bits, np.uint16)
    N, K = W_bits.shape
    idx = np.zeros(max(p, 1), np.int32)
    scores = np.zeros(N, np.float64)
    gg = None if g is None else _c(g, np.float32)
    rc = _load().or_select_rows(_ptr(W_bits), _ptr(gg), N, K, p, _ptr(idx), _ptr(scores))
    if rc:
        raise OracleError(rc)
    return idx[:p].copy(), scores


def select_coupled(Wg_bits, Wu_bits, Wd_bits, p, gg=None, gu=None, gd=None):
    """Eq. 9: the coupled intermediate-channel set of a gated MLP (gate/up
    [F][H], down [H][F]).  Returns (idx ascending int32[p], scores float64[F])."""
    Wg_bits, Wu_bits, Wd_bits = (_c(w, np.uint16) for w in (Wg_bits, Wu_bits, Wd_bits))
    F, H = Wg_bits.shape
    if Wu_bits.shape != (F, H) or Wd_bits.shape != (H, F):
        raise OracleError(ERR_INVALID_ARG)
    idx = np.zeros(max(p, 1), np.int32)
    scores = np.zeros(F, np.float64)
    g3 = [None if g is None else _c(g, np.float32) for g in (gg, gu, gd)]
    rc = _load().or_select_coupled(_ptr(Wg_bits), _ptr(Wu_bits), _ptr(Wd_bits), _ptr(g3[0]),
                                   _ptr(g3[1]), _ptr(g3[2]), F, H, p, _ptr(idx), _ptr(scores))
    if rc:
        raise OracleError(rc)
    return idx[:p].copy(), scores


def encode_rows(W_bits, S, p, g=None, idx=None):
    """Encoder with output-row protection (axis 1).  The protected rows come
    from :func:`select_rows` unless ``idx`` gives them.  Returns a dict like
    :func:`encode` with axis=1, q8 int8[p][pad16(K)], scale/idx per row."""
    W_bits = _c(W_bits, np.uint16)
    N, K = W_bits.shape
    C = K // 8 if K % 8 == 0 else 1
    kp = pad16(K)
    codes = np.zeros((S, N, C), np.uint8)
    norms = np.zeros((S, N, C), np.uint16)
    q8 = np.zeros((max(p, 1), kp), np.int8)
    scale = np.zeros(max(p, 1), np.uint16)
    out_idx = np.zeros(max(p, 1), np.int32)
    gg = None if g is None else _c(g, np.float32)
    given = None if idx is None else _c(idx, np.int32)
    if given is not None and len(given) != p:
        raise OracleError(ERR_INVALID_ARG)
    rc = _load().or_encode_rows(_ptr(W_bits), _ptr(gg), N, K, S, p, _ptr(given), _ptr(codes),
                                _ptr(norms), _ptr(q8), _ptr(scale), _ptr(out_idx))
    if rc:
        raise OracleError(rc)
    return dict(N=N, K=K, S=S, p=p, axis=1, codes=codes, norms=norms, q8=q8[:p].copy(),
                scale=scale[:p].copy(), idx=out_idx[:p].copy())


def encode_given(W_bits, S, idx):
    """Column protection (axis 0) with a given ascending column set, e.g. the
    down projection's share of the coupled MLP set: Eq. 10 on those columns,
    then the stages on the masked complement."""
    W_bits = _c(W_bits, np.uint16)
    N, K = W_bits.shape
    idx = _c(idx, np.int32)
    p = len(idx)
    if (K % 8 or np.any(idx < 0) or np.any(idx >= K) or np.any(np.diff(idx) <= 0)):
        raise OracleError(ERR_INVALID_ARG)
    if not np.all(np.isfinite(_bf16_bits_to_f64(W_bits))):
        raise OracleError(ERR_RANGE)
    q8 = np.zeros((N, max(pad16(p), 16)), np.int8)
    scale = np.zeros(max(p, 1), np.uint16)
    codes = np.zeros((S, N, K // 8), np.uint8)
    norms = np.zeros((S, N, K // 8), np.uint16)
    lib = _load()
    idx_arg = idx if p else np.zeros(1, np.int32)
    rc = lib.or_quantize_protected(_ptr(W_bits), N, K, _ptr(idx_arg), p, _ptr(q8), _ptr(scale))
    if rc == 0:
        rc = lib.or_encode_stages(_ptr(W_bits), N, K, S, _ptr(idx_arg), p, _ptr(codes), _ptr(norms))
    if rc:
        raise OracleError(rc)
    return dict(N=N, K=K, S=S, p=p, codes=codes, norms=norms, q8=q8[:, :pad16(p)].copy(),
                scale=scale[:p].copy(), idx=idx.copy())


def encode_coupled(Wg_bits, Wu_bits, Wd_bits, S, p):
    """Eq. 9 + Eq. 10 for a gated MLP: one protected intermediate set P
    (:func:`select_coupled`), the rows P of gate and up and the columns P of
    down kept in 8 bits.  Returns (gate, up, down) layer dicts."""
    idx, _ = select_coupled(Wg_bits, Wu_bits, Wd_bits, p)
    return (encode_rows(Wg_bits, S, p, idx=idx), encode_rows(Wu_bits, S, p, idx=idx),
            encode_given(Wd_bits, S, idx))


def _bf16_bits_to_f64(bits):
    """bf16 bit patterns -> float64 (exact), without importing the generators."""
    return (np.asarray(bits, np.uint16).astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def _layer_args(L):
    codes = _c(L["codes"], np.uint8)
    norms = _c(L["norms"], np.uint16)
    q8 = _c(L["q8"], np.int8) if L["p"] > 0 else np.zeros((L["N"], 16), np.int8)
    scale = _c(L["scale"], np.uint16) if L["p"] > 0 else np.zeros(1, np.uint16)
    idx = _c(L["idx"], np.int32) if L["p"] > 0 else np.zeros(1, np.int32)
    return codes, norms, q8, scale, idx


def decode_rows(L, row0=0, nrows=None):
    """Eq. 12 + Eq. 10: dense float64 rows [row0, row0+nrows) of What (input
    columns protected, or output rows for a layer with axis=1)."""
    N, K = L["N"], L["K"]
    if nrows is None:
        nrows = N - row0
    out = np.zeros((nrows, K), np.float64)
    if L.get("axis", 0) == 1:
        codes = _c(L["codes"], np.uint8)
        norms = _c(L["norms"], np.uint16)
        p = L["p"]
        q8 = _c(L["q8"], np.int8) if p > 0 else np.zeros((1, pad16(K)), np.int8)
        scale = _c(L["scale"], np.uint16) if p > 0 else np.zeros(1, np.uint16)
        idx = _c(L["idx"], np.int32) if p > 0 else np.zeros(1, np.int32)
        _load().or_decode_rows_axis1(_ptr(codes), _ptr(norms), _ptr(q8), _ptr(scale), _ptr(idx),
                                     N, K, L["S"], p, row0, nrows, _ptr(out))
        return out
    codes, norms, q8, scale, idx = _layer_args(L)
    _load().or_decode_rows(_ptr(codes), _ptr(norms), _ptr(q8), _ptr(scale), _ptr(idx),
                           N, K, L["S"], L["p"], row0, nrows, _ptr(out))
    return out


def matmul(What, X_bits):
    """y[b][i] = sum_j What[i][j] * x[b][j] in float64 (X_bits: bf16 bits)."""
    What = _c(What, np.float64)
    X_bits = _c(np.atleast_2d(X_bits), np.uint16)
    nrows, K = What.shape
    B = X_bits.shape[0]
    Y = np.zeros((B, nrows), np.float64)
    _load().or_matmul(_ptr(What), nrows, K, _ptr(X_bits), B, _ptr(Y))
    return Y


def double_to_fp8(x: float, fmt: int) -> int:
    """FP8 bits of x (FMT_E4M3 / FMT_E5M2): nearest even, saturating."""
    return int(_load().or_double_to_fp8(float(x), int(fmt)))


def fp8_to_double(v: int, fmt: int) -> float:
    return _load().or_fp8_to_double(int(v), int(fmt))


def quantize_protected_fmt(W_bits, idx, fmt):
    """Eq. 10 with the protected payload in format ``fmt``: returns
    (q [N][pad16(p)] uint8 FP8 bits / uint16 bf16 bits / int8, scale uint16[p])."""
    W_bits = _c(W_bits, np.uint16)
    N, K = W_bits.shape
    idx = _c(idx, np.int32)
    p = len(idx)
    pp = max(pad16(p), 16)
    dt = {FMT_INT8: np.int8, FMT_E4M3: np.uint8, FMT_E5M2: np.uint8, FMT_BF16: np.uint16}[fmt]
    q = np.zeros((N, pp), dt)
    scale = np.zeros(max(p, 1), np.uint16)
    idx_arg = idx if p else np.zeros(1, np.int32)
    if fmt == FMT_INT8:
        rc = _load().or_quantize_protected(_ptr(W_bits), N, K, _ptr(idx_arg), p, _ptr(q), _ptr(scale))
    else:
        rc = _load().or_quantize_protected_fmt(_ptr(W_bits), N, K, _ptr(idx_arg), p, int(fmt),
                                               _ptr(q), _ptr(scale))
    if rc:
        raise OracleError(rc)
    return q[:, :pad16(p)].copy(), scale[:p].copy()


def quantize_protected_rows_fmt(W_bits, idx, fmt):
    """Eq. 10 on protected output rows with the payload in format ``fmt``
    (the row axis of Eq. 9 under the protected-format ablation): row i of W
    is column i of W^T, so this is :func:`quantize_protected_fmt` on the
    transpose.  Returns (q [p][pad16(K)], scale uint16[p]); one scale per
    row, zero padding past K."""
    W_bits = _c(W_bits, np.uint16)
    N, K = W_bits.shape
    idx = _c(idx, np.int32)
    p = len(idx)
    qt, scale = quantize_protected_fmt(np.ascontiguousarray(W_bits.T), idx, fmt)
    q = np.zeros((p, pad16(K)), qt.dtype)
    q[:, :K] = qt[:, :p].T
    return q, scale


def protected_values_fmt(q, scale, fmt):
    """Decoded protected values [N][p] = scale_t * value(q[i][t])."""
    q = np.ascontiguousarray(q)
    scale = _c(scale, np.uint16)
    N, pp = q.shape
    p = len(scale)
    assert pp == pad16(p)
    out = np.zeros((N, p), np.float64)
    lib = _load()
    for i in range(N):
        for t in range(p):
            out[i, t] = lib.or_protected_value_fmt(_ptr(q), _ptr(scale), p, int(fmt), i, t)
    return out


def decoder_table_linear(A):
    """Table [256][8] (float64) of the linear decoder D(q) = A q, A [8][8]."""
    A = _c(A, np.float64)
    assert A.shape == (8, 8)
    T = np.zeros((256, 8), np.float64)
    _load().or_decoder_table_linear(_ptr(A), _ptr(T))
    return T


def decoder_table_mlp(W1, W2, Wr=None):
    """Table [256][8] (float64) of the odd decoder W2 (h + tanh(Wr h)),
    h = tanh(W1 q); W1 [hdim][8], W2 [8][hdim], Wr [hdim][hdim] or None
    (no residual block)."""
    W1 = _c(W1, np.float64)
    W2 = _c(W2, np.float64)
    hdim = W1.shape[0]
    assert W1.shape == (hdim, 8) and W2.shape == (8, hdim)
    if Wr is not None:
        Wr = _c(Wr, np.float64)
        assert Wr.shape == (hdim, hdim)
    T = np.zeros((256, 8), np.float64)
    rc = _load().or_decoder_table_mlp(_ptr(W1), hdim, _ptr(Wr) if Wr is not None else None,
                                      _ptr(W2), _ptr(T))
    if rc:
        raise OracleError(rc)
    return T


def table_to_fp16(T):
    """Binary16 bits of a float64 decoder table, each value rounded once
    (nearest even) by the oracle's own conversion."""
    T = np.asarray(T, np.float64)
    return np.array([double_to_fp16(float(v)) for v in T.ravel()], np.uint16).reshape(T.shape)


def decode_rows_table(L, tables16, row0=0, nrows=None):
    """Dense float64 rows of What with per-stage decoder tables
    (tables16 [S][256][8] binary16 bits): Eq. 12 with Eq. 1, and the Eq. 10
    protected columns."""
    N, K, S = L["N"], L["K"], L["S"]
    tables16 = _c(tables16, np.uint16)
    assert tables16.shape == (S, 256, 8)
    if nrows is None:
        nrows = N - row0
    out = np.zeros((nrows, K), np.float64)
    codes, norms, q8, scale, idx = _layer_args(L)
    _load().or_decode_rows_table(_ptr(codes), _ptr(norms), _ptr(tables16), _ptr(q8), _ptr(scale),
                                 _ptr(idx), N, K, S, L["p"], row0, nrows, _ptr(out))
    return out


def lora_apply(A_bits, Bm_bits, X_bits, Y0, scale=1.0):
    """Y0 + scale * (X A^T) Bm^T in float64: A [rank][K], Bm [N][rank] and
    X [B][K] as bf16 bits, Y0 [B][N]."""
    A_bits = _c(A_bits, np.uint16)
    Bm_bits = _c(Bm_bits, np.uint16)
    X_bits = _c(np.atleast_2d(X_bits), np.uint16)
    rank, K = A_bits.shape
    N = Bm_bits.shape[0]
    B = X_bits.shape[0]
    if Bm_bits.shape[1] != rank or X_bits.shape[1] != K:
        raise OracleError(ERR_INVALID_ARG)
    Y0 = _c(np.asarray(Y0, np.float64).reshape(B, N), np.float64)
    Y = np.zeros((B, N), np.float64)
    rc = _load().or_lora_apply(_ptr(A_bits), _ptr(Bm_bits), rank, N, K, float(scale),
                               _ptr(X_bits), B, _ptr(Y0), _ptr(Y))
    if rc:
        raise OracleError(rc)
    return Y


def apply_rows(L, rows, X_bits):
    """Y[b][t] = What[rows[t], :] . x_b, decoding one row at a time."""
    rows = _c(rows, np.int32)
    X_bits = _c(np.atleast_2d(X_bits), np.uint16)
    codes, norms, q8, scale, idx = _layer_args(L)
    B = X_bits.shape[0]
    Y = np.zeros((B, len(rows)), np.float64)
    rc = _load().or_apply_rows(_ptr(codes), _ptr(norms), _ptr(q8), _ptr(scale), _ptr(idx),
                               L["N"], L["K"], L["S"], L["p"], _ptr(rows), len(rows),
                               _ptr(X_bits), B, _ptr(Y))
    if rc:
        raise OracleError(rc)
    return Y


def gemv(L, X_bits):
    """Full output Y[B][N] = X What^T (decode to dense, then the naive matmul)."""
    return matmul(decode_rows(L), X_bits)
