"""Thin ctypes binding of libbisco.so (include/bisco.h), same entry-point
names.  It only marshals arguments: PyTorch supplies device memory and the
stream; every step of the computation runs in the library's CUDA kernels.
There is no fallback -- if the library is missing this module raises.
"""
from __future__ import annotations

import ctypes
import os

HERE = os.path.dirname(os.path.abspath(__file__))
# BISCO_LIB selects another build of the same library (for A/B timing).
LIB_PATH = os.environ.get("BISCO_LIB") or os.path.join(HERE, "libbisco.so")

OK, ERR_INVALID_ARG, ERR_UNSUPPORTED, ERR_RANGE, ERR_CUDA, ERR_TIMEOUT = range(6)

# Functions declared in include/bisco.h (kept in sync by tests/test_abi.py).
EXPORTS = (
    "bisco_abi_version", "bisco_status_string", "bisco_encoded_sizes",
    "bisco_layer_sizes", "bisco_encode_workspace_bytes",
    "bisco_encode_workspace_bytes_axis", "bisco_encode", "bisco_encode_with_set",
    "bisco_select_coupled_workspace_bytes", "bisco_select_coupled",
    "bisco_encode_noalloc", "bisco_gemv", "bisco_gemv_multi", "bisco_gemv_multi_lora",
    "bisco_gemv_lora",
    "bisco_gemm_workspace_bytes", "bisco_gemm", "bisco_decode_dense", "bisco_decode_dense_stage",
    "bisco_gemv_table",
    "bisco_decode_dense_table", "bisco_lora_apply",
    "bisco_get_device_error",
)

DENSE_F32, DENSE_BF16, DENSE_F16 = 0, 1, 2
PROT_INT8, PROT_E4M3, PROT_E5M2, PROT_BF16 = 0, 1, 2, 3


class BiscoError(RuntimeError):
    def __init__(self, code: int, where: str = ""):
        self.code = code
        super().__init__("%s: bisco status %d (%s)" % (where, code, status_string(code)))


class bisco_lora(ctypes.Structure):
    """struct bisco_lora of include/bisco.h."""
    _fields_ = [("A", ctypes.c_void_p), ("Bm", ctypes.c_void_p), ("rank", ctypes.c_int32),
                ("scale", ctypes.c_float)]


class bisco_layer(ctypes.Structure):
    _fields_ = [
        ("n_out", ctypes.c_int32), ("k_in", ctypes.c_int32), ("chunk_dim", ctypes.c_int32),
        ("stages", ctypes.c_int32), ("n_protected", ctypes.c_int32),
        ("protect_axis", ctypes.c_int32),
        ("codes", ctypes.c_void_p), ("norms", ctypes.c_void_p), ("q8", ctypes.c_void_p),
        ("q8_scale", ctypes.c_void_p), ("prot_idx", ctypes.c_void_p),
        ("protect_format", ctypes.c_int32),
    ]


_lib = None


def load(path: str = LIB_PATH):
    """Loads the CUDA library; raises if it has not been built."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise RuntimeError("libbisco.so not built (run __graft_entry__.build())")
    lib = ctypes.CDLL(path)
    P, i32, sz = ctypes.c_void_p, ctypes.c_int32, ctypes.c_size_t
    st = ctypes.c_int
    Lp = ctypes.POINTER(bisco_layer)
    lib.bisco_abi_version.restype = i32
    lib.bisco_abi_version.argtypes = []
    lib.bisco_status_string.restype = ctypes.c_char_p
    lib.bisco_status_string.argtypes = [i32]
    lib.bisco_encoded_sizes.restype = st
    lib.bisco_encoded_sizes.argtypes = [i32, i32, i32, i32, i32, ctypes.POINTER(sz)]
    lib.bisco_layer_sizes.restype = st
    lib.bisco_layer_sizes.argtypes = [Lp, ctypes.POINTER(sz)]
    lib.bisco_encode_workspace_bytes.restype = sz
    lib.bisco_encode_workspace_bytes.argtypes = [i32, i32]
    lib.bisco_encode_workspace_bytes_axis.restype = sz
    lib.bisco_encode_workspace_bytes_axis.argtypes = [i32, i32, i32]
    lib.bisco_encode.restype = st
    lib.bisco_encode.argtypes = [P, P, Lp, P, sz, P]
    lib.bisco_encode_with_set.restype = st
    lib.bisco_encode_with_set.argtypes = [P, P, Lp, P, sz, P]
    lib.bisco_select_coupled_workspace_bytes.restype = sz
    lib.bisco_select_coupled_workspace_bytes.argtypes = [i32]
    lib.bisco_select_coupled.restype = st
    lib.bisco_select_coupled.argtypes = [P, P, P, P, P, P, i32, i32, i32, P, P, sz, P]
    lib.bisco_encode_noalloc.restype = st
    lib.bisco_encode_noalloc.argtypes = [P, P, Lp, P]
    lib.bisco_gemv.restype = st
    lib.bisco_gemv.argtypes = [Lp, P, i32, P, P]
    lib.bisco_gemv_multi.restype = st
    lib.bisco_gemv_multi.argtypes = [Lp, i32, P, i32, ctypes.POINTER(P), P]
    lib.bisco_gemv_multi_lora.restype = st
    lib.bisco_gemv_multi_lora.argtypes = [Lp, ctypes.POINTER(bisco_lora), i32, P, ctypes.POINTER(P), P]
    lib.bisco_gemv_lora.restype = st
    lib.bisco_gemv_lora.argtypes = [Lp, ctypes.POINTER(bisco_lora), P, P, P]
    lib.bisco_gemm_workspace_bytes.restype = sz
    lib.bisco_gemm_workspace_bytes.argtypes = [Lp, i32]
    lib.bisco_gemm.restype = st
    lib.bisco_gemm.argtypes = [Lp, P, i32, P, P, sz, P]
    lib.bisco_decode_dense.restype = st
    lib.bisco_decode_dense.argtypes = [Lp, P, i32, P]
    lib.bisco_decode_dense_stage.restype = st
    lib.bisco_decode_dense_stage.argtypes = [Lp, i32, P, i32, P]
    lib.bisco_gemv_table.restype = st
    lib.bisco_gemv_table.argtypes = [Lp, P, P, i32, P, P]
    lib.bisco_decode_dense_table.restype = st
    lib.bisco_decode_dense_table.argtypes = [Lp, P, P, i32, P]
    lib.bisco_lora_apply.restype = st
    lib.bisco_lora_apply.argtypes = [P, P, i32, i32, i32, ctypes.c_float, P, i32, P, P, P]
    lib.bisco_get_device_error.restype = st
    lib.bisco_get_device_error.argtypes = [P]
    _lib = lib
    return lib


def status_string(code: int) -> str:
    return load().bisco_status_string(int(code)).decode()


def _check(code: int, where: str):
    if code != OK:
        raise BiscoError(code, where)


def _stream(stream):
    import torch
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def bisco_abi_version() -> int:
    return int(load().bisco_abi_version())


def bisco_encoded_sizes(N, K, S, p, d=8):
    out = (ctypes.c_size_t * 5)()
    _check(load().bisco_encoded_sizes(N, K, d, S, p, out), "bisco_encoded_sizes")
    return [int(v) for v in out]


def bisco_layer_sizes(N, K, S, p, axis=0, fmt=PROT_INT8, d=8):
    """Byte sizes of the five buffers of a layer with these sizes, protection
    axis and protected payload format."""
    c = bisco_layer(N, K, d, S, p, axis, None, None, None, None, None, fmt)
    out = (ctypes.c_size_t * 5)()
    _check(load().bisco_layer_sizes(ctypes.byref(c), out), "bisco_layer_sizes")
    return [int(v) for v in out]


def bisco_encode_workspace_bytes(N, K) -> int:
    return int(load().bisco_encode_workspace_bytes(N, K))


def bisco_encode_workspace_bytes_axis(N, K, axis) -> int:
    return int(load().bisco_encode_workspace_bytes_axis(N, K, axis))


def bisco_select_coupled_workspace_bytes(F) -> int:
    return int(load().bisco_select_coupled_workspace_bytes(F))


def bisco_gemm_workspace_bytes(L, M) -> int:
    """Workspace bytes bisco_gemm needs for layer L (a Layer or its C struct)."""
    c = L.c if isinstance(L, Layer) else L
    return int(load().bisco_gemm_workspace_bytes(ctypes.byref(c), M))


class Layer:
    """A coded layer in device memory (torch tensors) plus its C struct.
    axis 0 protects input columns (q8 [N][p_pad]); axis 1 protects output
    rows (q8 [p][roundup(K, 16)]).  fmt is the protected payload's format
    (PROT_*; BF16 payloads are [N][p_pad] uint16)."""

    def __init__(self, N, K, S, p, device="cuda", d=8, axis=0, fmt=PROT_INT8):
        import torch
        sizes = bisco_encoded_sizes(N, K, S, p, d) if (axis, fmt) == (0, PROT_INT8) else \
            bisco_layer_sizes(N, K, S, p, axis, fmt, d)
        self.N, self.K, self.S, self.p, self.axis, self.fmt = N, K, S, p, axis, fmt
        self.p_pad = (p + 15) // 16 * 16
        self.kp = (K + 15) // 16 * 16
        dev = torch.device(device)
        self.codes = torch.empty((S, N, K // 8), dtype=torch.uint8, device=dev)
        self.norms = torch.empty((S, N, K // 8), dtype=torch.int16, device=dev)
        qdt = {PROT_INT8: torch.int8, PROT_E4M3: torch.uint8, PROT_E5M2: torch.uint8,
               PROT_BF16: torch.int16}[fmt]
        if axis == 1:
            self.q8 = torch.empty((max(p, 1), self.kp), dtype=qdt, device=dev)
        else:
            self.q8 = torch.empty((N, max(self.p_pad, 16)), dtype=qdt, device=dev)
        self.scale = torch.empty((max(p, 8),), dtype=torch.int16, device=dev)
        self.idx = torch.empty((max(p, 4),), dtype=torch.int32, device=dev)
        assert sizes[0] == self.codes.numel() and sizes[1] == 2 * self.norms.numel()
        assert sizes[2] <= self.q8.numel() * self.q8.element_size()
        self.c = bisco_layer(N, K, d, S, p, axis, self.codes.data_ptr(), self.norms.data_ptr(),
                             self.q8.data_ptr(), self.scale.data_ptr(), self.idx.data_ptr(), fmt)

    @property
    def compressed_bytes(self) -> int:
        """Algorithmic payload: signs + norms + unpadded q8 + scales + indices."""
        q8 = self.p * (self.K if self.axis == 1 else self.N) * (2 if self.fmt == PROT_BF16 else 1)
        return self.S * self.N * (self.K // 8) * 3 + q8 + 6 * self.p

    def to_numpy(self):
        """Host copy in the oracle's dict layout."""
        p = self.p
        L = dict(N=self.N, K=self.K, S=self.S, p=p,
                 codes=self.codes.cpu().numpy(),
                 norms=self.norms.cpu().numpy().view("uint16"),
                 scale=self.scale[:p].cpu().numpy().view("uint16"),
                 idx=self.idx[:p].cpu().numpy())
        if self.axis == 1:
            L["axis"] = 1
            L["q8"] = self.q8[:p].cpu().numpy()
        else:
            L["q8"] = self.q8[:, :self.p_pad].cpu().numpy()
        if self.fmt == PROT_BF16:
            L["q8"] = L["q8"].view("uint16")
        if self.fmt != PROT_INT8:
            L["fmt"] = self.fmt
        return L

    @classmethod
    def from_numpy(cls, L, device="cuda"):
        import numpy as np
        import torch
        axis = L.get("axis", 0)
        fmt = L.get("fmt", PROT_INT8)
        obj = cls(L["N"], L["K"], L["S"], L["p"], device, axis=axis, fmt=fmt)
        obj.codes.copy_(torch.from_numpy(np.ascontiguousarray(L["codes"])))
        obj.norms.copy_(torch.from_numpy(np.ascontiguousarray(L["norms"]).view(np.int16)))
        if L["p"]:
            q8 = np.ascontiguousarray(L["q8"])
            q8 = torch.from_numpy(q8.view(np.int16) if q8.dtype == np.uint16 else q8)
            if axis == 1:
                obj.q8[:L["p"]].copy_(q8)
            else:
                obj.q8[:, :obj.p_pad].copy_(q8)
            obj.scale[:L["p"]].copy_(torch.from_numpy(np.ascontiguousarray(L["scale"]).view(np.int16)))
            obj.idx[:L["p"]].copy_(torch.from_numpy(np.ascontiguousarray(L["idx"])))
        return obj


def _bits2d(W_bits):
    import torch
    if W_bits.dtype == torch.bfloat16:
        W_bits = W_bits.view(torch.int16)
    assert W_bits.is_cuda and W_bits.is_contiguous() and W_bits.dim() == 2
    return W_bits


def bisco_encode(W_bits, S, p, g=None, workspace=None, stream=None, axis=0,
                 fmt=PROT_INT8) -> Layer:
    """Encodes a device tensor of bf16 bits [N][K] (int16 or bfloat16);
    axis 1 protects the p output rows of largest norm instead of columns;
    fmt selects the protected payload's format."""
    import torch
    W_bits = _bits2d(W_bits)
    N, K = W_bits.shape
    L = Layer(N, K, S, p, W_bits.device, axis=axis, fmt=fmt)
    need = bisco_encode_workspace_bytes_axis(N, K, axis)
    if workspace is None:
        workspace = torch.empty(max(need, 16), dtype=torch.uint8, device=W_bits.device)
    if g is not None:
        assert g.dtype == torch.float32 and g.is_cuda and g.numel() == (N if axis == 1 else K)
    _check(load().bisco_encode(_ptr(W_bits), _ptr(g), ctypes.byref(L.c), _ptr(workspace),
                               workspace.numel(), _stream(stream)), "bisco_encode")
    return L


def bisco_encode_with_set(W_bits, S, idx, axis, workspace=None, stream=None,
                          fmt=PROT_INT8) -> Layer:
    """Encodes with the protected set given (device int32 [p], ascending):
    columns for axis 0, rows for axis 1; fmt is the payload's format."""
    import torch
    W_bits = _bits2d(W_bits)
    N, K = W_bits.shape
    p = int(idx.numel())
    assert idx.dtype == torch.int32 and idx.is_cuda and idx.is_contiguous()
    L = Layer(N, K, S, p, W_bits.device, axis=axis, fmt=fmt)
    need = bisco_encode_workspace_bytes_axis(N, K, axis)
    if workspace is None:
        workspace = torch.empty(max(need, 16), dtype=torch.uint8, device=W_bits.device)
    _check(load().bisco_encode_with_set(_ptr(W_bits), _ptr(idx) if p else None, ctypes.byref(L.c),
                                        _ptr(workspace), workspace.numel(), _stream(stream)),
           "bisco_encode_with_set")
    return L


def bisco_select_coupled(Wg_bits, Wu_bits, Wd_bits, p, gg=None, gu=None, gd=None,
                         workspace=None, stream=None):
    """The coupled protected set (Eq. 9) of a gated MLP: gate/up [F][H],
    down [H][F]; returns the p channels as a device int32 tensor."""
    import torch
    Wg_bits, Wu_bits, Wd_bits = _bits2d(Wg_bits), _bits2d(Wu_bits), _bits2d(Wd_bits)
    F, H = Wg_bits.shape
    assert tuple(Wu_bits.shape) == (F, H) and tuple(Wd_bits.shape) == (H, F)
    idx = torch.empty((max(p, 1),), dtype=torch.int32, device=Wg_bits.device)
    need = bisco_select_coupled_workspace_bytes(F)
    if workspace is None:
        workspace = torch.empty(max(need, 16), dtype=torch.uint8, device=Wg_bits.device)
    for g in (gg, gu, gd):
        assert g is None or (g.dtype == torch.float32 and g.is_cuda and g.numel() == F)
    _check(load().bisco_select_coupled(_ptr(Wg_bits), _ptr(Wu_bits), _ptr(Wd_bits), _ptr(gg),
                                       _ptr(gu), _ptr(gd), F, H, p, _ptr(idx), _ptr(workspace),
                                       workspace.numel(), _stream(stream)),
           "bisco_select_coupled")
    return idx[:p]


def bisco_encode_noalloc(W_bits, S, p, g=None, stream=None) -> Layer:
    """bisco_encode with the library's fixed scratch array instead of a
    workspace (for callers that cannot allocate device memory; K up to
    BISCO_ENCODE_NOALLOC_MAX_K = 32768).  The output Layer's tensors are
    still allocated here, by PyTorch."""
    import torch
    if W_bits.dtype == torch.bfloat16:
        W_bits = W_bits.view(torch.int16)
    assert W_bits.is_cuda and W_bits.is_contiguous() and W_bits.dim() == 2
    N, K = W_bits.shape
    L = Layer(N, K, S, p, W_bits.device)
    if g is not None:
        assert g.dtype == torch.float32 and g.is_cuda and g.numel() == K
    _check(load().bisco_encode_noalloc(_ptr(W_bits), _ptr(g), ctypes.byref(L.c), _stream(stream)),
           "bisco_encode_noalloc")
    return L


def bisco_gemv(L: Layer, x_bits, y=None, stream=None):
    """y[B][N] (float32) = x What^T for B <= 16 activation rows (bf16 bits)."""
    import torch
    if x_bits.dtype == torch.bfloat16:
        x_bits = x_bits.view(torch.int16)
    if x_bits.dim() == 1:
        x_bits = x_bits.unsqueeze(0)
    B = x_bits.shape[0]
    assert x_bits.is_contiguous() and x_bits.shape[1] == L.K
    if y is None:
        y = torch.empty((B, L.N), dtype=torch.float32, device=x_bits.device)
    _check(load().bisco_gemv(ctypes.byref(L.c), _ptr(x_bits), B, _ptr(y), _stream(stream)),
           "bisco_gemv")
    return y


def bisco_gemv_multi(layers, x_bits, ys=None, stream=None):
    """[y_g] = x What_g^T for layers sharing K and S, one launch (q/k/v)."""
    import torch
    if x_bits.dtype == torch.bfloat16:
        x_bits = x_bits.view(torch.int16)
    if x_bits.dim() == 1:
        x_bits = x_bits.unsqueeze(0)
    B = x_bits.shape[0]
    G = len(layers)
    assert x_bits.is_contiguous() and all(L.K == x_bits.shape[1] for L in layers)
    if ys is None:
        ys = [torch.empty((B, L.N), dtype=torch.float32, device=x_bits.device) for L in layers]
    structs = (bisco_layer * G)(*[L.c for L in layers])
    yp = (ctypes.c_void_p * G)(*[y.data_ptr() for y in ys])
    _check(load().bisco_gemv_multi(structs, G, _ptr(x_bits), B, yp, _stream(stream)),
           "bisco_gemv_multi")
    return ys


def _lora_struct(lora):
    """(A, Bm, scale) of bf16 device tensors, or None for no compensation."""
    if lora is None:
        return bisco_lora(None, None, 0, 0.0)
    A, Bm, scale = lora
    return bisco_lora(A.data_ptr(), Bm.data_ptr(), int(A.shape[0]), float(scale))


def bisco_gemv_multi_lora(layers, loras, x_bits, ys=None, stream=None):
    """[y_g] = x What_g^T + scale_g (x A_g^T) Bm_g^T at batch 1 in one launch;
    loras[g] = (A [rank][K] bf16, Bm [N][rank] bf16, scale) or None."""
    import torch
    if x_bits.dtype == torch.bfloat16:
        x_bits = x_bits.view(torch.int16)
    if x_bits.dim() == 1:
        x_bits = x_bits.unsqueeze(0)
    G = len(layers)
    assert x_bits.shape[0] == 1 and x_bits.is_contiguous() and len(loras) == G
    for r in loras:
        if r is not None:
            assert r[0].is_contiguous() and r[1].is_contiguous()
    if ys is None:
        ys = [torch.empty((1, L.N), dtype=torch.float32, device=x_bits.device) for L in layers]
    structs = (bisco_layer * G)(*[L.c for L in layers])
    lstructs = (bisco_lora * G)(*[_lora_struct(r) for r in loras])
    yp = (ctypes.c_void_p * G)(*[y.data_ptr() for y in ys])
    _check(load().bisco_gemv_multi_lora(structs, lstructs, G, _ptr(x_bits), yp, _stream(stream)),
           "bisco_gemv_multi_lora")
    return ys


def bisco_gemv_lora(L: Layer, lora, x_bits, y=None, stream=None):
    """y = x What^T + scale (x A^T) Bm^T at batch 1 (lora = (A, Bm, scale))."""
    import torch
    if x_bits.dtype == torch.bfloat16:
        x_bits = x_bits.view(torch.int16)
    if x_bits.dim() == 1:
        x_bits = x_bits.unsqueeze(0)
    assert x_bits.shape[0] == 1 and x_bits.is_contiguous()
    if y is None:
        y = torch.empty((1, L.N), dtype=torch.float32, device=x_bits.device)
    ls = _lora_struct(lora)
    _check(load().bisco_gemv_lora(ctypes.byref(L.c), ctypes.byref(ls), _ptr(x_bits), y.data_ptr(),
                                  _stream(stream)), "bisco_gemv_lora")
    return y


def bisco_gemm(L: Layer, X_bits, Y=None, workspace=None, stream=None):
    """Y[M][N] (float32) = X What^T for any M (prefill)."""
    import torch
    if X_bits.dtype == torch.bfloat16:
        X_bits = X_bits.view(torch.int16)
    M = X_bits.shape[0]
    assert X_bits.is_contiguous() and X_bits.shape[1] == L.K
    if Y is None:
        Y = torch.empty((M, L.N), dtype=torch.float32, device=X_bits.device)
    need = bisco_gemm_workspace_bytes(L, M)
    if need and workspace is None:
        workspace = torch.empty(need, dtype=torch.uint8, device=X_bits.device)
    nbytes = 0 if workspace is None else workspace.numel()
    _check(load().bisco_gemm(ctypes.byref(L.c), _ptr(X_bits), M, _ptr(Y), _ptr(workspace),
                             nbytes, _stream(stream)), "bisco_gemm")
    return Y


def bisco_decode_dense(L: Layer, dtype: str = "f32", out=None, stream=None):
    """The layer's decoded weight What [N][K] as a dense tensor ("f32", "bf16"
    or "f16"): the materialise-then-multiply path."""
    import torch
    code = {"f32": DENSE_F32, "bf16": DENSE_BF16, "f16": DENSE_F16}[dtype]
    tdt = {"f32": torch.float32, "bf16": torch.bfloat16, "f16": torch.float16}[dtype]
    if out is None:
        out = torch.empty((L.N, L.K), dtype=tdt, device=L.codes.device)
    assert out.is_contiguous() and out.dtype == tdt and tuple(out.shape) == (L.N, L.K)
    _check(load().bisco_decode_dense(ctypes.byref(L.c), _ptr(out), code, _stream(stream)),
           "bisco_decode_dense")
    return out


def bisco_decode_dense_stage(L: Layer, stage: int, out, accumulate: bool, stream=None):
    """Adds (or writes) one stage's term of What into the fp32 [N][K] tensor
    `out`; the last stage also writes the protected set."""
    import torch
    assert out.is_contiguous() and out.dtype == torch.float32 and tuple(out.shape) == (L.N, L.K)
    _check(load().bisco_decode_dense_stage(ctypes.byref(L.c), int(stage), _ptr(out), int(bool(accumulate)),
                                           _stream(stream)), "bisco_decode_dense_stage")
    return out


def bisco_decode_dense_sequential(L: Layer, out=None, stream=None):
    """What [N][K] fp32 decoded stage by stage (one pass per stage)."""
    import torch
    if out is None:
        out = torch.empty((L.N, L.K), dtype=torch.float32, device=L.codes.device)
    for s in range(L.c.stages):
        bisco_decode_dense_stage(L, s, out, s > 0, stream)
    return out


def _tables(L: Layer, tables):
    import torch
    if tables.dtype == torch.float16:
        tables = tables.view(torch.int16)
    assert tables.is_cuda and tables.is_contiguous() and tuple(tables.shape) == (L.S, 256, 8)
    return tables


def bisco_gemv_table(L: Layer, tables, x_bits, y=None, stream=None):
    """y[B][N] = x What^T with the learned decoder step given as per-stage
    tables [S][256][8] (float16 or their int16 bits) of the decoded unit code
    of every code byte."""
    import torch
    tables = _tables(L, tables)
    if x_bits.dtype == torch.bfloat16:
        x_bits = x_bits.view(torch.int16)
    if x_bits.dim() == 1:
        x_bits = x_bits.unsqueeze(0)
    B = x_bits.shape[0]
    assert x_bits.is_contiguous() and x_bits.shape[1] == L.K
    if y is None:
        y = torch.empty((B, L.N), dtype=torch.float32, device=x_bits.device)
    _check(load().bisco_gemv_table(ctypes.byref(L.c), _ptr(tables), _ptr(x_bits), B, _ptr(y),
                                   _stream(stream)), "bisco_gemv_table")
    return y


def bisco_decode_dense_table(L: Layer, tables, dtype: str = "f32", out=None, stream=None):
    """The layer decoded with per-stage decoder tables, as a dense [N][K]
    tensor ("f32", "bf16" or "f16")."""
    import torch
    tables = _tables(L, tables)
    code = {"f32": DENSE_F32, "bf16": DENSE_BF16, "f16": DENSE_F16}[dtype]
    tdt = {"f32": torch.float32, "bf16": torch.bfloat16, "f16": torch.float16}[dtype]
    if out is None:
        out = torch.empty((L.N, L.K), dtype=tdt, device=L.codes.device)
    assert out.is_contiguous() and out.dtype == tdt and tuple(out.shape) == (L.N, L.K)
    _check(load().bisco_decode_dense_table(ctypes.byref(L.c), _ptr(tables), _ptr(out), code,
                                           _stream(stream)), "bisco_decode_dense_table")
    return out


def bisco_lora_apply(A, Bm, x_bits, y, scale: float = 1.0, t=None, stream=None):
    """y[B][N] += scale * (x A^T) Bm^T in place: the low-rank compensation of a
    layer's output.  A [rank][K] and Bm [N][rank] bf16, x [B][K] bf16 bits,
    y [B][N] float32; t [B][rank] float32 scratch (allocated if None)."""
    import torch
    if x_bits.dtype == torch.bfloat16:
        x_bits = x_bits.view(torch.int16)
    if x_bits.dim() == 1:
        x_bits = x_bits.unsqueeze(0)
    A = A.view(torch.int16) if A.dtype == torch.bfloat16 else A
    Bm = Bm.view(torch.int16) if Bm.dtype == torch.bfloat16 else Bm
    rank, K = A.shape
    N = Bm.shape[0]
    batch = x_bits.shape[0]
    assert Bm.shape[1] == rank and x_bits.shape[1] == K and tuple(y.shape) == (batch, N)
    assert A.is_contiguous() and Bm.is_contiguous() and x_bits.is_contiguous() and y.is_contiguous()
    assert y.dtype == torch.float32
    if t is None:
        t = torch.empty((batch, rank), dtype=torch.float32, device=y.device)
    _check(load().bisco_lora_apply(_ptr(A), _ptr(Bm), rank, N, K, float(scale), _ptr(x_bits),
                                   batch, _ptr(y), _ptr(t), _stream(stream)),
           "bisco_lora_apply")
    return y


def bisco_get_device_error(stream=None) -> int:
    return int(load().bisco_get_device_error(_stream(stream)))
