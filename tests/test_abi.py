"""C-ABI checks that need no GPU: the library loads, exports every function
include/bisco.h declares, and rejects bad arguments before touching the
device."""
import ctypes
import os
import re

import pytest

import oracle
from paper_2607_08643_gb300 import bisco, synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "bisco.h")


@pytest.fixture(scope="module")
def lib():
    from paper_2607_08643_gb300 import build
    build.build()
    return bisco.load()


def declared_functions():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(bisco_[a-z_0-9]+)\s*\(", src)))


def test_header_declarations_are_exported(lib):
    names = declared_functions()
    assert set(names) == set(bisco.EXPORTS)
    for n in names:
        assert getattr(lib, n) is not None


def test_abi_version_and_status_strings(lib):
    assert bisco.bisco_abi_version() == 107
    for code in range(6):
        assert bisco.status_string(code)
    assert bisco.status_string(99) == "unknown status"


def test_encoded_sizes_match_oracle_accounting(lib):
    for (N, K, S, rho) in [(1024, 1024, 2, 1), (4096, 4096, 2, 1), (12288, 4096, 3, 2),
                           (4096, 12288, 3, 2), (37, 136, 1, 0)]:
        p = synth.protected_count(K, rho)
        assert bisco.bisco_encoded_sizes(N, K, S, p) == oracle.encoded_sizes(N, K, S, p)


@pytest.mark.parametrize("args,code", [
    ((0, 64, 8, 1, 0), bisco.ERR_INVALID_ARG),
    ((4, 60, 8, 1, 0), bisco.ERR_INVALID_ARG),
    ((4, 64, 8, 4, 0), bisco.ERR_INVALID_ARG),
    ((4, 64, 8, 1, 65), bisco.ERR_INVALID_ARG),
    ((4, 64, 16, 1, 0), bisco.ERR_UNSUPPORTED),
])
def test_encoded_sizes_rejects(lib, args, code):
    out = (ctypes.c_size_t * 5)()
    assert lib.bisco_encoded_sizes(*args, out) == code


def _fake_layer(**kw):
    base = dict(n_out=64, k_in=256, chunk_dim=8, stages=2, n_protected=3, protect_axis=0,
                codes=0x10000, norms=0x20000, q8=0x30000, q8_scale=0x40000, prot_idx=0x50000)
    base.update(kw)
    return bisco.bisco_layer(**base)


@pytest.mark.parametrize("kw,code", [
    (dict(k_in=252), bisco.ERR_INVALID_ARG),
    (dict(stages=0), bisco.ERR_INVALID_ARG),
    (dict(n_protected=-1), bisco.ERR_INVALID_ARG),
    (dict(chunk_dim=16), bisco.ERR_UNSUPPORTED),
    (dict(protect_axis=1, n_protected=65), bisco.ERR_INVALID_ARG),   # p > N for rows
    (dict(n_protected=257), bisco.ERR_INVALID_ARG),                 # p > K for columns
    (dict(protect_axis=2), bisco.ERR_INVALID_ARG),
    (dict(codes=0x10004), bisco.ERR_INVALID_ARG),
    (dict(codes=0), bisco.ERR_INVALID_ARG),
    (dict(q8=0), bisco.ERR_INVALID_ARG),
])
def test_layer_validation_before_any_device_call(lib, kw, code):
    L = _fake_layer(**kw)
    x = ctypes.c_void_p(0x60000)
    y = ctypes.c_void_p(0x70000)
    assert lib.bisco_gemv(ctypes.byref(L), x, 1, y, None) == code
    assert lib.bisco_gemm(ctypes.byref(L), x, 4, y, None, 0, None) == code
    assert lib.bisco_encode(x, None, ctypes.byref(L), ctypes.c_void_p(0x80000), 1 << 20, None) == code


def test_call_argument_validation(lib):
    L = _fake_layer()
    x, y = ctypes.c_void_p(0x60000), ctypes.c_void_p(0x70000)
    assert lib.bisco_gemv(ctypes.byref(L), x, 17, y, None) == bisco.ERR_INVALID_ARG
    assert lib.bisco_gemv(ctypes.byref(L), x, -1, y, None) == bisco.ERR_INVALID_ARG
    assert lib.bisco_gemv(ctypes.byref(L), ctypes.c_void_p(0x60002), 1, y, None) == bisco.ERR_INVALID_ARG
    assert lib.bisco_gemv(ctypes.byref(L), None, 1, y, None) == bisco.ERR_INVALID_ARG
    assert lib.bisco_gemv(None, x, 1, y, None) == bisco.ERR_INVALID_ARG
    assert lib.bisco_gemv(ctypes.byref(L), x, 0, y, None) == bisco.OK          # empty batch
    assert lib.bisco_gemm(ctypes.byref(L), x, -3, y, None, 0, None) == bisco.ERR_INVALID_ARG
    assert lib.bisco_gemm(ctypes.byref(L), x, 0, y, None, 0, None) == bisco.OK  # empty prefill
    # encode: workspace too small / misaligned weights / misaligned g
    ws = bisco.bisco_encode_workspace_bytes(64, 256)
    assert ws >= 64 * 256 // 8 and ws % 256 == 0
    assert lib.bisco_encode(x, None, ctypes.byref(L), ctypes.c_void_p(0x80000), ws - 1, None) \
        == bisco.ERR_INVALID_ARG
    assert lib.bisco_encode(ctypes.c_void_p(0x60008), None, ctypes.byref(L),
                            ctypes.c_void_p(0x80000), ws, None) == bisco.ERR_INVALID_ARG
    assert lib.bisco_encode(x, ctypes.c_void_p(0x90002), ctypes.byref(L),
                            ctypes.c_void_p(0x80000), ws, None) == bisco.ERR_INVALID_ARG
    assert lib.bisco_encode_workspace_bytes(0, 64) == 0
    assert lib.bisco_gemm_workspace_bytes(ctypes.byref(_fake_layer(k_in=12)), 128) == 0
    assert lib.bisco_gemm_workspace_bytes(ctypes.byref(L), -1) == 0
    assert lib.bisco_gemm_workspace_bytes(ctypes.byref(L), 16) == 0        # decode-kernel path
    assert lib.bisco_gemm_workspace_bytes(ctypes.byref(L), 17) == \
        17 * (256 + 128) * 2 + 160 * 2 * 128 * 128 * 4                    # tensor cores from 17
    # tensor-core path: fp16 activations plus hi/lo protected columns (rounded
    # up to 256 bytes), then the partial tiles of the stream-K split (160 CTAs
    # x 2 slots x TN tokens x 128 features, fp32)
    L2 = _fake_layer(k_in=4096, n_protected=41)
    assert lib.bisco_gemm_workspace_bytes(ctypes.byref(L2), 2048) == \
        2048 * (4096 + 128) * 2 + 160 * 2 * 256 * 128 * 4
    assert lib.bisco_gemm_workspace_bytes(ctypes.byref(L2), 100) == \
        100 * (4096 + 128) * 2 + 160 * 2 * 128 * 128 * 4
    assert lib.bisco_gemm_workspace_bytes(ctypes.byref(_fake_layer(k_in=128, n_protected=1)), 65) == \
        (65 * 256 * 2 + 255) // 256 * 256 + 160 * 2 * 128 * 128 * 4
    assert lib.bisco_gemm(ctypes.byref(L2), x, 2048, y, None, 0, None) == bisco.ERR_INVALID_ARG


def test_decode_dense_validation(lib):
    L = _fake_layer()
    out = ctypes.c_void_p(0x70000)
    assert lib.bisco_decode_dense(ctypes.byref(L), out, 3, None) == bisco.ERR_INVALID_ARG     # dtype
    assert lib.bisco_decode_dense(ctypes.byref(L), out, -1, None) == bisco.ERR_INVALID_ARG
    assert lib.bisco_decode_dense(ctypes.byref(L), None, bisco.DENSE_F32, None) == bisco.ERR_INVALID_ARG
    assert lib.bisco_decode_dense(ctypes.byref(L), ctypes.c_void_p(0x70004), bisco.DENSE_BF16,
                                  None) == bisco.ERR_INVALID_ARG                               # alignment
    assert lib.bisco_decode_dense(None, out, bisco.DENSE_F16, None) == bisco.ERR_INVALID_ARG
    assert lib.bisco_decode_dense(ctypes.byref(_fake_layer(codes=0x10004)), out, bisco.DENSE_F32,
                                  None) == bisco.ERR_INVALID_ARG


def test_gemv_multi_validation(lib):
    L = _fake_layer()
    x = ctypes.c_void_p(0x60000)
    ys = (ctypes.c_void_p * 4)(0x70000, 0x71000, 0x72000, 0x73000)
    arr = (bisco.bisco_layer * 4)(L, L, L, L)
    assert lib.bisco_gemv_multi(arr, 0, x, 1, ys, None) == bisco.ERR_INVALID_ARG
    assert lib.bisco_gemv_multi(arr, 5, x, 1, ys, None) == bisco.ERR_INVALID_ARG
    assert lib.bisco_gemv_multi(None, 1, x, 1, ys, None) == bisco.ERR_INVALID_ARG
    assert lib.bisco_gemv_multi(arr, 2, x, 1, None, None) == bisco.ERR_INVALID_ARG
    mixed = (bisco.bisco_layer * 2)(L, _fake_layer(k_in=512))          # K differs
    assert lib.bisco_gemv_multi(mixed, 2, x, 1, ys, None) == bisco.ERR_INVALID_ARG
    mixed = (bisco.bisco_layer * 2)(L, _fake_layer(stages=3))          # S differs
    assert lib.bisco_gemv_multi(mixed, 2, x, 1, ys, None) == bisco.ERR_INVALID_ARG
    bad = (bisco.bisco_layer * 2)(L, _fake_layer(codes=0x10004))       # layer invalid
    assert lib.bisco_gemv_multi(bad, 2, x, 1, ys, None) == bisco.ERR_INVALID_ARG
    assert lib.bisco_gemv_multi(arr, 2, x, 17, ys, None) == bisco.ERR_INVALID_ARG
    assert lib.bisco_gemv_multi(arr, 2, ctypes.c_void_p(0x60002), 1, ys, None) \
        == bisco.ERR_INVALID_ARG
    odd = (ctypes.c_void_p * 2)(0x70000, 0x70004)                       # y[1] misaligned
    assert lib.bisco_gemv_multi(arr, 2, x, 1, odd, None) == bisco.ERR_INVALID_ARG
    assert lib.bisco_gemv_multi(arr, 2, x, 0, ys, None) == bisco.OK   # empty batch


def test_lora_validation(lib):
    A, Bm, x, y, t = (ctypes.c_void_p(a) for a in (0x10000, 0x20000, 0x30000, 0x40000, 0x50000))
    f = lib.bisco_lora_apply
    E = bisco.ERR_INVALID_ARG
    for rank in (0, 4, 12, 264, -8):                                   # rank: 8..256, % 8
        assert f(A, Bm, rank, 64, 64, 1.0, x, 1, y, t, None) == E
    for N, K in ((0, 64), (64, 0), (64, 4), (64, 12)):                 # N >= 1, K >= 8, K % 8
        assert f(A, Bm, 16, N, K, 1.0, x, 1, y, t, None) == E
    for batch in (0, -1, 65536):
        assert f(A, Bm, 16, 64, 64, 1.0, x, batch, y, t, None) == E
    for scale in (float("nan"), float("inf"), -float("inf")):
        assert f(A, Bm, 16, 64, 64, scale, x, 1, y, t, None) == E
    ptrs = [A, Bm, x, y, t]
    for i in range(5):                                                  # NULL, misaligned
        for bad in (None, ctypes.c_void_p(0x60008)):
            p = list(ptrs)
            p[i] = bad
            assert f(p[0], p[1], 16, 64, 64, 1.0, p[2], 1, p[3], p[4], None) == E


def test_gemv_lora_validation(lib):
    """The fused compensation entry points check every argument before any
    device call; shapes the batch-1 kernel does not take are UNSUPPORTED."""
    L = _fake_layer()                                                   # k_in 256
    L4 = _fake_layer(k_in=4096)
    x = ctypes.c_void_p(0x60000)
    ys = (ctypes.c_void_p * 2)(0x70000, 0x80000)
    ok = bisco.bisco_lora(0x90000, 0xA0000, 16, 1.0)
    E = bisco.ERR_INVALID_ARG
    f = lib.bisco_gemv_multi_lora
    arr = (bisco.bisco_layer * 2)(L, L)
    lor = (bisco.bisco_lora * 2)(ok, ok)
    assert f(arr, lor, 2, x, ys, None) == bisco.ERR_UNSUPPORTED       # K != 4096
    for bad in (bisco.bisco_lora(0x90000, 0xA0000, r, 1.0) for r in (4, 12, 72, -8)):
        assert f(arr, (bisco.bisco_lora * 2)(ok, bad), 2, x, ys, None) == E
    for bad in (bisco.bisco_lora(0x90008, 0xA0000, 16, 1.0), bisco.bisco_lora(0x90000, None, 16, 1.0),
                bisco.bisco_lora(0x90000, 0xA0000, 16, float("nan"))):
        assert f(arr, (bisco.bisco_lora * 2)(bad, ok), 2, x, ys, None) == E
    # rank 0: no compensation, A and Bm not looked at
    none = bisco.bisco_lora(None, None, 0, float("nan"))
    assert f(arr, (bisco.bisco_lora * 2)(none, none), 2, x, ys, None) == bisco.ERR_UNSUPPORTED
    assert f(arr, None, 2, x, ys, None) == E
    assert f(arr, lor, 0, x, ys, None) == E
    assert f(arr, lor, 5, x, ys, None) == E
    assert f(arr, lor, 2, ctypes.c_void_p(0x60002), ys, None) == E      # x misaligned
    mixed = (bisco.bisco_layer * 2)(L4, L)                              # K differs
    assert f(mixed, lor, 2, x, ys, None) == E
    g = lib.bisco_gemv_lora
    assert g(ctypes.byref(L), ctypes.byref(ok), x, ctypes.c_void_p(0x70000), None) == bisco.ERR_UNSUPPORTED
    assert g(ctypes.byref(L), None, x, ctypes.c_void_p(0x70000), None) == E
    assert g(ctypes.byref(L), ctypes.byref(ok), x, ctypes.c_void_p(0x70004), None) == E


def test_binding_argument_counts_match_header(lib):
    """Every prototype in bisco.h has as many parameters as the ctypes
    binding declares for it (a drifted binding would pass garbage)."""
    src = re.sub(r"/\*.*?\*/", "", open(HEADER).read(), flags=re.S)
    protos = re.findall(r"\b(bisco_[a-z_0-9]+)\s*\(([^;{]*?)\)\s*;", src, flags=re.S)
    assert protos
    seen = set()
    for name, params in protos:
        params = params.strip()
        n = 0 if params in ("", "void") else params.count(",") + 1
        assert len(getattr(lib, name).argtypes) == n, name
        seen.add(name)
    assert seen == set(bisco.EXPORTS)


def test_layer_sizes_match_oracle_layouts(lib):
    """bisco_layer_sizes: the buffers the oracle's encoders fill, byte for
    byte, for protected rows and for every protected payload format."""
    for (N, K, S, p) in [(64, 136, 2, 3), (12288, 4096, 2, 123), (40, 64, 1, 0), (16, 64, 3, 16)]:
        sizes = bisco.bisco_layer_sizes(N, K, S, p, axis=1)
        kp = oracle.pad16(K)
        assert sizes == [S * N * (K // 8), 2 * S * N * (K // 8), p * kp, 2 * p, 4 * p]
        if N * K <= 1 << 14:
            L = oracle.encode_rows(synth.layer_weights(N, K, seed=7), S, p)
            assert sizes[:2] == [L["codes"].nbytes, L["norms"].nbytes]
            assert sizes[2:] == [L["q8"].nbytes, L["scale"].nbytes, L["idx"].nbytes]
    W = synth.layer_weights(48, 256, seed=8)
    for fmt in (bisco.PROT_INT8, bisco.PROT_E4M3, bisco.PROT_E5M2, bisco.PROT_BF16):
        sizes = bisco.bisco_layer_sizes(48, 256, 2, 5, axis=0, fmt=fmt)
        assert sizes[:2] == bisco.bisco_encoded_sizes(48, 256, 2, 5)[:2]
        idx = oracle.select_protected(W, 5)[0]
        q, scale = oracle.quantize_protected_fmt(W, idx, fmt)
        padded = q.itemsize * 48 * oracle.pad16(5)          # the oracle returns q[:, :p_pad]
        assert sizes[2:] == [padded, scale.nbytes, 4 * 5]
    assert bisco.bisco_layer_sizes(64, 64, 2, 5) == bisco.bisco_encoded_sizes(64, 64, 2, 5)
    f = lib.bisco_layer_sizes
    out = (ctypes.c_size_t * 5)()

    def c(**kw):
        base = dict(n_out=64, k_in=64, chunk_dim=8, stages=2, n_protected=4, protect_axis=0,
                    protect_format=0)
        base.update(kw)
        return ctypes.byref(bisco.bisco_layer(**base))

    assert f(c(), out) == bisco.OK
    assert f(c(protect_axis=1, n_protected=65), out) == bisco.ERR_INVALID_ARG   # p > N
    assert f(c(protect_axis=1, k_in=128, n_protected=65), out) == bisco.ERR_INVALID_ARG
    assert f(c(protect_axis=1, n_out=128, n_protected=65), out) == bisco.OK      # rows may exceed K
    assert f(c(protect_axis=2), out) == bisco.ERR_INVALID_ARG
    assert f(c(chunk_dim=16), out) == bisco.ERR_UNSUPPORTED
    assert f(c(protect_format=4), out) == bisco.ERR_INVALID_ARG
    assert f(c(protect_format=-1), out) == bisco.ERR_INVALID_ARG
    assert f(c(protect_format=1, protect_axis=1), out) == bisco.OK               # FP8 rows
    f(c(protect_format=3, protect_axis=1, n_protected=5), out)                   # BF16 rows
    assert out[2] == 5 * 64 * 2
    assert f(c(), None) == bisco.ERR_INVALID_ARG
    assert f(None, out) == bisco.ERR_INVALID_ARG


def test_protect_format_validation_before_any_device_call(lib):
    x, y = ctypes.c_void_p(0x60000), ctypes.c_void_p(0x70000)
    tab = ctypes.c_void_p(0x90000)
    for fmt, code in ((5, bisco.ERR_INVALID_ARG), (-2, bisco.ERR_INVALID_ARG)):
        L = _fake_layer(protect_format=fmt)
        assert lib.bisco_gemv(ctypes.byref(L), x, 1, y, None) == code
        assert lib.bisco_gemm(ctypes.byref(L), x, 4, y, None, 0, None) == code
        assert lib.bisco_decode_dense(ctypes.byref(L), y, bisco.DENSE_F32, None) == code
    for fmt in (bisco.PROT_E4M3, bisco.PROT_E5M2, bisco.PROT_BF16):       # tables: INT8 only
        L = _fake_layer(protect_format=fmt)
        assert lib.bisco_gemv_table(ctypes.byref(L), tab, x, 1, y, None) == bisco.ERR_UNSUPPORTED
        assert lib.bisco_decode_dense_table(ctypes.byref(L), tab, y, 0, None) == bisco.ERR_UNSUPPORTED
        assert lib.bisco_encode_noalloc(x, None, ctypes.byref(L), None) == bisco.ERR_UNSUPPORTED


def test_noalloc_validates_the_layer_as_bisco_encode_does(lib):
    """Sizes, axis and format outside the layer's range give the same
    INVALID_ARG as bisco_encode; the row axis alone is UNSUPPORTED."""
    w, ws = ctypes.c_void_p(0x30000), ctypes.c_void_p(0x40000)
    for bad in (dict(protect_format=5), dict(protect_format=-1), dict(protect_axis=2),
                dict(k_in=12), dict(stages=4), dict(n_protected=-1), dict(n_protected=257)):
        L = _fake_layer(**bad)
        assert lib.bisco_encode(w, None, ctypes.byref(L), ws, 1 << 20, None) == bisco.ERR_INVALID_ARG
        assert lib.bisco_encode_noalloc(w, None, ctypes.byref(L), None) == bisco.ERR_INVALID_ARG, bad
    L = _fake_layer(protect_axis=1, n_protected=3)
    assert lib.bisco_encode_noalloc(w, None, ctypes.byref(L), None) == bisco.ERR_UNSUPPORTED
    assert lib.bisco_encode_noalloc(None, None, ctypes.byref(_fake_layer()), None) \
        == bisco.ERR_INVALID_ARG


def test_encode_workspace_by_axis(lib):
    assert bisco.bisco_encode_workspace_bytes_axis(300, 64, 0) == bisco.bisco_encode_workspace_bytes(300, 64)
    ws = bisco.bisco_encode_workspace_bytes_axis(300, 64, 1)
    assert ws % 256 == 0 and ws >= 13 * 300
    assert bisco.bisco_encode_workspace_bytes_axis(300, 64, 2) == 0
    assert bisco.bisco_encode_workspace_bytes_axis(300, 60, 1) == 0
    assert bisco.bisco_select_coupled_workspace_bytes(0) == 0
    assert bisco.bisco_select_coupled_workspace_bytes(1000) >= 13 * 1000
    # a row-protected encode wants the row workspace
    L = _fake_layer(n_out=300, k_in=64, n_protected=3, protect_axis=1)
    x = ctypes.c_void_p(0x60000)
    small = bisco.bisco_encode_workspace_bytes_axis(300, 64, 0)
    assert small < ws
    assert lib.bisco_encode(x, None, ctypes.byref(L), ctypes.c_void_p(0x80000), small, None) \
        == bisco.ERR_INVALID_ARG


def test_encode_with_set_validation(lib):
    f = lib.bisco_encode_with_set
    E = bisco.ERR_INVALID_ARG
    x, idx, ws = ctypes.c_void_p(0x60000), ctypes.c_void_p(0x50000), ctypes.c_void_p(0x80000)
    big = 1 << 20
    for axis in (0, 1):
        L = _fake_layer(protect_axis=axis)
        assert f(None, idx, ctypes.byref(L), ws, big, None) == E                 # weights
        assert f(ctypes.c_void_p(0x60008), idx, ctypes.byref(L), ws, big, None) == E
        assert f(x, None, ctypes.byref(L), ws, big, None) == E                   # p > 0, no set
        assert f(x, ctypes.c_void_p(0x50002), ctypes.byref(L), ws, big, None) == E
        assert f(x, idx, ctypes.byref(L), None, big, None) == E                  # workspace
        assert f(x, idx, ctypes.byref(L), ws, 16, None) == E
        assert f(x, idx, None, ws, big, None) == E
    assert f(x, idx, ctypes.byref(_fake_layer(protect_axis=1, n_protected=65)), ws, big, None) == E
    assert f(x, idx, ctypes.byref(_fake_layer(chunk_dim=16)), ws, big, None) == bisco.ERR_UNSUPPORTED


def test_select_coupled_validation(lib):
    f = lib.bisco_select_coupled
    E = bisco.ERR_INVALID_ARG
    g, u, d = ctypes.c_void_p(0x10000), ctypes.c_void_p(0x20000), ctypes.c_void_p(0x30000)
    idx, ws = ctypes.c_void_p(0x40000), ctypes.c_void_p(0x80000)
    big = 1 << 20
    ok = [g, u, d, None, None, None, 96, 64, 4, idx, ws, big, None]

    def call(**kw):
        a = list(ok)
        names = ["g", "u", "d", "gg", "gu", "gd", "F", "H", "p", "idx", "ws", "bytes", "s"]
        for k, v in kw.items():
            a[names.index(k)] = v
        return f(*a)

    for bad in (dict(F=0), dict(H=0), dict(p=-1), dict(p=97), dict(g=None), dict(d=None),
                dict(u=ctypes.c_void_p(0x20008)), dict(gg=ctypes.c_void_p(0x90002)),
                dict(gd=ctypes.c_void_p(0x90001)), dict(idx=None), dict(idx=ctypes.c_void_p(0x40002)),
                dict(ws=None), dict(ws=ctypes.c_void_p(0x80008)), dict(bytes=64)):
        assert call(**bad) == E, bad


def test_decoder_table_validation(lib):
    E = bisco.ERR_INVALID_ARG
    L = _fake_layer()
    tab, x, y = ctypes.c_void_p(0x90000), ctypes.c_void_p(0x60000), ctypes.c_void_p(0x70000)
    g, d = lib.bisco_gemv_table, lib.bisco_decode_dense_table
    for bad_tab in (None, ctypes.c_void_p(0x90008)):
        assert g(ctypes.byref(L), bad_tab, x, 1, y, None) == E
        assert d(ctypes.byref(L), bad_tab, y, bisco.DENSE_F32, None) == E
    assert g(ctypes.byref(L), tab, x, 17, y, None) == E
    assert g(ctypes.byref(L), tab, x, -1, y, None) == E
    assert g(ctypes.byref(L), tab, ctypes.c_void_p(0x60002), 1, y, None) == E
    assert g(ctypes.byref(L), tab, x, 1, None, None) == E
    assert g(ctypes.byref(L), tab, x, 0, y, None) == bisco.OK                  # empty batch
    assert g(None, tab, x, 1, y, None) == E
    assert g(ctypes.byref(_fake_layer(chunk_dim=16)), tab, x, 1, y, None) == bisco.ERR_UNSUPPORTED
    assert d(ctypes.byref(L), tab, y, 3, None) == E
    assert d(ctypes.byref(L), tab, None, bisco.DENSE_BF16, None) == E
    assert d(ctypes.byref(L), tab, ctypes.c_void_p(0x70004), bisco.DENSE_F16, None) == E
    assert d(ctypes.byref(_fake_layer(stages=4)), tab, y, bisco.DENSE_F32, None) == E


@pytest.mark.parametrize("name", ["bisco_layer", "bisco_lora"])
def test_struct_layout_matches_the_header(tmp_path, name):
    """The ctypes mirrors of bisco_layer and bisco_lora have the C structs'
    sizes and field offsets (arrays of them cross the ABI in
    bisco_gemv_multi and bisco_gemv_multi_lora)."""
    import subprocess
    cls = getattr(bisco, name)
    fields = [f for f, _ in cls._fields_]
    src = tmp_path / "layout.c"
    src.write_text('#include <stdio.h>\n#include <stddef.h>\n#include "bisco.h"\nint main(void) {\n'
                   '  printf("%%zu\\n", sizeof(%s));\n' % name +
                   "".join('  printf("%%zu\\n", offsetof(%s, %s));\n' % (name, f) for f in fields) +
                   "  return 0;\n}\n")
    exe = tmp_path / "layout"
    subprocess.check_call(["gcc", "-std=c11", "-I", os.path.join(ROOT, "include"), "-o", str(exe), str(src)])
    out = [int(v) for v in subprocess.check_output([str(exe)]).split()]
    assert out[0] == ctypes.sizeof(cls)
    assert out[1:] == [getattr(cls, f).offset for f in fields]


@pytest.mark.parametrize("axis,fmt", [(0, bisco.PROT_INT8), (0, bisco.PROT_E4M3), (0, bisco.PROT_E5M2),
                                      (0, bisco.PROT_BF16), (1, bisco.PROT_INT8), (1, bisco.PROT_E4M3),
                                      (1, bisco.PROT_BF16)])
def test_layer_marshalling_round_trip(lib, axis, fmt):
    """Layer.from_numpy / to_numpy carry the oracle's layer dicts exactly for
    every protection axis and payload format (host tensors; no device call),
    and the C struct describes the tensors it points at."""
    import numpy as np
    N, K, S, p = 40, 136, 2, 3
    W = synth.layer_weights(N, K, seed=5)
    if axis == 1:
        ref = oracle.encode_rows(W, S, p)
        if fmt != bisco.PROT_INT8:
            q, scale = oracle.quantize_protected_rows_fmt(W, ref["idx"], fmt)
            ref = dict(ref, q8=q, scale=scale, fmt=fmt)
    else:
        ref = oracle.encode(W, S=S, p=p)
        if fmt != bisco.PROT_INT8:
            q, scale = oracle.quantize_protected_fmt(W, ref["idx"], fmt)
            ref = dict(ref, q8=q, scale=scale, fmt=fmt)
    L = bisco.Layer.from_numpy(ref, device="cpu")
    got = L.to_numpy()
    for k in ("codes", "norms", "q8", "scale", "idx"):
        assert got[k].dtype == ref[k].dtype and np.array_equal(got[k], ref[k]), k
    assert got.get("axis", 0) == axis and got.get("fmt", 0) == ref.get("fmt", 0)
    c = L.c
    assert (c.n_out, c.k_in, c.stages, c.n_protected, c.protect_axis, c.protect_format) == \
        (N, K, S, p, axis, fmt)
    assert c.codes == L.codes.data_ptr() and c.q8 == L.q8.data_ptr() and c.prot_idx == L.idx.data_ptr()
    sizes = bisco.bisco_layer_sizes(N, K, S, p, axis, fmt)
    assert sizes[2] <= L.q8.numel() * L.q8.element_size()
    extra = 2 if fmt == bisco.PROT_BF16 else 1
    assert L.compressed_bytes == S * N * (K // 8) * 3 + p * (K if axis else N) * extra + 6 * p
