"""The batch-1 table-lookup decode's arithmetic (its reading of Eq. 12:
per chunk, the 16 signed sums of each half of the chunk's activations,
summed in fp32 and rounded once to fp16; each chunk-stage adds
n * T_lo + n * T_hi in fp32) emulated in numpy at full layer sizes and held
against the fp64 oracle.  The kernel's own parity is checked on the GPU;
this checks the error budget of the arithmetic it uses: its max-relative
error per activation row stays well inside the 2e-3 bar (about 1e-4 to
2e-4 for q_proj, growing slowly with K and S)."""
import numpy as np
import pytest

import oracle
from paper_2607_08643_gb300 import synth


def _table_decode_model(L, x_bits):
    N, K, S, p = L["N"], L["K"], L["S"], L["p"]
    C = K // 8
    xf = synth.bf16_bits_to_f32(x_bits)[0].astype(np.float32)
    xm = xf.copy()
    xm[L["idx"]] = 0.0                     # protected columns count as zero (Eq. 10)
    xc = xm.reshape(C, 8)
    v = np.arange(16)
    sg = (1.0 - 2.0 * ((v[:, None] >> np.arange(4)[None, :]) & 1)).astype(np.float32)
    lo = (xc[:, None, 0:4] * sg[None]).sum(axis=2, dtype=np.float32).astype(np.float16)
    hi = (xc[:, None, 4:8] * sg[None]).sum(axis=2, dtype=np.float32).astype(np.float16)
    acc = np.zeros(N, np.float32)
    cols = np.arange(C)[None, :]
    for s in range(S):
        cb = L["codes"][s].astype(np.int64)
        n = L["norms"][s].view(np.float16).astype(np.float32)
        tl = lo[cols, cb & 15].astype(np.float32)
        th = hi[cols, cb >> 4].astype(np.float32)
        acc += (n * tl + n * th).sum(axis=1, dtype=np.float32)
    y = acc * np.float32(1.0 / np.sqrt(8.0))
    sc = L["scale"].view(np.float16).astype(np.float32)
    y += (L["q8"][:, :p].astype(np.float32) * (sc * xf[L["idx"]])[None, :]).sum(axis=1)
    return y


@pytest.mark.parametrize("name,S,rho,dist", [("q_proj", 2, 1, "normal"), ("down_proj", 3, 2, "t4")])
def test_table_decode_arithmetic_error_budget(name, S, rho, dist):
    N, K = synth.QWEN3_8B_SHAPES[name]
    p = synth.protected_count(K, rho)
    L = oracle.encode(synth.layer_weights(N, K, seed=3, dist=dist), S=S, p=p)
    for seed in (10, 11):
        x = synth.activations(1, K, seed=seed)
        ref = oracle.gemv(L, x)[0]
        err = np.abs(_table_decode_model(L, x) - ref).max() / np.abs(ref).max()
        assert err <= 5e-4, (name, seed, err)
