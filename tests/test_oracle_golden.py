"""Regression anchor for the fp64 oracle (no GPU): it still computes the
stored small worked example (tests/golden/make_oracle_golden.py wrote it from
the oracle alone) bit for bit.  This file is kept apart from
test_oracle_pins.py, whose independent pins the planted-mistake suite runs
alone: the anchor would catch any change and hide whether the pins do."""
import json
import os

import numpy as np

import oracle

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def test_oracle_reproduces_its_stored_worked_example():
    """Regression anchor: the oracle still computes the stored small example
    bit for bit (tests/golden/make_oracle_golden.py wrote it)."""
    with open(os.path.join(GOLDEN, "oracle_small_layer.json")) as f:
        g = json.load(f)
    N, K, S, p = g["N"], g["K"], g["S"], g["p"]
    W = np.array([int(h, 16) for h in g["W_bf16_hex"]], np.uint16).reshape(N, K)
    x = np.array([int(h, 16) for h in g["x_bf16_hex"]], np.uint16).reshape(-1, K)
    L = oracle.encode(W, S=S, p=p)
    assert L["codes"].ravel().tolist() == g["codes"]
    assert [format(int(v), "04x") for v in L["norms"].ravel()] == g["norms_fp16_hex"]
    assert L["q8"].ravel().tolist() == g["q8"]
    assert [format(int(v), "04x") for v in L["scale"]] == g["scale_fp16_hex"]
    assert L["idx"].tolist() == g["idx"]
    What = oracle.decode_rows(L)
    assert [float(v).hex() for v in What.ravel()] == g["What_f64_hex"]
    assert [float(v).hex() for v in oracle.matmul(What, x).ravel()] == g["y_f64_hex"]
