"""Writes tests/golden/oracle_small_layer.json: a small worked example of
the encoder (Eq. 8, Eq. 10, Eq. 3, Eq. 5-7), the dense decode (Eq. 12) and
the product, computed by the fp64 oracle alone.  It anchors the oracle's
arithmetic: a later change to it must regenerate this file, and its commit
must name the paper passage (or the reading) that justifies the change.

    python tests/golden/make_oracle_golden.py
"""
import json
import os
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(os.path.dirname(HERE))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

import oracle  # noqa: E402
from paper_2607_08643_gb300 import synth  # noqa: E402

N, K, S, P = 8, 32, 2, 2


def example():
    W = synth.layer_weights(N, K, seed=2024)
    x = synth.activations(2, K, seed=2025)
    L = oracle.encode(W, S=S, p=P)
    What = oracle.decode_rows(L)
    y = oracle.matmul(What, x)
    return {
        "_source": "fp64 oracle (oracle/bisco_oracle.c) on seeded synthetic inputs; written by "
                   "tests/golden/make_oracle_golden.py",
        "_cite": "encode: Sec. III-E Eq. 8 and Eq. 10, Sec. III-C Eq. 3, Sec. III-D Eq. 5-7; "
                 "decode: Sec. III-G Eq. 12 with the Eq. 10 overwrite; product: plain definition",
        "N": N, "K": K, "S": S, "p": P,
        "W_bf16_hex": [format(int(v), "04x") for v in W.ravel()],
        "x_bf16_hex": [format(int(v), "04x") for v in x.ravel()],
        "codes": [int(v) for v in L["codes"].ravel()],
        "norms_fp16_hex": [format(int(v), "04x") for v in L["norms"].ravel()],
        "q8": [int(v) for v in L["q8"].ravel()],
        "scale_fp16_hex": [format(int(v), "04x") for v in L["scale"].ravel()],
        "idx": [int(v) for v in L["idx"]],
        "What_f64_hex": [float(v).hex() for v in What.ravel()],
        "y_f64_hex": [float(v).hex() for v in y.ravel()],
    }


if __name__ == "__main__":
    g = example()
    with open(os.path.join(HERE, "oracle_small_layer.json"), "w") as f:   # one key per line
        f.write("{\n" + ",\n".join("%s: %s" % (json.dumps(k), json.dumps(v)) for k, v in g.items())
                + "\n}\n")
