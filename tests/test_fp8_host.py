"""The library's FP8 conversions (csrc/fp8.cuh, the header its encoder and
decode kernels use) compiled for the host and compared with the fp64 oracle
bit for bit: every code's value, and the rounding of every midpoint between
neighbouring codes, subnormals, both zeros, saturation and random values.
This checks the rounding logic of the protected-format encoder on the CPU;
the GPU parity tests check the kernels themselves."""
import math
import os
import subprocess

import numpy as np
import pytest

import oracle

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
CSRC = os.path.join(ROOT, "paper_2607_08643_gb300", "csrc")

PROBE = r"""
#include <stdio.h>
#include <stdlib.h>
#include "fp8.cuh"
// usage: probe FMT IN OUT -- IN: float64 values, OUT: one FP8 code each;
//        probe FMT - OUT    -- OUT: the float32 value of each of the 256 codes
int main(int argc, char **argv) {
    if (argc != 4) return 2;
    const int fmt = atoi(argv[1]);
    FILE *o = fopen(argv[3], "wb");
    if (!o) return 3;
    if (argv[2][0] == '-') {
        for (unsigned v = 0; v < 256; ++v) {
            const float f = bisco::fp8_to_f32(v, fmt);
            fwrite(&f, sizeof f, 1, o);
        }
    } else {
        FILE *in = fopen(argv[2], "rb");
        if (!in) return 4;
        const bisco::Fp8Format f = bisco::fp8_format(fmt);
        double x;
        while (fread(&x, sizeof x, 1, in) == 1) {
            const unsigned char c = bisco::f64_to_fp8(x, f);
            fwrite(&c, 1, 1, o);
        }
        fclose(in);
    }
    fclose(o);
    return 0;
}
"""

FMTS = [oracle.FMT_E4M3, oracle.FMT_E5M2]


@pytest.fixture(scope="module")
def probe(tmp_path_factory):
    d = tmp_path_factory.mktemp("fp8probe")
    src = d / "probe.cpp"
    src.write_text(PROBE)
    exe = d / "probe"
    subprocess.check_call(["g++", "-std=c++17", "-O2", "-ffp-contract=off", "-I", CSRC,
                           "-o", str(exe), str(src), "-lm"])
    return d, exe


def _encode(probe, fmt, xs):
    d, exe = probe
    inp, out = d / ("in%d.bin" % fmt), d / ("out%d.bin" % fmt)
    np.asarray(xs, np.float64).tofile(inp)
    subprocess.check_call([str(exe), str(fmt), str(inp), str(out)])
    return np.fromfile(out, np.uint8)


@pytest.mark.parametrize("fmt", FMTS)
def test_fp8_values_of_all_codes_match_oracle(probe, fmt):
    d, exe = probe
    out = d / ("codes%d.bin" % fmt)
    subprocess.check_call([str(exe), str(fmt), "-", str(out)])
    mine = np.fromfile(out, np.float32).astype(np.float64)
    ref = np.array([oracle.fp8_to_double(v, fmt) for v in range(256)])
    assert np.array_equal(mine, ref, equal_nan=True)


@pytest.mark.parametrize("fmt", FMTS)
def test_fp8_rounding_matches_oracle(probe, fmt):
    vals = np.array([oracle.fp8_to_double(v, fmt) for v in range(256)])
    fin = np.sort(np.unique(vals[np.isfinite(vals) & (vals >= 0)]))
    maxf = fin[-1]
    mids = (fin[1:] + fin[:-1]) / 2
    rng = np.random.default_rng(17)
    xs = np.concatenate([
        mids, -mids, np.nextafter(mids, 0), np.nextafter(mids, np.inf), fin, -fin,
        rng.uniform(-maxf, maxf, 4000), rng.normal(0, 1, 4000),
        rng.normal(0, fin[1] * 4, 2000),                       # subnormal range
        [0.0, -0.0, maxf, -maxf, maxf * 1.0004, maxf * 1.5, -maxf * 1e9, math.inf, -math.inf,
         5e-324, -1e-300],
    ])
    got = _encode(probe, fmt, xs)
    want = np.array([oracle.double_to_fp8(float(x), fmt) for x in xs], np.uint8)
    bad = np.flatnonzero(got != want)
    assert bad.size == 0, [(float(xs[i]), int(got[i]), int(want[i])) for i in bad[:5]]
    nan = _encode(probe, fmt, [math.nan])
    assert math.isnan(oracle.fp8_to_double(int(nan[0]), fmt))
