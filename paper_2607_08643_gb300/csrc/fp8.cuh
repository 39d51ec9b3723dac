// fp8.cuh -- FP8 E4M3 / E5M2 conversions of the protected payload formats
// (the paper's protected-format ablation, variants of Eq. 10).  Host and
// device: the kernels in formats.cu use them, and a host build of the same
// header lets the CPU tests compare them with the fp64 oracle bit for bit.
//
//   E4M3: sign, 4 exponent bits (bias 7), 3 mantissa bits; largest finite
//         448 (code 0x7E); S.1111.111 is NaN; no infinities.
//   E5M2: sign, 5 exponent bits (bias 15), 2 mantissa bits; largest finite
//         57344 (code 0x7B); exponent 31 holds infinities and NaNs.
#pragma once

#include <math.h>
#include <stdint.h>

#include "../../include/bisco.h"

#ifdef __CUDACC__
#define BISCO_HD __host__ __device__ __forceinline__
#else
#define BISCO_HD inline
#endif

namespace bisco {

struct Fp8Format {
    int mbits, bias;
    double maxf;
    uint8_t maxcode;
};

BISCO_HD Fp8Format fp8_format(int fmt) {
    if (fmt == BISCO_PROT_E4M3) return {3, 7, 448.0, 0x7E};
    return {2, 15, 57344.0, 0x7B};   // BISCO_PROT_E5M2
}

// binary64 -> FP8 bits, nearest even: the significand is scaled by a power
// of two (exact) so that the kept bits are its integer part and rounded once
// by rint; subnormals share the least normal exponent; a value that rounds
// above the largest finite one takes that one (saturation); NaN gives the
// format's NaN.
BISCO_HD uint8_t f64_to_fp8(double x, const Fp8Format &f) {
    const uint8_t sign = signbit(x) ? 0x80 : 0x00;
    if (isnan(x)) return sign | (f.mbits == 3 ? 0x7F : 0x7E);
    const double a = fabs(x);
    if (a == 0.0) return sign;
    if (isinf(a)) return sign | f.maxcode;
    int E = ilogb(a);
    if (E < 1 - f.bias) E = 1 - f.bias;
    double m = rint(ldexp(a, f.mbits - E));
    if (m == ldexp(1.0, f.mbits + 1)) {   // rounded up into the next binade
        m = ldexp(1.0, f.mbits);
        E += 1;
    }
    if (ldexp(m, E - f.mbits) > f.maxf) return sign | f.maxcode;
    const int mi = static_cast<int>(m);
    if (mi >= (1 << f.mbits))
        return sign | static_cast<uint8_t>(((E + f.bias) << f.mbits) | (mi - (1 << f.mbits)));
    return sign | static_cast<uint8_t>(mi);
}

// FP8 bits -> value (exact in fp32).
BISCO_HD float fp8_to_f32(uint32_t v, int fmt) {
    const int mb = fmt == BISCO_PROT_E4M3 ? 3 : 2;
    const int bias = fmt == BISCO_PROT_E4M3 ? 7 : 15;
    const int emax = (1 << (7 - mb)) - 1;
    const int e = static_cast<int>((v >> mb) & static_cast<uint32_t>(emax));
    const int mn = static_cast<int>(v & ((1u << mb) - 1u));
    float r;
    if (mb == 3 && e == emax && mn == 7)
        r = NAN;
    else if (mb == 2 && e == emax)
        r = mn ? NAN : INFINITY;
    else if (e == 0)
        r = ldexpf(static_cast<float>(mn), 1 - bias - mb);
    else
        r = ldexpf(static_cast<float>((1 << mb) + mn), e - bias - mb);
    return (v & 0x80u) ? -r : r;
}

}  // namespace bisco
