// formats.cu -- protected payloads other than INT8 (the paper's
// protected-format ablation: FP8 E4M3, FP8 E5M2, BF16 for the protected
// channels of Sec. III-E Eq. 10).
//
// Encode: per protected column j, scale = fp16(max_i |W_ij| / F) with F the
// format's largest finite value, and q_ij = fp8(W_ij / scale) (binary64
// quotient rounded once to FP8, nearest even, gradual underflow, saturating
// at F); BF16 keeps the weight itself with scale 1.0.
//
// Decode: the binary spherical kernels run without the protected set, so a
// protected column carries its decoded stage value w_b; this file then adds
//   y[m][i] += sum_t (scale_t * value(q[i][t]) - w_b(i, j_t)) * x[m][j_t]
// which leaves scale * value(q) in place of the stage value (Eq. 10's
// overwrite).  All of it in fp32 except the encoder (binary64).
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "bisco_dev.cuh"
#include "bisco_host.h"
#include "convert.cuh"
#include "fp8.cuh"

namespace bisco {
namespace {

using cvt::bf16_to_f64;
using cvt::f16_to_f64;
using cvt::f64_to_f16_rn;
using cvt::from_f32;

// The value of a protected payload element (exact in fp32).
__device__ __forceinline__ float payload_value(const void *q, int64_t e, int fmt) {
    if (fmt == BISCO_PROT_BF16)
        return __uint_as_float(static_cast<uint32_t>(static_cast<const uint16_t *>(q)[e]) << 16);
    return fp8_to_f32(static_cast<const uint8_t *>(q)[e], fmt);
}

// Encoder: one CTA per payload column t < p_pad (t >= p: zero padding).
__global__ void __launch_bounds__(256) k_q_fmt(const uint16_t *__restrict__ W, int N, int K, int p,
                                               int p_pad, const int32_t *__restrict__ idx, int fmt,
                                               void *__restrict__ q, uint16_t *__restrict__ scale,
                                               int *err) {
    const int t = blockIdx.x;
    uint8_t *q8 = static_cast<uint8_t *>(q);
    uint16_t *q16 = static_cast<uint16_t *>(q);
    if (t >= p) {
        for (int i = threadIdx.x; i < N; i += blockDim.x) {
            const int64_t e = static_cast<int64_t>(i) * p_pad + t;
            if (fmt == BISCO_PROT_BF16) q16[e] = 0; else q8[e] = 0;
        }
        return;
    }
    const int j = idx[t];
    if (fmt == BISCO_PROT_BF16) {
        if (threadIdx.x == 0) scale[t] = 0x3C00u;   // 1.0
        for (int i = threadIdx.x; i < N; i += blockDim.x)
            q16[static_cast<int64_t>(i) * p_pad + t] = W[static_cast<int64_t>(i) * K + j];
        return;
    }
    const Fp8Format f = fp8_format(fmt);
    double m = 0.0;
    for (int i = threadIdx.x; i < N; i += blockDim.x)
        m = fmax(m, fabs(bf16_to_f64(W[static_cast<int64_t>(i) * K + j])));
    __shared__ double red[256];
    red[threadIdx.x] = m;
    __syncthreads();
    for (int w = 128; w > 0; w >>= 1) {
        if (threadIdx.x < w) red[threadIdx.x] = fmax(red[threadIdx.x], red[threadIdx.x + w]);
        __syncthreads();
    }
    const uint16_t s16 = f64_to_f16_rn(__ddiv_rn(red[0], f.maxf));
    if ((s16 & 0x7C00u) == 0x7C00u) {
        if (threadIdx.x == 0) latch_error(err, BISCO_ERR_RANGE);
        return;
    }
    if (threadIdx.x == 0) scale[t] = s16;
    const double s = f16_to_f64(s16);
    for (int i = threadIdx.x; i < N; i += blockDim.x) {
        const double w = bf16_to_f64(W[static_cast<int64_t>(i) * K + j]);
        q8[static_cast<int64_t>(i) * p_pad + t] = s != 0.0 ? f64_to_fp8(__ddiv_rn(w, s), f) : 0;
    }
}

// Encoder on protected output rows: one CTA per protected row t < p, one
// scale per row (the row is the protected channel), q [p][kp] with
// kp = roundup(K, 16) and zero padding past K.
__global__ void __launch_bounds__(256) k_q_fmt_rows(const uint16_t *__restrict__ W, int N, int K,
                                                    int kp, const int32_t *__restrict__ idx,
                                                    int fmt, void *__restrict__ q,
                                                    uint16_t *__restrict__ scale, int *err) {
    const int t = blockIdx.x;
    const int i = idx[t];
    uint8_t *q8 = static_cast<uint8_t *>(q) + static_cast<int64_t>(t) * kp;
    uint16_t *q16 = static_cast<uint16_t *>(q) + static_cast<int64_t>(t) * kp;
    if (i < 0 || i >= N) {   // only after a latched k_set_map error
        for (int k = threadIdx.x; k < kp; k += blockDim.x) {
            if (fmt == BISCO_PROT_BF16) q16[k] = 0; else q8[k] = 0;
        }
        return;
    }
    const uint16_t *wrow = W + static_cast<int64_t>(i) * K;
    if (fmt == BISCO_PROT_BF16) {
        if (threadIdx.x == 0) scale[t] = 0x3C00u;   // 1.0
        for (int k = threadIdx.x; k < kp; k += blockDim.x) q16[k] = k < K ? wrow[k] : 0;
        return;
    }
    const Fp8Format f = fp8_format(fmt);
    double m = 0.0;
    for (int k = threadIdx.x; k < K; k += blockDim.x) m = fmax(m, fabs(bf16_to_f64(wrow[k])));
    __shared__ double red[256];
    red[threadIdx.x] = m;
    __syncthreads();
    for (int w = 128; w > 0; w >>= 1) {
        if (threadIdx.x < w) red[threadIdx.x] = fmax(red[threadIdx.x], red[threadIdx.x + w]);
        __syncthreads();
    }
    const uint16_t s16 = f64_to_f16_rn(__ddiv_rn(red[0], f.maxf));
    if ((s16 & 0x7C00u) == 0x7C00u) {
        if (threadIdx.x == 0) latch_error(err, BISCO_ERR_RANGE);
        return;
    }
    if (threadIdx.x == 0) scale[t] = s16;
    const double s = f16_to_f64(s16);
    for (int k = threadIdx.x; k < kp; k += blockDim.x)
        q8[k] = (k < K && s != 0.0) ? f64_to_fp8(__ddiv_rn(bf16_to_f64(wrow[k]), s), f) : 0;
}

constexpr int kFixRows = 32, kFixTok = 32, kFixT = 32;

// The correction of the decode kernels' output, for a tile of 32 output
// rows x 32 activation rows, the protected columns taken 32 at a time
// through shared memory.  Thread (r = tid / 8, c = tid % 8) owns rows r and
// activation rows 4c..4c+3 of the tile; every (m, i) belongs to one thread.
__global__ void __launch_bounds__(256) k_prot_fix(const uint8_t *__restrict__ codes,
                                                  const uint16_t *__restrict__ norms,
                                                  const void *__restrict__ q,
                                                  const uint16_t *__restrict__ scale,
                                                  const int32_t *__restrict__ idx, int fmt, int N,
                                                  int K, int S, int p,
                                                  const uint16_t *__restrict__ X, int M,
                                                  float *__restrict__ Y, int *err) {
    __shared__ float s_d[kFixRows][kFixT + 1];
    __shared__ float s_x[kFixTok][kFixT + 1];
    const int tid = threadIdx.x;
    const int r = tid >> 3, c = tid & 7;
    const int i0 = blockIdx.x * kFixRows;
    const int C = K / 8, p_pad = (p + 15) / 16 * 16;
    const float inv_sqrt8 = 0.35355339059327373f;   // the decode kernels' 1/sqrt(8) in fp32
    // token tiles stride by the grid (its y extent is capped at 65535)
    for (int m0 = blockIdx.y * kFixTok; m0 < M; m0 += gridDim.y * kFixTok) {
        float acc[4] = {0.f, 0.f, 0.f, 0.f};
        for (int t0 = 0; t0 < p; t0 += kFixT) {
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const int tt = 4 * c + u, t = t0 + tt;
                // d = scale * value(q) - (stage value of that weight), row i0 + r
                float d = 0.f;
                const int i = i0 + r;
                if (t < p && i < N) {
                    const int j = idx[t];
                    if (j >= 0 && j < K) {
                        float wb = 0.f;
                        for (int s = 0; s < S; ++s) {
                            const int64_t e = (static_cast<int64_t>(s) * N + i) * C + j / 8;
                            const float n = __half2float(__ushort_as_half(norms[e]));
                            wb += ((codes[e] >> (j % 8)) & 1u) ? -n : n;
                        }
                        const float sc = __half2float(__ushort_as_half(scale[t]));
                        d = sc * payload_value(q, static_cast<int64_t>(i) * p_pad + t, fmt) -
                            wb * inv_sqrt8;
                    } else if (r == 0) {
                        latch_error(err, BISCO_ERR_INVALID_ARG);   // not a column of this layer
                    }
                }
                s_d[r][tt] = d;
                // activation (m0 + r, column j_t)
                float xv = 0.f;
                const int m = m0 + r;
                if (t < p && m < M) {
                    const int j = idx[t];
                    if (j >= 0 && j < K)
                        xv = __uint_as_float(static_cast<uint32_t>(X[static_cast<int64_t>(m) * K + j]) << 16);
                }
                s_x[r][tt] = xv;
            }
            __syncthreads();
#pragma unroll 8
            for (int tt = 0; tt < kFixT; ++tt) {
                const float d = s_d[r][tt];
#pragma unroll
                for (int u = 0; u < 4; ++u) acc[u] = fmaf(d, s_x[4 * c + u][tt], acc[u]);
            }
            __syncthreads();
        }
        const int i = i0 + r;
        if (i < N) {
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const int m = m0 + 4 * c + u;
                if (m < M) Y[static_cast<int64_t>(m) * N + i] += acc[u];
            }
        }
    }
}

// Dense decode: out[i][idx[u]] = scale_u * value(q[i][u]), one thread per (i, u).
template <typename T>
__global__ void __launch_bounds__(256) k_dense_fmt(const void *__restrict__ q,
                                                   const uint16_t *__restrict__ scale,
                                                   const int32_t *__restrict__ idx, int fmt, int N,
                                                   int K, int p, T *__restrict__ out, int *err) {
    const int64_t e = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (e >= static_cast<int64_t>(N) * p) return;
    const int i = static_cast<int>(e / p), u = static_cast<int>(e % p);
    const int j = idx[u];
    if (j < 0 || j >= K) {
        latch_error(err, BISCO_ERR_INVALID_ARG);   // not a column of this layer
        return;
    }
    const int p_pad = (p + 15) / 16 * 16;
    const float sc = __half2float(__ushort_as_half(scale[u]));
    out[static_cast<int64_t>(i) * K + j] =
        from_f32<T>(sc * payload_value(q, static_cast<int64_t>(i) * p_pad + u, fmt));
}

template <typename T>
bisco_status launch_dense_fmt_t(const bisco_layer &L, T *out, int *err, cudaStream_t stream) {
    const int64_t n = static_cast<int64_t>(L.n_out) * L.n_protected;
    k_dense_fmt<T><<<static_cast<unsigned>((n + 255) / 256), 256, 0, stream>>>(
        L.q8, L.q8_scale, L.prot_idx, L.protect_format, L.n_out, L.k_in, L.n_protected, out, err);
    return cudaGetLastError() == cudaSuccess ? BISCO_OK : BISCO_ERR_CUDA;
}

}  // namespace

bisco_status launch_q_fmt(const uint16_t *W, const bisco_layer &L, int *err, cudaStream_t stream) {
    const int p = L.n_protected, p_pad = (p + 15) / 16 * 16;
    if (p_pad == 0) return BISCO_OK;
    k_q_fmt<<<p_pad, 256, 0, stream>>>(W, L.n_out, L.k_in, p, p_pad, L.prot_idx, L.protect_format,
                                       L.q8, L.q8_scale, err);
    return cudaGetLastError() == cudaSuccess ? BISCO_OK : BISCO_ERR_CUDA;
}

bisco_status launch_q_fmt_rows(const uint16_t *W, const bisco_layer &L, int *err,
                               cudaStream_t stream) {
    if (L.n_protected <= 0) return BISCO_OK;
    const int kp = (L.k_in + 15) / 16 * 16;
    k_q_fmt_rows<<<L.n_protected, 256, 0, stream>>>(W, L.n_out, L.k_in, kp, L.prot_idx,
                                                    L.protect_format, L.q8, L.q8_scale, err);
    return cudaGetLastError() == cudaSuccess ? BISCO_OK : BISCO_ERR_CUDA;
}

bisco_status launch_prot_fix(const bisco_layer &L, const uint16_t *X, int M, float *Y, int *err,
                             cudaStream_t stream) {
    if (L.n_protected <= 0 || M <= 0) return BISCO_OK;
    const int tiles = (M + kFixTok - 1) / kFixTok;
    const dim3 grid((L.n_out + kFixRows - 1) / kFixRows, tiles < 65535 ? tiles : 65535);
    k_prot_fix<<<grid, 256, 0, stream>>>(L.codes, L.norms, L.q8, L.q8_scale, L.prot_idx,
                                         L.protect_format, L.n_out, L.k_in, L.stages,
                                         L.n_protected, X, M, Y, err);
    return cudaGetLastError() == cudaSuccess ? BISCO_OK : BISCO_ERR_CUDA;
}

bisco_status launch_dense_fmt(const bisco_layer &L, void *out, int dtype, int *err,
                              cudaStream_t stream) {
    if (L.n_protected <= 0) return BISCO_OK;
    switch (dtype) {
        case BISCO_DENSE_F32: return launch_dense_fmt_t(L, static_cast<float *>(out), err, stream);
        case BISCO_DENSE_BF16:
            return launch_dense_fmt_t(L, static_cast<__nv_bfloat16 *>(out), err, stream);
        case BISCO_DENSE_F16: return launch_dense_fmt_t(L, static_cast<__half *>(out), err, stream);
        default: return BISCO_ERR_INVALID_ARG;
    }
}

}  // namespace bisco
