// rows.cu -- output-row protection at decode time (Sec. III-E Eq. 9 with
// Eq. 10 on rows): the protected output rows of a layer are kept as payload
// rows (INT8, FP8 E4M3 / E5M2 or BF16) with one fp16 scale each, and their
// outputs overwrite what the binary spherical stages give for those rows.
//
//   Y[m][idx[t]] = scale[t] * sum_k value(q8[t][k]) * X[m][k]        t < p
//
// value() is exact in fp32, and so are its products with bf16 activations.
// The sum runs in fp32, each lane over the columns k = 8 * lane + 256 * j,
// then a fixed butterfly over the warp, so the result does not depend on
// the launch.
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

constexpr int kRowWarps = 8;

using cvt::bf16_hi;
using cvt::bf16_lo;
using cvt::from_f32;

// Eight consecutive payload elements of a protected row, from element `off`
// (a multiple of 8): INT8 and FP8 are one 8-byte load, BF16 one 16-byte
// load; every value is exact in fp32.
template <int FMT>
__device__ __forceinline__ void load_payload8(const void *q, int64_t off, float (&v)[8]) {
    if (FMT == BISCO_PROT_BF16) {
        const uint4 w = *reinterpret_cast<const uint4 *>(static_cast<const uint16_t *>(q) + off);
        const uint32_t ww[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
        for (int e = 0; e < 8; ++e) v[e] = (e & 1) ? bf16_hi(ww[e >> 1]) : bf16_lo(ww[e >> 1]);
    } else {
        const uint2 w = *reinterpret_cast<const uint2 *>(static_cast<const uint8_t *>(q) + off);
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            const uint32_t b = ((e < 4 ? w.x : w.y) >> (8 * (e & 3))) & 0xFFu;
            v[e] = FMT == BISCO_PROT_INT8 ? static_cast<float>(static_cast<int8_t>(b))
                                          : fp8_to_f32(b, FMT);
        }
    }
}

__device__ __forceinline__ float payload_elem(const void *q, int64_t e, int fmt) {
    if (fmt == BISCO_PROT_BF16)
        return __uint_as_float(static_cast<uint32_t>(static_cast<const uint16_t *>(q)[e]) << 16);
    const uint32_t b = static_cast<const uint8_t *>(q)[e];
    return fmt == BISCO_PROT_INT8 ? static_cast<float>(static_cast<int8_t>(b)) : fp8_to_f32(b, fmt);
}

// One warp per task of RT protected rows x TOK activation rows; the tasks
// are spread over the grid, neighbouring warps sharing their activation
// rows.  Rows t >= p and tokens m >= M load row p-1 / token M-1 and store
// nothing, so every load stays inside the buffers.
template <int RT, int TOK, int FMT>
__global__ void __launch_bounds__(32 * kRowWarps) k_rows_apply(
    const void *__restrict__ q8, const uint16_t *__restrict__ scale,
    const int32_t *__restrict__ idx, int p, int kp, int K, int N,
    const uint16_t *__restrict__ X, int M, float *__restrict__ Y, int *err) {
    const int lane = threadIdx.x & 31;
    const int warp = threadIdx.x >> 5;
    const int64_t nrb = (p + RT - 1) / RT;
    const int64_t ntb = (M + TOK - 1) / TOK;
    const int64_t tasks = nrb * ntb;
    for (int64_t task = static_cast<int64_t>(blockIdx.x) * kRowWarps + warp; task < tasks;
         task += static_cast<int64_t>(gridDim.x) * kRowWarps) {
        const int rb = static_cast<int>(task % nrb);
        const int tb = static_cast<int>(task / nrb);
        int64_t qrow[RT];   // element offset of each protected row
        const uint16_t *xrow[TOK];
#pragma unroll
        for (int r = 0; r < RT; ++r) qrow[r] = static_cast<int64_t>(min(rb * RT + r, p - 1)) * kp;
#pragma unroll
        for (int m = 0; m < TOK; ++m)
            xrow[m] = X + static_cast<int64_t>(min(tb * TOK + m, M - 1)) * K;
        float acc[RT][TOK];
#pragma unroll
        for (int r = 0; r < RT; ++r)
#pragma unroll
            for (int m = 0; m < TOK; ++m) acc[r][m] = 0.f;
        for (int k = 8 * lane; k < K; k += 256) {
            uint4 xv[TOK];
            float qv[RT][8];
#pragma unroll
            for (int m = 0; m < TOK; ++m) xv[m] = *reinterpret_cast<const uint4 *>(xrow[m] + k);
#pragma unroll
            for (int r = 0; r < RT; ++r) load_payload8<FMT>(q8, qrow[r] + k, qv[r]);
#pragma unroll
            for (int e = 0; e < 8; ++e) {
                float xe[TOK];
#pragma unroll
                for (int m = 0; m < TOK; ++m) {
                    const uint32_t w = e < 2 ? xv[m].x : e < 4 ? xv[m].y : e < 6 ? xv[m].z : xv[m].w;
                    xe[m] = (e & 1) ? bf16_hi(w) : bf16_lo(w);
                }
#pragma unroll
                for (int r = 0; r < RT; ++r)
#pragma unroll
                    for (int m = 0; m < TOK; ++m) acc[r][m] = fmaf(qv[r][e], xe[m], acc[r][m]);
            }
        }
#pragma unroll
        for (int r = 0; r < RT; ++r)
#pragma unroll
            for (int m = 0; m < TOK; ++m)
#pragma unroll
                for (int off = 16; off > 0; off >>= 1)
                    acc[r][m] += __shfl_xor_sync(0xFFFFFFFFu, acc[r][m], off);
        if (lane == 0) {
#pragma unroll
            for (int r = 0; r < RT; ++r) {
                const int t = rb * RT + r;
                if (t >= p) continue;
                const int i = idx[t];
                if (i < 0 || i >= N) {
                    latch_error(err, BISCO_ERR_INVALID_ARG);   // not a row of this layer
                    continue;
                }
                const float s = __half2float(__ushort_as_half(scale[t]));
#pragma unroll
                for (int m = 0; m < TOK; ++m) {
                    const int mm = tb * TOK + m;
                    if (mm < M) Y[static_cast<int64_t>(mm) * N + i] = s * acc[r][m];
                }
            }
        }
    }
}

// Dense protected rows, one CTA per row t: out[idx[t]][k] = scale[t] * value(q8[t][k])
// (exact in fp32, rounded once to the output type).
template <typename T>
__global__ void __launch_bounds__(256) k_rows_dense(const void *__restrict__ q8,
                                                    const uint16_t *__restrict__ scale,
                                                    const int32_t *__restrict__ idx, int fmt,
                                                    int kp, int K, int N, T *__restrict__ out,
                                                    int *err) {
    const int t = blockIdx.x;
    const int i = idx[t];
    if (i < 0 || i >= N) {
        if (threadIdx.x == 0) latch_error(err, BISCO_ERR_INVALID_ARG);
        return;
    }
    const float s = __half2float(__ushort_as_half(scale[t]));
    const int64_t q0 = static_cast<int64_t>(t) * kp;
    T *orow = out + static_cast<int64_t>(i) * K;
    for (int k = threadIdx.x; k < K; k += blockDim.x)
        orow[k] = from_f32<T>(s * payload_elem(q8, q0 + k, fmt));
}

template <int RT, int TOK, int FMT>
bisco_status launch_apply_t(const bisco_layer &L, const uint16_t *X, int M, float *Y, int *err,
                            cudaStream_t stream) {
    const int p = L.n_protected, K = L.k_in, N = L.n_out;
    const int kp = (K + 15) / 16 * 16;
    const int64_t tasks = static_cast<int64_t>((p + RT - 1) / RT) * ((M + TOK - 1) / TOK);
    const int64_t cap = static_cast<int64_t>(num_sms()) * 8;
    const int64_t blocks = (tasks + kRowWarps - 1) / kRowWarps;
    const unsigned grid = static_cast<unsigned>(blocks < cap ? blocks : cap);
    k_rows_apply<RT, TOK, FMT><<<grid, 32 * kRowWarps, 0, stream>>>(L.q8, L.q8_scale, L.prot_idx,
                                                                    p, kp, K, N, X, M, Y, err);
    return cudaGetLastError() == cudaSuccess ? BISCO_OK : BISCO_ERR_CUDA;
}

template <typename T>
bisco_status launch_rows_dense_t(const bisco_layer &L, T *out, int *err, cudaStream_t stream) {
    const int K = L.k_in;
    const int kp = (K + 15) / 16 * 16;
    k_rows_dense<T><<<L.n_protected, 256, 0, stream>>>(L.q8, L.q8_scale, L.prot_idx,
                                                       L.protect_format, kp, K, L.n_out, out, err);
    return cudaGetLastError() == cudaSuccess ? BISCO_OK : BISCO_ERR_CUDA;
}

}  // namespace

bisco_status launch_rows_apply(const bisco_layer &L, const uint16_t *X, int M, float *Y, int *err,
                               cudaStream_t stream) {
    if (L.n_protected <= 0 || M <= 0) return BISCO_OK;
    const bool small = M <= 16;
    switch (L.protect_format) {
        case BISCO_PROT_INT8:
            return small ? launch_apply_t<1, 1, BISCO_PROT_INT8>(L, X, M, Y, err, stream)
                         : launch_apply_t<4, 4, BISCO_PROT_INT8>(L, X, M, Y, err, stream);
        case BISCO_PROT_E4M3:
            return small ? launch_apply_t<1, 1, BISCO_PROT_E4M3>(L, X, M, Y, err, stream)
                         : launch_apply_t<4, 4, BISCO_PROT_E4M3>(L, X, M, Y, err, stream);
        case BISCO_PROT_E5M2:
            return small ? launch_apply_t<1, 1, BISCO_PROT_E5M2>(L, X, M, Y, err, stream)
                         : launch_apply_t<4, 4, BISCO_PROT_E5M2>(L, X, M, Y, err, stream);
        case BISCO_PROT_BF16:
            return small ? launch_apply_t<1, 1, BISCO_PROT_BF16>(L, X, M, Y, err, stream)
                         : launch_apply_t<4, 4, BISCO_PROT_BF16>(L, X, M, Y, err, stream);
        default: return BISCO_ERR_INVALID_ARG;
    }
}

bisco_status launch_rows_dense(const bisco_layer &L, void *out, int dtype, int *err,
                               cudaStream_t stream) {
    if (L.n_protected <= 0) return BISCO_OK;
    switch (dtype) {
        case BISCO_DENSE_F32: return launch_rows_dense_t(L, static_cast<float *>(out), err, stream);
        case BISCO_DENSE_BF16:
            return launch_rows_dense_t(L, static_cast<__nv_bfloat16 *>(out), err, stream);
        case BISCO_DENSE_F16: return launch_rows_dense_t(L, static_cast<__half *>(out), err, stream);
        default: return BISCO_ERR_INVALID_ARG;
    }
}

}  // namespace bisco
