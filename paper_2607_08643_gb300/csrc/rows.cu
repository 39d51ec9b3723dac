// rows.cu -- output-row protection at decode time (Sec. III-E Eq. 9 with
// Eq. 10 on rows): the protected output rows of a layer are kept as int8
// rows with one fp16 scale each, and their outputs overwrite what the
// binary spherical stages give for those rows.
//
//   Y[m][idx[t]] = scale[t] * sum_k q8[t][k] * X[m][k]        t < p
//
// The products int8 x bf16 are exact in fp32; the sum runs in fp32, each
// lane over the columns k = 8 * lane + 256 * j, then a fixed butterfly over
// the warp, so the result does not depend on the launch.
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "bisco_dev.cuh"
#include "bisco_host.h"

namespace bisco {
namespace {

constexpr int kRowWarps = 8;

__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }

// One warp per task of RT protected rows x TOK activation rows; the tasks
// are spread over the grid, neighbouring warps sharing their activation
// rows.  Rows t >= p and tokens m >= M load row p-1 / token M-1 and store
// nothing, so every load stays inside the buffers.
template <int RT, int TOK>
__global__ void __launch_bounds__(32 * kRowWarps) k_rows_apply(
    const int8_t *__restrict__ q8, const uint16_t *__restrict__ scale,
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
        const int8_t *qrow[RT];
        const uint16_t *xrow[TOK];
#pragma unroll
        for (int r = 0; r < RT; ++r)
            qrow[r] = q8 + static_cast<int64_t>(min(rb * RT + r, p - 1)) * kp;
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
            uint2 qv[RT];
#pragma unroll
            for (int m = 0; m < TOK; ++m) xv[m] = *reinterpret_cast<const uint4 *>(xrow[m] + k);
#pragma unroll
            for (int r = 0; r < RT; ++r) qv[r] = *reinterpret_cast<const uint2 *>(qrow[r] + k);
#pragma unroll
            for (int e = 0; e < 8; ++e) {
                float xe[TOK];
#pragma unroll
                for (int m = 0; m < TOK; ++m) {
                    const uint32_t w = e < 2 ? xv[m].x : e < 4 ? xv[m].y : e < 6 ? xv[m].z : xv[m].w;
                    xe[m] = (e & 1) ? bf16_hi(w) : bf16_lo(w);
                }
#pragma unroll
                for (int r = 0; r < RT; ++r) {
                    const uint32_t w = e < 4 ? qv[r].x : qv[r].y;
                    const float q = static_cast<float>(static_cast<int8_t>((w >> (8 * (e & 3))) & 0xFFu));
#pragma unroll
                    for (int m = 0; m < TOK; ++m) acc[r][m] = fmaf(q, xe[m], acc[r][m]);
                }
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

template <typename T>
__device__ __forceinline__ T from_f32(float v);
template <>
__device__ __forceinline__ float from_f32<float>(float v) { return v; }
template <>
__device__ __forceinline__ __nv_bfloat16 from_f32<__nv_bfloat16>(float v) { return __float2bfloat16_rn(v); }
template <>
__device__ __forceinline__ __half from_f32<__half>(float v) { return __float2half_rn(v); }

// Dense protected rows, one CTA per row t: out[idx[t]][k] = scale[t] * q8[t][k]
// (exact in fp32, rounded once to the output type).
template <typename T>
__global__ void __launch_bounds__(256) k_rows_dense(const int8_t *__restrict__ q8,
                                                    const uint16_t *__restrict__ scale,
                                                    const int32_t *__restrict__ idx, int kp, int K,
                                                    int N, T *__restrict__ out, int *err) {
    const int t = blockIdx.x;
    const int i = idx[t];
    if (i < 0 || i >= N) {
        if (threadIdx.x == 0) latch_error(err, BISCO_ERR_INVALID_ARG);
        return;
    }
    const float s = __half2float(__ushort_as_half(scale[t]));
    const int8_t *qrow = q8 + static_cast<int64_t>(t) * kp;
    T *orow = out + static_cast<int64_t>(i) * K;
    for (int k = threadIdx.x; k < K; k += blockDim.x)
        orow[k] = from_f32<T>(s * static_cast<float>(qrow[k]));
}

template <int RT, int TOK>
bisco_status launch_apply_t(const bisco_layer &L, const uint16_t *X, int M, float *Y, int *err,
                            cudaStream_t stream) {
    const int p = L.n_protected, K = L.k_in, N = L.n_out;
    const int kp = (K + 15) / 16 * 16;
    const int64_t tasks = static_cast<int64_t>((p + RT - 1) / RT) * ((M + TOK - 1) / TOK);
    const int64_t cap = static_cast<int64_t>(num_sms()) * 8;
    const int64_t blocks = (tasks + kRowWarps - 1) / kRowWarps;
    const unsigned grid = static_cast<unsigned>(blocks < cap ? blocks : cap);
    k_rows_apply<RT, TOK><<<grid, 32 * kRowWarps, 0, stream>>>(L.q8, L.q8_scale, L.prot_idx, p, kp,
                                                               K, N, X, M, Y, err);
    return cudaGetLastError() == cudaSuccess ? BISCO_OK : BISCO_ERR_CUDA;
}

template <typename T>
bisco_status launch_rows_dense_t(const bisco_layer &L, T *out, int *err, cudaStream_t stream) {
    const int K = L.k_in;
    const int kp = (K + 15) / 16 * 16;
    k_rows_dense<T><<<L.n_protected, 256, 0, stream>>>(L.q8, L.q8_scale, L.prot_idx, kp, K, L.n_out,
                                                       out, err);
    return cudaGetLastError() == cudaSuccess ? BISCO_OK : BISCO_ERR_CUDA;
}

}  // namespace

bisco_status launch_rows_apply(const bisco_layer &L, const uint16_t *X, int M, float *Y, int *err,
                               cudaStream_t stream) {
    if (L.n_protected <= 0 || M <= 0) return BISCO_OK;
    if (M <= 16) return launch_apply_t<1, 1>(L, X, M, Y, err, stream);
    return launch_apply_t<4, 4>(L, X, M, Y, err, stream);
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
