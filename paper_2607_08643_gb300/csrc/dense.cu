// dense.cu -- the coded layer decoded to a dense matrix in device memory
// (Sec. III-G Eq. 12 with the Eq. 10 overwrite):
//     What[i][j] = sum_s (bit_{s,i,j} ? -1 : +1) * n16_{s,i,j/8} / sqrt(8)   j not protected
//     What[i][j] = scale_j * q8[i][j]                                         j protected
// This is the materialise-then-multiply path (the decoded weight written to
// HBM once, then a dense library product), kept next to the fused kernels
// as their measured comparison and as a second check of the decode.
//
// One thread per 8-column chunk of a row: S sign bytes and S fp16 norms in
// (consecutive threads read consecutive bytes), 8 values out (consecutive
// threads write consecutive 16- or 32-byte pieces).  The stage sum is formed
// in fp32, exact for the norm magnitudes of real layers, and rounded once
// after the 1/sqrt(8) scale; a second kernel overwrites the protected
// columns with scale * q8, exact in fp32.  HBM-bound: reads S*N*K/8*3
// bytes, writes N*K*sizeof(out).
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "bisco_dev.cuh"
#include "bisco_host.h"

namespace bisco {
namespace {

constexpr float kInvSqrt8 = 0.35355339059327373f;
constexpr int kDenseThreads = 256;

__device__ __forceinline__ void store8(float *dst, const float (&v)[8]) {
    reinterpret_cast<float4 *>(dst)[0] = make_float4(v[0], v[1], v[2], v[3]);
    reinterpret_cast<float4 *>(dst)[1] = make_float4(v[4], v[5], v[6], v[7]);
}

__device__ __forceinline__ void store8(__nv_bfloat16 *dst, const float (&v)[8]) {
    uint32_t w[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const __nv_bfloat162 h = __floats2bfloat162_rn(v[2 * i], v[2 * i + 1]);
        w[i] = *reinterpret_cast<const uint32_t *>(&h);
    }
    *reinterpret_cast<uint4 *>(dst) = make_uint4(w[0], w[1], w[2], w[3]);
}

__device__ __forceinline__ void store8(__half *dst, const float (&v)[8]) {
    uint32_t w[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const __half2 h = __floats2half2_rn(v[2 * i], v[2 * i + 1]);
        w[i] = *reinterpret_cast<const uint32_t *>(&h);
    }
    *reinterpret_cast<uint4 *>(dst) = make_uint4(w[0], w[1], w[2], w[3]);
}

template <typename T>
__device__ __forceinline__ T from_f32(float v);
template <>
__device__ __forceinline__ float from_f32<float>(float v) { return v; }
template <>
__device__ __forceinline__ __nv_bfloat16 from_f32<__nv_bfloat16>(float v) { return __float2bfloat16_rn(v); }
template <>
__device__ __forceinline__ __half from_f32<__half>(float v) { return __float2half_rn(v); }

template <typename T>
__global__ void __launch_bounds__(kDenseThreads) k_decode_dense(const uint8_t *__restrict__ codes,
                                                                const uint16_t *__restrict__ norms,
                                                                int N, int K, int S, T *__restrict__ out) {
    const int C = K / 8;
    const int64_t chunks = static_cast<int64_t>(N) * C;
    const int64_t e = static_cast<int64_t>(blockIdx.x) * kDenseThreads + threadIdx.x;
    if (e >= chunks) return;
    float v[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
    for (int s = 0; s < S; ++s) {
        const uint32_t b = codes[static_cast<int64_t>(s) * chunks + e];
        const float n = __half2float(__ushort_as_half(norms[static_cast<int64_t>(s) * chunks + e]));
#pragma unroll
        for (int k = 0; k < 8; ++k) v[k] += ((b >> k) & 1u) ? -n : n;
    }
#pragma unroll
    for (int k = 0; k < 8; ++k) v[k] *= kInvSqrt8;
    store8(out + e * 8, v);   // row i = e / C, columns 8 (e % C) .. + 7
}

template <typename T>
__global__ void __launch_bounds__(kDenseThreads) k_dense_protected(const int8_t *__restrict__ q8,
                                                                   const uint16_t *__restrict__ q8_scale,
                                                                   const int32_t *__restrict__ prot_idx,
                                                                   int N, int K, int p, int p_pad,
                                                                   T *__restrict__ out, int *err) {
    const int64_t e = static_cast<int64_t>(blockIdx.x) * kDenseThreads + threadIdx.x;
    if (e >= static_cast<int64_t>(N) * p) return;
    const int i = static_cast<int>(e / p), u = static_cast<int>(e % p);
    const int j = prot_idx[u];
    if (j < 0 || j >= K) {
        latch_error(err, BISCO_ERR_INVALID_ARG);   // not a column of this layer
        return;
    }
    const float sc = __half2float(__ushort_as_half(q8_scale[u]));
    out[static_cast<int64_t>(i) * K + j] =
        from_f32<T>(sc * static_cast<float>(q8[static_cast<int64_t>(i) * p_pad + u]));
}

// One stage of Eq. 12 into a dense fp32 matrix: out (=, or += when ACC)
// (bit ? -1 : +1) * n16 / sqrt(8), one thread per 8-column chunk.  Calling it
// stage after stage is the sequential residual decode that Sec. III-G's
// packed decode (k_decode_dense: every stage in one pass) replaces.
template <bool ACC>
__global__ void __launch_bounds__(kDenseThreads) k_decode_stage(const uint8_t *__restrict__ codes,
                                                                const uint16_t *__restrict__ norms,
                                                                int64_t chunks, float *__restrict__ out) {
    const int64_t e = static_cast<int64_t>(blockIdx.x) * kDenseThreads + threadIdx.x;
    if (e >= chunks) return;
    const uint32_t b = codes[e];
    const float t = __half2float(__ushort_as_half(norms[e])) * kInvSqrt8;
    float v[8];
#pragma unroll
    for (int k = 0; k < 8; ++k) v[k] = ((b >> k) & 1u) ? -t : t;
    if constexpr (ACC) {
        const float4 a = reinterpret_cast<const float4 *>(out + e * 8)[0];
        const float4 c = reinterpret_cast<const float4 *>(out + e * 8)[1];
        v[0] += a.x; v[1] += a.y; v[2] += a.z; v[3] += a.w;
        v[4] += c.x; v[5] += c.y; v[6] += c.z; v[7] += c.w;
    }
    store8(out + e * 8, v);
}

template <typename T>
bisco_status launch_dense_t(const bisco_layer &L, T *out, int *err, cudaStream_t stream) {
    const int N = L.n_out, K = L.k_in, S = L.stages, p = L.n_protected;
    const int64_t chunks = static_cast<int64_t>(N) * (K / 8);
    k_decode_dense<T><<<static_cast<unsigned>((chunks + kDenseThreads - 1) / kDenseThreads), kDenseThreads,
                        0, stream>>>(reinterpret_cast<const uint8_t *>(L.codes), L.norms, N, K, S, out);
    if (cudaGetLastError() != cudaSuccess) return BISCO_ERR_CUDA;
    if (p > 0) {
        const int64_t n = static_cast<int64_t>(N) * p;
        k_dense_protected<T><<<static_cast<unsigned>((n + kDenseThreads - 1) / kDenseThreads),
                               kDenseThreads, 0, stream>>>(L.q8, L.q8_scale, L.prot_idx, N, K, p,
                                                           (p + 15) / 16 * 16, out, err);
        if (cudaGetLastError() != cudaSuccess) return BISCO_ERR_CUDA;
    }
    return BISCO_OK;
}

}  // namespace

bisco_status launch_decode_stage(const bisco_layer &L, int stage, float *out, bool accumulate,
                                 cudaStream_t stream) {
    const int64_t chunks = static_cast<int64_t>(L.n_out) * (L.k_in / 8);
    const uint8_t *codes = reinterpret_cast<const uint8_t *>(L.codes) + stage * chunks;
    const uint16_t *norms = L.norms + stage * chunks;
    const unsigned grid = static_cast<unsigned>((chunks + kDenseThreads - 1) / kDenseThreads);
    if (accumulate)
        k_decode_stage<true><<<grid, kDenseThreads, 0, stream>>>(codes, norms, chunks, out);
    else
        k_decode_stage<false><<<grid, kDenseThreads, 0, stream>>>(codes, norms, chunks, out);
    return cudaGetLastError() == cudaSuccess ? BISCO_OK : BISCO_ERR_CUDA;
}

bisco_status launch_dense_protected_f32(const bisco_layer &L, float *out, int *err, cudaStream_t stream) {
    const int N = L.n_out, K = L.k_in, p = L.n_protected;
    if (p == 0) return BISCO_OK;
    const int64_t n = static_cast<int64_t>(N) * p;
    k_dense_protected<float><<<static_cast<unsigned>((n + kDenseThreads - 1) / kDenseThreads), kDenseThreads,
                               0, stream>>>(L.q8, L.q8_scale, L.prot_idx, N, K, p, (p + 15) / 16 * 16, out, err);
    return cudaGetLastError() == cudaSuccess ? BISCO_OK : BISCO_ERR_CUDA;
}

bisco_status launch_decode_dense(const bisco_layer &L, void *out, int dtype, int *err,
                                 cudaStream_t stream) {
    switch (dtype) {
        case BISCO_DENSE_F32: return launch_dense_t(L, static_cast<float *>(out), err, stream);
        case BISCO_DENSE_BF16: return launch_dense_t(L, static_cast<__nv_bfloat16 *>(out), err, stream);
        case BISCO_DENSE_F16: return launch_dense_t(L, static_cast<__half *>(out), err, stream);
        default: return BISCO_ERR_INVALID_ARG;
    }
}

}  // namespace bisco
