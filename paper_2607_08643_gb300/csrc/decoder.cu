// decoder.cu -- the learned decoder step (Sec. III-A Eq. 1, decoded per
// Sec. III-G Eq. 12) in table form.  Stage s of a chunk decodes to
// n16 * D_s(q), and since the code q of a chunk takes only 256 values, D_s
// is held as its table T_s[v][k] = D_s(q(v))_k in binary16 ([S][256][8],
// 4 KB per stage): a linear decoder A q, a sign-symmetric perceptron, or
// any other map the caller evaluated.  The identity decoder is the table
// (bit k of v ? -1 : +1) / sqrt(8).
//
//   What[i][8c + k] = sum_s n16_{s,i,c} * T_s[code_{s,i,c}][k]   (column not protected)
//   What[i][j]      = scale_t * q8[i][t]                          (j = prot_idx[t])
//
// Products fp16 x fp16 are exact in fp32; every sum runs in fp32.
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "bisco_dev.cuh"
#include "bisco_host.h"
#include "convert.cuh"

namespace bisco {
namespace {

constexpr int kTableEntries = 256 * 8;   // halves per stage

using cvt::bf16_to_f32;
using cvt::from_f32;

// Stages S tables into shared memory (S * 4 KB, 16-byte copies).
__device__ __forceinline__ void stage_tables(const uint16_t *__restrict__ tables, int S,
                                             uint4 *s_tab) {
    const uint4 *src = reinterpret_cast<const uint4 *>(tables);
    for (int u = threadIdx.x; u < S * kTableEntries / 8; u += blockDim.x) s_tab[u] = src[u];
    __syncthreads();
}

// The 8 decoded values of one chunk: w[k] = sum_s n_s * T_s[code_s][k].
__device__ __forceinline__ void decode_chunk(const uint8_t *__restrict__ codes,
                                             const uint16_t *__restrict__ norms,
                                             const uint4 *s_tab, int S, int64_t e0,
                                             int64_t stage_stride, float (&w)[8]) {
#pragma unroll
    for (int k = 0; k < 8; ++k) w[k] = 0.f;
    for (int s = 0; s < S; ++s) {
        const int64_t e = e0 + s * stage_stride;
        const uint32_t v = codes[e];
        const float n = __half2float(__ushort_as_half(norms[e]));
        const uint4 row = s_tab[s * 256 + v];
        const uint32_t hw[4] = {row.x, row.y, row.z, row.w};
#pragma unroll
        for (int h = 0; h < 4; ++h) {
            const float2 t = __half22float2(*reinterpret_cast<const __half2 *>(&hw[h]));
            w[2 * h] = fmaf(n, t.x, w[2 * h]);
            w[2 * h + 1] = fmaf(n, t.y, w[2 * h + 1]);
        }
    }
}

// Decode GEMV with a decoder table: one warp per output row, B <= 16.
// Protected columns replace their decoded value by scale * q8 (Eq. 10).
__global__ void __launch_bounds__(256) k_gemv_table(const uint8_t *__restrict__ codes,
                                                    const uint16_t *__restrict__ norms,
                                                    const uint16_t *__restrict__ tables,
                                                    const int8_t *__restrict__ q8,
                                                    const uint16_t *__restrict__ q8_scale,
                                                    const int32_t *__restrict__ prot_idx, int N,
                                                    int K, int S, int p,
                                                    const uint16_t *__restrict__ x, int B,
                                                    float *__restrict__ y, int *err) {
    __shared__ uint4 s_tab[3 * kTableEntries / 8];
    stage_tables(tables, S, s_tab);
    const int C = K / 8, p_pad = (p + 15) / 16 * 16;
    const int lane = threadIdx.x & 31;
    const int i = blockIdx.x * (blockDim.x / 32) + (threadIdx.x >> 5);
    if (i >= N) return;
    const int64_t stride = static_cast<int64_t>(N) * C;
    float acc[16];
#pragma unroll
    for (int b = 0; b < 16; ++b) acc[b] = 0.f;
    for (int c = lane; c < C; c += 32) {
        float w[8];
        decode_chunk(codes, norms, s_tab, S, static_cast<int64_t>(i) * C + c, stride, w);
#pragma unroll
        for (int b = 0; b < 16; ++b) {
            if (b >= B) break;
            const uint4 xr = *reinterpret_cast<const uint4 *>(x + static_cast<int64_t>(b) * K + 8 * c);
            const uint32_t xw[4] = {xr.x, xr.y, xr.z, xr.w};
            float d = 0.f;
#pragma unroll
            for (int h = 0; h < 4; ++h) {
                d = fmaf(w[2 * h], __uint_as_float(xw[h] << 16), d);
                d = fmaf(w[2 * h + 1], __uint_as_float(xw[h] & 0xFFFF0000u), d);
            }
            acc[b] += d;
        }
    }
    // Eq. 10: the protected columns' decoded value is replaced by scale * q8
    for (int t = lane; t < p; t += 32) {
        const int j = prot_idx[t];
        if (j < 0 || j >= K) {   // not a column of this layer
            latch_error(err, BISCO_ERR_INVALID_ARG);
            continue;
        }
        float w[8];
        decode_chunk(codes, norms, s_tab, S, static_cast<int64_t>(i) * C + j / 8, stride, w);
        float wb = 0.f;
#pragma unroll
        for (int k = 0; k < 8; ++k) wb = (k == j % 8) ? w[k] : wb;
        const float wq = __half2float(__ushort_as_half(q8_scale[t])) *
                         static_cast<float>(q8[static_cast<int64_t>(i) * p_pad + t]);
#pragma unroll
        for (int b = 0; b < 16; ++b) {
            if (b >= B) break;
            acc[b] += (wq - wb) * bf16_to_f32(x[static_cast<int64_t>(b) * K + j]);
        }
    }
#pragma unroll
    for (int b = 0; b < 16; ++b)
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) acc[b] += __shfl_xor_sync(0xffffffffu, acc[b], o);
    if (lane == 0) {
#pragma unroll
        for (int b = 0; b < 16; ++b)
            if (b < B) y[static_cast<int64_t>(b) * N + i] = acc[b];
    }
}

// k_gemv_table for K % 32 == 0: each lane takes groups of 4 consecutive
// chunks, one 32-bit code word and one 8-byte norm word per stage, and
// issues the loads of UNROLL groups before decoding any of them; S is a
// template parameter so that the words stay in registers.
template <int S, int UNROLL>
__global__ void __launch_bounds__(256) k_gemv_table_v(const uint8_t *__restrict__ codes,
                                                      const uint16_t *__restrict__ norms,
                                                      const uint16_t *__restrict__ tables,
                                                      const int8_t *__restrict__ q8,
                                                      const uint16_t *__restrict__ q8_scale,
                                                      const int32_t *__restrict__ prot_idx, int N,
                                                      int K, int p,
                                                      const uint16_t *__restrict__ x, int B,
                                                      float *__restrict__ y, int *err) {
    __shared__ uint4 s_tab[3 * kTableEntries / 8];
    stage_tables(tables, S, s_tab);
    const int C = K / 8, G = C / 4, p_pad = (p + 15) / 16 * 16;
    const int lane = threadIdx.x & 31;
    const int i = blockIdx.x * (blockDim.x / 32) + (threadIdx.x >> 5);
    if (i >= N) return;
    const uint32_t *cw32 = reinterpret_cast<const uint32_t *>(codes);
    const uint2 *nw64 = reinterpret_cast<const uint2 *>(norms);
    float acc[16];
#pragma unroll
    for (int b = 0; b < 16; ++b) acc[b] = 0.f;
    for (int g0 = lane; g0 < G; g0 += 32 * UNROLL) {
        uint32_t cw[UNROLL][S];
        uint2 nw[UNROLL][S];
#pragma unroll
        for (int u = 0; u < UNROLL; ++u) {
            const int g = min(g0 + 32 * u, G - 1);   // groups past the row reload the last one
#pragma unroll
            for (int s = 0; s < S; ++s) {
                const int64_t e = (static_cast<int64_t>(s) * N + i) * G + g;
                cw[u][s] = cw32[e];
                nw[u][s] = nw64[e];
            }
        }
#pragma unroll
        for (int u = 0; u < UNROLL; ++u) {
            const int g = g0 + 32 * u;
            if (g >= G) break;
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                float w[8];
#pragma unroll
                for (int k = 0; k < 8; ++k) w[k] = 0.f;
#pragma unroll
                for (int s = 0; s < S; ++s) {
                    const uint32_t v = (cw[u][s] >> (8 * q)) & 0xFFu;
                    const uint32_t nh = q < 2 ? nw[u][s].x : nw[u][s].y;
                    const float n = __half2float(__ushort_as_half(
                        static_cast<uint16_t>((q & 1) ? (nh >> 16) : (nh & 0xFFFFu))));
                    const uint4 row = s_tab[s * 256 + v];
                    const uint32_t hw[4] = {row.x, row.y, row.z, row.w};
#pragma unroll
                    for (int h = 0; h < 4; ++h) {
                        const float2 t = __half22float2(*reinterpret_cast<const __half2 *>(&hw[h]));
                        w[2 * h] = fmaf(n, t.x, w[2 * h]);
                        w[2 * h + 1] = fmaf(n, t.y, w[2 * h + 1]);
                    }
                }
                const int c = 4 * g + q;
#pragma unroll
                for (int b = 0; b < 16; ++b) {
                    if (b >= B) break;
                    const uint4 xr =
                        *reinterpret_cast<const uint4 *>(x + static_cast<int64_t>(b) * K + 8 * c);
                    const uint32_t xw[4] = {xr.x, xr.y, xr.z, xr.w};
                    float d = 0.f;
#pragma unroll
                    for (int h = 0; h < 4; ++h) {
                        d = fmaf(w[2 * h], __uint_as_float(xw[h] << 16), d);
                        d = fmaf(w[2 * h + 1], __uint_as_float(xw[h] & 0xFFFF0000u), d);
                    }
                    acc[b] += d;
                }
            }
        }
    }
    // Eq. 10, as in k_gemv_table
    const int64_t stride = static_cast<int64_t>(N) * C;
    for (int t = lane; t < p; t += 32) {
        const int j = prot_idx[t];
        if (j < 0 || j >= K) {
            latch_error(err, BISCO_ERR_INVALID_ARG);
            continue;
        }
        float w[8];
        decode_chunk(codes, norms, s_tab, S, static_cast<int64_t>(i) * C + j / 8, stride, w);
        float wb = 0.f;
#pragma unroll
        for (int k = 0; k < 8; ++k) wb = (k == j % 8) ? w[k] : wb;
        const float wq = __half2float(__ushort_as_half(q8_scale[t])) *
                         static_cast<float>(q8[static_cast<int64_t>(i) * p_pad + t]);
#pragma unroll
        for (int b = 0; b < 16; ++b) {
            if (b >= B) break;
            acc[b] += (wq - wb) * bf16_to_f32(x[static_cast<int64_t>(b) * K + j]);
        }
    }
#pragma unroll
    for (int b = 0; b < 16; ++b)
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) acc[b] += __shfl_xor_sync(0xffffffffu, acc[b], o);
    if (lane == 0) {
#pragma unroll
        for (int b = 0; b < 16; ++b)
            if (b < B) y[static_cast<int64_t>(b) * N + i] = acc[b];
    }
}

// Dense decode with a decoder table: one thread per chunk.
template <typename T>
__global__ void __launch_bounds__(256) k_dense_table(const uint8_t *__restrict__ codes,
                                                     const uint16_t *__restrict__ norms,
                                                     const uint16_t *__restrict__ tables, int N,
                                                     int K, int S, T *__restrict__ out) {
    __shared__ uint4 s_tab[3 * kTableEntries / 8];
    stage_tables(tables, S, s_tab);
    const int64_t chunks = static_cast<int64_t>(N) * (K / 8);
    const int64_t e = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (e >= chunks) return;
    float w[8];
    decode_chunk(codes, norms, s_tab, S, e, chunks, w);
    T *o = out + e * 8;   // chunk e covers out[i][8c .. 8c+7], i*K + 8c = 8e
#pragma unroll
    for (int k = 0; k < 8; ++k) o[k] = from_f32<T>(w[k]);
}

// Protected columns of the dense decode: out[i][prot_idx[u]] = scale_u * q8[i][u].
template <typename T>
__global__ void __launch_bounds__(256) k_dense_table_protected(const int8_t *__restrict__ q8,
                                                               const uint16_t *__restrict__ q8_scale,
                                                               const int32_t *__restrict__ prot_idx,
                                                               int N, int K, int p,
                                                               T *__restrict__ out, int *err) {
    const int64_t e = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (e >= static_cast<int64_t>(N) * p) return;
    const int i = static_cast<int>(e / p), u = static_cast<int>(e % p);
    const int j = prot_idx[u];
    if (j < 0 || j >= K) {
        latch_error(err, BISCO_ERR_INVALID_ARG);   // not a column of this layer
        return;
    }
    const int p_pad = (p + 15) / 16 * 16;
    const float sc = __half2float(__ushort_as_half(q8_scale[u]));
    out[static_cast<int64_t>(i) * K + j] =
        from_f32<T>(sc * static_cast<float>(q8[static_cast<int64_t>(i) * p_pad + u]));
}

template <typename T>
bisco_status launch_dense_table_t(const bisco_layer &L, const uint16_t *tables, T *out, int *err,
                                  cudaStream_t stream) {
    const int N = L.n_out, K = L.k_in, S = L.stages, p = L.n_protected;
    const int64_t chunks = static_cast<int64_t>(N) * (K / 8);
    k_dense_table<T><<<static_cast<unsigned>((chunks + 255) / 256), 256, 0, stream>>>(
        L.codes, L.norms, tables, N, K, S, out);
    if (cudaGetLastError() != cudaSuccess) return BISCO_ERR_CUDA;
    if (p > 0) {
        const int64_t n = static_cast<int64_t>(N) * p;
        k_dense_table_protected<T><<<static_cast<unsigned>((n + 255) / 256), 256, 0, stream>>>(
            L.q8, L.q8_scale, L.prot_idx, N, K, p, out, err);
        if (cudaGetLastError() != cudaSuccess) return BISCO_ERR_CUDA;
    }
    return BISCO_OK;
}

}  // namespace

bisco_status launch_gemv_table(const bisco_layer &L, const uint16_t *tables, const uint16_t *x,
                               int B, float *y, int *err, cudaStream_t stream) {
    const int rows_per_block = 8;
    const unsigned grid = (L.n_out + rows_per_block - 1) / rows_per_block;
    const int N = L.n_out, K = L.k_in, p = L.n_protected;
    if (K % 32 == 0) {   // 4-chunk code and norm words are aligned
        switch (L.stages) {
            case 1:
                k_gemv_table_v<1, 2><<<grid, 32 * rows_per_block, 0, stream>>>(
                    L.codes, L.norms, tables, L.q8, L.q8_scale, L.prot_idx, N, K, p, x, B, y, err);
                break;
            case 2:
                k_gemv_table_v<2, 2><<<grid, 32 * rows_per_block, 0, stream>>>(
                    L.codes, L.norms, tables, L.q8, L.q8_scale, L.prot_idx, N, K, p, x, B, y, err);
                break;
            default:
                k_gemv_table_v<3, 2><<<grid, 32 * rows_per_block, 0, stream>>>(
                    L.codes, L.norms, tables, L.q8, L.q8_scale, L.prot_idx, N, K, p, x, B, y, err);
                break;
        }
    } else {
        k_gemv_table<<<grid, 32 * rows_per_block, 0, stream>>>(L.codes, L.norms, tables, L.q8,
                                                              L.q8_scale, L.prot_idx, N, K,
                                                              L.stages, p, x, B, y, err);
    }
    return cudaGetLastError() == cudaSuccess ? BISCO_OK : BISCO_ERR_CUDA;
}

bisco_status launch_dense_table(const bisco_layer &L, const uint16_t *tables, void *out, int dtype,
                                int *err, cudaStream_t stream) {
    switch (dtype) {
        case BISCO_DENSE_F32:
            return launch_dense_table_t(L, tables, static_cast<float *>(out), err, stream);
        case BISCO_DENSE_BF16:
            return launch_dense_table_t(L, tables, static_cast<__nv_bfloat16 *>(out), err, stream);
        case BISCO_DENSE_F16:
            return launch_dense_table_t(L, tables, static_cast<__half *>(out), err, stream);
        default: return BISCO_ERR_INVALID_ARG;
    }
}

}  // namespace bisco
