// lora.cu -- low-rank compensation added to a coded layer's output (the
// optional LoRA path of Sec. III-F: adapters trained while the codes stay
// fixed, stored apart from the coded layer):
//     t[b][r]  = sum_k A[r][k] x[b][k]
//     y[b][n] += scale * sum_r Bm[n][r] t[b][r]
// Two kernels, both bound by reading the adapter (rank * (K + N) bf16):
//  * k_lora_down: one warp per rank row r and block of up to 8 activation
//    rows; lane l reads 16-byte pieces l, l + 32, ... of A[r] and of each
//    x[b] (coalesced), keeps one fp32 sum per activation row, then a fixed
//    butterfly over the warp.  A is read once per 8 activation rows.
//  * k_lora_up: one thread per output n of one activation row; it reads its
//    row of Bm (rank bf16, contiguous rows: the warp reads one contiguous
//    block) and t[b] (broadcast), and adds scale * sum into y.
// The summation order depends only on the sizes, never on the launch, so the
// result is deterministic.
#include <cuda_runtime.h>
#include <stdint.h>
#include <stdlib.h>

#include "bisco_dev.cuh"
#include "bisco_host.h"

namespace bisco {
namespace {

constexpr int kDownWarps = 8;    // rank rows per CTA
constexpr int kDownRows = 8;     // activation rows per CTA
constexpr int kUpThreads = 256;

__device__ __forceinline__ float bf16f(uint32_t w, int hi) {
    return __uint_as_float(hi ? (w & 0xFFFF0000u) : (w << 16));
}

__global__ void __launch_bounds__(kDownWarps * 32) k_lora_down(const uint16_t *__restrict__ A,
                                                               const uint16_t *__restrict__ x,
                                                               int rank, int K, int batch,
                                                               float *__restrict__ t) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int r = blockIdx.x * kDownWarps + warp;
    const int b0 = blockIdx.y * kDownRows;
    const int nb = min(kDownRows, batch - b0);
    if (r >= rank) return;
    float acc[kDownRows];
#pragma unroll
    for (int i = 0; i < kDownRows; ++i) acc[i] = 0.f;
    const uint4 *arow = reinterpret_cast<const uint4 *>(A + static_cast<int64_t>(r) * K);
    for (int q = lane; q < K / 8; q += 32) {
        const uint4 a = arow[q];
        const uint32_t aw[4] = {a.x, a.y, a.z, a.w};
#pragma unroll
        for (int i = 0; i < kDownRows; ++i) {
            if (i >= nb) break;
            const uint4 v = reinterpret_cast<const uint4 *>(x + static_cast<int64_t>(b0 + i) * K)[q];
            const uint32_t vw[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
            for (int e = 0; e < 8; ++e)
                acc[i] = fmaf(bf16f(aw[e >> 1], e & 1), bf16f(vw[e >> 1], e & 1), acc[i]);
        }
    }
#pragma unroll
    for (int i = 0; i < kDownRows; ++i) {
        float v = acc[i];
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xFFFFFFFFu, v, o);
        if (lane == 0 && i < nb) t[static_cast<int64_t>(b0 + i) * rank + r] = v;
    }
}

// k_lora_down with one CTA per rank row r (and block of up to 8 activation
// rows): warp w takes the 16-byte pieces w*32 + lane + 256*i of A[r] and of
// each x[b], the warps' sums meet in shared memory and are added in warp
// order.  Eight times the warps of k_lora_down at the same bytes, for the
// small grids of decode (rank 16, batch 1: 16 CTAs instead of 2); the order
// still depends only on the sizes.
__global__ void __launch_bounds__(kDownWarps * 32) k_lora_down_split(
    const uint16_t *__restrict__ A, const uint16_t *__restrict__ x, int rank, int K, int batch,
    float *__restrict__ t) {
    __shared__ float s_part[kDownWarps][kDownRows];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int r = blockIdx.x;
    const int b0 = blockIdx.y * kDownRows;
    const int nb = min(kDownRows, batch - b0);
    float acc[kDownRows];
#pragma unroll
    for (int i = 0; i < kDownRows; ++i) acc[i] = 0.f;
    const uint4 *arow = reinterpret_cast<const uint4 *>(A + static_cast<int64_t>(r) * K);
    for (int q = warp * 32 + lane; q < K / 8; q += kDownWarps * 32) {
        const uint4 a = arow[q];
        const uint32_t aw[4] = {a.x, a.y, a.z, a.w};
#pragma unroll
        for (int i = 0; i < kDownRows; ++i) {
            if (i >= nb) break;
            const uint4 v = reinterpret_cast<const uint4 *>(x + static_cast<int64_t>(b0 + i) * K)[q];
            const uint32_t vw[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
            for (int e = 0; e < 8; ++e)
                acc[i] = fmaf(bf16f(aw[e >> 1], e & 1), bf16f(vw[e >> 1], e & 1), acc[i]);
        }
    }
#pragma unroll
    for (int i = 0; i < kDownRows; ++i) {
        float v = acc[i];
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xFFFFFFFFu, v, o);
        if (lane == 0) s_part[warp][i] = v;
    }
    __syncthreads();
    if (threadIdx.x < nb) {
        float v = 0.f;
#pragma unroll
        for (int w = 0; w < kDownWarps; ++w) v += s_part[w][threadIdx.x];
        t[static_cast<int64_t>(b0 + threadIdx.x) * rank + r] = v;
    }
}

__global__ void __launch_bounds__(kUpThreads) k_lora_up(const uint16_t *__restrict__ Bm,
                                                        const float *__restrict__ t, int rank, int N,
                                                        float scale, float *__restrict__ y) {
    const int n = blockIdx.x * kUpThreads + threadIdx.x;
    const int b = blockIdx.y;
    if (n >= N) return;
    const uint4 *brow = reinterpret_cast<const uint4 *>(Bm + static_cast<int64_t>(n) * rank);
    const float4 *trow = reinterpret_cast<const float4 *>(t + static_cast<int64_t>(b) * rank);
    float sum = 0.f;
    for (int q = 0; q < rank / 8; ++q) {
        const uint4 w = brow[q];
        const float4 t0 = trow[2 * q], t1 = trow[2 * q + 1];
        sum = fmaf(bf16f(w.x, 0), t0.x, sum);
        sum = fmaf(bf16f(w.x, 1), t0.y, sum);
        sum = fmaf(bf16f(w.y, 0), t0.z, sum);
        sum = fmaf(bf16f(w.y, 1), t0.w, sum);
        sum = fmaf(bf16f(w.z, 0), t1.x, sum);
        sum = fmaf(bf16f(w.z, 1), t1.y, sum);
        sum = fmaf(bf16f(w.w, 0), t1.z, sum);
        sum = fmaf(bf16f(w.w, 1), t1.w, sum);
    }
    float *out = y + static_cast<int64_t>(b) * N + n;
    *out = fmaf(scale, sum, *out);
}

}  // namespace

bisco_status launch_lora_apply(const uint16_t *A, const uint16_t *Bm, int rank, int N, int K,
                               float scale, const uint16_t *x, int batch, float *y, float *t,
                               cudaStream_t stream) {
    // BISCO_LORA_SPLIT=1 selects the K-split down projection (measured
    // against the default before it becomes one)
    const char *split = getenv("BISCO_LORA_SPLIT");
    if (split && split[0] == '1') {
        const dim3 gs(rank, (batch + kDownRows - 1) / kDownRows);
        k_lora_down_split<<<gs, kDownWarps * 32, 0, stream>>>(A, x, rank, K, batch, t);
    } else {
        const dim3 gd((rank + kDownWarps - 1) / kDownWarps, (batch + kDownRows - 1) / kDownRows);
        k_lora_down<<<gd, kDownWarps * 32, 0, stream>>>(A, x, rank, K, batch, t);
    }
    if (cudaGetLastError() != cudaSuccess) return BISCO_ERR_CUDA;
    const dim3 gu((N + kUpThreads - 1) / kUpThreads, batch);
    k_lora_up<<<gu, kUpThreads, 0, stream>>>(Bm, t, rank, N, scale, y);
    if (cudaGetLastError() != cudaSuccess) return BISCO_ERR_CUDA;
    return BISCO_OK;
}

}  // namespace bisco
