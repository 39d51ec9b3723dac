// encode.cu -- offline BiSCo encoder on the GPU (Sec. III-E Eq. 8 and
// Eq. 10, Sec. III-C Eq. 3, Sec. III-D Eq. 5-7), with output-row
// protection and the coupled MLP channel set of Sec. III-E Eq. 9.
//
// Every floating-point step is binary64 with an explicit rounding intrinsic
// (no FMA contraction; this file is also compiled with --fmad=false), sums
// run in a fixed order, and narrowing to binary16 uses the hardware's
// round-to-nearest-even conversion, so the produced bytes are a pure
// function of the input bits.
#include <cuda_runtime.h>
#include <stdint.h>

#include "bisco_dev.cuh"
#include "bisco_host.h"

namespace bisco {
namespace {

__device__ __forceinline__ uint16_t f64_to_f16_rn(double x) {
    unsigned short r;
    asm("cvt.rn.f16.f64 %0, %1;" : "=h"(r) : "d"(x));
    return r;
}

__device__ __forceinline__ double f16_to_f64(uint16_t h) {
    return static_cast<double>(__half2float(__ushort_as_half(h)));
}

__device__ __forceinline__ double bf16_to_f64(uint16_t b) {
    return static_cast<double>(__uint_as_float(static_cast<uint32_t>(b) << 16));
}

__device__ __forceinline__ bool bf16_nonfinite(uint16_t b) { return (b & 0x7F80u) == 0x7F80u; }

// Eq. 8 score of every input column: g_j * sqrt(sum_{i ascending} W_ij^2).
// One thread per column; also rejects non-finite weights.
__global__ void __launch_bounds__(128) k_colscore(const uint16_t *__restrict__ W,
                                                  const float *__restrict__ g, int N, int K,
                                                  double *__restrict__ score, int *err) {
    const int j = blockIdx.x * blockDim.x + threadIdx.x;
    if (j >= K) return;
    double sum = 0.0;
    bool bad = false;
    const uint16_t *col = W + j;
    int i = 0;
    for (; i + 8 <= N; i += 8) {
        uint16_t b[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) b[u] = col[static_cast<int64_t>(i + u) * K];
#pragma unroll
        for (int u = 0; u < 8; ++u) {
            bad |= bf16_nonfinite(b[u]);
            const double w = bf16_to_f64(b[u]);
            sum = __dadd_rn(sum, __dmul_rn(w, w));
        }
    }
    for (; i < N; ++i) {
        const uint16_t b = col[static_cast<int64_t>(i) * K];
        bad |= bf16_nonfinite(b);
        const double w = bf16_to_f64(b);
        sum = __dadd_rn(sum, __dmul_rn(w, w));
    }
    if (bad) latch_error(err, BISCO_ERR_RANGE);
    double s = __dsqrt_rn(sum);
    if (g) s = __dmul_rn(static_cast<double>(g[j]), s);
    score[j] = s;
}

// Eq. 8 TopK, step 1: rank_j = number of columns that precede j in the
// order (score descending, index ascending); column j is protected iff
// rank_j < p.  One thread per column, scores staged through shared memory;
// counting stops once every thread of the block has reached p.
constexpr int kRankThreads = 256;
constexpr int kRankTile = 2048;

__global__ void __launch_bounds__(kRankThreads) k_rank(const double *__restrict__ score, int K,
                                                       int p, int32_t *__restrict__ rank_out) {
    __shared__ double s[kRankTile];
    const int j = blockIdx.x * blockDim.x + threadIdx.x;
    const double sj = j < K ? score[j] : 0.0;
    int rank = 0;
    for (int q0 = 0; q0 < K; q0 += kRankTile) {
        const int n = min(kRankTile, K - q0);
        __syncthreads();
        for (int q = threadIdx.x; q < n; q += blockDim.x) s[q] = score[q0 + q];
        __syncthreads();
        if (j < K && rank < p) {
            for (int q = 0; q < n; ++q) {
                const double sq = s[q];
                rank += (sq > sj) || (sq == sj && q0 + q < j);
            }
        }
        if (__syncthreads_and(j >= K || rank >= p)) break;
    }
    if (j < K) rank_out[j] = rank;
}

// Eq. 8 TopK, step 2 (one CTA): protected-column map and the ascending list
// of protected columns, by an ordered compaction over contiguous ranges.
constexpr int kCompactThreads = 1024;

__global__ void __launch_bounds__(kCompactThreads) k_compact(const int32_t *__restrict__ rank,
                                                             int K, int p,
                                                             uint8_t *__restrict__ prot,
                                                             int32_t *__restrict__ idx) {
    __shared__ int counts[kCompactThreads];
    const int per = (K + kCompactThreads - 1) / kCompactThreads;
    const int j0 = min(K, static_cast<int>(threadIdx.x) * per);
    const int j1 = min(K, j0 + per);
    int mine = 0;
    for (int j = j0; j < j1; ++j) {
        const uint8_t f = rank[j] < p ? 1 : 0;
        prot[j] = f;
        mine += f;
    }
    counts[threadIdx.x] = mine;
    __syncthreads();
    if (threadIdx.x == 0) {
        int run = 0;
        for (int t = 0; t < kCompactThreads; ++t) {
            const int c = counts[t];
            counts[t] = run;
            run += c;
        }
    }
    __syncthreads();
    int pos = counts[threadIdx.x];
    for (int j = j0; j < j1; ++j)
        if (prot[j]) idx[pos++] = j;
}

// Eq. 10 per-channel 8-bit quantiser, one CTA per q8 column t < p_pad
// (columns t >= p are the zero padding).
__global__ void __launch_bounds__(256) k_q8(const uint16_t *__restrict__ W, int N, int K, int p,
                                            int p_pad, const int32_t *__restrict__ idx,
                                            int8_t *__restrict__ q8, uint16_t *__restrict__ scale,
                                            int *err) {
    const int t = blockIdx.x;
    if (t >= p) {
        for (int i = threadIdx.x; i < N; i += blockDim.x) q8[static_cast<int64_t>(i) * p_pad + t] = 0;
        return;
    }
    const int j = idx[t];
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
    const uint16_t s16 = f64_to_f16_rn(__ddiv_rn(red[0], 127.0));
    if ((s16 & 0x7C00u) == 0x7C00u) {
        if (threadIdx.x == 0) latch_error(err, BISCO_ERR_RANGE);
        return;
    }
    if (threadIdx.x == 0) scale[t] = s16;
    const double s = f16_to_f64(s16);
    for (int i = threadIdx.x; i < N; i += blockDim.x) {
        double q = 0.0;
        if (s != 0.0) {
            q = rint(__ddiv_rn(bf16_to_f64(W[static_cast<int64_t>(i) * K + j]), s));
            q = fmin(127.0, fmax(-127.0, q));
        }
        q8[static_cast<int64_t>(i) * p_pad + t] = static_cast<int8_t>(static_cast<int>(q));
    }
}

// Eq. 3 + Eq. 5-7: one thread per (row, chunk); S sign/norm stages on the
// residual, protected entries held at zero in every stage.  `prot` maps the
// protected input columns ([K] bytes), or with kRows the protected output
// rows ([N] bytes), whose chunks then code as norm 0, sign byte 0.
template <bool kRows>
__global__ void __launch_bounds__(256) k_stages(const uint16_t *__restrict__ W, int N, int K, int S,
                                                const uint8_t *__restrict__ prot,
                                                uint8_t *__restrict__ codes,
                                                uint16_t *__restrict__ norms, int *err) {
    const int C = K / 8;
    const int64_t e = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (e >= static_cast<int64_t>(N) * C) return;
    const int i = static_cast<int>(e / C);
    const int c = static_cast<int>(e % C);
    const uint4 raw = *reinterpret_cast<const uint4 *>(W + static_cast<int64_t>(i) * K + 8 * c);
    uint32_t pv[2];
    if (kRows) {
        pv[0] = pv[1] = prot[i] ? 0xFFFFFFFFu : 0u;
    } else {
        const uint2 pm = *reinterpret_cast<const uint2 *>(prot + 8 * c);
        pv[0] = pm.x;
        pv[1] = pm.y;
    }
    const uint32_t wv[4] = {raw.x, raw.y, raw.z, raw.w};
    bool pr[8];
    double v[8];
#pragma unroll
    for (int k = 0; k < 8; ++k) {
        pr[k] = ((pv[k / 4] >> (8 * (k % 4))) & 0xFFu) != 0;
        const uint16_t b = static_cast<uint16_t>(wv[k / 2] >> (16 * (k % 2)));
        v[k] = pr[k] ? 0.0 : bf16_to_f64(b);
    }
    const double inv_sqrt8 = __ddiv_rn(1.0, __dsqrt_rn(8.0));
    for (int s = 0; s < S; ++s) {
        double sum = __dmul_rn(v[0], v[0]);
#pragma unroll
        for (int k = 1; k < 8; ++k) sum = __dadd_rn(sum, __dmul_rn(v[k], v[k]));
        const uint16_t n16 = f64_to_f16_rn(__dsqrt_rn(sum));
        if ((n16 & 0x7C00u) == 0x7C00u) latch_error(err, BISCO_ERR_RANGE);
        uint32_t bits = 0;
#pragma unroll
        for (int k = 0; k < 8; ++k) bits |= (v[k] < 0.0 ? 1u : 0u) << k;
        const double t = __dmul_rn(f16_to_f64(n16), inv_sqrt8);
#pragma unroll
        for (int k = 0; k < 8; ++k) {
            const double rhat = ((bits >> k) & 1u) ? -t : t;
            v[k] = pr[k] ? 0.0 : __dsub_rn(v[k], rhat);
        }
        const int64_t o = (static_cast<int64_t>(s) * N + i) * C + c;
        codes[o] = static_cast<uint8_t>(bits);
        norms[o] = n16;
    }
}

// Row score for output-row protection: g_i * sqrt(sum_{k ascending} W_ik^2).
// One thread per row; also rejects non-finite weights.
__global__ void __launch_bounds__(128) k_rowscore(const uint16_t *__restrict__ W,
                                                  const float *__restrict__ g, int N, int K,
                                                  double *__restrict__ score, int *err) {
    const int i = blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= N) return;
    const uint4 *row = reinterpret_cast<const uint4 *>(W + static_cast<int64_t>(i) * K);
    double sum = 0.0;
    bool bad = false;
    for (int c = 0; c < K / 8; ++c) {
        const uint4 raw = row[c];
        const uint32_t wv[4] = {raw.x, raw.y, raw.z, raw.w};
#pragma unroll
        for (int k = 0; k < 8; ++k) {
            const uint16_t b = static_cast<uint16_t>(wv[k / 2] >> (16 * (k % 2)));
            bad |= bf16_nonfinite(b);
            const double w = bf16_to_f64(b);
            sum = __dadd_rn(sum, __dmul_rn(w, w));
        }
    }
    if (bad) latch_error(err, BISCO_ERR_RANGE);
    double s = __dsqrt_rn(sum);
    if (g) s = __dmul_rn(static_cast<double>(g[i]), s);
    score[i] = s;
}

// Eq. 9 coupled score of intermediate channel j of a gated MLP (gate and up
// [F][H], down [H][F]): the gate row norm, the up row norm and the down
// column norm, each weighted by its own g (NULL = 1) and added in that
// order.  One thread per channel.
__global__ void __launch_bounds__(128) k_coupled_score(
    const uint16_t *__restrict__ Wg, const uint16_t *__restrict__ Wu,
    const uint16_t *__restrict__ Wd, const float *__restrict__ gg, const float *__restrict__ gu,
    const float *__restrict__ gd, int F, int H, double *__restrict__ score, int *err) {
    const int j = blockIdx.x * blockDim.x + threadIdx.x;
    if (j >= F) return;
    double sg = 0.0, su = 0.0, sd = 0.0;
    bool bad = false;
    for (int h = 0; h < H; ++h) {
        const uint16_t a = Wg[static_cast<int64_t>(j) * H + h];
        const uint16_t b = Wu[static_cast<int64_t>(j) * H + h];
        const uint16_t c = Wd[static_cast<int64_t>(h) * F + j];
        bad |= bf16_nonfinite(a) | bf16_nonfinite(b) | bf16_nonfinite(c);
        const double da = bf16_to_f64(a), db = bf16_to_f64(b), dc = bf16_to_f64(c);
        sg = __dadd_rn(sg, __dmul_rn(da, da));
        su = __dadd_rn(su, __dmul_rn(db, db));
        sd = __dadd_rn(sd, __dmul_rn(dc, dc));
    }
    if (bad) latch_error(err, BISCO_ERR_RANGE);
    double tg = __dsqrt_rn(sg), tu = __dsqrt_rn(su), td = __dsqrt_rn(sd);
    if (gg) tg = __dmul_rn(static_cast<double>(gg[j]), tg);
    if (gu) tu = __dmul_rn(static_cast<double>(gu[j]), tu);
    if (gd) td = __dmul_rn(static_cast<double>(gd[j]), td);
    score[j] = __dadd_rn(__dadd_rn(tg, tu), td);
}

// A caller-given protected set (one CTA): the map over the n channels and
// the stored index list.  An index outside [0, n) or out of ascending
// order latches BISCO_ERR_INVALID_ARG; an out-of-range one is stored as 0
// so that the kernels after this one stay inside the weight.
__global__ void __launch_bounds__(1024) k_set_map(const int32_t *__restrict__ idx_in, int p, int n,
                                                  uint8_t *__restrict__ map,
                                                  int32_t *__restrict__ idx_out, int *err) {
    for (int j = threadIdx.x; j < n; j += blockDim.x) map[j] = 0;
    __syncthreads();
    for (int t = threadIdx.x; t < p; t += blockDim.x) {
        const int i = idx_in[t];
        const bool in_range = i >= 0 && i < n;
        if (!in_range || (t > 0 && idx_in[t - 1] >= i)) latch_error(err, BISCO_ERR_INVALID_ARG);
        idx_out[t] = in_range ? i : 0;
        if (in_range) map[i] = 1;
    }
}

// Eq. 10 on protected output rows, one CTA per row t < p: one fp16 scale
// per row, q8 [p][kp] with kp = roundup(K, 16), zero padding.
__global__ void __launch_bounds__(256) k_q8_rows(const uint16_t *__restrict__ W, int N, int K,
                                                 int kp, const int32_t *__restrict__ idx,
                                                 int8_t *__restrict__ q8,
                                                 uint16_t *__restrict__ scale, int *err) {
    const int t = blockIdx.x;
    const int i = idx[t];
    int8_t *qrow = q8 + static_cast<int64_t>(t) * kp;
    if (i < 0 || i >= N) {   // only after a latched k_set_map error
        for (int k = threadIdx.x; k < kp; k += blockDim.x) qrow[k] = 0;
        return;
    }
    const uint16_t *wrow = W + static_cast<int64_t>(i) * K;
    double m = 0.0;
    for (int k = threadIdx.x; k < K; k += blockDim.x) m = fmax(m, fabs(bf16_to_f64(wrow[k])));
    __shared__ double red[256];
    red[threadIdx.x] = m;
    __syncthreads();
    for (int w = 128; w > 0; w >>= 1) {
        if (threadIdx.x < w) red[threadIdx.x] = fmax(red[threadIdx.x], red[threadIdx.x + w]);
        __syncthreads();
    }
    const uint16_t s16 = f64_to_f16_rn(__ddiv_rn(red[0], 127.0));
    if ((s16 & 0x7C00u) == 0x7C00u) {
        if (threadIdx.x == 0) latch_error(err, BISCO_ERR_RANGE);
        return;
    }
    if (threadIdx.x == 0) scale[t] = s16;
    const double s = f16_to_f64(s16);
    for (int k = threadIdx.x; k < kp; k += blockDim.x) {
        double q = 0.0;
        if (k < K && s != 0.0) {
            q = rint(__ddiv_rn(bf16_to_f64(wrow[k]), s));
            q = fmin(127.0, fmax(-127.0, q));
        }
        qrow[k] = static_cast<int8_t>(static_cast<int>(q));
    }
}

// Empty kernel that ends every encode.  bisco_gemv starts reading a layer
// before it waits on the kernels ahead of it in the stream (programmatic
// dependent launch); with this ordinary launch between them, the stage
// kernel has completed, with its writes visible, before the GEMV starts.
__global__ void k_encode_done() {}

}  // namespace

static size_t round_up(size_t v, size_t a) { return (v + a - 1) / a * a; }

size_t encode_workspace_bytes(int N, int K) {
    if (N < 1 || K < 8 || K % 8) return 0;
    const size_t k = static_cast<size_t>(K);
    return round_up(8 * k, 256) + round_up(4 * k, 256) + round_up(k, 256);
}

bisco_status launch_encode(const uint16_t *W, const float *g, const bisco_layer &L,
                           void *workspace, int *err, cudaStream_t stream) {
    const int N = L.n_out, K = L.k_in, S = L.stages, p = L.n_protected;
    const int p_pad = (p + 15) / 16 * 16;
    const size_t k = static_cast<size_t>(K);
    unsigned char *ws = static_cast<unsigned char *>(workspace);
    double *score = reinterpret_cast<double *>(ws);
    int32_t *rank = reinterpret_cast<int32_t *>(ws + round_up(8 * k, 256));
    uint8_t *prot = ws + round_up(8 * k, 256) + round_up(4 * k, 256);

    k_colscore<<<(K + 127) / 128, 128, 0, stream>>>(W, g, N, K, score, err);
    k_rank<<<(K + kRankThreads - 1) / kRankThreads, kRankThreads, 0, stream>>>(score, K, p, rank);
    k_compact<<<1, kCompactThreads, 0, stream>>>(rank, K, p, prot, L.prot_idx);
    if (L.protect_format != BISCO_PROT_INT8) {
        if (launch_q_fmt(W, L, err, stream) != BISCO_OK) return BISCO_ERR_CUDA;
    } else if (p_pad > 0) {
        k_q8<<<p_pad, 256, 0, stream>>>(W, N, K, p, p_pad, L.prot_idx, L.q8, L.q8_scale, err);
    }
    const int64_t chunks = static_cast<int64_t>(N) * (K / 8);
    k_stages<false><<<static_cast<unsigned>((chunks + 255) / 256), 256, 0, stream>>>(
        W, N, K, S, prot, L.codes, L.norms, err);
    k_encode_done<<<1, 32, 0, stream>>>();
    return cudaGetLastError() == cudaSuccess ? BISCO_OK : BISCO_ERR_CUDA;
}

// Scratch of the selection paths over n channels: scores (8n), ranks (4n)
// and the protected map (n), each 256-byte aligned.
static size_t select_ws_bytes(size_t n) {
    return round_up(8 * n, 256) + round_up(4 * n, 256) + round_up(n, 256);
}

size_t encode_workspace_bytes_axis(int N, int K, int axis) {
    if (N < 1 || K < 8 || K % 8) return 0;
    if (axis == 0) return encode_workspace_bytes(N, K);
    if (axis == 1) return select_ws_bytes(static_cast<size_t>(N));
    return 0;
}

size_t select_coupled_workspace_bytes(int F) {
    return F < 1 ? 0 : select_ws_bytes(static_cast<size_t>(F));
}

// Output-row protection: row scores, TopK over rows, Eq. 10 on the rows, and
// the stages of the row-masked weight.
bisco_status launch_encode_rows(const uint16_t *W, const float *g, const bisco_layer &L,
                                void *workspace, int *err, cudaStream_t stream) {
    const int N = L.n_out, K = L.k_in, S = L.stages, p = L.n_protected;
    const int kp = (K + 15) / 16 * 16;
    const size_t n = static_cast<size_t>(N);
    unsigned char *ws = static_cast<unsigned char *>(workspace);
    double *score = reinterpret_cast<double *>(ws);
    int32_t *rank = reinterpret_cast<int32_t *>(ws + round_up(8 * n, 256));
    uint8_t *prot = ws + round_up(8 * n, 256) + round_up(4 * n, 256);

    k_rowscore<<<(N + 127) / 128, 128, 0, stream>>>(W, g, N, K, score, err);
    k_rank<<<(N + kRankThreads - 1) / kRankThreads, kRankThreads, 0, stream>>>(score, N, p, rank);
    k_compact<<<1, kCompactThreads, 0, stream>>>(rank, N, p, prot, L.prot_idx);
    if (L.protect_format != BISCO_PROT_INT8) {
        if (launch_q_fmt_rows(W, L, err, stream) != BISCO_OK) return BISCO_ERR_CUDA;
    } else if (p > 0) {
        k_q8_rows<<<p, 256, 0, stream>>>(W, N, K, kp, L.prot_idx, L.q8, L.q8_scale, err);
    }
    const int64_t chunks = static_cast<int64_t>(N) * (K / 8);
    k_stages<true><<<static_cast<unsigned>((chunks + 255) / 256), 256, 0, stream>>>(
        W, N, K, S, prot, L.codes, L.norms, err);
    k_encode_done<<<1, 32, 0, stream>>>();
    return cudaGetLastError() == cudaSuccess ? BISCO_OK : BISCO_ERR_CUDA;
}

// The encoder with a caller-given protected set (columns for axis 0, rows
// for axis 1), for example the coupled MLP set of launch_select_coupled.
bisco_status launch_encode_with_set(const uint16_t *W, const int32_t *idx_in,
                                    const bisco_layer &L, void *workspace, int *err,
                                    cudaStream_t stream) {
    const int N = L.n_out, K = L.k_in, S = L.stages, p = L.n_protected;
    const bool rows = L.protect_axis == 1;
    const size_t n = static_cast<size_t>(rows ? N : K);
    uint8_t *prot = static_cast<unsigned char *>(workspace) + round_up(8 * n, 256) +
                    round_up(4 * n, 256);
    k_set_map<<<1, 1024, 0, stream>>>(idx_in, p, static_cast<int>(n), prot, L.prot_idx, err);
    const int64_t chunks = static_cast<int64_t>(N) * (K / 8);
    const unsigned sgrid = static_cast<unsigned>((chunks + 255) / 256);
    if (rows) {
        const int kp = (K + 15) / 16 * 16;
        if (L.protect_format != BISCO_PROT_INT8) {
            if (launch_q_fmt_rows(W, L, err, stream) != BISCO_OK) return BISCO_ERR_CUDA;
        } else if (p > 0) {
            k_q8_rows<<<p, 256, 0, stream>>>(W, N, K, kp, L.prot_idx, L.q8, L.q8_scale, err);
        }
        k_stages<true><<<sgrid, 256, 0, stream>>>(W, N, K, S, prot, L.codes, L.norms, err);
    } else {
        const int p_pad = (p + 15) / 16 * 16;
        if (L.protect_format != BISCO_PROT_INT8) {
            if (launch_q_fmt(W, L, err, stream) != BISCO_OK) return BISCO_ERR_CUDA;
        } else if (p_pad > 0) {
            k_q8<<<p_pad, 256, 0, stream>>>(W, N, K, p, p_pad, L.prot_idx, L.q8, L.q8_scale, err);
        }
        k_stages<false><<<sgrid, 256, 0, stream>>>(W, N, K, S, prot, L.codes, L.norms, err);
    }
    k_encode_done<<<1, 32, 0, stream>>>();
    return cudaGetLastError() == cudaSuccess ? BISCO_OK : BISCO_ERR_CUDA;
}

// Eq. 9 coupled selection over the F intermediate channels of a gated MLP.
bisco_status launch_select_coupled(const uint16_t *Wg, const uint16_t *Wu, const uint16_t *Wd,
                                   const float *gg, const float *gu, const float *gd, int F,
                                   int H, int p, int32_t *idx_out, void *workspace, int *err,
                                   cudaStream_t stream) {
    const size_t n = static_cast<size_t>(F);
    unsigned char *ws = static_cast<unsigned char *>(workspace);
    double *score = reinterpret_cast<double *>(ws);
    int32_t *rank = reinterpret_cast<int32_t *>(ws + round_up(8 * n, 256));
    uint8_t *prot = ws + round_up(8 * n, 256) + round_up(4 * n, 256);
    k_coupled_score<<<(F + 127) / 128, 128, 0, stream>>>(Wg, Wu, Wd, gg, gu, gd, F, H, score, err);
    k_rank<<<(F + kRankThreads - 1) / kRankThreads, kRankThreads, 0, stream>>>(score, F, p, rank);
    k_compact<<<1, kCompactThreads, 0, stream>>>(rank, F, p, prot, idx_out);
    k_encode_done<<<1, 32, 0, stream>>>();
    return cudaGetLastError() == cudaSuccess ? BISCO_OK : BISCO_ERR_CUDA;
}

}  // namespace bisco
