// gemv.cu -- decode-time y = What x straight from the coded layer
// (Sec. III-G Eq. 12 with the Eq. 10 protected scatter), batch 1..16.
//
// Shared decode scheme (GB300, HBM-bound):
//  * A producer thread streams ring slots of the sign bytes and fp16 norms
//    of all S stages (rows x 512*WQ input columns) into shared memory with
//    TMA (cp.async.bulk.tensor, mbarrier complete_tx).  Weights never depend
//    on earlier kernels, so this starts before the wait on the previous grid
//    (programmatic dependent launch), and every CTA lets the next kernel in
//    the stream be scheduled at once: CTAs of consecutive layers share an SM
//    and the next layer's weights stream in while this one finishes.
//  * Consumer warps decode in registers: for a 32-bit code word holding
//    chunks c..c+3 (byte per chunk), one shift brings the sign bits of
//    element i of chunk c and of chunk c+2 to bits 15 and 31, and one LOP3
//    ((w << s) & 0x80008000) ^ (n_c | n_{c+2} << 16) yields the fp16 pair
//    (+-n_c, +-n_{c+2}) exactly.  These pairs are the A fragments of
//    mma.m16n8k16 (fp16 in, fp32 accumulate), one MMA per stage, so the
//    stage sum of Eq. 12 is exact in fp32.  The activations are staged once
//    per CTA, as fp16 in the matching permuted order, with the protected
//    columns zeroed (Eq. 10's overwrite); lanes whose activation row is >= B
//    read a zero block, so every fragment load is unconditional.
//  * The int8 protected columns are a few more k tiles on the same MMA: q8
//    as exact fp16 integers against scale_j * x_j split into fp16 hi + lo;
//    y = acc / sqrt(8) + acc_protected.
//
// k_gemv_stream (batch <= 8, at least one 16-row tile per SM): one
// persistent CTA per SM walks its 16-row tiles while the ring keeps
// streaming across tile boundaries; a reducer warp computes each tile's
// protected term and writes y, so the consumer warps never stop decoding.
// k_gemv (short layers, batch > 8): a cluster of CK CTAs splits K; ranks 1..
// store their partial sums into rank 0's shared memory and arrive on an
// mbarrier there; rank 0 adds them in rank order (deterministic, no atomics).
#include <cuda_runtime.h>
#include <stdint.h>
#include <stdio.h>
#include <stdlib.h>

#include <algorithm>

#include "bisco_dev.cuh"
#include "bisco_host.h"

namespace bisco {
namespace {

constexpr int kSlab = 512;   // input columns one consumer warp covers per slot
constexpr float kInvSqrt8 = 0.35355339059327373f;

struct GemvArgs {
    const uint16_t *x;
    float *y;
    const uint16_t *q8_scale;
    const int32_t *prot_idx;
    int *err;
    int N, K, B, p;
    int wide_per_rank;   // ring slots' worth of columns per cluster rank (k_gemv)
    int nslot;           // ring depth
    uint32_t off_xt, off_q8, off_red, off_cl, off_bar, off_pidx, off_pmask, off_pu, off_zero,
        off_prot;
    int pidx_cap;        // protected entries staged per CTA (multiple of 16)
    int xt_pitch;        // bytes per activation row in the staged operand
};

__device__ __forceinline__ uint32_t word_of(const uint4 &v, int i) {
    return i == 0 ? v.x : (i == 1 ? v.y : (i == 2 ? v.z : v.w));
}

// A fragment of one k16 tile from the code words of rows lo/hi: pairs i0
// and i0+1 of each word, ((w << (15-i)) & 0x80008000) ^ norm pair.
__device__ __forceinline__ void decode_pairs(int i0, uint32_t cl, uint32_t ch, uint32_t nl,
                                             uint32_t nh, uint32_t (&af)[4]) {
    af[0] = lop3_and_xor(cl << (15 - i0), 0x80008000u, nl);
    af[1] = lop3_and_xor(ch << (15 - i0), 0x80008000u, nh);
    af[2] = lop3_and_xor(cl << (14 - i0), 0x80008000u, nl);
    af[3] = lop3_and_xor(ch << (14 - i0), 0x80008000u, nh);
}

__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }

// A-byte aligned base of the dynamic shared memory (1024 for the 128-byte
// swizzle, 128 for plain TMA boxes), derived by pointer arithmetic on the
// shared array so that accesses stay shared-space ones.
template <uint32_t A = 1024>
__device__ __forceinline__ unsigned char *aligned_smem(unsigned char *raw) {
    return raw + ((A - (smem_u32(raw) & (A - 1u))) & (A - 1u));
}

constexpr int kMaxGroup = 4;   // layers sharing one activation in a grouped launch

// Per-layer shared-memory view used by the activation staging.
struct StageView {
    unsigned char *xt;        // [B][xt_pitch] staged fp16 operand
    const uint32_t *pmask;    // protected-column bits per 32-column group
    const int *pu;            // protected columns before each group
    const float *pscale;      // scale of each protected column
    float *xs;                // [B][cap] scale * x of each protected column
    const int *pidx;          // the protected columns (absolute indices)
    int np;                   // how many
};

// Activation staging for the input columns [k_begin, k_begin + cols) of G
// layers that share x: bf16 rows from global memory -> fp16 in the permuted
// fragment order [512-column slab][w][m][t][4 pairs], converted once, then
// stored per layer with that layer's protected columns zeroed; then
// scale_u * x[b][j_u] of the protected columns (exact in fp32: 11 x 8
// significant bits) in a flat second loop, whose loads are all independent
// (gathering them inside the first loop put a dependent round trip on every
// job with a protected column: 7 us of a 17.6 us launch at batch 16).
// Job = one 32-column group of one row.  Pair i of a
// 32-column group is element i&7 of chunk (i>>3) and of chunk (i>>3)+2 --
// bits i and i+16 of its code word, columns (i>>3)*8 + (i&7) and that + 16.
template <int MAXG, bool kHalfXs = false, int kBatch = 1>
__device__ __forceinline__ void stage_activations(const uint16_t *x, int K, int B, int k_begin,
                                                  int cols, int nnar, int xt_pitch, int cap,
                                                  int G, const StageView (&v)[MAXG]) {
    const int groups_per_row = cols >> 5;   // cols % 128 == 0 on this path
    const int njobs = B * nnar * 16;
    const int nthr = static_cast<int>(blockDim.x);
    // kBatch jobs per thread have their loads in flight together (one round
    // trip to memory per batch; more than one job per batch measured no
    // faster at batch 8..16)
    for (int e0 = threadIdx.x; e0 < njobs; e0 += kBatch * nthr) {
        uint32_t rr[kBatch][16];
#pragma unroll
        for (int i = 0; i < kBatch; ++i) {
            const int e = e0 + i * nthr;
            const int t = e & 3, w = (e >> 2) & 3, sb = e >> 4;
            const int b = sb / nnar, slab = sb - b * nnar;
            const int g32 = slab * 16 + t * 4 + w;
            if (e < njobs && g32 < groups_per_row) {
                const uint16_t *src = x + static_cast<int64_t>(b) * K + k_begin + g32 * 32;
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    const uint4 u4 = reinterpret_cast<const uint4 *>(src)[q];
                    rr[i][4 * q] = u4.x; rr[i][4 * q + 1] = u4.y; rr[i][4 * q + 2] = u4.z; rr[i][4 * q + 3] = u4.w;
                }
            } else {
#pragma unroll
                for (int q = 0; q < 16; ++q) rr[i][q] = 0u;
            }
        }
#pragma unroll
        for (int i = 0; i < kBatch; ++i) {
            const int e = e0 + i * nthr;
            if (e >= njobs) break;
            const int t = e & 3, w = (e >> 2) & 3, sb = e >> 4;
            const int b = sb / nnar, slab = sb - b * nnar;
            const int g32 = slab * 16 + t * 4 + w;
            const int dst_off = b * xt_pitch + slab * 1024 + t * 16 + w * 256;
            uint32_t o[16];
#pragma unroll
            for (int j = 0; j < 16; ++j) {
                // pair j: columns c0 = (j>>3)*8 + (j&7) (low half) and c0 + 16
                const int c0 = (j >> 3) * 8 + (j & 7);
                const uint32_t f = rr[i][c0 >> 1], sw = rr[i][(c0 + 16) >> 1];
                const __half2 h = __floats2half2_rn((c0 & 1) ? bf16_hi(f) : bf16_lo(f),
                                                    (c0 & 1) ? bf16_hi(sw) : bf16_lo(sw));
                o[j] = *reinterpret_cast<const uint32_t *>(&h);
            }
#pragma unroll
            for (int g = 0; g < MAXG; ++g) {
                if (g >= G) break;
                uint32_t pm = g32 < groups_per_row ? v[g].pmask[g32] : 0u;
                unsigned char *dst = v[g].xt + dst_off;
                if (pm == 0u) {
#pragma unroll
                    for (int m = 0; m < 4; ++m)
                        *reinterpret_cast<uint4 *>(dst + m * 64) =
                            make_uint4(o[4 * m], o[4 * m + 1], o[4 * m + 2], o[4 * m + 3]);
                    continue;
                }
                // protected columns of this group: zero their halves
                uint32_t om[16];
#pragma unroll
                for (int j = 0; j < 16; ++j) {
                    const int c0 = (j >> 3) * 8 + (j & 7);
                    const uint32_t keep = (((pm >> c0) & 1u) ? 0u : 0x0000FFFFu) |
                                          (((pm >> (c0 + 16)) & 1u) ? 0u : 0xFFFF0000u);
                    om[j] = o[j] & keep;
                }
#pragma unroll
                for (int m = 0; m < 4; ++m)
                    *reinterpret_cast<uint4 *>(dst + m * 64) =
                        make_uint4(om[4 * m], om[4 * m + 1], om[4 * m + 2], om[4 * m + 3]);
            }
        }
    }
    // scale * x of every protected column of every layer and row
#pragma unroll
    for (int g = 0; g < MAXG; ++g) {
        if (g >= G) break;
        const int np = v[g].np;
        for (int e = threadIdx.x; e < B * np; e += nthr) {
            const int b = e / np, u = e - b * np;
            const float sx = v[g].pscale[u] * bf16_bits_to_f32(x[static_cast<int64_t>(b) * K + v[g].pidx[u]]);
            if constexpr (kHalfXs) {
                __half *xh = reinterpret_cast<__half *>(v[g].xs);
                const __half hi = __float2half_rn(sx);
                xh[b * cap + u] = hi;
                xh[(B + b) * cap + u] = __float2half_rn(sx - __half2float(hi));
            } else {
                v[g].xs[b * cap + u] = sx;
            }
        }
    }
}

// One ring slot's share of one consumer warp: rows lo/hi of column quarter
// q (512 columns) for all S stages, accumulated into four MMA chains.
template <int S, int BM, int kCodeRow, int kNormRow, bool kSwz, int NT>
__device__ __forceinline__ void decode_slot(const unsigned char *cs, const unsigned char *ns,
                                            int q, int rlo, int rhi, int t,
                                            const unsigned char *const (&xr)[NT],
                                            float (&acc)[4][NT][4]) {
    // stages one after another: keeps one stage's codes and norms live
#pragma unroll 1
    for (int s = 0; s < S; ++s) {
        const uint4 clo = *reinterpret_cast<const uint4 *>(cs + (s * BM + rlo) * kCodeRow + q * 64 + t * 16);
        const uint4 chi = *reinterpret_cast<const uint4 *>(cs + (s * BM + rhi) * kCodeRow + q * 64 + t * 16);
        const unsigned char *nlo = ns + (s * BM + rlo) * kNormRow + q * 128;
        const unsigned char *nhi = ns + (s * BM + rhi) * kNormRow + q * 128;
        const int sl = kSwz ? (rlo & 7) : 0, sh = kSwz ? (rhi & 7) : 0;
        const uint4 nl0 = *reinterpret_cast<const uint4 *>(nlo + (((2 * t) ^ sl) << 4));
        const uint4 nl1 = *reinterpret_cast<const uint4 *>(nlo + (((2 * t + 1) ^ sl) << 4));
        const uint4 nh0 = *reinterpret_cast<const uint4 *>(nhi + (((2 * t) ^ sh) << 4));
        const uint4 nh1 = *reinterpret_cast<const uint4 *>(nhi + (((2 * t + 1) ^ sh) << 4));
#pragma unroll
        for (int w = 0; w < 4; ++w) {
            const uint32_t cl = word_of(clo, w), ch = word_of(chi, w);
            const uint32_t la = word_of(w < 2 ? nl0 : nl1, (2 * w) & 3);
            const uint32_t lb = word_of(w < 2 ? nl0 : nl1, (2 * w + 1) & 3);
            const uint32_t ha = word_of(w < 2 ? nh0 : nh1, (2 * w) & 3);
            const uint32_t hb = word_of(w < 2 ? nh0 : nh1, (2 * w + 1) & 3);
            // norm pairs (n_c, n_{c+2}) for chunks 0/2 and 1/3 of the word
            const uint32_t np0l = prmt(la, lb, 0x5410), np1l = prmt(la, lb, 0x7632);
            const uint32_t np0h = prmt(ha, hb, 0x5410), np1h = prmt(ha, hb, 0x7632);
#pragma unroll
            for (int m = 0; m < 4; ++m) {
                uint4 xf[NT];
#pragma unroll
                for (int nt = 0; nt < NT; ++nt)
                    xf[nt] = *reinterpret_cast<const uint4 *>(xr[nt] + (w * 4 + m) * 64);
                // k tiles 2m, 2m+1: pairs 4m..4m+3 of the word
                uint32_t af[2][4];
                decode_pairs(4 * m, cl, ch, m < 2 ? np0l : np1l, m < 2 ? np0h : np1h, af[0]);
                decode_pairs(4 * m + 2, cl, ch, m < 2 ? np0l : np1l, m < 2 ? np0h : np1h, af[1]);
#pragma unroll
                for (int nt = 0; nt < NT; ++nt) {
                    mma_16816(acc[(w & 1) * 2][nt], af[0], xf[nt].x, xf[nt].y);
                    mma_16816(acc[(w & 1) * 2 + 1][nt], af[1], xf[nt].z, xf[nt].w);
                }
            }
        }
    }
}

// Protected k tile u16..u16+15 for rows lo/hi (Eq. 10): q8 bytes from the
// int8 slab in shared memory (column col0 + u; box-major [box][BM][128]
// storage, or rows of q8_pitch bytes when q8_pitch > 0) as exact fp16
// integers against scale * x (s_xs) split into fp16 hi + lo.
template <int BM, int NT>
__device__ __forceinline__ void protected_tile(const int8_t *q8s, int col0, int u16, int p_loc,
                                               int rlo, int rhi, int g, int t, const float *s_xs,
                                               int xs_pitch, int B, float (&accp)[NT][4],
                                               int q8_pitch = 0) {
    auto q8v = [&](int r, int u) -> float {
        if (u >= p_loc) return 0.f;
        const int col = col0 + u;
        return static_cast<float>(q8_pitch > 0 ? q8s[r * q8_pitch + col]
                                               : q8s[((col >> 7) * BM + r) * 128 + (col & 127)]);
    };
    const int u0 = u16 + 2 * t;
    uint32_t af[4];
    const int uu[4] = {u0, u0, u0 + 8, u0 + 8};
#pragma unroll
    for (int e = 0; e < 4; ++e) {
        const int r = (e & 1) ? rhi : rlo;
        const __half2 h = __floats2half2_rn(q8v(r, uu[e]), q8v(r, uu[e] + 1));
        af[e] = *reinterpret_cast<const uint32_t *>(&h);
    }
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) {
        const int bg = nt * 8 + g;
        uint32_t hi[2] = {0u, 0u}, lo[2] = {0u, 0u};
        if (bg < B) {
#pragma unroll
            for (int h = 0; h < 2; ++h) {
                const int u = u0 + 8 * h;
                const float v0 = u < p_loc ? s_xs[bg * xs_pitch + u] : 0.f;
                const float v1 = u + 1 < p_loc ? s_xs[bg * xs_pitch + u + 1] : 0.f;
                const __half2 vh = __floats2half2_rn(v0, v1);
                const float2 back = __half22float2(vh);
                const __half2 vl = __floats2half2_rn(v0 - back.x, v1 - back.y);
                hi[h] = *reinterpret_cast<const uint32_t *>(&vh);
                lo[h] = *reinterpret_cast<const uint32_t *>(&vl);
            }
        }
        mma_16816(accp[nt], af, hi[0], hi[1]);
        mma_16816(accp[nt], af, lo[0], lo[1]);
    }
}

// Protected k tile u16..u16+15 of rows g and g + 8 (Eq. 10), batch columns
// nt * 8 + g of the MMA n-tiles: q8 from a tile slab of rows of `pitch`
// bytes (16-bit loads of column pairs, exact int8 -> fp16), scale * x as fp16
// hi + lo halves xsh/xsl [B][cap], zero past the layer's p, so no bounds
// checks.
template <int NT>
__device__ __forceinline__ void protected_rows(const int8_t *q8s, int pitch, int u16, int g, int t,
                                               const __half *xsh, const __half *xsl, int cap, int B,
                                               float (&acc)[NT][4]) {
    const int u0 = u16 + 2 * t;
    auto pair = [&](int r, int u) {
        return i8x2_to_h2(*reinterpret_cast<const uint16_t *>(q8s + r * pitch + u));
    };
    const uint32_t af[4] = {pair(g, u0), pair(g + 8, u0), pair(g, u0 + 8), pair(g + 8, u0 + 8)};
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) {
        const int bg = nt * 8 + g;
        uint32_t h0 = 0u, h1 = 0u, l0 = 0u, l1 = 0u;
        if (bg < B) {
            h0 = *reinterpret_cast<const uint32_t *>(xsh + bg * cap + u0);
            h1 = *reinterpret_cast<const uint32_t *>(xsh + bg * cap + u0 + 8);
            l0 = *reinterpret_cast<const uint32_t *>(xsl + bg * cap + u0);
            l1 = *reinterpret_cast<const uint32_t *>(xsl + bg * cap + u0 + 8);
        }
        mma_16816(acc[nt], af, h0, h1);
        mma_16816(acc[nt], af, l0, l1);
    }
}

// Protected-column bookkeeping of one CTA (warp 0): indices in [k_begin,
// k_end) (prot_idx is ascending), their scales, a bit mask over the CTA's
// 32-column groups and the number of protected columns before each group.
// Returns the index range [lo, hi) in prot_idx via s_lohi.
__device__ __forceinline__ void stage_protected_meta(const GemvArgs &a, int k_begin, int k_end,
                                                     int mwords, int *s_pidx, float *s_pscale,
                                                     uint32_t *s_pmask, int *s_pu, int *s_lohi) {
    const int lane = threadIdx.x & 31;
    for (int i = lane; i < mwords; i += 32) s_pmask[i] = 0u;
    int lo = 0, hi = a.p;
    if (k_begin > 0 || k_end < a.K) {
        // position of [k_begin, k_end) in the ascending list; four loads in
        // flight per lane
        hi = 0;
        for (int t0 = 0; t0 < a.p; t0 += 128) {
            int v[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const int t = t0 + 32 * i + lane;
                v[i] = t < a.p ? a.prot_idx[t] : 0x7FFFFFFF;
            }
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                lo += __popc(__ballot_sync(0xFFFFFFFFu, v[i] < k_begin));
                hi += __popc(__ballot_sync(0xFFFFFFFFu, v[i] < k_end));
            }
        }
    }
    __syncwarp();
    // an ascending index list puts at most pidx_cap entries in [k_begin,
    // k_end); anything else is not a valid layer and is reported, not used
    if (hi - lo > a.pidx_cap) {
        if (lane == 0) latch_error(a.err, BISCO_ERR_INVALID_ARG);
        hi = lo + a.pidx_cap;
    }
#pragma unroll 4
    for (int u = lane; u < hi - lo; u += 32) {
        const int j = a.prot_idx[lo + u];
        const bool in_range = j >= k_begin && j < k_end;
        if (!in_range) latch_error(a.err, BISCO_ERR_INVALID_ARG);
        s_pidx[u] = in_range ? j : k_begin;
        s_pscale[u] = in_range ? __half2float(__ushort_as_half(a.q8_scale[lo + u])) : 0.f;
        if (in_range) atomicOr(&s_pmask[(j - k_begin) >> 5], 1u << ((j - k_begin) & 31));
    }
    __syncwarp();
    int run = 0;
    for (int base = 0; base < mwords; base += 32) {
        const int i = base + lane;
        const int c = i < mwords ? __popc(s_pmask[i]) : 0;
        int incl = c;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int v = __shfl_up_sync(0xFFFFFFFFu, incl, o);
            if (lane >= o) incl += v;
        }
        if (i < mwords) s_pu[i] = run + incl - c;
        run += __shfl_sync(0xFFFFFFFFu, incl, 31);
    }
    if (lane == 0) {
        s_lohi[0] = lo;
        s_lohi[1] = hi;
    }
}

// ------------------------------------------------------------------------
// Clustered kernel: BM = 16*WM rows x one K range per CTA.
template <int WM, int WQ, int NT, int S>
__global__ void __launch_bounds__((WM * WQ + 1) * 32, (NT == 1 && (WM * WQ + 1) * 32 <= 320) ? 2 : 1)
k_gemv(const __grid_constant__ CUtensorMap tm_codes, const __grid_constant__ CUtensorMap tm_norms,
       const __grid_constant__ CUtensorMap tm_q8, const GemvArgs a) {
    constexpr int BM = 16 * WM;
    constexpr int BP = 8 * NT;
    constexpr int NCW = WM * WQ;             // consumer warps; warp NCW is the producer
    constexpr int SW = kSlab * WQ;           // columns per ring slot
    constexpr int kCodeRow = SW / 8;
    constexpr int kNormRow = SW / 4;
    constexpr bool kSwz = (WQ == 1);         // 128-byte swizzle when a norm row is 128 B
    constexpr uint32_t kCodesBytes = S * BM * kCodeRow;
    constexpr uint32_t kSlotBytes = S * BM * (kCodeRow + kNormRow);

    extern __shared__ unsigned char smem_raw[];
    unsigned char *sm = aligned_smem(smem_raw);
    const uint32_t sbase = smem_u32(sm);
    __shared__ int s_abort, s_lohi[2];

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int rank = static_cast<int>(cluster_ctarank());
    const int nrank = static_cast<int>(cluster_nctarank());
    const int row0 = blockIdx.y * BM;
    const int k_begin = min(a.K, rank * a.wide_per_rank * SW);
    const int k_end = min(a.K, k_begin + a.wide_per_rank * SW);
    const int nwide = (k_end - k_begin + SW - 1) / SW;
    const int nnar = (k_end - k_begin + kSlab - 1) / kSlab;
    const int nslot = a.nslot;
    const uint32_t bar_full = sbase + a.off_bar;
    const uint32_t bar_empty = bar_full + 8 * nslot;
    const uint32_t bar_q8 = bar_full + 16 * nslot;
    const uint32_t bar_cl = bar_q8 + 8;
    const bool producer = (warp == NCW) && (lane == 0);
    const uint64_t pol = l2_evict_first_policy();
    int *s_pidx = reinterpret_cast<int *>(sm + a.off_pidx);
    float *s_pscale = reinterpret_cast<float *>(s_pidx + a.pidx_cap);
    float *s_xs = s_pscale + a.pidx_cap;
    uint32_t *s_pmask = reinterpret_cast<uint32_t *>(sm + a.off_pmask);
    int *s_pu = reinterpret_cast<int *>(sm + a.off_pu);

    int issued = 0;
    if (producer) {
        for (int i = 0; i < nslot; ++i) {
            mbar_init(bar_full + 8 * i, 1);
            mbar_init(bar_empty + 8 * i, NCW);
        }
        mbar_init(bar_q8, 1);
        mbar_init(bar_cl, nrank > 1 ? (nrank - 1) * blockDim.x : 1);
        fence_mbar_init();
        s_abort = 0;
        prefetch_tmap(&tm_codes);
        prefetch_tmap(&tm_norms);
        for (; issued < nwide && issued < nslot; ++issued) {
            const uint32_t dst = sbase + issued * kSlotBytes;
            mbar_arrive_expect_tx(bar_full + 8 * issued, kSlotBytes);
            const int kx = (k_begin + issued * SW) / 8;
            tma_load_3d_hint(dst, &tm_codes, bar_full + 8 * issued, kx, row0, 0, pol);
            tma_load_3d_hint(dst + kCodesBytes, &tm_norms, bar_full + 8 * issued, kx, row0, 0, pol);
        }
    }
    if (warp == 0)
        stage_protected_meta(a, k_begin, k_end, nnar * (kSlab / 32), s_pidx, s_pscale, s_pmask,
                             s_pu, s_lohi);
    if (producer && k_end > k_begin) {
        for (int b = 0; b < a.B; ++b)
            prefetch_l2(a.x + static_cast<int64_t>(b) * a.K + k_begin,
                        static_cast<uint32_t>(k_end - k_begin) * 2);
    }
    __syncthreads();
    // the next kernel in the stream may start streaming its own weights now
    pdl_launch_dependents();
    // rank 0's reduction barrier is initialised before any rank arrives on
    // it: arrive here, wait just before the hand-over at the end
    if (nrank > 1) cluster_arrive();
    const int lo_t = s_lohi[0], p_loc = s_lohi[1] - s_lohi[0];
    const int q8x0 = lo_t & ~15;   // 16-byte aligned TMA start
    const int q8_boxes = p_loc > 0 ? (lo_t + p_loc - q8x0 + 127) >> 7 : 0;
    if (producer && q8_boxes > 0) {
        mbar_arrive_expect_tx(bar_q8, static_cast<uint32_t>(q8_boxes * BM * 128));
        for (int q = 0; q < q8_boxes; ++q)
            tma_load_2d_hint(sbase + a.off_q8 + q * BM * 128, &tm_q8, bar_q8, q8x0 + 128 * q, row0,
                             pol);
    }

    // activations may be written by the previous kernel
    pdl_wait();
    {
        StageView v[1] = {{sm + a.off_xt, s_pmask, s_pu, s_pscale, s_xs, s_pidx, p_loc}};
        stage_activations<1>(a.x, a.K, a.B, k_begin, k_end - k_begin, nnar, a.xt_pitch, a.pidx_cap,
                             1, v);
    }
    for (int i = threadIdx.x; i < 1024 / 16; i += blockDim.x)
        reinterpret_cast<uint4 *>(sm + a.off_zero)[i] = make_uint4(0, 0, 0, 0);
    __syncthreads();

    float *red = reinterpret_cast<float *>(sm + a.off_red);

    if (warp == NCW) {
        // ------------------------------------------------ producer: refill
        if (producer) {
            for (; issued < nwide; ++issued) {
                const int slot = issued % nslot;
                if (!mbar_wait(bar_empty + 8 * slot, ((issued / nslot) - 1) & 1)) {
                    latch_error(a.err, BISCO_ERR_TIMEOUT);
                    atomicExch(&s_abort, 1);
                    break;
                }
                if (*reinterpret_cast<volatile int *>(&s_abort)) break;
                const uint32_t dst = sbase + slot * kSlotBytes;
                mbar_arrive_expect_tx(bar_full + 8 * slot, kSlotBytes);
                const int kx = (k_begin + issued * SW) / 8;
                tma_load_3d_hint(dst, &tm_codes, bar_full + 8 * slot, kx, row0, 0, pol);
                tma_load_3d_hint(dst + kCodesBytes, &tm_norms, bar_full + 8 * slot, kx, row0, 0, pol);
            }
            if (*reinterpret_cast<volatile int *>(&s_abort)) {
                // let every copy already in flight land before the CTA exits
                for (int slot = 0; slot < nslot && slot < issued; ++slot) {
                    const int last = slot + ((issued - 1 - slot) / nslot) * nslot;
                    mbar_wait(bar_full + 8 * slot, (last / nslot) & 1);
                }
                if (q8_boxes > 0) mbar_wait(bar_q8, 0);
            }
        }
    } else {
        // ----------------------------------------------- consumers: decode
        // warp (wm, q) owns rows 16*wm.. and column quarter q of every slot
        const int wm = warp % WM, q = warp / WM;
        const int g = lane >> 2, t = lane & 3;
        const int rlo = 16 * wm + g, rhi = rlo + 8;
        const unsigned char *xb[NT];
        int xstep[NT];
#pragma unroll
        for (int nt = 0; nt < NT; ++nt) {
            const int bg = nt * 8 + g;
            xb[nt] = bg < a.B ? sm + a.off_xt + bg * a.xt_pitch + t * 16 : sm + a.off_zero + t * 16;
            xstep[nt] = bg < a.B ? 1024 : 0;
        }
        float acc[4][NT][4];
#pragma unroll
        for (int c = 0; c < 4; ++c)
#pragma unroll
            for (int nt = 0; nt < NT; ++nt)
#pragma unroll
                for (int k = 0; k < 4; ++k) acc[c][nt][k] = 0.f;

        for (int it = 0; it < nwide; ++it) {
            const int slot = it % nslot;
            if (*reinterpret_cast<volatile int *>(&s_abort)) break;
            if (!mbar_wait(bar_full + 8 * slot, (it / nslot) & 1)) {
                latch_error(a.err, BISCO_ERR_TIMEOUT);
                atomicExch(&s_abort, 1);
                break;
            }
            const int nar = it * WQ + q;   // this warp's 512-column slab
            if (nar < nnar) {
                const unsigned char *cs = sm + slot * kSlotBytes;
                const unsigned char *xr[NT];
#pragma unroll
                for (int nt = 0; nt < NT; ++nt) xr[nt] = xb[nt] + nar * xstep[nt];
                decode_slot<S, BM, kCodeRow, kNormRow, kSwz, NT>(cs, cs + kCodesBytes, q, rlo, rhi, t,
                                                                 xr, acc);
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(bar_empty + 8 * slot);
        }

        // protected columns: k tiles of a row group shared out over its WQ warps
        float accp[NT][4];
#pragma unroll
        for (int nt = 0; nt < NT; ++nt)
#pragma unroll
            for (int k = 0; k < 4; ++k) accp[nt][k] = 0.f;
        if (q8_boxes > 0 && q * 16 < p_loc) {
            if (!mbar_wait(bar_q8, 0)) {
                latch_error(a.err, BISCO_ERR_TIMEOUT);
                atomicExch(&s_abort, 1);
            } else {
                for (int u16 = 16 * q; u16 < p_loc; u16 += 16 * WQ)
                    protected_tile<BM, NT>(reinterpret_cast<const int8_t *>(sm + a.off_q8),
                                           lo_t - q8x0, u16, p_loc, rlo, rhi, g, t, s_xs,
                                           a.pidx_cap, a.B, accp);
            }
        }
#pragma unroll
        for (int nt = 0; nt < NT; ++nt)
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                const int r = k < 2 ? rlo : rhi;
                const int b = nt * 8 + 2 * t + (k & 1);
                const float sum = (acc[0][nt][k] + acc[1][nt][k]) + (acc[2][nt][k] + acc[3][nt][k]);
                red[(q * BM + r) * BP + b] = sum * kInvSqrt8 + accp[nt][k];
            }
    }

    __syncthreads();
    // this CTA's partial for each (row, batch): column quarters in order
    if (WQ > 1) {
        for (int e = threadIdx.x; e < BM * BP; e += blockDim.x) {
            float v = red[e];
#pragma unroll
            for (int qq = 1; qq < WQ; ++qq) v += red[qq * BM * BP + e];
            red[e] = v;
        }
        __syncthreads();
    }
    if (nrank == 1) {
        for (int e = threadIdx.x; e < a.B * BM; e += blockDim.x) {
            const int b = e / BM, r = e - b * BM;
            if (row0 + r < a.N) a.y[static_cast<int64_t>(b) * a.N + row0 + r] = red[r * BP + b];
        }
        return;
    }
    cluster_wait();
    if (rank != 0) {
        // hand the partial to rank 0; every thread releases its own stores
        const uint32_t dst = mapa_shared(sbase + a.off_cl + (rank - 1) * BM * BP * 4, 0);
        for (int e = threadIdx.x; e < BM * BP; e += blockDim.x) st_shared_cluster_f32(dst + e * 4, red[e]);
        mbar_arrive_cluster(mapa_shared(bar_cl, 0));
        return;
    }
    if (!mbar_wait_cluster(bar_cl, 0)) {
        latch_error(a.err, BISCO_ERR_TIMEOUT);
        return;
    }
    const float *cl = reinterpret_cast<const float *>(sm + a.off_cl);
    for (int e = threadIdx.x; e < a.B * BM; e += blockDim.x) {
        const int b = e / BM, r = e - b * BM;
        float v = red[r * BP + b];
        for (int qq = 1; qq < nrank; ++qq) v += cl[((qq - 1) * BM + r) * BP + b];
        if (row0 + r < a.N) a.y[static_cast<int64_t>(b) * a.N + row0 + r] = v;
    }
}

// ------------------------------------------------------------------------
// Streaming kernel: persistent CTA over 16-row tiles x all K of G <= 4 layers
// that share the activations (G = 1 for a plain bisco_gemv), batch <= 8.
// Warp (q, k) decodes column quarter q of every slot whose global index is
// k modulo WK; warp NCW produces; warp NCW+1 reduces.  A slot's full
// barrier is split into WK barriers taken in turn by its fills, so that a
// consumer group always waits on a barrier whose previous phase it observed
// itself, whatever the ring depth.

// ------------------------------------------------------------------------
// Table-lookup decode for a single activation row (batch 1).
//
// Per sign byte b of chunk c, Eq. 12's inner product sum_e s_e x[8c+e] is
// the sum of two signed sums of four activations, one per half of the byte.
// The tables hold them for every chunk and every v = 0..15:
//   T_lo(c, v) = sum_{e<4} (bit e of v ? -x[8c+e] : +x[8c+e])
//   T_hi(c, v) = the same over x[8c+4+e]
// as one fp16 pair (T_lo low, T_hi high) per 32-bit word.  A chunk-stage
// then costs two shared-memory lookups, T_lo(c, b & 15) and T_hi(c, b >> 4),
// and two fp16 x fp16 -> fp32 FMAs with its norm, instead of decoding eight
// signs.  Rounding T to fp16 is this path's one approximation (relative
// 2^-11 of each half sum).
//
// Placement: chunk c sits at position P, where within each group of 128
// chunks chunk 4l + j is at 32j + l, and entry (P, v) is at byte
//   (P >> 6) * 4096 + v * 256 + (P & 63) * 4.
// Lane l reading chunk 4l + j of its code word thus hits bank l, and the
// address is one byte permute: byte 0 the lane's slot (P & 63) * 4, byte 1
// the nibble with (P >> 6) & 15 above it, byte 2 (P >> 6) >> 4.
constexpr int kLutSlotCols = 2048;                    // ring slot width the placement assumes
constexpr int kLutSlotBytes = kLutSlotCols / 8 * 64;  // table bytes per slot of columns

// Tables of x[0, K) for nchunk chunk positions (a multiple of 128; chunks at
// or past K/8 get zero tables, so a ragged last slot reads zeros).  With a
// protected-column mask (a bit per column, 32 per word) those columns count
// as zero, which is Eq. 10's overwrite for a launch of one layer.
__device__ __forceinline__ void build_nibble_tables(const uint16_t *x, int K, int nchunk,
                                                    const uint32_t *pmask, unsigned char *tab) {
    // a warp's jobs go in batches whose loads are all issued before any
    // table is written: one round trip to memory per batch (one in all for
    // K up to 2 * 32 * 8 * warps columns; larger batches measured slower on
    // the short layers)
    constexpr int kBatch = 2;
    const int lane = threadIdx.x & 31, nwarp = static_cast<int>(blockDim.x >> 5);
    const int njobs = nchunk / 32;
    for (int J0 = static_cast<int>(threadIdx.x >> 5); J0 < njobs; J0 += kBatch * nwarp) {
        uint4 u[kBatch];
        uint32_t m[kBatch];
#pragma unroll
        for (int i = 0; i < kBatch; ++i) {
            const int J = J0 + i * nwarp;
            const int c = (J >> 2) * 128 + 4 * lane + (J & 3);
            u[i] = make_uint4(0u, 0u, 0u, 0u);
            m[i] = 0u;
            if (J < njobs && 8 * c < K) {
                u[i] = *reinterpret_cast<const uint4 *>(x + 8 * c);
                if (pmask != nullptr) m[i] = (pmask[c >> 2] >> ((c & 3) * 8)) & 0xFFu;
            }
        }
#pragma unroll
        for (int i = 0; i < kBatch; ++i) {
            const int J = J0 + i * nwarp;
            if (J >= njobs) break;
            const int P = (J >> 2) * 128 + 32 * (J & 3) + lane;
            float e[8] = {bf16_lo(u[i].x), bf16_hi(u[i].x), bf16_lo(u[i].y), bf16_hi(u[i].y),
                          bf16_lo(u[i].z), bf16_hi(u[i].z), bf16_lo(u[i].w), bf16_hi(u[i].w)};
#pragma unroll
            for (int k = 0; k < 8; ++k)
                if ((m[i] >> k) & 1u) e[k] = 0.f;
            // signed sums of element pairs: index bit 0 negates the first, bit 1 the second
            float a[2][4], d[2][4];
#pragma unroll
            for (int h = 0; h < 2; ++h) {
                const float x0 = e[4 * h], x1 = e[4 * h + 1], x2 = e[4 * h + 2], x3 = e[4 * h + 3];
                a[h][0] = x0 + x1; a[h][1] = x1 - x0; a[h][2] = x0 - x1; a[h][3] = -(x0 + x1);
                d[h][0] = x2 + x3; d[h][1] = x3 - x2; d[h][2] = x2 - x3; d[h][3] = -(x2 + x3);
            }
            unsigned char *dst = tab + (P >> 6) * 4096 + (P & 63) * 4;
#pragma unroll
            for (int v = 0; v < 16; ++v) {
                const __half2 t = __floats2half2_rn(a[0][v & 3] + d[0][v >> 2], a[1][v & 3] + d[1][v >> 2]);
                *reinterpret_cast<__half2 *>(dst + v * 256) = t;
            }
        }
    }
}

// One ring slot (2048 columns, slot index w along K) for rows row0..row0+R-1
// and all S stages: lane l takes code words l and 32 + l of each row, i.e.
// chunks 4(32m + l) + j at table positions 256w + 128m + 32j + l.
template <int S, int R, int kCodeRow, int kNormRow>
__device__ __forceinline__ void lut_slot(uint32_t cs, uint32_t ns, uint32_t tab, int w, int row0,
                                         int lane, float (&acc)[R]) {
    uint32_t sgpat[2], base[2][4];
#pragma unroll
    for (int m = 0; m < 2; ++m) {
        // 64-position table blocks of chunks j = 0, 1 and j = 2, 3 of word m
        const uint32_t g0 = 4u * static_cast<uint32_t>(w) + 2u * m, g1 = g0 + 1u;
        sgpat[m] = (g0 & 15u) * 0x1010u | (g1 & 15u) * 0x10100000u;
#pragma unroll
        for (int j = 0; j < 4; ++j)
            base[m][j] = static_cast<uint32_t>(lane) * 4u + (j & 1) * 128u + (((j < 2 ? g0 : g1) >> 4) << 16);
    }
    // every code and norm word of the slot first, so that no lookup waits
    // behind another stage's or row's code load
    uint32_t cw[S][R][2];
    uint2 nw[S][R][2];
#pragma unroll
    for (int s = 0; s < S; ++s)
#pragma unroll
        for (int r = 0; r < R; ++r) {
            const uint32_t crow = cs + (s * 16 + row0 + r) * kCodeRow + lane * 4;
            const uint32_t nrow = ns + (s * 16 + row0 + r) * kNormRow + lane * 8;
#pragma unroll
            for (int m = 0; m < 2; ++m) {
                cw[s][r][m] = lds_u32(crow + m * 128);
                nw[s][r][m] = lds_u64(nrow + m * 256);
            }
        }
#pragma unroll
    for (int s = 0; s < S; ++s)
#pragma unroll
        for (int r = 0; r < R; ++r)
#pragma unroll
            for (int m = 0; m < 2; ++m) {
                const uint32_t wl = lop3_and_or(cw[s][r][m], 0x0F0F0F0Fu, sgpat[m]);
                const uint32_t wh = lop3_and_or(cw[s][r][m] >> 4, 0x0F0F0F0Fu, sgpat[m]);
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    const uint32_t sel = 0x7604u | (static_cast<uint32_t>(j) << 4);
                    const uint32_t tl = lds_u32(tab + prmt(wl, base[m][j], sel));
                    const uint32_t th = lds_u32(tab + prmt(wh, base[m][j], sel));
                    const uint32_t nj = j < 2 ? nw[s][r][m].x : nw[s][r][m].y;
                    const uint16_t n = (j & 1) ? hi_half(nj) : lo_half(nj);
                    acc[r] = fma_f16_f32(lo_half(tl), n, acc[r]);
                    acc[r] = fma_f16_f32(hi_half(th), n, acc[r]);
                }
            }
}

// A launch over several layers shares one set of tables built from x itself,
// so the BSQ terms of a layer's protected columns (Eq. 10 replaces them) are
// removed here: for the protected columns u0..u1 of slot w, acc[r] of row
// row0 + r loses sum_s (+-n_s) * x_j.  One column per lane (all R rows and S
// stages loaded at once); the warp sum of acc[r] then carries the total.
template <int S, int R, int kCodeRow, int kNormRow>
__device__ __forceinline__ void lut_protected(const unsigned char *cs, const unsigned char *ns,
                                              int w, int row0, int lane, const int *pidx,
                                              const float *xj, int u0, int u1, float (&acc)[R]) {
    for (int u = u0 + lane; u < u1; u += 32) {
        const int jc = pidx[u] - w * kLutSlotCols;   // column within the slot
        if (jc < 0 || jc >= kLutSlotCols) continue;   // only for a list that is not ascending
        const int ch = jc >> 3, e = jc & 7;
        const float xv = xj[u];
        uint32_t b[R][S];
        uint16_t n[R][S];
#pragma unroll
        for (int r = 0; r < R; ++r)
#pragma unroll
            for (int s = 0; s < S; ++s) {
                b[r][s] = cs[(s * 16 + row0 + r) * kCodeRow + ch];
                n[r][s] = *reinterpret_cast<const uint16_t *>(ns + (s * 16 + row0 + r) * kNormRow + 2 * ch);
            }
#pragma unroll
        for (int r = 0; r < R; ++r) {
            float sum = 0.f;
#pragma unroll
            for (int s = 0; s < S; ++s) {
                const float v = __half2float(__ushort_as_half(n[r][s]));
                sum += ((b[r][s] >> e) & 1u) ? -v : v;
            }
            acc[r] = fmaf(-sum, xv, acc[r]);
        }
    }
}

// Sum of acc[r] over the warp's 32 lanes for r = 0, 1: afterwards every lane
// holds the total of row bit4(lane).
__device__ __forceinline__ float reduce_rows2(const float (&acc)[2], int lane) {
    const bool h16 = (lane & 16) != 0;
    float k = h16 ? acc[1] : acc[0];
    k += __shfl_xor_sync(0xFFFFFFFFu, h16 ? acc[0] : acc[1], 16);
    k += __shfl_xor_sync(0xFFFFFFFFu, k, 8);
    k += __shfl_xor_sync(0xFFFFFFFFu, k, 4);
    k += __shfl_xor_sync(0xFFFFFFFFu, k, 2);
    k += __shfl_xor_sync(0xFFFFFFFFu, k, 1);
    return k;
}

struct StreamLayer {
    float *y;
    const uint16_t *q8_scale;
    const int32_t *prot_idx;
    int N, p;
    int tile0;       // first tile of this layer in the launch's tile list
    const int8_t *q8;
    int q8_pitch;    // bytes per row of q8 (p rounded up to 16), 0 without protection
};

template <int MAXG>
struct StreamArgs {
    CUtensorMap mc[MAXG], mn[MAXG];
    StreamLayer L[MAXG];
    const uint16_t *x;
    int *err;
    int K, B, G, ntiles, nslot;
    int q8_pitch;    // the largest of the layers' (int8 double buffer size)
    int pidx_cap, xt_pitch, mwords;
    int pblk;        // ints per layer in the protected-column block
    uint32_t off_xt, off_q8, off_red, off_bar, off_pidx, off_pmask, off_zero, off_prot, off_tab;
};

// LUT: batch 1 through the nibble tables (x staged as tables); otherwise the
// MMA decode for batch <= 8 * NT (NT n-tiles of 8 activation rows; at NT = 2
// the staged activations fill most of the shared memory: one CTA per SM).
template <int WQ, int WK, int S, int MAXG, bool LUT, int NT = 1>
__global__ void __launch_bounds__((WQ * WK + 2) * 32, NT == 1 ? 2 : 1)
k_gemv_stream(const __grid_constant__ StreamArgs<MAXG> a) {
    constexpr int BM = 16;
    constexpr int BP = 8 * NT;
    static_assert(!LUT || NT == 1, "the table decode is batch 1");
    constexpr int NCW = WQ * WK;
    constexpr int SW = kSlab * WQ;
    constexpr int kCodeRow = SW / 8;
    constexpr int kNormRow = SW / 4;
    constexpr uint32_t kCodesBytes = S * BM * kCodeRow;
    constexpr uint32_t kSlotBytes = S * BM * (kCodeRow + kNormRow);
    static_assert(!LUT || (SW == kLutSlotCols && NCW == 8), "table decode: 2048-column slots, 8 warps");
    // table decode: every consumer warp takes every slot, two rows each; a
    // launch of one layer masks its protected columns in the tables, a
    // grouped launch shares unmasked tables and corrects per layer
    constexpr int kLutRows = BM / NCW;
    constexpr bool kLutMasked = (MAXG == 1);

    extern __shared__ unsigned char smem_raw[];
    unsigned char *sm = aligned_smem<128>(smem_raw);   // unswizzled boxes only
    const uint32_t sbase = smem_u32(sm);
    __shared__ int s_abort, s_lohi[MAXG][2];
    // layer descriptors, read with a run-time layer index: from shared memory
    // (a run-time index into the parameter block is a slow generic load)
    __shared__ StreamLayer s_L[MAXG];

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int Gd = static_cast<int>(gridDim.x), cta = static_cast<int>(blockIdx.x);
    if (threadIdx.x < MAXG) {
#pragma unroll
        for (int i = 0; i < MAXG; ++i)
            if (static_cast<int>(threadIdx.x) == i) s_L[i] = a.L[i];
    }
    __syncthreads();
    // every scalar the loops use, read once: the tensor maps are addressed
    // with a run-time layer index, after which parameter reads inside loops
    // are not hoisted
    const int K = a.K, B = a.B, G = a.G, xt_pitch = a.xt_pitch, mwords = a.mwords;
    const uint32_t off_xt = a.off_xt, off_q8 = a.off_q8, off_zero = a.off_zero;
    const uint32_t off_pidx = a.off_pidx, off_pmask = a.off_pmask, off_prot = a.off_prot;
    const int pblk = a.pblk;
    const uint16_t *const x = a.x;
    int *const err = a.err;
    int tile0[MAXG];
#pragma unroll
    for (int i = 0; i < MAXG; ++i) tile0[i] = a.L[i].tile0;
    const CUtensorMap *const maps_c = &a.mc[0];
    const CUtensorMap *const maps_n = &a.mn[0];
    const int my_tiles = a.ntiles > cta ? (a.ntiles - 1 - cta) / Gd + 1 : 0;
    const int nwide = (K + SW - 1) / SW;
    const int nnar = (K + kSlab - 1) / kSlab;
    const int total = my_tiles * nwide;   // ring fills of this CTA
    const int nslot = a.nslot;
    const int cap = a.pidx_cap;
    const uint32_t q8_buf_bytes = static_cast<uint32_t>(a.q8_pitch * BM);
    const uint32_t bar_full = sbase + a.off_bar;            // [nslot][WK]
    const uint32_t bar_empty = bar_full + 8 * nslot * WK;   // [nslot]
    const uint32_t bar_q8f = bar_empty + 8 * nslot;         // [2] int8 slab landed
    const uint32_t bar_rf = bar_q8f + 32;                   // [2] tile partials written
    const uint32_t bar_re = bar_rf + 16;                    // [2] tile partials read
    const bool producer = (warp == NCW) && (lane == 0);
    const uint64_t pol = l2_evict_first_policy();
    float *red = reinterpret_cast<float *>(sm + a.off_red);   // [2][NCW][BM][B]

    // per-layer shared-memory views
    // per layer: indices, scales, scale * x [B][cap]; the table decode adds
    // x of each protected column [cap] and the first protected column of
    // every slot [nwide + 1]
    auto pidx_of = [&](int g) { return reinterpret_cast<int *>(sm + off_pidx) + g * pblk; };
    auto pscale_of = [&](int g) { return reinterpret_cast<float *>(pidx_of(g) + cap); };
    auto xs_of = [&](int g) { return pscale_of(g) + cap; };
    auto xj_of = [&](int g) { return xs_of(g) + B * cap; };
    auto su_of = [&](int g) { return reinterpret_cast<int *>(xj_of(g) + cap); };
    auto pmask_of = [&](int g) {
        return reinterpret_cast<uint32_t *>(sm + off_pmask) + g * 2 * mwords;
    };
    auto pu_of = [&](int g) { return reinterpret_cast<int *>(pmask_of(g) + mwords); };
    auto xt_of = [&](int g) { return sm + off_xt + g * B * xt_pitch; };
    // tile ii of this CTA -> (layer, first row)
    auto layer_of = [&](int ii) {
        const int T = cta + ii * Gd;
        int g = 0;
#pragma unroll
        for (int i = 1; i < MAXG; ++i)
            if (i < G && T >= tile0[i]) g = i;
        return g;
    };
    auto row0_of = [&](int ii, int g) { return (cta + ii * Gd - s_L[g].tile0) * BM; };
    auto full_bar = [&](int gidx) {
        const int ph = gidx / nslot;
        return bar_full + 8 * ((gidx % nslot) * WK + ph % WK);
    };
    auto full_parity = [&](int gidx) { return static_cast<uint32_t>((gidx / nslot) / WK) & 1u; };
    // the producer walks its tiles in order: layer and first row of the
    // current tile are kept in registers
    int cur_ii = -1, cur_g = 0, cur_row0 = 0;
    auto issue_slot = [&](int gidx) {
        const int ii = gidx / nwide, w = gidx - ii * nwide;
        if (ii != cur_ii) {
            cur_ii = ii;
            cur_g = layer_of(ii);
            cur_row0 = row0_of(ii, cur_g);
        }
        const uint32_t dst = sbase + (gidx % nslot) * kSlotBytes;
        const uint32_t bar = full_bar(gidx);
        const CUtensorMap *mc = maps_c + cur_g, *mn = maps_n + cur_g;
        mbar_arrive_expect_tx(bar, kSlotBytes);
        tma_load_3d_hint(dst, mc, bar, w * (SW / 8), cur_row0, 0, pol);
        tma_load_3d_hint(dst + kCodesBytes, mn, bar, w * (SW / 8), cur_row0, 0, pol);
    };
    // the int8 slab of tile ii (a plain arrive when its layer has none): the
    // tile's rows of q8 are contiguous, one bulk copy (no tensor map)
    auto issue_q8 = [&](int ii) {
        const int g = layer_of(ii);
        const uint32_t bar = bar_q8f + 8 * (ii & 1);
        const int pitch = s_L[g].q8_pitch;
        if (pitch == 0) {
            mbar_arrive(bar);
            return;
        }
        const int row0 = row0_of(ii, g);
        const int rows = min(BM, s_L[g].N - row0);
        const uint32_t bytes = static_cast<uint32_t>(rows * pitch);
        const uint32_t dst = sbase + off_q8 + (ii & 1) * q8_buf_bytes;
        mbar_arrive_expect_tx(bar, bytes);
        bulk_load(dst, s_L[g].q8 + static_cast<int64_t>(row0) * pitch, bytes, bar);
    };

    int issued = 0;
    if (producer) {
        for (int i = 0; i < nslot; ++i) {
            for (int k = 0; k < WK; ++k) mbar_init(bar_full + 8 * (i * WK + k), 1);
            mbar_init(bar_empty + 8 * i, LUT ? NCW : WQ);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(bar_q8f + 8 * i, 1);
            mbar_init(bar_rf + 8 * i, NCW);
            mbar_init(bar_re + 8 * i, 1);
        }
        fence_mbar_init();
        s_abort = 0;
        for (int g = 0; g < G; ++g) {
            prefetch_tmap(maps_c + g);
            prefetch_tmap(maps_n + g);
        }
        // the first ring fills, then the int8 slabs of the first two tiles
        // (two buffers; the reducer issues the rest as it frees them)
        for (; issued < total && issued < nslot; ++issued) issue_slot(issued);
        for (int t = 0; t < 2 && t < my_tiles; ++t) issue_q8(t);
        // activations: into L2 now, into the CTA after the wait
        for (int b = 0; b < B; ++b)
            prefetch_l2(x + static_cast<int64_t>(b) * K, static_cast<uint32_t>(K) * 2);
    }
    if (warp < G) {
        // one warp per layer: its protected columns, scales and masks
        GemvArgs la = {};
        la.q8_scale = s_L[warp].q8_scale;
        la.prot_idx = s_L[warp].prot_idx;
        la.err = err;
        la.K = K;
        la.p = s_L[warp].p;
        la.pidx_cap = cap;
        stage_protected_meta(la, 0, K, nnar * (kSlab / 32), pidx_of(warp), pscale_of(warp),
                             pmask_of(warp), pu_of(warp), s_lohi[warp]);
        __syncwarp();
        {
            // scale * x halves past the layer's protected count are zero (the
            // protected k tiles run to a multiple of 16); the staging after the
            // wait writes the others
            const int np = s_lohi[warp][1] - s_lohi[warp][0];
            __half *xh = reinterpret_cast<__half *>(xs_of(warp));
            for (int b = 0; b < B; ++b)
                for (int u = np + lane; u < cap; u += 32) {
                    xh[b * cap + u] = __float2half_rn(0.f);
                    xh[(B + b) * cap + u] = __float2half_rn(0.f);
                }
        }
        if constexpr (LUT) {
            // protected columns before each slot (the masks live in the table
            // area until the tables are built)
            __syncwarp();
            const int *pu = pu_of(warp);
            int *su = su_of(warp);
            const int np = s_lohi[warp][1] - s_lohi[warp][0];
            for (int w = lane; w <= nwide; w += 32) su[w] = w < nwide ? pu[w * (kLutSlotCols / 32)] : np;
        }
    }
    __syncthreads();
    pdl_launch_dependents();

    // activations may be written by the previous kernel
    pdl_wait();
    if constexpr (LUT) {
        // protected activations of every layer (flat list over layers), x and
        // scale * x as fp16 hi + lo; the first blockDim.x are loaded before the
        // table build so that both share one round trip to memory
        auto protected_entry = [&](int e, int &g, int &u) {
            for (g = 0; g < G; ++g) {
                const int np = s_lohi[g][1] - s_lohi[g][0];
                if (e < np) {
                    u = e;
                    return true;
                }
                e -= np;
            }
            return false;
        };
        auto store_protected = [&](int g, int u, float xv) {
            const float sx = pscale_of(g)[u] * xv;
            __half *xh = reinterpret_cast<__half *>(xs_of(g));
            const __half hi = __float2half_rn(sx);
            xh[u] = hi;
            xh[cap + u] = __float2half_rn(sx - __half2float(hi));
            xj_of(g)[u] = xv;
        };
        int g0 = 0, u0 = 0;
        const bool has0 = protected_entry(threadIdx.x, g0, u0);
        const float x0 = has0 ? bf16_bits_to_f32(x[pidx_of(g0)[u0]]) : 0.f;
        build_nibble_tables(x, K, nwide * (kLutSlotCols / 8), kLutMasked ? pmask_of(0) : nullptr,
                            sm + a.off_tab);
        if (has0) store_protected(g0, u0, x0);
        for (int e = threadIdx.x + blockDim.x;; e += blockDim.x) {
            int g, u;
            if (!protected_entry(e, g, u)) break;
            store_protected(g, u, bf16_bits_to_f32(x[pidx_of(g)[u]]));
        }
    } else {
        StageView v[MAXG] = {};
#pragma unroll
        for (int g = 0; g < MAXG; ++g)
            if (g < G)
                v[g] = {xt_of(g), pmask_of(g), pu_of(g), pscale_of(g), xs_of(g), pidx_of(g),
                        s_lohi[g][1] - s_lohi[g][0]};
        stage_activations<MAXG, true>(x, K, B, 0, K, nnar, xt_pitch, cap, G, v);
        for (int i = threadIdx.x; i < 1024 / 16; i += blockDim.x)
            reinterpret_cast<uint4 *>(sm + off_zero)[i] = make_uint4(0, 0, 0, 0);
    }
    __syncthreads();

    if (warp == NCW) {
        // ------------------------------------------------ producer: refill
        if (producer) {
            bool ok = true;
            for (; issued < total; ++issued) {
                const int slot = issued % nslot;
                if (!mbar_wait(bar_empty + 8 * slot, ((issued / nslot) - 1) & 1)) {
                    ok = false;
                    break;
                }
                if (*reinterpret_cast<volatile int *>(&s_abort)) break;
                issue_slot(issued);
            }
            if (!ok) {
                latch_error(err, BISCO_ERR_TIMEOUT);
                atomicExch(&s_abort, 1);
            }
            // every copy issued has landed before this thread leaves
            for (int gi = (issued > nslot ? issued - nslot : 0); gi < issued; ++gi)
                mbar_wait(full_bar(gi), full_parity(gi));
        }
    } else if (warp == NCW + 1) {
        // ------------------------------------------- reducer: protected + y
        const int gq = lane >> 2, t = lane & 3;
        const int8_t *q8base = reinterpret_cast<const int8_t *>(sm + off_q8);
        float *prot = reinterpret_cast<float *>(sm + off_prot);   // [BM][BP]
        int ii = 0;
        for (; ii < my_tiles; ++ii) {
            if (*reinterpret_cast<volatile int *>(&s_abort)) break;
            const int g = layer_of(ii);
            float accp[NT][4] = {};
            if (!mbar_wait_all(bar_q8f + 8 * (ii & 1), (ii >> 1) & 1)) {
                if (lane == 0) {
                    latch_error(err, BISCO_ERR_TIMEOUT);
                    atomicExch(&s_abort, 1);
                }
                break;
            }
            const int pg = s_L[g].p;
            const __half *xsh = reinterpret_cast<const __half *>(xs_of(g)), *xsl = xsh + B * cap;
            const int8_t *slab = q8base + (ii & 1) * q8_buf_bytes;
            for (int u16 = 0; u16 < pg; u16 += 16)
                protected_rows<NT>(slab, s_L[g].q8_pitch, u16, gq, t, xsh, xsl, cap, B, accp);
            __syncwarp();
            // buffer ii & 1 is free: the slab of tile ii + 2 goes into it
            if (lane == 0 && ii + 2 < my_tiles) {
                fence_proxy_async_smem();
                issue_q8(ii + 2);
            }
#pragma unroll
            for (int nt = 0; nt < NT; ++nt)
#pragma unroll
                for (int e = 0; e < 4; ++e)
                    prot[(e < 2 ? gq : gq + 8) * BP + nt * 8 + 2 * t + (e & 1)] = accp[nt][e];
            __syncwarp();
            if (!mbar_wait_all(bar_rf + 8 * (ii & 1), (ii >> 1) & 1)) {
                if (lane == 0) {
                    latch_error(err, BISCO_ERR_TIMEOUT);
                    atomicExch(&s_abort, 1);
                }
                break;
            }
            const float *rb = red + (ii & 1) * NCW * BM * B;
            const int row0 = row0_of(ii, g), N = s_L[g].N;
            float *y = s_L[g].y;
            for (int e = lane; e < B * BM; e += 32) {
                const int b = e / BM, r = e - b * BM;
                float v = 0.f;
                // table decode: one partial per row; MMA decode: one per warp
#pragma unroll
                for (int wq = 0; wq < (LUT ? 1 : NCW); ++wq) v += rb[(wq * BM + r) * B + b];
                v += prot[r * BP + b];
                if (row0 + r < N) y[static_cast<int64_t>(b) * N + row0 + r] = v;
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(bar_re + 8 * (ii & 1));
        }
        // the slabs of the two tiles after the last one consumed (issued by the
        // prologue or above) have landed before this warp leaves
        if (lane == 0)
            for (int t2 = ii; t2 < my_tiles && t2 < ii + 2; ++t2)
                mbar_wait(bar_q8f + 8 * (t2 & 1), (t2 >> 1) & 1);
    } else if constexpr (LUT) {
        // --------------------------------- consumers: table decode, batch 1
        const int row0 = warp * kLutRows;
        const uint32_t tab = sbase + a.off_tab;
        for (int ii = 0; ii < my_tiles; ++ii) {
            if (*reinterpret_cast<volatile int *>(&s_abort)) break;
            const int g = layer_of(ii);
            const int *pidx = pidx_of(g), *su = su_of(g);
            const float *xj = xj_of(g);
            float acc[kLutRows] = {};
            bool ok = true;
            for (int w = 0; w < nwide; ++w) {
                const int gidx = ii * nwide + w;
                if (!mbar_wait_all(full_bar(gidx), full_parity(gidx)) ||
                    __any_sync(0xFFFFFFFFu, *reinterpret_cast<volatile int *>(&s_abort) != 0)) {
                    ok = false;
                    break;
                }
                const unsigned char *cs = sm + (gidx % nslot) * kSlotBytes;
                lut_slot<S, kLutRows, kCodeRow, kNormRow>(smem_u32(cs), smem_u32(cs) + kCodesBytes, tab,
                                                          w, row0, lane, acc);
                if constexpr (!kLutMasked) {
                    const int u0 = su[w], u1 = su[w + 1];
                    if (u1 > u0)
                        lut_protected<S, kLutRows, kCodeRow, kNormRow>(cs, cs + kCodesBytes, w, row0, lane,
                                                                       pidx, xj, u0, u1, acc);
                }
                __syncwarp();
                if (lane == 0) mbar_arrive(bar_empty + 8 * (gidx % nslot));
            }
            if (ok && ii >= 2 && !mbar_wait_all(bar_re + 8 * (ii & 1), ((ii >> 1) - 1) & 1)) ok = false;
            if (!ok) {
                if (lane == 0) {
                    latch_error(err, BISCO_ERR_TIMEOUT);
                    atomicExch(&s_abort, 1);
                }
                break;
            }
            const float v = reduce_rows2(acc, lane);
            if ((lane & 15) == 0) {
                float *rb = red + (ii & 1) * NCW * BM * B;
                rb[row0 + (lane >> 4)] = v * kInvSqrt8;
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(bar_rf + 8 * (ii & 1));
        }
    } else {
        // ----------------------------------------------- consumers: decode
        const int q = warp % WQ, k = warp / WQ;
        const int gq = lane >> 2, t = lane & 3;
        for (int ii = 0; ii < my_tiles; ++ii) {
            if (*reinterpret_cast<volatile int *>(&s_abort)) break;
            const int g = layer_of(ii);
            // activation row nt * 8 + gq of each n-tile (rows >= B read a zero block)
            const unsigned char *xb[NT];
            int xstep[NT];
#pragma unroll
            for (int nt = 0; nt < NT; ++nt) {
                const int bg = nt * 8 + gq;
                xb[nt] = bg < B ? xt_of(g) + bg * xt_pitch + t * 16 : sm + off_zero + t * 16;
                xstep[nt] = bg < B ? 1024 : 0;
            }
            float acc[4][NT][4] = {};
            bool ok = true;
            // this warp's slots of tile ii: global index ii*nwide + w == k (mod WK)
            for (int w = (k - (ii * nwide) % WK + WK) % WK; w < nwide; w += WK) {
                const int gidx = ii * nwide + w;
                if (!mbar_wait_all(full_bar(gidx), full_parity(gidx)) ||
                    __any_sync(0xFFFFFFFFu, *reinterpret_cast<volatile int *>(&s_abort) != 0)) {
                    ok = false;
                    break;
                }
                const int nar = w * WQ + q;
                if (nar < nnar) {
                    const unsigned char *cs = sm + (gidx % nslot) * kSlotBytes;
                    const unsigned char *xr[NT];
#pragma unroll
                    for (int nt = 0; nt < NT; ++nt) xr[nt] = xb[nt] + nar * xstep[nt];
                    decode_slot<S, BM, kCodeRow, kNormRow, false, NT>(cs, cs + kCodesBytes, q, gq,
                                                                      gq + 8, t, xr, acc);
                }
                __syncwarp();
                if (lane == 0) mbar_arrive(bar_empty + 8 * (gidx % nslot));
            }
            // hand this warp's partial of tile ii to the reducer (buffer ii & 1,
            // free once the reducer has finished tile ii - 2)
            if (ok && ii >= 2 && !mbar_wait_all(bar_re + 8 * (ii & 1), ((ii >> 1) - 1) & 1)) ok = false;
            if (!ok) {
                if (lane == 0) {
                    latch_error(err, BISCO_ERR_TIMEOUT);
                    atomicExch(&s_abort, 1);
                }
                break;
            }
            float *rb = red + (ii & 1) * NCW * BM * B;
#pragma unroll
            for (int nt = 0; nt < NT; ++nt)
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const int r = e < 2 ? gq : gq + 8;
                    const int b = nt * 8 + 2 * t + (e & 1);
                    if (b < B)
                        rb[(warp * BM + r) * B + b] =
                            ((acc[0][nt][e] + acc[1][nt][e]) + (acc[2][nt][e] + acc[3][nt][e])) * kInvSqrt8;
                }
            __syncwarp();
            if (lane == 0) mbar_arrive(bar_rf + 8 * (ii & 1));
        }
    }
}

// ------------------------------------------------------------------------
// Correctness path for layers whose row pitch rules out TMA (K % 128 != 0)
// or whose protected set is too large for the fast kernels' shared memory:
// one warp per output row, fp32 throughout.
__global__ void __launch_bounds__(256) k_gemv_generic(const uint8_t *__restrict__ codes,
                                                      const uint16_t *__restrict__ norms,
                                                      const int8_t *__restrict__ q8,
                                                      const uint16_t *__restrict__ q8_scale,
                                                      const int32_t *__restrict__ prot_idx,
                                                      int N, int K, int S, int p,
                                                      const uint16_t *__restrict__ x, int B,
                                                      float *__restrict__ y, int *err) {
    const int C = K / 8, p_pad = (p + 15) / 16 * 16;
    const int lane = threadIdx.x & 31;
    const int i = blockIdx.x * (blockDim.x / 32) + (threadIdx.x >> 5);
    if (i >= N) return;
    float acc[16];
#pragma unroll
    for (int b = 0; b < 16; ++b) acc[b] = 0.f;
    for (int c = lane; c < C; c += 32) {
        for (int s = 0; s < S; ++s) {
            const int64_t e = (static_cast<int64_t>(s) * N + i) * C + c;
            const uint32_t bits = codes[e];
            const float n = __half2float(__ushort_as_half(norms[e]));
#pragma unroll
            for (int b = 0; b < 16; ++b) {
                if (b >= B) break;
                float d = 0.f;
#pragma unroll
                for (int k = 0; k < 8; ++k) {
                    const float xv = bf16_bits_to_f32(x[static_cast<int64_t>(b) * K + 8 * c + k]);
                    d += ((bits >> k) & 1u) ? -xv : xv;
                }
                acc[b] += n * d;
            }
        }
    }
    // Eq. 10: replace the BSQ value of each protected column by scale * q8
    // (kept in the same 1/sqrt(8) units as acc until the final scaling)
    for (int t = lane; t < p; t += 32) {
        const int j = prot_idx[t], c = j / 8, k = j % 8;
        if (j < 0 || j >= K) {   // not a column of this layer
            latch_error(err, BISCO_ERR_INVALID_ARG);
            continue;
        }
        float wb = 0.f;
        for (int s = 0; s < S; ++s) {
            const int64_t e = (static_cast<int64_t>(s) * N + i) * C + c;
            const float v = __half2float(__ushort_as_half(norms[e]));
            wb += ((codes[e] >> k) & 1u) ? -v : v;
        }
        const float wq = __half2float(__ushort_as_half(q8_scale[t])) *
                         static_cast<float>(q8[static_cast<int64_t>(i) * p_pad + t]) / kInvSqrt8;
#pragma unroll
        for (int b = 0; b < 16; ++b) {
            if (b >= B) break;
            acc[b] += (wq - wb) * bf16_bits_to_f32(x[static_cast<int64_t>(b) * K + j]);
        }
    }
#pragma unroll
    for (int b = 0; b < 16; ++b)
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) acc[b] += __shfl_xor_sync(0xffffffffu, acc[b], o);
    if (lane == 0)
        for (int b = 0; b < B; ++b) y[static_cast<int64_t>(b) * N + i] = acc[b] * kInvSqrt8;
}

// ------------------------------------------------------------- planning

constexpr size_t kMaxSmem = 227 * 1024;
// Two CTAs (this layer's and the next one's) share an SM when each needs at
// most this much dynamic shared memory (228 KB per SM, 1 KB reserved per CTA).
constexpr size_t kCoresident = 112 * 1024;

struct Plan {
    int wm, wq, ck, nslot;
};

// (WM, WQ) tilings of k_gemv that are instantiated.
constexpr int kTilings[][2] = {{1, 4}, {2, 4}, {4, 4}, {2, 2}, {4, 2}, {4, 1}, {8, 1}, {1, 2}};

bool tiling_known(int wm, int wq) {
    for (const auto &t : kTilings)
        if (t[0] == wm && t[1] == wq) return true;
    return false;
}

// Tuning overrides, read on every call (sweeps, and tests that cover every
// path):  BISCO_GEMV_MODE  = "stream" | "cluster"   force a kernel
//         BISCO_GEMV_PLAN  = "WM,CK,NSLOT[,WQ]"     k_gemv tiling
//         BISCO_GEMV_NSLOT = n                      k_gemv_stream ring depth
bool plan_override(Plan *pl) {
    const char *e = getenv("BISCO_GEMV_PLAN");
    if (!e) return false;
    int v[4] = {0, 0, 0, 1};
    const int n = sscanf(e, "%d,%d,%d,%d", &v[0], &v[1], &v[2], &v[3]);
    if (n < 3 || !tiling_known(v[0], v[3]) || v[1] < 1 || v[1] > 8 || v[2] < 0 || v[2] > 16)
        return false;
    *pl = {v[0], v[3], v[1], v[2]};
    return true;
}

size_t align_up(size_t v, size_t a) { return (v + a - 1) / a * a; }

// Shared-memory carve-up after the ring (common to both kernels).
size_t layout_tail(size_t off, int B, int nar, int q8_bytes, int pidx_cap, int red_bytes,
                   int cl_bytes, int prot_bytes, int nbars, GemvArgs *a) {
    a->off_xt = static_cast<uint32_t>(off);
    a->xt_pitch = nar * 1024 + 64;   // +64 B: rows g and g+1 land in different banks
    off += static_cast<size_t>(B) * a->xt_pitch;
    off = align_up(off, 128);
    a->off_q8 = static_cast<uint32_t>(off);
    off += q8_bytes;
    a->pidx_cap = pidx_cap;
    a->off_pidx = static_cast<uint32_t>(off);
    off += static_cast<size_t>(2 + B) * pidx_cap * 4;   // indices, scales, scale * x
    a->off_pmask = static_cast<uint32_t>(off);
    off += static_cast<size_t>(nar) * (kSlab / 32) * 4;
    a->off_pu = static_cast<uint32_t>(off);
    off += static_cast<size_t>(nar) * (kSlab / 32) * 4;
    off = align_up(off, 16);
    a->off_zero = static_cast<uint32_t>(off);
    off += 1024;
    a->off_red = static_cast<uint32_t>(off);
    off += red_bytes;
    a->off_cl = static_cast<uint32_t>(off);
    off += cl_bytes;
    a->off_prot = static_cast<uint32_t>(off);
    off += prot_bytes;
    off = align_up(off, 8);
    a->off_bar = static_cast<uint32_t>(off);
    off += static_cast<size_t>(nbars) * 8;
    return off + 1024;   // slack for the 1024-byte aligned base
}

size_t cluster_smem(int wm, int wq, int ck, int S, int B, int p, int wide_per_rank, int nslot,
                    GemvArgs *a) {
    const int BM = 16 * wm, BP = B > 8 ? 16 : 8, SW = kSlab * wq;
    const int nar = wide_per_rank * wq;
    const int cap = static_cast<int>(align_up(static_cast<size_t>(std::min(p, nar * kSlab)), 16));
    const int q8_boxes = p > 0 ? (cap + 15 + 127) / 128 : 0;   // bound per CTA
    const size_t ring = static_cast<size_t>(nslot) * S * BM * (SW / 8 + SW / 4);
    return layout_tail(ring, B, nar, q8_boxes * BM * 128, cap, wq * BM * BP * 4,
                       (ck > 1 ? ck - 1 : 0) * BM * BP * 4, 0, nslot * 2 + 2, a);
}

// Shared memory of k_gemv_stream for G layers (largest protected count
// p_max, largest int8 row pitch q8_pitch).  The table decode (lut) keeps nibble
// tables of x instead of staged fp16 copies.  A grouped launch (MAXG > 1)
// keeps the protected-column masks of its prologue as scratch in the table
// area, built over afterwards; a single layer's tables are built from the
// masks, which therefore get their own area.
template <int MAXG>
size_t stream_smem(int wq, int wk, int S, int B, int K, int G, int p_max, int q8_pitch, int nslot,
                   bool lut, StreamArgs<MAXG> *a) {
    const int BM = 16, BP = B > 8 ? 16 : 8, SW = kSlab * wq;
    const int nar = (K + kSlab - 1) / kSlab;
    const int nwide = (K + SW - 1) / SW;
    a->pidx_cap = static_cast<int>(align_up(static_cast<size_t>(p_max), 16));
    a->mwords = nar * (kSlab / 32);
    // indices, scales, scale * x [B]; the table decode adds x and slot starts
    a->pblk = lut ? (3 + B) * a->pidx_cap + static_cast<int>(align_up(nwide + 1, 4))
                  : (2 + B) * a->pidx_cap;
    size_t off = static_cast<size_t>(nslot) * S * BM * (SW / 8 + SW / 4);
    if (lut) {
        a->off_tab = static_cast<uint32_t>(off);
        a->off_pmask = static_cast<uint32_t>(off);   // G * 2 * mwords words <= K bytes
        a->off_xt = a->off_zero = 0;
        a->xt_pitch = 0;
        off += static_cast<size_t>(nwide) * kLutSlotBytes;
        if (MAXG == 1) {
            a->off_pmask = static_cast<uint32_t>(off);
            off += static_cast<size_t>(2) * a->mwords * 4;
        }
    } else {
        a->off_tab = 0;
        a->off_xt = static_cast<uint32_t>(off);
        a->xt_pitch = nar * 1024 + 64;   // +64 B: rows g and g+1 land in different banks
        off += static_cast<size_t>(G) * B * a->xt_pitch;
    }
    off = align_up(off, 128);
    a->off_q8 = static_cast<uint32_t>(off);
    off += static_cast<size_t>(2) * q8_pitch * BM;
    a->off_pidx = static_cast<uint32_t>(off);
    off += static_cast<size_t>(G) * a->pblk * 4;
    if (!lut) {
        a->off_pmask = static_cast<uint32_t>(off);
        off += static_cast<size_t>(G) * 2 * a->mwords * 4;       // masks, prefix counts
        off = align_up(off, 16);
        a->off_zero = static_cast<uint32_t>(off);
        off += 1024;
    }
    off = align_up(off, 16);
    a->off_red = static_cast<uint32_t>(off);
    off += static_cast<size_t>(2) * wq * wk * BM * B * 4;   // partials of the B rows
    a->off_prot = static_cast<uint32_t>(off);
    off += static_cast<size_t>(BM) * BP * 4;
    off = align_up(off, 8);
    a->off_bar = static_cast<uint32_t>(off);
    off += static_cast<size_t>(nslot * (wk + 1) + 8) * 8;
    return off + 128;   // slack for the 128-byte aligned base
}

// k_gemv tiling rule: 2048-column slots (four column-quarter warps per row
// group), 32 rows per CTA (16 for short layers, 64 at batch > 8); the K split
// grows until about one CTA per SM.
Plan choose_plan(int N, int K, int B) {
    const int sms = num_sms();
    Plan pl = B > 8 ? Plan{4, 4, 1, 0} : Plan{2, 4, 1, 0};
    if (B <= 8 && N <= 2048) pl = {1, 4, 1, 0};
    const int SW = kSlab * pl.wq;
    const int total_wide = (K + SW - 1) / SW;
    const int mblocks = (N + 16 * pl.wm - 1) / (16 * pl.wm);
    while (pl.ck < 8 && pl.ck < total_wide && static_cast<long>(mblocks) * pl.ck < (sms * 4) / 5)
        ++pl.ck;
    return pl;
}

template <typename Kern>
bool set_smem(Kern kern, size_t smem, size_t (&configured)[64]) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return false;
    if (smem > configured[dev]) {
        if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 static_cast<int>(smem)) != cudaSuccess)
            return false;
        configured[dev] = smem;
    }
    return true;
}

template <int WM, int WQ, int NT, int S>
bisco_status launch_t(const CUtensorMap &mc, const CUtensorMap &mn, const CUtensorMap &mq,
                      const GemvArgs &a, int ck, size_t smem, cudaStream_t stream) {
    auto kern = k_gemv<WM, WQ, NT, S>;
    static size_t configured[64] = {};
    if (!set_smem(kern, smem, configured)) return BISCO_ERR_CUDA;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(ck, (a.N + 16 * WM - 1) / (16 * WM), 1);
    cfg.blockDim = dim3((WM * WQ + 1) * 32, 1, 1);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = ck;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 2;
    return cudaLaunchKernelEx(&cfg, kern, mc, mn, mq, a) == cudaSuccess ? BISCO_OK : BISCO_ERR_CUDA;
}

template <int WM, int WQ, int NT>
bisco_status launch_s(int S, const CUtensorMap &mc, const CUtensorMap &mn, const CUtensorMap &mq,
                      const GemvArgs &a, int ck, size_t smem, cudaStream_t stream) {
    switch (S) {
        case 1: return launch_t<WM, WQ, NT, 1>(mc, mn, mq, a, ck, smem, stream);
        case 2: return launch_t<WM, WQ, NT, 2>(mc, mn, mq, a, ck, smem, stream);
        default: return launch_t<WM, WQ, NT, 3>(mc, mn, mq, a, ck, smem, stream);
    }
}

template <int WM, int WQ>
bisco_status launch_w(bool two, int S, const CUtensorMap &mc, const CUtensorMap &mn,
                      const CUtensorMap &mq, const GemvArgs &a, int ck, size_t smem,
                      cudaStream_t stream) {
    if (two) {
        if constexpr (WM >= 2) return launch_s<WM, WQ, 2>(S, mc, mn, mq, a, ck, smem, stream);
        return BISCO_ERR_UNSUPPORTED;
    }
    return launch_s<WM, WQ, 1>(S, mc, mn, mq, a, ck, smem, stream);
}

template <int WQ, int WK, int S, int MAXG, bool LUT, int NT = 1>
bisco_status launch_stream_t(const StreamArgs<MAXG> &a, int grid, size_t smem, cudaStream_t stream) {
    auto kern = k_gemv_stream<WQ, WK, S, MAXG, LUT, NT>;
    static size_t configured[64] = {};
    if (!set_smem(kern, smem, configured)) return BISCO_ERR_CUDA;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid, 1, 1);
    cfg.blockDim = dim3((WQ * WK + 2) * 32, 1, 1);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kern, a) == cudaSuccess ? BISCO_OK : BISCO_ERR_CUDA;
}

// Tensor maps of one layer: signs and norms as [S][N][K/8] boxes of
// rows x SW columns (all S stages), q8 as [N][p_pad] boxes of rows x 128.
bool layer_maps(const bisco_layer &L, int rows, int SW, bool swz, CUtensorMap *mc, CUtensorMap *mn,
                CUtensorMap *mq) {
    const int N = L.n_out, K = L.k_in, S = L.stages, p = L.n_protected;
    const uint64_t dims[3] = {static_cast<uint64_t>(K / 8), static_cast<uint64_t>(N),
                              static_cast<uint64_t>(S)};
    const uint64_t strides[2] = {static_cast<uint64_t>(K / 8), static_cast<uint64_t>(N) * (K / 8)};
    const uint32_t box[3] = {static_cast<uint32_t>(SW / 8), static_cast<uint32_t>(rows),
                             static_cast<uint32_t>(S)};
    const uint64_t nstrides[2] = {static_cast<uint64_t>(K / 4), static_cast<uint64_t>(N) * (K / 4)};
    if (!encode_tensor_map(mc, CU_TENSOR_MAP_DATA_TYPE_UINT8, 3, L.codes, dims, strides, box,
                           CU_TENSOR_MAP_SWIZZLE_NONE) ||
        !encode_tensor_map(mn, CU_TENSOR_MAP_DATA_TYPE_UINT16, 3, L.norms, dims, nstrides, box,
                           swz ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_NONE))
        return false;
    if (p > 0) {
        const int p_pad = (p + 15) / 16 * 16;
        const uint64_t qd[2] = {static_cast<uint64_t>(p_pad), static_cast<uint64_t>(N)};
        const uint64_t qs[1] = {static_cast<uint64_t>(p_pad)};
        const uint32_t qb[2] = {128, static_cast<uint32_t>(rows)};
        if (!encode_tensor_map(mq, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, L.q8, qd, qs, qb,
                               CU_TENSOR_MAP_SWIZZLE_NONE))
            return false;
    } else {
        *mq = *mc;   // never dereferenced when p == 0
    }
    return true;
}

// Ring depth: as many slots as fit next to `rest` bytes within `budget`,
// clamped to [lo, hi].
int fit_slots(size_t rest, size_t slot, size_t budget, int lo, int hi) {
    const long fit = rest < budget ? static_cast<long>((budget - rest) / slot) : 0;
    return static_cast<int>(fit < lo ? lo : (fit > hi ? hi : fit));
}

// One k_gemv_stream launch over G layers that share x (same K and S).
// *launched stays false when the shared memory does not fit.
template <int MAXG>
bisco_status launch_stream_g(const bisco_layer *Ls, int G, const uint16_t *x, int B,
                             float *const *y, int *err, int sms, cudaStream_t stream, bool *launched) {
    constexpr int WQ = 4, WK = 2;
    const int K = Ls[0].k_in, S = Ls[0].stages;
    // batch 1 decodes through nibble tables of x unless BISCO_GEMV_LUT=0
    const char *lut_env = getenv("BISCO_GEMV_LUT");
    const bool lut = B == 1 && !(lut_env && lut_env[0] == '0');
    *launched = false;
    // batch 9..16 (two MMA n-tiles) for single layers only
    if (B > 8 && (MAXG > 1 || B > 16)) return BISCO_OK;
    StreamArgs<MAXG> a = {};
    a.x = x;
    a.err = err;
    a.K = K;
    a.B = B;
    a.G = G;
    int p_max = 0, q8_max = 0, tiles = 0;
    for (int g = 0; g < G; ++g) {
        const bisco_layer &L = Ls[g];
        StreamLayer &sl = a.L[g];
        sl.y = y[g];
        sl.q8_scale = L.q8_scale;
        sl.prot_idx = L.prot_idx;
        sl.N = L.n_out;
        sl.p = L.n_protected;
        sl.tile0 = tiles;
        sl.q8 = L.q8;
        sl.q8_pitch = L.n_protected > 0 ? (L.n_protected + 15) / 16 * 16 : 0;
        tiles += (L.n_out + 15) / 16;
        p_max = p_max > sl.p ? p_max : sl.p;
        q8_max = q8_max > sl.q8_pitch ? q8_max : sl.q8_pitch;
    }
    a.ntiles = tiles;
    a.q8_pitch = q8_max;
    const size_t slot = static_cast<size_t>(S) * 16 * (kSlab * WQ / 8 + kSlab * WQ / 4);
    int nslot = 0;
    if (const char *e = getenv("BISCO_GEMV_NSLOT")) nslot = atoi(e);
    if (nslot <= 0 || nslot > 16) {
        // at least three slots: with two, the refills of a long launch are
        // exposed (measured -15 % on the S = 3 MLP shapes), which costs more
        // than sharing the SM with the next kernel gains
        nslot = fit_slots(stream_smem(WQ, WK, S, B, K, G, p_max, q8_max, 0, lut, &a), slot,
                          kCoresident, 3, 8);
        if (stream_smem(WQ, WK, S, B, K, G, p_max, q8_max, nslot, lut, &a) > kMaxSmem) nslot = 2;
    }
    const size_t smem = stream_smem(WQ, WK, S, B, K, G, p_max, q8_max, nslot, lut, &a);
    if (smem > kMaxSmem) return BISCO_OK;
    a.nslot = nslot;
    for (int g = 0; g < G; ++g) {
        CUtensorMap unused_q8;   // the int8 slab goes by bulk copy
        if (!layer_maps(Ls[g], 16, kSlab * WQ, false, &a.mc[g], &a.mn[g], &unused_q8))
            return BISCO_ERR_CUDA;
    }
    const int grid = tiles < sms ? tiles : sms;
    *launched = true;
    if (lut) {
        switch (S) {
            case 1: return launch_stream_t<WQ, WK, 1, MAXG, true>(a, grid, smem, stream);
            case 2: return launch_stream_t<WQ, WK, 2, MAXG, true>(a, grid, smem, stream);
            default: return launch_stream_t<WQ, WK, 3, MAXG, true>(a, grid, smem, stream);
        }
    }
    if constexpr (MAXG == 1) {
        if (B > 8) {
            switch (S) {
                case 1: return launch_stream_t<WQ, WK, 1, MAXG, false, 2>(a, grid, smem, stream);
                case 2: return launch_stream_t<WQ, WK, 2, MAXG, false, 2>(a, grid, smem, stream);
                default: return launch_stream_t<WQ, WK, 3, MAXG, false, 2>(a, grid, smem, stream);
            }
        }
    }
    switch (S) {
        case 1: return launch_stream_t<WQ, WK, 1, MAXG, false>(a, grid, smem, stream);
        case 2: return launch_stream_t<WQ, WK, 2, MAXG, false>(a, grid, smem, stream);
        default: return launch_stream_t<WQ, WK, 3, MAXG, false>(a, grid, smem, stream);
    }
}

// A single layer gets the one-layer instantiation: a run-time layer index
// (and the larger parameter block) cost about 5 % per launch.
bisco_status launch_stream(const bisco_layer *Ls, int G, const uint16_t *x, int B, float *const *y,
                           int *err, int sms, cudaStream_t stream, bool *launched) {
    if (G == 1) return launch_stream_g<1>(Ls, G, x, B, y, err, sms, stream, launched);
    return launch_stream_g<kMaxGroup>(Ls, G, x, B, y, err, sms, stream, launched);
}

}  // namespace

bisco_status launch_gemv(const bisco_layer &L, const uint16_t *x, int B, float *y, int *err,
                         cudaStream_t stream) {
    const int N = L.n_out, K = L.k_in, S = L.stages, p = L.n_protected;
    auto generic = [&]() -> bisco_status {
        const int rows_per_block = 8;
        k_gemv_generic<<<(N + rows_per_block - 1) / rows_per_block, 32 * rows_per_block, 0, stream>>>(
            L.codes, L.norms, L.q8, L.q8_scale, L.prot_idx, N, K, S, p, x, B, y, err);
        return cudaGetLastError() == cudaSuccess ? BISCO_OK : BISCO_ERR_CUDA;
    };
    if (K % 128 != 0) return generic();   // row pitch rules out TMA

    GemvArgs a = {};
    a.x = x;
    a.y = y;
    a.q8_scale = L.q8_scale;
    a.prot_idx = L.prot_idx;
    a.err = err;
    a.N = N;
    a.K = K;
    a.B = B;
    a.p = p;

    // batch 1: the row-split kernel of gemv_b1.cu where it applies (K a
    // multiple of 4096), unless a kernel of this file is forced
    const char *mode = getenv("BISCO_GEMV_MODE");
    if (B == 1 && !mode) {
        bool launched = false;
        const bisco_status st = launch_gemv_b1(&L, 1, x, &y, err, stream, &launched);
        if (launched || st != BISCO_OK) return st;
    }

    // streaming kernel: small batch and at least one 16-row tile per SM
    const int sms = num_sms();
    bool use_stream = B <= 16 && (N + 15) / 16 >= sms;
    if (mode && mode[0] == 's') use_stream = B <= 16;
    if (mode && mode[0] == 'c') use_stream = false;
    if (use_stream) {
        bool launched = false;
        const bisco_status st = launch_stream(&L, 1, x, B, &y, err, sms, stream, &launched);
        if (launched || st != BISCO_OK) return st;
    }

    // k_gemv plan: the preferred tiling (or BISCO_GEMV_PLAN), then smaller
    // ones; for each, split K further until the staged activations and a
    // 2-slot ring fit (at batch 9..16 the activations alone are 16 rows of
    // K fp16, so large K needs narrow slots and wide splits)
    Plan first = choose_plan(N, K, B);
    const bool forced = plan_override(&first);
    if (B > 8 && first.wm < 2) first = {2, first.wq, first.ck, first.nslot};
    if (!tiling_known(first.wm, first.wq)) first = {2, 4, first.ck, first.nslot};
    Plan cands[1 + sizeof(kTilings) / sizeof(kTilings[0])];
    int ncand = 0;
    cands[ncand++] = first;
    if (!forced) {
        // fallbacks, largest row block first (two MMA n-tiles need WM >= 2)
        static const int order[][2] = {{4, 4}, {2, 4}, {4, 2}, {2, 2}, {1, 4}, {1, 2}, {4, 1}, {8, 1}};
        for (const auto &t : order) {
            if (B > 8 && t[0] < 2) continue;
            if (t[0] == first.wm && t[1] == first.wq) continue;
            cands[ncand++] = {t[0], t[1], 1, 0};
        }
    }
    Plan pl = {};
    int wpr = 0, nslot = 0;
    size_t smem = 0;
    bool fits = false;
    for (int ci = 0; ci < ncand && !fits; ++ci) {
        pl = cands[ci];
        const int BMc = 16 * pl.wm, SWc = kSlab * pl.wq;
        const int total_wide_c = (K + SWc - 1) / SWc;
        if (pl.ck > total_wide_c) pl.ck = total_wide_c;
        const size_t slot = static_cast<size_t>(S) * BMc * (SWc / 8 + SWc / 4);
        for (;;) {
            wpr = (total_wide_c + pl.ck - 1) / pl.ck;
            nslot = pl.nslot;
            if (nslot <= 0) {
                nslot = fit_slots(cluster_smem(pl.wm, pl.wq, pl.ck, S, B, p, wpr, 0, &a), slot,
                                  kCoresident, 2, 8);
                if (nslot > wpr && wpr >= 2) nslot = wpr;
            }
            if (nslot < 2) nslot = 2;
            smem = cluster_smem(pl.wm, pl.wq, pl.ck, S, B, p, wpr, nslot, &a);
            if (smem <= kMaxSmem) {
                fits = true;
                break;
            }
            if (pl.ck >= 8 || pl.ck >= total_wide_c) break;
            ++pl.ck;
        }
    }
    if (!fits) return generic();   // e.g. p close to K
    const int BM = 16 * pl.wm;
    const int SW = kSlab * pl.wq;
    a.wide_per_rank = wpr;
    a.nslot = nslot;
    CUtensorMap mc, mn, mq;
    if (!layer_maps(L, BM, SW, pl.wq == 1, &mc, &mn, &mq)) return BISCO_ERR_CUDA;

    const bool two = B > 8;
    const int ck = pl.ck;
    if (pl.wm == 1 && pl.wq == 4) return launch_w<1, 4>(two, S, mc, mn, mq, a, ck, smem, stream);
    if (pl.wm == 2 && pl.wq == 4) return launch_w<2, 4>(two, S, mc, mn, mq, a, ck, smem, stream);
    if (pl.wm == 4 && pl.wq == 4) return launch_w<4, 4>(two, S, mc, mn, mq, a, ck, smem, stream);
    if (pl.wm == 2 && pl.wq == 2) return launch_w<2, 2>(two, S, mc, mn, mq, a, ck, smem, stream);
    if (pl.wm == 4 && pl.wq == 2) return launch_w<4, 2>(two, S, mc, mn, mq, a, ck, smem, stream);
    if (pl.wm == 4 && pl.wq == 1) return launch_w<4, 1>(two, S, mc, mn, mq, a, ck, smem, stream);
    if (pl.wm == 8 && pl.wq == 1) return launch_w<8, 1>(two, S, mc, mn, mq, a, ck, smem, stream);
    if (pl.wm == 1 && pl.wq == 2) return launch_w<1, 2>(two, S, mc, mn, mq, a, ck, smem, stream);
    return BISCO_ERR_UNSUPPORTED;
}

bisco_status launch_gemv_multi(const bisco_layer *Ls, int G, const uint16_t *x, int B,
                               float *const *y, int *err, cudaStream_t stream) {
    if (B == 1 && !getenv("BISCO_GEMV_MODE")) {
        bool launched = false;
        const bisco_status st = launch_gemv_b1(Ls, G, x, y, err, stream, &launched);
        if (launched || st != BISCO_OK) return st;
    }
    if (B <= 8 && Ls[0].k_in % 128 == 0) {
        bool launched = false;
        const bisco_status st = launch_stream(Ls, G, x, B, y, err, num_sms(), stream, &launched);
        if (launched || st != BISCO_OK) return st;
    }
    for (int g = 0; g < G; ++g) {   // one launch per layer
        const bisco_status st = launch_gemv(Ls[g], x, B, y[g], err, stream);
        if (st != BISCO_OK) return st;
    }
    return BISCO_OK;
}

}  // namespace bisco
