// gemv.cu -- decode-time y = What x straight from the coded layer
// (Sec. III-F Eq. 12 with the Eq. 10 protected scatter), batch 1..16.
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

// 1024-byte aligned base of the dynamic shared memory, derived by pointer
// arithmetic on the shared array so that accesses stay shared-space ones.
__device__ __forceinline__ unsigned char *aligned_smem(unsigned char *raw) {
    return raw + ((1024u - (smem_u32(raw) & 1023u)) & 1023u);
}

constexpr int kMaxGroup = 4;   // layers sharing one activation in a grouped launch

// Per-layer shared-memory view used by the activation staging.
struct StageView {
    unsigned char *xt;        // [B][xt_pitch] staged fp16 operand
    const uint32_t *pmask;    // protected-column bits per 32-column group
    const int *pu;            // protected columns before each group
    const float *pscale;      // scale of each protected column
    float *xs;                // [B][cap] scale * x of each protected column
};

// Activation staging for the input columns [k_begin, k_begin + cols) of G
// layers that share x: bf16 rows from global memory -> fp16 in the permuted
// fragment order [512-column slab][w][m][t][4 pairs], converted once, then
// stored per layer with that layer's protected columns zeroed; scale_u *
// x[b][j_u] of the protected columns (exact in fp32: 11 x 8 significant
// bits) is taken from the same cache lines, so the activations cost one
// round trip to memory.  Job = one 32-column group of one row.  Pair i of a
// 32-column group is element i&7 of chunk (i>>3) and of chunk (i>>3)+2 --
// bits i and i+16 of its code word, columns (i>>3)*8 + (i&7) and that + 16.
template <int MAXG>
__device__ __forceinline__ void stage_activations(const uint16_t *x, int K, int B, int k_begin,
                                                  int cols, int nnar, int xt_pitch, int cap,
                                                  int G, const StageView (&v)[MAXG]) {
    const int groups_per_row = cols >> 5;   // cols % 128 == 0 on this path
    const int njobs = B * nnar * 16;
    for (int e = threadIdx.x; e < njobs; e += blockDim.x) {
        const int t = e & 3, w = (e >> 2) & 3, sb = e >> 4;
        const int b = sb / nnar, slab = sb - b * nnar;
        const int g32 = slab * 16 + t * 4 + w;
        const int dst_off = b * xt_pitch + slab * 1024 + t * 16 + w * 256;
        uint32_t o[16];
        const uint16_t *src = x + static_cast<int64_t>(b) * K + k_begin + g32 * 32;
        if (g32 < groups_per_row) {
            uint32_t r[16];
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const uint4 u4 = reinterpret_cast<const uint4 *>(src)[q];
                r[4 * q] = u4.x; r[4 * q + 1] = u4.y; r[4 * q + 2] = u4.z; r[4 * q + 3] = u4.w;
            }
#pragma unroll
            for (int i = 0; i < 16; ++i) {
                // pair i: columns c0 = (i>>3)*8 + (i&7) (low half) and c0 + 16
                const int c0 = (i >> 3) * 8 + (i & 7);
                const uint32_t f = r[c0 >> 1], sw = r[(c0 + 16) >> 1];
                const __half2 h = __floats2half2_rn((c0 & 1) ? bf16_hi(f) : bf16_lo(f),
                                                    (c0 & 1) ? bf16_hi(sw) : bf16_lo(sw));
                o[i] = *reinterpret_cast<const uint32_t *>(&h);
            }
        } else {
#pragma unroll
            for (int i = 0; i < 16; ++i) o[i] = 0u;
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
            // protected columns of this group: record scale * x, zero the halves
            const int u0 = v[g].pu[g32];   // protected columns before this group
            for (uint32_t bits = pm; bits; bits &= bits - 1u) {
                const int k = __ffs(bits) - 1;
                const int u = u0 + __popc(pm & ((1u << k) - 1u));
                v[g].xs[b * cap + u] = v[g].pscale[u] * bf16_bits_to_f32(src[k]);
            }
            uint32_t om[16];
#pragma unroll
            for (int i = 0; i < 16; ++i) {
                const int c0 = (i >> 3) * 8 + (i & 7);
                const uint32_t keep = (((pm >> c0) & 1u) ? 0u : 0x0000FFFFu) |
                                      (((pm >> (c0 + 16)) & 1u) ? 0u : 0xFFFF0000u);
                om[i] = o[i] & keep;
            }
#pragma unroll
            for (int m = 0; m < 4; ++m)
                *reinterpret_cast<uint4 *>(dst + m * 64) =
                    make_uint4(om[4 * m], om[4 * m + 1], om[4 * m + 2], om[4 * m + 3]);
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
// TMA'd int8 slab (column col0 + u of box-major [box][BM][128] storage) as
// exact fp16 integers against scale * x (s_xs) split into fp16 hi + lo.
template <int BM, int NT>
__device__ __forceinline__ void protected_tile(const int8_t *q8s, int col0, int u16, int p_loc,
                                               int rlo, int rhi, int g, int t, const float *s_xs,
                                               int xs_pitch, int B, float (&accp)[NT][4]) {
    auto q8v = [&](int r, int u) -> float {
        if (u >= p_loc) return 0.f;
        const int col = col0 + u;
        return static_cast<float>(q8s[((col >> 7) * BM + r) * 128 + (col & 127)]);
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
        StageView v[1] = {{sm + a.off_xt, s_pmask, s_pu, s_pscale, s_xs}};
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

struct StreamLayer {
    float *y;
    const uint16_t *q8_scale;
    const int32_t *prot_idx;
    int N, p;
    int tile0;       // first tile of this layer in the launch's tile list
    int q8_boxes;    // 128-column boxes of the int8 slab of one tile
};

template <int MAXG>
struct StreamArgs {
    CUtensorMap mc[MAXG], mn[MAXG], mq[MAXG];
    StreamLayer L[MAXG];
    const uint16_t *x;
    int *err;
    int K, B, G, ntiles, nslot;
    int q8_boxes;    // the largest of the layers' (int8 double buffer size)
    int pidx_cap, xt_pitch, mwords;
    uint32_t off_xt, off_q8, off_red, off_bar, off_pidx, off_pmask, off_zero, off_prot;
};

template <int WQ, int WK, int S, int MAXG>
__global__ void __launch_bounds__((WQ * WK + 2) * 32, 2)
k_gemv_stream(const __grid_constant__ StreamArgs<MAXG> a) {
    constexpr int BM = 16;
    constexpr int BP = 8;
    constexpr int NCW = WQ * WK;
    constexpr int SW = kSlab * WQ;
    constexpr int kCodeRow = SW / 8;
    constexpr int kNormRow = SW / 4;
    constexpr uint32_t kCodesBytes = S * BM * kCodeRow;
    constexpr uint32_t kSlotBytes = S * BM * (kCodeRow + kNormRow);

    extern __shared__ unsigned char smem_raw[];
    unsigned char *sm = aligned_smem(smem_raw);
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
    const uint16_t *const x = a.x;
    int *const err = a.err;
    int tile0[MAXG];
#pragma unroll
    for (int i = 0; i < MAXG; ++i) tile0[i] = a.L[i].tile0;
    const CUtensorMap *const maps_c = &a.mc[0];
    const CUtensorMap *const maps_n = &a.mn[0];
    const CUtensorMap *const maps_q = &a.mq[0];
    const int my_tiles = a.ntiles > cta ? (a.ntiles - 1 - cta) / Gd + 1 : 0;
    const int nwide = (K + SW - 1) / SW;
    const int nnar = (K + kSlab - 1) / kSlab;
    const int total = my_tiles * nwide;   // ring fills of this CTA
    const int nslot = a.nslot;
    const int cap = a.pidx_cap;
    const uint32_t q8_buf_bytes = static_cast<uint32_t>(a.q8_boxes * BM * 128);
    const uint32_t bar_full = sbase + a.off_bar;            // [nslot][WK]
    const uint32_t bar_empty = bar_full + 8 * nslot * WK;   // [nslot]
    const uint32_t bar_q8f = bar_empty + 8 * nslot;         // [2] int8 slab landed
    const uint32_t bar_q8e = bar_q8f + 16;                  // [2] int8 slab consumed
    const uint32_t bar_rf = bar_q8e + 16;                   // [2] tile partials written
    const uint32_t bar_re = bar_rf + 16;                    // [2] tile partials read
    const bool producer = (warp == NCW) && (lane == 0);
    const uint64_t pol = l2_evict_first_policy();
    float *red = reinterpret_cast<float *>(sm + a.off_red);   // [2][NCW][BM][B]

    // per-layer shared-memory views
    auto pidx_of = [&](int g) {
        return reinterpret_cast<int *>(sm + off_pidx) + g * (2 + B) * cap;
    };
    auto pscale_of = [&](int g) { return reinterpret_cast<float *>(pidx_of(g) + cap); };
    auto xs_of = [&](int g) { return pscale_of(g) + cap; };
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
    // the int8 slab of tile ii (a plain arrive when its layer has none)
    auto issue_q8 = [&](int ii) {
        const int g = layer_of(ii);
        const uint32_t bar = bar_q8f + 8 * (ii & 1);
        const int boxes = s_L[g].q8_boxes;
        if (boxes == 0) {
            mbar_arrive(bar);
            return;
        }
        const uint32_t dst = sbase + off_q8 + (ii & 1) * q8_buf_bytes;
        mbar_arrive_expect_tx(bar, static_cast<uint32_t>(boxes * BM * 128));
        for (int q = 0; q < boxes; ++q)
            tma_load_2d_hint(dst + q * BM * 128, maps_q + g, bar, 128 * q, row0_of(ii, g), pol);
    };

    int issued = 0, q8_issued = 0;
    if (producer) {
        for (int i = 0; i < nslot; ++i) {
            for (int k = 0; k < WK; ++k) mbar_init(bar_full + 8 * (i * WK + k), 1);
            mbar_init(bar_empty + 8 * i, WQ);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(bar_q8f + 8 * i, 1);
            mbar_init(bar_q8e + 8 * i, 1);
            mbar_init(bar_rf + 8 * i, NCW);
            mbar_init(bar_re + 8 * i, 1);
        }
        fence_mbar_init();
        s_abort = 0;
        for (int g = 0; g < G; ++g) {
            prefetch_tmap(maps_c + g);
            prefetch_tmap(maps_n + g);
        }
        for (; issued < total && issued < nslot; ++issued) {
            // a tile's int8 slab goes out with its first slot (two buffers)
            if (issued % nwide == 0 && issued / nwide < 2) issue_q8(q8_issued++);
            issue_slot(issued);
        }
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
    }
    __syncthreads();
    pdl_launch_dependents();

    // activations may be written by the previous kernel
    pdl_wait();
    {
        StageView v[MAXG] = {};
#pragma unroll
        for (int g = 0; g < MAXG; ++g)
            if (g < G) v[g] = {xt_of(g), pmask_of(g), pu_of(g), pscale_of(g), xs_of(g)};
        stage_activations<MAXG>(x, K, B, 0, K, nnar, xt_pitch, cap, G, v);
    }
    for (int i = threadIdx.x; i < 1024 / 16; i += blockDim.x)
        reinterpret_cast<uint4 *>(sm + off_zero)[i] = make_uint4(0, 0, 0, 0);
    __syncthreads();

    if (warp == NCW) {
        // ------------------------------------------------ producer: refill
        if (producer) {
            // The int8 slab of tile ii (buffer ii & 1) goes out just before the
            // tile's first slot, once tile ii-2 released the buffer; every slot
            // of tile ii-1 is issued by then, so this never starves the decode.
            auto issue_q8_upto = [&](int ii) -> bool {
                while (q8_issued <= ii && q8_issued < my_tiles) {
                    if (q8_issued >= 2 &&
                        !mbar_wait(bar_q8e + 8 * (q8_issued & 1), ((q8_issued >> 1) - 1) & 1))
                        return false;
                    issue_q8(q8_issued);
                    ++q8_issued;
                }
                return true;
            };
            bool ok = true;
            for (; issued < total; ++issued) {
                const int slot = issued % nslot;
                if (issued % nwide == 0 && !issue_q8_upto(issued / nwide)) {
                    ok = false;
                    break;
                }
                if (!mbar_wait(bar_empty + 8 * slot, ((issued / nslot) - 1) & 1)) {
                    ok = false;
                    break;
                }
                if (*reinterpret_cast<volatile int *>(&s_abort)) break;
                issue_slot(issued);
            }
            if (ok && !*reinterpret_cast<volatile int *>(&s_abort) && !issue_q8_upto(my_tiles - 1))
                ok = false;
            if (!ok) {
                latch_error(err, BISCO_ERR_TIMEOUT);
                atomicExch(&s_abort, 1);
            }
            // every copy issued has landed before this thread leaves
            for (int gi = (issued > nslot ? issued - nslot : 0); gi < issued; ++gi)
                mbar_wait(full_bar(gi), full_parity(gi));
            for (int ii = (q8_issued > 2 ? q8_issued - 2 : 0); ii < q8_issued; ++ii)
                mbar_wait(bar_q8f + 8 * (ii & 1), (ii >> 1) & 1);
        }
    } else if (warp == NCW + 1) {
        // ------------------------------------------- reducer: protected + y
        const int gq = lane >> 2, t = lane & 3;
        const int8_t *q8base = reinterpret_cast<const int8_t *>(sm + off_q8);
        float *prot = reinterpret_cast<float *>(sm + off_prot);   // [BM][BP]
        for (int ii = 0; ii < my_tiles; ++ii) {
            if (*reinterpret_cast<volatile int *>(&s_abort)) break;
            const int g = layer_of(ii);
            float accp[1][4] = {{0.f, 0.f, 0.f, 0.f}};
            if (!mbar_wait_all(bar_q8f + 8 * (ii & 1), (ii >> 1) & 1)) {
                if (lane == 0) {
                    latch_error(err, BISCO_ERR_TIMEOUT);
                    atomicExch(&s_abort, 1);
                }
                break;
            }
            const int pg = s_L[g].p;
            for (int u16 = 0; u16 < pg; u16 += 16)
                protected_tile<BM, 1>(q8base + (ii & 1) * q8_buf_bytes, 0, u16, pg, gq, gq + 8, gq,
                                      t, xs_of(g), cap, B, accp);
            __syncwarp();
            if (lane == 0) mbar_arrive(bar_q8e + 8 * (ii & 1));
#pragma unroll
            for (int e = 0; e < 4; ++e) prot[(e < 2 ? gq : gq + 8) * BP + 2 * t + (e & 1)] = accp[0][e];
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
#pragma unroll
                for (int wq = 0; wq < NCW; ++wq) v += rb[(wq * BM + r) * B + b];
                v += prot[r * BP + b];
                if (row0 + r < N) y[static_cast<int64_t>(b) * N + row0 + r] = v;
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(bar_re + 8 * (ii & 1));
        }
    } else {
        // ----------------------------------------------- consumers: decode
        const int q = warp % WQ, k = warp / WQ;
        const int gq = lane >> 2, t = lane & 3;
        const int xstep = gq < B ? 1024 : 0;
        for (int ii = 0; ii < my_tiles; ++ii) {
            if (*reinterpret_cast<volatile int *>(&s_abort)) break;
            const int g = layer_of(ii);
            const unsigned char *xb = gq < B ? xt_of(g) + gq * xt_pitch + t * 16
                                             : sm + off_zero + t * 16;
            float acc[4][1][4];
#pragma unroll
            for (int c = 0; c < 4; ++c)
#pragma unroll
                for (int e = 0; e < 4; ++e) acc[c][0][e] = 0.f;
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
                    const unsigned char *xr[1] = {xb + nar * xstep};
                    decode_slot<S, BM, kCodeRow, kNormRow, false, 1>(cs, cs + kCodesBytes, q, gq,
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
            for (int e = 0; e < 4; ++e) {
                const int r = e < 2 ? gq : gq + 8;
                const int b = 2 * t + (e & 1);
                if (b < B)
                    rb[(warp * BM + r) * B + b] =
                        ((acc[0][0][e] + acc[1][0][e]) + (acc[2][0][e] + acc[3][0][e])) * kInvSqrt8;
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
// p_max, largest int8 slab q8_boxes).
template <int MAXG>
size_t stream_smem(int wq, int wk, int S, int B, int K, int G, int p_max, int q8_boxes, int nslot,
                   StreamArgs<MAXG> *a) {
    const int BM = 16, BP = 8, SW = kSlab * wq;
    const int nar = (K + kSlab - 1) / kSlab;
    a->pidx_cap = static_cast<int>(align_up(static_cast<size_t>(p_max), 16));
    a->mwords = nar * (kSlab / 32);
    size_t off = static_cast<size_t>(nslot) * S * BM * (SW / 8 + SW / 4);
    a->off_xt = static_cast<uint32_t>(off);
    a->xt_pitch = nar * 1024 + 64;   // +64 B: rows g and g+1 land in different banks
    off += static_cast<size_t>(G) * B * a->xt_pitch;
    off = align_up(off, 128);
    a->off_q8 = static_cast<uint32_t>(off);
    off += static_cast<size_t>(2) * q8_boxes * BM * 128;
    a->off_pidx = static_cast<uint32_t>(off);
    off += static_cast<size_t>(G) * (2 + B) * a->pidx_cap * 4;   // indices, scales, scale * x
    a->off_pmask = static_cast<uint32_t>(off);
    off += static_cast<size_t>(G) * 2 * a->mwords * 4;           // masks, prefix counts
    off = align_up(off, 16);
    a->off_zero = static_cast<uint32_t>(off);
    off += 1024;
    a->off_red = static_cast<uint32_t>(off);
    off += static_cast<size_t>(2) * wq * wk * BM * B * 4;   // partials of the B rows
    a->off_prot = static_cast<uint32_t>(off);
    off += static_cast<size_t>(BM) * BP * 4;
    off = align_up(off, 8);
    a->off_bar = static_cast<uint32_t>(off);
    off += static_cast<size_t>(nslot * (wk + 1) + 8) * 8;
    return off + 1024;   // slack for the 1024-byte aligned base
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

template <int WQ, int WK, int S, int MAXG>
bisco_status launch_stream_t(const StreamArgs<MAXG> &a, int grid, size_t smem, cudaStream_t stream) {
    auto kern = k_gemv_stream<WQ, WK, S, MAXG>;
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
    *launched = false;
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
        sl.q8_boxes = L.n_protected > 0 ? ((L.n_protected + 15) / 16 * 16 + 127) / 128 : 0;
        tiles += (L.n_out + 15) / 16;
        p_max = p_max > sl.p ? p_max : sl.p;
        q8_max = q8_max > sl.q8_boxes ? q8_max : sl.q8_boxes;
    }
    a.ntiles = tiles;
    a.q8_boxes = q8_max;
    const size_t slot = static_cast<size_t>(S) * 16 * (kSlab * WQ / 8 + kSlab * WQ / 4);
    int nslot = 0;
    if (const char *e = getenv("BISCO_GEMV_NSLOT")) nslot = atoi(e);
    if (nslot <= 0 || nslot > 16) {
        // at least three slots: with two, the refills of a long launch are
        // exposed (measured -15 % on the S = 3 MLP shapes), which costs more
        // than sharing the SM with the next kernel gains
        nslot = fit_slots(stream_smem(WQ, WK, S, B, K, G, p_max, q8_max, 0, &a), slot, kCoresident,
                          3, 8);
        if (stream_smem(WQ, WK, S, B, K, G, p_max, q8_max, nslot, &a) > kMaxSmem) nslot = 2;
    }
    const size_t smem = stream_smem(WQ, WK, S, B, K, G, p_max, q8_max, nslot, &a);
    if (smem > kMaxSmem) return BISCO_OK;
    a.nslot = nslot;
    for (int g = 0; g < G; ++g)
        if (!layer_maps(Ls[g], 16, kSlab * WQ, false, &a.mc[g], &a.mn[g], &a.mq[g]))
            return BISCO_ERR_CUDA;
    const int grid = tiles < sms ? tiles : sms;
    *launched = true;
    switch (S) {
        case 1: return launch_stream_t<WQ, WK, 1, MAXG>(a, grid, smem, stream);
        case 2: return launch_stream_t<WQ, WK, 2, MAXG>(a, grid, smem, stream);
        default: return launch_stream_t<WQ, WK, 3, MAXG>(a, grid, smem, stream);
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

    // streaming kernel: small batch and at least one 16-row tile per SM
    const char *mode = getenv("BISCO_GEMV_MODE");
    const int sms = num_sms();
    bool use_stream = B <= 8 && (N + 15) / 16 >= sms;
    if (mode && mode[0] == 's') use_stream = B <= 8;
    if (mode && mode[0] == 'c') use_stream = false;
    if (use_stream) {
        bool launched = false;
        const bisco_status st = launch_stream(&L, 1, x, B, &y, err, sms, stream, &launched);
        if (launched || st != BISCO_OK) return st;
    }

    Plan pl = choose_plan(N, K, B);
    plan_override(&pl);
    if (B > 8 && pl.wm < 2) pl = {2, pl.wq, pl.ck, pl.nslot};
    if (!tiling_known(pl.wm, pl.wq)) pl = {2, 4, pl.ck, pl.nslot};
    const int BM = 16 * pl.wm;
    const int SW = kSlab * pl.wq;
    const int total_wide = (K + SW - 1) / SW;
    if (pl.ck > total_wide) pl.ck = total_wide;
    const size_t slot = static_cast<size_t>(S) * BM * (SW / 8 + SW / 4);
    // split K further until the staged activations and a 2-slot ring fit
    int wpr = 0, nslot = 0;
    size_t smem = 0;
    for (;;) {
        wpr = (total_wide + pl.ck - 1) / pl.ck;
        nslot = pl.nslot;
        if (nslot <= 0) {
            nslot = fit_slots(cluster_smem(pl.wm, pl.wq, pl.ck, S, B, p, wpr, 0, &a), slot,
                              kCoresident, 2, 8);
            if (nslot > wpr && wpr >= 2) nslot = wpr;
        }
        if (nslot < 2) nslot = 2;
        smem = cluster_smem(pl.wm, pl.wq, pl.ck, S, B, p, wpr, nslot, &a);
        if (smem <= kMaxSmem) break;
        if (pl.ck >= 8 || pl.ck >= total_wide) return generic();   // e.g. p close to K
        ++pl.ck;
    }
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
