// gemv.cu -- decode-time y = What x straight from the coded layer
// (Sec. III-F Eq. 12 with the Eq. 10 protected scatter), batch 1..16.
//
// Design (GB300, HBM-bound):
//  * Each CTA owns BM = 16*WM output rows and one K range; a cluster of CK
//    CTAs splits K and reduces its partial sums in a fixed rank order
//    through distributed shared memory (deterministic, no atomics).
//  * One producer thread streams 512-column slabs of the sign bytes and the
//    fp16 norms of all S stages into a shared-memory ring with TMA
//    (cp.async.bulk.tensor, mbarrier complete_tx); the norm tile uses the
//    128-byte swizzle so the consumers' 16-byte reads are conflict-free.
//  * Consumer warps own 16 rows each and decode in registers: for a 32-bit
//    code word holding chunks c..c+3 (byte per chunk), one shift brings the
//    sign bits of element j of chunk c and of chunk c+2 to bits 15 and 31,
//    and one LOP3 ((w << s) & 0x80008000) ^ (n_c | n_{c+2} << 16) yields the
//    fp16 pair (+-n_c, +-n_{c+2}) exactly.  These pairs are the A fragments
//    of mma.m16n8k16 (fp16 in, fp32 accumulate), one MMA per stage, so the
//    stage sum of Eq. 12 is exact in fp32.  The activation operand is staged
//    once per CTA as fp16 in the matching permuted order, with protected
//    columns zeroed (Eq. 10's overwrite).
//  * Epilogue: the int8 protected columns are one more small MMA pass
//    (q8 as exact fp16 integers against scale_j * x_j split into fp16
//    hi + lo parts), then y = acc / sqrt(8) + acc_protected.
#include <cuda_runtime.h>
#include <stdint.h>
#include <stdio.h>
#include <stdlib.h>


#include "bisco_dev.cuh"
#include "bisco_host.h"

namespace bisco {
namespace {

constexpr int kSlab = 512;            // input columns per ring slot
constexpr int kCodeRow = kSlab / 8;   // 64 bytes of signs per row per stage
constexpr int kNormRow = kSlab / 4;   // 128 bytes of norms per row per stage
constexpr float kInvSqrt8 = 0.35355339059327373f;

struct GemvArgs {
    const uint16_t *x;
    float *y;
    const uint16_t *q8_scale;
    const int32_t *prot_idx;
    int *err;
    int N, K, B, p;
    int slabs_per_rank, total_slabs, nslot;
    uint32_t off_xt, off_q8, off_xs, off_red, off_bar;
    int xt_pitch;   // bytes per activation row in the staged operand
    int xs_pitch;   // halves per activation row of the protected operand
    int q8_boxes;   // 128-column TMA boxes of q8 reserved per CTA
};

__device__ __forceinline__ uint32_t word_of(const uint4 &v, int i) {
    return i == 0 ? v.x : (i == 1 ? v.y : (i == 2 ? v.z : v.w));
}

// Position (in halves, within one activation row) of slab-relative column
// kk in the permuted operand layout [slab][w][m][t][4 pairs][2].
__device__ __forceinline__ int xt_pos(int kk) {
    const int slab = kk >> 9, col = kk & 511;
    const int t = col >> 7, cc = col & 127;
    const int w = cc >> 5, cw = cc & 31;
    const int c4 = cw >> 3, j = cw & 7;
    const int i = 8 * (c4 & 1) + j, half = c4 >> 1;
    return slab * 512 + (((w * 4 + (i >> 2)) * 4 + t) * 4 + (i & 3)) * 2 + half;
}

__device__ __forceinline__ int lower_bound_i32(const int32_t *a, int n, int v) {
    int lo = 0, hi = n;
    while (lo < hi) {
        const int mid = (lo + hi) >> 1;
        if (a[mid] < v) lo = mid + 1; else hi = mid;
    }
    return lo;
}

__device__ __forceinline__ uint32_t pack_q8_pair(int8_t a, int8_t b) {
    const __half2 h = __floats2half2_rn(static_cast<float>(a), static_cast<float>(b));
    return *reinterpret_cast<const uint32_t *>(&h);
}

template <int WM, int NT, int S>
__global__ void __launch_bounds__((WM + 1) * 32, 1)
k_gemv(const __grid_constant__ CUtensorMap tm_codes, const __grid_constant__ CUtensorMap tm_norms,
       const __grid_constant__ CUtensorMap tm_q8, const GemvArgs a) {
    constexpr int BM = 16 * WM;
    constexpr int BP = 8 * NT;
    constexpr uint32_t kCodesBytes = S * BM * kCodeRow;
    constexpr uint32_t kSlotBytes = S * BM * (kCodeRow + kNormRow);

    extern __shared__ unsigned char smem_raw[];
    unsigned char *sm = reinterpret_cast<unsigned char *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const uint32_t sbase = smem_u32(sm);
    __shared__ int s_abort, s_lo, s_hi;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int rank = static_cast<int>(cluster_ctarank());
    const int nrank = static_cast<int>(cluster_nctarank());
    const int row0 = blockIdx.y * BM;
    const int slab0 = rank * a.slabs_per_rank;
    const int nsl = max(0, min(a.slabs_per_rank, a.total_slabs - slab0));
    const int k_begin = slab0 * kSlab;
    const int k_end = min(a.K, k_begin + nsl * kSlab);
    const int nslot = a.nslot;
    const uint32_t bar_full = sbase + a.off_bar;
    const uint32_t bar_empty = bar_full + 8 * nslot;
    const uint32_t bar_q8 = bar_full + 16 * nslot;

    if (threadIdx.x == 0) {
        for (int i = 0; i < nslot; ++i) {
            mbar_init(bar_full + 8 * i, 1);
            mbar_init(bar_empty + 8 * i, WM);
        }
        mbar_init(bar_q8, 1);
        fence_mbar_init();
        s_abort = 0;
    }
    if (threadIdx.x == 32) {
        s_lo = a.p ? lower_bound_i32(a.prot_idx, a.p, k_begin) : 0;
        s_hi = a.p ? lower_bound_i32(a.prot_idx, a.p, k_end) : 0;
    }
    __syncthreads();
    const int lo_t = s_lo, p_loc = s_hi - s_lo;
    const bool producer = (warp == WM) && (lane == 0);

    // Weights do not depend on earlier kernels: start streaming them before
    // waiting on the previous grid (programmatic dependent launch).
    int issued = 0;
    if (producer) {
        prefetch_tmap(&tm_codes);
        prefetch_tmap(&tm_norms);
        if (p_loc > 0) {
            const int qx0 = lo_t & ~15;
            const int nq = (lo_t + p_loc - qx0 + 127) >> 7;
            mbar_arrive_expect_tx(bar_q8, static_cast<uint32_t>(nq * BM * 128));
            for (int q = 0; q < nq; ++q)
                tma_load_2d(sbase + a.off_q8 + q * BM * 128, &tm_q8, bar_q8, qx0 + 128 * q, row0);
        }
        for (; issued < nsl && issued < nslot; ++issued) {
            const uint32_t dst = sbase + issued * kSlotBytes;
            mbar_arrive_expect_tx(bar_full + 8 * issued, kSlotBytes);
            const int kx = (k_begin + issued * kSlab) / 8;
            tma_load_3d(dst, &tm_codes, bar_full + 8 * issued, kx, row0, 0);
            tma_load_3d(dst + kCodesBytes, &tm_norms, bar_full + 8 * issued, kx, row0, 0);
        }
    }

    pdl_wait();

    // Stage the activation operand: fp16, permuted to fragment order,
    // protected columns zeroed; and scale_j * x_j as fp16 hi + lo.
    {
        uint16_t *xt = reinterpret_cast<uint16_t *>(sm + a.off_xt);
        const int cols = nsl * kSlab;
        const int pitch_h = a.xt_pitch / 2;
        for (int e = threadIdx.x; e < a.B * cols; e += blockDim.x) {
            const int b = e / cols, kk = e - b * cols;
            const int k = k_begin + kk;
            const uint16_t v = k < k_end ? bf16_bits_to_f16_bits(a.x[static_cast<int64_t>(b) * a.K + k]) : 0;
            xt[b * pitch_h + xt_pos(kk)] = v;
        }
        __syncthreads();
        __half *xs_hi = reinterpret_cast<__half *>(sm + a.off_xs);
        __half *xs_lo = xs_hi + a.B * a.xs_pitch;
        const int p16 = (p_loc + 15) & ~15;
        for (int e = threadIdx.x; e < a.B * p16; e += blockDim.x) {
            const int b = e / p16, u = e - b * p16;
            float v = 0.f;
            if (u < p_loc) {
                const int j = a.prot_idx[lo_t + u];
                xt[b * pitch_h + xt_pos(j - k_begin)] = 0;
                v = __half2float(__ushort_as_half(a.q8_scale[lo_t + u])) *
                    bf16_bits_to_f32(a.x[static_cast<int64_t>(b) * a.K + j]);
            }
            const __half h = __float2half_rn(v);
            xs_hi[b * a.xs_pitch + u] = h;
            xs_lo[b * a.xs_pitch + u] = __float2half_rn(v - __half2float(h));
        }
    }
    __syncthreads();
    pdl_launch_dependents();

    float *red = reinterpret_cast<float *>(sm + a.off_red);

    if (warp == WM) {
        // ------------------------------------------------ producer: refill
        if (producer) {
            for (; issued < nsl; ++issued) {
                const int slot = issued % nslot;
                const uint32_t par = ((issued / nslot) - 1) & 1;
                if (!mbar_wait(bar_empty + 8 * slot, par)) {
                    latch_error(a.err, BISCO_ERR_TIMEOUT);
                    atomicExch(&s_abort, 1);
                    break;
                }
                if (*reinterpret_cast<volatile int *>(&s_abort)) break;
                const uint32_t dst = sbase + slot * kSlotBytes;
                mbar_arrive_expect_tx(bar_full + 8 * slot, kSlotBytes);
                const int kx = (k_begin + issued * kSlab) / 8;
                tma_load_3d(dst, &tm_codes, bar_full + 8 * slot, kx, row0, 0);
                tma_load_3d(dst + kCodesBytes, &tm_norms, bar_full + 8 * slot, kx, row0, 0);
            }
            if (*reinterpret_cast<volatile int *>(&s_abort)) {
                // let every copy already in flight land before the CTA exits
                for (int slot = 0; slot < nslot && slot < issued; ++slot) {
                    const int last = slot + ((issued - 1 - slot) / nslot) * nslot;
                    mbar_wait(bar_full + 8 * slot, (last / nslot) & 1);
                }
                if (p_loc > 0) mbar_wait(bar_q8, 0);
            }
        }
    } else {
        // ----------------------------------------------- consumers: decode
        const int g = lane >> 2, t = lane & 3;
        const int rlo = 16 * warp + g, rhi = rlo + 8;
        float acc[NT][4];
#pragma unroll
        for (int nt = 0; nt < NT; ++nt)
#pragma unroll
            for (int k = 0; k < 4; ++k) acc[nt][k] = 0.f;

        for (int it = 0; it < nsl; ++it) {
            const int slot = it % nslot;
            if (*reinterpret_cast<volatile int *>(&s_abort)) break;
            if (!mbar_wait(bar_full + 8 * slot, (it / nslot) & 1)) {
                latch_error(a.err, BISCO_ERR_TIMEOUT);
                atomicExch(&s_abort, 1);
                break;
            }
            const unsigned char *cs = sm + slot * kSlotBytes;
            const unsigned char *ns = cs + kCodesBytes;
            const unsigned char *xrow = sm + a.off_xt + it * 1024 + t * 16;
#pragma unroll
            for (int s = 0; s < S; ++s) {
                const uint4 clo = *reinterpret_cast<const uint4 *>(cs + (s * BM + rlo) * kCodeRow + t * 16);
                const uint4 chi = *reinterpret_cast<const uint4 *>(cs + (s * BM + rhi) * kCodeRow + t * 16);
                const unsigned char *nlo = ns + (s * BM + rlo) * kNormRow;
                const unsigned char *nhi = ns + (s * BM + rhi) * kNormRow;
                const uint4 nl0 = *reinterpret_cast<const uint4 *>(nlo + (((2 * t) ^ (rlo & 7)) << 4));
                const uint4 nl1 = *reinterpret_cast<const uint4 *>(nlo + (((2 * t + 1) ^ (rlo & 7)) << 4));
                const uint4 nh0 = *reinterpret_cast<const uint4 *>(nhi + (((2 * t) ^ (rhi & 7)) << 4));
                const uint4 nh1 = *reinterpret_cast<const uint4 *>(nhi + (((2 * t + 1) ^ (rhi & 7)) << 4));
#pragma unroll
                for (int w = 0; w < 4; ++w) {
                    const uint32_t cl = word_of(clo, w), ch = word_of(chi, w);
                    const uint32_t la = word_of(w < 2 ? nl0 : nl1, (2 * w) & 3);
                    const uint32_t lb = word_of(w < 2 ? nl0 : nl1, (2 * w + 1) & 3);
                    const uint32_t ha = word_of(w < 2 ? nh0 : nh1, (2 * w) & 3);
                    const uint32_t hb = word_of(w < 2 ? nh0 : nh1, (2 * w + 1) & 3);
                    const uint32_t np0l = prmt(la, lb, 0x5410), np1l = prmt(la, lb, 0x7632);
                    const uint32_t np0h = prmt(ha, hb, 0x5410), np1h = prmt(ha, hb, 0x7632);
#pragma unroll
                    for (int m = 0; m < 4; ++m) {
                        uint4 xf[NT];
#pragma unroll
                        for (int nt = 0; nt < NT; ++nt) {
                            const int bg = nt * 8 + g;
                            xf[nt] = bg < a.B ? *reinterpret_cast<const uint4 *>(
                                                    xrow + bg * a.xt_pitch + (w * 4 + m) * 64)
                                              : make_uint4(0, 0, 0, 0);
                        }
#pragma unroll
                        for (int qq = 0; qq < 2; ++qq) {
                            const int q = 2 * m + qq;
                            const int i0 = 2 * q, i1 = 2 * q + 1;
                            const uint32_t nl = q < 4 ? np0l : np1l;
                            const uint32_t nh = q < 4 ? np0h : np1h;
                            uint32_t af[4];
                            af[0] = lop3_and_xor(cl << (15 - i0), 0x80008000u, nl);
                            af[1] = lop3_and_xor(ch << (15 - i0), 0x80008000u, nh);
                            af[2] = lop3_and_xor(cl << (15 - i1), 0x80008000u, nl);
                            af[3] = lop3_and_xor(ch << (15 - i1), 0x80008000u, nh);
#pragma unroll
                            for (int nt = 0; nt < NT; ++nt)
                                mma_16816(acc[nt], af, word_of(xf[nt], 2 * qq), word_of(xf[nt], 2 * qq + 1));
                        }
                    }
                }
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(bar_empty + 8 * slot);
        }

        // protected int8 columns (Eq. 10) as a second MMA pass
        float accp[NT][4];
#pragma unroll
        for (int nt = 0; nt < NT; ++nt)
#pragma unroll
            for (int k = 0; k < 4; ++k) accp[nt][k] = 0.f;
        if (p_loc > 0) {
            if (!mbar_wait(bar_q8, 0)) {
                latch_error(a.err, BISCO_ERR_TIMEOUT);
                atomicExch(&s_abort, 1);
            } else {
                const int8_t *q8s = reinterpret_cast<const int8_t *>(sm + a.off_q8);
                const int qoff = lo_t - (lo_t & ~15);
                const __half *xs_hi = reinterpret_cast<const __half *>(sm + a.off_xs);
                const __half *xs_lo = xs_hi + a.B * a.xs_pitch;
                auto q8at = [&](int r, int u) -> int8_t {
                    if (u >= p_loc) return 0;
                    const int col = qoff + u;
                    return q8s[((col >> 7) * BM + r) * 128 + (col & 127)];
                };
                for (int u16 = 0; u16 < p_loc; u16 += 16) {
                    const int u0 = u16 + 2 * t;
                    uint32_t af[4];
                    af[0] = pack_q8_pair(q8at(rlo, u0), q8at(rlo, u0 + 1));
                    af[1] = pack_q8_pair(q8at(rhi, u0), q8at(rhi, u0 + 1));
                    af[2] = pack_q8_pair(q8at(rlo, u0 + 8), q8at(rlo, u0 + 9));
                    af[3] = pack_q8_pair(q8at(rhi, u0 + 8), q8at(rhi, u0 + 9));
#pragma unroll
                    for (int nt = 0; nt < NT; ++nt) {
                        const int bg = nt * 8 + g;
                        uint32_t h0 = 0, h1 = 0, l0 = 0, l1 = 0;
                        if (bg < a.B) {
                            h0 = *reinterpret_cast<const uint32_t *>(xs_hi + bg * a.xs_pitch + u0);
                            h1 = *reinterpret_cast<const uint32_t *>(xs_hi + bg * a.xs_pitch + u0 + 8);
                            l0 = *reinterpret_cast<const uint32_t *>(xs_lo + bg * a.xs_pitch + u0);
                            l1 = *reinterpret_cast<const uint32_t *>(xs_lo + bg * a.xs_pitch + u0 + 8);
                        }
                        mma_16816(accp[nt], af, h0, h1);
                        mma_16816(accp[nt], af, l0, l1);
                    }
                }
            }
        }
#pragma unroll
        for (int nt = 0; nt < NT; ++nt)
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                const int r = k < 2 ? rlo : rhi;
                const int b = nt * 8 + 2 * t + (k & 1);
                red[r * BP + b] = acc[nt][k] * kInvSqrt8 + accp[nt][k];
            }
    }

    __syncthreads();
    __syncwarp();
    if (nrank > 1) {
        cluster_sync();
        if (rank == 0) {
            const uint32_t red_addr = sbase + a.off_red;
            for (int e = threadIdx.x; e < a.B * BM; e += blockDim.x) {
                const int b = e / BM, r = e - b * BM;
                const uint32_t off = static_cast<uint32_t>((r * BP + b) * 4);
                float v = 0.f;
                for (int q = 0; q < nrank; ++q) v += ld_shared_cluster_f32(mapa_shared(red_addr + off, q));
                if (row0 + r < a.N) a.y[static_cast<int64_t>(b) * a.N + row0 + r] = v;
            }
        }
        __syncwarp();
        cluster_sync();
    } else {
        for (int e = threadIdx.x; e < a.B * BM; e += blockDim.x) {
            const int b = e / BM, r = e - b * BM;
            if (row0 + r < a.N) a.y[static_cast<int64_t>(b) * a.N + row0 + r] = red[r * BP + b];
        }
    }
}

// Correctness path for layers whose row pitch rules out TMA (K % 128 != 0):
// one warp per output row, fp32 throughout.
__global__ void __launch_bounds__(256) k_gemv_generic(const uint8_t *__restrict__ codes,
                                                      const uint16_t *__restrict__ norms,
                                                      const int8_t *__restrict__ q8,
                                                      const uint16_t *__restrict__ q8_scale,
                                                      const int32_t *__restrict__ prot_idx,
                                                      int N, int K, int S, int p,
                                                      const uint16_t *__restrict__ x, int B,
                                                      float *__restrict__ y) {
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

struct Plan {
    int wm, ck, nslot;
};

// "WM,CK,NSLOT" from BISCO_GEMV_PLAN overrides the tiling (tuning sweeps and
// tests that cover every cluster/tile shape); read on every call.
bool plan_override(Plan *pl) {
    const char *e = getenv("BISCO_GEMV_PLAN");
    if (!e) return false;
    int v[3] = {0, 0, 0};
    if (sscanf(e, "%d,%d,%d", &v[0], &v[1], &v[2]) != 3) return false;
    if ((v[0] != 1 && v[0] != 2 && v[0] != 4) || v[1] < 1 || v[1] > 8 || v[2] < 0 || v[2] > 16)
        return false;
    *pl = {v[0], v[1], v[2]};
    return true;
}

constexpr int kSmemBudget = 110 * 1024;

size_t smem_bytes_for(int wm, int S, int B, int p, int slabs_per_rank, int nslot, GemvArgs *a) {
    const int BM = 16 * wm;
    const int NT = B > 8 ? 2 : 1;
    size_t off = static_cast<size_t>(nslot) * S * BM * (kCodeRow + kNormRow);
    a->off_xt = static_cast<uint32_t>(off);
    a->xt_pitch = slabs_per_rank * 1024 + 64;
    off += static_cast<size_t>(B) * a->xt_pitch;
    off = (off + 127) & ~size_t(127);
    a->off_q8 = static_cast<uint32_t>(off);
    a->q8_boxes = p > 0 ? (p + 15 + 127) / 128 : 0;
    off += static_cast<size_t>(a->q8_boxes) * BM * 128;
    a->off_xs = static_cast<uint32_t>(off);
    a->xs_pitch = ((p + 15) & ~15) + 8;
    off += static_cast<size_t>(2) * B * a->xs_pitch * 2;
    off = (off + 15) & ~size_t(15);
    a->off_red = static_cast<uint32_t>(off);
    off += static_cast<size_t>(BM) * 8 * NT * 4;
    a->off_bar = static_cast<uint32_t>(off);
    off += static_cast<size_t>(2 * nslot + 1) * 8;
    return off + 1024;   // alignment slack for the 1024-byte aligned base
}

Plan choose_plan(int N, int K, int B, int S) {
    const int sms = num_sms();
    const int total_slabs = (K + kSlab - 1) / kSlab;
    Plan best{4, 1, 2};
    long best_score = -1;
    for (int wm : {4, 2, 1}) {
        if (B > 8 && wm < 2) continue;
        const int BM = 16 * wm;
        const int mblocks = (N + BM - 1) / BM;
        for (int ck = 1; ck <= 8; ++ck) {
            const int spr = (total_slabs + ck - 1) / ck;
            if ((ck - 1) * spr >= total_slabs) continue;          // an empty rank
            if (static_cast<long>(B) * (spr * 1024 + 64) > 64 * 1024) continue;
            const long ctas = static_cast<long>(mblocks) * ck;
            // prefer ~2 resident CTAs per SM, then bigger tiles, then less split
            const long fill = ctas >= 2L * sms ? 2L * sms : ctas;
            const long score = fill * 64 + wm * 8 - ck;
            if (score > best_score) {
                best_score = score;
                best = {wm, ck, 0};
            }
        }
    }
    return best;
}

template <int WM, int NT, int S>
bisco_status launch_t(const CUtensorMap &mc, const CUtensorMap &mn, const CUtensorMap &mq,
                      const GemvArgs &a, int ck, size_t smem, cudaStream_t stream) {
    auto kern = k_gemv<WM, NT, S>;
    static size_t configured[64] = {};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return BISCO_ERR_CUDA;
    if (smem > configured[dev]) {
        if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 static_cast<int>(smem)) != cudaSuccess)
            return BISCO_ERR_CUDA;
        if (cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) !=
            cudaSuccess)
            return BISCO_ERR_CUDA;
        configured[dev] = smem;
    }
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(ck, (a.N + 16 * WM - 1) / (16 * WM), 1);
    cfg.blockDim = dim3((WM + 1) * 32, 1, 1);
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

template <int WM, int NT>
bisco_status launch_s(int S, const CUtensorMap &mc, const CUtensorMap &mn, const CUtensorMap &mq,
                      const GemvArgs &a, int ck, size_t smem, cudaStream_t stream) {
    switch (S) {
        case 1: return launch_t<WM, NT, 1>(mc, mn, mq, a, ck, smem, stream);
        case 2: return launch_t<WM, NT, 2>(mc, mn, mq, a, ck, smem, stream);
        default: return launch_t<WM, NT, 3>(mc, mn, mq, a, ck, smem, stream);
    }
}

}  // namespace

bisco_status launch_gemv(const bisco_layer &L, const uint16_t *x, int B, float *y, int *err,
                         cudaStream_t stream) {
    const int N = L.n_out, K = L.k_in, S = L.stages, p = L.n_protected;
    if (K % 128 != 0) {
        const int rows_per_block = 8;
        k_gemv_generic<<<(N + rows_per_block - 1) / rows_per_block, 32 * rows_per_block, 0, stream>>>(
            L.codes, L.norms, L.q8, L.q8_scale, L.prot_idx, N, K, S, p, x, B, y);
        return cudaGetLastError() == cudaSuccess ? BISCO_OK : BISCO_ERR_CUDA;
    }
    Plan pl = choose_plan(N, K, B, S);
    plan_override(&pl);
    if (B > 8 && pl.wm < 2) pl.wm = 2;
    const int BM = 16 * pl.wm;
    const int total_slabs = (K + kSlab - 1) / kSlab;
    if (pl.ck > total_slabs) pl.ck = total_slabs;
    const int spr = (total_slabs + pl.ck - 1) / pl.ck;

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
    a.slabs_per_rank = spr;
    a.total_slabs = total_slabs;
    // ring depth: as many slots as fit next to the rest, 2..8
    int nslot = pl.nslot;
    if (nslot <= 0) {
        const size_t rest = smem_bytes_for(pl.wm, S, B, p, spr, 0, &a);
        const size_t slot = static_cast<size_t>(S) * BM * (kCodeRow + kNormRow);
        long fit = rest < static_cast<size_t>(kSmemBudget) ? (kSmemBudget - static_cast<long>(rest)) / static_cast<long>(slot) : 0;
        nslot = static_cast<int>(fit < 2 ? 2 : (fit > 8 ? 8 : fit));
        if (nslot > spr && spr >= 2) nslot = spr;
        if (nslot < 2) nslot = 2;
    }
    a.nslot = nslot;
    const size_t smem = smem_bytes_for(pl.wm, S, B, p, spr, nslot, &a);
    if (smem > 227 * 1024) return BISCO_ERR_UNSUPPORTED;

    CUtensorMap mc, mn, mq;
    {
        const uint64_t dims[3] = {static_cast<uint64_t>(K / 8), static_cast<uint64_t>(N),
                                  static_cast<uint64_t>(S)};
        const uint64_t strides[2] = {static_cast<uint64_t>(K / 8),
                                     static_cast<uint64_t>(N) * (K / 8)};
        const uint32_t box[3] = {static_cast<uint32_t>(kCodeRow), static_cast<uint32_t>(BM),
                                 static_cast<uint32_t>(S)};
        if (!encode_tensor_map(&mc, CU_TENSOR_MAP_DATA_TYPE_UINT8, 3, L.codes, dims, strides, box,
                               CU_TENSOR_MAP_SWIZZLE_NONE))
            return BISCO_ERR_CUDA;
        const uint64_t nstrides[2] = {static_cast<uint64_t>(K / 4),
                                      static_cast<uint64_t>(N) * (K / 4)};
        const uint32_t nbox[3] = {static_cast<uint32_t>(kCodeRow), static_cast<uint32_t>(BM),
                                  static_cast<uint32_t>(S)};
        if (!encode_tensor_map(&mn, CU_TENSOR_MAP_DATA_TYPE_UINT16, 3, L.norms, dims, nstrides,
                               nbox, CU_TENSOR_MAP_SWIZZLE_128B))
            return BISCO_ERR_CUDA;
    }
    if (p > 0) {
        const int p_pad = (p + 15) / 16 * 16;
        const uint64_t dims[2] = {static_cast<uint64_t>(p_pad), static_cast<uint64_t>(N)};
        const uint64_t strides[1] = {static_cast<uint64_t>(p_pad)};
        const uint32_t box[2] = {128, static_cast<uint32_t>(BM)};
        if (!encode_tensor_map(&mq, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, L.q8, dims, strides, box,
                               CU_TENSOR_MAP_SWIZZLE_NONE))
            return BISCO_ERR_CUDA;
    } else {
        mq = mc;   // never dereferenced when p == 0
    }

    const bool two = B > 8;
    switch (pl.wm) {
        case 1: return two ? BISCO_ERR_UNSUPPORTED : launch_s<1, 1>(S, mc, mn, mq, a, pl.ck, smem, stream);
        case 2: return two ? launch_s<2, 2>(S, mc, mn, mq, a, pl.ck, smem, stream)
                           : launch_s<2, 1>(S, mc, mn, mq, a, pl.ck, smem, stream);
        default: return two ? launch_s<4, 2>(S, mc, mn, mq, a, pl.ck, smem, stream)
                            : launch_s<4, 1>(S, mc, mn, mq, a, pl.ck, smem, stream);
    }
}

}  // namespace bisco
