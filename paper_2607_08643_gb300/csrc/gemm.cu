// gemm.cu -- prefill Y = X What^T (Sec. III-G Eq. 12 with the Eq. 10
// protected scatter) on the 5th-generation tensor cores.
//
// Prefill is a dense contraction, so the decoded weight feeds tcgen05.mma
// (kind::f16, fp32 accumulation in tensor memory).  The weight is never
// written out: per 128-column step, decoder warps expand the TMA-staged sign
// bytes and fp16 norms of 128 output features into fp16 values in registers
// (shift + LOP3 per element pair, the S stages summed with one fp16 add per
// stage, Eq. 12) and store them straight into tensor memory, where they are
// the MMA's A operand (M = 128 features).  The activations are the B operand
// (N = 256 tokens), TMA-staged in the 128-byte swizzle.
//
// The activations are bf16 and the decoded weight fp16; one MMA needs one
// type, so a pre-pass writes an fp16 copy of X into the workspace with the
// protected columns zeroed (Eq. 10's overwrite) and, appended after the
// K columns, sqrt(8) * scale_j * x_j split into fp16 hi and lo parts in
// blocks of 64 protected columns [hi | lo].  The matching A columns are the
// int8 q8 values (exact in fp16), so the protected term is a few more k
// steps of the same MMA, and the epilogue is Y = D / sqrt(8).
//
// CTA roles (512 threads, one CTA per SM, persistent over whole tiles
// taken round robin, or over a range of the tiles' k-steps in a stream-K
// split; gemm_sched.cuh):
//   warps 0-3  epilogue: TMEM -> registers -> Y (fp32), or to a partial
//              tile in the workspace; lane quarter w
//   warp 4     TMA producer of the compressed-weight ring
//   warp 5     TMEM allocator and MMA issuer (one thread)
//   warp 6     TMA producer of the activation ring
//   warps 8-15 decoders: lane quarter w % 4, K half (w - 8) / 4
#include <cuda_runtime.h>
#include <stdint.h>

#include "bisco_dev.cuh"
#include "bisco_host.h"
#include "gemm_sched.cuh"

namespace bisco {
namespace {

constexpr int GM = 128;     // output features per tile (MMA M, TMEM lanes)
constexpr int GN = 256;     // tokens per tile (MMA N); 128 when M <= 128
constexpr int GK = 128;     // K columns per weight step (one TMEM A stage)
// Ring depths are template parameters (NX activation stages of 64 columns
// = 32 KB, NW compressed-weight stages of 128 columns): the activation ring
// must cover the L2 latency of a stream consumed at 64 B/clk, so it takes
// what the weight ring leaves of the 227 KB.
constexpr int NA = 3;       // TMEM A ring (128 K columns = 64 TMEM columns each)
constexpr int kThreads = 512;
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kColD = 0;     // accumulator: TN <= 256 fp32 columns
constexpr uint32_t kColA = 256;   // A stages
// one 64-column activation stage of a TN-token tile: TN rows x 64 fp16
constexpr uint32_t x_stage_bytes(int tn) { return static_cast<uint32_t>(tn) * 128; }
constexpr float kInvSqrt8 = 0.35355339059327373f;
constexpr float kSqrt8 = 2.8284271247461903f;

struct GemmArgs {
    float *Y;
    int *err;
    float *part;    // partial tiles of the stream-K split: [G][2][TN tokens][GM features] fp32
    int M, N, S;
    int ks_main;    // 128-column weight steps over K (K_pad / 128)
    int ks_ext;     // extension steps (one per 64 protected columns)
    int tiles_t;    // token tiles
    SkPlan sk;      // the split of the tiles' k-steps over the CTAs (gemm_sched.cuh)
    uint32_t w_stage;   // bytes of one compressed-weight stage
};

// idesc of kind::f16: D f32, A = B = f16, both K-major, N = tn, M = GM.
constexpr uint32_t idesc_f16(int tn) {
    return (1u << 4) | (static_cast<uint32_t>(tn >> 3) << 17) | (static_cast<uint32_t>(GM >> 4) << 24);
}

// Decoded fp16 pairs of 8 chunks (64 columns) of one row and S stages:
// element pair (2j, 2j+1) of chunk c is ((t << (15-2j)) & 0x80008000) ^
// (n|n<<16) with t = byte * 0x8001 (bit k at k and at k+15), stages summed
// in fp16.  out[4c + j] holds K columns 8c + 2j, 8c + 2j + 1.
__device__ __forceinline__ void decode_row64(const unsigned char *codes, const unsigned char *norms,
                                             int S, int r, int h, uint32_t (&out)[32]) {
#pragma unroll 1
    for (int s = 0; s < S; ++s) {
        const uint2 cw = *reinterpret_cast<const uint2 *>(codes + (s * GM + r) * 16 + h * 8);
        const uint4 nw = *reinterpret_cast<const uint4 *>(norms + (s * GM + r) * 32 + h * 16);
        const uint32_t nv[4] = {nw.x, nw.y, nw.z, nw.w};
#pragma unroll
        for (int c = 0; c < 8; ++c) {
            const uint32_t word = c < 4 ? cw.x : cw.y;
            const uint32_t b = prmt(word, 0u, 0x4440u + (c & 3));       // byte c, zero-extended
            const uint32_t t = b * 0x8001u;
            const uint32_t np = prmt(nv[c >> 1], 0u, (c & 1) ? 0x3232u : 0x1010u);   // n | n << 16
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const uint32_t v = lop3_and_xor(t << (15 - 2 * j), 0x80008000u, np);
                if (s == 0) {
                    out[4 * c + j] = v;
                } else {
                    __half2 a = *reinterpret_cast<const __half2 *>(&out[4 * c + j]);
                    a = __hadd2(a, *reinterpret_cast<const __half2 *>(&v));
                    out[4 * c + j] = *reinterpret_cast<const uint32_t *>(&a);
                }
            }
        }
    }
}

// 64 int8 q8 values of one row -> fp16 pairs (exact): bytes biased by 128
// become the mantissa of 1024 + u, minus 1152.
__device__ __forceinline__ void decode_q8_row(const unsigned char *q8s, int r, uint32_t (&out)[32]) {
    const __half2 bias = __floats2half2_rn(1152.f, 1152.f);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const uint4 v = *reinterpret_cast<const uint4 *>(q8s + r * 64 + 16 * i);
        const uint32_t w4[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const uint32_t x = w4[q] ^ 0x80808080u;
            uint32_t lo = prmt(x, 0x64646464u, 0x5140u);
            uint32_t hi = prmt(x, 0x64646464u, 0x7362u);
            __half2 a = __hsub2(*reinterpret_cast<const __half2 *>(&lo), bias);
            __half2 b = __hsub2(*reinterpret_cast<const __half2 *>(&hi), bias);
            out[8 * i + 2 * q] = *reinterpret_cast<const uint32_t *>(&a);
            out[8 * i + 2 * q + 1] = *reinterpret_cast<const uint32_t *>(&b);
        }
    }
}

template <int NX, int NW, int TN>
__global__ void __launch_bounds__(kThreads, 1)
k_gemm(const __grid_constant__ CUtensorMap tm_x, const __grid_constant__ CUtensorMap tm_codes,
       const __grid_constant__ CUtensorMap tm_norms, const __grid_constant__ CUtensorMap tm_q8,
       const GemmArgs a) {
    constexpr uint32_t kXStage = x_stage_bytes(TN);
    constexpr uint32_t kIdesc = idesc_f16(TN);
    extern __shared__ unsigned char smem_raw[];
    unsigned char *sm = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
    const uint32_t sbase = smem_u32(sm);
    __shared__ uint32_t s_tmem;
    __shared__ int s_abort;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t x_ring = sbase;
    const uint32_t w_ring = sbase + NX * kXStage;
    const uint32_t bars = w_ring + NW * a.w_stage;
    const uint32_t xfull = bars, xempty = xfull + 8 * NX;
    const uint32_t wfull = xempty + 8 * NX, wempty = wfull + 8 * NW;
    const uint32_t afull = wempty + 8 * NW, aempty = afull + 8 * NA;
    const uint32_t dfull = aempty + 8 * NA, dempty = dfull + 8, drain = dempty + 8;
    const int S = a.S;
    const SkSched sch(blockIdx.x, a.sk);
    const uint32_t wbytes_main = static_cast<uint32_t>(S) * GM * 48;

    if (threadIdx.x == 0) {
        for (int i = 0; i < NX; ++i) {
            mbar_init(xfull + 8 * i, 1);
            mbar_init(xempty + 8 * i, 1);
        }
        for (int i = 0; i < NW; ++i) {
            mbar_init(wfull + 8 * i, 1);
            mbar_init(wempty + 8 * i, 8);
        }
        for (int i = 0; i < NA; ++i) {
            mbar_init(afull + 8 * i, 8);
            mbar_init(aempty + 8 * i, 1);
        }
        mbar_init(dfull, 1);
        mbar_init(dempty, 4);
        mbar_init(drain, 1);
        fence_mbar_init();
        s_abort = 0;
    }
    if (warp == 5) tmem_alloc(smem_u32(&s_tmem), kTmemCols);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    // the kernel launched after this one (the fixup, or the next call's
    // pre-pass) may take its place on the SMs now and wait there for this
    // grid's completion
    pdl_launch_dependents();
    const uint32_t tmem = s_tmem;
    auto aborted = [&]() { return *reinterpret_cast<volatile int *>(&s_abort) != 0; };
    auto fail = [&]() {
        latch_error(a.err, BISCO_ERR_TIMEOUT);
        atomicExch(&s_abort, 1);
    };

    if (warp == 4) {
        // ----------------------------------- producer: compressed weights
        // (its own thread: the weight ring runs ahead of the decoders without
        // waiting for the MMAs to free activation stages)
        if (lane == 0) {
            prefetch_tmap(&tm_codes);
            prefetch_tmap(&tm_norms);
            int wi = 0;
            bool ok = true;
            for (int j = 0; ok && j < sch.n; ++j) {
                const SkPiece pc = sch.at(j, blockIdx.x, a.sk);
                const int f0 = (pc.t / a.tiles_t) * GM;
                for (int ks = pc.k0; ks < pc.k1; ++ks) {
                    const int ws = wi % NW;
                    if (wi >= NW && !mbar_wait(wempty + 8 * ws, ((wi / NW) - 1) & 1)) { ok = false; break; }
                    if (aborted()) { ok = false; break; }
                    const uint32_t wdst = w_ring + ws * a.w_stage;
                    if (ks < a.ks_main) {
                        mbar_arrive_expect_tx(wfull + 8 * ws, wbytes_main);
                        // weights are re-read by the CTAs working on the other token tiles
                        // of this feature tile: normal L2 policy
                        tma_load_3d(wdst, &tm_codes, wfull + 8 * ws, ks * (GK / 8), f0, 0);
                        tma_load_3d(wdst + S * GM * 16, &tm_norms, wfull + 8 * ws, ks * (GK / 8), f0, 0);
                    } else {
                        mbar_arrive_expect_tx(wfull + 8 * ws, GM * 64);
                        tma_load_2d(wdst, &tm_q8, wfull + 8 * ws, (ks - a.ks_main) * 64, f0);
                    }
                    ++wi;
                }
            }
            if (!ok) fail();
            // every copy issued has landed before this thread leaves (in the
            // normal case the consumers saw them all, so this returns at once)
            for (int i = (wi > NW ? wi - NW : 0); i < wi; ++i) mbar_wait(wfull + 8 * (i % NW), (i / NW) & 1);
        }
    } else if (warp == 6) {
        // ----------------------------------------- producer: activations
        if (lane == 0) {
            prefetch_tmap(&tm_x);
            // the activation copy X16 is written by the pre-pass launched just
            // before this kernel (programmatic dependent launch)
            pdl_wait();
            int xi = 0;
            bool ok = true;
            for (int j = 0; ok && j < sch.n; ++j) {
                const SkPiece pc = sch.at(j, blockIdx.x, a.sk);
                const int t0 = (pc.t % a.tiles_t) * TN;
                for (int ks = pc.k0; ok && ks < pc.k1; ++ks) {
                    for (int hh = 0; hh < 2; ++hh) {
                        const int xs = xi % NX;
                        if (xi >= NX && !mbar_wait(xempty + 8 * xs, ((xi / NX) - 1) & 1)) { ok = false; break; }
                        if (aborted()) { ok = false; break; }
                        mbar_arrive_expect_tx(xfull + 8 * xs, kXStage);
                        tma_load_2d(x_ring + xs * kXStage, &tm_x, xfull + 8 * xs, ks * GK + hh * 64, t0);
                        ++xi;
                    }
                }
            }
            if (!ok) fail();
            for (int i = (xi > NX ? xi - NX : 0); i < xi; ++i) mbar_wait(xfull + 8 * (i % NX), (i / NX) & 1);
        }
    } else if (warp == 5) {
        // --------------------------------------------------- MMA issuer
        if (lane == 0) {
            int xi = 0, ai = 0;
            bool ok = true;
            for (int ti = 0; ok && ti < sch.n; ++ti) {
                const SkPiece pc = sch.at(ti, blockIdx.x, a.sk);
                if (ti > 0 && !mbar_wait(dempty, (ti - 1) & 1)) { ok = false; break; }
                tc_fence_after();
                for (int ks = pc.k0; ks < pc.k1 && ok; ++ks) {
                    const int as = ai % NA;
                    if (!mbar_wait(afull + 8 * as, (ai / NA) & 1) || aborted()) { ok = false; break; }
                    tc_fence_after();
                    for (int hh = 0; hh < 2; ++hh) {
                        const int xs = xi % NX;
                        if (!mbar_wait(xfull + 8 * xs, (xi / NX) & 1)) { ok = false; break; }
                        tc_fence_after();
#pragma unroll
                        for (int kk = 0; kk < 4; ++kk) {
                            const uint32_t a_tmem = tmem + kColA + as * 64 + hh * 32 + kk * 8;
                            const uint64_t bdesc = smem_desc_sw128(x_ring + xs * kXStage + kk * 32);
                            tc_mma_f16_ta(tmem + kColD, a_tmem, bdesc, kIdesc, (ks != pc.k0) | hh | kk);
                        }
                        tc_commit(xempty + 8 * xs);
                        ++xi;
                    }
                    tc_commit(aempty + 8 * as);
                    ++ai;
                }
                if (ok) tc_commit(dfull);
            }
            if (!ok) fail();
            // nothing may still be running on the tensor core when TMEM is freed
            tc_commit(drain);
            mbar_wait(drain, 0);
        }
    } else if (warp >= 8) {
        // ------------------------------------------------------ decoders
        const int q = warp & 3, h = (warp - 8) >> 2;
        const int r = 32 * q + lane;
        int wi = 0, ai = 0;
        for (int j = 0; j < sch.n; ++j) {
            const SkPiece pc = sch.at(j, blockIdx.x, a.sk);
            bool ok = true;
            for (int ks = pc.k0; ks < pc.k1; ++ks) {
                const int ws = wi % NW, as = ai % NA;
                if (!mbar_wait_all(wfull + 8 * ws, (wi / NW) & 1)) { ok = false; break; }
                if (__any_sync(0xFFFFFFFFu, aborted())) { ok = false; break; }
                const unsigned char *wst = sm + (w_ring - sbase) + ws * a.w_stage;
                uint32_t out[32];
                if (ks < a.ks_main)
                    decode_row64(wst, wst + S * GM * 16, S, r, h, out);
                else
                    decode_q8_row(wst, r, out);
                __syncwarp();
                if (lane == 0) mbar_arrive(wempty + 8 * ws);
                // the TMEM stage is needed only for the store: decode first, so
                // the decode overlaps the MMAs still reading this stage
                if (ai >= NA && !mbar_wait_all(aempty + 8 * as, ((ai / NA) - 1) & 1)) { ok = false; break; }
                tc_fence_after();
                tmem_st32(tmem + (static_cast<uint32_t>(32 * q) << 16) + kColA + as * 64 + h * 32, out);
                tmem_wait_st();
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(afull + 8 * as);
                ++wi;
                ++ai;
            }
            if (!ok) {
                if (lane == 0) fail();
                break;
            }
        }
    } else if (warp < 4) {
        // ------------------------------------------------------ epilogue
        const int q = warp;
        for (int ti = 0; ti < sch.n; ++ti) {
            const SkPiece pc = sch.at(ti, blockIdx.x, a.sk);
            if (!mbar_wait_all(dfull, ti & 1) || __any_sync(0xFFFFFFFFu, aborted())) {
                if (lane == 0) fail();
                break;
            }
            tc_fence_after();
            const int f0 = (pc.t / a.tiles_t) * GM, t0 = (pc.t % a.tiles_t) * TN;
            const int feat = f0 + 32 * q + lane;
            const uint32_t dcol = tmem + (static_cast<uint32_t>(32 * q) << 16) + kColD;
            if (pc.k0 == 0 && pc.k1 == a.sk.KS) {
                // the whole tile: Y directly
#pragma unroll 1
                for (int c = 0; c < TN / 32; ++c) {
                    uint32_t v[32];
                    tmem_ld32(dcol + c * 32, v);
                    tmem_wait_ld();
                    if (feat < a.N) {
#pragma unroll
                        for (int i = 0; i < 32; ++i) {
                            const int tok = t0 + c * 32 + i;
                            if (tok < a.M)
                                a.Y[static_cast<int64_t>(tok) * a.N + feat] = __uint_as_float(v[i]) * kInvSqrt8;
                        }
                    }
                }
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(dempty);
                continue;
            }
            // a piece of a split tile: its sum to this CTA's slot (sk_slot: the
            // first piece of the range in slot 0, a later one in slot 1)
            float *mine = a.part + (static_cast<int64_t>(blockIdx.x) * 2 + (ti == 0 ? 0 : 1)) * (GM * TN);
#pragma unroll 1
            for (int c = 0; c < TN / 32; ++c) {
                uint32_t v[32];
                tmem_ld32(dcol + c * 32, v);
                tmem_wait_ld();
#pragma unroll
                for (int i = 0; i < 32; ++i) __stcg(mine + (c * 32 + i) * GM + 32 * q + lane, __uint_as_float(v[i]));
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(dempty);
        }
    }

    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 5) tmem_dealloc(tmem, kTmemCols);
}

// Sum of the pieces of the tiles split by the stream-K schedule, in CTA
// order, into Y.  Block (c - 1, j) takes the tile that holds the boundary
// between CTAs c - 1 and c, if that boundary is the first inside it, and its
// 32-token chunk j: 256 threads, 4 features x 4 tokens each.
constexpr int kFixThreads = 256;

__global__ void __launch_bounds__(kFixThreads) k_gemm_fixup(const GemmArgs a, int TN) {
    // the partial tiles are written by the GEMM launched just before; the
    // next kernel may launch meanwhile
    pdl_launch_dependents();
    pdl_wait();
    const int c = blockIdx.x + 1;
    const int t = sk_fixup_tile(c, a.sk);
    if (t < 0) return;   // no split here, or not the first boundary inside the tile
    const int64_t ts = static_cast<int64_t>(t) * a.sk.KS;
    const int c_lo = sk_owner(ts, a.sk), c_hi = sk_owner(ts + a.sk.KS - 1, a.sk);
    const int f0 = (t / a.tiles_t) * GM, t0 = (t % a.tiles_t) * TN;
    const int fl = (threadIdx.x & 31) * 4, tl0 = blockIdx.y * 32 + (threadIdx.x >> 5) * 4;
    float4 acc[4];
#pragma unroll 1
    for (int cc = c_lo; cc <= c_hi; ++cc) {
        const float *src = a.part + (static_cast<int64_t>(cc) * 2 + sk_slot(cc, t, a.sk)) * (GM * TN);
        float4 v[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) v[i] = __ldcg(reinterpret_cast<const float4 *>(src + (tl0 + i) * GM + fl));
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            if (cc == c_lo) {
                acc[i] = v[i];
            } else {
                acc[i].x += v[i].x;
                acc[i].y += v[i].y;
                acc[i].z += v[i].z;
                acc[i].w += v[i].w;
            }
        }
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int tok = t0 + tl0 + i;
        if (tok >= a.M) break;
        float *yr = a.Y + static_cast<int64_t>(tok) * a.N + f0 + fl;
        const float o[4] = {acc[i].x, acc[i].y, acc[i].z, acc[i].w};
#pragma unroll
        for (int u = 0; u < 4; ++u)
            if (f0 + fl + u < a.N) yr[u] = o[u] * kInvSqrt8;
    }
}

// Activation pre-pass: X16[m][k] = fp16(x[m][k]) for k < K (0 for
// protected k and for K <= k < K_pad); for protected block bq and u < 64,
// X16[m][K_pad + 128 bq + u] = hi(v), X16[m][K_pad + 128 bq + 64 + u] = lo(v)
// with v = sqrt(8) * scale_{64bq+u} * x[m][j_{64bq+u}] (0 past p).
constexpr int kPrepThreads = 256;
constexpr int kPrepJobs = 4;   // 8-column groups per thread, their loads in flight together

__global__ void __launch_bounds__(kPrepThreads) k_gemm_prep(const uint16_t *__restrict__ X, int M, int K,
                                                            int K_pad, int K_ext, int p,
                                                            const int32_t *__restrict__ prot_idx,
                                                            const uint16_t *__restrict__ q8_scale,
                                                            uint16_t *__restrict__ X16, int *err) {
    extern __shared__ uint32_t s_mask[];   // K_pad / 32 words
    // the GEMM launched after this kernel may set itself up meanwhile; it
    // waits for this grid's completion before it reads X16
    pdl_launch_dependents();
    // launched as a programmatic dependent of the kernel before it (which
    // may write X, or still read the X16 of an earlier call): nothing is
    // read or written before that kernel has completed
    pdl_wait();
    const int groups = K_ext / 8;
    const int64_t njobs = static_cast<int64_t>(M) * groups;
    const int64_t base = static_cast<int64_t>(blockIdx.x) * kPrepThreads * kPrepJobs + threadIdx.x;
    // the plain columns' loads go out first; the protected-column mask is
    // built while they are in flight
    uint4 v[kPrepJobs];
#pragma unroll
    for (int i = 0; i < kPrepJobs; ++i) {
        const int64_t e = base + static_cast<int64_t>(i) * kPrepThreads;
        v[i] = make_uint4(0u, 0u, 0u, 0u);
        if (e < njobs) {
            const int m = static_cast<int>(e / groups), k = static_cast<int>(e % groups) * 8;
            if (k < K) v[i] = *reinterpret_cast<const uint4 *>(X + static_cast<int64_t>(m) * K + k);
        }
    }
    const int mw = K_pad / 32;
    for (int i = threadIdx.x; i < mw; i += blockDim.x) s_mask[i] = 0u;
    __syncthreads();
    for (int u = threadIdx.x; u < p; u += blockDim.x) {
        const int j = prot_idx[u];
        if (j < 0 || j >= K) {
            latch_error(err, BISCO_ERR_INVALID_ARG);   // not a column of this layer
            continue;
        }
        atomicOr(&s_mask[j >> 5], 1u << (j & 31));
    }
    __syncthreads();
#pragma unroll
    for (int i = 0; i < kPrepJobs; ++i) {
        const int64_t e = base + static_cast<int64_t>(i) * kPrepThreads;
        if (e >= njobs) break;
        const int m = static_cast<int>(e / groups), k = static_cast<int>(e % groups) * 8;
        uint32_t o[4] = {0u, 0u, 0u, 0u};
        if (k < K_pad) {
            if (k < K) {
                const uint32_t w[4] = {v[i].x, v[i].y, v[i].z, v[i].w};
                const uint32_t pm = (s_mask[k >> 5] >> (k & 31)) & 0xFFu;
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    const float lo = (pm >> (2 * q)) & 1u ? 0.f : __uint_as_float(w[q] << 16);
                    const float hi = (pm >> (2 * q + 1)) & 1u ? 0.f : __uint_as_float(w[q] & 0xFFFF0000u);
                    const __half2 h2 = __floats2half2_rn(lo, hi);
                    o[q] = *reinterpret_cast<const uint32_t *>(&h2);
                }
            }
        } else {
            // protected block bq, part hi (0) or lo (1): sqrt(8) * scale_u * x[m][j_u]
            const uint16_t *xr = X + static_cast<int64_t>(m) * K;
            const int e2 = k - K_pad, bq = e2 >> 7, part = (e2 >> 6) & 1, u0 = bq * 64 + (e2 & 63);
            uint16_t hv[8];
#pragma unroll
            for (int q = 0; q < 8; ++q) {
                const int u = u0 + q;
                float val = 0.f;
                const int j = u < p ? prot_idx[u] : -1;
                if (j >= 0 && j < K)
                    val = (__half2float(__ushort_as_half(q8_scale[u])) *
                           __uint_as_float(static_cast<uint32_t>(xr[j]) << 16)) * kSqrt8;
                const __half vh = __float2half_rn(val);
                hv[q] = part ? __half_as_ushort(__float2half_rn(val - __half2float(vh)))
                             : __half_as_ushort(vh);
            }
#pragma unroll
            for (int q = 0; q < 4; ++q) o[q] = hv[2 * q] | (static_cast<uint32_t>(hv[2 * q + 1]) << 16);
        }
        *reinterpret_cast<uint4 *>(X16 + static_cast<int64_t>(m) * K_ext + k) =
            make_uint4(o[0], o[1], o[2], o[3]);
    }
}

int k_pad_of(int K) { return (K + GK - 1) / GK * GK; }
int p_ext_of(int p) { return (p + 63) / 64 * 64; }
int k_ext_of(int K, int p) { return k_pad_of(K) + 2 * p_ext_of(p); }

// The tcgen05 path needs TMA-legal strides.  Up to 16 tokens the batch-16
// decode kernels are faster (one pass over the weights that feeds every
// token); from 17 on they need a second pass, while the stream-K split keeps
// every SM busy on the tensor cores even with one token tile.
bool tensor_path(const bisco_layer &L, int M) { return M > 16 && L.k_in % 128 == 0; }

// Token tile: 256 (the decode of a weight step feeds the most MMA work);
// 128 when M fits in it.  The stream-K split keeps every SM busy either way.
int tile_tokens(int M) { return M <= 128 ? 128 : GN; }

size_t round256(size_t b) { return (b + 255) / 256 * 256; }

// Workspace: [X16: M x K_ext fp16][partial tiles: kSkMaxCtas x 2 x TN x GM
// fp32], each part rounded up to 256 bytes.
struct GemmWs {
    size_t x16, part, total;
    int ntiles;
};
GemmWs gemm_ws(const bisco_layer &L, int M) {
    GemmWs w;
    const int TN = tile_tokens(M);
    w.ntiles = ((M + TN - 1) / TN) * ((L.n_out + GM - 1) / GM);
    w.x16 = 0;
    w.part = round256(static_cast<size_t>(M) * k_ext_of(L.k_in, L.n_protected) * 2);
    w.total = w.part + static_cast<size_t>(kSkMaxCtas) * 2 * GM * TN * 4;
    return w;
}

bisco_status gemm_via_gemv(const bisco_layer &L, const uint16_t *X, int M, float *Y, int *err,
                           cudaStream_t stream) {
    for (int m0 = 0; m0 < M; m0 += 16) {
        const int b = M - m0 < 16 ? M - m0 : 16;
        const bisco_status st = launch_gemv(L, X + static_cast<int64_t>(m0) * L.k_in, b,
                                            Y + static_cast<int64_t>(m0) * L.n_out, err, stream);
        if (st != BISCO_OK) return st;
    }
    return BISCO_OK;
}

template <int NX, int NW, int TN>
bisco_status launch_gemm_t(const CUtensorMap &mx, const CUtensorMap &mc, const CUtensorMap &mn,
                           const CUtensorMap &mq, const GemmArgs &a, int grid, cudaStream_t stream) {
    const size_t smem =
        1024 + NX * x_stage_bytes(TN) + NW * a.w_stage + 8 * (2 * NX + 2 * NW + 2 * NA + 3);
    if (smem > 227 * 1024) return BISCO_ERR_UNSUPPORTED;
    static size_t configured[64] = {};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return BISCO_ERR_CUDA;
    if (smem > configured[dev]) {
        if (cudaFuncSetAttribute(k_gemm<NX, NW, TN>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 static_cast<int>(smem)) != cudaSuccess)
            return BISCO_ERR_CUDA;
        configured[dev] = smem;
    }
    // programmatic dependent launch after the pre-pass: barrier set-up and
    // the TMEM allocation overlap it; the producer waits before its first copy
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid, 1, 1);
    cfg.blockDim = dim3(kThreads, 1, 1);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, k_gemm<NX, NW, TN>, mx, mc, mn, mq, a) == cudaSuccess
               ? BISCO_OK
               : BISCO_ERR_CUDA;
}

}  // namespace

size_t gemm_workspace_bytes(const bisco_layer &L, int M) {
    if (!tensor_path(L, M)) return 0;
    return gemm_ws(L, M).total;
}

bisco_status launch_gemm(const bisco_layer &L, const uint16_t *X, int M, float *Y,
                         void *workspace, size_t ws_bytes, int *err, cudaStream_t stream) {
    if (!tensor_path(L, M)) return gemm_via_gemv(L, X, M, Y, err, stream);
    const int N = L.n_out, K = L.k_in, S = L.stages, p = L.n_protected;
    const int K_pad = k_pad_of(K), K_ext = k_ext_of(K, p);
    const GemmWs wl = gemm_ws(L, M);
    if (ws_bytes < wl.total) return BISCO_ERR_INVALID_ARG;
    unsigned char *wsb = static_cast<unsigned char *>(workspace);
    uint16_t *X16 = reinterpret_cast<uint16_t *>(wsb + wl.x16);

    const size_t prep_smem = static_cast<size_t>(K_pad / 32) * 4;
    if (prep_smem > 48 * 1024) {
        static size_t configured[64] = {};
        int dev = 0;
        if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return BISCO_ERR_CUDA;
        if (prep_smem > configured[dev]) {
            if (cudaFuncSetAttribute(k_gemm_prep, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     static_cast<int>(prep_smem)) != cudaSuccess)
                return BISCO_ERR_CUDA;
            configured[dev] = prep_smem;
        }
    }
    const int64_t prep_jobs = static_cast<int64_t>(M) * (K_ext / 8);
    const int prep_grid = static_cast<int>((prep_jobs + kPrepThreads * kPrepJobs - 1) / (kPrepThreads * kPrepJobs));
    {
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3(prep_grid, 1, 1);
        cfg.blockDim = dim3(kPrepThreads, 1, 1);
        cfg.dynamicSmemBytes = prep_smem;
        cfg.stream = stream;
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attr[0].val.programmaticStreamSerializationAllowed = 1;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        if (cudaLaunchKernelEx(&cfg, k_gemm_prep, X, M, K, K_pad, K_ext, p, L.prot_idx, L.q8_scale, X16,
                               err) != cudaSuccess)
            return BISCO_ERR_CUDA;
    }

    const int TN = tile_tokens(M);
    CUtensorMap mx, mc, mn, mq;
    {
        const uint64_t dims[2] = {static_cast<uint64_t>(K_ext), static_cast<uint64_t>(M)};
        const uint64_t strides[1] = {static_cast<uint64_t>(K_ext) * 2};
        const uint32_t box[2] = {64, static_cast<uint32_t>(TN)};
        if (!encode_tensor_map(&mx, CU_TENSOR_MAP_DATA_TYPE_UINT16, 2, X16, dims, strides, box,
                               CU_TENSOR_MAP_SWIZZLE_128B))
            return BISCO_ERR_CUDA;
    }
    {
        const uint64_t dims[3] = {static_cast<uint64_t>(K / 8), static_cast<uint64_t>(N),
                                  static_cast<uint64_t>(S)};
        const uint64_t cs[2] = {static_cast<uint64_t>(K / 8), static_cast<uint64_t>(N) * (K / 8)};
        const uint64_t ns[2] = {static_cast<uint64_t>(K / 4), static_cast<uint64_t>(N) * (K / 4)};
        const uint32_t box[3] = {GK / 8, GM, static_cast<uint32_t>(S)};
        if (!encode_tensor_map(&mc, CU_TENSOR_MAP_DATA_TYPE_UINT8, 3, L.codes, dims, cs, box,
                               CU_TENSOR_MAP_SWIZZLE_NONE) ||
            !encode_tensor_map(&mn, CU_TENSOR_MAP_DATA_TYPE_UINT16, 3, L.norms, dims, ns, box,
                               CU_TENSOR_MAP_SWIZZLE_NONE))
            return BISCO_ERR_CUDA;
    }
    if (p > 0) {
        const int p_pad = (p + 15) / 16 * 16;
        const uint64_t dims[2] = {static_cast<uint64_t>(p_pad), static_cast<uint64_t>(N)};
        const uint64_t strides[1] = {static_cast<uint64_t>(p_pad)};
        const uint32_t box[2] = {64, GM};
        if (!encode_tensor_map(&mq, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, L.q8, dims, strides, box,
                               CU_TENSOR_MAP_SWIZZLE_NONE))
            return BISCO_ERR_CUDA;
    } else {
        mq = mc;   // never dereferenced when p == 0
    }

    GemmArgs a = {};
    a.Y = Y;
    a.err = err;
    a.part = reinterpret_cast<float *>(wsb + wl.part);
    a.M = M;
    a.N = N;
    a.S = S;
    a.ks_main = K_pad / GK;
    a.ks_ext = p_ext_of(p) / 64;
    a.tiles_t = (M + TN - 1) / TN;
    a.sk = sk_plan(wl.ntiles, a.ks_main + a.ks_ext, num_sms());
    a.w_stage = static_cast<uint32_t>(S * GM * 48 > GM * 64 ? S * GM * 48 : GM * 64);
    const int grid = a.sk.G;
    // 256 tokens: S = 1: 6 x 32 KB + 3 x 8 KB; S = 2, 3: 5 x 32 KB + 3 x 12/18 KB;
    // 128 tokens: 8 x 16 KB + 3 x 8/12/18 KB (all <= 227 KB)
    bisco_status st;
    if (TN == 128) st = launch_gemm_t<8, 3, 128>(mx, mc, mn, mq, a, grid, stream);
    else if (S == 1) st = launch_gemm_t<6, 3, GN>(mx, mc, mn, mq, a, grid, stream);
    else st = launch_gemm_t<5, 3, GN>(mx, mc, mn, mq, a, grid, stream);
    if (st != BISCO_OK || a.sk.whole || a.sk.G < 2) return st;
    // the split tiles, summed once the GEMM is done (programmatic dependent
    // launch: its set-up overlaps the GEMM's last CTAs)
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(a.sk.G - 1, TN / 32, 1);
    cfg.blockDim = dim3(kFixThreads, 1, 1);
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, k_gemm_fixup, a, TN) == cudaSuccess ? BISCO_OK : BISCO_ERR_CUDA;
}

}  // namespace bisco
