// gemv_b1.cu -- batch-1 decode-time y = What x straight from the coded
// layer (Sec. III-G Eq. 12 with Eq. 10's protected columns) for G <= 4
// layers that share x and have K a multiple of 4096 (every Qwen3-8B
// projection); optionally with each layer's low-rank compensation
// (Sec. III-F) in the same launch.
//
// Work split.  The CTAs of the grid are shared out among the G layers so
// that the longest row run per CTA is as short as it can be (q/k/v of
// Qwen3-8B: 102/25/25 CTAs of 40-41 rows); each CTA takes a contiguous run
// of one layer's rows.  A launch with at least kB1TwoPerSm items per SM runs
// two of its own CTAs per SM, others one.  A row's work is S * K/4096 items,
// one per (stage, 4096-column span): 512 sign bytes and 512 fp16 norms,
// 1536 bytes.  A CTA orders its items span by span, then stage by stage and
// row by row (within a span and stage, consecutive rows are consecutive in
// memory), and each of its 16 warps takes the same contiguous run of every
// span.
//
// Data path.  Every warp owns a ring of `depth` one-item slots in shared
// memory.  Lane 0 fills a slot with two 1-D bulk copies (cp.async.bulk:
// 512 B of signs, 1 KB of norms) that complete on the slot's mbarrier, and
// refills it with the item `depth` further on as soon as the warp has read
// it into registers, before decoding it.  The first `depth` items of every
// warp are requested before the wait on the previous kernel, and a CTA
// takes at most the shared memory at which two CTAs share an SM, so the
// next call's CTAs request theirs while this one finishes.
//
// Decode (Eq. 12 per chunk-stage): for a sign byte b of chunk c the signed
// sum of the chunk's 8 activations is T_lo(c, b & 15) + T_hi(c, b >> 4),
// where T_lo(c, v) = sum_{e<4} (bit e of v ? -x[8c+e] : x[8c+e]) and T_hi the
// same over x[8c+4..8c+7].  Each is rounded once to fp16 (2^-11 relative),
// held as one fp16 pair (T_lo, T_hi) per (c, v), and meets the chunk's fp16
// norm in an fp16 x fp16 -> fp32 FMA (exact product).  The layer's protected
// columns are zero in its tables, which is Eq. 10's overwrite of their BSQ
// value; the 1/sqrt(8) of Eq. 3 is applied once per output.  A CTA holds
// the table of one span at a time (32 KB) and rebuilds it between spans.
//
// Table placement.  Lane l of an item handles chunks 8l+j (j = 0..7) of each
// 256-chunk half h of its span; chunk c = 512*span + 256*h + 8l + j sits at
// position P = 256*h + 32*j + l of the span's table, and entry (P, v) at
// byte
//   (P >> 6) * 4096 + v * 256 + (P & 63) * 4,
// so a lane's lookups always hit bank l.  With the table 4 KB aligned, the
// lane's base address has bits 8..11 clear and the lookup address is one
// shift and one LOP3 ((w >> s) & 0xF00 | base) plus a compile-time offset.
//
// Outputs.  The lane sums of a ring pass's items are added across the warp
// (fixed shuffle order) into one float per item.  A warp that has decoded
// its items computes the protected term sum_u value(q[r][u]) * (scale_u *
// x[idx_u]) of its share of the rows (int8, FP8 E4M3 / E5M2 or bf16
// payloads; staged in shared memory before the wait where they fit) while
// the others may still decode; after one CTA barrier a thread per row adds
// the row's items in item order, scales by 1/sqrt(8) and adds the protected
// term (and the compensation).  No atomics: the result depends only on the
// sizes.
#include <cuda_runtime.h>
#include <stdint.h>
#include <stdlib.h>

#include <type_traits>

#include "bisco_dev.cuh"
#include "bisco_host.h"
#include "fp8.cuh"

namespace bisco {
namespace {

constexpr int kB1Span = 512;                  // chunks per item
constexpr uint32_t kB1Item = 1536;            // bytes per item slot: signs, then norms
constexpr int kB1MaxG = 4;                    // layers per launch
constexpr float kB1InvSqrt8 = 0.35355339059327373f;
// kernel instances by the protected set's kind (see k_gemv_b1)
constexpr int kB1Int8 = 0, kB1Fmt = 1, kB1Rows = 2, kB1Tab = 3, kB1Lora = 4;
// dynamic shared memory of one CTA at most (227 KB per block less the
// kernel's static shared memory, rounded down)
constexpr size_t kB1MaxSmem = 226 * 1024;
// A launch with at least this many items per SM runs two of its own CTAs per
// SM: twice the copies in flight and twice the decoding warps outweigh the
// lost overlap with the neighbouring launches (for 2 x 12288 x 4096 at S = 2,
// 323 items per SM: 22.1 -> 18.6 us).
constexpr int kB1TwoPerSm = 256;

struct B1Layer {
    const uint8_t *codes;      // [S][N][K/8]
    const uint16_t *norms;     // [S][N][K/8] fp16
    const int8_t *q8;          // [N][p_pad] elements of the protected format
    const uint16_t *q8_scale;  // [p] fp16
    const int32_t *prot_idx;   // [p]
    float *y;                  // [N]
    const uint16_t *la;        // low-rank compensation: A [rank][K] bf16
    const uint16_t *lb;        //                        Bm [N][rank] bf16
    int rank;                  // 0: none
    float lscale;
    int N, p, p_pad;
    int fmt;                   // BISCO_PROT_*: int8, FP8 E4M3 / E5M2 or bf16 payload
    int prow;                  // payload bytes per row: p_pad elements of 1 or 2 bytes
    int axis;                  // 1: the protected channels are output rows (payload
                               // [p][kp], kp = roundup(K, 16) elements a row)
    int cta0, ctas;            // the CTAs of the grid that take this layer's rows
};

struct B1Args {
    B1Layer L[kB1MaxG];
    const uint16_t *x;
    const uint16_t *tab;       // decoder tables [S][256][8] fp16 (table mode), else null
    int *err;
    int K, G;
    int nspan;                 // K / 4096
    int S;                     // stages
    int depth;                 // item slots per warp
    int q8_staged;             // payload rows in shared memory (else read at the end)
    uint32_t sleep_ns;         // suspend-time hint of the item waits
    int withhold;              // test of the bounded waits: request no copies
    int lrank;                 // the largest compensation rank of the launch (0: none)
    uint32_t off_ring, off_pm, off_pidx, off_sx, off_part, off_prot, off_lt, off_q8, off_bar;   // table at 0
};

template <uint32_t A>
__device__ __forceinline__ unsigned char *align_smem(unsigned char *raw) {
    return raw + ((A - (smem_u32(raw) & (A - 1u))) & (A - 1u));
}

__device__ __forceinline__ uint4 lds_u128(uint32_t addr) {
    uint4 v;
    asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(addr));
    return v;
}

// (w >> sh) for sh >= 0, (w << -sh) otherwise (sh a compile-time constant)
template <int SH>
__device__ __forceinline__ uint32_t shift_by(uint32_t w) {
    if constexpr (SH >= 0) return w >> SH;
    else return w << (-SH);
}

// Lane sums of one item: 16 chunks (8 per half) through the tables at base0.
__device__ __forceinline__ float b1_item(const uint2 (&cw)[2], const uint4 (&nw)[2], uint32_t base0) {
    float acc4[2][2] = {{0.f, 0.f}, {0.f, 0.f}};   // four short FMA chains, one per word
#pragma unroll
    for (int h = 0; h < 2; ++h) {
#pragma unroll
        for (int jw = 0; jw < 2; ++jw) {
            const uint32_t w = jw ? cw[h].y : cw[h].x;
            const uint32_t n01 = jw ? nw[h].z : nw[h].x;
            const uint32_t n23 = jw ? nw[h].w : nw[h].y;
            uint32_t lo[4], hi[4];
            // v << 8 for the low and high nibble of byte jj: bits 8jj.. and 8jj+4..
            lo[0] = lop3_and_or(shift_by<-8>(w), 0xF00u, base0);
            lo[1] = lop3_and_or(w, 0xF00u, base0);
            lo[2] = lop3_and_or(shift_by<8>(w), 0xF00u, base0);
            lo[3] = lop3_and_or(shift_by<16>(w), 0xF00u, base0);
            hi[0] = lop3_and_or(shift_by<-4>(w), 0xF00u, base0);
            hi[1] = lop3_and_or(shift_by<4>(w), 0xF00u, base0);
            hi[2] = lop3_and_or(shift_by<12>(w), 0xF00u, base0);
            hi[3] = lop3_and_or(shift_by<20>(w), 0xF00u, base0);
            uint32_t tl[4], th[4];
#pragma unroll
            for (int jj = 0; jj < 4; ++jj) {
                const int j = 4 * jw + jj;
                const uint32_t off = h * 16384u + (j >> 1) * 4096u + (j & 1) * 128u;
                tl[jj] = lds_u32(lo[jj] + off);
                th[jj] = lds_u32(hi[jj] + off);
            }
            float &acc = acc4[h][jw];
#pragma unroll
            for (int jj = 0; jj < 4; ++jj) {
                const uint32_t nn = jj < 2 ? n01 : n23;
                const uint16_t n = (jj & 1) ? hi_half(nn) : lo_half(nn);
                acc = fma_f16_f32(lo_half(tl[jj]), n, acc);
                acc = fma_f16_f32(hi_half(th[jj]), n, acc);
            }
        }
    }
    return (acc4[0][0] + acc4[0][1]) + (acc4[1][0] + acc4[1][1]);
}

// Lane 0 of the warp requests one item into a ring slot: after a proxy fence
// (the warp's reads of the slot are done) it arms the slot's mbarrier for
// 1536 bytes and issues the two bulk copies (signs to the slot, norms 512
// bytes on); the other lanes run the same instructions with the predicate
// off, so the warp never diverges.
__device__ __forceinline__ void b1_request(uint32_t lead, uint32_t slot, uint32_t bar, const void *csrc,
                                           const void *nsrc, uint64_t pol) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.u32 p, %0, 0;\n\t"
        "@p fence.proxy.async.shared::cta;\n\t"
        "@p mbarrier.arrive.expect_tx.release.cta.shared::cta.b64 _, [%2], 1536;\n\t"
        "@p cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint"
        " [%1], [%3], 512, [%2], %5;\n\t"
        "@p cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint"
        " [%6], [%4], 1024, [%2], %5;\n\t}"
        ::"r"(lead), "r"(slot), "r"(bar), "l"(csrc), "l"(nsrc), "l"(pol), "r"(slot + 512u)
        : "memory");
}

// The table of one 4096-column span (32 KB): job J (of 16) of a warp,
// lane l: chunk 256*h + 8l + j of the span, h = J >> 3 & 1,
// j = J & 7, from its 8 activations xv (bf16, the span's column base c0)
// with the layer's protected columns (bits of pm) zeroed.
__device__ __forceinline__ void b1_table_job(uint32_t tab, const uint32_t *pm, int c0, int J, int lane,
                                             uint4 xv) {
    const int h = (J >> 3) & 1, j = J & 7;
    const int c = c0 + h * 256 + 8 * lane + j;   // chunk of the layer
    const uint32_t m = (pm[c >> 2] >> ((c & 3) * 8)) & 0xFFu;
    float e[8] = {__uint_as_float(xv.x << 16), __uint_as_float(xv.x & 0xFFFF0000u),
                  __uint_as_float(xv.y << 16), __uint_as_float(xv.y & 0xFFFF0000u),
                  __uint_as_float(xv.z << 16), __uint_as_float(xv.z & 0xFFFF0000u),
                  __uint_as_float(xv.w << 16), __uint_as_float(xv.w & 0xFFFF0000u)};
#pragma unroll
    for (int k = 0; k < 8; ++k)
        if ((m >> k) & 1u) e[k] = 0.f;
    // signed sums of element pairs: index bit 0 negates the first, bit 1 the second
    float p01[2][4], p23[2][4];
#pragma unroll
    for (int hh = 0; hh < 2; ++hh) {
        const float x0 = e[4 * hh], x1 = e[4 * hh + 1], x2 = e[4 * hh + 2], x3 = e[4 * hh + 3];
        p01[hh][0] = x0 + x1; p01[hh][1] = x1 - x0; p01[hh][2] = x0 - x1; p01[hh][3] = -(x0 + x1);
        p23[hh][0] = x2 + x3; p23[hh][1] = x3 - x2; p23[hh][2] = x2 - x3; p23[hh][3] = -(x2 + x3);
    }
    const int P = h * 256 + 32 * j + lane;
    const uint32_t dst = tab + static_cast<uint32_t>((P >> 6) * 4096 + (P & 63) * 4);
#pragma unroll
    for (int v = 0; v < 16; ++v) {
        const __half2 hv = __floats2half2_rn(p01[0][v & 3] + p23[0][v >> 2], p01[1][v & 3] + p23[1][v >> 2]);
        asm volatile("st.shared.b32 [%0], %1;" ::"r"(dst + v * 256), "r"(*reinterpret_cast<const uint32_t *>(&hv)));
    }
}

// Sums of four values over the warp with six shuffles: the values are folded
// in halves (lanes with bit 4 set keep c, d; with bit 3 set, the second of
// their pair), then added over the remaining eight lanes.  Every lane returns
// the total of value lane >> 3 (a, b, c, d); the order of the additions is
// fixed.
__device__ __forceinline__ float warp_sum4(float a, float b, float c, float d, int lane) {
    const bool h4 = (lane & 16) != 0, h3 = (lane & 8) != 0;
    const float r0 = __shfl_xor_sync(0xFFFFFFFFu, h4 ? a : c, 16);
    const float r1 = __shfl_xor_sync(0xFFFFFFFFu, h4 ? b : d, 16);
    const float k0 = (h4 ? c : a) + r0, k1 = (h4 ? d : b) + r1;
    float k = (h3 ? k1 : k0) + __shfl_xor_sync(0xFFFFFFFFu, h3 ? k0 : k1, 8);
    k += __shfl_xor_sync(0xFFFFFFFFu, k, 4);
    k += __shfl_xor_sync(0xFFFFFFFFu, k, 2);
    k += __shfl_xor_sync(0xFFFFFFFFu, k, 1);
    return k;
}

// x of job J's chunk in span sp (see b1_table_job).
__device__ __forceinline__ uint4 b1_table_x(const uint16_t *x, int sp, int J, int lane) {
    const int c = sp * kB1Span + ((J >> 3) & 1) * 256 + 8 * lane + (J & 7);
    return *reinterpret_cast<const uint4 *>(x + 8 * c);
}

// Table mode (the learned decoder step, Eq. 1 with Eq. 12): a chunk of
// stage s with code byte v decodes to n * T_s[v][0..7], so its term is
// n * sum_k T_s[v][k] x[8c+k].  The span's activations (protected columns
// zeroed, fp16) sit at position P = 256h + 32j + l of a 16-byte-per-chunk
// buffer, so lane l's loads hit consecutive words; the S decoder tables
// (4 KB each) follow it.
constexpr uint32_t kB1TabOff = 8192;   // the tables' offset in the table region

// Job J of the span's activation buffer (see b1_table_job for J and lane):
// chunk c = c0 + 256h + 8l + j, its 8 activations with the layer's
// protected columns zeroed, as fp16, at position 256h + 32j + l.
__device__ __forceinline__ void b1_xspan_job(uint32_t xs, const uint32_t *pm, int c0, int J, int lane,
                                             uint4 xv) {
    const int h = (J >> 3) & 1, j = J & 7;
    const int c = c0 + h * 256 + 8 * lane + j;
    const uint32_t m = (pm[c >> 2] >> ((c & 3) * 8)) & 0xFFu;
    const uint32_t w[4] = {xv.x, xv.y, xv.z, xv.w};
    uint32_t o[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        const float lo = (m >> (2 * q)) & 1u ? 0.f : __uint_as_float(w[q] << 16);
        const float hi = (m >> (2 * q + 1)) & 1u ? 0.f : __uint_as_float(w[q] & 0xFFFF0000u);
        const __half2 hv = __floats2half2_rn(lo, hi);
        o[q] = *reinterpret_cast<const uint32_t *>(&hv);
    }
    const uint32_t dst = xs + static_cast<uint32_t>((h * 256 + 32 * j + lane) * 16);
    asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(dst), "r"(o[0]), "r"(o[1]), "r"(o[2]), "r"(o[3]));
}

// Lane sums of one item in table mode: chunks 8l + j of each half through
// the stage's table at tb and the activations at xs_lane (the buffer plus
// 16 * lane).  fp16 x fp16 products are exact in fp32.
__device__ __forceinline__ float b1_item_tab(const uint2 (&cw)[2], const uint4 (&nw)[2], uint32_t xs_lane,
                                             uint32_t tb) {
    float acc4[2][2] = {{0.f, 0.f}, {0.f, 0.f}};
#pragma unroll
    for (int h = 0; h < 2; ++h) {
#pragma unroll
        for (int jw = 0; jw < 2; ++jw) {
            const uint32_t w = jw ? cw[h].y : cw[h].x;
            const uint32_t n01 = jw ? nw[h].z : nw[h].x;
            const uint32_t n23 = jw ? nw[h].w : nw[h].y;
            float &acc = acc4[h][jw];
            // (unrolled by two: fully unrolled, the kernel spills)
#pragma unroll 2
            for (int jj = 0; jj < 4; ++jj) {
                const int j = 4 * jw + jj;
                const uint32_t v = (w >> (8 * jj)) & 0xFFu;
                const uint4 t = lds_u128(tb + v * 16u);
                const uint4 xx = lds_u128(xs_lane + static_cast<uint32_t>((h * 256 + 32 * j) * 16));
                const uint32_t tw[4] = {t.x, t.y, t.z, t.w}, xw[4] = {xx.x, xx.y, xx.z, xx.w};
                float d = 0.f;
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    d = fma_f16_f32(lo_half(tw[q]), lo_half(xw[q]), d);
                    d = fma_f16_f32(hi_half(tw[q]), hi_half(xw[q]), d);
                }
                const uint32_t nn = jj < 2 ? n01 : n23;
                const uint16_t n = (jj & 1) ? hi_half(nn) : lo_half(nn);
                acc = fmaf(__half2float(__ushort_as_half(n)), d, acc);
            }
        }
    }
    return (acc4[0][0] + acc4[0][1]) + (acc4[1][0] + acc4[1][1]);
}

// NW warps; D ring slots (one item each) per warp; NSPAN 4096-column spans
// per row (0: a.nspan > 1, at run time).  With one span, every ring address
// is an immediate offset; with several, a CTA holds the table of one span at
// a time and walks its items span by span, rebuilding the table between
// spans (x of the next span is loaded while the current one is decoded).
// MODE: the protected set's kind, one instance each -- kB1Int8 (int8
// columns, the common case), kB1Fmt (columns in any payload format: the
// FP8 / bf16 conversions compiled in), kB1Rows (output rows in any format)
// or kB1Tab (table mode: the decoder tables of a.tab instead of the sign
// decode; one layer, int8 columns), or kB1Lora (int8 columns with each
// layer's low-rank compensation).
template <int NW, int D, int NSPAN, int MODE>
__global__ void __launch_bounds__(NW * 32, 2) k_gemv_b1(const __grid_constant__ B1Args a) {
    static_assert(D <= 4, "one folded reduction covers a ring pass");
    constexpr int kThreads = NW * 32;
    extern __shared__ unsigned char smem_raw[];
    unsigned char *sm = align_smem<4096>(smem_raw);
    const uint32_t sbase = smem_u32(sm);
    __shared__ int s_abort, s_lnext, s_r0, s_r1;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int K = a.K, C = K / 8, nspan = NSPAN ? NSPAN : a.nspan, S = a.S;
    // this CTA's layer and rows [ra, ra + nrows)
    int g = 0;
#pragma unroll
    for (int i = 1; i < kB1MaxG; ++i)
        if (i < a.G && static_cast<int>(blockIdx.x) >= a.L[i].cta0) g = i;
    const B1Layer &L = a.L[g];
    const int N = L.N, prow = L.prow, fmt = L.fmt;
    // protected input columns (Eq. 10) or, with axis 1, output rows (Eq. 9;
    // taken by the FMT instances only)
    constexpr bool FMT = MODE == kB1Fmt || MODE == kB1Rows, ROWS = MODE == kB1Rows,
                   TAB = MODE == kB1Tab, LORA = MODE == kB1Lora;
    const int lrank = LORA ? L.rank : 0;   // the compensation's rank (0: none)
    const int p = ROWS ? 0 : L.p, prows = ROWS ? L.p : 0;
    const int ci = static_cast<int>(blockIdx.x) - L.cta0;
    const int ra = static_cast<int>(static_cast<int64_t>(N) * ci / L.ctas);
    const int rb = static_cast<int>(static_cast<int64_t>(N) * (ci + 1) / L.ctas);
    const int nrows = rb - ra;
    const uint8_t *const codes = L.codes;
    const uint16_t *const norms = L.norms;
    const int8_t *const q8 = L.q8;
    float *const y = L.y;

    uint32_t *pm = reinterpret_cast<uint32_t *>(sm + a.off_pm);   // protected bits, 32 columns a word
    int *spidx = reinterpret_cast<int *>(sm + a.off_pidx);        // [p]
    float *ssc = reinterpret_cast<float *>(spidx + (p + 3) / 4 * 4);
    float *sx = reinterpret_cast<float *>(sm + a.off_sx);         // scale * x [p]
    float *part = reinterpret_cast<float *>(sm + a.off_part);     // [S * nrows * nspan]
    float *prot = reinterpret_cast<float *>(sm + a.off_prot);     // protected term [nrows]
    int8_t *q8s = reinterpret_cast<int8_t *>(sm + a.off_q8);
    const uint64_t pol = l2_evict_first_policy();

    // Items, span by span; within a span stage by stage, row by row (the
    // order of the [S][N][K/8] buffers for one span).  Every warp takes the
    // same contiguous run [kb0, kb0 + cnt0) of each span's S * nrows items.
    const int per_span = S * nrows;
    const int kb0 = per_span * warp / NW;
    const int cnt0 = per_span * (warp + 1) / NW - kb0;
    const int total = cnt0 * nspan;   // this warp's items
    const uint32_t wring = sbase + a.off_ring + static_cast<uint32_t>(warp * D) * kB1Item;
    const uint32_t wbar = sbase + a.off_bar + static_cast<uint32_t>(warp * D) * 8u;
    // request cursor (uniform over the warp): byte offset of the next item's
    // signs in codes (its norms at twice that in norms; below 2^32, checked
    // on the host), items left in its row run (at the end of a run the next
    // stage's rows follow, N - nrows rows on) and in its span's run
    const int s0 = nrows > 0 ? kb0 / nrows : 0, r0 = kb0 - s0 * nrows;
    const uint32_t off0 = (static_cast<uint32_t>(s0) * N + ra + r0) * static_cast<uint32_t>(C);
    const uint32_t gap = static_cast<uint32_t>(N - nrows) * C;
    uint32_t off = off0;
    int rleft = nrows - r0, cleft = cnt0, csp = 0;
    const uint32_t lead = lane == 0;
    const unsigned char *const nbytes = reinterpret_cast<const unsigned char *>(norms);
    // items still to request (withheld: none, every wait runs out with
    // nothing in flight)
    const int to_request = a.withhold ? 0 : total;
    int left = to_request;
    auto fill = [&](int d) {
        b1_request(lead, wring + d * kB1Item, wbar + d * 8u, codes + off, nbytes + 2ull * off, pol);
        --left;
        off += C;
        if (--rleft == 0) {
            off += gap;
            rleft = nrows;
        }
        if constexpr (NSPAN != 1) {
            if (--cleft == 0) {
                ++csp;
                off = off0 + static_cast<uint32_t>(csp) * kB1Span;
                rleft = nrows - r0;
                cleft = cnt0;
            }
        }
    };

    // ---- before the wait: barriers, first items, protected metadata, int8 rows
    if (lane == 0) {
        for (int d = 0; d < D; ++d) mbar_init(wbar + 8 * d, 1);
        fence_mbar_init();
    }
    __syncwarp();
#pragma unroll
    for (int d = 0; d < D; ++d)
        if (left > 0) fill(d);
    if (threadIdx.x == 0) {
        s_abort = 0;
        s_lnext = 0;
        // protected output rows of this CTA: [s_r0, s_r1) of the ascending list
        int t0 = 0, t1 = 0;
        if (ROWS && prows > 0) {
            int lo = 0, hi = prows;
            while (lo < hi) {
                const int mid = (lo + hi) >> 1;
                if (L.prot_idx[mid] < ra) lo = mid + 1;
                else hi = mid;
            }
            t0 = lo;
            hi = prows;
            while (lo < hi) {
                const int mid = (lo + hi) >> 1;
                if (L.prot_idx[mid] < rb) lo = mid + 1;
                else hi = mid;
            }
            t1 = lo;
        }
        s_r0 = t0;
        s_r1 = t1;
    }
    if (ROWS && prows > 0)
        for (int rr = threadIdx.x; rr < nrows; rr += kThreads) prot[rr] = 0.f;
    for (int i = threadIdx.x; i < C / 4; i += kThreads) pm[i] = 0u;
    __syncthreads();
    for (int u = threadIdx.x; u < p; u += kThreads) {
        int j = L.prot_idx[u];
        float sc = __half2float(__ushort_as_half(L.q8_scale[u]));
        if (j < 0 || j >= K) {   // not a valid layer: reported, and the entry dropped
            latch_error(a.err, BISCO_ERR_INVALID_ARG);
            j = -1;
            sc = 0.f;
        } else {
            atomicOr(&pm[j >> 5], 1u << (j & 31));
        }
        spidx[u] = j;
        ssc[u] = sc;
    }
    // x into L2 now (a prefetch moves no data into the CTA, so it is safe
    // ahead of the wait on a kernel that may still be writing x); read after
    if (threadIdx.x == 32) prefetch_l2(a.x, static_cast<uint32_t>(K) * 2u);
    // the compensation's weights into L2 as well: this CTA's share of A
    // (every CTA of the layer reads all of it) and Bm's rows of its rows
    if (lrank > 0 && threadIdx.x == 64) {
        const uint32_t abytes = static_cast<uint32_t>(lrank) * K * 2u;
        const uint32_t share = (abytes / L.ctas + 15u) / 16u * 16u;
        const uint32_t b0 = share * static_cast<uint32_t>(ci);
        if (b0 < abytes)
            prefetch_l2(reinterpret_cast<const unsigned char *>(L.la) + b0, min(share, abytes - b0));
        if (nrows > 0)
            prefetch_l2(L.lb + static_cast<size_t>(ra) * lrank, static_cast<uint32_t>(nrows * lrank) * 2u);
    }
    if (p > 0 && nrows > 0) {
        if (a.q8_staged) {
            const int n16 = nrows * prow / 16;
            const uint4 *src = reinterpret_cast<const uint4 *>(q8 + static_cast<int64_t>(ra) * prow);
            for (int i = threadIdx.x; i < n16; i += kThreads) reinterpret_cast<uint4 *>(q8s)[i] = src[i];
        } else if (threadIdx.x == 0) {
            // read at the end from global memory: into L2 now
            prefetch_l2(q8 + static_cast<int64_t>(ra) * prow, static_cast<uint32_t>(nrows * prow));
        }
    }
    __syncthreads();
    pdl_launch_dependents();

    // ---- after the wait: the first span's table, scale * x.  The x of this
    // thread's protected column and of its table jobs share one round trip.
    pdl_wait();
    const int uj = threadIdx.x < p ? spidx[threadIdx.x] : -1;
    const uint16_t xj = uj >= 0 ? a.x[uj] : static_cast<uint16_t>(0);
    {
        uint4 xv[(16 + NW - 1) / NW];
#pragma unroll
        for (int q = 0; q < (16 + NW - 1) / NW; ++q)
            if (warp + q * NW < 16) xv[q] = b1_table_x(a.x, 0, warp + q * NW, lane);
        if constexpr (TAB) {
            // the decoder tables, S x 4 KB, beside the activation buffer
            for (int q = threadIdx.x; q < S * 256; q += kThreads) {
                const uint4 t = reinterpret_cast<const uint4 *>(a.tab)[q];
                asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(sbase + kB1TabOff + q * 16u),
                             "r"(t.x), "r"(t.y), "r"(t.z), "r"(t.w));
            }
        }
#pragma unroll
        for (int q = 0; q < (16 + NW - 1) / NW; ++q)
            if (warp + q * NW < 16) {
                if constexpr (TAB)
                    b1_xspan_job(sbase, pm, 0, warp + q * NW, lane, xv[q]);
                else
                    b1_table_job(sbase, pm, 0, warp + q * NW, lane, xv[q]);
            }
    }
    if (threadIdx.x < p) sx[threadIdx.x] = uj >= 0 ? ssc[threadIdx.x] * bf16_bits_to_f32(xj) : 0.f;
    for (int u = threadIdx.x + kThreads; u < p; u += kThreads) {
        const int j = spidx[u];
        sx[u] = j >= 0 ? ssc[u] * bf16_bits_to_f32(a.x[j]) : 0.f;
    }
    __syncthreads();

    const uint32_t base0 = sbase + lane * 4u;
    // table mode: this lane's activation words, and the stage and the items
    // left in the row run of the next item to decode (the consumer's walk of
    // the same run the requests take)
    const uint32_t xs_lane = sbase + lane * 16u;
    int tst = s0, trl = nrows - r0;
    int i = 0;   // items consumed
    // slot d: wait for it, decode its item into this lane's partial sum,
    // request the next item into it; false on a timeout
    auto slot_item = [&](int d, uint32_t phase, float &v) -> bool {
        const uint32_t slot = wring + d * kB1Item, bar = wbar + d * 8u;
        if (!__all_sync(0xFFFFFFFFu, mbar_try_wait(bar, phase)) &&
            !__all_sync(0xFFFFFFFFu, mbar_wait_sleep(bar, phase, a.sleep_ns))) {
            if (lane == 0) {
                latch_error(a.err, BISCO_ERR_TIMEOUT);
                atomicExch(&s_abort, 1);
            }
            return false;
        }
        uint2 cw[2];
        uint4 nw[2];
        cw[0] = lds_u64(slot + lane * 8u);
        cw[1] = lds_u64(slot + 256u + lane * 8u);
        nw[0] = lds_u128(slot + 512u + lane * 16u);
        nw[1] = lds_u128(slot + 1024u + lane * 16u);
        // the slot's reads are done (the values are in registers, ordered
        // before the refill by the warp barrier and the proxy fence): refill
        // it before the decode, so the copy's latency overlaps the decode
        __syncwarp();
        if (left > 0) fill(d);
        if constexpr (TAB) {
            // this item's stage: the consumer's own walk of the run
            v = b1_item_tab(cw, nw, xs_lane, sbase + kB1TabOff + static_cast<uint32_t>(tst) * 4096u);
            if (--trl == 0) {
                ++tst;
                trl = nrows;
            }
        } else {
            v = b1_item(cw, nw, base0);
        }
        return true;
    };
    if constexpr (NSPAN == 1) {
        // ---- decode: D items a pass; their partial sums are added over the
        // warp together
        uint32_t phase = 0;
        for (int i0 = 0; i0 < total; i0 += D, phase ^= 1u) {
            float v[4] = {0.f, 0.f, 0.f, 0.f};
            const int n = min(D, total - i0);
            bool ok = true;
#pragma unroll
            for (int d = 0; d < D; ++d)
                if (ok && d < n) ok = slot_item(d, phase, v[d]);
            if (!ok) break;
            const float r = warp_sum4(v[0], v[1], v[2], v[3], lane);   // value lane >> 3, every lane
            if ((lane & 7) == 0 && (lane >> 3) < n) part[kb0 + i0 + (lane >> 3)] = r;
            i = i0 + n;
        }
    } else {
        // ---- decode span by span; the table of span sp replaces that of sp - 1
        bool ok = true;
        int d = 0;
        uint32_t phase = 0;
        uint4 xn[(16 + NW - 1) / NW];
#pragma unroll
        for (int q = 0; q < (16 + NW - 1) / NW; ++q)
            if (warp + q * NW < 16 && nspan > 1) xn[q] = b1_table_x(a.x, 1, warp + q * NW, lane);
        // (after a timeout the warp still passes every span's barriers)
        for (int sp = 0; sp < nspan; ++sp) {
            tst = s0;   // every span walks the same run of stages and rows
            trl = nrows - r0;
            if (sp > 0) {
                __syncthreads();   // every warp is done with the table of span sp - 1
#pragma unroll
                for (int q = 0; q < (16 + NW - 1) / NW; ++q)
                    if (warp + q * NW < 16) {
                        if constexpr (TAB)
                            b1_xspan_job(sbase, pm, sp * kB1Span, warp + q * NW, lane, xn[q]);
                        else
                            b1_table_job(sbase, pm, sp * kB1Span, warp + q * NW, lane, xn[q]);
                    }
                __syncthreads();
#pragma unroll
                for (int q = 0; q < (16 + NW - 1) / NW; ++q)
                    if (warp + q * NW < 16 && sp + 1 < nspan) xn[q] = b1_table_x(a.x, sp + 1, warp + q * NW, lane);
            }
            // four items at a time, their partial sums added over the warp together
            for (int j0 = 0; j0 < cnt0 && ok; j0 += 4) {
                float v[4] = {0.f, 0.f, 0.f, 0.f};
                const int n = min(4, cnt0 - j0);
#pragma unroll
                for (int q = 0; q < 4; ++q)
                    if (ok && q < n) {
                        ok = slot_item(d, phase, v[q]);
                        if (++d == D) {
                            d = 0;
                            phase ^= 1u;
                        }
                    }
                if (!ok) break;
                const float r = warp_sum4(v[0], v[1], v[2], v[3], lane);
                if ((lane & 7) == 0 && (lane >> 3) < n) part[sp * per_span + kb0 + j0 + (lane >> 3)] = r;
                i += n;
            }
        }
    }
    // every copy this warp requested has landed before it leaves the ring:
    // the slots of the items requested and not consumed (only after a
    // timeout; their slot for item j is j % D, its phase (j / D) & 1)
    const int requested = to_request - left;
    if (lane == 0)
        for (int j = i; j < requested; ++j)
            mbar_wait(wbar + static_cast<uint32_t>(j % D) * 8u, static_cast<uint32_t>(j / D) & 1u);

    // ---- the protected term of rows warp, warp + NW, ... (Eq. 10), while
    // other warps may still decode: four rows at a time, all their payload
    // loads issued before the first product, then added over the warp
    // together (load: a payload element's bits; value: its value, exact in
    // fp32 -- Eq. 10's int8, or the FP8 / bf16 payload of the protected-
    // format variants; one instance per format)
    auto prot_term = [&](auto load, auto value) {
        for (int rr0 = warp; rr0 < nrows; rr0 += 4 * NW) {
            float pr[4] = {0.f, 0.f, 0.f, 0.f};
            for (int u0 = 0; u0 < p; u0 += 64) {
                uint32_t qv[4][2];
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                    const int rr = rr0 + k * NW;
                    const int8_t *q8r = a.q8_staged ? q8s + rr * prow : q8 + static_cast<int64_t>(ra + rr) * prow;
#pragma unroll
                    for (int h = 0; h < 2; ++h) {
                        const int u = u0 + 32 * h + lane;
                        qv[k][h] = rr < nrows && u < p ? load(q8r, u) : 0u;
                    }
                }
#pragma unroll
                for (int k = 0; k < 4; ++k)
#pragma unroll
                    for (int h = 0; h < 2; ++h) {
                        const int u = u0 + 32 * h + lane;
                        if (u < p) pr[k] = fmaf(value(qv[k][h]), sx[u], pr[k]);
                    }
            }
            const float r = warp_sum4(pr[0], pr[1], pr[2], pr[3], lane);   // row rr0 + (lane >> 3) * NW
            const int rr = rr0 + (lane >> 3) * NW;
            if ((lane & 7) == 0 && rr < nrows) prot[rr] = r;
        }
    };
    auto load_byte = [](const int8_t *r, int u) { return static_cast<uint32_t>(static_cast<uint8_t>(r[u])); };
    if (p > 0) {
        if (!FMT || fmt == BISCO_PROT_INT8)
            prot_term(load_byte, [](uint32_t b) { return static_cast<float>(static_cast<int8_t>(b)); });
        else if (fmt == BISCO_PROT_BF16)
            prot_term([](const int8_t *r, int u) { return static_cast<uint32_t>(reinterpret_cast<const uint16_t *>(r)[u]); },
                      [](uint32_t b) { return __uint_as_float(b << 16); });
        else
            prot_term(load_byte, [fmt](uint32_t b) { return fp8_to_f32(b, fmt); });
    }

    // ---- the layer's low-rank compensation (Sec. III-F), first t = A x:
    // units of eight ranks x 256 columns, each taken by whichever warp is
    // free first (a unit's result does not depend on the warp), its sums
    // into lt[column slice][rank]
    float *lt = reinterpret_cast<float *>(sm + a.off_lt);   // [K / 256][rank], then t [rank]
    const int nsl = K / 256;
    if (lrank > 0) {
        const int nunit = (lrank / 8) * nsl;
        for (;;) {
            int u = 0;
            if (lane == 0) u = atomicAdd(&s_lnext, 1);
            u = __shfl_sync(0xFFFFFFFFu, u, 0);
            if (u >= nunit) break;
            const int sl = u % nsl, r0 = (u / nsl) * 8;
            const int col = sl * 256 + lane * 8;
            const uint4 xv = *reinterpret_cast<const uint4 *>(a.x + col);
            uint4 av[8];
#pragma unroll
            for (int q = 0; q < 8; ++q)
                av[q] = *reinterpret_cast<const uint4 *>(L.la + static_cast<size_t>(r0 + q) * K + col);
            const float xf[8] = {bf16_bits_to_f32(static_cast<uint16_t>(xv.x)), bf16_bits_to_f32(static_cast<uint16_t>(xv.x >> 16)),
                                 bf16_bits_to_f32(static_cast<uint16_t>(xv.y)), bf16_bits_to_f32(static_cast<uint16_t>(xv.y >> 16)),
                                 bf16_bits_to_f32(static_cast<uint16_t>(xv.z)), bf16_bits_to_f32(static_cast<uint16_t>(xv.z >> 16)),
                                 bf16_bits_to_f32(static_cast<uint16_t>(xv.w)), bf16_bits_to_f32(static_cast<uint16_t>(xv.w >> 16))};
            float d[8];
#pragma unroll
            for (int q = 0; q < 8; ++q) {
                const uint32_t w[4] = {av[q].x, av[q].y, av[q].z, av[q].w};
                float acc = 0.f;
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    acc = fmaf(bf16_bits_to_f32(static_cast<uint16_t>(w[e])), xf[2 * e], acc);
                    acc = fmaf(bf16_bits_to_f32(static_cast<uint16_t>(w[e] >> 16)), xf[2 * e + 1], acc);
                }
                d[q] = acc;
            }
            const float s0 = warp_sum4(d[0], d[1], d[2], d[3], lane);   // rank r0 + (lane >> 3)
            const float s1 = warp_sum4(d[4], d[5], d[6], d[7], lane);   // rank r0 + 4 + (lane >> 3)
            if ((lane & 7) == 0) {
                lt[sl * lrank + r0 + (lane >> 3)] = s0;
                lt[sl * lrank + r0 + 4 + (lane >> 3)] = s1;
            }
        }
    }
    __syncthreads();
    if (*reinterpret_cast<volatile int *>(&s_abort)) return;
    // t[r]: the slices' sums in slice order
    float *lt_t = lt + nsl * a.lrank;
    if (lrank > 0) {
        if (static_cast<int>(threadIdx.x) < lrank) {
            float t = 0.f;
            for (int sl = 0; sl < nsl; ++sl) t += lt[sl * lrank + threadIdx.x];
            lt_t[threadIdx.x] = t;
        }
        __syncthreads();
    }
    // ---- protected output rows (Eq. 9 with Eq. 10 on rows): their chunks
    // store norm 0, so the decode gave them 0; each is the dot product of
    // its payload row with x, times the row's scale.  Every warp takes K/16
    // columns of each of the CTA's protected rows (lane l eight of them per
    // 256), its sums go to the now idle ring, and a thread per row adds the
    // 16 in warp order.
    if constexpr (ROWS) {
        // rows in batches the ring holds (depth * 1536 bytes a warp)
        const int cap = a.depth * static_cast<int>(kB1Item) / 4;
        for (int b0 = s_r0; b0 < s_r1; b0 += cap) {
            const int b1 = min(s_r1, b0 + cap), nr = b1 - b0;
            float *rp = reinterpret_cast<float *>(sm + a.off_ring);   // [row][warp]
            const int kp = (K + 15) / 16 * 16, kw = K / NW;
            const bool bf = fmt == BISCO_PROT_BF16;
            for (int t = b0; t < b1; ++t) {
                const unsigned char *qr =
                    reinterpret_cast<const unsigned char *>(q8) + static_cast<int64_t>(t) * kp * (bf ? 2 : 1);
                float d = 0.f;
                for (int k0 = warp * kw + lane * 8; k0 < (warp + 1) * kw; k0 += 256) {
                    const uint4 xv = *reinterpret_cast<const uint4 *>(a.x + k0);
                    const uint32_t xw[4] = {xv.x, xv.y, xv.z, xv.w};
                    float qf[8];
                    if (bf) {
                        const uint4 q = *reinterpret_cast<const uint4 *>(qr + 2 * k0);
                        const uint32_t qw[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
                        for (int e = 0; e < 4; ++e) {
                            qf[2 * e] = __uint_as_float(qw[e] << 16);
                            qf[2 * e + 1] = __uint_as_float(qw[e] & 0xFFFF0000u);
                        }
                    } else {
                        const uint2 q = *reinterpret_cast<const uint2 *>(qr + k0);
#pragma unroll
                        for (int e = 0; e < 8; ++e) {
                            const uint32_t b8 = ((e < 4 ? q.x : q.y) >> (8 * (e & 3))) & 0xFFu;
                            qf[e] = fmt == BISCO_PROT_INT8 ? static_cast<float>(static_cast<int8_t>(b8))
                                                           : fp8_to_f32(b8, fmt);
                        }
                    }
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        d = fmaf(qf[2 * e], __uint_as_float(xw[e] << 16), d);
                        d = fmaf(qf[2 * e + 1], __uint_as_float(xw[e] & 0xFFFF0000u), d);
                    }
                }
#pragma unroll
                for (int o = 16; o > 0; o >>= 1) d += __shfl_xor_sync(0xFFFFFFFFu, d, o);
                if (lane == 0) rp[(t - b0) * NW + warp] = d;
            }
            __syncthreads();
            for (int i = threadIdx.x; i < nr; i += kThreads) {
                const int rr = L.prot_idx[b0 + i] - ra;
                if (rr < 0 || rr >= nrows) {   // not an ascending list
                    latch_error(a.err, BISCO_ERR_INVALID_ARG);
                    continue;
                }
                float d = 0.f;
                for (int w = 0; w < NW; ++w) d += rp[i * NW + w];
                prot[rr] = __half2float(__ushort_as_half(L.q8_scale[b0 + i])) * d;
            }
            __syncthreads();
        }
    }

    // ---- outputs: a thread per row; the row's item sums in order, then the
    // protected term, then scale * (Bm t) of the compensation
    for (int rr = threadIdx.x; rr < nrows; rr += kThreads) {
        float v = 0.f;
        for (int sp = 0; sp < nspan; ++sp)
            for (int s = 0; s < S; ++s) v += part[sp * per_span + s * nrows + rr];
        // (the sign decode's 1/sqrt(8) of Eq. 3; a decoder table holds its
        // outputs as they are)
        v = v * (TAB ? 1.f : kB1InvSqrt8) + (L.p > 0 ? prot[rr] : 0.f);
        if (lrank > 0) {
            const uint16_t *bm = L.lb + static_cast<size_t>(ra + rr) * lrank;
            float bt = 0.f;
            for (int r0 = 0; r0 < lrank; r0 += 8) {
                const uint4 bv = *reinterpret_cast<const uint4 *>(bm + r0);
                const uint32_t w[4] = {bv.x, bv.y, bv.z, bv.w};
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    bt = fmaf(bf16_bits_to_f32(static_cast<uint16_t>(w[e])), lt_t[r0 + 2 * e], bt);
                    bt = fmaf(bf16_bits_to_f32(static_cast<uint16_t>(w[e] >> 16)), lt_t[r0 + 2 * e + 1], bt);
                }
            }
            v = fmaf(L.lscale, bt, v);
        }
        y[ra + rr] = v;
    }
}

size_t align_up_b1(size_t v, size_t a) { return (v + a - 1) / a * a; }

template <int NW, int D, int NSPAN, int MODE>
bisco_status launch_b1_t(const B1Args &a, int grid, size_t smem, cudaStream_t stream) {
    auto kern = k_gemv_b1<NW, D, NSPAN, MODE>;
    static size_t configured[64] = {};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return BISCO_ERR_CUDA;
    if (smem > configured[dev]) {
        if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 static_cast<int>(smem)) != cudaSuccess)
            return BISCO_ERR_CUDA;
        configured[dev] = smem;
    }
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid, 1, 1);
    cfg.blockDim = dim3(NW * 32, 1, 1);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kern, a) == cudaSuccess ? BISCO_OK : BISCO_ERR_CUDA;
}

// The most dynamic shared memory at which two CTAs of the kernel (this
// layer's and the next one's) share an SM, from the runtime's occupancy
// calculator (every instantiation has the same block size and static
// shared memory); found once per device.
size_t b1_coresident_budget() {
    static size_t budget[64] = {};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 0;
    if (budget[dev] != 0) return budget[dev];
    auto kern = k_gemv_b1<16, 3, 1, kB1Int8>;
    constexpr size_t kHi = 160 * 1024;   // more than two CTAs of an SM can hold
    if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(kHi)) !=
        cudaSuccess) {
        (void)cudaGetLastError();
        return 0;
    }
    auto two = [&](size_t smem) {
        int n = 0;
        const bool ok = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, kern, 16 * 32, smem) == cudaSuccess;
        if (!ok) (void)cudaGetLastError();
        return ok && n >= 2;
    };
    size_t lo = 0, hi = kHi;   // two(lo) or lo = 0; not two(hi)
    while (hi - lo > 16) {
        const size_t mid = (lo + hi) / 2 / 16 * 16;
        if (two(mid)) lo = mid;
        else hi = mid;
    }
    budget[dev] = lo > 0 ? lo : 1;
    return budget[dev];
}

// Shared memory of one CTA of nw warps with `depth` one-item slots per
// warp, past the 4 KB aligned base (the span table first); fills the offsets
// of `a`.
size_t b1_layout(int C, int nw, int depth, int p_max, int rows_max, int items_max, size_t q8_bytes,
                 B1Args *a) {
    size_t off = static_cast<size_t>(kB1Span) * 64;   // the table of one span: 64 bytes per chunk
    a->off_ring = static_cast<uint32_t>(off);
    off += static_cast<size_t>(nw) * depth * kB1Item;
    a->off_pm = static_cast<uint32_t>(off);
    off += static_cast<size_t>(C);                          // one bit per column
    a->off_pidx = static_cast<uint32_t>(off);
    off += static_cast<size_t>((p_max + 3) / 4 * 4) * 8;    // indices, scales
    a->off_sx = static_cast<uint32_t>(off);
    off += static_cast<size_t>(p_max) * 4;
    off = align_up_b1(off, 16);
    a->off_part = static_cast<uint32_t>(off);
    off += static_cast<size_t>(items_max) * 4;
    a->off_prot = static_cast<uint32_t>(off);
    off += static_cast<size_t>(rows_max) * 4;
    a->off_lt = static_cast<uint32_t>(off);                 // compensation: slice sums, t
    off += a->lrank > 0 ? static_cast<size_t>(C / 32 + 1) * a->lrank * 4 : 0;
    off = align_up_b1(off, 16);
    a->off_q8 = static_cast<uint32_t>(off);
    off += q8_bytes;
    off = align_up_b1(off, 8);
    a->off_bar = static_cast<uint32_t>(off);
    off += static_cast<size_t>(nw) * depth * 8;
    return off + 4096;   // slack for the 4 KB aligned base
}

// The instantiated (warps, slots per warp, items per slot) shapes, in order
// of preference: one span per row, then several.  Measured on GB300: 12
// warps with two-item slots (the per-slot work paid once per two items, 80
// registers) run the 36x7 step 8 % slower than 16 warps with one item per
// slot -- latency is hidden by warps more than by the slot work saved.
struct B1Shape {
    int nw, depth;
};
constexpr B1Shape kB1Shapes[] = {{16, 3}, {16, 2}};

}  // namespace

bisco_status launch_gemv_b1(const bisco_layer *Ls, int G, const uint16_t *x, float *const *y,
                            int *err, cudaStream_t stream, bool *launched, const bisco_lora *loras,
                            const uint16_t *tables) {
    *launched = false;
    if (const char *e = getenv("BISCO_GEMV_B1"))
        if (e[0] == '0') return BISCO_OK;
    if (G < 1 || G > kB1MaxG) return BISCO_OK;
    const int K = Ls[0].k_in, S = Ls[0].stages;
    if (K % 4096 != 0 || S < 1 || S > 3) return BISCO_OK;
    B1Args a = {};
    a.x = x;
    a.err = err;
    a.K = K;
    a.G = G;
    a.nspan = K / 4096;
    int p_max = 0;
    for (int g = 0; g < G; ++g) {
        const bisco_layer &L = Ls[g];
        if (L.k_in != K || L.stages != S) return BISCO_OK;
        // the kernel's byte offsets into the sign planes are 32-bit
        if (static_cast<uint64_t>(S) * L.n_out * (K / 8) >= (1ull << 32)) return BISCO_OK;
        B1Layer &b = a.L[g];
        b.codes = reinterpret_cast<const uint8_t *>(L.codes);
        b.norms = L.norms;
        b.q8 = L.q8;
        b.q8_scale = L.q8_scale;
        b.prot_idx = L.prot_idx;
        b.y = y[g];
        b.N = L.n_out;
        b.p = L.n_protected;
        b.p_pad = (L.n_protected + 15) / 16 * 16;
        b.fmt = L.protect_format;
        b.axis = L.protect_axis;
        // int8 rows staged per CTA: the column payload only
        b.prow = L.protect_axis ? 0 : b.p_pad * (L.protect_format == BISCO_PROT_BF16 ? 2 : 1);
        if (!b.axis) p_max = p_max > b.p ? p_max : b.p;   // the column sets' metadata
        if (loras != nullptr && loras[g].rank > 0) {
            // the compensation's slices are 256 columns of one span
            if (a.nspan != 1) return BISCO_OK;
            b.la = loras[g].A;
            b.lb = loras[g].Bm;
            b.rank = loras[g].rank;
            b.lscale = loras[g].scale;
            a.lrank = a.lrank > b.rank ? a.lrank : b.rank;
        }
    }
    const int sms = num_sms();
    if (G > sms) return BISCO_OK;
    const size_t coresident = b1_coresident_budget();
    int items_all = 0;
    for (int g = 0; g < G; ++g) items_all += a.L[g].N * S * a.nspan;
    const int C = K / 8;
    const bool one = a.nspan == 1;
    const B1Shape *shapes = kB1Shapes;
    const int nshapes = 2;
    int total = 0;
    B1Shape pick = {0, 0};
    size_t smem = 0;
    // CTAs per layer: one each, then one at a time to the layer with the
    // longest row run per CTA, up to `slots` CTAs; then the first shape that
    // leaves room for a second CTA on the SM (int8 rows staged if they fit),
    // else, with one CTA per SM, the first that fits
    auto plan = [&](int slots) {
        int ctas[kB1MaxG] = {};
        total = G;
        for (int g = 0; g < G; ++g) ctas[g] = 1;
        auto run = [&](int g) { return (a.L[g].N + ctas[g] - 1) / ctas[g]; };
        while (total < slots) {
            int best = -1;
            for (int g = 0; g < G; ++g)
                if (ctas[g] < a.L[g].N && (best < 0 || run(g) > run(best))) best = g;
            if (best < 0) break;
            ++ctas[best];
            ++total;
        }
        int rows_max = 0;
        size_t q8_max = 0;
        for (int g = 0, c0 = 0; g < G; ++g) {
            a.L[g].cta0 = c0;
            a.L[g].ctas = ctas[g];
            c0 += ctas[g];
            rows_max = rows_max > run(g) ? rows_max : run(g);
            const size_t q8b = static_cast<size_t>(run(g)) * a.L[g].prow;
            q8_max = q8_max > q8b ? q8_max : q8b;
        }
        const int items_max = rows_max * S * a.nspan;
        pick = {0, 0};
        const int passes = slots > sms ? 1 : 2;
        for (int pass = 0; pass < passes && pick.nw == 0; ++pass) {
            const size_t budget = pass == 0 ? coresident : kB1MaxSmem;
            for (int k = 0; k < nshapes && pick.nw == 0; ++k)
                for (int staged = 1; staged >= 0 && pick.nw == 0; --staged) {
                    const B1Shape &sh = shapes[k];
                    const size_t need = b1_layout(C, sh.nw, sh.depth, p_max, rows_max, items_max,
                                                  staged ? q8_max : 0, &a);
                    if (need <= budget) {
                        pick = sh;
                        smem = need;
                        a.q8_staged = staged;
                    }
                }
        }
        if (pick.nw != 0)
            b1_layout(C, pick.nw, pick.depth, p_max, rows_max, items_max, a.q8_staged ? q8_max : 0, &a);
    };
    if (items_all >= kB1TwoPerSm * sms) plan(2 * sms);
    if (pick.nw == 0) plan(sms);
    if (pick.nw == 0) return BISCO_OK;
    a.depth = pick.depth;
    a.S = S;
    a.sleep_ns = 200;
    // test hook for the bounded waits: with BISCO_TEST_WITHHOLD_COPIES set the
    // kernel requests no data, so its waits expire, it latches
    // BISCO_ERR_TIMEOUT and returns with no copy in flight
    a.withhold = getenv("BISCO_TEST_WITHHOLD_COPIES") != nullptr;
    *launched = true;
    int mode = kB1Int8;
    if (tables != nullptr) {
        // table mode: one layer, int8 columns
        if (G != 1 || (a.L[0].p > 0 && (a.L[0].fmt != BISCO_PROT_INT8 || a.L[0].axis != 0)) || a.lrank > 0) {
            *launched = false;
            return BISCO_OK;
        }
        a.tab = tables;
        mode = kB1Tab;
    } else {
        // the kind of every protected set of the launch: one instance takes
        // int8 columns, one any column format, one rows (not mixed)
        bool cols_fmt = false, rows = false, cols = false;
        for (int g = 0; g < G; ++g) {
            if (a.L[g].p == 0) continue;
            if (a.L[g].axis) rows = true;
            else {
                cols = true;
                cols_fmt |= a.L[g].fmt != BISCO_PROT_INT8;
            }
        }
        if ((rows && cols) || (a.lrank > 0 && (rows || cols_fmt))) {
            *launched = false;
            return BISCO_OK;
        }
        mode = a.lrank > 0 ? kB1Lora : rows ? kB1Rows : cols_fmt ? kB1Fmt : kB1Int8;
    }
    auto go = [&](auto mode_c) {
        constexpr int M = decltype(mode_c)::value;
        if (one) {
            if (pick.depth == 3) return launch_b1_t<16, 3, 1, M>(a, total, smem, stream);
            return launch_b1_t<16, 2, 1, M>(a, total, smem, stream);
        }
        if (pick.depth == 3) return launch_b1_t<16, 3, 0, M>(a, total, smem, stream);
        return launch_b1_t<16, 2, 0, M>(a, total, smem, stream);
    };
    switch (mode) {
        case kB1Fmt: return go(std::integral_constant<int, kB1Fmt>());
        case kB1Rows: return go(std::integral_constant<int, kB1Rows>());
        case kB1Tab: return go(std::integral_constant<int, kB1Tab>());
        case kB1Lora: return go(std::integral_constant<int, kB1Lora>());
        default: return go(std::integral_constant<int, kB1Int8>());
    }
}
}  // namespace bisco
