// gemm_sched.cuh -- how the prefill GEMM shares its work out among its
// persistent CTAs, host and device: gemm.cu's kernels and launcher use it,
// and a host build lets the CPU tests check that every k-step of every tile
// runs exactly once and every tile split between CTAs is summed once.
//
// Output tiles t = 0..T-1 of KS k-steps each (one k-step: 128 columns of K,
// or 64 protected columns).  Two schedules:
//   whole tiles  CTA c runs tiles c, c + G, c + 2G, ...
//   stream-K     the tiles' k-steps laid end to end (tile t holds steps
//                [t*KS, (t+1)*KS), W = T*KS in all) and CTA c runs steps
//                [c*W/G, (c+1)*W/G): every CTA has the same work.  A tile
//                covered by one CTA goes straight to Y; the pieces of a tile
//                split between CTAs go to the workspace (the first piece of
//                a CTA's range in its slot 0, any later one in slot 1) and a
//                second kernel adds them in CTA order.
// sk_plan takes stream-K when its range plus kSkOverheadSteps is shorter
// than the whole-tile schedule's longest range.
#pragma once

#include <stdint.h>

#ifndef BISCO_HD
#ifdef __CUDACC__
#define BISCO_HD __host__ __device__ __forceinline__
#else
#define BISCO_HD inline
#endif
#endif

namespace bisco {

constexpr int kSkMaxCtas = 160;   // partial-tile slots in the workspace: 2 per CTA
constexpr int kSkMinSteps = 8;    // fewer CTAs when the pieces would be shorter
// The cost of stream-K's extra pieces (the partial tiles' stores, the
// pipeline drain at each piece boundary, the fixup kernel) in k-steps:
// measured on the Qwen3-8B shapes at 2048 tokens as 16-27.
constexpr int kSkOverheadSteps = 16;

struct SkPlan {
    int ntiles;   // output tiles T
    int KS;       // k-steps per tile
    int G;        // CTAs
    int whole;    // 1: whole tiles; 0: stream-K
    int64_t W;    // T * KS
};

// The schedule for T tiles of KS k-steps on `sms` SMs (T, KS >= 1).
BISCO_HD SkPlan sk_plan(int ntiles, int KS, int sms) {
    SkPlan p;
    p.ntiles = ntiles;
    p.KS = KS;
    p.W = static_cast<int64_t>(ntiles) * KS;
    const int cap = sms < kSkMaxCtas ? sms : kSkMaxCtas;
    int64_t g = p.W / kSkMinSteps;
    if (g > cap) g = cap;
    if (g < 1) g = 1;
    const int g_whole = ntiles < cap ? ntiles : cap;
    const int64_t whole_steps = static_cast<int64_t>((ntiles + g_whole - 1) / g_whole) * KS;
    p.whole = whole_steps <= p.W / g + kSkOverheadSteps ? 1 : 0;
    p.G = p.whole ? g_whole : static_cast<int>(g);
    return p;
}

// stream-K: the first step of CTA c's range (c = G gives W)
BISCO_HD int64_t sk_begin(int c, const SkPlan &p) { return static_cast<int64_t>(c) * p.W / p.G; }

// stream-K: the CTA whose range holds step w, the largest c with
// sk_begin(c) <= w
BISCO_HD int sk_owner(int64_t w, const SkPlan &p) { return static_cast<int>(((w + 1) * p.G - 1) / p.W); }

struct SkPiece {
    int t, k0, k1;   // tile, its k-steps [k0, k1)
};

// The pieces of CTA c, in the order it runs them.
struct SkSched {
    int n;            // pieces
    int64_t w0, w1;   // stream-K: the range

    BISCO_HD SkSched(int c, const SkPlan &p) {
        if (p.whole) {
            n = c < p.ntiles ? (p.ntiles - c + p.G - 1) / p.G : 0;
            w0 = w1 = 0;
        } else {
            w0 = sk_begin(c, p);
            w1 = sk_begin(c + 1, p);
            n = w1 > w0 ? static_cast<int>((w1 - 1) / p.KS - w0 / p.KS) + 1 : 0;
        }
    }

    BISCO_HD SkPiece at(int j, int c, const SkPlan &p) const {
        SkPiece pc;
        if (p.whole) {
            pc.t = c + j * p.G;
            pc.k0 = 0;
            pc.k1 = p.KS;
        } else {
            const int ta = static_cast<int>(w0 / p.KS), tb = static_cast<int>((w1 - 1) / p.KS);
            pc.t = ta + j;
            pc.k0 = pc.t == ta ? static_cast<int>(w0 - static_cast<int64_t>(ta) * p.KS) : 0;
            pc.k1 = pc.t == tb ? static_cast<int>(w1 - static_cast<int64_t>(tb) * p.KS) : p.KS;
        }
        return pc;
    }
};

// stream-K: the workspace slot of CTA cc's piece of tile t -- 0 if t is the
// first tile of cc's range, else 1
BISCO_HD int sk_slot(int cc, int t, const SkPlan &p) { return sk_begin(cc, p) / p.KS == t ? 0 : 1; }

// stream-K fixup: the tile that block c - 1 sums (c = 1..G-1: the boundary
// between CTAs c - 1 and c), or -1 when that boundary is at a tile's edge or
// is not the first boundary inside its tile (so each split tile is summed by
// exactly one block)
BISCO_HD int sk_fixup_tile(int c, const SkPlan &p) {
    const int64_t b = sk_begin(c, p);
    const int t = static_cast<int>(b / p.KS);
    const int64_t ts = static_cast<int64_t>(t) * p.KS;
    if (b == ts || sk_begin(c - 1, p) > ts) return -1;
    return t;
}

}  // namespace bisco
