"""The prefill GEMM's split of its tiles' k-steps over the persistent CTAs
(csrc/gemm_sched.cuh, the header the GEMM kernel, its fixup kernel and its
launcher use) compiled for the host: for every plan, every k-step of every
tile runs in exactly one CTA's pieces, a tile split between CTAs has its
pieces in the CTAs sk_owner names and in the workspace slots sk_slot names
(no two pieces of a CTA in one slot), and exactly one fixup block sums each
split tile while no whole tile is summed.  The GPU tests check the kernels
themselves."""
import os
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
CSRC = os.path.join(ROOT, "paper_2607_08643_gb300", "csrc")

PROBE = r"""
#include <stdio.h>
#include <vector>
#include "gemm_sched.cuh"
using namespace bisco;
// stdin: lines "T KS SMS"; stdout: "G whole" per line, or "FAIL reason"
static const char *check(const SkPlan &p, int sms) {
    const int cap = sms < kSkMaxCtas ? sms : kSkMaxCtas;
    if (p.G < 1 || p.G > cap) return "grid outside [1, min(sms, kSkMaxCtas)]";
    if (p.W != (long long)p.ntiles * p.KS) return "W != T * KS";
    std::vector<int> cover((size_t)p.W, 0), npieces(p.ntiles, 0), whole(p.ntiles, 0);
    std::vector<std::vector<int>> owners(p.ntiles);
    for (int c = 0; c < p.G; ++c) {
        const SkSched s(c, p);
        if (s.n < 1) return "a CTA with no work";
        int used[2] = {0, 0};
        long long next = s.w0;
        for (int j = 0; j < s.n; ++j) {
            const SkPiece pc = s.at(j, c, p);
            if (pc.t < 0 || pc.t >= p.ntiles) return "piece outside the tiles";
            if (!(0 <= pc.k0 && pc.k0 < pc.k1 && pc.k1 <= p.KS)) return "empty or out-of-range k-steps";
            if (!p.whole) {
                if ((long long)pc.t * p.KS + pc.k0 != next) return "stream-K pieces not contiguous";
                next = (long long)pc.t * p.KS + pc.k1;
            }
            for (int k = pc.k0; k < pc.k1; ++k) cover[(size_t)pc.t * p.KS + k] += 1;
            npieces[pc.t] += 1;
            owners[pc.t].push_back(c);
            if (pc.k0 == 0 && pc.k1 == p.KS) {
                whole[pc.t] = 1;
            } else {
                if (p.whole) return "a partial piece under whole tiles";
                const int slot = j == 0 ? 0 : 1;   // the GEMM epilogue's slot
                if (slot != sk_slot(c, pc.t, p)) return "epilogue slot != sk_slot";
                if (used[slot]++) return "two pieces of a CTA in one slot";
            }
        }
        if (!p.whole && next != s.w1) return "stream-K range not covered";
    }
    for (size_t i = 0; i < cover.size(); ++i)
        if (cover[i] != 1) return "a k-step run zero or several times";
    std::vector<int> fixed(p.ntiles, 0);
    if (!p.whole)
        for (int c = 1; c < p.G; ++c) {
            const int t = sk_fixup_tile(c, p);
            if (t < -1 || t >= p.ntiles) return "fixup tile out of range";
            if (t >= 0) fixed[t] += 1;
        }
    for (int t = 0; t < p.ntiles; ++t) {
        if (whole[t] != (npieces[t] == 1)) return "a tile both whole and split";
        if (npieces[t] > 1) {
            if (fixed[t] != 1) return "a split tile not summed exactly once";
            const long long ts = (long long)t * p.KS;
            const int lo = sk_owner(ts, p), hi = sk_owner(ts + p.KS - 1, p);
            if (hi - lo + 1 != npieces[t]) return "sk_owner range != the tile's CTAs";
            for (int i = 0; i < npieces[t]; ++i)
                if (owners[t][i] != lo + i) return "the tile's CTAs not lo..hi in order";
        } else if (fixed[t]) {
            return "a whole tile summed by the fixup";
        }
    }
    return nullptr;
}
int main() {
    int T, KS, sms;
    while (scanf("%d %d %d", &T, &KS, &sms) == 3) {
        const SkPlan p = sk_plan(T, KS, sms);
        const char *e = check(p, sms);
        if (e) printf("FAIL %s\n", e);
        else printf("%d %d\n", p.G, p.whole);
    }
    return 0;
}
"""


@pytest.fixture(scope="module")
def probe(tmp_path_factory):
    d = tmp_path_factory.mktemp("schedprobe")
    src = d / "probe.cpp"
    src.write_text(PROBE)
    exe = d / "probe"
    subprocess.check_call(["g++", "-std=c++17", "-O2", "-I", CSRC, "-o", str(exe), str(src)])
    return exe


def run(probe, triples):
    inp = "".join("%d %d %d\n" % t for t in triples)
    out = subprocess.run([str(probe)], input=inp, capture_output=True, text=True, check=True).stdout
    lines = out.split("\n")[:len(triples)]
    for t, line in zip(triples, lines):
        assert not line.startswith("FAIL"), (t, line)
    return [tuple(int(v) for v in line.split()) for line in lines]


def test_every_step_once_and_every_split_tile_summed_once(probe):
    triples = [(T, KS, sms)
               for T in (1, 2, 3, 7, 8, 63, 64, 151, 152, 153, 255, 256, 300, 768, 1000, 1536)
               for KS in (1, 2, 3, 5, 8, 13, 33, 98)
               for sms in (1, 2, 7, 148, 152, 160, 200)]
    assert len(run(probe, triples)) == len(triples)


@pytest.mark.parametrize("name,T,KS,whole", [
    ("q_proj 4096x4096", 256, 33, 1),     # 2 x 33 steps against 55 + 16: whole tiles
    ("k_proj 1024x4096", 64, 33, 0),      # 33 against 13 + 16
    ("gate_proj 12288x4096", 768, 33, 0),  # 6 x 33 against 166 + 16
    ("down_proj 4096x12288", 256, 98, 0),  # 2 x 98 against 165 + 16
])
def test_plans_of_qwen3_shapes_at_2048_tokens(probe, name, T, KS, whole):
    """The schedules the GB300 measurements chose (152 SMs): 128 features x
    256 tokens per tile, S = 2, 1 % protected columns (one extension step
    per 64 protected columns)."""
    (G, w), = run(probe, [(T, KS, 152)])
    assert w == whole, name
    assert G == 152, name


def test_small_problems_keep_pieces_long(probe):
    """Few k-steps: no more CTAs than W / 8, so a piece is never shorter
    than 8 k-steps unless the whole problem is."""
    for T, KS in ((1, 33), (2, 13), (1, 5), (3, 3)):
        (G, w), = run(probe, [(T, KS, 152)])
        if not w:
            assert T * KS // G >= 8
