// Work partition of the step kernel (host only).
//
// The gradient of a unit is one or more segments of the arena (a transformer
// block spans several weight tensors).  Segments are ordered by unit, and the
// segments of all units are concatenated into one stream of "points": a
// segment of L elements contributes max(L, 1) points (a unit with no element
// still needs one warp to run its Algorithm 1 update).  A unit costs
// kUnitCostBytes plus the bytes of its segments.  The stream is cut into runs
// of about equal cost, so skewed sizes (a 256-element unit next to a
// 70M-element one) balance across the grid: large segments are split over
// many runs, small ones are packed many to a run.  The small-unit loop gives
// every warp one run; the large-unit loop plans several runs per warp, which
// the warps take in turn.
//
// Cuts inside a segment fall on multiples of kSplitBytes from its start, so
// the body of every piece keeps the segment's 16-byte alignment.  Runs are
// strictly increasing and never empty, and a unit's segments are contiguous in
// the stream, so the runs that touch a unit are a contiguous range
// first_run[b] .. first_run[b] + num_parts[b] - 1; the kernel stores the
// partial sum of run r for unit b in slot part_base[b] + (r - first_run[b]),
// so the reduction order of a unit is fixed by the plan (whichever warp
// streams a run) and results are bitwise reproducible run to run.
#include <algorithm>
#include <cstdint>
#include <vector>

#include "gnmr_internal.h"

namespace gnmr {

namespace {

struct Point {
    int64_t seg;
    int64_t pos;
    bool operator<(const Point &o) const { return seg != o.seg ? seg < o.seg : pos < o.pos; }
};

}  // namespace

bool plan_partition(int64_t num_segments, const int64_t *seg_lengths, const int32_t *seg_unit,
                    int32_t num_units, int elem_bytes, int32_t max_runs, Plan &out)
{
    if (num_segments < 1 || num_units < 1 || !seg_lengths || !seg_unit ||
        (elem_bytes != 2 && elem_bytes != 4) || max_runs < 1)
        return false;
    const int64_t S = num_segments, U = num_units;
    // segments must be grouped by unit, every unit present
    for (int64_t g = 0; g < S; ++g) {
        const int64_t u = seg_unit[g];
        if (u < 0 || u >= U || (g > 0 && u < seg_unit[g - 1]) || (g > 0 && u > seg_unit[g - 1] + 1) ||
            (g == 0 && u != 0))
            return false;
    }
    if (seg_unit[S - 1] != U - 1)
        return false;

    std::vector<int64_t> cstart(S + 1, 0);     // cost at the start of segment g
    for (int64_t g = 0; g < S; ++g) {
        const int64_t L = seg_lengths[g];
        if (L < 0 || L > (INT64_MAX / 8) / elem_bytes)
            return false;
        const bool first = g == 0 || seg_unit[g] != seg_unit[g - 1];
        const int64_t cost = (first ? kUnitCostBytes : 0) + std::max<int64_t>(L, 1) * elem_bytes;
        if (cstart[g] > INT64_MAX / 2 - cost)
            return false;
        cstart[g + 1] = cstart[g] + cost;
    }
    const int64_t total = cstart[S];
    const int64_t want = (total + kMinRunBytes - 1) / kMinRunBytes;
    const int64_t W = std::max<int64_t>(1, std::min<int64_t>(want, max_runs));
    const int64_t align = std::max<int64_t>(1, kSplitBytes / elem_bytes);

    std::vector<Point> cuts;
    cuts.reserve(W + 1);
    cuts.push_back({0, 0});
    for (int64_t w = 1; w < W; ++w) {
        const int64_t target = (int64_t)((__int128)total * w / W);
        // segment g with cstart[g] <= target < cstart[g + 1]
        int64_t g = (int64_t)(std::upper_bound(cstart.begin(), cstart.end(), target) - cstart.begin()) - 1;
        g = std::min<int64_t>(std::max<int64_t>(g, 0), S - 1);
        const bool first = g == 0 || seg_unit[g] != seg_unit[g - 1];
        const int64_t local = target - cstart[g] - (first ? kUnitCostBytes : 0);
        int64_t pos = local <= 0 ? 0 : (local + elem_bytes - 1) / elem_bytes;
        pos = (pos + align - 1) / align * align;
        Point p{g, pos};
        if (pos >= std::max<int64_t>(seg_lengths[g], 1))
            p = {g + 1, 0};
        if (cuts.back() < p)
            cuts.push_back(p);
    }
    const Point end{S, 0};
    while (!(cuts.back() < end) && cuts.size() > 1)
        cuts.pop_back();
    cuts.push_back(end);

    const int64_t nw = (int64_t)cuts.size() - 1;
    out.num_runs = (int32_t)nw;
    out.run_seg.resize(nw + 1);
    out.run_pos.resize(nw + 1);
    for (int64_t w = 0; w <= nw; ++w) {
        out.run_seg[w] = cuts[w].seg;
        out.run_pos[w] = cuts[w].pos;
    }
    out.first_run.assign(U, -1);
    out.num_parts.assign(U, 0);
    for (int64_t w = 0; w < nw; ++w) {
        const int64_t g0 = cuts[w].seg;
        const int64_t last = cuts[w + 1].pos > 0 ? cuts[w + 1].seg : cuts[w + 1].seg - 1;
        int64_t prev_unit = -1;
        for (int64_t g = g0; g <= last; ++g) {
            const int64_t b = seg_unit[g];
            if (b == prev_unit)
                continue;
            prev_unit = b;
            if (out.first_run[b] < 0)
                out.first_run[b] = (int32_t)w;
            out.num_parts[b] += 1;
        }
    }
    out.part_base.resize(U);
    int64_t acc = 0;
    for (int64_t b = 0; b < U; ++b) {
        if (out.num_parts[b] < 1)
            return false;  // unreachable: every unit holds at least one point
        out.part_base[b] = acc;
        acc += out.num_parts[b];
    }
    out.num_partials = acc;
    return true;
}

}  // namespace gnmr
