// Work partition of the step kernel (host only).
//
// The units are concatenated in index order into one stream of "points": a
// unit of L elements contributes max(L, 1) points (an empty unit still needs
// one warp to run its Algorithm 1 update).  Each unit costs
// kUnitCostBytes + max(L, 1) * elem_bytes.  The stream is cut into runs of
// about equal cost, one run per warp, so skewed unit sizes (a 256-element
// unit next to a 70M-element one) balance across the grid: large units are
// split over many warps, small ones are packed many to a warp.
//
// Cuts inside a unit fall on multiples of kSplitBytes from the unit's start,
// so the body of every piece keeps the unit's 16-byte alignment.  Runs are
// strictly increasing and never empty, which makes the warps that touch a
// unit a contiguous range first_warp[b] .. first_warp[b] + num_parts[b] - 1;
// the kernel stores the partial sum of warp w for unit b in slot
// part_base[b] + (w - first_warp[b]), so the reduction order of a unit is
// fixed by the plan and results are bitwise reproducible run to run.
#include <algorithm>
#include <cstdint>
#include <utility>
#include <vector>

#include "gnmr_internal.h"

namespace gnmr {

namespace {

struct Point {
    int32_t unit;
    int64_t pos;
    bool operator<(const Point &o) const { return unit != o.unit ? unit < o.unit : pos < o.pos; }
    bool operator==(const Point &o) const { return unit == o.unit && pos == o.pos; }
};

}  // namespace

bool plan_partition(int32_t num_units, const int64_t *lengths, int elem_bytes,
                    int32_t max_warps, Plan &out)
{
    if (num_units < 1 || !lengths || (elem_bytes != 2 && elem_bytes != 4) || max_warps < 1)
        return false;
    const int64_t U = num_units;
    std::vector<int64_t> cstart(U + 1, 0);     // cost at the start of unit b
    for (int64_t b = 0; b < U; ++b) {
        int64_t L = lengths[b];
        if (L < 0 || L > (INT64_MAX / 8) / elem_bytes)
            return false;
        int64_t pts = std::max<int64_t>(L, 1);
        int64_t cost = kUnitCostBytes + pts * elem_bytes;
        if (cstart[b] > INT64_MAX / 2 - cost)
            return false;
        cstart[b + 1] = cstart[b] + cost;
    }
    const int64_t total = cstart[U];
    int64_t want = (total + kMinRunBytes - 1) / kMinRunBytes;
    const int64_t W = std::max<int64_t>(1, std::min<int64_t>(want, max_warps));
    const int64_t align = std::max<int64_t>(1, kSplitBytes / elem_bytes);

    std::vector<Point> cuts;
    cuts.reserve(W + 1);
    cuts.push_back({0, 0});
    for (int64_t w = 1; w < W; ++w) {
        const int64_t target = (int64_t)((__int128)total * w / W);
        // unit b with cstart[b] <= target < cstart[b + 1]
        int64_t b = (int64_t)(std::upper_bound(cstart.begin(), cstart.end(), target) - cstart.begin()) - 1;
        b = std::min<int64_t>(std::max<int64_t>(b, 0), U - 1);
        const int64_t local = target - cstart[b] - kUnitCostBytes;
        int64_t pos = local <= 0 ? 0 : (local + elem_bytes - 1) / elem_bytes;
        pos = (pos + align - 1) / align * align;
        Point p{(int32_t)b, pos};
        if (pos >= std::max<int64_t>(lengths[b], 1))
            p = {(int32_t)(b + 1), 0};
        if (cuts.back() < p)
            cuts.push_back(p);
    }
    const Point end{(int32_t)U, 0};
    while (!(cuts.back() < end) && cuts.size() > 1)
        cuts.pop_back();
    cuts.push_back(end);

    const int64_t nw = (int64_t)cuts.size() - 1;
    out.num_warps = (int32_t)nw;
    out.run_unit.resize(nw + 1);
    out.run_pos.resize(nw + 1);
    for (int64_t w = 0; w <= nw; ++w) {
        out.run_unit[w] = cuts[w].unit;
        out.run_pos[w] = cuts[w].pos;
    }
    out.first_warp.assign(U, -1);
    out.num_parts.assign(U, 0);
    for (int64_t w = 0; w < nw; ++w) {
        const int64_t u0 = cuts[w].unit;
        const int64_t last = cuts[w + 1].pos > 0 ? cuts[w + 1].unit : cuts[w + 1].unit - 1;
        for (int64_t b = u0; b <= last; ++b) {
            if (out.first_warp[b] < 0)
                out.first_warp[b] = (int32_t)w;
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
