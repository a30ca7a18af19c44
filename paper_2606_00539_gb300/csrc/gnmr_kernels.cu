// GNMR per-step monitor: one kernel launch per training step on sm_103a.
//
// Phase 1, every warp (the hot loop).  The segment stream (a unit is one or
// more segments of the arena) is cut by gnmr_plan.cpp into contiguous runs.
// With the small-unit loop each warp owns one run.  With the large-unit loop
// there are about 16 runs per warp: each warp starts on its own run and then
// takes the next untaken one from a counter, so warps that stream faster take
// more runs and all warps finish within about one run of each other (with one
// run per warp, HBM's uneven service left the slowest warps ~8 % of the step
// behind the median).  For every segment (or part of one) in a run the warp streams the
// gradient with 16-byte read-only loads (8 or 16 in flight per lane, by the
// loop shape), squares in fp32, sums blocks of 16 iterations in fp32 and the
// blocks as float pairs (error-free TwoSum), and all-reduces the lanes' totals
// across the warp with shuffles, converting to fp64 once per segment:
// n_b = ||g_b||_2 (Sec. 2, Eq. local_gradient).  No shared memory, no block
// barrier on this path.  (The streaming reduction lives in gnmr_stream.cuh.)
//
// Phase 2, the warp that completes unit b.  A unit split over several runs
// collects their partial sums through fixed slots (one per run, whichever
// warp streams it) and a per-unit ticket; the warp that takes the last ticket
// sums the slots in slot order (so the result does not depend on timing); a
// unit of two parts trades its partial in one atomic exchange.  Completed units queue up in the warp's lanes and run the
// unit epilogue 32 at a time, one unit per lane: Algorithm 1 (GNMR,
// Delta-GNMR, incremental mean, window queue), the combined risk
// R = max{GNMR/alpha_t, Delta-GNMR/beta_t} and the candidate test
// R > 1 or Lock > 0 (Sec. 3.3).  Candidates go to a compact list; members of
// the capped pool also count in a global risk histogram and, at or above the
// bin predicted from the previous step's cut, go to a short hot list.  Every
// unit's outcome if it is not selected is written here.
//
// Phase 3, the last CTA to finish (grid ticket): Top_maxO.  The histogram
// gives the bin that holds the maxO-th largest risk; one read of the hot list
// (or, if the prediction missed, of the whole list) commits every candidate
// above that bin, and the bin's own members are ranked on the 96-bit key
// (R descending, unit index ascending) in shared memory.  Then the lock
// bookkeeping of Algorithm 2 for the selected units, the counts, and the
// reset of the counters for the next launch.  No CTA ever waits for another:
// the tickets and the run counter decide who continues, so the kernel cannot
// hang whatever the grid size or residency.
//
// The same kernel also runs either half of a sharded step: phase 1 alone
// (per-unit sums of squares of a shard) or phases 2-3 alone on sums that the
// caller has added up across shards.
#include <cstdint>

#include <cuda_runtime.h>
#include <math_constants.h>

#include "gnmr_internal.h"
#include "gnmr_stream.cuh"

namespace gnmr {
namespace {

// Two compiled shapes of the streaming loop, chosen per handle from the mean
// unit size (both measured on GB300): many small units run best with 8
// 16-byte loads in flight per lane and two CTAs per SM; large units with 16
// loads per lane and one CTA per SM (fewer, deeper streams) and runs of at
// most 256 KiB taken dynamically.
template <int V> struct Shape;
template <> struct Shape<kVariantSmall> {
    static constexpr int kUnroll = 8;
    static constexpr int kMinCtas = 2;
    static constexpr bool kDynamic = false;           // one planned run per warp
};
template <> struct Shape<kVariantBulk> {
    static constexpr int kUnroll = 16;
    static constexpr int kMinCtas = 1;
    static constexpr bool kDynamic = true;            // further runs taken from a counter
};

__device__ __forceinline__ double pick_threshold(double override_value, int64_t t, int64_t warmup,
                                                 double init_value, double main_value)
{
    if (!isnan(override_value))
        return override_value;
    return t <= warmup ? init_value : main_value;
}

// Order-preserving keys: R >= 0 (never NaN), so its IEEE bits order like its
// value; the low word ranks lower unit indices higher.
__device__ __forceinline__ uint64_t risk_key(double r)
{
    const uint64_t bits = static_cast<uint64_t>(__double_as_longlong(r));
    return (bits << 1) == 0 ? 0ull : bits;           // -0 and +0 share the key 0 (integer test)
}
__device__ __forceinline__ uint32_t index_key(int32_t b, int32_t num_units)
{
    return static_cast<uint32_t>(num_units - 1 - b);
}

// Bin of the risk histogram for a risk key (non-decreasing in the key): 0 for
// R < 1, else 1 + the key's exponent and top three mantissa bits counted
// from those of 1.0, the last bin open-ended.
__device__ __forceinline__ uint32_t risk_bin(uint64_t key)
{
    constexpr uint32_t kOne = 1023u << 3;                 // exponent of 1.0, three mantissa bits 0
    const uint32_t e8 = static_cast<uint32_t>(key >> 49); // sign (0), exponent, top three mantissa bits
    if (e8 < kOne)
        return 0;
    const uint32_t b = e8 - kOne + 1;
    return b < static_cast<uint32_t>(kRiskBins) ? b : static_cast<uint32_t>(kRiskBins - 1);
}

// Appends the lanes' entries (flag set) to a list with one atomic per warp;
// slots at or past cap are counted but not written.  Called by all 32 lanes.
__device__ __forceinline__ void warp_append(Candidate *list, uint32_t *count, uint32_t cap, bool flag, double r,
                                            int32_t b, uint32_t lk)
{
    const unsigned want = __ballot_sync(kFull, flag);
    if (!want)
        return;
    const int lane = threadIdx.x & 31;
    const int leader = __ffs(want) - 1;
    uint32_t base = 0;
    if (lane == leader)
        base = atomicAdd(count, static_cast<uint32_t>(__popc(want)));
    base = __shfl_sync(kFull, base, leader);
    if (flag) {
        const uint32_t slot = base + __popc(want & ((1u << lane) - 1u));
        if (slot < cap) {
            list[slot].risk = r;
            list[slot].unit = b;
            list[slot].lock = lk;
        }
    }
}

// Unit epilogue for up to 32 units at once, one per lane (lanes with
// `active` false only take part in the collective append): Algorithm 1, the
// combined risk of Sec. 3.3, the statistics outputs and the candidate test of
// Algorithm 2.  Every lane issues its unit's loads together, so a batch costs
// about one memory round trip; candidates are appended with one atomic per
// warp.  Called by all 32 lanes.
__device__ void unit_epilogue(const StepParams &p, bool active, int32_t b, double sumsq,
                              double alpha, double beta, int64_t t)
{
    bool cand = false;
    double r = 0.0;
    uint32_t cand_lock = 0;
    // read now, used after the risk: the step's hot-list bin (only the
    // selection, after every CTA, rewrites it)
    const uint32_t hot_bin = __ldcg(&p.ctl->hot_bin);
    if (active) {
        const double n = sqrt(sumsq);
        const int w = p.window;
        double *Q = p.queue + static_cast<int64_t>(b) * w;
        // the window's lines travel with the state load: the window reads,
        // which need the state's head, then hit in L1
        asm volatile("prefetch.global.L1 [%0];" ::"l"(Q));
        asm volatile("prefetch.global.L1 [%0];" ::"l"(Q + (w - 1)));
        UnitState s = p.state[b];
        const bool rec = p.recoverable[b] != 0;
        // The risk first (its chain of dependent divisions decides the
        // epilogue's latency), the state update after it.
        double g, d;
        if (!isfinite(n)) {
            // Non-finite gradient: maximal risk, no change to A_b, Q_b, k_b.
            g = CUDART_INF;
            d = CUDART_INF;
        } else {
            // mean of the window, summed oldest to newest; its loads are issued
            // as soon as the state's head is known, before the division for g
            const bool full = s.fill == w;
            double q = 0.0;
            if (full) {
                int idx = s.head, k = 0;
                for (; k + 8 <= w; k += 8) {
                    double v[8];
#pragma unroll
                    for (int j = 0; j < 8; ++j) {
                        const int ix = idx + j < w ? idx + j : idx + j - w;
                        v[j] = Q[ix];
                    }
#pragma unroll
                    for (int j = 0; j < 8; ++j)
                        q += v[j];
                    idx = idx + 8 < w ? idx + 8 : idx + 8 - w;
                }
                for (; k < w; ++k) {
                    q += Q[idx];
                    idx = (idx + 1 == w) ? 0 : idx + 1;
                }
            }
            g = (s.count == 0 || s.mean == 0.0) ? 1.0 : n / (s.mean + p.eps);
            if (full) {
                const double den = q / static_cast<double>(w) + p.eps;
                d = (den == 0.0) ? (g > 0.0 ? CUDART_INF : 1.0) : g / den;
            } else {
                d = 1.0;
            }
        }
        const double x = g / alpha, y = d / beta;
        r = x > y ? x : y;
        if (isfinite(n)) {
            s.count += 1;
            s.mean = s.mean + (n - s.mean) / static_cast<double>(s.count);
            if (s.fill < w) {                        // still filling: head stays 0
                Q[s.fill] = g;
                s.fill += 1;
            } else {                                 // overwrite the oldest
                Q[s.head] = g;
                s.head = (s.head + 1 == w) ? 0 : s.head + 1;
            }
            p.state[b].mean = s.mean;
            p.state[b].count = s.count;
            p.state[b].fill = s.fill;
            p.state[b].head = s.head;
        }

        if (p.out_norm) p.out_norm[b] = n;
        if (p.out_gnmr) p.out_gnmr[b] = g;
        if (p.out_dgnmr) p.out_dgnmr[b] = d;
        if (p.out_risk) p.out_risk[b] = r;

        const bool stat = p.policy == 2;
        if (stat && t <= p.static_warmup && rec)
            p.state[b].gsum = s.gsum + g;
        if (t <= p.forced_steps || (stat && t <= p.static_warmup)) {
            // every recoverable unit on the recovery path; locks untouched
            p.mask[b] = rec ? 1 : 0;
            p.state[b].active = rec ? 1 : 0;
            if (p.out_lock) p.out_lock[b] = s.lock;
        } else if (stat) {
            if (t == p.static_warmup + 1 && rec) {
                cand = true;                          // ranked once by the warm-up's GNMR sum
                r = s.gsum;
                // outcome if not kept (the last CTA rewrites the kept units)
                p.mask[b] = 0;
                p.state[b].active = 0;
                if (p.out_lock) p.out_lock[b] = s.lock;
            } else {
                p.mask[b] = (rec && t > p.static_warmup + 1 && s.active) ? 1 : 0;
                if (t == p.static_warmup + 1)
                    p.state[b].active = 0;
                if (p.out_lock) p.out_lock[b] = s.lock;
            }
        } else {
            cand = rec && (r > 1.0 || s.lock > 0);
            // The outcome of a unit outside A_t (Algorithm 2: Lock_b = 0, low-cost
            // path), written here for every unit; the last CTA rewrites only the
            // selected ones.  A non-candidate's Lock_b is already 0.
            p.mask[b] = 0;
            p.state[b].active = 0;
            if (cand)
                p.state[b].lock = 0;
            if (p.out_lock) p.out_lock[b] = 0;
        }
        cand_lock = static_cast<uint32_t>(s.lock) | (s.active ? kCandActive : 0u);
    }
    // The capped pool: every candidate, or under the admission cap those not
    // active at t-1 (the retained ones are selected without ranking).  Pool
    // members count in the risk histogram; the hot list takes those at or
    // above this step's predicted bin, and every retained candidate.
    const bool retained = cand && p.policy == 1 && (cand_lock & kCandActive);
    bool hot = retained;
    if (cand && !retained) {
        const uint32_t bin = risk_bin(risk_key(r));
        atomicAdd(&p.risk_hist[bin], 1u);
        hot = bin >= hot_bin;
    }
    warp_append(p.cand, &p.ctl->n_cand, static_cast<uint32_t>(p.num_units), cand, r, b, cand_lock);
    warp_append(p.hot, &p.ctl->n_hot, p.hot_cap, hot, r, b, cand_lock);
}

// A unit split over several warps: stores this warp's partial and takes a
// ticket.  Returns true (with the unit's total in s) for the warp that takes
// the last ticket; that warp sums the partials in slot order.  A unit of two
// parts trades its partial through the first slot in one atomic exchange:
// the first warp finds the slot empty and leaves its partial there, the
// second takes it, adds it to its own (IEEE addition is commutative, so the
// bits are those of the slot-order sum) and empties the slot again.
__device__ __forceinline__ bool combine_parts(const StepParams &p, int32_t b, int32_t parts, int32_t run,
                                              double &s, int lane)
{
    const int64_t base = p.part_base[b];
    if (parts == 2) {
        unsigned long long other = 0;
        if (lane == 0) {
            const double mine = isnan(s) ? CUDART_NAN : s;          // never the empty pattern
            other = atomicExch(reinterpret_cast<unsigned long long *>(p.partial + base),
                               static_cast<unsigned long long>(__double_as_longlong(mine)));
        }
        other = __shfl_sync(kFull, other, 0);
        if (other == kEmptyPartial)
            return false;
        if (lane == 0)
            __stcg(reinterpret_cast<unsigned long long *>(p.partial + base), kEmptyPartial);
        s = s + __longlong_as_double(static_cast<long long>(other));
        return true;
    }
    uint32_t last = 0;
    if (lane == 0) {
        __stcg(&p.partial[base + (run - p.first_run[b])], s);
        last = ticket_acq_rel(&p.unit_ticket[b]) == static_cast<uint32_t>(parts - 1);
    }
    last = __shfl_sync(kFull, last, 0);
    if (!last)
        return false;
    __syncwarp();                                    // lane 0's acquire orders the lanes' loads
    double acc = 0.0;
    for (int32_t j = lane; j < parts; j += 32)
        acc += __ldcg(&p.partial[base + j]);
    s = warp_allreduce_sum(acc);
    if (lane == 0)
        p.unit_ticket[b] = 0;                        // ready for the next step
    return true;
}

__device__ __forceinline__ void load_candidate(const Candidate *c, double &r, int32_t &b, uint32_t &lock)
{
    const double2 v = __ldcg(reinterpret_cast<const double2 *>(c));
    const uint64_t w = static_cast<uint64_t>(__double_as_longlong(v.y));
    r = v.x;
    b = static_cast<int32_t>(w & 0xffffffffu);
    lock = static_cast<uint32_t>(w >> 32);
}

// Bucket of the r-th largest digit in hist[256] (r >= 1): misc[1] = the
// bucket, misc[2] = r minus the count above it, misc[3] = its count.  Warp 0
// scans; the caller synchronises before and after.
__device__ __forceinline__ void find_bucket(const uint32_t *hist, uint32_t r, uint32_t *misc)
{
    if (threadIdx.x >= 32)
        return;
    const int l = threadIdx.x;                       // lane l owns buckets 255-8l down to 248-8l
    const uint4 *v = reinterpret_cast<const uint4 *>(hist + 248 - 8 * l);
    const uint4 a = v[0], b = v[1];                  // buckets 248-8l .. 255-8l, ascending
    const uint32_t c8[8] = {b.w, b.z, b.y, b.x, a.w, a.z, a.y, a.x};   // descending
    uint32_t sum = 0;
#pragma unroll
    for (int j = 0; j < 8; ++j)
        sum += c8[j];
    uint32_t incl = sum;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const uint32_t v = __shfl_up_sync(kFull, incl, o);
        if (l >= o)
            incl += v;
    }
    const uint32_t excl = incl - sum;
    if (excl < r && r <= incl) {                     // exactly one lane
        uint32_t above = excl;
#pragma unroll
        for (int j = 0; j < 8; ++j) {
            if (above + c8[j] >= r) {
                misc[1] = static_cast<uint32_t>(255 - 8 * l - j);
                misc[2] = r - above;
                misc[3] = c8[j];
                break;
            }
            above += c8[j];
        }
    }
}

// Candidate loads a thread keeps in flight in each selection pass.
constexpr int kSelectIlp = 6;

// K-th largest 96-bit key (risk_key : index_key) among the m candidates (or
// among those not active at t-1 when only_new), 1 <= K < that count, by
// most-significant-digit radix select with 8-bit digits.
// Returns the threshold: exactly K keys compare >= it.  All threads of the
// CTA call this.
__device__ void radix_select(const StepParams &p, uint32_t m, uint32_t K, bool only_new, uint32_t *hist,
                             uint32_t *misc, uint64_t &thr_hi, uint32_t &thr_lo)
{
    const int lo_bits = p.num_units > 1 ? 32 - __clz(static_cast<uint32_t>(p.num_units - 1)) : 0;
    const int lo_digits = (lo_bits + 7) / 8;
    uint64_t pre_hi = 0, msk_hi = 0;
    uint32_t pre_lo = 0, msk_lo = 0;
    uint32_t r = K;
    for (int dgt = 0; dgt < 8 + lo_digits; ++dgt) {
        const bool in_hi = dgt < 8;
        const int shift = in_hi ? 56 - 8 * dgt : 8 * (lo_digits - 1 - (dgt - 8));
        for (int i = threadIdx.x; i < 256; i += blockDim.x)
            hist[i] = 0;
        __syncthreads();
        for (uint32_t i0 = threadIdx.x; i0 < m; i0 += kSelectIlp * blockDim.x) {
            double rr[kSelectIlp];
            int32_t bb[kSelectIlp];
            uint32_t ll[kSelectIlp];
#pragma unroll
            for (int j = 0; j < kSelectIlp; ++j) {  // loads in flight per thread
                const uint32_t i = i0 + j * blockDim.x;
                if (i < m)
                    load_candidate(p.cand + i, rr[j], bb[j], ll[j]);
            }
#pragma unroll
            for (int j = 0; j < kSelectIlp; ++j) {
                if (i0 + j * blockDim.x >= m)
                    break;
                if (only_new && (ll[j] & kCandActive))
                    continue;
                const uint64_t hi = risk_key(rr[j]);
                const uint32_t lo = index_key(bb[j], p.num_units);
                if ((hi & msk_hi) == pre_hi && (lo & msk_lo) == pre_lo) {
                    const uint32_t dig = in_hi ? static_cast<uint32_t>(hi >> shift) & 0xffu
                                               : (lo >> shift) & 0xffu;
                    atomicAdd(&hist[dig], 1u);
                }
            }
        }
        __syncthreads();
        find_bucket(hist, r, misc);
        __syncthreads();
        const uint32_t bucket = misc[1];
        const uint32_t in_bucket = misc[3];
        r = misc[2];
        if (in_hi) {
            pre_hi |= static_cast<uint64_t>(bucket) << shift;
            msk_hi |= 0xffull << shift;
        } else {
            pre_lo |= bucket << shift;
            msk_lo |= 0xffu << shift;
        }
        __syncthreads();
        if (in_bucket == r)                          // every key with this prefix is in
            break;
    }
    thr_hi = pre_hi;
    thr_lo = pre_lo;
}

// Delta M_t = sum of c_b over the units on the recovery path, in a fixed
// order (thread-strided partial sums, then a fixed tree), so the value is
// reproducible run to run.
__device__ void delta_mem(const StepParams &p, double *red)
{
    double acc = 0.0;
    for (int32_t b = threadIdx.x; b < p.num_units; b += blockDim.x)
        if (__ldcg(p.mask + b))
            acc += p.unit_cost[b];
    red[threadIdx.x] = acc;
    __syncthreads();
    for (unsigned o = blockDim.x / 2; o > 0; o >>= 1) {
        if (threadIdx.x < o)
            red[threadIdx.x] += red[threadIdx.x + o];
        __syncthreads();
    }
    if (threadIdx.x == 0)
        *p.out_delta_mem = red[0];
}

// Algorithm 2's outcome for a unit in A_t (the epilogue has already written
// the outcome for every unit outside it).
__device__ __forceinline__ void commit_selected(const StepParams &p, bool stat, int32_t b, double r, uint32_t lk)
{
    p.mask[b] = 1;
    if (stat) {
        p.state[b].active = 1;                       // the static policy keeps no locks
    } else {
        const int32_t prev = static_cast<int32_t>(lk & ~kCandActive);
        const int32_t next = r > 1.0 ? p.lock_len : (prev - 1 > 0 ? prev - 1 : 0);
        *reinterpret_cast<int2 *>(&p.state[b].lock) = make_int2(next, 1);   // lock, active
        if (p.out_lock) p.out_lock[b] = next;
    }
}

// The selecting CTA's shared memory: the cut list (the pool members of the
// bin that holds the maxO-th largest risk, when only part of that bin is
// selected: key, unit, lock word) and, for a cut bin too large to rank
// directly, the histogram of an in-CTA radix select over it.
constexpr int kWideBits = 11;
constexpr int kWideBins = 1 << kWideBits;
static_assert(kWideBins == 4 * kThreads, "four histogram bins per thread of the selecting CTA");
static_assert(kRiskBins == 4 * kThreads, "four risk-histogram bins per thread of the selecting CTA");
constexpr uint32_t kCutCap = 3072;
constexpr size_t kCutUnitOffset = sizeof(uint64_t) * kCutCap;
constexpr size_t kCutLockOffset = kCutUnitOffset + sizeof(int32_t) * kCutCap;
constexpr size_t kCutHistOffset = kCutLockOffset + sizeof(uint32_t) * kCutCap;
constexpr size_t kKeyCacheBytes = kCutHistOffset + sizeof(uint32_t) * kWideBins;
static_assert(kCutHistOffset % 16 == 0, "the histogram is read as 16-byte vectors");

// Slots of the selecting CTA's misc[] words.
constexpr int kMiscLast = 0;      // this CTA took the last grid ticket
constexpr int kMiscBin = 1;       // find_*: the bin holding the r-th largest
constexpr int kMiscRank = 2;      // r minus the count above that bin
constexpr int kMiscCount = 3;     // that bin's count
constexpr int kMiscHint = 5;      // scan_risk_hist: the bin holding the hint-th largest
constexpr int kMiscPool = 6;      // scan_risk_hist: the pool size
constexpr int kMiscFill = 7;      // cut-list entries appended

// Bin of the r-th largest digit in hist[kWideBins] (r >= 1), by the whole
// CTA: thread t owns the four bins just below those of thread t - 1 (thread
// 0 the highest); the counts above each thread's bins come from a warp scan
// and a scan of the 16 warp totals (in wsum[16]).
__device__ __forceinline__ void find_bucket_wide(const uint32_t *hist, uint32_t r, uint32_t *misc, uint32_t *wsum)
{
    const int t = threadIdx.x, lane = t & 31, wid = t >> 5;
    const int q4 = kWideBins / 4 - 1 - t;
    const uint4 q = reinterpret_cast<const uint4 *>(hist)[q4];      // bins 4 q4 .. 4 q4 + 3
    const uint32_t c4[4] = {q.w, q.z, q.y, q.x};                     // descending
    const uint32_t sum = c4[0] + c4[1] + c4[2] + c4[3];
    uint32_t incl = sum;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const uint32_t u = __shfl_up_sync(kFull, incl, o);
        if (lane >= o)
            incl += u;
    }
    if (lane == 31)
        wsum[wid] = incl;
    __syncthreads();
    if (wid == 0) {
        const uint32_t tot = lane < kWarpsPerCta ? wsum[lane] : 0u;
        uint32_t x = tot;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const uint32_t u = __shfl_up_sync(kFull, x, o);
            if (lane >= o)
                x += u;
        }
        if (lane < kWarpsPerCta)
            wsum[lane] = x - tot;                    // counts in the warps' higher bins
    }
    __syncthreads();
    uint32_t above = wsum[wid] + incl - sum;
    if (above < r && r <= above + sum) {             // exactly one thread
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            if (above + c4[j] >= r) {
                misc[kMiscBin] = static_cast<uint32_t>(4 * q4 + 3 - j);
                misc[kMiscRank] = r - above;
                misc[kMiscCount] = c4[j];
                break;
            }
            above += c4[j];
        }
    }
}

// Reads and clears the global risk histogram (four bins per thread, thread 0
// the highest).  misc[kMiscPool] = the pool size P; with K = min(P, cap),
// if 1 <= K < P: misc[kMiscBin/Rank/Count] describe the bin holding the K-th
// largest risk, and misc[kMiscHint] the bin holding the min(P, K + extra)-th
// largest (the next step's hot-list prediction).  Callers synchronise after.
__device__ void scan_risk_hist(const StepParams &p, uint32_t cap, uint32_t extra, uint32_t *misc, uint32_t *wsum)
{
    const int t = threadIdx.x, lane = t & 31, wid = t >> 5;
    const int q4 = kRiskBins / 4 - 1 - t;
    uint4 *gh = reinterpret_cast<uint4 *>(p.risk_hist) + q4;
    const uint4 q = __ldcg(gh);                                      // bins 4 q4 .. 4 q4 + 3
    __stcg(gh, make_uint4(0u, 0u, 0u, 0u));                          // empty for the next step
    const uint32_t c4[4] = {q.w, q.z, q.y, q.x};                     // descending
    const uint32_t sum = c4[0] + c4[1] + c4[2] + c4[3];
    uint32_t incl = sum;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const uint32_t u = __shfl_up_sync(kFull, incl, o);
        if (lane >= o)
            incl += u;
    }
    if (lane == 31)
        wsum[wid] = incl;
    __syncthreads();
    if (wid == 0) {
        const uint32_t tot = lane < kWarpsPerCta ? wsum[lane] : 0u;
        uint32_t x = tot;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const uint32_t u = __shfl_up_sync(kFull, x, o);
            if (lane >= o)
                x += u;
        }
        if (lane < kWarpsPerCta)
            wsum[lane] = x - tot;
        if (lane == kWarpsPerCta - 1)
            misc[kMiscPool] = x;
    }
    __syncthreads();
    const uint32_t pool = misc[kMiscPool];
    const uint32_t K = pool < cap ? pool : cap;
    if (K == 0 || K >= pool)
        return;
    const uint32_t r2 = pool - K > extra ? K + extra : pool;
    const uint32_t above0 = wsum[wid] + incl - sum;
    if (above0 < K && K <= above0 + sum) {
        uint32_t above = above0;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            if (above + c4[j] >= K) {
                misc[kMiscBin] = static_cast<uint32_t>(4 * q4 + 3 - j);
                misc[kMiscRank] = K - above;
                misc[kMiscCount] = c4[j];
                break;
            }
            above += c4[j];
        }
    }
    if (above0 < r2 && r2 <= above0 + sum) {
        uint32_t above = above0;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            if (above + c4[j] >= r2) {
                misc[kMiscHint] = static_cast<uint32_t>(4 * q4 + 3 - j);
                break;
            }
            above += c4[j];
        }
    }
}

// One read of n list entries: commits every retained entry (admission cap)
// and every pool entry in a bin above c; the pool entries of bin c are
// committed too when the whole bin is selected, else collected in the cut
// list (misc[kMiscFill] counts them; at most kCutCap are stored).
__device__ void gather_commit(const StepParams &p, const Candidate *src, uint32_t n, bool admission, bool stat,
                              uint32_t c, bool whole_bin, uint64_t *ck, int32_t *cu, uint32_t *cl, uint32_t *misc)
{
    for (uint32_t i0 = threadIdx.x; i0 < n; i0 += kSelectIlp * blockDim.x) {
        double rr[kSelectIlp];
        int32_t bb[kSelectIlp];
        uint32_t ll[kSelectIlp];
#pragma unroll
        for (int j = 0; j < kSelectIlp; ++j) {      // loads in flight per thread
            const uint32_t i = i0 + j * blockDim.x;
            if (i < n)
                load_candidate(src + i, rr[j], bb[j], ll[j]);
        }
#pragma unroll
        for (int j = 0; j < kSelectIlp; ++j) {
            if (i0 + j * blockDim.x >= n)
                break;
            if (admission && (ll[j] & kCandActive)) {
                commit_selected(p, stat, bb[j], rr[j], ll[j]);
                continue;
            }
            const uint64_t key = risk_key(rr[j]);
            const uint32_t bin = risk_bin(key);
            if (bin > c || (bin == c && whole_bin)) {
                commit_selected(p, stat, bb[j], rr[j], ll[j]);
            } else if (bin == c) {
                const uint32_t at = atomicAdd(&misc[kMiscFill], 1u);
                if (at < kCutCap) {
                    ck[at] = key;
                    cu[at] = bb[j];
                    cl[at] = ll[j];
                }
            }
        }
    }
}

// r-th largest (key : index_key) among the n <= kCutCap cut-list entries,
// 1 <= r < n: MSD radix select with 11-bit digits on shared memory, starting
// at bit `start` of the 64-bit key (the bits above it are equal for every
// entry), then over the unit indices when whole keys tie.  Exactly r entries
// compare >= the returned threshold.  All threads of the CTA call this.
__device__ void radix_select_cut(const uint64_t *keys, const int32_t *units, uint32_t n, uint32_t r, int start,
                                 int32_t num_units, uint32_t *hist, uint32_t *wsum, uint32_t *misc,
                                 uint64_t &thr_hi, uint32_t &thr_lo)
{
    const int lo_bits = num_units > 1 ? 32 - __clz(static_cast<uint32_t>(num_units - 1)) : 0;
    uint64_t pre_hi = 0, msk_hi = start < 64 ? ~0ull << start : 0ull;
    if (start < 64)
        pre_hi = keys[0] & msk_hi;
    uint32_t pre_lo = 0, msk_lo = 0;
    int pos_hi = start, pos_lo = lo_bits;
    while (pos_hi > 0 || pos_lo > 0) {
        const bool in_hi = pos_hi > 0;
        int &pos = in_hi ? pos_hi : pos_lo;
        const int width = pos < kWideBits ? pos : kWideBits;
        pos -= width;
        const int shift = pos;
        const uint32_t dmask = (1u << width) - 1u;
        reinterpret_cast<uint4 *>(hist)[threadIdx.x] = make_uint4(0u, 0u, 0u, 0u);
        __syncthreads();
        for (uint32_t i = threadIdx.x; i < n; i += blockDim.x) {
            const uint64_t hi = keys[i];
            if ((hi & msk_hi) != pre_hi)
                continue;
            uint32_t dig;
            if (in_hi) {
                dig = static_cast<uint32_t>(hi >> shift) & dmask;
            } else {                                  // whole keys tie: rank by unit index
                const uint32_t lo = index_key(units[i], num_units);
                if ((lo & msk_lo) != pre_lo)
                    continue;
                dig = (lo >> shift) & dmask;
            }
            atomicAdd(&hist[dig], 1u);
        }
        __syncthreads();
        find_bucket_wide(hist, r, misc, wsum);
        __syncthreads();
        const uint32_t bucket = misc[kMiscBin];
        const uint32_t in_bucket = misc[kMiscCount];
        r = misc[kMiscRank];
        if (in_hi) {
            pre_hi |= static_cast<uint64_t>(bucket) << shift;
            msk_hi |= static_cast<uint64_t>(dmask) << shift;
        } else {
            pre_lo |= bucket << shift;
            msk_lo |= dmask << shift;
        }
        __syncthreads();
        if (in_bucket == r)                          // every key with this prefix is in
            break;
    }
    thr_hi = pre_hi;
    thr_lo = pre_lo;
}

// Does entry (kj, uj) rank above (k, u)?  Risk descending, then unit ascending.
__device__ __forceinline__ uint32_t ranks_above(uint64_t kj, int32_t uj, uint64_t k, int32_t u)
{
    return (kj > k) | ((kj == k) & (uj < u));
}

// Commits the r largest (key desc, unit asc) of the n cut-list entries,
// 1 <= r < n <= kCutCap.  Each entry's rank is counted against all others
// directly: up to 32 entries in warp 0's registers (shuffles), up to one per
// thread from shared memory (eight entries per step, loads issued together);
// larger lists use the radix select.
__device__ void select_cut(const StepParams &p, bool stat, uint32_t c, uint32_t n, uint32_t r, const uint64_t *ck,
                           const int32_t *cu, const uint32_t *cl, uint32_t *hist, uint32_t *wsum, uint32_t *misc)
{
    if (n <= 32) {
        if (threadIdx.x < 32) {
            const uint32_t i = threadIdx.x;
            const bool mine = i < n;
            const uint64_t k = mine ? ck[i] : 0ull;
            const int32_t u = mine ? cu[i] : 0;
            uint32_t rank = 0;
#pragma unroll
            for (int j = 0; j < 32; ++j) {
                const uint64_t kj = __shfl_sync(kFull, k, j);
                const int32_t uj = __shfl_sync(kFull, u, j);
                rank += (static_cast<uint32_t>(j) < n) ? ranks_above(kj, uj, k, u) : 0u;
            }
            if (mine && rank < r)
                commit_selected(p, stat, u, __longlong_as_double(static_cast<long long>(k)), cl[i]);
        }
        return;
    }
    if (n <= blockDim.x) {
        const uint32_t i = threadIdx.x;
        if (i < n) {
            const uint64_t k = ck[i];
            const int32_t u = cu[i];
            uint32_t rank = 0;
            uint32_t j = 0;
            for (; j + 8 <= n; j += 8) {
                uint64_t kj[8];
                int32_t uj[8];
#pragma unroll
                for (int q = 0; q < 8; ++q) {
                    kj[q] = ck[j + q];
                    uj[q] = cu[j + q];
                }
#pragma unroll
                for (int q = 0; q < 8; ++q)
                    rank += ranks_above(kj[q], uj[q], k, u);
            }
            for (; j < n; ++j)
                rank += ranks_above(ck[j], cu[j], k, u);
            if (rank < r)
                commit_selected(p, stat, u, __longlong_as_double(static_cast<long long>(k)), cl[i]);
        }
        return;
    }
    // every key of an interior bin shares the sign, exponent and top three mantissa bits
    const int start = (c > 0 && c + 1 < static_cast<uint32_t>(kRiskBins)) ? 49 : 64;
    uint64_t thr_hi = 0;
    uint32_t thr_lo = 0;
    radix_select_cut(ck, cu, n, r, start, p.num_units, hist, wsum, misc, thr_hi, thr_lo);
    for (uint32_t i = threadIdx.x; i < n; i += blockDim.x) {
        const uint64_t k = ck[i];
        if (k > thr_hi || (k == thr_hi && index_key(cu[i], p.num_units) >= thr_lo))
            commit_selected(p, stat, cu[i], __longlong_as_double(static_cast<long long>(k)), cl[i]);
    }
}

// Last CTA: Top_maxO (or the policy's choice), Algorithm 2's lock
// bookkeeping, mask, counts, Delta M_t, reset.  The unit epilogues have
// already written the outcome of every unit outside A_t; this writes A_t.
//
// The risk histogram gives the pool size and the bin c that holds the
// maxO-th largest risk.  One read of a list then commits every entry above c
// (and the retained ones), and the pool members of bin c are ranked among
// themselves.  The list read is the hot list when the previous step's
// prediction was at or below c and the hot list did not overflow (it then
// holds every entry at or above c), else the whole candidate list.
__device__ void select_and_commit(const StepParams &p, int64_t t, uint32_t *hist, uint32_t *misc, double *red,
                                  unsigned char *smem)
{
    uint32_t m = __ldcg(&p.ctl->n_cand);
    m = m < static_cast<uint32_t>(p.num_units) ? m : static_cast<uint32_t>(p.num_units);
    const bool all_on = t <= p.forced_steps || (p.policy == 2 && t <= p.static_warmup);
    const bool stat = p.policy == 2 && !all_on;
    const bool admission = p.policy == 1 && !all_on;
    uint32_t n_sel = 0;
    uint32_t next_hot = kNoHot + 1;                  // > kNoHot: keep the current prediction
    if (all_on) {
        m = 0;
        n_sel = static_cast<uint32_t>(p.num_recoverable);
    } else if (stat && t > p.static_warmup + 1) {
        m = 0;
        n_sel = static_cast<uint32_t>(p.static_keep);
    } else if (!admission && m <= (stat ? static_cast<uint32_t>(p.static_keep) : static_cast<uint32_t>(p.max_o))) {
        // every candidate is in the pool and the pool fits the budget: one read of the
        // list commits all of it and empties the histogram bins it filled (no scan)
        for (uint32_t i = threadIdx.x; i < m; i += blockDim.x) {
            double r;
            int32_t b;
            uint32_t lk;
            load_candidate(p.cand + i, r, b, lk);
            commit_selected(p, stat, b, r, lk);
            __stcg(p.risk_hist + risk_bin(risk_key(r)), 0u);
        }
        n_sel = m;
        next_hot = 0;                                // a small pool: every candidate is hot next step
    } else {
        const uint32_t cap = stat ? static_cast<uint32_t>(p.static_keep) : static_cast<uint32_t>(p.max_o);
        scan_risk_hist(p, cap, 3 * cap + 64, misc, hist);
        __syncthreads();
        const uint32_t pool = misc[kMiscPool];
        const uint32_t retained = admission && m > pool ? m - pool : 0u;
        const uint32_t K = pool < cap ? pool : cap;
        if (K == 0 || K >= pool) {
            // the whole pool is selected (or none of it): one read of the list
            const bool take_all = K >= pool;
            for (uint32_t i = threadIdx.x; i < m; i += blockDim.x) {
                double r;
                int32_t b;
                uint32_t lk;
                load_candidate(p.cand + i, r, b, lk);
                if (take_all || (admission && (lk & kCandActive)))
                    commit_selected(p, stat, b, r, lk);
            }
            next_hot = 0;                            // a small pool: every candidate is hot next step
        } else {
            uint64_t *ck = reinterpret_cast<uint64_t *>(smem);
            int32_t *cu = reinterpret_cast<int32_t *>(smem + kCutUnitOffset);
            uint32_t *cl = reinterpret_cast<uint32_t *>(smem + kCutLockOffset);
            uint32_t *wide_hist = reinterpret_cast<uint32_t *>(smem + kCutHistOffset);
            const uint32_t c = misc[kMiscBin], rc = misc[kMiscRank], nc = misc[kMiscCount];
            next_hot = misc[kMiscHint];
            const uint32_t hot_bin = __ldcg(&p.ctl->hot_bin);
            const uint32_t n_hot = __ldcg(&p.ctl->n_hot);
            const bool use_hot = hot_bin <= c && n_hot <= p.hot_cap;
            __syncthreads();                         // every thread has read misc
            if (threadIdx.x == 0)
                misc[kMiscFill] = 0;
            __syncthreads();
            gather_commit(p, use_hot ? p.hot : p.cand, use_hot ? n_hot : m, admission, stat, c, rc == nc,
                          ck, cu, cl, misc);
            __syncthreads();
            if (rc < nc) {
                if (nc <= kCutCap) {
                    select_cut(p, stat, c, nc, rc, ck, cu, cl, wide_hist, hist, misc);
                } else {
                    // a cut bin larger than the shared list: radix passes over the
                    // whole candidate list in global memory (commits are idempotent)
                    uint64_t thr_hi = 0;
                    uint32_t thr_lo = 0;
                    radix_select(p, m, K, admission, hist, misc, thr_hi, thr_lo);
                    for (uint32_t i = threadIdx.x; i < m; i += blockDim.x) {
                        double r;
                        int32_t b;
                        uint32_t lk;
                        load_candidate(p.cand + i, r, b, lk);
                        const uint64_t key = risk_key(r);
                        if ((admission && (lk & kCandActive)) || key > thr_hi ||
                            (key == thr_hi && index_key(b, p.num_units) >= thr_lo))
                            commit_selected(p, stat, b, r, lk);
                    }
                }
            }
        }
        n_sel = K + retained;
    }
    if (threadIdx.x == 0 && p.out_counts) {
        p.out_counts[0] = static_cast<int32_t>(m);
        p.out_counts[1] = static_cast<int32_t>(n_sel);
    }
    __syncthreads();
    if (p.unit_cost && p.out_delta_mem) {
        __threadfence_block();
        delta_mem(p, red);
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        p.ctl->next_run = 0;                         // every CTA, so every warp, is done
        p.ctl->n_cand = 0;
        p.ctl->n_hot = 0;
        if (next_hot <= kNoHot)
            p.ctl->hot_bin = next_hot;
        p.ctl->ctas_done = 0;
        p.ctl->steps += 1;
    }
}

// MODE kStepFull: the whole step.  kStepPartials: phase 1 only, each unit's
// sum of squares written to out_sumsq (the first half of a sharded step).
// kStepFinish: no gradient read; phases 2-3 on the sums in in_sumsq (the
// second half, after the caller has reduced the shards' sums).
template <int DT, int MODE, int V>
__global__ void __launch_bounds__(kThreads, Shape<V>::kMinCtas)
gnmr_step_kernel(const __grid_constant__ StepParams p)
{
    __shared__ __align__(16) uint32_t s_hist[256];
    __shared__ uint32_t s_misc[8];
    __shared__ double s_red[kThreads];
    extern __shared__ __align__(16) unsigned char s_keys[];   // kKeyCacheBytes unless MODE == kStepPartials
    constexpr int kEB = Elem<DT>::kBytes;
    const int lane = threadIdx.x & 31;
    const int warp = blockIdx.x * kWarpsPerCta + (threadIdx.x >> 5);
    // Launched as a programmatic dependent of whatever precedes it on the
    // stream: wait here until that kernel has completed and its writes are
    // visible (the arena, the previous step's state), then let the next step
    // launch as soon as it finds room on an SM (it waits here too).
    asm volatile("griddepcontrol.wait;" ::: "memory");
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

    if (MODE == kStepFinish) {
        const int64_t t = __ldcg(&p.ctl->steps) + 1;
        const double alpha = pick_threshold(p.alpha_override, t, p.warmup_steps, p.alpha_init, p.alpha_main);
        const double beta = pick_threshold(p.beta_override, t, p.warmup_steps, p.beta_init, p.beta_main);
        const int64_t warps = static_cast<int64_t>(gridDim.x) * kWarpsPerCta;
        for (int64_t b0 = static_cast<int64_t>(warp) * 32; b0 < p.num_units; b0 += warps * 32) {
            const int64_t b = b0 + lane;
            const bool active = b < p.num_units;
            const double s = active ? p.in_sumsq[b] : 0.0;
            unit_epilogue(p, active, active ? static_cast<int32_t>(b) : 0, s, alpha, beta, t);
        }
    } else if (warp < p.num_warps) {
        // t, alpha_t and beta_t are fixed for the whole step.
        const int64_t t = __ldcg(&p.ctl->steps) + 1;
        const double alpha = pick_threshold(p.alpha_override, t, p.warmup_steps, p.alpha_init, p.alpha_main);
        const double beta = pick_threshold(p.beta_override, t, p.warmup_steps, p.beta_init, p.beta_main);
        const char *arena = static_cast<const char *>(p.arena);
        // Units this warp completes wait here, lane j holding the j-th, and run
        // their epilogues 32 at a time.
        int32_t pend_b = 0;
        double pend_s = 0.0;
        int npend = 0;
        int32_t run = warp;                              // every warp starts on its own run
        auto complete = [&](int32_t b, double s) {
            const int32_t parts = p.num_parts[b];
            if (parts == 1 || combine_parts(p, b, parts, run, s, lane)) {
                if (MODE == kStepPartials) {
                    if (lane == 0)
                        p.out_sumsq[b] = s;
                } else {
                    if (lane == npend) {
                        pend_b = b;
                        pend_s = s;
                    }
                    if (++npend == 32) {
                        unit_epilogue(p, true, pend_b, pend_s, alpha, beta, t);
                        npend = 0;
                    }
                }
            }
        };
        for (;;) {
            // Large-unit loop: the index of the warp's next run is taken now, so
            // the atomic's round trip hides under this run's stream.
            uint32_t next = 0;
            if (Shape<V>::kDynamic && lane == 0)
                next = atomicAdd(&p.ctl->next_run, 1u);
            int64_t g = p.run_seg[run];
            int64_t pos = p.run_pos[run];
            const int64_t g_end = p.run_seg[run + 1];
            const int64_t pos_end = p.run_pos[run + 1];
            // Segments of one unit are consecutive: their sums add up in segment
            // order until the unit changes.
            int32_t cur = -1;
            double cur_s = 0.0;
            while (g < g_end || (g == g_end && pos < pos_end)) {
                const int32_t b = p.seg_unit[g];
                const int64_t len = p.length[g];
                int64_t stop = (g == g_end) ? pos_end : len;
                stop = stop < len ? stop : len;
                const int64_t n = stop > pos ? stop - pos : 0;
                const char *seg = arena + (p.offset[g] + pos) * kEB;
                bool suspect;
                double s = warp_segment_sumsq<DT, Shape<V>::kUnroll>(seg, n, lane, suspect);
                if (suspect)
                    s = warp_segment_sumsq_f64<DT>(seg, n, lane);
                if (b != cur) {
                    if (cur >= 0)
                        complete(cur, cur_s);
                    cur = b;
                    cur_s = s;
                } else {
                    cur_s += s;
                }
                ++g;
                pos = 0;
            }
            if (cur >= 0)
                complete(cur, cur_s);
            if (!Shape<V>::kDynamic)
                break;
            run = p.num_warps + static_cast<int32_t>(__shfl_sync(kFull, next, 0));
            if (run >= p.num_runs)
                break;
        }
        // The run counter is reset for the next launch (which starts only
        // after this grid has completed) by the selecting CTA, after every
        // warp has drawn its last index.  The partial-sums half has no
        // selecting CTA: there the last warp to draw past the end resets it.
        if (Shape<V>::kDynamic && MODE == kStepPartials && lane == 0 &&
            ticket_acq_rel(&p.ctl->warps_done) == static_cast<uint32_t>(p.num_warps - 1)) {
            p.ctl->next_run = 0;
            p.ctl->warps_done = 0;
        }
        if (MODE != kStepPartials && npend > 0)
            unit_epilogue(p, lane < npend, pend_b, pend_s, alpha, beta, t);
    }
    if (MODE == kStepPartials)
        return;

    // Grid completion: the last CTA through runs the selection.  The barrier
    // orders the CTA's writes before thread 0's release; the last ticket's
    // acquire, then the barrier, orders the selecting CTA's reads after
    // every CTA's writes.
    __syncthreads();
    if (threadIdx.x == 0)
        s_misc[kMiscLast] = ticket_acq_rel(&p.ctl->ctas_done) == gridDim.x - 1 ? 1u : 0u;
    __syncthreads();
    if (s_misc[kMiscLast]) {
        select_and_commit(p, __ldcg(&p.ctl->steps) + 1, s_hist, s_misc, s_red, s_keys);
    }
}

template <int MODE, int V>
cudaError_t launch_mode(const StepParams &p, int dtype, int num_ctas, cudaStream_t stream)
{
    constexpr size_t smem = MODE == kStepPartials ? 0 : kKeyCacheBytes;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(static_cast<unsigned>(num_ctas));
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    if (dtype == 1)
        return cudaLaunchKernelEx(&cfg, gnmr_step_kernel<1, MODE, V>, p);
    return cudaLaunchKernelEx(&cfg, gnmr_step_kernel<0, MODE, V>, p);
}

template <int V>
cudaError_t launch_variant(const StepParams &p, int dtype, int num_ctas, cudaStream_t stream, int mode)
{
    if (mode == kStepPartials)
        return launch_mode<kStepPartials, V>(p, dtype, num_ctas, stream);
    return launch_mode<kStepFull, V>(p, dtype, num_ctas, stream);
}

}  // namespace

cudaError_t launch_step(const StepParams &p, int dtype, int num_ctas, cudaStream_t stream, int mode,
                        int variant)
{
    if (mode == kStepFinish)                      // no gradient read: one shape is enough
        return launch_mode<kStepFinish, kVariantSmall>(p, 0, num_ctas, stream);
    if (variant == kVariantBulk)
        return launch_variant<kVariantBulk>(p, dtype, num_ctas, stream, mode);
    return launch_variant<kVariantSmall>(p, dtype, num_ctas, stream, mode);
}

namespace {

// The key cache is dynamic shared memory above the 48 KiB default, an opt-in
// that is a per-device function attribute: set for every instance a handle
// launches, on the current device.
template <int DT, int V>
cudaError_t prepare_variant(int *ctas_per_sm)
{
    const int bytes = static_cast<int>(kKeyCacheBytes);
    cudaError_t e = cudaFuncSetAttribute(gnmr_step_kernel<DT, kStepFull, V>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
    if (e == cudaSuccess)
        e = cudaFuncSetAttribute(gnmr_step_kernel<0, kStepFinish, kVariantSmall>,
                                 cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
    if (e == cudaSuccess)
        e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(ctas_per_sm, gnmr_step_kernel<DT, kStepFull, V>,
                                                          kThreads, kKeyCacheBytes);
    return e;
}

}  // namespace

cudaError_t step_occupancy(int dtype, int variant, int *ctas_per_sm)
{
    if (variant == kVariantBulk)
        return dtype == 1 ? prepare_variant<1, kVariantBulk>(ctas_per_sm)
                          : prepare_variant<0, kVariantBulk>(ctas_per_sm);
    return dtype == 1 ? prepare_variant<1, kVariantSmall>(ctas_per_sm)
                      : prepare_variant<0, kVariantSmall>(ctas_per_sm);
}

}  // namespace gnmr
