// Host side of the libgnmr C ABI (include/gnmr.h): argument and layout
// validation, the work plan, the single device allocation that holds all
// library-owned state, and the per-step launch.
#include <algorithm>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <limits>
#include <new>
#include <string>
#include <vector>

#include <cuda_runtime_api.h>

#include "gnmr.h"
#include "gnmr_internal.h"

struct gnmr_handle {
    gnmr_config cfg{};            // layout pointers cleared after create
    int32_t num_units = 0;
    int elem_bytes = 0;
    int32_t num_ctas = 0;
    int32_t finish_ctas = 0;      // grid of the controller-only launch
    int32_t variant = 0;          // streaming-loop shape (gnmr::kVariant*)
    int32_t num_warps = 0;        // warps with a first run
    int32_t num_runs = 0;
    int64_t num_segments = 0;
    int64_t num_partials = 0;
    int64_t device_bytes = 0;
    int64_t max_end = 0;
    int64_t steps = 0;
    double alpha_override = std::numeric_limits<double>::quiet_NaN();
    double beta_override = std::numeric_limits<double>::quiet_NaN();
    bool broken = false;
    std::string err;
    void *dmem = nullptr;
    gnmr::StepParams params{};    // device pointers filled at create
};

namespace {

thread_local std::string g_create_error;

std::string format(const char *fmt, ...)
{
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    std::vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    return buf;
}

gnmr_status fail_create(gnmr_status s, const std::string &why)
{
    g_create_error = why;
    return s;
}

gnmr_status fail(gnmr_handle *h, gnmr_status s, const std::string &why)
{
    h->err = why;
    return s;
}

// Makes `dev` current for the scope of a call and restores the caller's.
class DeviceScope {
public:
    explicit DeviceScope(int dev)
    {
        if (cudaGetDevice(&prev_) != cudaSuccess) {
            prev_ = -1;
            status_ = cudaErrorNoDevice;
            return;
        }
        switched_ = prev_ != dev;
        status_ = switched_ ? cudaSetDevice(dev) : cudaSuccess;
    }
    ~DeviceScope()
    {
        if (switched_)
            cudaSetDevice(prev_);
    }
    cudaError_t status() const { return status_; }

private:
    int prev_ = -1;
    bool switched_ = false;
    cudaError_t status_ = cudaSuccess;
};

bool positive_finite(double x) { return std::isfinite(x) && x > 0.0; }

// Carves sub-buffers out of one allocation, each 256-byte aligned.
struct Carver {
    size_t size = 0;
    size_t take(size_t bytes)
    {
        size_t at = size;
        size += (bytes + 255) / 256 * 256;
        return at;
    }
};

}  // namespace

extern "C" {

void gnmr_config_defaults(gnmr_config *cfg)
{
    if (!cfg)
        return;
    std::memset(cfg, 0, sizeof *cfg);
    cfg->dtype = GNMR_DTYPE_BF16;
    cfg->window = 8;
    cfg->max_o = 4;
    cfg->lock_len = 1;
    cfg->alpha_init = 1.5;
    cfg->alpha_main = 1.1;
    cfg->beta_init = 1.5;
    cfg->beta_main = 1.5;
    cfg->warmup_steps = 0;
    cfg->eps = 1e-8;
    cfg->device = 0;
    cfg->policy = GNMR_POLICY_ACTIVE_CAP;
    cfg->static_fraction = 0.25;
}

const char *gnmr_status_string(gnmr_status s)
{
    switch (s) {
    case GNMR_OK: return "GNMR_OK";
    case GNMR_ERR_INVALID_ARG: return "GNMR_ERR_INVALID_ARG: invalid argument";
    case GNMR_ERR_LAYOUT: return "GNMR_ERR_LAYOUT: unit layout does not fit the arena";
    case GNMR_ERR_CUDA: return "GNMR_ERR_CUDA: CUDA call failed";
    case GNMR_ERR_OOM: return "GNMR_ERR_OOM: out of memory";
    case GNMR_ERR_STATE: return "GNMR_ERR_STATE: handle unusable after an earlier CUDA error";
    }
    return "unknown gnmr_status";
}

const char *gnmr_last_error(const gnmr_handle *h)
{
    return h ? h->err.c_str() : g_create_error.c_str();
}

gnmr_status gnmr_plan_partition(int32_t num_units, const int64_t *lengths, int32_t dtype,
                                int32_t max_warps, int32_t *num_warps, int32_t *run_unit,
                                int64_t *run_pos, int32_t *first_warp, int32_t *num_parts)
{
    if (num_units < 1 || !lengths || (dtype != GNMR_DTYPE_F32 && dtype != GNMR_DTYPE_BF16) ||
        max_warps < 1 || !num_warps || !run_unit || !run_pos || !first_warp || !num_parts)
        return GNMR_ERR_INVALID_ARG;
    gnmr::Plan plan;
    try {
        std::vector<int32_t> ident(num_units);
        for (int32_t u = 0; u < num_units; ++u)
            ident[u] = u;
        if (!gnmr::plan_partition(num_units, lengths, ident.data(), num_units,
                                  dtype == GNMR_DTYPE_BF16 ? 2 : 4, max_warps, plan))
            return GNMR_ERR_INVALID_ARG;
    } catch (const std::bad_alloc &) {
        return GNMR_ERR_OOM;
    }
    *num_warps = plan.num_runs;
    for (int32_t w = 0; w <= plan.num_runs; ++w)
        run_unit[w] = static_cast<int32_t>(plan.run_seg[w]);
    std::memcpy(run_pos, plan.run_pos.data(), sizeof(int64_t) * (plan.num_runs + 1));
    std::memcpy(first_warp, plan.first_run.data(), sizeof(int32_t) * num_units);
    std::memcpy(num_parts, plan.num_parts.data(), sizeof(int32_t) * num_units);
    return GNMR_OK;
}

gnmr_status gnmr_create(const gnmr_config *cfg, gnmr_handle **out)
{
    if (out)
        *out = nullptr;
    if (!cfg || !out)
        return fail_create(GNMR_ERR_INVALID_ARG, "cfg and out must not be NULL");
    const gnmr_config &c = *cfg;
    if (c.num_units < 1)
        return fail_create(GNMR_ERR_INVALID_ARG, format("num_units must be >= 1 (got %d)", c.num_units));
    if (!c.offsets || !c.lengths)
        return fail_create(GNMR_ERR_INVALID_ARG, "offsets and lengths must not be NULL");
    if (c.dtype != GNMR_DTYPE_F32 && c.dtype != GNMR_DTYPE_BF16)
        return fail_create(GNMR_ERR_INVALID_ARG, format("unknown dtype %d", c.dtype));
    if (c.window < 1 || c.window > (1 << 16))
        return fail_create(GNMR_ERR_INVALID_ARG, format("window must be in [1, 65536] (got %d)", c.window));
    if (c.max_o < 0 || c.lock_len < 0 || c.warmup_steps < 0)
        return fail_create(GNMR_ERR_INVALID_ARG, "max_o, lock_len and warmup_steps must be >= 0");
    if (!positive_finite(c.alpha_init) || !positive_finite(c.alpha_main) ||
        !positive_finite(c.beta_init) || !positive_finite(c.beta_main))
        return fail_create(GNMR_ERR_INVALID_ARG, "thresholds alpha/beta must be finite and > 0");
    if (!std::isfinite(c.eps) || c.eps < 0.0)
        return fail_create(GNMR_ERR_INVALID_ARG, "eps must be finite and >= 0");
    if (c.policy < GNMR_POLICY_ACTIVE_CAP || c.policy > GNMR_POLICY_STATIC_TOP || c.forced_recovery_steps < 0 ||
        c.static_warmup_steps < 0 || !(c.static_fraction >= 0.0 && c.static_fraction <= 1.0))
        return fail_create(GNMR_ERR_INVALID_ARG,
                           "policy, forced_recovery_steps, static_warmup_steps or static_fraction out of range");
    if (c.loop_shape < GNMR_LOOP_AUTO || c.loop_shape > GNMR_LOOP_LARGE_UNITS)
        return fail_create(GNMR_ERR_INVALID_ARG, "loop_shape out of range");
    if (c.unit_cost)
        for (int32_t b = 0; b < c.num_units; ++b)
            if (!std::isfinite(c.unit_cost[b]))
                return fail_create(GNMR_ERR_INVALID_ARG, format("unit_cost[%d] is not finite", b));
    if (c.num_segments < 0 || (c.num_segments > 0 && !c.segment_unit))
        return fail_create(GNMR_ERR_INVALID_ARG, "num_segments must be >= 0, with segment_unit when > 0");
    const int eb = c.dtype == GNMR_DTYPE_BF16 ? 2 : 4;
    const int64_t limit = std::numeric_limits<int64_t>::max() / 8;
    const int64_t S_in = c.num_segments > 0 ? c.num_segments : c.num_units;
    int64_t max_end = 0;
    for (int64_t g = 0; g < S_in; ++g) {
        const int64_t o = c.offsets[g], l = c.lengths[g];
        if (o < 0 || l < 0 || o > limit - l)
            return fail_create(GNMR_ERR_INVALID_ARG,
                               format("%s %lld: offset %lld / length %lld out of range",
                                      c.num_segments > 0 ? "segment" : "unit", (long long)g,
                                      (long long)o, (long long)l));
        if (c.num_segments > 0 && (c.segment_unit[g] < 0 || c.segment_unit[g] >= c.num_units))
            return fail_create(GNMR_ERR_INVALID_ARG,
                               format("segment %lld: unit %d out of range", (long long)g, c.segment_unit[g]));
        if (l > 0 && o + l > max_end)
            max_end = o + l;
    }

    int ndev = 0;
    if (cudaGetDeviceCount(&ndev) != cudaSuccess || ndev < 1)
        return fail_create(GNMR_ERR_CUDA, "no CUDA device available");
    if (c.device < 0 || c.device >= ndev)
        return fail_create(GNMR_ERR_INVALID_ARG, format("device %d out of range (%d devices)", c.device, ndev));
    DeviceScope scope(c.device);
    if (scope.status() != cudaSuccess)
        return fail_create(GNMR_ERR_CUDA, format("cudaSetDevice(%d): %s", c.device,
                                                 cudaGetErrorString(scope.status())));
    // the streaming-loop variant follows the mean unit size
    int64_t grad_bytes = 0;
    for (int64_t g = 0; g < S_in; ++g)
        grad_bytes += c.lengths[g] * eb;
    const bool large = c.loop_shape == GNMR_LOOP_AUTO ? grad_bytes / c.num_units >= gnmr::kBulkUnitBytes
                                                      : c.loop_shape == GNMR_LOOP_LARGE_UNITS;
    const int variant = large ? gnmr::kVariantBulk : gnmr::kVariantSmall;
    int sms = 0, per_sm = 0;
    cudaError_t e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, c.device);
    if (e == cudaSuccess)
        e = gnmr::step_occupancy(c.dtype, variant, &per_sm);
    if (e != cudaSuccess || sms < 1 || per_sm < 1)
        return fail_create(GNMR_ERR_CUDA, format("device query failed: %s", cudaGetErrorString(e)));

    gnmr_handle *h = new (std::nothrow) gnmr_handle;
    if (!h)
        return fail_create(GNMR_ERR_OOM, "host allocation failed");
    const int64_t U = c.num_units;
    try {
        // Segments grouped by unit (stable: a unit keeps its segments' order);
        // a unit without segments gets one empty segment.
        std::vector<int64_t> seg_off, seg_len;
        std::vector<int32_t> seg_unit;
        if (c.num_segments > 0) {
            std::vector<int64_t> order(S_in);
            for (int64_t g = 0; g < S_in; ++g)
                order[g] = g;
            std::stable_sort(order.begin(), order.end(), [&](int64_t a, int64_t b) {
                return c.segment_unit[a] < c.segment_unit[b];
            });
            seg_off.reserve(S_in + U);
            size_t k = 0;
            for (int32_t u = 0; u < c.num_units; ++u) {
                const size_t before = seg_off.size();
                while (k < order.size() && c.segment_unit[order[k]] == u) {
                    seg_off.push_back(c.offsets[order[k]]);
                    seg_len.push_back(c.lengths[order[k]]);
                    seg_unit.push_back(u);
                    ++k;
                }
                if (seg_off.size() == before) {
                    seg_off.push_back(0);
                    seg_len.push_back(0);
                    seg_unit.push_back(u);
                }
            }
        } else {
            seg_off.assign(c.offsets, c.offsets + U);
            seg_len.assign(c.lengths, c.lengths + U);
            seg_unit.resize(U);
            for (int32_t u = 0; u < c.num_units; ++u)
                seg_unit[u] = u;
        }
        const int64_t S = static_cast<int64_t>(seg_off.size());
        // The small-unit loop plans one run per resident warp.  The large-unit
        // loop plans about kRunsPerWarp runs per warp (never fewer runs than
        // the one-per-warp plan), which the warps take dynamically.
        const int64_t grid_warps = int64_t(sms) * per_sm * gnmr::kWarpsPerCta;
        int64_t max_runs = grid_warps;
        if (variant == gnmr::kVariantBulk) {
            const int64_t cost = grad_bytes + U * gnmr::kUnitCostBytes;
            int64_t run = cost / (grid_warps * gnmr::kRunsPerWarp);
            run = std::min(std::max(run, gnmr::kBulkRunMin), gnmr::kBulkRunMax);
            max_runs = std::max(max_runs, (cost + run - 1) / run);
            if (max_runs > INT32_MAX / 2) {
                delete h;
                return fail_create(GNMR_ERR_INVALID_ARG, "work partition failed (too many runs)");
            }
        }
        gnmr::Plan plan;
        if (!gnmr::plan_partition(S, seg_len.data(), seg_unit.data(), c.num_units, eb,
                                  static_cast<int32_t>(max_runs), plan)) {
            delete h;
            return fail_create(GNMR_ERR_INVALID_ARG, "work partition failed (sizes out of range)");
        }
        const int64_t W = plan.num_runs;
        Carver cv;
        const size_t o_off = cv.take(sizeof(int64_t) * S);
        const size_t o_len = cv.take(sizeof(int64_t) * S);
        const size_t o_segu = cv.take(sizeof(int32_t) * S);
        const size_t o_rec = cv.take(U);
        const size_t o_run_seg = cv.take(sizeof(int64_t) * (W + 1));
        const size_t o_run_pos = cv.take(sizeof(int64_t) * (W + 1));
        const size_t o_first = cv.take(sizeof(int32_t) * U);
        const size_t o_parts = cv.take(sizeof(int32_t) * U);
        const size_t o_pbase = cv.take(sizeof(int64_t) * U);
        const size_t o_partial = cv.take(sizeof(double) * plan.num_partials);
        const size_t o_ticket = cv.take(sizeof(uint32_t) * U);
        const size_t o_state = cv.take(sizeof(gnmr::UnitState) * U);
        const size_t o_queue = cv.take(sizeof(double) * U * c.window);
        const size_t o_cand = cv.take(sizeof(gnmr::Candidate) * U);
        const uint32_t hot_cap = static_cast<uint32_t>(std::min<int64_t>(U, gnmr::kHotCapMax));
        const size_t o_hot = cv.take(sizeof(gnmr::Candidate) * hot_cap);
        const size_t o_hist = cv.take(sizeof(uint32_t) * gnmr::kRiskBins);
        const size_t o_ctl = cv.take(sizeof(gnmr::Control));
        const size_t o_cost = c.unit_cost ? cv.take(sizeof(double) * U) : 0;

        // Host image of the whole block: static tables plus zeroed state.
        std::vector<unsigned char> img(cv.size, 0);
        std::memcpy(&img[o_off], seg_off.data(), sizeof(int64_t) * S);
        std::memcpy(&img[o_len], seg_len.data(), sizeof(int64_t) * S);
        std::memcpy(&img[o_segu], seg_unit.data(), sizeof(int32_t) * S);
        int32_t num_rec = 0;
        for (int64_t b = 0; b < U; ++b) {
            img[o_rec + b] = c.recoverable ? (c.recoverable[b] != 0) : 1;
            num_rec += img[o_rec + b];
        }
        if (c.unit_cost)
            std::memcpy(&img[o_cost], c.unit_cost, sizeof(double) * U);
        std::memcpy(&img[o_run_seg], plan.run_seg.data(), sizeof(int64_t) * (W + 1));
        std::memcpy(&img[o_run_pos], plan.run_pos.data(), sizeof(int64_t) * (W + 1));
        std::memcpy(&img[o_first], plan.first_run.data(), sizeof(int32_t) * U);
        std::memcpy(&img[o_parts], plan.num_parts.data(), sizeof(int32_t) * U);
        std::memcpy(&img[o_pbase], plan.part_base.data(), sizeof(int64_t) * U);
        std::memset(&img[o_partial], 0xff, sizeof(double) * plan.num_partials);   // every slot empty
        static_assert(gnmr::kEmptyPartial == ~0ull, "empty partial slots are all-ones bytes");
        {
            gnmr::Control ctl{};
            ctl.hot_bin = gnmr::kNoHot;              // no prediction before the first selection
            std::memcpy(&img[o_ctl], &ctl, sizeof ctl);
        }

        e = cudaMalloc(&h->dmem, cv.size);
        if (e != cudaSuccess) {
            cudaGetLastError();
            delete h;
            return fail_create(e == cudaErrorMemoryAllocation ? GNMR_ERR_OOM : GNMR_ERR_CUDA,
                               format("cudaMalloc(%zu): %s", cv.size, cudaGetErrorString(e)));
        }
        e = cudaMemcpy(h->dmem, img.data(), cv.size, cudaMemcpyHostToDevice);
        if (e != cudaSuccess) {
            cudaFree(h->dmem);
            delete h;
            return fail_create(GNMR_ERR_CUDA, format("cudaMemcpy: %s", cudaGetErrorString(e)));
        }

        char *base = static_cast<char *>(h->dmem);
        gnmr::StepParams &p = h->params;
        p.offset = reinterpret_cast<const int64_t *>(base + o_off);
        p.length = reinterpret_cast<const int64_t *>(base + o_len);
        p.seg_unit = reinterpret_cast<const int32_t *>(base + o_segu);
        p.recoverable = reinterpret_cast<const uint8_t *>(base + o_rec);
        p.run_seg = reinterpret_cast<const int64_t *>(base + o_run_seg);
        p.run_pos = reinterpret_cast<const int64_t *>(base + o_run_pos);
        p.first_run = reinterpret_cast<const int32_t *>(base + o_first);
        p.num_parts = reinterpret_cast<const int32_t *>(base + o_parts);
        p.part_base = reinterpret_cast<const int64_t *>(base + o_pbase);
        p.partial = reinterpret_cast<double *>(base + o_partial);
        p.unit_ticket = reinterpret_cast<uint32_t *>(base + o_ticket);
        p.state = reinterpret_cast<gnmr::UnitState *>(base + o_state);
        p.queue = reinterpret_cast<double *>(base + o_queue);
        p.cand = reinterpret_cast<gnmr::Candidate *>(base + o_cand);
        p.hot = reinterpret_cast<gnmr::Candidate *>(base + o_hot);
        p.hot_cap = hot_cap;
        p.risk_hist = reinterpret_cast<uint32_t *>(base + o_hist);
        p.ctl = reinterpret_cast<gnmr::Control *>(base + o_ctl);
        p.unit_cost = c.unit_cost ? reinterpret_cast<const double *>(base + o_cost) : nullptr;
        p.policy = c.policy;
        p.num_recoverable = num_rec;
        p.forced_steps = c.forced_recovery_steps;
        p.static_warmup = c.static_warmup_steps;
        p.static_keep = static_cast<int32_t>(std::min<double>(std::ceil(c.static_fraction * num_rec), num_rec));
        p.num_units = c.num_units;
        const int32_t step_warps = static_cast<int32_t>(std::min<int64_t>(plan.num_runs, grid_warps));
        p.num_warps = step_warps;
        p.num_runs = plan.num_runs;
        p.window = c.window;
        p.max_o = c.max_o;
        p.lock_len = c.lock_len;
        p.warmup_steps = c.warmup_steps;
        p.alpha_init = c.alpha_init;
        p.alpha_main = c.alpha_main;
        p.beta_init = c.beta_init;
        p.beta_main = c.beta_main;
        p.eps = c.eps;

        h->cfg = c;
        h->cfg.offsets = nullptr;
        h->cfg.lengths = nullptr;
        h->cfg.recoverable = nullptr;
        h->cfg.segment_unit = nullptr;
        h->cfg.unit_cost = nullptr;
        h->num_segments = S;
        h->variant = variant;
        h->num_units = c.num_units;
        h->elem_bytes = eb;
        h->num_warps = step_warps;
        h->num_runs = plan.num_runs;
        h->num_ctas = (step_warps + gnmr::kWarpsPerCta - 1) / gnmr::kWarpsPerCta;
        {
            const int64_t warps = (U + 31) / 32;
            const int64_t ctas = (warps + gnmr::kWarpsPerCta - 1) / gnmr::kWarpsPerCta;
            h->finish_ctas = static_cast<int32_t>(std::min<int64_t>(ctas, int64_t(sms) * per_sm));
        }
        h->num_partials = plan.num_partials;
        h->device_bytes = static_cast<int64_t>(cv.size);
        h->max_end = max_end;
    } catch (const std::bad_alloc &) {
        if (h->dmem)
            cudaFree(h->dmem);
        delete h;
        return fail_create(GNMR_ERR_OOM, "host allocation failed while planning");
    }
    *out = h;
    return GNMR_OK;
}

gnmr_status gnmr_step(gnmr_handle *h, const void *d_arena, int64_t arena_elems, void *stream,
                      uint8_t *d_mask, const gnmr_stats *stats)
{
    if (!h)
        return GNMR_ERR_INVALID_ARG;
    if (h->broken)
        return fail(h, GNMR_ERR_STATE, "an earlier step failed in CUDA; destroy the handle");
    if (!d_mask)
        return fail(h, GNMR_ERR_INVALID_ARG, "d_mask must not be NULL");
    if (arena_elems < 0)
        return fail(h, GNMR_ERR_INVALID_ARG, "arena_elems must be >= 0");
    if (!d_arena && h->max_end > 0)
        return fail(h, GNMR_ERR_INVALID_ARG, "d_arena is NULL but units are not empty");
    if (reinterpret_cast<uintptr_t>(d_arena) % static_cast<uintptr_t>(h->elem_bytes) != 0)
        return fail(h, GNMR_ERR_INVALID_ARG, "d_arena is not aligned to the element size");
    if (arena_elems < h->max_end)
        return fail(h, GNMR_ERR_LAYOUT,
                    format("arena holds %lld elements but the layout needs %lld",
                           (long long)arena_elems, (long long)h->max_end));
    DeviceScope scope(h->cfg.device);
    if (scope.status() != cudaSuccess)
        return fail(h, GNMR_ERR_CUDA, format("cudaSetDevice: %s", cudaGetErrorString(scope.status())));

    gnmr::StepParams p = h->params;
    p.arena = d_arena;
    p.mask = d_mask;
    if (stats) {
        p.out_norm = stats->norm;
        p.out_gnmr = stats->gnmr;
        p.out_dgnmr = stats->dgnmr;
        p.out_risk = stats->risk;
        p.out_lock = stats->lock;
        p.out_counts = stats->counts;
        p.out_delta_mem = stats->delta_mem;
    }
    p.alpha_override = h->alpha_override;
    p.beta_override = h->beta_override;
    const cudaError_t e = gnmr::launch_step(p, h->cfg.dtype, h->num_ctas, static_cast<cudaStream_t>(stream),
                                            gnmr::kStepFull, h->variant);
    if (e != cudaSuccess) {
        h->broken = true;
        return fail(h, GNMR_ERR_CUDA, format("step launch: %s", cudaGetErrorString(e)));
    }
    h->steps += 1;
    return GNMR_OK;
}

gnmr_status gnmr_step_partials(gnmr_handle *h, const void *d_arena, int64_t arena_elems, void *stream,
                               double *d_sumsq)
{
    if (!h)
        return GNMR_ERR_INVALID_ARG;
    if (h->broken)
        return fail(h, GNMR_ERR_STATE, "an earlier step failed in CUDA; destroy the handle");
    if (!d_sumsq)
        return fail(h, GNMR_ERR_INVALID_ARG, "d_sumsq must not be NULL");
    if (arena_elems < 0)
        return fail(h, GNMR_ERR_INVALID_ARG, "arena_elems must be >= 0");
    if (!d_arena && h->max_end > 0)
        return fail(h, GNMR_ERR_INVALID_ARG, "d_arena is NULL but units are not empty");
    if (reinterpret_cast<uintptr_t>(d_arena) % static_cast<uintptr_t>(h->elem_bytes) != 0)
        return fail(h, GNMR_ERR_INVALID_ARG, "d_arena is not aligned to the element size");
    if (arena_elems < h->max_end)
        return fail(h, GNMR_ERR_LAYOUT,
                    format("arena holds %lld elements but the layout needs %lld",
                           (long long)arena_elems, (long long)h->max_end));
    DeviceScope scope(h->cfg.device);
    if (scope.status() != cudaSuccess)
        return fail(h, GNMR_ERR_CUDA, format("cudaSetDevice: %s", cudaGetErrorString(scope.status())));
    gnmr::StepParams p = h->params;
    p.arena = d_arena;
    p.out_sumsq = d_sumsq;
    const cudaError_t e = gnmr::launch_step(p, h->cfg.dtype, h->num_ctas, static_cast<cudaStream_t>(stream),
                                            gnmr::kStepPartials, h->variant);
    if (e != cudaSuccess) {
        h->broken = true;
        return fail(h, GNMR_ERR_CUDA, format("partials launch: %s", cudaGetErrorString(e)));
    }
    return GNMR_OK;
}

gnmr_status gnmr_finish(gnmr_handle *h, const double *d_sumsq, void *stream, uint8_t *d_mask,
                        const gnmr_stats *stats)
{
    if (!h)
        return GNMR_ERR_INVALID_ARG;
    if (h->broken)
        return fail(h, GNMR_ERR_STATE, "an earlier step failed in CUDA; destroy the handle");
    if (!d_sumsq || !d_mask)
        return fail(h, GNMR_ERR_INVALID_ARG, "d_sumsq and d_mask must not be NULL");
    DeviceScope scope(h->cfg.device);
    if (scope.status() != cudaSuccess)
        return fail(h, GNMR_ERR_CUDA, format("cudaSetDevice: %s", cudaGetErrorString(scope.status())));
    gnmr::StepParams p = h->params;
    p.in_sumsq = d_sumsq;
    p.mask = d_mask;
    if (stats) {
        p.out_norm = stats->norm;
        p.out_gnmr = stats->gnmr;
        p.out_dgnmr = stats->dgnmr;
        p.out_risk = stats->risk;
        p.out_lock = stats->lock;
        p.out_counts = stats->counts;
        p.out_delta_mem = stats->delta_mem;
    }
    p.alpha_override = h->alpha_override;
    p.beta_override = h->beta_override;
    const cudaError_t e = gnmr::launch_step(p, h->cfg.dtype, h->finish_ctas, static_cast<cudaStream_t>(stream),
                                            gnmr::kStepFinish);
    if (e != cudaSuccess) {
        h->broken = true;
        return fail(h, GNMR_ERR_CUDA, format("finish launch: %s", cudaGetErrorString(e)));
    }
    h->steps += 1;
    return GNMR_OK;
}

static int64_t state_blob_bytes(const gnmr_handle *h)
{
    return static_cast<int64_t>(sizeof(gnmr::StateHeader)) +
           static_cast<int64_t>(sizeof(gnmr::UnitState)) * h->num_units +
           static_cast<int64_t>(sizeof(double)) * h->num_units * h->cfg.window;
}

gnmr_status gnmr_get_state(gnmr_handle *h, void *stream, void *host_buf, int64_t buf_bytes,
                           int64_t *state_bytes)
{
    if (!h)
        return GNMR_ERR_INVALID_ARG;
    const int64_t need = state_blob_bytes(h);
    if (state_bytes)
        *state_bytes = need;
    if (!host_buf)
        return GNMR_OK;
    if (buf_bytes < need)
        return fail(h, GNMR_ERR_INVALID_ARG, format("state needs %lld bytes", (long long)need));
    if (h->broken)
        return fail(h, GNMR_ERR_STATE, "an earlier step failed in CUDA; destroy the handle");
    DeviceScope scope(h->cfg.device);
    if (scope.status() != cudaSuccess)
        return fail(h, GNMR_ERR_CUDA, format("cudaSetDevice: %s", cudaGetErrorString(scope.status())));
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    char *out = static_cast<char *>(host_buf);
    gnmr::Control ctl{};
    const size_t units_bytes = sizeof(gnmr::UnitState) * h->num_units;
    const size_t queue_bytes = sizeof(double) * h->num_units * h->cfg.window;
    cudaError_t e = cudaMemcpyAsync(&ctl, h->params.ctl, sizeof ctl, cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess)
        e = cudaMemcpyAsync(out + sizeof(gnmr::StateHeader), h->params.state, units_bytes,
                            cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess)
        e = cudaMemcpyAsync(out + sizeof(gnmr::StateHeader) + units_bytes, h->params.queue, queue_bytes,
                            cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess)
        e = cudaStreamSynchronize(st);
    if (e != cudaSuccess)
        return fail(h, GNMR_ERR_CUDA, format("state copy: %s", cudaGetErrorString(e)));
    gnmr::StateHeader hdr{};
    std::memcpy(hdr.magic, "GNMR", 4);
    hdr.version = 2;
    hdr.num_units = h->num_units;
    hdr.window = h->cfg.window;
    hdr.steps = ctl.steps;
    std::memcpy(out, &hdr, sizeof hdr);
    return GNMR_OK;
}

gnmr_status gnmr_set_state(gnmr_handle *h, void *stream, const void *host_buf, int64_t buf_bytes)
{
    if (!h || !host_buf)
        return h ? fail(h, GNMR_ERR_INVALID_ARG, "host_buf must not be NULL") : GNMR_ERR_INVALID_ARG;
    const int64_t need = state_blob_bytes(h);
    if (buf_bytes < need)
        return fail(h, GNMR_ERR_INVALID_ARG, format("state needs %lld bytes", (long long)need));
    gnmr::StateHeader hdr{};
    std::memcpy(&hdr, host_buf, sizeof hdr);
    if (std::memcmp(hdr.magic, "GNMR", 4) != 0 || hdr.version != 2)
        return fail(h, GNMR_ERR_INVALID_ARG, "not a GNMR state blob (magic/version)");
    if (hdr.num_units != h->num_units || hdr.window != h->cfg.window || hdr.steps < 0)
        return fail(h, GNMR_ERR_INVALID_ARG,
                    format("state is for %d units / window %d; handle has %d / %d", hdr.num_units,
                           hdr.window, h->num_units, h->cfg.window));
    const char *in = static_cast<const char *>(host_buf);
    const size_t units_bytes = sizeof(gnmr::UnitState) * h->num_units;
    const size_t queue_bytes = sizeof(double) * h->num_units * h->cfg.window;
    for (int32_t b = 0; b < h->num_units; ++b) {
        gnmr::UnitState u;
        std::memcpy(&u, in + sizeof hdr + sizeof u * b, sizeof u);
        if (u.count < 0 || u.fill < 0 || u.fill > h->cfg.window || u.head < 0 || u.head >= h->cfg.window ||
            u.lock < 0 || u.lock > h->cfg.lock_len || (u.active != 0 && u.active != 1))
            return fail(h, GNMR_ERR_INVALID_ARG, format("state of unit %d is out of range", b));
    }
    if (h->broken)
        return fail(h, GNMR_ERR_STATE, "an earlier step failed in CUDA; destroy the handle");
    DeviceScope scope(h->cfg.device);
    if (scope.status() != cudaSuccess)
        return fail(h, GNMR_ERR_CUDA, format("cudaSetDevice: %s", cudaGetErrorString(scope.status())));
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    gnmr::Control ctl{};
    ctl.steps = hdr.steps;
    ctl.hot_bin = gnmr::kNoHot;
    cudaError_t e = cudaMemcpyAsync(h->params.state, in + sizeof hdr, units_bytes, cudaMemcpyHostToDevice, st);
    if (e == cudaSuccess)
        e = cudaMemcpyAsync(h->params.queue, in + sizeof hdr + units_bytes, queue_bytes,
                            cudaMemcpyHostToDevice, st);
    if (e == cudaSuccess)
        e = cudaMemcpyAsync(h->params.ctl, &ctl, sizeof ctl, cudaMemcpyHostToDevice, st);
    if (e == cudaSuccess)
        e = cudaMemsetAsync(h->params.unit_ticket, 0, sizeof(uint32_t) * h->num_units, st);
    if (e == cudaSuccess)
        e = cudaMemsetAsync(h->params.risk_hist, 0, sizeof(uint32_t) * gnmr::kRiskBins, st);
    if (e == cudaSuccess)
        e = cudaMemsetAsync(h->params.partial, 0xff, sizeof(double) * h->num_partials, st);
    if (e == cudaSuccess)
        e = cudaStreamSynchronize(st);
    if (e != cudaSuccess) {
        h->broken = true;
        return fail(h, GNMR_ERR_CUDA, format("state copy: %s", cudaGetErrorString(e)));
    }
    h->steps = hdr.steps;
    return GNMR_OK;
}

gnmr_status gnmr_set_thresholds(gnmr_handle *h, double alpha, double beta)
{
    if (!h)
        return GNMR_ERR_INVALID_ARG;
    if ((!std::isnan(alpha) && !positive_finite(alpha)) || (!std::isnan(beta) && !positive_finite(beta)))
        return fail(h, GNMR_ERR_INVALID_ARG, "thresholds must be finite and > 0, or NaN");
    h->alpha_override = alpha;
    h->beta_override = beta;
    return GNMR_OK;
}

gnmr_status gnmr_get_info(const gnmr_handle *h, gnmr_info *info)
{
    if (!h || !info)
        return GNMR_ERR_INVALID_ARG;
    info->num_units = h->num_units;
    info->dtype = h->cfg.dtype;
    info->device = h->cfg.device;
    info->num_ctas = h->num_ctas;
    info->threads_per_cta = gnmr::kThreads;
    info->num_warps = h->num_warps;
    info->num_partials = h->num_partials;
    info->device_bytes = h->device_bytes;
    info->arena_elems_min = h->max_end;
    info->steps = h->steps;
    info->loop_shape = h->variant == gnmr::kVariantBulk ? GNMR_LOOP_LARGE_UNITS : GNMR_LOOP_SMALL_UNITS;
    info->num_runs = h->num_runs;
    return GNMR_OK;
}

gnmr_status gnmr_destroy(gnmr_handle *h)
{
    if (!h)
        return GNMR_OK;
    gnmr_status st = GNMR_OK;
    {
        DeviceScope scope(h->cfg.device);
        if (scope.status() == cudaSuccess) {
            // cudaFree waits for work in flight on the device before freeing.
            if (h->dmem && cudaFree(h->dmem) != cudaSuccess)
                st = GNMR_ERR_CUDA;
        } else {
            st = GNMR_ERR_CUDA;
        }
    }
    delete h;
    return st;
}

}  // extern "C"

namespace gnmr {

void record_thread_error(const char *why)
{
    g_create_error = why ? why : "";
}

}  // namespace gnmr
