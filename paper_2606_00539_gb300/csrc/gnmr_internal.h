// Internal declarations shared by the host API (gnmr_api.cpp, gnmr_plan.cpp)
// and the device code (gnmr_kernels.cu).  Not part of the public ABI.
#pragma once

#include <cstddef>
#include <cstdint>
#include <vector>

#include <cuda_runtime_api.h>

namespace gnmr {

// Launch shape of the step kernel: 512 threads = 16 warps per CTA.  Two
// compiled variants of the streaming loop (gnmr_kernels.cu): kVariantSmall
// (two resident CTAs per SM, one planned run per warp) for layouts of many
// small units, kVariantBulk (one CTA per SM, deeper per-warp streams, runs
// taken from a shared counter) for layouts whose mean unit holds at least
// kBulkUnitBytes.
constexpr int kThreads = 512;
constexpr int kWarpsPerCta = kThreads / 32;
constexpr int kVariantSmall = 0;
constexpr int kVariantBulk = 1;
constexpr int64_t kBulkUnitBytes = int64_t(1) << 20;

// Work partition: a unit costs its element bytes plus this many bytes of
// equivalent fixed work (reduction, Algorithm 1 update, bookkeeping); runs
// are cut at multiples of kSplitBytes inside a unit, and no run is planned
// smaller than kMinRunBytes unless the whole problem is.
constexpr int64_t kUnitCostBytes = 4096;
constexpr int64_t kSplitBytes = 512;
constexpr int64_t kMinRunBytes = 4096;   // one 4 KiB load round per warp: small problems spread over more SMs
// Large-unit loop: the stream is cut into about kRunsPerWarp runs per warp of
// kBulkRunMin..kBulkRunMax bytes each.  Each warp starts on its own run and
// then takes the next untaken one, so warps that stream faster take more runs
// and all finish together (static equal runs left the slowest warps ~8 % of
// the step behind the median one).
constexpr int64_t kRunsPerWarp = 16;
constexpr int64_t kBulkRunMin = int64_t(64) << 10;
constexpr int64_t kBulkRunMax = int64_t(256) << 10;

// Persistent per-unit controller state (Algorithm 1 and 2), 40 bytes.
struct UnitState {
    double mean;      // A_b, historical mean of n_b
    int64_t count;    // k_b, steps at which b was observed
    int32_t fill;     // |Q_b|, valid entries of the GNMR queue (<= window)
    int32_t head;     // ring position of the oldest queue entry once full
    int32_t lock;     // Lock_b
    int32_t active;   // 1 if b was on the recovery path at the previous step
    double gsum;      // GNMR summed over the static policy's warm-up
};
// lock and active are written together as one 8-byte store
static_assert(offsetof(UnitState, lock) % 8 == 0 && offsetof(UnitState, active) == offsetof(UnitState, lock) + 4,
              "UnitState lock/active pair");

// Bit pattern of an empty partial slot (a NaN that no partial sum takes:
// partials are non-negative, +inf or the canonical NaN).  The first slot of
// every unit split in two holds it between steps.
constexpr unsigned long long kEmptyPartial = ~0ull;

// Candidate-pool entry written by the unit epilogue, read by the selection
// (one 16-byte load).
struct Candidate {
    double risk;      // R_{b,t} (the static policy ranks by the GNMR sum)
    int32_t unit;
    uint32_t lock;    // Lock_b before this step, bit 31: active at the previous step
};
constexpr uint32_t kCandActive = 0x80000000u;

// Risk histogram of the candidate pool, built by the unit epilogues with one
// atomic per pool member and read (and cleared) by the selecting CTA.  Bin 0
// holds R < 1 (lock-only candidates); bin i >= 1 holds the R >= 1 whose
// exponent and top three mantissa bits are the (i-1)-th such pattern above
// 1.0: eight bins per octave, [1, 1.125), [1.125, 1.25), ..., [1.875, 2),
// [2, 2.25), ...; the last bin also holds everything larger (+inf included).
constexpr int kRiskBins = 2048;
// Hot list: the candidates a step appends because their bin is at or above a
// bin predicted from the previous step's cut (plus, under the admission cap,
// every retained unit).  When the prediction holds, the selecting CTA reads
// this short list instead of the whole candidate list.
constexpr uint32_t kHotCapMax = 8192;
constexpr uint32_t kNoHot = kRiskBins;   // hot_bin: no prediction, no pool member is hot

// Device-resident step control block.
struct Control {
    uint32_t ctas_done;   // CTA completion ticket of the current launch
    uint32_t n_cand;      // |C_t| appended so far
    int64_t steps;        // completed steps (t of the last step)
    uint32_t n_hot;       // hot-list entries appended so far (may exceed the capacity)
    uint32_t hot_bin;     // lowest bin whose pool members go to the hot list this step
    uint32_t pad[26];     // the run counters below on a 128-byte line of their own
    uint32_t next_run;    // runs taken beyond the warps' first ones (large-unit loop)
    uint32_t warps_done;  // partial-sums half: warps that have taken their last run
                          // (both zero between launches)
};
static_assert(offsetof(Control, next_run) == 128, "run counters on their own line");

// Checkpoint blob: this header, then UnitState[num_units], then the GNMR ring
// buffers double[num_units * window] (little-endian, as on the device).
struct StateHeader {
    char magic[4];        // "GNMR"
    uint32_t version;     // 2
    int32_t num_units;
    int32_t window;
    int64_t steps;
    int64_t reserved;
};

struct StepParams {
    const void *arena;
    const int64_t *offset;       // [S] segment offsets, segments grouped by unit
    const int64_t *length;       // [S] segment lengths
    const int32_t *seg_unit;     // [S] unit of each segment (non-decreasing)
    const uint8_t *recoverable;  // [U]
    const int64_t *run_seg;      // [R + 1] first segment of each run
    const int64_t *run_pos;      // [R + 1]
    const int32_t *first_run;    // [U] first run touching unit b
    const int32_t *num_parts;    // [U]
    const int64_t *part_base;    // [U] first partial slot of unit b
    double *partial;             // [num_partials]
    uint32_t *unit_ticket;       // [U]
    UnitState *state;            // [U]
    double *queue;               // [U * window] GNMR ring buffers
    Candidate *cand;             // [U]
    Candidate *hot;              // [hot_cap] the hot list
    uint32_t *risk_hist;         // [kRiskBins], zero between steps
    Control *ctl;
    uint8_t *mask;               // [U], caller
    double *out_norm, *out_gnmr, *out_dgnmr, *out_risk;  // caller, optional
    int32_t *out_lock, *out_counts;                       // caller, optional
    double *out_sumsq;                                    // kStepPartials output [U]
    const double *in_sumsq;                               // kStepFinish input [U]
    double *out_delta_mem;                                // caller, optional [1]
    const double *unit_cost;                              // [U] or null
    int32_t policy;
    int32_t num_recoverable;
    int64_t forced_steps;
    int64_t static_warmup;
    int32_t static_keep;                                  // ceil(static_fraction * |B_rec|)
    uint32_t hot_cap;                                     // min(U, kHotCapMax)
    int32_t num_units;
    int32_t num_warps;           // warps with a first run: runs 0 .. num_warps - 1
    int32_t window;
    int32_t max_o;
    int32_t lock_len;
    int32_t num_runs;            // R; runs num_warps .. R - 1 are taken dynamically
    int64_t warmup_steps;
    double alpha_init, alpha_main, beta_init, beta_main, eps;
    double alpha_override, beta_override;  // NaN = two-stage schedule
};

// Step kernel modes: the full step, its gradient half (per-unit sums of
// squares only) and its controller half (Algorithms 1-2 on given sums).
constexpr int kStepFull = 0;
constexpr int kStepPartials = 1;
constexpr int kStepFinish = 2;

// Enqueues one launch of the step kernel in `mode`; returns the launch status.
cudaError_t launch_step(const StepParams &p, int dtype, int num_ctas, cudaStream_t stream,
                        int mode = kStepFull, int variant = kVariantSmall);

// Resident CTAs per SM of the step kernel for `dtype` and `variant`.
cudaError_t step_occupancy(int dtype, int variant, int *ctas_per_sm);

// Records the failure detail that gnmr_last_error(NULL) reports on the
// calling thread (used by calls that have no handle).
void record_thread_error(const char *why);

// Host-side work partition (gnmr_plan.cpp).
struct Plan {
    int32_t num_runs = 0;
    std::vector<int64_t> run_seg;     // [num_runs + 1]
    std::vector<int64_t> run_pos;     // [num_runs + 1]
    std::vector<int32_t> first_run;   // [U]
    std::vector<int32_t> num_parts;   // [U]
    std::vector<int64_t> part_base;   // [U]
    int64_t num_partials = 0;
};

// Segments must be grouped by unit (seg_unit non-decreasing, every unit
// 0..num_units-1 present).  Cuts the stream into at most max_runs runs, none
// smaller than kMinRunBytes unless the whole problem is.  Returns false if
// the inputs are out of range.
bool plan_partition(int64_t num_segments, const int64_t *seg_lengths, const int32_t *seg_unit,
                    int32_t num_units, int elem_bytes, int32_t max_runs, Plan &out);

}  // namespace gnmr
