// gnmr_unit_norms_static: per-unit gradient L2 norms with no memory
// allocation of any kind.
//
// Some callers cannot call cudaMalloc: code that runs inside a framework
// whose caching allocator already owns the device memory (a raw cudaMalloc
// there fragments the pool or fails outright once it is reserved), hooks
// called in the middle of a training step (cudaMalloc and cudaFree
// synchronise the device and would stall the step), and deployments that fix
// their memory footprint at start-up.  They cannot create a gnmr_handle, whose
// state and scratch come from one cudaMalloc, so this entry point computes the
// first stage of the monitor -- n_b = ||g_b||_2 for every unit, the values
// gnmr_step reports in stats->norm -- with every piece of scratch in one
// file-scope device array sized at compile time.
//
// The array (kScratchBytes, about 5.6 MiB) is reserved on every GPU that
// loads the library until the process exits.  Every call shares it and it
// keeps the last call's contents; the per-unit tickets that must start at
// zero are cleared by each call.  Calls whose work overlaps on the GPU (two
// streams, or two host threads) race on the array: serialise them.
#include <cmath>
#include <cstdint>
#include <cstddef>
#include <cstring>
#include <mutex>

#include <cuda_runtime.h>
#include <math_constants.h>

#include "gnmr.h"
#include "gnmr_internal.h"
#include "gnmr_stream.cuh"

namespace {

using gnmr::kFull;

constexpr int64_t kMaxUnits = int64_t(1) << 17;        // 131,072 units
constexpr int64_t kMaxWarps = int64_t(1) << 14;        // streaming warps of one call
constexpr int64_t kChunkBytes = int64_t(64) << 10;     // gradient bytes per chunk
constexpr int kThreads = 512;
constexpr int kWarpsPerCta = kThreads / 32;
constexpr int kUnroll = 8;                             // 16-byte loads in flight per lane
constexpr int kMaxDevices = 64;

constexpr size_t align256(size_t x) { return (x + 255) / 256 * 256; }
constexpr size_t kOffGeneration = 0;                   // layout generation of the tables below
constexpr size_t kOffOffsets = align256(kOffGeneration + 8);
constexpr size_t kOffLengths = align256(kOffOffsets + 8 * kMaxUnits);
constexpr size_t kOffStart = align256(kOffLengths + 8 * kMaxUnits);
constexpr size_t kOffTicket = align256(kOffStart + 8 * (kMaxUnits + 1));
constexpr size_t kOffPartBase = align256(kOffTicket + 4 * kMaxUnits);
constexpr size_t kOffWarpUnit = align256(kOffPartBase + 8 * kMaxUnits);
constexpr size_t kOffBound = align256(kOffWarpUnit + 4 * kMaxWarps);
constexpr size_t kOffPieces = align256(kOffBound + 8 * (kMaxWarps + 1));
constexpr size_t kOffPartial = align256(kOffPieces + 8 * kMaxUnits);
constexpr size_t kScratchBytes = align256(kOffPartial + 8 * (kMaxUnits + kMaxWarps));

// All scratch of gnmr_unit_norms_static: the generation number of the layout
// the tables hold, unit offsets and lengths (copied from the caller's host arrays), each unit's first chunk index, per-unit tickets,
// each unit's first partial slot, each warp's first unit and first chunk,
// each unit's first warp and piece count, and one fp64 partial per
// (warp, unit) piece.
static __device__ __align__(256) unsigned char g_norm_scratch[kScratchBytes];

struct View {
    unsigned long long *generation;
    int64_t *offset;
    int64_t *length;
    int64_t *chunk_start;   // [U + 1]
    uint32_t *ticket;
    int64_t *part_base;     // [U]
    int32_t *warp_unit;     // [W] the unit holding warp w's first chunk
    int64_t *bound;         // [W + 1] warp w streams chunks [bound[w], bound[w + 1])
    int64_t *pieces;        // [U] first warp (low 32 bits) and number of warps of unit b
    double *partial;
};

__host__ __device__ inline View carve(unsigned char *base)
{
    return View{reinterpret_cast<unsigned long long *>(base + kOffGeneration),
                reinterpret_cast<int64_t *>(base + kOffOffsets),
                reinterpret_cast<int64_t *>(base + kOffLengths),
                reinterpret_cast<int64_t *>(base + kOffStart),
                reinterpret_cast<uint32_t *>(base + kOffTicket),
                reinterpret_cast<int64_t *>(base + kOffPartBase),
                reinterpret_cast<int32_t *>(base + kOffWarpUnit),
                reinterpret_cast<int64_t *>(base + kOffBound),
                reinterpret_cast<int64_t *>(base + kOffPieces),
                reinterpret_cast<double *>(base + kOffPartial)};
}

// Chunks of unit b: ceil(length / chunk_elems), at least one (an empty unit
// still gets its norm, 0, written).  chunk_elems = 2^chunk_shift.
__host__ __device__ inline int64_t unit_chunks(int64_t len, int chunk_shift)
{
    return len > 0 ? ((len - 1) >> chunk_shift) + 1 : 1;
}

// Work split (host, at upload): the chunks (units in order, each unit's
// chunks in order) are cut into contiguous warp ranges of about equal cost, a
// chunk costing its bytes and a unit's first chunk kUnitCostBytes more (the
// per-unit work), so skewed unit sizes still balance; cut points that
// coincide are merged, so every warp range is non-empty.  The warps touching
// unit b are then w0(b) .. w0(b) + pieces(b) - 1, and the partial of warp w
// for b lives in slot part_base[b] + w - w0(b): the reduction order of every
// unit is fixed.

// Warp w streams its contiguous range of chunks with the step kernel's
// segment reduction, adding the chunks of one unit in order; a unit held by
// one warp is finished there, a unit spread over several by the warp that
// takes its last ticket, which adds the pieces in slot order.
//
// `generation` is the layout generation the call enqueued its work for.  If
// the tables in the scratch array hold another one (a call with a different
// layout replaced them before this kernel ran: calls that overlap on the
// GPU), the kernel writes NaN for every unit instead of reading them.
template <int DT>
__global__ void __launch_bounds__(kThreads, 2) static_norms_kernel(const void *arena, unsigned char *base,
                                                                   int32_t num_units, int64_t W,
                                                                   int64_t chunk_elems, double *norms,
                                                                   unsigned long long generation)
{
    constexpr int kEB = gnmr::Elem<DT>::kBytes;
    const View v = carve(base);
    const int lane = threadIdx.x & 31;
    const int64_t w = static_cast<int64_t>(blockIdx.x) * kWarpsPerCta + (threadIdx.x >> 5);
    if (__ldcg(v.generation) != generation) {
        const int64_t threads = static_cast<int64_t>(gridDim.x) * blockDim.x;
        for (int64_t u = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; u < num_units; u += threads)
            norms[u] = CUDART_NAN;
        return;
    }
    if (w >= W)
        return;
    const int64_t c0 = v.bound[w], c1 = v.bound[w + 1];
    // Unit metadata travels in batches of 32 consecutive units, loaded by the
    // warp's lanes together (one memory round trip per 32 units instead of a
    // dependent chain per unit) into the warp's slice of shared memory.
    __shared__ int64_t s_next[kWarpsPerCta][32], s_off[kWarpsPerCta][32], s_len[kWarpsPerCta][32];
    __shared__ int64_t s_pieces[kWarpsPerCta][32];
    __shared__ int64_t s_first0[kWarpsPerCta];
    const int wid = threadIdx.x >> 5;
    int32_t mb = 0;
    auto load_batch = [&](int32_t from) {                // warp-uniform
        mb = from;
        const int32_t u = from + lane;
        const bool ok = u < num_units;
        s_next[wid][lane] = ok ? v.chunk_start[u + 1] : 0;
        s_off[wid][lane] = ok ? v.offset[u] : 0;
        s_len[wid][lane] = ok ? v.length[u] : 0;
        s_pieces[wid][lane] = ok ? v.pieces[u] : 0;
        if (lane == 0)
            s_first0[wid] = v.chunk_start[from];
        __syncwarp();
    };
    int64_t first = 0, next = 0, off = 0, len = 0, wp = 0;
    auto meta = [&](int32_t u) {                         // warp-uniform
        if (u >= mb + 32) {
            __syncwarp();                                // every lane is done with the old batch
            load_batch(u);
        }
        const int j = u - mb;
        first = j ? s_next[wid][j - 1] : s_first0[wid];
        next = s_next[wid][j];
        off = s_off[wid][j];
        len = s_len[wid][j];
        wp = s_pieces[wid][j];
    };
    int32_t b = v.warp_unit[w];
    load_batch(b);
    meta(b);
    double s = 0.0;

    auto finish = [&](int32_t u, int64_t u_wp, double sum) {
        const int64_t w0 = static_cast<uint32_t>(u_wp);
        const int64_t pieces = u_wp >> 32;
        if (pieces > 1) {
            uint32_t last = 0;
            if (lane == 0) {
                __stcg(&v.partial[v.part_base[u] + (w - w0)], sum);
                last = gnmr::ticket_acq_rel(&v.ticket[u]) == static_cast<uint32_t>(pieces - 1);
            }
            last = __shfl_sync(kFull, last, 0);
            if (!last)
                return;
            __syncwarp();                                // lane 0's acquire orders the lanes' loads
            double acc = 0.0;
            for (int64_t j = lane; j < pieces; j += 32)
                acc += __ldcg(&v.partial[v.part_base[u] + j]);
            sum = gnmr::warp_allreduce_sum(acc);
            if (lane == 0)
                v.ticket[u] = 0;                         // ready for the next call
        }
        if (lane == 0)
            norms[u] = sqrt(sum);
    };

    for (int64_t c = c0; c < c1; ++c) {
        if (c >= next) {                                 // the range moves on to the next unit
            finish(b, wp, s);
            s = 0.0;
            do {
                if (b + 1 >= num_units) {                // tables not of this layout: stop
                    if (lane == 0)
                        norms[b] = CUDART_NAN;
                    return;
                }
                meta(++b);
            } while (c >= next);
        }
        const int64_t a = (c - first) * chunk_elems;
        const int64_t e = a + chunk_elems < len ? a + chunk_elems : len;
        const int64_t n = e > a ? e - a : 0;
        const char *seg = static_cast<const char *>(arena) + (off + a) * kEB;
        bool suspect;
        double x = gnmr::warp_segment_sumsq<DT, kUnroll>(seg, n, lane, suspect);
        if (suspect)
            x = gnmr::warp_segment_sumsq_f64<DT>(seg, n, lane);
        s += x;
    }
    finish(b, wp, s);
}

std::mutex g_setup_mu;
void *g_scratch_addr[kMaxDevices] = {};

// The host computes each call's chunk and slot tables into these static
// arrays (no allocation) and copies them to the device scratch; the copy
// from pageable memory is staged before cudaMemcpyAsync returns, so the
// arrays are free again once the copies are enqueued.
std::mutex g_plan_mu;
int64_t g_host_chunk_start[kMaxUnits + 1];
int64_t g_host_part_base[kMaxUnits];
int32_t g_host_warp_unit[kMaxWarps];
int64_t g_host_bound[kMaxWarps + 1];
int64_t g_host_pieces[kMaxUnits];

// The layout last uploaded to a device's scratch (one device at a time): a
// call with the same device, dtype and layout -- every step of a training
// loop -- finds the tables already there and skips the uploads, whose
// pageable host->device copies would otherwise dominate a call on many small
// units.  Compared element by element, so a match is exact.
struct Uploaded {
    int device = -1;
    unsigned long long generation = 0;   // written with the tables to the device scratch
    int sms = 0;
    int32_t dtype = -1;
    int32_t num_units = 0;
    int64_t chunks = 0;
    int64_t warps = 0;
    int64_t offsets[kMaxUnits];
    int64_t lengths[kMaxUnits];
};
Uploaded g_uploaded;
unsigned long long g_next_generation = 1;   // the device scratch starts at 0: no layout

bool same_layout(int dev, int sms, int32_t dtype, int32_t num_units, const int64_t *offsets,
                 const int64_t *lengths)
{
    const Uploaded &u = g_uploaded;
    return u.device == dev && u.sms == sms && u.dtype == dtype && u.num_units == num_units &&
           std::memcmp(u.offsets, offsets, sizeof(int64_t) * num_units) == 0 &&
           std::memcmp(u.lengths, lengths, sizeof(int64_t) * num_units) == 0;
}

// Device address of g_norm_scratch on the current device.  In host code the
// name g_norm_scratch is only a host-side stand-in, so the address is looked
// up once per device, with that device current, and cached.
cudaError_t scratch_address(void **out)
{
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess)
        return e;
    if (dev < 0 || dev >= kMaxDevices)
        return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lock(g_setup_mu);
    if (!g_scratch_addr[dev]) {
        void *p = nullptr;
        e = cudaGetSymbolAddress(&p, g_norm_scratch);
        if (e != cudaSuccess)
            return e;
        g_scratch_addr[dev] = p;
    }
    *out = g_scratch_addr[dev];
    return cudaSuccess;
}

// Failure details are short enough (<= 15 characters) to live in the
// thread's error string without a heap allocation.
constexpr char kErrDtype[] = "dtype unknown";
constexpr char kErrUnits[] = "units > 131072";
constexpr char kErrNull[] = "NULL pointer";
constexpr char kErrLayout[] = "unit off arena";
constexpr char kErrArena[] = "arena misalign";
constexpr char kErrCuda[] = "CUDA failed";
constexpr char kErrDevice[] = "device query";
static_assert(sizeof(kErrDtype) <= 16 && sizeof(kErrUnits) <= 16 && sizeof(kErrNull) <= 16 &&
                  sizeof(kErrLayout) <= 16 && sizeof(kErrArena) <= 16 &&
                  sizeof(kErrCuda) <= 16 && sizeof(kErrDevice) <= 16,
              "failure details must fit a short string");

template <size_t N>
gnmr_status reject(gnmr_status s, const char (&why)[N])
{
    gnmr::record_thread_error(why);
    return s;
}

}  // namespace

extern "C" gnmr_status gnmr_unit_norms_static(const void *d_arena, int64_t arena_elems, int32_t dtype,
                                              int32_t num_units, const int64_t *offsets,
                                              const int64_t *lengths, double *d_norms, void *stream)
{
    if (dtype != GNMR_DTYPE_F32 && dtype != GNMR_DTYPE_BF16)
        return reject(GNMR_ERR_INVALID_ARG, kErrDtype);
    if (num_units < 1 || num_units > kMaxUnits)
        return reject(GNMR_ERR_INVALID_ARG, kErrUnits);
    if (!offsets || !lengths || !d_norms || arena_elems < 0)
        return reject(GNMR_ERR_INVALID_ARG, kErrNull);
    const int eb = dtype == GNMR_DTYPE_BF16 ? 2 : 4;
    const int chunk_shift = eb == 2 ? 15 : 14;             // 64 KiB chunks
    const int64_t chunk_elems = int64_t(1) << chunk_shift;
    static_assert(kChunkBytes == (int64_t(1) << 16), "chunk_shift assumes 64 KiB chunks");
    int64_t max_end = 0;
    for (int32_t b = 0; b < num_units; ++b) {
        const int64_t o = offsets[b], l = lengths[b];
        if (o < 0 || l < 0 || o > arena_elems - l)
            return reject(GNMR_ERR_LAYOUT, kErrLayout);
        if (l > 0 && o + l > max_end)
            max_end = o + l;
    }
    if ((!d_arena && max_end > 0) || reinterpret_cast<uintptr_t>(d_arena) % eb != 0)
        return reject(GNMR_ERR_INVALID_ARG, kErrArena);

    void *addr = nullptr;
    cudaError_t e = scratch_address(&addr);
    if (e != cudaSuccess)
        return reject(GNMR_ERR_CUDA, kErrCuda);
    unsigned char *base = static_cast<unsigned char *>(addr);
    const View v = carve(base);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    int dev = 0, sms = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || sms < 1)
        return reject(GNMR_ERR_CUDA, kErrDevice);

    std::lock_guard<std::mutex> lock(g_plan_mu);
    if (!same_layout(dev, sms, dtype, num_units, offsets, lengths)) {
        g_uploaded.device = -1;                             // until the uploads are enqueued
        int64_t T = 0, total = 0;
        for (int32_t b = 0; b < num_units; ++b) {
            g_host_chunk_start[b] = T;
            T += unit_chunks(lengths[b], chunk_shift);
            total += gnmr::kUnitCostBytes + lengths[b] * eb;
        }
        g_host_chunk_start[num_units] = T;
        int64_t want = int64_t(sms) * 2 * kWarpsPerCta;    // two resident CTAs per SM
        want = want < kMaxWarps ? want : kMaxWarps;
        want = want < T ? want : T;
        // cut points: the first chunk starting at or after cost total * k / want
        int64_t nb = 0, k = 1, ucost = 0;
        g_host_bound[nb++] = 0;
        for (int32_t b = 0; b < num_units; ++b) {
            const int64_t uend = ucost + gnmr::kUnitCostBytes + lengths[b] * eb;
            const int64_t nch = unit_chunks(lengths[b], chunk_shift);
            for (; k < want; ++k) {
                const int64_t t = total / want * k + total % want * k / want;
                if (t >= uend)
                    break;
                // chunk j >= 1 of b starts at cost ucost + kUnitCostBytes + j * kChunkBytes
                const int64_t r = t - ucost - gnmr::kUnitCostBytes;
                const int64_t j = t <= ucost ? 0 : (r <= kChunkBytes ? 1 : (r + kChunkBytes - 1) / kChunkBytes);
                const int64_t c = j < nch ? g_host_chunk_start[b] + j : g_host_chunk_start[b + 1];
                if (c > g_host_bound[nb - 1])
                    g_host_bound[nb++] = c;
            }
            ucost = uend;
        }
        if (g_host_bound[nb - 1] != T)
            g_host_bound[nb++] = T;
        const int64_t W = nb - 1;
        int64_t slot = 0, wi = 0;
        for (int32_t b = 0; b < num_units; ++b) {
            const int64_t first = g_host_chunk_start[b], last = g_host_chunk_start[b + 1] - 1;
            while (g_host_bound[wi + 1] <= first)
                ++wi;
            int64_t wj = wi;
            while (g_host_bound[wj + 1] <= last)
                ++wj;
            g_host_part_base[b] = slot;
            slot += wj - wi + 1;
            g_host_pieces[b] = static_cast<int64_t>(static_cast<uint64_t>(wi) | (static_cast<uint64_t>(wj - wi + 1) << 32));
        }
        int32_t u = 0;                                      // unit of each warp's first chunk
        for (int64_t w = 0; w < W; ++w) {
            while (g_host_chunk_start[u + 1] <= g_host_bound[w])
                ++u;
            g_host_warp_unit[w] = u;
        }
        // the generation goes last: a kernel of this call sees it only with
        // every table of this layout already in place (stream order)
        static unsigned long long host_generation;
        host_generation = g_next_generation++;
        e = cudaMemcpyAsync(v.offset, offsets, sizeof(int64_t) * num_units, cudaMemcpyHostToDevice, st);
        if (e == cudaSuccess)
            e = cudaMemcpyAsync(v.length, lengths, sizeof(int64_t) * num_units, cudaMemcpyHostToDevice, st);
        if (e == cudaSuccess)
            e = cudaMemcpyAsync(v.chunk_start, g_host_chunk_start, sizeof(int64_t) * (num_units + 1),
                                cudaMemcpyHostToDevice, st);
        if (e == cudaSuccess)
            e = cudaMemcpyAsync(v.part_base, g_host_part_base, sizeof(int64_t) * num_units,
                                cudaMemcpyHostToDevice, st);
        if (e == cudaSuccess)
            e = cudaMemcpyAsync(v.warp_unit, g_host_warp_unit, sizeof(int32_t) * W, cudaMemcpyHostToDevice,
                                st);
        if (e == cudaSuccess)
            e = cudaMemcpyAsync(v.bound, g_host_bound, sizeof(int64_t) * (W + 1), cudaMemcpyHostToDevice, st);
        if (e == cudaSuccess)
            e = cudaMemcpyAsync(v.pieces, g_host_pieces, sizeof(int64_t) * num_units, cudaMemcpyHostToDevice,
                                st);
        if (e == cudaSuccess)
            e = cudaMemcpyAsync(v.generation, &host_generation, sizeof host_generation, cudaMemcpyHostToDevice,
                                st);
        if (e != cudaSuccess)
            return reject(GNMR_ERR_CUDA, kErrCuda);
        g_uploaded.generation = host_generation;
        std::memcpy(g_uploaded.offsets, offsets, sizeof(int64_t) * num_units);
        std::memcpy(g_uploaded.lengths, lengths, sizeof(int64_t) * num_units);
        g_uploaded.device = dev;
        g_uploaded.sms = sms;
        g_uploaded.dtype = dtype;
        g_uploaded.num_units = num_units;
        g_uploaded.chunks = T;
        g_uploaded.warps = W;
    }
    const int64_t W = g_uploaded.warps;
    e = cudaMemsetAsync(v.ticket, 0, sizeof(uint32_t) * num_units, st);
    if (e != cudaSuccess)
        return reject(GNMR_ERR_CUDA, kErrCuda);
    const int grid = static_cast<int>((W + kWarpsPerCta - 1) / kWarpsPerCta);
    const unsigned long long gen = g_uploaded.generation;
    if (dtype == GNMR_DTYPE_BF16)
        static_norms_kernel<1><<<grid, kThreads, 0, st>>>(d_arena, base, num_units, W, chunk_elems, d_norms, gen);
    else
        static_norms_kernel<0><<<grid, kThreads, 0, st>>>(d_arena, base, num_units, W, chunk_elems, d_norms, gen);
    e = cudaGetLastError();
    if (e != cudaSuccess)
        return reject(GNMR_ERR_CUDA, kErrCuda);
    return GNMR_OK;
}
