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
// The array (kScratchBytes, about 11.5 MiB) is reserved on every GPU that
// loads the library until the process exits.  Every call shares it and it
// keeps the last call's contents; the per-unit tickets that must start at
// zero are cleared by each call.  Calls whose work overlaps on the GPU (two
// streams, or two host threads) race on the array: serialise them.
#include <cmath>
#include <cstdint>
#include <cstddef>
#include <mutex>

#include <cuda_runtime.h>

#include "gnmr.h"
#include "gnmr_internal.h"

namespace {

constexpr int64_t kMaxUnits = int64_t(1) << 17;        // 131,072 units
constexpr int64_t kMaxChunks = int64_t(1) << 20;       // 1,048,576 chunks
constexpr int64_t kChunkBytes = int64_t(64) << 10;     // gradient bytes per chunk
constexpr int kThreads = 512;
constexpr int kMaxDevices = 64;
constexpr unsigned kFull = 0xffffffffu;

constexpr size_t align256(size_t x) { return (x + 255) / 256 * 256; }
constexpr size_t kOffOffsets = 0;
constexpr size_t kOffLengths = align256(kOffOffsets + 8 * kMaxUnits);
constexpr size_t kOffStart = align256(kOffLengths + 8 * kMaxUnits);
constexpr size_t kOffTicket = align256(kOffStart + 8 * (kMaxUnits + 1));
constexpr size_t kOffPartial = align256(kOffTicket + 4 * kMaxUnits);
constexpr size_t kScratchBytes = align256(kOffPartial + 8 * kMaxChunks);

// All scratch of gnmr_unit_norms_static: unit offsets and lengths (copied from
// the caller's host arrays), each unit's first chunk index, per-unit tickets,
// and one fp64 partial sum per chunk.
static __device__ __align__(256) unsigned char g_norm_scratch[kScratchBytes];

struct View {
    int64_t *offset;
    int64_t *length;
    int64_t *chunk_start;   // [U + 1]
    uint32_t *ticket;
    double *partial;
};

__host__ __device__ inline View carve(unsigned char *base)
{
    return View{reinterpret_cast<int64_t *>(base + kOffOffsets),
                reinterpret_cast<int64_t *>(base + kOffLengths),
                reinterpret_cast<int64_t *>(base + kOffStart),
                reinterpret_cast<uint32_t *>(base + kOffTicket),
                reinterpret_cast<double *>(base + kOffPartial)};
}

// Chunks of unit b: ceil(length / chunk_elems), at least one (an empty unit
// still gets its norm, 0, written).
__host__ __device__ inline int64_t unit_chunks(int64_t len, int64_t chunk_elems)
{
    return len > 0 ? (len + chunk_elems - 1) / chunk_elems : 1;
}

// One CTA: chunk_start = exclusive prefix of unit_chunks, tickets cleared.
__global__ void __launch_bounds__(1024) plan_chunks_kernel(unsigned char *base, int32_t num_units,
                                                           int64_t chunk_elems)
{
    __shared__ int64_t part[1024];
    const View v = carve(base);
    const int64_t per = (num_units + blockDim.x - 1) / blockDim.x;
    const int64_t lo = threadIdx.x * per;
    const int64_t hi = lo + per < num_units ? lo + per : num_units;
    int64_t local = 0;
    for (int64_t b = lo; b < hi; ++b) {
        local += unit_chunks(v.length[b], chunk_elems);
        v.ticket[b] = 0;
    }
    part[threadIdx.x] = local;
    __syncthreads();
    for (unsigned o = 1; o < blockDim.x; o <<= 1) {     // inclusive scan
        const int64_t add = threadIdx.x >= o ? part[threadIdx.x - o] : 0;
        __syncthreads();
        part[threadIdx.x] += add;
        __syncthreads();
    }
    int64_t at = part[threadIdx.x] - local;
    for (int64_t b = lo; b < hi; ++b) {
        v.chunk_start[b] = at;
        at += unit_chunks(v.length[b], chunk_elems);
    }
    if (threadIdx.x == blockDim.x - 1)
        v.chunk_start[num_units] = part[threadIdx.x];
}

template <int DT> __device__ __forceinline__ float elem(uint32_t w, int half);
template <> __device__ __forceinline__ float elem<0>(uint32_t w, int) { return __uint_as_float(w); }
template <> __device__ __forceinline__ float elem<1>(uint32_t w, int half)
{
    return __uint_as_float(half ? (w & 0xffff0000u) : (w << 16));
}

template <int DT> __device__ __forceinline__ uint32_t load_elem(const char *p)
{
    if (DT == 1)
        return static_cast<uint32_t>(__ldg(reinterpret_cast<const unsigned short *>(p))) << 16;
    return __ldg(reinterpret_cast<const unsigned int *>(p));
}

__device__ __forceinline__ double warp_sum(double x)
{
#pragma unroll
    for (int o = 16; o > 0; o >>= 1)
        x += __shfl_xor_sync(kFull, x, o);
    return x;
}

// Sum of squares of n elements at seg by one warp: 16-byte body loads (4 in
// flight per lane), fp32 per load, fp64 across loads; exact fp64 squares if the
// fp32 result may have under- or overflowed.
template <int DT> __device__ double warp_sumsq(const char *seg, int64_t n, int lane)
{
    constexpr int kEB = DT == 1 ? 2 : 4;
    constexpr int kVE = 16 / kEB;
    const uint32_t mis = static_cast<uint32_t>(reinterpret_cast<uintptr_t>(seg) & 15u);
    int64_t head = ((16u - mis) & 15u) / kEB;
    head = head < n ? head : n;
    const int64_t nvec = (n - head) / kVE;
    const int64_t tail = n - head - nvec * kVE;
    uint32_t bits = 0;
    double acc = 0.0;
    if (lane < head) {
        const uint32_t w = load_elem<DT>(seg + lane * kEB);
        const float x = __uint_as_float(w);
        bits |= w;
        acc += static_cast<double>(x * x);
    }
    if (lane < tail) {
        const uint32_t w = load_elem<DT>(seg + (head + nvec * kVE + lane) * kEB);
        const float x = __uint_as_float(w);
        bits |= w;
        acc += static_cast<double>(x * x);
    }
    const uint4 *v = reinterpret_cast<const uint4 *>(seg + head * kEB);
    for (int64_t i = lane; i < nvec; i += 4 * 32) {
        uint4 r[4];
#pragma unroll
        for (int j = 0; j < 4; ++j)
            r[j] = (i + j * 32 < nvec) ? __ldg(v + i + j * 32) : make_uint4(0u, 0u, 0u, 0u);
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const uint32_t w[4] = {r[j].x, r[j].y, r[j].z, r[j].w};
            float s = 0.f;
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                bits |= w[k];
                const float a = elem<DT>(w[k], 0);
                s = fmaf(a, a, s);
                if (DT == 1) {
                    const float b = elem<DT>(w[k], 1);
                    s = fmaf(b, b, s);
                }
            }
            acc += static_cast<double>(s);
        }
    }
    acc = warp_sum(acc);
    bits = __reduce_or_sync(kFull, bits);
    const uint32_t magnitude = DT == 1 ? 0x7fff7fffu : 0x7fffffffu;
    if ((bits & magnitude) != 0u && !(acc >= 0x1p-100 && acc <= 0x1p+100)) {
        acc = 0.0;
        for (int64_t i = lane; i < n; i += 32) {
            const double x = static_cast<double>(__uint_as_float(load_elem<DT>(seg + i * kEB)));
            acc = fma(x, x, acc);
        }
        acc = warp_sum(acc);
    }
    return acc;
}

// Warps take chunks round-robin; a unit of one chunk is finished by its warp,
// a unit of several by the warp that takes its last ticket, summing the
// chunk partials in chunk order.
template <int DT>
__global__ void __launch_bounds__(kThreads) static_norms_kernel(const void *arena, unsigned char *base,
                                                                int32_t num_units, int64_t total_chunks,
                                                                int64_t chunk_elems, double *norms)
{
    constexpr int kEB = DT == 1 ? 2 : 4;
    const View v = carve(base);
    const int lane = threadIdx.x & 31;
    const int64_t warps = static_cast<int64_t>(gridDim.x) * (kThreads / 32);
    for (int64_t c = static_cast<int64_t>(blockIdx.x) * (kThreads / 32) + (threadIdx.x >> 5);
         c < total_chunks; c += warps) {
        int32_t lo = 0, hi = num_units - 1;                  // last b with chunk_start[b] <= c
        while (lo < hi) {
            const int32_t mid = lo + (hi - lo + 1) / 2;
            if (v.chunk_start[mid] <= c)
                lo = mid;
            else
                hi = mid - 1;
        }
        const int32_t b = lo;
        const int64_t first = v.chunk_start[b];
        const int64_t nch = v.chunk_start[b + 1] - first;
        const int64_t len = v.length[b];
        const int64_t a = (c - first) * chunk_elems;
        const int64_t e = a + chunk_elems < len ? a + chunk_elems : len;
        const int64_t n = e > a ? e - a : 0;
        const char *seg = static_cast<const char *>(arena) + (v.offset[b] + a) * kEB;
        double s = warp_sumsq<DT>(seg, n, lane);
        if (nch > 1) {
            uint32_t last = 0;
            if (lane == 0) {
                __stcg(&v.partial[c], s);
                __threadfence();
                last = atomicAdd(&v.ticket[b], 1u) == static_cast<uint32_t>(nch - 1);
            }
            last = __shfl_sync(kFull, last, 0);
            if (!last)
                continue;
            __threadfence();
            double acc = 0.0;
            for (int64_t j = lane; j < nch; j += 32)
                acc += __ldcg(&v.partial[first + j]);
            s = warp_sum(acc);
            if (lane == 0)
                v.ticket[b] = 0;
        }
        if (lane == 0)
            norms[b] = sqrt(s);
    }
}

std::mutex g_setup_mu;
void *g_scratch_addr[kMaxDevices] = {};

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
constexpr char kErrChunks[] = "chunks>1048576";
constexpr char kErrArena[] = "arena misalign";
constexpr char kErrCuda[] = "CUDA failed";
static_assert(sizeof(kErrDtype) <= 16 && sizeof(kErrUnits) <= 16 && sizeof(kErrNull) <= 16 &&
                  sizeof(kErrLayout) <= 16 && sizeof(kErrChunks) <= 16 && sizeof(kErrArena) <= 16 &&
                  sizeof(kErrCuda) <= 16,
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
    const int64_t chunk_elems = kChunkBytes / eb;
    int64_t chunks = 0, max_end = 0;
    for (int32_t b = 0; b < num_units; ++b) {
        const int64_t o = offsets[b], l = lengths[b];
        if (o < 0 || l < 0 || o > arena_elems - l)
            return reject(GNMR_ERR_LAYOUT, kErrLayout);
        if (l > 0 && o + l > max_end)
            max_end = o + l;
        chunks += unit_chunks(l, chunk_elems);
    }
    if (chunks > kMaxChunks)
        return reject(GNMR_ERR_INVALID_ARG, kErrChunks);
    if ((!d_arena && max_end > 0) || reinterpret_cast<uintptr_t>(d_arena) % eb != 0)
        return reject(GNMR_ERR_INVALID_ARG, kErrArena);

    void *addr = nullptr;
    cudaError_t e = scratch_address(&addr);
    if (e != cudaSuccess)
        return reject(GNMR_ERR_CUDA, kErrCuda);
    unsigned char *base = static_cast<unsigned char *>(addr);
    const View v = carve(base);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    e = cudaMemcpyAsync(v.offset, offsets, sizeof(int64_t) * num_units, cudaMemcpyHostToDevice, st);
    if (e == cudaSuccess)
        e = cudaMemcpyAsync(v.length, lengths, sizeof(int64_t) * num_units, cudaMemcpyHostToDevice, st);
    if (e != cudaSuccess)
        return reject(GNMR_ERR_CUDA, kErrCuda);
    plan_chunks_kernel<<<1, 1024, 0, st>>>(base, num_units, chunk_elems);
    int dev = 0, sms = 1;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    const int64_t warps_wanted = chunks < int64_t(sms) * 2 * (kThreads / 32) ? chunks
                                                                             : int64_t(sms) * 2 * (kThreads / 32);
    const int grid = static_cast<int>((warps_wanted + kThreads / 32 - 1) / (kThreads / 32));
    if (dtype == GNMR_DTYPE_BF16)
        static_norms_kernel<1><<<grid, kThreads, 0, st>>>(d_arena, base, num_units, chunks, chunk_elems, d_norms);
    else
        static_norms_kernel<0><<<grid, kThreads, 0, st>>>(d_arena, base, num_units, chunks, chunk_elems, d_norms);
    e = cudaGetLastError();
    if (e != cudaSuccess)
        return reject(GNMR_ERR_CUDA, kErrCuda);
    return GNMR_OK;
}
