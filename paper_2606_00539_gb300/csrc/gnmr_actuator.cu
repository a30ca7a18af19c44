// Recovery actuator: per-token fake quantization of every unit's saved
// activations, in the low-cost or the recovery format as the unit's mask bit
// says (App. E.2; the activation-quantization stress bench of Sec. 5.1).  For
// each token row: amax = max |x|; inv = fmax / amax; scale = amax / fmax;
// y = round_to_format(x * inv) * scale, rounding to the nearest representable
// value with ties to the even code and saturating at fmax.  All arithmetic is
// fp32, so the quantized codes are the same on any IEEE machine.  Rows whose
// max is 0, that hold a NaN or Inf, or whose scale factor fmax / amax
// overflows fp32 (amax below fmax / FLT_MAX) are copied unchanged.
//
// The rounding is the hardware minifloat conversion (cvt.rn.satfinite to
// e2m1x2 / e3m2x2 / e4m3x2 / e5m2x2, then back to f16x2, where every value of
// these formats is exact): round to nearest even, saturating -- the format
// definition itself, two values per instruction.
//
// One warp per token row: pass 1 reads the row for amax (integer max over the
// magnitude bits), pass 2 reads it again from L2 and writes the result, so
// HBM sees one read and one write per element.  The grid holds 16 warps per
// SM, whose rows (about 30 MB in all) stay resident in the 129 MB L2 between
// the two passes: pass 1 loads them with an L2 evict-last policy, pass 2
// reads and the output stores use evict-first, so the write stream does not
// push the waiting rows out.  (32 warps per SM left a fifth of the pass-2
// reads missing L2; 8 cannot keep enough loads in flight.)  No shared memory,
// no block barrier, no waits.
#include <algorithm>
#include <cmath>
#include <cstdint>
#include <cstring>
#include <new>
#include <string>
#include <vector>

#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include "gnmr.h"
#include "gnmr_internal.h"

struct gnmr_actuator {
    int32_t num_units = 0;
    int32_t dtype = 0;
    int32_t device = 0;
    int32_t grid = 0;
    int64_t total_rows = 0;
    int64_t max_end = 0;
    void *dmem = nullptr;
    const int64_t *offset = nullptr;      // [U]
    const int64_t *cols = nullptr;        // [U]
    const int64_t *row_start = nullptr;   // [U + 1]
};

namespace {

constexpr unsigned kFull = 0xffffffffu;
constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr int kMinCtas = 2;             // 16 resident warps per SM: their rows stay in L2
constexpr int kPass1Loads = 16;         // 16-byte loads in flight per lane in pass 1 (from HBM)
constexpr int kPass2Loads = 8;          // in pass 2 (from L2)

struct FqFmt {
    float fmax;
    int code;      // gnmr_fq_format; 0 = copy
};

bool fmt_of(int code, FqFmt &f)
{
    switch (code) {
    case GNMR_FQ_NONE: f = {1.0f, 0}; return true;
    case GNMR_FQ_E2M1: f = {6.0f, 1}; return true;
    case GNMR_FQ_E3M2: f = {28.0f, 2}; return true;
    case GNMR_FQ_E4M3: f = {448.0f, 3}; return true;
    case GNMR_FQ_E5M2: f = {57344.0f, 4}; return true;
    default: return false;
    }
}

// Rounds (a0, a1) to format CODE and returns them as fp32 (exact).
template <int CODE>
__device__ __forceinline__ float2 fq_round2(float a0, float a1)
{
    uint32_t h2;
    if (CODE == 1)
        asm("{ .reg .b8 t; cvt.rn.satfinite.e2m1x2.f32 t, %2, %1; cvt.rn.f16x2.e2m1x2 %0, t; }"
            : "=r"(h2) : "f"(a0), "f"(a1));
    else if (CODE == 2)
        asm("{ .reg .b16 t; cvt.rn.satfinite.e3m2x2.f32 t, %2, %1; cvt.rn.f16x2.e3m2x2 %0, t; }"
            : "=r"(h2) : "f"(a0), "f"(a1));
    else if (CODE == 3)
        asm("{ .reg .b16 t; cvt.rn.satfinite.e4m3x2.f32 t, %2, %1; cvt.rn.f16x2.e4m3x2 %0, t; }"
            : "=r"(h2) : "f"(a0), "f"(a1));
    else
        asm("{ .reg .b16 t; cvt.rn.satfinite.e5m2x2.f32 t, %2, %1; cvt.rn.f16x2.e5m2x2 %0, t; }"
            : "=r"(h2) : "f"(a0), "f"(a1));
    __half2 h;
    memcpy(&h, &h2, sizeof h);
    return make_float2(__low2float(h), __high2float(h));
}

template <int DT> struct Act;
template <> struct Act<0> {                     // fp32: 4 per vector
    static constexpr int kBytes = 4;
    static constexpr int kN = 4;
    __device__ static float load(const void *p, int64_t i) { return __ldg(static_cast<const float *>(p) + i); }
    __device__ static void store(void *p, int64_t i, float y) { static_cast<float *>(p)[i] = y; }
    __device__ static void copy(const void *s, void *d, int64_t i)
    {
        static_cast<unsigned int *>(d)[i] = __ldg(static_cast<const unsigned int *>(s) + i);
    }
    __device__ static void unpack(const uint4 v, float *x)
    {
        x[0] = __uint_as_float(v.x); x[1] = __uint_as_float(v.y);
        x[2] = __uint_as_float(v.z); x[3] = __uint_as_float(v.w);
    }
    __device__ static uint4 pack(const float *y)
    {
        return make_uint4(__float_as_uint(y[0]), __float_as_uint(y[1]), __float_as_uint(y[2]), __float_as_uint(y[3]));
    }
};
template <> struct Act<1> {                     // bf16: 8 per vector
    static constexpr int kBytes = 2;
    static constexpr int kN = 8;
    __device__ static float load(const void *p, int64_t i)
    {
        return __uint_as_float(static_cast<uint32_t>(__ldg(static_cast<const unsigned short *>(p) + i)) << 16);
    }
    __device__ static void store(void *p, int64_t i, float y)
    {
        static_cast<unsigned short *>(p)[i] = __bfloat16_as_ushort(__float2bfloat16_rn(y));
    }
    __device__ static void copy(const void *s, void *d, int64_t i)
    {
        static_cast<unsigned short *>(d)[i] = __ldg(static_cast<const unsigned short *>(s) + i);
    }
    __device__ static void unpack(const uint4 v, float *x)
    {
        const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            x[2 * i] = __uint_as_float(w[i] << 16);
            x[2 * i + 1] = __uint_as_float(w[i] & 0xffff0000u);
        }
    }
    __device__ static uint4 pack(const float *y)
    {
        uint32_t w[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const __nv_bfloat162 p = __floats2bfloat162_rn(y[2 * i], y[2 * i + 1]);
            memcpy(&w[i], &p, sizeof w[i]);
        }
        return make_uint4(w[0], w[1], w[2], w[3]);
    }
};

template <int DT, int CODE>
__device__ __forceinline__ uint4 quantize_vec(const uint4 v, float inv, float scale)
{
    float x[Act<DT>::kN], y[Act<DT>::kN];
    Act<DT>::unpack(v, x);
#pragma unroll
    for (int k = 0; k < Act<DT>::kN; k += 2) {
        const float2 q = fq_round2<CODE>(x[k] * inv, x[k + 1] * inv);
        y[k] = q.x * scale;
        y[k + 1] = q.y * scale;
    }
    return Act<DT>::pack(y);
}

// Largest magnitude of a 16-byte vector as an fp32 bit pattern without its
// sign: for non-negative floats the bit patterns order like the values, and
// Inf (0x7f800000) and NaN (above it) order above every finite value.
template <int DT> __device__ __forceinline__ uint32_t vec_max_bits(const uint4 v);
template <> __device__ __forceinline__ uint32_t vec_max_bits<0>(const uint4 v)
{
    return max(max(v.x & 0x7fffffffu, v.y & 0x7fffffffu), max(v.z & 0x7fffffffu, v.w & 0x7fffffffu));
}
template <> __device__ __forceinline__ uint32_t vec_max_bits<1>(const uint4 v)
{
    // two bf16 per word: per-halfword unsigned max of the magnitudes
    const uint32_t m = __vmaxu2(__vmaxu2(v.x & 0x7fff7fffu, v.y & 0x7fff7fffu),
                                __vmaxu2(v.z & 0x7fff7fffu, v.w & 0x7fff7fffu));
    return max(m << 16, m & 0xffff0000u);
}
template <int DT> __device__ __forceinline__ uint32_t elem_max_bits(const char *p, int64_t i)
{
    return __float_as_uint(Act<DT>::load(p, i)) & 0x7fffffffu;
}

// Where a row lives and how it splits into head / 16-byte body / tail (the
// body is vectorised only when input and output share 16-byte alignment).
struct RowRef {
    const char *src;
    char *dst;
    int64_t n, head, nvec, tail_at;
    FqFmt f;
};

// The unit holding row r: the cached unit when r is still inside it (the
// common case, rows advance by the number of warps), else a binary search.
struct UnitHint {
    int32_t unit = -1;
    int64_t begin = 0, end = 0;
};

__device__ __forceinline__ int32_t unit_of_row(int64_t r, const int64_t *row_start, int32_t num_units, UnitHint &h)
{
    if (r >= h.begin && r < h.end)
        return h.unit;
    int32_t lo = 0, hi = num_units - 1;          // last unit with row_start <= r
    while (lo < hi) {
        const int32_t mid = lo + (hi - lo + 1) / 2;
        if (row_start[mid] <= r)
            lo = mid;
        else
            hi = mid - 1;
    }
    h.unit = lo;
    h.begin = row_start[lo];
    h.end = row_start[lo + 1];
    return lo;
}

template <int DT>
__device__ __forceinline__ RowRef locate_row(int64_t r, const void *in, void *out, const int64_t *offset,
                                             const int64_t *cols, const int64_t *row_start, int32_t num_units,
                                             const uint8_t *mask, const FqFmt &low, const FqFmt &rec,
                                             UnitHint &hint)
{
    constexpr int kEB = Act<DT>::kBytes;
    const int32_t b = unit_of_row(r, row_start, num_units, hint);
    RowRef q;
    q.f = (mask != nullptr && mask[b]) ? rec : low;
    q.n = cols[b];
    const int64_t e0 = offset[b] + (r - row_start[b]) * q.n;
    q.src = static_cast<const char *>(in) + e0 * kEB;
    q.dst = static_cast<char *>(out) + e0 * kEB;
    const uint32_t mis = static_cast<uint32_t>(reinterpret_cast<uintptr_t>(q.src) & 15u);
    const bool aligned = mis == static_cast<uint32_t>(reinterpret_cast<uintptr_t>(q.dst) & 15u);
    q.head = aligned ? static_cast<int64_t>(((16u - mis) & 15u) / kEB) : q.n;
    q.head = q.head < q.n ? q.head : q.n;
    q.nvec = (q.n - q.head) / Act<DT>::kN;
    q.tail_at = q.head + q.nvec * Act<DT>::kN;
    return q;
}

// L2 eviction policies for a whole access (createpolicy), and 16-byte
// accesses that carry one.
__device__ __forceinline__ uint64_t policy_evict_last()
{
    uint64_t p;
    asm("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
    return p;
}
__device__ __forceinline__ uint64_t policy_evict_first()
{
    uint64_t p;
    asm("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
    return p;
}
__device__ __forceinline__ uint4 ld_policy(const uint4 *q, uint64_t pol)
{
    uint4 r;
    asm volatile("ld.global.L2::cache_hint.v4.u32 {%0, %1, %2, %3}, [%4], %5;"
                 : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w) : "l"(q), "l"(pol));
    return r;
}
__device__ __forceinline__ void st_policy(uint4 *q, uint4 v, uint64_t pol)
{
    asm volatile("st.global.L2::cache_hint.v4.u32 [%0], {%1, %2, %3, %4}, %5;"
                 ::"l"(q), "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w), "l"(pol) : "memory");
}

// Pass 1's load keeps the line in L2 for pass 2; pass 2's load is its last
// use, and the output is written once.
__device__ __forceinline__ uint4 ld_keep(const uint4 *p) { return ld_policy(p, policy_evict_last()); }
__device__ __forceinline__ uint4 ld_last(const uint4 *p) { return ld_policy(p, policy_evict_first()); }
__device__ __forceinline__ void st_once(uint4 *p, uint4 v) { st_policy(p, v, policy_evict_first()); }

// Pass 2 of one row in format CODE (one warp): quantize and write.
template <int DT, int CODE>
__device__ __forceinline__ void quantize_row_warp(const char *src, char *dst, const uint4 *vs, uint4 *vd,
                                                  int64_t head, int64_t nvec, int64_t tail_at, int64_t n,
                                                  float inv, float scale, int lane)
{
    for (int64_t i = lane; i < head; i += 32)
        Act<DT>::store(dst, i, fq_round2<CODE>(Act<DT>::load(src, i) * inv, 0.f).x * scale);
    int64_t i = lane;
    for (; i + (kPass2Loads - 1) * 32 < nvec; i += kPass2Loads * 32) {
        uint4 v[kPass2Loads];
#pragma unroll
        for (int j = 0; j < kPass2Loads; ++j)
            v[j] = ld_last(vs + i + j * 32);
#pragma unroll
        for (int j = 0; j < kPass2Loads; ++j)
            st_once(vd + i + j * 32, quantize_vec<DT, CODE>(v[j], inv, scale));
    }
    for (; i < nvec; i += 32)
        st_once(vd + i, quantize_vec<DT, CODE>(ld_last(vs + i), inv, scale));
    for (int64_t t = tail_at + lane; t < n; t += 32)
        Act<DT>::store(dst, t, fq_round2<CODE>(Act<DT>::load(src, t) * inv, 0.f).x * scale);
}

// One warp per token row, rows assigned round-robin.  Pass 1 reads the row
// (16 16-byte loads in flight per lane) for amax; pass 2 reads it again -- from
// L2, the resident warps' rows fit there -- and writes the result once.  No
// shared memory and no block barrier.
template <int DT>
__global__ void __launch_bounds__(kThreads, kMinCtas) fake_quant_kernel(
    const void *in, void *out, const int64_t *offset, const int64_t *cols, const int64_t *row_start,
    int32_t num_units, int64_t total_rows, const uint8_t *mask, FqFmt low, FqFmt rec)
{
    constexpr int kEB = Act<DT>::kBytes;
    const int lane = threadIdx.x & 31;
    const int64_t warps = static_cast<int64_t>(gridDim.x) * kWarps;
    UnitHint hint;
    for (int64_t r = static_cast<int64_t>(blockIdx.x) * kWarps + (threadIdx.x >> 5); r < total_rows;
         r += warps) {
        const RowRef q = locate_row<DT>(r, in, out, offset, cols, row_start, num_units, mask, low, rec, hint);
        const uint4 *vs = reinterpret_cast<const uint4 *>(q.src + q.head * kEB);
        uint4 *vd = reinterpret_cast<uint4 *>(q.dst + q.head * kEB);
        uint32_t mbits = 0;
        for (int64_t i = lane; i < q.head; i += 32)
            mbits = max(mbits, elem_max_bits<DT>(q.src, i));
        int64_t i = lane;
        for (; i + (kPass1Loads - 1) * 32 < q.nvec; i += kPass1Loads * 32) {
            uint4 v[kPass1Loads];
#pragma unroll
            for (int j = 0; j < kPass1Loads; ++j)
                v[j] = ld_keep(vs + i + j * 32);
#pragma unroll
            for (int j = 0; j < kPass1Loads; ++j)
                mbits = max(mbits, vec_max_bits<DT>(v[j]));
        }
        for (; i < q.nvec; i += 32)
            mbits = max(mbits, vec_max_bits<DT>(ld_keep(vs + i)));
        for (int64_t t = q.tail_at + lane; t < q.n; t += 32)
            mbits = max(mbits, elem_max_bits<DT>(q.src, t));
#pragma unroll
        for (int o = 16; o > 0; o >>= 1)
            mbits = max(mbits, __shfl_xor_sync(kFull, mbits, o));

        // kept (bit-for-bit copy): no format, a zero row, a non-finite value,
        // or a row so small that its scale factor fmax / amax overflows fp32
        if (q.f.code == 0 || mbits == 0u || mbits >= 0x7f800000u || isinf(q.f.fmax / __uint_as_float(mbits))) {
            if (q.src != q.dst) {
                for (int64_t t = lane; t < q.head; t += 32)
                    Act<DT>::copy(q.src, q.dst, t);
                for (int64_t t = lane; t < q.nvec; t += 32)
                    st_once(vd + t, ld_last(vs + t));
                for (int64_t t = q.tail_at + lane; t < q.n; t += 32)
                    Act<DT>::copy(q.src, q.dst, t);
            }
            continue;
        }
        const float amax = __uint_as_float(mbits);
        const float inv = q.f.fmax / amax;
        const float scale = amax / q.f.fmax;
        switch (q.f.code) {                       // one dispatch per row
        case 1: quantize_row_warp<DT, 1>(q.src, q.dst, vs, vd, q.head, q.nvec, q.tail_at, q.n, inv, scale, lane); break;
        case 2: quantize_row_warp<DT, 2>(q.src, q.dst, vs, vd, q.head, q.nvec, q.tail_at, q.n, inv, scale, lane); break;
        case 3: quantize_row_warp<DT, 3>(q.src, q.dst, vs, vd, q.head, q.nvec, q.tail_at, q.n, inv, scale, lane); break;
        default: quantize_row_warp<DT, 4>(q.src, q.dst, vs, vd, q.head, q.nvec, q.tail_at, q.n, inv, scale, lane); break;
        }
    }
}

gnmr_status act_fail(gnmr_status s, const std::string &why)
{
    gnmr::record_thread_error(why.c_str());
    return s;
}

}  // namespace

extern "C" {

gnmr_status gnmr_actuator_create(int32_t num_units, const int64_t *offsets, const int64_t *rows,
                                 const int64_t *cols, int32_t dtype, int32_t device, gnmr_actuator **out)
{
    if (out)
        *out = nullptr;
    if (!out || !offsets || !rows || !cols || num_units < 1)
        return act_fail(GNMR_ERR_INVALID_ARG, "actuator: NULL argument or num_units < 1");
    if (dtype != GNMR_DTYPE_F32 && dtype != GNMR_DTYPE_BF16)
        return act_fail(GNMR_ERR_INVALID_ARG, "actuator: unknown dtype");
    std::vector<int64_t> start(num_units + 1, 0);
    int64_t max_end = 0;
    const int64_t limit = INT64_MAX / 8;
    for (int32_t b = 0; b < num_units; ++b) {
        if (offsets[b] < 0 || rows[b] < 0 || cols[b] < 0 || (cols[b] > 0 && rows[b] > limit / cols[b]) ||
            offsets[b] > limit - rows[b] * cols[b] || start[b] > limit - rows[b])
            return act_fail(GNMR_ERR_INVALID_ARG, "actuator: unit " + std::to_string(b) + " out of range");
        start[b + 1] = start[b] + rows[b];
        max_end = std::max(max_end, offsets[b] + rows[b] * cols[b]);
    }
    int ndev = 0;
    if (cudaGetDeviceCount(&ndev) != cudaSuccess || device < 0 || device >= ndev)
        return act_fail(GNMR_ERR_CUDA, "actuator: device not available");
    int prev = 0;
    cudaGetDevice(&prev);
    cudaSetDevice(device);
    int sms = 1;
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, device);
    gnmr_actuator *a = new (std::nothrow) gnmr_actuator;
    if (!a) {
        cudaSetDevice(prev);
        return act_fail(GNMR_ERR_OOM, "actuator: host allocation failed");
    }
    const size_t U = static_cast<size_t>(num_units);
    std::vector<int64_t> img(2 * U + U + 1);
    std::memcpy(img.data(), offsets, 8 * U);
    std::memcpy(img.data() + U, cols, 8 * U);
    std::memcpy(img.data() + 2 * U, start.data(), 8 * (U + 1));
    cudaError_t e = cudaMalloc(&a->dmem, 8 * img.size());
    if (e == cudaSuccess)
        e = cudaMemcpy(a->dmem, img.data(), 8 * img.size(), cudaMemcpyHostToDevice);
    cudaSetDevice(prev);
    if (e != cudaSuccess) {
        if (a->dmem)
            cudaFree(a->dmem);
        delete a;
        return act_fail(e == cudaErrorMemoryAllocation ? GNMR_ERR_OOM : GNMR_ERR_CUDA,
                        std::string("actuator: ") + cudaGetErrorString(e));
    }
    const int64_t *base = static_cast<const int64_t *>(a->dmem);
    a->offset = base;
    a->cols = base + U;
    a->row_start = base + 2 * U;
    a->num_units = num_units;
    a->dtype = dtype;
    a->device = device;
    a->total_rows = start[U];
    a->max_end = max_end;
    const int64_t warps = std::min<int64_t>(std::max<int64_t>(a->total_rows, 1), int64_t(sms) * kMinCtas * kWarps);
    a->grid = static_cast<int32_t>((warps + kWarps - 1) / kWarps);
    *out = a;
    return GNMR_OK;
}

gnmr_status gnmr_actuator_apply(gnmr_actuator *a, const void *d_in, void *d_out, int64_t arena_elems,
                                const uint8_t *d_mask, int32_t lowcost_format, int32_t recovery_format,
                                void *stream)
{
    FqFmt low, rec;
    if (!a)
        return GNMR_ERR_INVALID_ARG;
    if (!fmt_of(lowcost_format, low) || !fmt_of(recovery_format, rec))
        return act_fail(GNMR_ERR_INVALID_ARG, "actuator: unknown format");
    if ((!d_in || !d_out) && a->max_end > 0)
        return act_fail(GNMR_ERR_INVALID_ARG, "actuator: NULL activation buffer");
    const int eb = a->dtype == GNMR_DTYPE_BF16 ? 2 : 4;
    if (reinterpret_cast<uintptr_t>(d_in) % eb || reinterpret_cast<uintptr_t>(d_out) % eb)
        return act_fail(GNMR_ERR_INVALID_ARG, "actuator: buffers not aligned to the element size");
    if (arena_elems < a->max_end)
        return act_fail(GNMR_ERR_LAYOUT, "actuator: buffer shorter than the layout");
    if (a->total_rows == 0)
        return GNMR_OK;
    int prev = 0;
    cudaGetDevice(&prev);
    cudaSetDevice(a->device);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    if (a->dtype == GNMR_DTYPE_BF16)
        fake_quant_kernel<1><<<a->grid, kThreads, 0, st>>>(d_in, d_out, a->offset, a->cols, a->row_start,
                                                          a->num_units, a->total_rows, d_mask, low, rec);
    else
        fake_quant_kernel<0><<<a->grid, kThreads, 0, st>>>(d_in, d_out, a->offset, a->cols, a->row_start,
                                                          a->num_units, a->total_rows, d_mask, low, rec);
    const cudaError_t e = cudaGetLastError();
    cudaSetDevice(prev);
    if (e != cudaSuccess)
        return act_fail(GNMR_ERR_CUDA, std::string("actuator launch: ") + cudaGetErrorString(e));
    return GNMR_OK;
}

gnmr_status gnmr_actuator_destroy(gnmr_actuator *a)
{
    if (!a)
        return GNMR_OK;
    int prev = 0;
    cudaGetDevice(&prev);
    cudaSetDevice(a->device);
    const cudaError_t e = a->dmem ? cudaFree(a->dmem) : cudaSuccess;
    cudaSetDevice(prev);
    delete a;
    return e == cudaSuccess ? GNMR_OK : GNMR_ERR_CUDA;
}

}  // extern "C"
