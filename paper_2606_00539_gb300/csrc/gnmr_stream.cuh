// Streaming sum of squares over a gradient segment and the completion
// ticket, shared by the step kernel and the allocation-free norms entry point
// (device code only).
//
// A warp reads a segment with 16-byte loads on the non-coherent path (no L1
// allocation, 256-byte L2 prefetch), squares in fp32, sums short blocks in
// fp32 and the blocks as an unevaluated pair of floats (hi + lo, about 48
// significant bits), then adds the 32 lanes' totals with an fp32 xor
// butterfly (non-negative terms: at most five roundings, about 3e-7
// relative) and converts to fp64 once per segment.  It flags segments whose fp32 squares
// may have lost accuracy (denormal or overflowing squares), which the caller
// recomputes with exact fp64 squares.  Any element alignment: a scalar head
// and tail around the 16-byte body.
//
// Why float pairs: on GB300 an fp64 add has a 64-cycle dependent latency and
// the SM retires one fp64 warp-instruction every 20 cycles, shared by all its
// warps.  A five-round fp64 shuffle reduction per segment held that pipe 40 %
// of the time on layouts of many small units and stalled the streams; the
// fp32 error-free additions run on the fp32 pipe.  The pairs keep a long run
// of blocks accurate; the final five-level tree over the lanes does not need
// them (measured: a pair-wise TwoSum butterfly there cost 1 us more on 100K
// units).
#ifndef GNMR_STREAM_CUH
#define GNMR_STREAM_CUH

#include <cstdint>

namespace gnmr {
namespace {

constexpr unsigned kFull = 0xffffffffu;
constexpr int kFlush = 16;   // main-loop iterations summed in fp32 before the pair add

template <int DT> struct Elem;
template <> struct Elem<0> {             // fp32
    static constexpr int kBytes = 4;
    static constexpr uint32_t kMagnitude = 0x7fffffffu;
};
template <> struct Elem<1> {             // bf16, two per 32-bit word
    static constexpr int kBytes = 2;
    static constexpr uint32_t kMagnitude = 0x7fff7fffu;
};

// 16-byte streaming load: non-coherent read-only path, no L1 allocation,
// 256-byte L2 prefetch granularity.
constexpr int kVecWords = 4;
constexpr int kVecBytes = 16;
struct alignas(kVecBytes) Vec {
    uint32_t w[kVecWords];
};

__device__ __forceinline__ Vec ld_stream(const Vec *p)
{
    Vec r;
    asm("ld.global.nc.L1::no_allocate.L2::256B.v4.u32 {%0, %1, %2, %3}, [%4];"
        : "=r"(r.w[0]), "=r"(r.w[1]), "=r"(r.w[2]), "=r"(r.w[3]) : "l"(p));
    return r;
}

__device__ __forceinline__ Vec zero_vec()
{
    Vec r;
#pragma unroll
    for (int i = 0; i < kVecWords; ++i)
        r.w[i] = 0u;
    return r;
}

__device__ __forceinline__ uint32_t vec_or(const Vec &v)
{
    uint32_t o = 0;
#pragma unroll
    for (int i = 0; i < kVecWords; ++i)
        o |= v.w[i];
    return o;
}

// One element as an fp32 bit pattern (bf16 is the upper half of an fp32).
template <int DT> __device__ __forceinline__ uint32_t ld_elem_bits(const char *p);
template <> __device__ __forceinline__ uint32_t ld_elem_bits<0>(const char *p)
{
    return __ldg(reinterpret_cast<const unsigned int *>(p));
}
template <> __device__ __forceinline__ uint32_t ld_elem_bits<1>(const char *p)
{
    return static_cast<uint32_t>(__ldg(reinterpret_cast<const unsigned short *>(p))) << 16;
}

// Sum of squares of the elements packed in one vector, in fp32 (two
// independent chains per vector).
template <int DT> __device__ __forceinline__ float vec_sumsq(const Vec &v);
template <> __device__ __forceinline__ float vec_sumsq<0>(const Vec &v)
{
    float s0 = 0.f, s1 = 0.f;
#pragma unroll
    for (int i = 0; i < kVecWords; i += 2) {
        const float a = __uint_as_float(v.w[i]), b = __uint_as_float(v.w[i + 1]);
        s0 = fmaf(a, a, s0);
        s1 = fmaf(b, b, s1);
    }
    return s0 + s1;
}
template <> __device__ __forceinline__ float vec_sumsq<1>(const Vec &v)
{
    float s0 = 0.f, s1 = 0.f;
#pragma unroll
    for (int i = 0; i < kVecWords; ++i) {
        const float lo = __uint_as_float(v.w[i] << 16);
        const float hi = __uint_as_float(v.w[i] & 0xffff0000u);
        s0 = fmaf(lo, lo, s0);
        s1 = fmaf(hi, hi, s1);
    }
    return s0 + s1;
}

__device__ __forceinline__ double warp_allreduce_sum(double v)
{
    // xor butterfly: both partners add the same two operands, so every lane
    // ends with the same bits.
#pragma unroll
    for (int o = 16; o > 0; o >>= 1)
        v += __shfl_xor_sync(kFull, v, o);
    return v;
}

// Knuth's TwoSum: s + e == a + b exactly, s = fl(a + b), in any operand
// order (fl(a + b) == fl(b + a), and e is the exact rounding error).
__device__ __forceinline__ void two_sum(float a, float b, float &s, float &e)
{
    s = __fadd_rn(a, b);
    const float bb = __fadd_rn(s, -a);
    e = __fadd_rn(__fadd_rn(a, -__fadd_rn(s, -bb)), __fadd_rn(b, -bb));
}

// (hi, lo) += x for an unevaluated pair hi + lo.
__device__ __forceinline__ void pair_add(float &hi, float &lo, float x)
{
    float s, e;
    two_sum(hi, x, s, e);
    hi = s;
    lo = __fadd_rn(lo, e);
}

// Sum of squares of n elements at seg, by the whole warp.  Returns the sum
// in every lane and sets `suspect` when fp32 squaring may have lost accuracy:
// a nonzero segment whose sum is below 2^-100 (denormal squares) or above
// 2^100 (possible fp32 overflow), or a NaN/Inf sum.
template <int DT, int kUnroll>
__device__ __forceinline__ double warp_segment_sumsq(const char *seg, int64_t n, int lane,
                                                     bool &suspect)
{
    constexpr int kEB = Elem<DT>::kBytes;
    constexpr int kVE = kVecBytes / kEB;
    constexpr uint32_t kAlign = kVecBytes - 1;
    const uint32_t mis = static_cast<uint32_t>(reinterpret_cast<uintptr_t>(seg) & kAlign);
    int64_t head = static_cast<int64_t>(((kVecBytes - mis) & kAlign) / kEB);
    head = head < n ? head : n;
    const int64_t nvec = (n - head) / kVE;
    const int64_t tail = n - head - nvec * kVE;

    uint32_t bits = 0;
    float blk = 0.f;
    if (lane < head) {
        const uint32_t w = ld_elem_bits<DT>(seg + lane * kEB);
        const float x = __uint_as_float(w);
        bits |= w;
        blk = fmaf(x, x, blk);
    }
    if (lane < tail) {
        const uint32_t w = ld_elem_bits<DT>(seg + (head + nvec * kVE + lane) * kEB);
        const float x = __uint_as_float(w);
        bits |= w;
        blk = fmaf(x, x, blk);
    }

    const Vec *v = reinterpret_cast<const Vec *>(seg + head * kEB);
    float acc_hi = 0.f, acc_lo = 0.f;
    int64_t i = lane;
    int cnt = 0;
    for (; i + (kUnroll - 1) * 32 < nvec; i += kUnroll * 32) {
        Vec r[kUnroll];
#pragma unroll
        for (int j = 0; j < kUnroll; ++j)
            r[j] = ld_stream(v + i + j * 32);
        float a[kUnroll];
#pragma unroll
        for (int j = 0; j < kUnroll; ++j) {
            a[j] = vec_sumsq<DT>(r[j]);
            bits |= vec_or(r[j]);
        }
#pragma unroll
        for (int w = kUnroll / 2; w > 0; w >>= 1)     // pairwise tree
#pragma unroll
            for (int j = 0; j < w; ++j)
                a[j] += a[j + w];
        blk += a[0];
        if (++cnt == kFlush) {
            pair_add(acc_hi, acc_lo, blk);
            blk = 0.f;
            cnt = 0;
        }
    }
    // Fewer than kUnroll vectors left for this lane: one predicated batch.
    {
        Vec r[kUnroll - 1];
#pragma unroll
        for (int j = 0; j < kUnroll - 1; ++j)
            r[j] = (i + j * 32 < nvec) ? ld_stream(v + i + j * 32) : zero_vec();
        float a = 0.f;
#pragma unroll
        for (int j = 0; j < kUnroll - 1; ++j) {
            a += vec_sumsq<DT>(r[j]);
            bits |= vec_or(r[j]);
        }
        blk += a;
    }
    pair_add(acc_hi, acc_lo, blk);
    // the lanes' totals (non-negative) summed by an fp32 xor butterfly: both
    // partners add the same two operands, so every lane ends with the same bits
    float tot = acc_hi + acc_lo;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1)
        tot += __shfl_xor_sync(kFull, tot, o);
    const float lead = tot;
    const double acc = static_cast<double>(tot);
    bits = __reduce_or_sync(kFull, bits);
    suspect = (bits & Elem<DT>::kMagnitude) != 0u && !(lead >= 0x1p-100f && lead <= 0x1p+100f);
    return acc;
}

// Exact-product fallback: each element squared in fp64 (exact for fp32 and
// bf16 inputs) and summed in fp64.  Taken only for segments flagged suspect.
template <int DT>
__device__ __noinline__ double warp_segment_sumsq_f64(const char *seg, int64_t n, int lane)
{
    constexpr int kEB = Elem<DT>::kBytes;
    double acc = 0.0;
    for (int64_t i = lane; i < n; i += 32) {
        const double x = static_cast<double>(__uint_as_float(ld_elem_bits<DT>(seg + i * kEB)));
        acc = fma(x, x, acc);
    }
    return warp_allreduce_sum(acc);
}

// Ticket increment with acquire-release semantics at GPU scope: it publishes
// the caller's earlier writes (and, after a barrier, those of its CTA) and,
// for the caller that draws the last ticket, makes every earlier holder's
// writes visible.
__device__ __forceinline__ uint32_t ticket_acq_rel(uint32_t *t)
{
    uint32_t old;
    asm volatile("atom.acq_rel.gpu.global.add.u32 %0, [%1], 1;" : "=r"(old) : "l"(t) : "memory");
    return old;
}

}  // namespace
}  // namespace gnmr

#endif  // GNMR_STREAM_CUH
