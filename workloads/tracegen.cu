// Synthetic gradient generator for the GNMR workloads (input generation only;
// no GNMR arithmetic).  Unit u at step t holds s_u * z, z ~ N(0, 1) iid,
// stored as fp32 or bf16 (round to nearest even).  z comes from the
// counter-based generator Philox4x32-10 (Salmon, Moraes, Dror, Shaw, "Parallel
// random numbers: as easy as 1, 2, 3", SC 2011) keyed by (seed, attempt) with
// counter (element quad index, unit, step), then the Box-Muller transform, so
// any unit can be regenerated alone and identically.
//
// C entry point (plain pointers, device memory unless noted):
//   int tracegen_fill(void *arena, int dtype, const int64_t *task_unit,
//                     const int64_t *task_start, const int64_t *task_count,
//                     int64_t num_tasks, const int64_t *unit_offset,
//                     const double *unit_scale, const int32_t *unit_attempt,
//                     uint32_t seed, uint32_t step, void *stream)
// Each task writes task_count elements of unit task_unit starting at element
// task_start of that unit.  Returns the CUDA launch status.
#include <cstdint>

#include <cuda_bf16.h>
#include <cuda_runtime.h>

namespace {

struct U4 {
    uint32_t x, y, z, w;
};

__device__ __forceinline__ U4 philox_round(U4 c, uint32_t k0, uint32_t k1)
{
    const uint32_t m0 = 0xD2511F53u, m1 = 0xCD9E8D57u;
    const uint32_t hi0 = __umulhi(m0, c.x), lo0 = m0 * c.x;
    const uint32_t hi1 = __umulhi(m1, c.z), lo1 = m1 * c.z;
    return U4{hi1 ^ c.y ^ k0, lo1, hi0 ^ c.w ^ k1, lo0};
}

__device__ __forceinline__ U4 philox4x32_10(U4 c, uint32_t k0, uint32_t k1)
{
#pragma unroll
    for (int r = 0; r < 10; ++r) {
        c = philox_round(c, k0, k1);
        k0 += 0x9E3779B9u;
        k1 += 0xBB67AE85u;
    }
    return c;
}

// Uniform in (0, 1): 24 random bits, offset by half an ulp.
__device__ __forceinline__ float unit_open(uint32_t x)
{
    return (static_cast<float>(x >> 8) + 0.5f) * (1.0f / 16777216.0f);
}

__global__ void fill_kernel(void *arena, int dtype, const int64_t *task_unit, const int64_t *task_start,
                            const int64_t *task_count, int64_t num_tasks, const int64_t *unit_offset,
                            const double *unit_scale, const int32_t *unit_attempt, uint32_t seed,
                            uint32_t step)
{
    for (int64_t task = blockIdx.x; task < num_tasks; task += gridDim.x) {
        const int64_t u = task_unit[task];
        const int64_t start = task_start[task];
        const int64_t count = task_count[task];
        const float s = static_cast<float>(unit_scale[u]);
        const uint32_t attempt = static_cast<uint32_t>(unit_attempt[u]);
        const int64_t base = unit_offset[u];
        // element i of the unit takes output (i % 4) of quad i / 4
        for (int64_t q = start / 4 + threadIdx.x; q * 4 < start + count; q += blockDim.x) {
            const U4 r = philox4x32_10(U4{static_cast<uint32_t>(q), static_cast<uint32_t>(q >> 32),
                                          static_cast<uint32_t>(u), step},
                                       seed, attempt);
            float z[4];
            {
                const float rad = sqrtf(-2.0f * logf(unit_open(r.x)));
                float sn, cs;
                sincospif(2.0f * unit_open(r.y), &sn, &cs);
                z[0] = rad * cs;
                z[1] = rad * sn;
            }
            {
                const float rad = sqrtf(-2.0f * logf(unit_open(r.z)));
                float sn, cs;
                sincospif(2.0f * unit_open(r.w), &sn, &cs);
                z[2] = rad * cs;
                z[3] = rad * sn;
            }
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const int64_t i = q * 4 + j;
                if (i < start || i >= start + count)
                    continue;
                const float v = s * z[j];
                if (dtype == 1)
                    reinterpret_cast<__nv_bfloat16 *>(arena)[base + i] = __float2bfloat16_rn(v);
                else
                    reinterpret_cast<float *>(arena)[base + i] = v;
            }
        }
    }
}

}  // namespace

extern "C" int tracegen_fill(void *arena, int dtype, const int64_t *task_unit, const int64_t *task_start,
                             const int64_t *task_count, int64_t num_tasks, const int64_t *unit_offset,
                             const double *unit_scale, const int32_t *unit_attempt, uint32_t seed,
                             uint32_t step, void *stream)
{
    if (num_tasks <= 0)
        return 0;
    int dev = 0, sms = 1;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    const int64_t want = sms * 8;
    const int grid = static_cast<int>(num_tasks < want ? num_tasks : want);
    fill_kernel<<<grid, 256, 0, static_cast<cudaStream_t>(stream)>>>(
        arena, dtype, task_unit, task_start, task_count, num_tasks, unit_offset, unit_scale,
        unit_attempt, seed, step);
    return static_cast<int>(cudaGetLastError());
}
