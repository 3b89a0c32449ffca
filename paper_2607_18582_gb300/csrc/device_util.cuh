// Small device helpers shared by the library's kernels.  Each one fixes a piece of
// arithmetic that must be identical wherever it is used (stage kernels, delta
// kernel, epilogue), because memoized and vanilla results are compared bit for bit.
#pragma once

#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>

namespace mure {

__host__ __device__ __forceinline__ int64_t round4(int64_t n) { return (n + 3) & ~int64_t(3); }

// ReLU returns +0 for every non-positive input (and for NaN), so the sign of a zero
// pre-activation never reaches later layers; ReLU6 also caps at 6.
__device__ __forceinline__ float act_apply(int act, float v)
{
    if (act == MURE_ACT_RELU) return v > 0.f ? v : 0.f;
    if (act == MURE_ACT_RELU6) return v > 0.f ? (v < 6.f ? v : 6.f) : 0.f;
    return v;
}

// 2x2 max pool of one window, top-left first; a later element replaces the
// running maximum only when strictly greater.
__device__ __forceinline__ float max4_first(float a, float b, float c, float d)
{
    float m = a;
    if (b > m) m = b;
    if (c > m) m = c;
    if (d > m) m = d;
    return m;
}

// Global average pooling of channel c of a [P][C] map: fp32 sum over positions in
// ascending order, divided by P.
__device__ __forceinline__ float gap_sum(const float *map, int P, int C, int c)
{
    float s = 0.f;
    for (int q = 0; q < P; ++q) s += map[(int64_t)q * C + c];
    return s / (float)P;
}

// argmax with the lowest index winning ties; a NaN counts as the maximum.
__device__ __forceinline__ int argmax_first(const float *v, int C)
{
    int best = 0;
    for (int c = 1; c < C; ++c) {
        if (isnan(v[best])) break;
        if (isnan(v[c]) || v[c] > v[best]) best = c;
    }
    return best;
}

// A logit vector is a near tie when its top-2 margin is below 1e-4 |max logit|.
__device__ __forceinline__ bool near_tie(const float *v, int C, int arg)
{
    if (C < 2) return false;
    const float top = v[arg];
    float second = -INFINITY;
    for (int c = 0; c < C; ++c)
        if (c != arg && v[c] > second) second = v[c];
    return (top - second) < 1e-4f * fabsf(top);
}

// SplitMix64 (Steele, Lea, Flood 2014): output number i (0-based) of the generator
// whose state starts at `seed` and advances by the golden-ratio increment.
__device__ __forceinline__ uint64_t splitmix64(uint64_t seed, uint64_t i)
{
    uint64_t z = seed + (i + 1) * 0x9E3779B97F4A7C15ull;
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

}  // namespace mure
