// The kill epilogue of a row whose logits a thread holds in registers, shared by the
// output-layer kernel and the tensor-core kernel that computes the output layer in
// its own epilogue: both must reach the same verdicts bit for bit.
#pragma once

#include "common.cuh"
#include "device_util.cuh"

namespace mure {

// argmax / near tie / kill of one row's logits held in registers (CP >= C, unrolled
// and predicated): the same rules as argmax_first and near_tie.
template <int CP>
__device__ __forceinline__ int argmax_reg(const float (&v)[CP], int C)
{
    int best = 0;
    float bv = v[0];
    bool bnan = isnan(v[0]);
#pragma unroll
    for (int c = 1; c < CP; ++c)
        if (c < C && !bnan && (isnan(v[c]) || v[c] > bv)) { best = c; bv = v[c]; bnan = isnan(v[c]); }
    return best;
}

template <int CP>
__device__ __forceinline__ void epilogue_reg(const FinalArgs &fa, int64_t t0, int T, int64_t row, bool in_range,
                                             const float (&v)[CP], int C)
{
    const int64_t lr = in_range ? logical_row(fa.lrow, row) : row;
    const int g = (int)(lr / T);
    const int64_t t = t0 + lr % T;
    const bool valid = in_range && t < fa.n_in;
    int arg = 0;
    bool near = false;
    if (valid) {
        arg = argmax_reg<CP>(v, C);
        float top = v[0], second = -INFINITY;
#pragma unroll
        for (int c = 0; c < CP; ++c) if (c == arg) top = v[c];
#pragma unroll
        for (int c = 0; c < CP; ++c)
            if (c < C && c != arg && v[c] > second) second = v[c];
        near = C >= 2 && (top - second) < 1e-4f * fabsf(top);
    }
    const bool kill = valid && fa.pred0[t] == fa.label[t] && arg != fa.label[t];
    const unsigned kb = __ballot_sync(0xffffffffu, kill);
    const unsigned nb = __ballot_sync(0xffffffffu, near);
    const int lane = threadIdx.x & 31;
    if (fa.compact) {
        // a compacted batch: the warp's rows are any (mutant, input) pairs; the matrix
        // was zeroed, each killed row sets its own bit
        if (kill) atomicOr(fa.kill32 + (int64_t)fa.mutant_id[g] * fa.words32 + (t >> 5), 1u << (t & 31));
        if (lane == 0 && nb && fa.near_ties) atomicAdd(fa.near_ties, (unsigned long long)__popc(nb));
    } else if (lane == 0 && in_range) {
        const int mid = fa.mutant_id[g];
        fa.kill32[(int64_t)mid * fa.words32 + (t >> 5)] = kb;
        if (nb && fa.near_ties) atomicAdd(fa.near_ties, (unsigned long long)__popc(nb));
    }
    if (valid && fa.logits_out) {
        float *o = fa.logits_out + ((int64_t)fa.mutant_id[g] * fa.n_in + t) * C;
#pragma unroll
        for (int c = 0; c < CP; ++c)
            if (c < C) o[c] = v[c];
    }
}

}  // namespace mure
