// Exact unchanged-row elimination (memoized mode; beyond the paper, sound by the
// argument of its soundness theorem).  A single-layer mutant changes only the
// channels of layer l it lists, so row r's suffix (layers l+1 .. L-1) is a function of
// its x_{l+1} alone, the tensor the first suffix stage reads: where every mutated
// channel of the row's patch equals the cached original x_{l+1} of its input bit for
// bit, the suffix reproduces the original forward pass (the kernels are deterministic
// and batch-invariant), so the row's prediction is the original's, its kill bit is 0
// and its logits are the cached original logits.  Such rows are dropped before the
// suffix; the others are listed in ascending order for a compacted batch.
#include "common.cuh"
#include "device_util.cuh"

namespace mure {

namespace {

constexpr int kRowsPerBlock = 256;   // 8 warps x 32 rows

// One warp per row (32 rows per warp in turn): flags[r] = 1 for a row to run, 0 for
// an unchanged row or a padding input; block_cnt[b] = the rows to run of block b.
__global__ void __launch_bounds__(256) k_unchanged_flags(const UnchangedArgs ua, int64_t t0, int T, int R,
                                                         int32_t *flags, int32_t *block_cnt)
{
    __shared__ int cnt;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (threadIdx.x == 0) cnt = 0;
    __syncthreads();
    int mine = 0;
    for (int i = 0; i < 32; ++i) {
        const int64_t r = (int64_t)blockIdx.x * kRowsPerBlock + warp * 32 + i;
        if (r >= R) break;
        const int g = (int)(r / T);
        const int64_t t = t0 + r % T;
        int run = 0;
        if (t < ua.fa.n_in) {
            const int k = ua.n_neurons[g];
            const int32_t *ids = ua.ids + ua.neuron_off[g];
            const float *prow = ua.patch + r * ua.row_stride;
            const float *orig = ua.base + t * ua.base_stride;
            bool same = true;
            for (int q = 0; q < k && same; ++q) {
                const int j = ids[q];
                for (int c = lane; c < ua.cells; c += 32)
                    same &= __float_as_uint(__ldg(prow + (int64_t)q * ua.cells + c)) ==
                            __float_as_uint(__ldg(orig + (int64_t)c * ua.ch + j));
                same = __all_sync(0xffffffffu, same);
            }
            run = same ? 0 : 1;
            if (same) {
                // the original logits stand for the row's
                const float *lg = ua.logits + t * ua.logits_stride;
                const int mid = ua.fa.mutant_id[g];
                if (ua.fa.logits_out)
                    for (int c = lane; c < ua.C; c += 32) ua.fa.logits_out[((int64_t)mid * ua.fa.n_in + t) * ua.C + c] = lg[c];
                if (lane == 0 && ua.fa.near_ties) {
                    float v[kMaxClasses];
                    for (int c = 0; c < ua.C; ++c) v[c] = lg[c];
                    const int arg = argmax_first(v, ua.C);
                    if (near_tie(v, ua.C, arg)) atomicAdd(ua.fa.near_ties, 1ull);
                }
            }
        }
        if (lane == 0) flags[r] = run;
        mine += run;
    }
    if (lane == 0 && mine) atomicAdd(&cnt, mine);
    __syncthreads();
    if (threadIdx.x == 0) block_cnt[blockIdx.x] = cnt;
}

// Exclusive scan of the block counts (one block); count = their sum.
__global__ void __launch_bounds__(1024) k_unchanged_scan(int32_t *block_cnt, int nb, int32_t *count)
{
    __shared__ int32_t part[1024];
    __shared__ int32_t carry;
    if (threadIdx.x == 0) carry = 0;
    __syncthreads();
    for (int base = 0; base < nb; base += 1024) {
        const int i = base + threadIdx.x;
        const int32_t v = i < nb ? block_cnt[i] : 0;
        part[threadIdx.x] = v;
        __syncthreads();
        // Hillis-Steele inclusive scan of the chunk
        for (int off = 1; off < 1024; off <<= 1) {
            const int32_t add = threadIdx.x >= off ? part[threadIdx.x - off] : 0;
            __syncthreads();
            part[threadIdx.x] += add;
            __syncthreads();
        }
        if (i < nb) block_cnt[i] = carry + part[threadIdx.x] - v;
        __syncthreads();
        if (threadIdx.x == 1023) carry += part[1023];
        __syncthreads();
    }
    if (threadIdx.x == 0) *count = carry;
}

// lrow[offset of block b + rank of r among its block's rows to run] = r.
__global__ void __launch_bounds__(256) k_unchanged_compact(const int32_t *flags, const int32_t *block_off, int R,
                                                           int32_t *lrow)
{
    __shared__ int32_t warp_cnt[8];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    int32_t total = 0;
    // rows of warp w: 32 consecutive groups of 32 rows? no: row = block * 256 + w * 32 + i
    // (the flags kernel's order); each lane takes row i = lane
    const int64_t r = (int64_t)blockIdx.x * kRowsPerBlock + warp * 32 + lane;
    const int f = r < R ? flags[r] : 0;
    const unsigned b = __ballot_sync(0xffffffffu, f);
    if (lane == 0) warp_cnt[warp] = __popc(b);
    __syncthreads();
    for (int w = 0; w < warp; ++w) total += warp_cnt[w];
    if (f) lrow[block_off[blockIdx.x] + total + __popc(b & ((1u << lane) - 1u))] = (int32_t)r;
}

}  // namespace

int launch_unchanged(const UnchangedArgs &ua, RowMap rm, int32_t *flags, int32_t *block_cnt, int32_t *lrow,
                     int32_t *count, cudaStream_t s)
{
    const int nb = (rm.R + kRowsPerBlock - 1) / kRowsPerBlock;
    k_unchanged_flags<<<nb, 256, 0, s>>>(ua, rm.t0, rm.T, rm.R, flags, block_cnt);
    k_unchanged_scan<<<1, 1024, 0, s>>>(block_cnt, nb, count);
    k_unchanged_compact<<<nb, 256, 0, s>>>(flags, block_cnt, rm.R, lrow);
    return 3;
}

}  // namespace mure
