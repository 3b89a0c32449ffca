// Mutant-side kernels: descriptor expansion (GF noise, WS shuffles), the delta
// kernel that rewrites only the mutated neurons' channels of a layer on top of its
// original output, and the score reduction.
#include <algorithm>

#include "common.cuh"
#include "device_util.cuh"

namespace mure {

// ------------------------------------------------------------------ expansion --

// Box-Muller in fp64 on SplitMix64 draws: standard normal number f of a stream.
__device__ double gauss_f64(uint64_t stream, int64_t f)
{
    const int64_t pr = f >> 1;
    const double u1 = (double)((splitmix64(stream, (uint64_t)(2 * pr)) >> 11) + 1) * (1.0 / 9007199254740992.0);
    const double u2 = (double)((splitmix64(stream, (uint64_t)(2 * pr + 1)) >> 11) + 1) * (1.0 / 9007199254740992.0);
    const double r = sqrt(-2.0 * log(u1));
    const double th = 6.283185307179586476925286766559 * u2;
    return (f & 1) ? r * sin(th) : r * cos(th);
}

__global__ void k_expand(const ExpandArgs a)
{
    const SlotJob jb = a.jobs[blockIdx.x];
    const uint64_t stream = splitmix64(jb.seed, (uint64_t)jb.q);
    float *out = a.patch + jb.out_off;
    const float *w = a.W[jb.layer] + (int64_t)jb.j * jb.F;
    if (jb.op == MURE_OP_GF) {
        const double sigma = (double)jb.param * a.sigma[jb.layer];
        for (int f = threadIdx.x; f < jb.F; f += blockDim.x) out[f] = (float)(sigma * gauss_f64(stream, f));
        return;
    }
    // WS: Fisher-Yates from the last index down, draw (F-1-i) picks j = floor(u (i+1))
    int32_t *perm = a.perm + jb.perm_off;
    for (int f = threadIdx.x; f < jb.F; f += blockDim.x) perm[f] = f;
    __syncthreads();
    if (threadIdx.x == 0) {
        for (int i = jb.F - 1; i >= 1; --i) {
            const uint64_t x = splitmix64(stream, (uint64_t)(jb.F - 1 - i));
            const double u = (double)(x >> 11) * (1.0 / 9007199254740992.0);
            int jj = (int)(u * (double)(i + 1));
            if (jj > i) jj = i;
            const int32_t t = perm[i];
            perm[i] = perm[jj];
            perm[jj] = t;
        }
    }
    __syncthreads();
    for (int f = threadIdx.x; f < jb.F; f += blockDim.x) {
        const float wp = __ldg(w + perm[f]);
        out[f] = a.ws_as_weights ? wp : wp - __ldg(w + f);
    }
}

int launch_expand(const ExpandArgs &ea, cudaStream_t s)
{
    if (ea.n_jobs <= 0) return 0;
    int launches = 0;
    for (int64_t j0 = 0; j0 < ea.n_jobs; j0 += 65535) {
        ExpandArgs a = ea;
        a.jobs = ea.jobs + j0;
        const int64_t n = ea.n_jobs - j0 < 65535 ? ea.n_jobs - j0 : 65535;
        k_expand<<<(unsigned)n, 256, 0, s>>>(a);
        ++launches;
    }
    return launches;
}

// Population standard deviation of each layer's weights: two passes in fp64, fixed
// block-reduction tree.
__global__ void k_layer_std(const float *const *W, const int64_t *n, double *out)
{
    __shared__ double red[256];
    const float *w = W[blockIdx.x];
    const int64_t cnt = n[blockIdx.x];
    double s = 0.0;
    for (int64_t i = threadIdx.x; i < cnt; i += 256) s += (double)w[i];
    red[threadIdx.x] = s;
    __syncthreads();
    for (int o = 128; o > 0; o >>= 1) {
        if (threadIdx.x < o) red[threadIdx.x] += red[threadIdx.x + o];
        __syncthreads();
    }
    const double mean = red[0] / (double)cnt;
    __syncthreads();
    double ss = 0.0;
    for (int64_t i = threadIdx.x; i < cnt; i += 256) {
        const double d = (double)w[i] - mean;
        ss += d * d;
    }
    red[threadIdx.x] = ss;
    __syncthreads();
    for (int o = 128; o > 0; o >>= 1) {
        if (threadIdx.x < o) red[threadIdx.x] += red[threadIdx.x + o];
        __syncthreads();
    }
    if (threadIdx.x == 0) out[blockIdx.x] = sqrt(red[0] / (double)cnt);
}

int launch_layer_std(const float *const *W, const int64_t *n, int L, double *out, cudaStream_t s)
{
    if (L <= 0) return 0;
    k_layer_std<<<L, 256, 0, s>>>(W, n, out);
    return 1;
}

// ---------------------------------------------------------------------- delta --
//
// The delta of a group at layer l: the values of the mutated neurons' channels of
// x_{l+1} (after layer l's activation, skip add, pooling and GAP), computed from the
// original pre-activation z_l and, for GF / WS, the layer's input x_l.  They go to a
// compact per-row patch buffer patch[r][q][c] (slot q < kmax, output cell c of layer
// l); the first kernel of the suffix applies it on top of the unmutated row.

struct PatchValsParams {
    int ih, iw, ic, kh, kw, stride, pad, oh, ow, oc, K;
    int act1, has_add, act2, pool, gap;
    int sk_w, sk_c, sk_stride;
    int cells;           // output cells of layer l (pooled positions; 1 with GAP)
    int mcells, mcw;     // cells of the post-op map (pooled or not) and its width
    const float *z; int64_t z_stride; int z_per_input;   // channel-major [oc][oh*ow]
    const float *x; int64_t x_stride; int x_per_input;
    const float *skip; int64_t skip_stride; int skip_per_input;
    int64_t t0; int T; int G;
    PatchArgs pa;
    int kmax;
    float *out; int64_t out_stride;
    int warp_dot;        // 1: fan-in sums split across a warp (layers with < 32 positions)
    int skip_dot_ops;    // 1: GF / WS values come from k_patch_dot
    int only_dot_ops;    // 1: the other operators come from k_patch_vals_staged
    int skip_copy_ops;   // 1: NEB / NS slots are applied by the consumer (window GEMM)
    int dw;              // depthwise layer: neuron j's fan-in is its kh x kw filter on input channel j
    int embed;           // embedding: channel j at step t is table entry W[j][id_t]; GF / WS add e[id_t]
    int vocab;
    const float *W, *b;  // the layer's weights [oc][K] and biases (depthwise NS)
};

struct SlotCtx {
    const float *z, *x, *s, *e;
    int op, j, sj;
};

// NS on a depthwise layer: the two neurons exchange filters and biases, but each filter
// stays on its own output channel's input channel, so the mutated channel j is
// recomputed, b[m] + sum_k W[m][k] x_j[k] (m its partner), not taken from channel m.
__device__ __forceinline__ bool dw_switch(const PatchValsParams &p, int op) { return p.dw && op == MURE_OP_NS; }

// Mutated output of neuron j at conv position (oy, ox) after act1, skip and act2;
// `dot` is the GF / WS correction sum_k e_k x_k at that position (depthwise NS: the
// partner's filter on channel j).
__device__ __forceinline__ float slot_post(const PatchValsParams &p, const SlotCtx &d, int oy, int ox, float dot)
{
    float zz = d.z[(int64_t)d.sj * (p.oh * p.ow) + oy * p.ow + ox];
    if (dw_switch(p, d.op)) zz = dot + __ldg(p.b + d.sj);   // the forward kernel's chain: taps from +0, then + b
    else if (d.op == MURE_OP_NAI) zz = -zz;
    else if (d.op == MURE_OP_GF || d.op == MURE_OP_WS) zz = zz + dot;
    float v = d.op == MURE_OP_NEB ? 0.f : act_apply(p.act1, zz);
    if (p.has_add) {
        const float sv = d.j < p.sk_c ? d.s[((int64_t)oy * p.sk_stride * p.sk_w + ox * p.sk_stride) * p.sk_c + d.j] : 0.f;
        v = act_apply(p.act2, v + sv);
    }
    return v;
}

// sum_k e_k x_k over the receptive field of (oy, ox): one thread, ascending k.
__device__ __forceinline__ float dot_serial(const PatchValsParams &p, const SlotCtx &d, int oy, int ox)
{
    float acc = 0.f;
    if (p.embed) {
        // the one-hot input of an embedding: the term of the step's id
        const int id = (int)__ldg(d.x + ox);
        return (unsigned)id < (unsigned)p.vocab ? acc + __ldg(d.e + id) : acc;
    }
    const int iy0 = oy * p.stride - p.pad, ix0 = ox * p.stride - p.pad;
    if (p.dw) {
        // a depthwise neuron: its filter taps (ky, kx) on input channel j
        for (int ky = 0; ky < p.kh; ++ky) {
            const int iy = iy0 + ky;
            for (int kx = 0; kx < p.kw; ++kx) {
                const int ix = ix0 + kx;
                if ((unsigned)iy < (unsigned)p.ih && (unsigned)ix < (unsigned)p.iw)
                    acc = fmaf(__ldg(d.e + ky * p.kw + kx), __ldg(d.x + ((int64_t)iy * p.iw + ix) * p.ic + d.j), acc);
            }
        }
        return acc;
    }
    int k = 0;
    for (int ky = 0; ky < p.kh; ++ky) {
        const int iy = iy0 + ky;
        for (int kx = 0; kx < p.kw; ++kx, k += p.ic) {
            const int ix = ix0 + kx;
            if ((unsigned)iy >= (unsigned)p.ih || (unsigned)ix >= (unsigned)p.iw) continue;
            const float *xp = d.x + ((int64_t)iy * p.iw + ix) * p.ic;
            const float *ep = d.e + k;
            for (int ci = 0; ci < p.ic; ++ci) acc = fmaf(__ldg(ep + ci), __ldg(xp + ci), acc);
        }
    }
    return acc;
}

// The same sum with a warp: lane i takes k = i, i+32, ... in ascending order, then a
// butterfly over the lanes; every lane ends with the same value.
__device__ __forceinline__ float dot_warp(const PatchValsParams &p, const SlotCtx &d, int oy, int ox, int lane)
{
    float acc = 0.f;
    if (p.embed) {
        // one term: every lane returns it (no butterfly)
        const int id = (int)__ldg(d.x + ox);
        return (unsigned)id < (unsigned)p.vocab ? acc + __ldg(d.e + id) : acc;
    }
    const int iy0 = oy * p.stride - p.pad, ix0 = ox * p.stride - p.pad;
    if (p.dw) {
        for (int k = lane; k < p.K; k += 32) {
            const int ky = k / p.kw, kx = k - ky * p.kw, iy = iy0 + ky, ix = ix0 + kx;
            if ((unsigned)iy < (unsigned)p.ih && (unsigned)ix < (unsigned)p.iw)
                acc = fmaf(__ldg(d.e + k), __ldg(d.x + ((int64_t)iy * p.iw + ix) * p.ic + d.j), acc);
        }
    } else if (p.kh == 1 && p.kw == 1 && p.ih == 1 && p.iw == 1) {
        for (int k = lane; k < p.K; k += 32) acc = fmaf(__ldg(d.e + k), __ldg(d.x + k), acc);
    } else {
        for (int k = lane; k < p.K; k += 32) {
            const int ci = k % p.ic, t = k / p.ic, kx = t % p.kw, ky = t / p.kw;
            const int iy = iy0 + ky, ix = ix0 + kx;
            if ((unsigned)iy < (unsigned)p.ih && (unsigned)ix < (unsigned)p.iw)
                acc = fmaf(__ldg(d.e + k), __ldg(d.x + ((int64_t)iy * p.iw + ix) * p.ic + ci), acc);
        }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
    return acc;
}

// Value of map cell c (a pooled window or one position) of slot d.  In warp-dot
// mode every lane of the warp must call it with the same c.
__device__ __forceinline__ float cell_value(const PatchValsParams &p, const SlotCtx &d, int c, int lane)
{
    const bool dot = d.op == MURE_OP_GF || d.op == MURE_OP_WS || dw_switch(p, d.op);
    const int cy = c / p.mcw, cx = c % p.mcw;
    if (!p.pool) {
        const float dv = dot ? (p.warp_dot ? dot_warp(p, d, cy, cx, lane) : dot_serial(p, d, cy, cx)) : 0.f;
        return slot_post(p, d, cy, cx, dv);
    }
    float w4[4];
#pragma unroll
    for (int sub = 0; sub < 4; ++sub) {
        const int oy = 2 * cy + (sub >> 1), ox = 2 * cx + (sub & 1);
        const float dv = dot ? (p.warp_dot ? dot_warp(p, d, oy, ox, lane) : dot_serial(p, d, oy, ox)) : 0.f;
        w4[sub] = slot_post(p, d, oy, ox, dv);
    }
    return max4_first(w4[0], w4[1], w4[2], w4[3]);
}

// One warp per (mutant g, slot q) of one input (blockIdx.y), so the mutants of an
// input read its z and x while they are in L2; the warp's lanes take the cells (one
// lane per cell), or, for layers with fewer than 32 positions, share each cell's dot
// product.
__global__ void __launch_bounds__(256) k_patch_vals(const PatchValsParams p)
{
    extern __shared__ float gap_buf[];  // [8][mcells] with GAP in lane mode
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int item = (int)blockIdx.x * 8 + warp;     // warp-uniform
    if (item >= p.G * p.kmax) return;
    const int g = item / p.kmax, q = item - g * p.kmax;
    if (q >= p.pa.n_neurons[g]) return;
    const int op = p.pa.op[g];
    const bool gfws = op == MURE_OP_GF || op == MURE_OP_WS;
    const bool dot = gfws || dw_switch(p, op);
    if (gfws && p.skip_dot_ops) return;
    if (!dot && p.only_dot_ops) return;
    const int32_t *ids = p.pa.ids + p.pa.neuron_off[g];
    SlotCtx d;
    d.op = op;
    d.j = ids[q];
    d.sj = op == MURE_OP_NS ? ids[q ^ 1] : d.j;
    // the fan-in terms of the sum: GF / WS patch, or (depthwise NS) the partner's filter
    const float *e = gfws ? p.pa.patch + p.pa.patch_off[g] + (int64_t)q * p.K
                          : dot ? p.W + (int64_t)d.sj * p.K : nullptr;
    if (!dot && (p.warp_dot || p.cells < 32)) {
        // no fan-in sum and few cells: one input per lane, its cells in order (a GAP
        // value is the same ascending sum over the map cells as below)
        for (int tl = blockIdx.y * 32 + lane; tl < p.T; tl += gridDim.y * 32) {
            const int64_t r = (int64_t)g * p.T + tl, t = p.t0 + tl;
            d.z = p.z + (p.z_per_input ? t : r) * p.z_stride;
            d.x = nullptr;
            d.s = p.has_add ? p.skip + (p.skip_per_input ? t : r) * p.skip_stride : nullptr;
            d.e = nullptr;
            float *o = p.out + r * p.out_stride + q * p.cells;
            if (p.gap) {
                float s = 0.f;
                for (int cc = 0; cc < p.mcells; ++cc) s += cell_value(p, d, cc, lane);
                o[0] = s / (float)p.mcells;
            } else {
                for (int c = 0; c < p.cells; ++c) o[c] = cell_value(p, d, c, lane);
            }
        }
        return;
    }
    for (int tl = blockIdx.y; tl < p.T; tl += gridDim.y) {
        const int64_t r = (int64_t)g * p.T + tl, t = p.t0 + tl;
        d.z = p.z + (p.z_per_input ? t : r) * p.z_stride;
        d.x = dot ? p.x + (p.x_per_input ? t : r) * p.x_stride : nullptr;
        d.s = p.has_add ? p.skip + (p.skip_per_input ? t : r) * p.skip_stride : nullptr;
        d.e = e;
        float *o = p.out + r * p.out_stride + q * p.cells;
        if (p.gap) {
            // the map cells, then their ascending fp32 sum / count
            float s = 0.f;
            if (p.warp_dot) {
                for (int cc = 0; cc < p.mcells; ++cc) s += cell_value(p, d, cc, lane);
            } else {
                float *gb = gap_buf + warp * p.mcells;
                for (int cc = lane; cc < p.mcells; cc += 32) gb[cc] = cell_value(p, d, cc, lane);
                __syncwarp();
                for (int cc = 0; cc < p.mcells; ++cc) s += gb[cc];
                __syncwarp();
            }
            if (lane == 0) o[0] = s / (float)p.mcells;
        } else if (p.warp_dot) {
            for (int c = 0; c < p.cells; ++c) {
                const float v = cell_value(p, d, c, lane);
                if (lane == 0) o[c] = v;
            }
        } else {
            for (int c = lane; c < p.cells; c += 32) o[c] = cell_value(p, d, c, lane);
        }
    }
}

// The operators without a fan-in sum (NAI, NEB, NS) of a convolution layer in
// memoized mode, one input per block: the input's cached pre-activation maps are
// staged in shared memory once and every mutant slot of the batch reads its channel
// there (the mutants of a batch share the inputs).  The arithmetic is slot_post's,
// so the values equal those of k_patch_vals bit for bit.
template <bool PAIR>
__global__ void __launch_bounds__(256) k_patch_vals_staged(const PatchValsParams p)
{
    extern __shared__ __align__(16) float zs[];   // [oc][oh * ow] of the block's input, then the cell table
    const int P = p.oh * p.ow, nz = p.oc * P;
    int *coff = reinterpret_cast<int *>(zs + nz);   // cell -> top-left position of its window
    const int tl = blockIdx.x;
    const float *z = p.z + (p.t0 + tl) * p.z_stride;
    for (int i = threadIdx.x; i < nz; i += blockDim.x) zs[i] = z[i];
    for (int c = threadIdx.x; c < p.mcells; c += blockDim.x)
        coff[c] = p.pool ? 2 * (c / p.mcw) * p.ow + 2 * (c % p.mcw) : c;
    __syncthreads();
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    // the batch's NEB / NAI / NS slots (listed by the host), one warp per slot
    for (int64_t sl = warp; sl < p.pa.n_vslot; sl += blockDim.x >> 5) {
        const int4 e = p.pa.vslot[sl];
        const int g = e.x - p.pa.dslot_g0, q = e.y, sj = e.z, op = e.w;
        if (p.skip_copy_ops && (op == MURE_OP_NEB || op == MURE_OP_NS)) continue;
        const float *zc = zs + sj * P;
        float *o = p.out + ((int64_t)g * p.T + tl) * p.out_stride + q * p.cells;
        auto post = [&](float zz) {
            if (op == MURE_OP_NAI) zz = -zz;
            return op == MURE_OP_NEB ? 0.f : act_apply(p.act1, zz);
        };
        auto cell = [&](int c) {
            const int b = coff[c];
            return p.pool ? max4_first(post(zc[b]), post(zc[b + 1]), post(zc[b + p.ow]), post(zc[b + p.ow + 1]))
                          : post(zc[b]);
        };
        if constexpr (PAIR) {
            // two neighbouring pooling windows per lane: their 2x4 inputs are two
            // 16-byte loads (the host checks the alignment), one 8-byte store
            for (int c = 2 * lane; c < p.cells; c += 64) {
                float2 r;
                if (op == MURE_OP_NEB) {
                    r = make_float2(0.f, 0.f);
                } else {
                    const int b = coff[c];
                    const float4 u = *reinterpret_cast<const float4 *>(zc + b);
                    const float4 v = *reinterpret_cast<const float4 *>(zc + b + p.ow);
                    r.x = max4_first(post(u.x), post(u.y), post(v.x), post(v.y));
                    r.y = max4_first(post(u.z), post(u.w), post(v.z), post(v.w));
                }
                *reinterpret_cast<float2 *>(o + c) = r;
            }
        } else {
            for (int c = lane; c < p.cells; c += 32) o[c] = cell(c);
        }
    }
}

// Dense layers in memoized mode, kDenseIn inputs per block: the inputs' cached rows
// x and pre-activations z are staged in shared memory; a thread per (slot, input)
// copies the operators without a fan-in sum, a warp per GF / WS slot (the host's list)
// keeps its delta row in registers and forms the dot products of the block's inputs
// exactly as dot_warp does (lane i sums k = i, i+32, ... ascending, then a butterfly).
constexpr int kDenseIn = 8;
constexpr int kDenseKMax = 1024;

template <int KPER>
__global__ void __launch_bounds__(256) k_patch_vals_dense_in(const PatchValsParams p)
{
    extern __shared__ float sm2[];
    const int K = p.K, OC = p.oc;
    float *xs = sm2;                     // [kDenseIn][K]
    float *zs = xs + kDenseIn * K;       // [kDenseIn][OC]
    const int tl0 = blockIdx.x * kDenseIn;
    const int ni = min(kDenseIn, p.T - tl0);
    for (int i = threadIdx.x; i < ni * K; i += blockDim.x) {
        const int a = i / K, k = i - a * K;
        xs[i] = __ldg(p.x + (p.t0 + tl0 + a) * p.x_stride + k);
    }
    for (int i = threadIdx.x; i < ni * OC; i += blockDim.x) {
        const int a = i / OC, c = i - a * OC;
        zs[i] = __ldg(p.z + (p.t0 + tl0 + a) * p.z_stride + c);
    }
    __syncthreads();
    // operators without a fan-in sum
    for (int it = threadIdx.x; it < p.G * p.kmax * kDenseIn; it += blockDim.x) {
        const int sl = it / kDenseIn, a = it - sl * kDenseIn;
        const int g = sl / p.kmax, q = sl - g * p.kmax;
        if (a >= ni || q >= p.pa.n_neurons[g]) continue;
        const int op = p.pa.op[g];
        if (op == MURE_OP_GF || op == MURE_OP_WS) continue;
        const int32_t *ids = p.pa.ids + p.pa.neuron_off[g];
        const int sj = op == MURE_OP_NS ? ids[q ^ 1] : ids[q];
        float zz = zs[a * OC + sj];
        if (op == MURE_OP_NAI) zz = -zz;
        p.out[((int64_t)g * p.T + tl0 + a) * p.out_stride + q] = op == MURE_OP_NEB ? 0.f : act_apply(p.act1, zz);
    }
    // GF / WS: a warp per slot
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    constexpr int kPer = KPER;   // >= ceil(K / 32): the unrolled loop has no dead steps
    for (int64_t s2 = warp; s2 < p.pa.n_dslot; s2 += blockDim.x >> 5) {
        const int g = p.pa.dslot[2 * s2] - p.pa.dslot_g0, q = p.pa.dslot[2 * s2 + 1];
        const int j = p.pa.ids[p.pa.neuron_off[g] + q];
        const float *e = p.pa.patch + p.pa.patch_off[g] + (int64_t)q * K;
        float ev[kPer];
#pragma unroll
        for (int i = 0; i < kPer; ++i) ev[i] = lane + 32 * i < K ? __ldg(e + lane + 32 * i) : 0.f;
        for (int a = 0; a < ni; ++a) {
            const float *xa = xs + a * K;
            float acc = 0.f;
#pragma unroll
            for (int i = 0; i < kPer; ++i)
                if (lane + 32 * i < K) acc = fmaf(ev[i], xa[lane + 32 * i], acc);
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
            if (lane == 0)
                p.out[((int64_t)g * p.T + tl0 + a) * p.out_stride + q] = act_apply(p.act1, zs[a * OC + j] + acc);
        }
    }
}

int launch_patch_vals(const Stage &S, Src z, Src x, Src skip, RowMap rm, const PatchArgs &pa, int kmax, float *out,
                      int64_t out_stride, cudaStream_t s, bool skip_dot_ops, bool skip_copy_ops)
{
    if (rm.R <= 0 || kmax <= 0) return 0;
    PatchValsParams p{};
    p.ih = S.ih; p.iw = S.iw; p.ic = S.ic; p.kh = S.kh; p.kw = S.kw; p.stride = S.stride; p.pad = S.pad;
    p.oh = S.oh; p.ow = S.ow; p.oc = S.oc; p.K = S.K;
    p.act1 = S.act1; p.has_add = S.has_add; p.act2 = S.act2; p.pool = S.pool; p.gap = S.gap;
    p.sk_w = S.sk_w; p.sk_c = S.sc_c; p.sk_stride = S.sc_stride;
    p.mcw = S.pool ? S.ow / 2 : S.ow;
    p.mcells = (S.pool ? S.oh / 2 : S.oh) * p.mcw;
    p.cells = S.gap ? 1 : p.mcells;
    p.z = z.p; p.z_stride = z.stride; p.z_per_input = z.per_input;
    p.x = x.p; p.x_stride = x.stride; p.x_per_input = x.per_input;
    p.skip = skip.p; p.skip_stride = skip.stride; p.skip_per_input = skip.per_input;
    p.t0 = rm.t0; p.T = rm.T; p.G = rm.R / rm.T;
    p.pa = pa;
    p.kmax = kmax;
    p.out = out; p.out_stride = out_stride;
    p.warp_dot = (S.oh * S.ow) < 32;
    p.skip_dot_ops = skip_dot_ops;
    p.skip_copy_ops = skip_copy_ops;
    p.dw = S.kind == MURE_NODE_DWCONV;
    p.embed = S.kind == MURE_NODE_EMBED;
    p.vocab = S.vocab;
    p.W = S.W;
    p.b = S.b;
    const int64_t n_items = (int64_t)p.G * kmax;
    // each warp walks several inputs (blockIdx.y, +gridDim.y, ...): enough blocks to
    // fill the GPU, few enough that block scheduling stays negligible.  Without fan-in
    // sums in the launch, a layer of fewer than 32 cells takes a lane per input (32 inputs
    // per block row), so more than ceil(T / 32) block rows would only idle (ncu: 4 x 608
    // blocks for 2,048 inputs of VGG's conv 256->256, most of them empty)
    const int64_t gx = (n_items + 7) / 8;
    const bool lane_per_input = skip_dot_ops && S.kind != MURE_NODE_DWCONV && (p.warp_dot || p.cells < 32);
    const int64_t gy = std::max<int64_t>(1, std::min<int64_t>(lane_per_input ? (rm.T + 31) / 32 : rm.T,
                                                              (152 * 16 + gx - 1) / gx));
    const dim3 grid((unsigned)gx, (unsigned)gy);
    const size_t smem = (S.gap && !p.warp_dot) ? 8 * (size_t)p.mcells * sizeof(float) : 0;
    // memoized dense layers: all operators per block of inputs
    if (z.per_input && x.per_input && S.kind == MURE_NODE_DENSE && !S.has_add && !S.gap && !S.pool &&
        S.K <= kDenseKMax && S.oh * S.ow == 1) {
        const size_t sm = (size_t)kDenseIn * (S.K + S.oc) * 4;
        if (sm <= 48 * 1024) {
            const unsigned blocks = (unsigned)((rm.T + kDenseIn - 1) / kDenseIn);
            // the unrolled dot loop sized to the fan-in (measured on the LeNet-5
            // workload: FC 400-120 0.222 -> 0.148 ms, FC 120-84 0.207 -> 0.106 ms)
            if (S.K <= 128) k_patch_vals_dense_in<4><<<blocks, 256, sm, s>>>(p);
            else if (S.K <= 256) k_patch_vals_dense_in<8><<<blocks, 256, sm, s>>>(p);
            else if (S.K <= 512) k_patch_vals_dense_in<16><<<blocks, 256, sm, s>>>(p);
            else k_patch_vals_dense_in<kDenseKMax / 32><<<blocks, 256, sm, s>>>(p);
            return 1;
        }
    }
    // memoized convolution layers whose maps fit in shared memory: the non-dot
    // operators per input, staged
    const size_t staged_smem = ((size_t)S.oc * S.oh * S.ow + p.mcells) * 4;
    const bool staged = z.per_input && S.kind == MURE_NODE_CONV2D && !S.has_add && !S.gap &&
                        staged_smem <= 48 * 1024;
    int launches = 0;
    if (staged) {
        if (pa.n_vslot > 0) {
            // pairs of windows: even window columns, 16-byte aligned rows and slots
            // (measured on conv 1->6: the delta of 400 mutants x 10,000 inputs
            // 3.20 -> 3.02 ms)
            const bool pair = S.pool && p.mcw % 2 == 0 && S.ow % 4 == 0 && p.cells % 2 == 0 && out_stride % 2 == 0 &&
                              (reinterpret_cast<uintptr_t>(out) & 7) == 0 && (S.oh * S.ow) % 4 == 0;
            if (pair) k_patch_vals_staged<true><<<(unsigned)rm.T, 256, staged_smem, s>>>(p);
            else k_patch_vals_staged<false><<<(unsigned)rm.T, 256, staged_smem, s>>>(p);
            ++launches;
        }
        if (skip_dot_ops) return launches;
        p.only_dot_ops = 1;
    }
    k_patch_vals<<<grid, 256, smem, s>>>(p);
    return launches + 1;
}

// Materialise rows: out = base with the overlay's channels written in (for suffix
// kernels that read plain rows).  out may alias a per-row base.
__global__ void __launch_bounds__(256) k_rows_overlay(const float *__restrict__ base, int64_t base_stride,
                                                      int base_per_input, int64_t t0, int T, int R, int64_t n_floats,
                                                      const Overlay ov, float *out, int64_t out_stride,
                                                      int rows_per_block, const int32_t *lrow)
{
    extern __shared__ float sm[];  // [rows_per_block][n_floats]
    __shared__ const float *src[64];
    __shared__ float *dst[64];
    __shared__ int gidx[64];
    __shared__ int64_t lidx[64];
    const int64_t r0 = (int64_t)blockIdx.x * rows_per_block;
    const int nr = (int)(R - r0 < rows_per_block ? R - r0 : rows_per_block);
    if (threadIdx.x < nr) {
        const int64_t r = r0 + threadIdx.x, lr = logical_row(lrow, r);
        src[threadIdx.x] = base + (base_per_input ? t0 + lr % T : r) * base_stride;
        dst[threadIdx.x] = out + r * out_stride;
        gidx[threadIdx.x] = (int)(lr / T);
        lidx[threadIdx.x] = lr;
    }
    __syncthreads();
    const int nf = (int)n_floats;
    for (int i = threadIdx.x; i < nr * nf; i += blockDim.x) {
        const int rl = i / nf;
        sm[i] = __ldg(src[rl] + (i - rl * nf));
    }
    __syncthreads();
    const int per_row = ov.kmax * ov.cells;
    for (int i = threadIdx.x; i < nr * per_row; i += blockDim.x) {
        const int rl = i / per_row, rem = i - rl * per_row, q = rem / ov.cells, c = rem - q * ov.cells;
        const int g = gidx[rl];
        if (q >= ov.n_neurons[g]) continue;
        const int j = ov.ids[ov.neuron_off[g] + q];
        sm[rl * nf + c * ov.ch + j] = ov.patch[lidx[rl] * ov.row_stride + q * ov.cells + c];
    }
    __syncthreads();
    for (int i = threadIdx.x; i < nr * nf; i += blockDim.x) {
        const int rl = i / nf;
        dst[rl][i - rl * nf] = sm[i];
    }
}

// Large rows: copy the base rows, then scatter the overlay (two ordered launches).
__global__ void k_copy_rows(const float4 *__restrict__ src, int64_t src_stride4, int per_input, int64_t n4, int64_t t0,
                            int T, int64_t R, float4 *__restrict__ dst, int64_t dst_stride4, const int32_t *lrow)
{
    const int64_t total = R * n4;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < total; i += (int64_t)gridDim.x * blockDim.x) {
        const int64_t r = i / n4, e = i - r * n4;
        dst[r * dst_stride4 + e] = __ldg(src + (per_input ? t0 + logical_row(lrow, r) % T : r) * src_stride4 + e);
    }
}

__global__ void k_overlay_scatter(int64_t T, int64_t R, const Overlay ov, float *out, int64_t out_stride,
                                  const int32_t *lrow)
{
    const int64_t per_row = (int64_t)ov.kmax * ov.cells;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < R * per_row;
         i += (int64_t)gridDim.x * blockDim.x) {
        const int64_t r = i / per_row, lr = logical_row(lrow, r);
        const int rem = (int)(i - r * per_row), q = rem / ov.cells, c = rem - q * ov.cells;
        const int g = (int)(lr / T);
        if (q >= ov.n_neurons[g]) continue;
        const int j = ov.ids[ov.neuron_off[g] + q];
        out[r * out_stride + (int64_t)c * ov.ch + j] = ov.patch[lr * ov.row_stride + q * ov.cells + c];
    }
}

int launch_rows_overlay(Src base, int64_t n_floats, RowMap rm, const Overlay &ov, float *out, int64_t out_stride,
                        cudaStream_t s)
{
    if (rm.R <= 0) return 0;
    // large rows, or rows patched in place (only the mutated channels are written)
    if (n_floats > 8192 || (base.p == out && !base.per_input)) {
        int launches = 0;
        if (!(base.p == out && !base.per_input)) {
            const int64_t n4 = (n_floats + 3) / 4, total = (int64_t)rm.R * n4;
            const int64_t blocks = std::min<int64_t>((total + 255) / 256, 152 * 64);
            k_copy_rows<<<(unsigned)blocks, 256, 0, s>>>(reinterpret_cast<const float4 *>(base.p), base.stride / 4,
                                                         base.per_input, n4, rm.t0, rm.T, rm.R,
                                                         reinterpret_cast<float4 *>(out), out_stride / 4, rm.lrow);
            ++launches;
        }
        const int64_t total = (int64_t)rm.R * ov.kmax * ov.cells;
        if (total > 0) {
            const int64_t blocks = std::min<int64_t>((total + 255) / 256, 152 * 64);
            k_overlay_scatter<<<(unsigned)blocks, 256, 0, s>>>(rm.T, rm.R, ov, out, out_stride, rm.lrow);
            ++launches;
        }
        return launches;
    }
    const int rows_per_block = (int)std::max<int64_t>(1, std::min<int64_t>(64, 8192 / std::max<int64_t>(n_floats, 1)));
    const size_t smem = (size_t)rows_per_block * n_floats * sizeof(float);
    if (smem > 48 * 1024)
        cudaFuncSetAttribute(k_rows_overlay, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    const int64_t blocks = (rm.R + rows_per_block - 1) / rows_per_block;
    k_rows_overlay<<<(unsigned)blocks, 256, smem, s>>>(base.p, base.stride, base.per_input, rm.t0, rm.T, rm.R,
                                                      n_floats, ov, out, out_stride, rows_per_block, rm.lrow);
    return 1;
}

// --------------------------------------------------------------------- scores --

__global__ void __launch_bounds__(128) k_scores(const uint32_t *__restrict__ kill32, int64_t n_mut, int64_t words32,
                                                const int32_t *__restrict__ label, unsigned long long *totals)
{
    const int lane = threadIdx.x & 31;
    const int64_t i = (int64_t)blockIdx.x * 4 + (threadIdx.x >> 5);
    if (i >= n_mut) return;
    // the set of killing labels as kLabelWords 32-bit words (up to kMaxClasses labels)
    uint32_t any = 0, labels[kLabelWords] = {};
    for (int64_t w = lane; w < words32; w += 32) {
        uint32_t bits = kill32[i * words32 + w];
        any |= bits;
        while (bits) {
            const int b = __ffs(bits) - 1;
            const int lb = label[w * 32 + b];
#pragma unroll
            for (int k = 0; k < kLabelWords; ++k)
                if ((lb >> 5) == k) labels[k] |= 1u << (lb & 31);
            bits &= bits - 1;
        }
    }
    int count = 0;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) any |= __shfl_xor_sync(0xffffffffu, any, o);
#pragma unroll
    for (int k = 0; k < kLabelWords; ++k) {
        uint32_t m = labels[k];
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) m |= __shfl_xor_sync(0xffffffffu, m, o);
        count += __popc(m);
    }
    if (lane == 0) {
        if (any) atomicAdd(&totals[0], 1ull);
        atomicAdd(&totals[1], (unsigned long long)count);
    }
}

int launch_scores(const uint32_t *kill32, int64_t n_mut, int64_t words32, const int32_t *label, int n_classes,
                  unsigned long long *totals, cudaStream_t s)
{
    (void)n_classes;
    if (n_mut <= 0) return 0;
    k_scores<<<(unsigned)((n_mut + 3) / 4), 128, 0, s>>>(kill32, n_mut, words32, label, totals);
    return 1;
}

__global__ void k_label_set(const int32_t *__restrict__ label, int64_t n, uint32_t *mask)
{
    uint32_t m[kLabelWords] = {};
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
        const int lb = label[i];
#pragma unroll
        for (int k = 0; k < kLabelWords; ++k)
            if ((lb >> 5) == k) m[k] |= 1u << (lb & 31);
    }
#pragma unroll
    for (int k = 0; k < kLabelWords; ++k) {
        uint32_t v = m[k];
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) v |= __shfl_xor_sync(0xffffffffu, v, o);
        if ((threadIdx.x & 31) == 0 && v) atomicOr(mask + k, v);
    }
}

int launch_label_set(const int32_t *label, int64_t n, uint32_t *mask, cudaStream_t s)
{
    if (n <= 0) return 0;
    int64_t blocks = (n + 255) / 256;
    if (blocks > 1024) blocks = 1024;
    k_label_set<<<(unsigned)blocks, 256, 0, s>>>(label, n, mask);
    return 1;
}

}  // namespace mure
