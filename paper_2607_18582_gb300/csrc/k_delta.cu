// Mutant-side kernels: descriptor expansion (GF noise, WS shuffles), the delta
// kernel that rewrites only the mutated neurons' channels of a layer on top of its
// original output, and the score reduction.
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

struct DeltaParams {
    int ih, iw, ic, kh, kw, stride, pad, oh, ow, oc, K;
    int act1, has_add, act2, pool, gap;
    int sk_w, sk_c, sk_stride;
    const float *z; int64_t z_stride; int z_per_input;
    const float *x; int64_t x_stride; int x_per_input;
    const float *skip; int64_t skip_stride; int skip_per_input;
    int64_t t0; int T; int R;
    PatchArgs pa;
    int kmax;
    float *y; int64_t y_stride;
    int lane_mode;
};

struct DeltaRow {
    const float *z, *x, *s, *e;
    int op, j, src_j;
};

// Mutated output of neuron j at conv position (oy, ox) after act1, skip and act2.
// `dot` is the GF/WS correction sum_k e_k x_k of that position.
__device__ __forceinline__ float delta_post(const DeltaParams &p, const DeltaRow &d, int oy, int ox, float dot)
{
    float zz = d.z[((int64_t)oy * p.ow + ox) * p.oc + d.src_j];
    if (d.op == MURE_OP_NAI) zz = -zz;
    else if (d.op == MURE_OP_GF || d.op == MURE_OP_WS) zz = zz + dot;
    float v = d.op == MURE_OP_NEB ? 0.f : act_apply(p.act1, zz);
    if (p.has_add) {
        const float s = d.j < p.sk_c ? d.s[((int64_t)oy * p.sk_stride * p.sk_w + ox * p.sk_stride) * p.sk_c + d.j] : 0.f;
        v = act_apply(p.act2, v + s);
    }
    return v;
}

// sum_k e_k x_k over the receptive field of (oy, ox): one lane, ascending k.
__device__ __forceinline__ float dot_serial(const DeltaParams &p, const DeltaRow &d, int oy, int ox)
{
    float acc = 0.f;
    const int iy0 = oy * p.stride - p.pad, ix0 = ox * p.stride - p.pad;
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

// The same sum with the warp: lane i takes k = i, i+32, ... in ascending order, then
// a butterfly over lanes; every lane ends with the same value.
__device__ __forceinline__ float dot_warp(const DeltaParams &p, const DeltaRow &d, int oy, int ox, int lane)
{
    float acc = 0.f;
    const int iy0 = oy * p.stride - p.pad, ix0 = ox * p.stride - p.pad;
    for (int k = lane; k < p.K; k += 32) {
        const int ci = k % p.ic, t = k / p.ic, kx = t % p.kw, ky = t / p.kw;
        const int iy = iy0 + ky, ix = ix0 + kx;
        if ((unsigned)iy < (unsigned)p.ih && (unsigned)ix < (unsigned)p.iw)
            acc = fmaf(__ldg(d.e + k), __ldg(d.x + ((int64_t)iy * p.iw + ix) * p.ic + ci), acc);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
    return acc;
}

__global__ void __launch_bounds__(128) k_delta(const DeltaParams p)
{
    extern __shared__ float gap_buf[];  // [4 warps][cells] when the layer ends in GAP
    const int lane = threadIdx.x & 31, wib = threadIdx.x >> 5;
    const int64_t wid = (int64_t)blockIdx.x * 4 + wib;
    const int64_t r = wid / p.kmax;
    const int q = (int)(wid % p.kmax);
    if (r >= p.R) return;
    const int g = (int)(r / p.T);
    const int64_t t = p.t0 + r % p.T;
    DeltaRow d;
    d.op = p.pa.op[g];
    if (q >= p.pa.n_neurons[g]) return;
    const int32_t *ids = p.pa.ids + p.pa.neuron_off[g];
    d.j = ids[q];
    d.src_j = d.op == MURE_OP_NS ? ids[q ^ 1] : d.j;
    d.z = p.z + (p.z_per_input ? t : r) * p.z_stride;
    const bool needs_dot = d.op == MURE_OP_GF || d.op == MURE_OP_WS;
    d.x = needs_dot ? p.x + (p.x_per_input ? t : r) * p.x_stride : nullptr;
    d.e = needs_dot ? p.pa.patch + p.pa.patch_off[g] + (int64_t)q * p.K : nullptr;
    d.s = p.has_add ? p.skip + (p.skip_per_input ? t : r) * p.skip_stride : nullptr;
    float *yrow = p.y + r * p.y_stride;

    const int cw = p.pool ? p.ow / 2 : p.ow;
    const int cells = (p.pool ? p.oh / 2 : p.oh) * cw;
    float gsum = 0.f;
    float *gb = gap_buf + wib * cells;
    for (int c0 = 0; c0 < cells; c0 += (p.lane_mode ? 32 : 1)) {
        const int c = p.lane_mode ? c0 + lane : c0;
        const bool active = c < cells;
        float v = 0.f;
        const int cy = active ? c / cw : 0, cx = active ? c % cw : 0;
        if (p.pool) {
            float w4[4];
            for (int sub = 0; sub < 4; ++sub) {
                const int oy = 2 * cy + (sub >> 1), ox = 2 * cx + (sub & 1);
                float dot = 0.f;
                if (needs_dot) dot = p.lane_mode ? (active ? dot_serial(p, d, oy, ox) : 0.f) : dot_warp(p, d, oy, ox, lane);
                w4[sub] = active ? delta_post(p, d, oy, ox, dot) : 0.f;
            }
            v = max4_first(w4[0], w4[1], w4[2], w4[3]);
        } else {
            float dot = 0.f;
            if (needs_dot) dot = p.lane_mode ? (active ? dot_serial(p, d, cy, cx) : 0.f) : dot_warp(p, d, cy, cx, lane);
            v = active ? delta_post(p, d, cy, cx, dot) : 0.f;
        }
        if (p.gap) {
            if (p.lane_mode) { if (active) gb[c] = v; }
            else gsum += v;  // cells in ascending order
        } else if (active && (p.lane_mode || lane == 0)) {
            yrow[(int64_t)c * p.oc + d.j] = v;
        }
    }
    if (p.gap) {
        if (p.lane_mode) {
            __syncwarp();
            if (lane == 0) {
                float s = 0.f;
                for (int c = 0; c < cells; ++c) s += gb[c];
                yrow[d.j] = s / (float)cells;
            }
        } else if (lane == 0) {
            yrow[d.j] = gsum / (float)cells;
        }
    }
}

int launch_delta(const Stage &S, Src z, Src x, Src skip, RowMap rm, const PatchArgs &pa, int kmax, float *y,
                 int64_t y_stride, cudaStream_t s)
{
    if (rm.R <= 0 || kmax <= 0) return 0;
    DeltaParams p{};
    p.ih = S.ih; p.iw = S.iw; p.ic = S.ic; p.kh = S.kh; p.kw = S.kw; p.stride = S.stride; p.pad = S.pad;
    p.oh = S.oh; p.ow = S.ow; p.oc = S.oc; p.K = S.K;
    p.act1 = S.act1; p.has_add = S.has_add; p.act2 = S.act2; p.pool = S.pool; p.gap = S.gap;
    p.sk_w = S.sk_w; p.sk_c = S.sc_c; p.sk_stride = S.sc_stride;
    p.z = z.p; p.z_stride = z.stride; p.z_per_input = z.per_input;
    p.x = x.p; p.x_stride = x.stride; p.x_per_input = x.per_input;
    p.skip = skip.p; p.skip_stride = skip.stride; p.skip_per_input = skip.per_input;
    p.t0 = rm.t0; p.T = rm.T; p.R = rm.R;
    p.pa = pa;
    p.kmax = kmax;
    p.y = y; p.y_stride = y_stride;
    const int cells = (S.pool ? S.oh / 2 : S.oh) * (S.pool ? S.ow / 2 : S.ow);
    // one lane per output position when there are at least 32 of them; otherwise
    // the warp splits each position's fan-in (dense layers)
    p.lane_mode = (S.oh * S.ow) >= 32;
    const size_t smem = S.gap ? (size_t)4 * cells * sizeof(float) : 0;
    const int64_t warps = (int64_t)rm.R * kmax;
    k_delta<<<(unsigned)((warps + 3) / 4), 128, smem, s>>>(p);
    return 1;
}

// --------------------------------------------------------------------- scores --

__global__ void __launch_bounds__(128) k_scores(const uint32_t *__restrict__ kill32, int64_t n_mut, int64_t words32,
                                                const int32_t *__restrict__ label, unsigned long long *totals)
{
    const int lane = threadIdx.x & 31;
    const int64_t i = (int64_t)blockIdx.x * 4 + (threadIdx.x >> 5);
    if (i >= n_mut) return;
    uint32_t any = 0, labels = 0;
    for (int64_t w = lane; w < words32; w += 32) {
        uint32_t bits = kill32[i * words32 + w];
        any |= bits;
        while (bits) {
            const int b = __ffs(bits) - 1;
            labels |= 1u << label[w * 32 + b];
            bits &= bits - 1;
        }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        any |= __shfl_xor_sync(0xffffffffu, any, o);
        labels |= __shfl_xor_sync(0xffffffffu, labels, o);
    }
    if (lane == 0) {
        if (any) atomicAdd(&totals[0], 1ull);
        atomicAdd(&totals[1], (unsigned long long)__popc(labels));
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
    uint32_t m = 0;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x)
        m |= 1u << label[i];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) m |= __shfl_xor_sync(0xffffffffu, m, o);
    if ((threadIdx.x & 31) == 0 && m) atomicOr(mask, m);
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
