// Direct convolution for layers whose per-row input fits in shared memory (the
// LeNet-5 convolutions): a block stages whole zero-padded input rows and the layer's
// weights in shared memory, and each thread computes a 2x2 pooling window (or four
// positions) for every output channel.  The receptive-field offsets are compile-time
// constants, so the inner loop is loads with immediate offsets and FMAs.
//
// Arithmetic: every output element is the same fp32 chain as in k_stage_simt, i.e.
// acc = fma(x_k, w_k, acc) over k = (ky, kx, ci) ascending from +0 (zero-padding taps
// give x = 0), then + bias; the post-ops are the same helpers.  The two kernels give
// identical bits, so which one runs a layer does not change any result.
#include <algorithm>

#include "common.cuh"
#include "device_util.cuh"

namespace mure {

struct ConvSmallParams {
    const float *x; int64_t x_stride; int x_per_input;
    int64_t t0; int T; int R;
    int ih, iw, oh, ow;
    const float *Wt;  // [K][OC]
    const float *b;
    int act1;
    float *z; int64_t z_stride;
    float *y; int64_t y_stride;
    int rows_per_block, cells;
    Overlay ov;       // mutated channels of the input rows (ov.patch null: none)
};

// KH x KW filter, IC input channels, OC output channels (OCT of them per thread),
// WP / HP padded input width / height, PAD zero padding, POOL: 2x2 max pool after
// the activation.
template <int KH, int KW, int IC, int OC, int OCT, int WP, int HP, int PAD, bool POOL>
__global__ void __launch_bounds__(256, 3) k_conv_small(const ConvSmallParams p)
{
    constexpr int K = KH * KW * IC;
    constexpr int TILE = HP * WP * IC;
    constexpr int NSPLIT = OC / OCT;
    extern __shared__ __align__(16) float sm[];
    float *ws = sm;              // [K][OC]
    float *xs = sm + K * OC;     // [rows_per_block][TILE]
    __shared__ const float *src_row[32];
    __shared__ int row_g[32];
    const int tid = threadIdx.x;
    const int64_t row0 = (int64_t)blockIdx.x * p.rows_per_block;
    const int nrows = (int)(p.R - row0 < p.rows_per_block ? p.R - row0 : p.rows_per_block);
    if (tid < nrows) {
        const int64_t row = row0 + tid;
        src_row[tid] = p.x + (p.x_per_input ? (p.t0 + row % p.T) : row) * p.x_stride;
        row_g[tid] = (int)(row / p.T);
    }
    __syncthreads();

    for (int i = tid; i < K * OC; i += blockDim.x) ws[i] = __ldg(p.Wt + i);
    if (PAD == 0 && TILE % 4 == 0 && p.x_stride % 4 == 0) {
        // the padded tile is the row itself: 16-byte copies, several in flight
        constexpr int T4 = TILE / 4;
#pragma unroll 4
        for (int i = tid; i < nrows * T4; i += blockDim.x) {
            const int rl = i / T4, e = i - rl * T4;
            reinterpret_cast<float4 *>(xs)[i] = __ldg(reinterpret_cast<const float4 *>(src_row[rl]) + e);
        }
    } else {
#pragma unroll 4
        for (int i = tid; i < nrows * TILE; i += blockDim.x) {
            const int rl = i / TILE, e = i - rl * TILE;
            const int ci = e % IC, pix = e / IC, px = pix % WP, py = pix / WP;
            const int iy = py - PAD, ix = px - PAD;
            float v = 0.f;
            if ((unsigned)iy < (unsigned)p.ih && (unsigned)ix < (unsigned)p.iw)
                v = __ldg(src_row[rl] + (iy * p.iw + ix) * IC + ci);
            xs[i] = v;
        }
    }
    __syncthreads();
    if (p.ov.patch) {
        // the mutant's channels of each input row, written over the staged tile
        const int per_row = p.ov.kmax * p.ov.cells;
        for (int i = tid; i < nrows * per_row; i += blockDim.x) {
            const int rl = i / per_row, rem = i - rl * per_row, q = rem / p.ov.cells, c = rem - q * p.ov.cells;
            const int g = row_g[rl];
            if (q >= p.ov.n_neurons[g]) continue;
            const int j = p.ov.ids[p.ov.neuron_off[g] + q];
            const int py = c / p.iw, px = c - py * p.iw;
            xs[rl * TILE + ((py + PAD) * WP + px + PAD) * IC + j] =
                p.ov.patch[(row0 + rl) * p.ov.row_stride + q * p.ov.cells + c];
        }
        __syncthreads();
    }

    const int per_row = p.cells * NSPLIT;
    const int rl = tid / per_row, cell = (tid % per_row) / NSPLIT, n0 = (tid % NSPLIT) * OCT;
    if (rl >= nrows) return;
    const int64_t row = row0 + rl;
    // the four positions this thread computes: a pooling window, or 4 consecutive
    // positions of one output row (ow % 4 == 0 when not pooling)
    int oy[4], ox[4];
    if (POOL) {
        const int pw = p.ow / 2, py = cell / pw, px = cell % pw;
#pragma unroll
        for (int s = 0; s < 4; ++s) { oy[s] = 2 * py + (s >> 1); ox[s] = 2 * px + (s & 1); }
    } else {
        const int q = cell * 4;
#pragma unroll
        for (int s = 0; s < 4; ++s) { oy[s] = (q + s) / p.ow; ox[s] = (q + s) % p.ow; }
    }
    const float *xt = xs + rl * TILE;
    float acc[4][OCT];
#pragma unroll
    for (int s = 0; s < 4; ++s)
#pragma unroll
        for (int n = 0; n < OCT; ++n) acc[s][n] = 0.f;
    int base[4];
#pragma unroll
    for (int s = 0; s < 4; ++s) base[s] = (oy[s] * WP + ox[s]) * IC;
#pragma unroll 1
    for (int ky = 0; ky < KH; ++ky)
#pragma unroll
        for (int kx = 0; kx < KW; ++kx)
#pragma unroll
            for (int ci = 0; ci < IC; ++ci) {
                const int k = (ky * KW + kx) * IC + ci;
                float w[OCT];
#pragma unroll
                for (int n = 0; n < OCT; ++n) w[n] = ws[k * OC + n0 + n];
#pragma unroll
                for (int s = 0; s < 4; ++s) {
                    const float a = xt[base[s] + (ky * WP + kx) * IC + ci];
#pragma unroll
                    for (int n = 0; n < OCT; ++n) acc[s][n] = fmaf(a, w[n], acc[s][n]);
                }
            }

    float *yrow = p.y + row * p.y_stride;
#pragma unroll
    for (int nn = 0; nn < OCT; ++nn) {
        const int n = n0 + nn;
        const float bias = __ldg(p.b + n);
        float v[4];
#pragma unroll
        for (int s = 0; s < 4; ++s) {
            const float zz = acc[s][nn] + bias;
            if (p.z) p.z[row * p.z_stride + (int64_t)n * (p.oh * p.ow) + oy[s] * p.ow + ox[s]] = zz;
            v[s] = act_apply(p.act1, zz);
        }
        if (POOL) {
            yrow[(int64_t)cell * OC + n] = max4_first(v[0], v[1], v[2], v[3]);
        } else {
#pragma unroll
            for (int s = 0; s < 4; ++s) yrow[((int64_t)oy[s] * p.ow + ox[s]) * OC + n] = v[s];
        }
    }
}

namespace {

template <int KH, int KW, int IC, int OC, int OCT, int WP, int HP, int PAD, bool POOL>
int launch_small(const Stage &S, Src x, RowMap rm, float *z_out, int64_t z_stride, float *y_out, int64_t y_stride,
                 cudaStream_t s, const Overlay *ov)
{
    ConvSmallParams p{};
    if (ov) p.ov = *ov;
    p.x = x.p; p.x_stride = x.stride; p.x_per_input = x.per_input;
    p.t0 = rm.t0; p.T = rm.T; p.R = rm.R;
    p.ih = S.ih; p.iw = S.iw; p.oh = S.oh; p.ow = S.ow;
    p.Wt = S.Wt; p.b = S.b; p.act1 = S.act1;
    p.z = z_out; p.z_stride = z_stride;
    p.y = y_out; p.y_stride = y_stride;
    p.cells = POOL ? (S.oh / 2) * (S.ow / 2) : S.oh * S.ow / 4;
    p.rows_per_block = std::min(32, 256 / (p.cells * (OC / OCT)));
    const size_t smem = ((size_t)KH * KW * IC * OC + (size_t)p.rows_per_block * HP * WP * IC) * sizeof(float);
    // per device, cheap: allow more than the default 48 KiB of dynamic shared memory
    cudaFuncSetAttribute(k_conv_small<KH, KW, IC, OC, OCT, WP, HP, PAD, POOL>,
                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    const int64_t blocks = (rm.R + p.rows_per_block - 1) / p.rows_per_block;
    k_conv_small<KH, KW, IC, OC, OCT, WP, HP, PAD, POOL>
        <<<(unsigned)blocks, p.rows_per_block * p.cells * (OC / OCT), smem, s>>>(p);
    return 1;
}

}  // namespace

// Which layers the shared-memory kernel takes: stride 1, no residual add or GAP, and
// one of the compiled geometries.
int conv_small_variant(const Stage &S)
{
    if (S.kind != MURE_NODE_CONV2D || S.stride != 1 || S.has_add || S.gap) return 0;
    if (S.kh == 5 && S.kw == 5 && S.ic == 6 && S.oc == 16 && S.pad == 0 && S.ih == 14 && S.iw == 14 && S.pool) return 1;
    if (S.kh == 5 && S.kw == 5 && S.ic == 1 && S.oc == 6 && S.pad == 2 && S.ih == 28 && S.iw == 28 && S.pool) return 2;
    return 0;
}

int launch_conv_small(const Stage &S, Src x, RowMap rm, float *z_out, int64_t z_stride, float *y_out,
                      int64_t y_stride, cudaStream_t s, const Overlay *ov)
{
    if (rm.R <= 0) return 0;
    switch (S.variant) {
    case 1: return launch_small<5, 5, 6, 16, 4, 14, 14, 0, true>(S, x, rm, z_out, z_stride, y_out, y_stride, s, ov);
    case 2: return launch_small<5, 5, 1, 6, 6, 32, 32, 2, true>(S, x, rm, z_out, z_stride, y_out, y_stride, s, ov);
    }
    return 0;
}

}  // namespace mure

// ------------------------------------------------ GF / WS delta, small layers --
//
// For the geometries above, the GF / WS correction sum_k e_k x_k of every output
// position is a one-channel convolution of the layer input with the mutant's patch
// vector e.  A block takes one mutant and several inputs: e and the zero-padded input
// tiles sit in shared memory and the taps are unrolled, in the generic kernel's order
// (k = (ky, kx, ci) ascending, fma chain from +0; a padding tap adds e * 0, which
// leaves the chain unchanged), so both kernels give the same bits.

namespace mure {

struct PatchDotParams {
    const float *z; int64_t z_stride; int z_per_input;   // channel-major [oc][oh*ow]
    const float *x; int64_t x_stride; int x_per_input;
    int64_t t0; int T; int G;
    int ih, iw, oh, ow, act1;
    const int32_t *op, *n_neurons, *ids;
    const int64_t *neuron_off, *patch_off;
    const int32_t *dslot; int64_t n_dslot; int32_t dslot_g0;   // the batch's GF / WS slots
    const float *e_all;
    float *out; int64_t out_stride;
    int cells, rows_per_block;
    int oc;
};

template <int KH, int KW, int IC, int WP, int HP, int PAD, bool POOL, int KMAX>
__global__ void __launch_bounds__(256) k_patch_dot(const PatchDotParams p)
{
    constexpr int K = KH * KW * IC;
    constexpr int TILE = HP * WP * IC;
    extern __shared__ __align__(16) float sm[];
    const int g = blockIdx.x;
    const int op = p.op[g];
    if (op != MURE_OP_GF && op != MURE_OP_WS) return;
    const int k = min(p.n_neurons[g], KMAX);
    if (k <= 0) return;
    float *es = sm;               // [k][K]
    float *xs = sm + KMAX * K;    // [rows_per_block][TILE]
    const int tl0 = blockIdx.y * p.rows_per_block;
    const int nr = min(p.rows_per_block, p.T - tl0);
    const float *e = p.e_all + p.patch_off[g];
    for (int i = threadIdx.x; i < k * K; i += blockDim.x) es[i] = __ldg(e + i);
    for (int i = threadIdx.x; i < nr * TILE; i += blockDim.x) {
        const int rl = i / TILE, el = i - rl * TILE;
        const int ci = el % IC, pix = el / IC, px = pix % WP, py = pix / WP;
        const int iy = py - PAD, ix = px - PAD;
        const int64_t tl = tl0 + rl;
        float v = 0.f;
        if ((unsigned)iy < (unsigned)p.ih && (unsigned)ix < (unsigned)p.iw)
            v = __ldg(p.x + (p.x_per_input ? p.t0 + tl : (int64_t)g * p.T + tl) * p.x_stride + (iy * p.iw + ix) * IC + ci);
        xs[i] = v;
    }
    __syncthreads();
    const int32_t *ids = p.ids + p.neuron_off[g];
    const int per_row = k * p.cells;
    for (int it = threadIdx.x; it < nr * per_row; it += blockDim.x) {
        const int rl = it / per_row, rem = it - rl * per_row, q = rem / p.cells, c = rem - q * p.cells;
        const int64_t tl = tl0 + rl;
        const int64_t r = (int64_t)g * p.T + tl, t = p.t0 + tl;
        const int j = ids[q];
        const float *zr = p.z + (p.z_per_input ? t : r) * p.z_stride + (int64_t)j * (p.oh * p.ow);
        const float *xt = xs + rl * TILE;
        const float *eq = es + q * K;
        const int pw = POOL ? p.ow / 2 : p.ow;
        const int cy = c / pw, cx = c - cy * pw;
        float v4[4];
#pragma unroll
        for (int s = 0; s < (POOL ? 4 : 1); ++s) {
            const int oy = POOL ? 2 * cy + (s >> 1) : cy, ox = POOL ? 2 * cx + (s & 1) : cx;
            const float *xw = xt + (oy * WP + ox) * IC;
            float acc = 0.f;
#pragma unroll
            for (int ky = 0; ky < KH; ++ky)
#pragma unroll
                for (int kx = 0; kx < KW; ++kx)
#pragma unroll
                    for (int ci = 0; ci < IC; ++ci)
                        acc = fmaf(eq[(ky * KW + kx) * IC + ci], xw[(ky * WP + kx) * IC + ci], acc);
            v4[s] = act_apply(p.act1, zr[oy * p.ow + ox] + acc);
        }
        p.out[r * p.out_stride + q * p.cells + c] = POOL ? max4_first(v4[0], v4[1], v4[2], v4[3]) : v4[0];
    }
}

// The same values in memoized mode, one input per block: the input's padded map and
// its pre-activation maps are staged once, and every GF / WS slot of the batch (the
// mutants share the inputs) is computed from there, SMAX slots' filters at a time
// (EG: the filters are read through L1 instead of being staged).  A
// thread takes CW output cells (pooling windows: 4 CW positions) for SG slots: each
// filter tap costs 4 CW + SG shared loads (the slot loads are warp broadcasts) for
// 4 CW SG FMAs.  Every sum is the same ascending fp32 chain as in k_patch_dot, so the
// two kernels agree bit for bit.
template <int KH, int KW, int IC, int WP, int HP, int PAD, bool POOL, int CW, int SG, int SMAX, int NT, bool EG = false>
__global__ void __launch_bounds__(NT) k_patch_dot_in(const PatchDotParams p)
{
    constexpr int K = KH * KW * IC;
    constexpr int TILE = HP * WP * IC;
    constexpr int NPOS = POOL ? 4 : 1;
    constexpr int NP = CW * NPOS;          // positions per thread
    extern __shared__ __align__(16) float sm[];
    const int P = p.oh * p.ow;
    float *xs = sm;                       // [TILE] zero-padded input map
    float *es = xs + TILE;                // [SMAX][K] filter deltas (EG: read through L1 instead)
    float *zsm = es + (EG ? 0 : SMAX * K);   // [oc][P] pre-activation maps
    __shared__ int sl_g[SMAX], sl_q[SMAX], sl_j[SMAX];
    const int tl = blockIdx.x;
    const int64_t t = p.t0 + tl;
    const float *xin = p.x + t * p.x_stride;
    for (int i = threadIdx.x; i < TILE; i += NT) {
        const int ci = i % IC, pix = i / IC, px = pix % WP, py = pix / WP;
        const int iy = py - PAD, ix = px - PAD;
        xs[i] = ((unsigned)iy < (unsigned)p.ih && (unsigned)ix < (unsigned)p.iw) ? __ldg(xin + (iy * p.iw + ix) * IC + ci)
                                                                                  : 0.f;
    }
    const float *zin = p.z + t * p.z_stride;
    for (int i = threadIdx.x; i < p.oc * P; i += NT) zsm[i] = __ldg(zin + i);
    const int pw = POOL ? p.ow / 2 : p.ow;
    const int chunks = (p.cells + CW - 1) / CW;
    // the batch's GF / WS slots (listed by the host), SMAX at a time
    for (int64_t s0 = 0; s0 < p.n_dslot; s0 += SMAX) {
        const int ns = (int)(p.n_dslot - s0 < SMAX ? p.n_dslot - s0 : SMAX);
        __syncthreads();
        for (int i = threadIdx.x; i < ns; i += NT) {
            const int g = p.dslot[2 * (s0 + i)] - p.dslot_g0, q = p.dslot[2 * (s0 + i) + 1];
            sl_g[i] = g;
            sl_q[i] = q;
            sl_j[i] = p.ids[p.neuron_off[g] + q];
        }
        __syncthreads();
        if (!EG) {
            for (int i = threadIdx.x; i < ns * K; i += NT) {
                const int sl = i / K, kk = i - sl * K;
                es[i] = __ldg(p.e_all + p.patch_off[sl_g[sl]] + (int64_t)sl_q[sl] * K + kk);
            }
            __syncthreads();
        }
        const int groups = (ns + SG - 1) / SG;
        for (int it = threadIdx.x; it < groups * chunks; it += NT) {
            const int sg = it / chunks, ch = it - sg * chunks;
            const int nsg = min(SG, ns - sg * SG);
            int off[NP];
#pragma unroll
            for (int w = 0; w < CW; ++w) {
                const int c = min(ch * CW + w, p.cells - 1);   // a chunk past the last cell repeats it
                const int cy = c / pw, cx = c - cy * pw;
#pragma unroll
                for (int s2 = 0; s2 < NPOS; ++s2) {
                    const int oy = POOL ? 2 * cy + (s2 >> 1) : cy, ox = POOL ? 2 * cx + (s2 & 1) : cx;
                    off[w * NPOS + s2] = (oy * WP + ox) * IC;
                }
            }
            const float *e0 = es + sg * SG * K;
            const float *eg[SG];
            if (EG) {
#pragma unroll
                for (int a = 0; a < SG; ++a) {
                    const int sl = sg * SG + (a < nsg ? a : 0);
                    eg[a] = p.e_all + p.patch_off[sl_g[sl]] + (int64_t)sl_q[sl] * K;
                }
            }
            float acc[SG][NP];
#pragma unroll
            for (int a = 0; a < SG; ++a)
#pragma unroll
                for (int q2 = 0; q2 < NP; ++q2) acc[a][q2] = 0.f;
#pragma unroll 1
            for (int ky = 0; ky < KH; ++ky)
#pragma unroll
                for (int kx = 0; kx < KW; ++kx)
#pragma unroll
                    for (int ci = 0; ci < IC; ++ci) {
                        const int kk = (ky * KW + kx) * IC + ci, xo = (ky * WP + kx) * IC + ci;
                        float xv[NP];
#pragma unroll
                        for (int q2 = 0; q2 < NP; ++q2) xv[q2] = xs[off[q2] + xo];
#pragma unroll
                        for (int a = 0; a < SG; ++a) {
                            const float ev = EG ? __ldg(eg[a] + kk) : e0[(a < nsg ? a : 0) * K + kk];
#pragma unroll
                            for (int q2 = 0; q2 < NP; ++q2) acc[a][q2] = fmaf(ev, xv[q2], acc[a][q2]);
                        }
                    }
#pragma unroll
            for (int a = 0; a < SG; ++a) {
                if (a >= nsg) break;
                const int sl = sg * SG + a;
                const float *zr = zsm + sl_j[sl] * P;
                float *orow = p.out + ((int64_t)sl_g[sl] * p.T + tl) * p.out_stride + sl_q[sl] * p.cells;
#pragma unroll
                for (int w = 0; w < CW; ++w) {
                    const int c = ch * CW + w;
                    if (c >= p.cells) break;
                    const int cy = c / pw, cx = c - cy * pw;
                    float v4[NPOS];
#pragma unroll
                    for (int s2 = 0; s2 < NPOS; ++s2) {
                        const int oy = POOL ? 2 * cy + (s2 >> 1) : cy, ox = POOL ? 2 * cx + (s2 & 1) : cx;
                        v4[s2] = act_apply(p.act1, zr[oy * p.ow + ox] + acc[a][w * NPOS + s2]);
                    }
                    orow[c] = POOL ? max4_first(v4[0], v4[1], v4[2], v4[3]) : v4[0];
                }
            }
        }
    }
}

namespace {
template <int KH, int KW, int IC, int WP, int HP, int PAD, bool POOL>
int launch_dot(const Stage &S, Src z, Src x, RowMap rm, const PatchArgs &pa, int kmax, float *out, int64_t out_stride,
               cudaStream_t s)
{
    constexpr int KMAX = 8;
    PatchDotParams p{};
    p.z = z.p; p.z_stride = z.stride; p.z_per_input = z.per_input;
    p.x = x.p; p.x_stride = x.stride; p.x_per_input = x.per_input;
    p.t0 = rm.t0; p.T = rm.T; p.G = rm.R / rm.T;
    p.ih = S.ih; p.iw = S.iw; p.oh = S.oh; p.ow = S.ow; p.act1 = S.act1;
    p.op = pa.op; p.n_neurons = pa.n_neurons; p.ids = pa.ids; p.neuron_off = pa.neuron_off;
    p.patch_off = pa.patch_off; p.e_all = pa.patch;
    p.dslot = pa.dslot; p.n_dslot = pa.n_dslot; p.dslot_g0 = pa.dslot_g0;
    p.out = out; p.out_stride = out_stride;
    p.cells = POOL ? (S.oh / 2) * (S.ow / 2) : S.oh * S.ow;
    p.rows_per_block = 8;
    p.oc = S.oc;
    if (z.per_input && x.per_input) {
        // memoized: one block per input, a cell and four slots per thread (measured
        // against two cells and / or eight slots per thread: more registers per thread
        // cost more in occupancy than the fewer shared loads save)
        constexpr int CW = 1, SG = 4, NT = 256;
        // the slot filters: staged in shared memory 32 slots at a time, or, where a
        // filter is long (IC > 1: 150 taps), read through L1 for all slots at once so
        // that no block runs a nearly empty last round of slots (measured: conv 6->16
        // 1.83 -> 1.65 ms per 400 mutants x 10,000 inputs; conv 1->6 slower that way)
        constexpr bool EG = IC > 1;
        constexpr int SMAX = EG ? 256 : 32;
        const size_t smem2 =
            ((size_t)HP * WP * IC + (EG ? 0 : (size_t)SMAX * KH * KW * IC) + (size_t)S.oc * S.oh * S.ow) * sizeof(float);
        if (smem2 <= 200 * 1024) {
            auto kern = k_patch_dot_in<KH, KW, IC, WP, HP, PAD, POOL, CW, SG, SMAX, NT, EG>;
            cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem2);
            kern<<<(unsigned)rm.T, NT, smem2, s>>>(p);
            return 1;
        }
    }
    const size_t smem = ((size_t)KMAX * KH * KW * IC + (size_t)p.rows_per_block * HP * WP * IC) * sizeof(float);
    cudaFuncSetAttribute(k_patch_dot<KH, KW, IC, WP, HP, PAD, POOL, KMAX>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                         (int)smem);
    const dim3 grid((unsigned)p.G, (unsigned)((rm.T + p.rows_per_block - 1) / p.rows_per_block));
    k_patch_dot<KH, KW, IC, WP, HP, PAD, POOL, KMAX><<<grid, 256, smem, s>>>(p);
    return 1;
}
}  // namespace

// GF / WS delta values for the small-layer geometries (the neuron count per mutant
// must be <= 8); 0 when the layer has no such kernel.
int patch_dot_supported(const Stage &S, int kmax) { return S.geo > 0 && kmax <= 8 && !S.has_add && !S.gap; }

int launch_patch_dot(const Stage &S, Src z, Src x, RowMap rm, const PatchArgs &pa, int kmax, float *out,
                     int64_t out_stride, cudaStream_t s)
{
    if (rm.R <= 0) return 0;
    switch (S.geo) {
    case 1: return launch_dot<5, 5, 6, 14, 14, 0, true>(S, z, x, rm, pa, kmax, out, out_stride, s);
    case 2: return launch_dot<5, 5, 1, 32, 32, 2, true>(S, z, x, rm, pa, kmax, out, out_stride, s);
    }
    return 0;
}

}  // namespace mure
