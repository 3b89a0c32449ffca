// Layer kernels of the FP32 arithmetic: implicit-GEMM convolution / dense on the
// CUDA cores, the output layer with the fused argmax / compare / kill epilogue, and
// small row-movement kernels.
//
// Determinism contract (what makes memoized == vanilla bit for bit): every output
// element z[row][pos][n] is the fp32 FMA chain acc = fma(x_k, w_k, acc) over the
// fan-in k = (ky, kx, ci) in ascending order starting from +0 (zero-padding taps
// contribute x = 0), then z = acc + b[n].  Nothing depends on the batch size, the
// tile a row lands in or the number of mutants, so one row gives the same bits in
// the cache build, in a vanilla prefix and in a memoized suffix.
#include "common.cuh"
#include "device_util.cuh"
#include "epilogue.cuh"

namespace mure {

struct StageParams {
    const float *x; int64_t x_stride; int x_per_input;
    int64_t t0; int T; int R;
    const int32_t *lrow;   // compacted batch: logical rows (per-input reads), else null
    int ih, iw, ic, kh, kw, stride, pad, oh, ow, oc, K;
    const float *Wt;  // [K][oc]
    const float *b;
    int act1, has_add, act2, pool;
    const float *skip; int64_t skip_stride; int skip_per_input; int sk_w, sk_c, sk_stride;
    float *z; int64_t z_stride;
    float *y; int64_t y_stride;
    int P;   // GEMM rows per batch row: oh*ow, ordered (oy, ox), or with pooling
             // 4 * (oh/2) * (ow/2) ordered (py, px, dy, dx)
    int pw;  // pooled width
};

template <int BN>
__global__ void __launch_bounds__(256) k_stage_simt(const StageParams p)
{
    constexpr int BM = 4096 / BN, BK = 16;
    constexpr int A_SPLIT = 256 / BM, A_PER = BK / A_SPLIT;
    constexpr int B_SPLIT = 256 / BN, B_PER = BK / B_SPLIT;
    __shared__ __align__(16) float As[BK][BM];
    __shared__ __align__(16) float Bs[BK][BN];

    const int tid = threadIdx.x;
    const int tn = tid % (BN / 4), tm = tid / (BN / 4);
    const int64_t M = (int64_t)p.R * p.P;
    const int64_t m0 = (int64_t)blockIdx.x * BM;
    const int n0 = blockIdx.y * BN;

    // this thread's A-load row
    const int m_l = tid % BM, kl0 = (tid / BM) * A_PER;
    const int64_t m = m0 + m_l;
    const bool valid_m = m < M;
    int iy0 = 0, ix0 = 0;
    const float *xrow = p.x;
    if (valid_m) {
        const int64_t row = m / p.P;
        const int q = (int)(m % p.P);
        int oy, ox;
        if (p.pool) {
            const int w = q >> 2, sub = q & 3;
            oy = 2 * (w / p.pw) + (sub >> 1);
            ox = 2 * (w % p.pw) + (sub & 1);
        } else {
            oy = q / p.ow;
            ox = q % p.ow;
        }
        iy0 = oy * p.stride - p.pad;
        ix0 = ox * p.stride - p.pad;
        xrow = p.x + (p.x_per_input ? (p.t0 + logical_row(p.lrow, row) % p.T) : row) * p.x_stride;
    }
    const int n_l = tid % BN, kb0 = (tid / BN) * B_PER;

    float acc[4][4];
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = 0.f;

    for (int k0 = 0; k0 < p.K; k0 += BK) {
        {
            int k = k0 + kl0;
            int ci = k % p.ic, t = k / p.ic, kx = t % p.kw, ky = t / p.kw;
#pragma unroll
            for (int i = 0; i < A_PER; ++i) {
                float v = 0.f;
                if (valid_m && k + i < p.K) {
                    const int iy = iy0 + ky, ix = ix0 + kx;
                    if ((unsigned)iy < (unsigned)p.ih && (unsigned)ix < (unsigned)p.iw)
                        v = __ldg(xrow + ((int64_t)iy * p.iw + ix) * p.ic + ci);
                }
                As[kl0 + i][m_l] = v;
                if (++ci == p.ic) { ci = 0; if (++kx == p.kw) { kx = 0; ++ky; } }
            }
        }
#pragma unroll
        for (int i = 0; i < B_PER; ++i) {
            const int k = k0 + kb0 + i, n = n0 + n_l;
            Bs[kb0 + i][n_l] = (k < p.K && n < p.oc) ? __ldg(p.Wt + (int64_t)k * p.oc + n) : 0.f;
        }
        __syncthreads();
#pragma unroll
        for (int kk = 0; kk < BK; ++kk) {
            const float4 a = *reinterpret_cast<const float4 *>(&As[kk][tm * 4]);
            const float4 b = *reinterpret_cast<const float4 *>(&Bs[kk][tn * 4]);
            const float av[4] = {a.x, a.y, a.z, a.w}, bv[4] = {b.x, b.y, b.z, b.w};
#pragma unroll
            for (int i = 0; i < 4; ++i)
#pragma unroll
                for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(av[i], bv[j], acc[i][j]);
        }
        __syncthreads();
    }

    // epilogue: bias, activation, skip, pooling
    const int64_t mb = m0 + tm * 4;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        const int n = n0 + tn * 4 + j;
        if (n >= p.oc) continue;
        const float bias = __ldg(p.b + n);
        float win[4];
        int64_t row = 0;
        int py = 0, px = 0;
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const int64_t mm = mb + i;
            win[i] = 0.f;
            if (mm >= M) continue;
            row = mm / p.P;
            const int q = (int)(mm % p.P);
            int oy, ox;
            if (p.pool) {
                const int w = q >> 2, sub = q & 3;
                py = w / p.pw; px = w % p.pw;
                oy = 2 * py + (sub >> 1);
                ox = 2 * px + (sub & 1);
            } else {
                oy = q / p.ow;
                ox = q % p.ow;
            }
            const float z = acc[i][j] + bias;
            if (p.z) p.z[row * p.z_stride + (int64_t)n * (p.oh * p.ow) + oy * p.ow + ox] = z;  // channel-major
            float v = act_apply(p.act1, z);
            if (p.has_add) {
                const float *sr =
                    p.skip + (p.skip_per_input ? (p.t0 + logical_row(p.lrow, row) % p.T) : row) * p.skip_stride;
                const float s = n < p.sk_c ? sr[((int64_t)oy * p.sk_stride * p.sk_w + ox * p.sk_stride) * p.sk_c + n] : 0.f;
                v = act_apply(p.act2, v + s);
            }
            if (p.pool) win[i] = v;
            else p.y[row * p.y_stride + ((int64_t)oy * p.ow + ox) * p.oc + n] = v;
        }
        if (p.pool && mb < M)
            p.y[row * p.y_stride + ((int64_t)py * p.pw + px) * p.oc + n] = max4_first(win[0], win[1], win[2], win[3]);
    }
}

// Global average pooling: y[r][c] = (sum over positions, ascending, in fp32) / P.
__global__ void k_gap(const float *__restrict__ in, int64_t in_stride, int P, int C, int R, float *__restrict__ y,
                      int64_t y_stride)
{
    const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= (int64_t)R * C) return;
    const int64_t r = i / C;
    const int c = (int)(i % C);
    y[r * y_stride + c] = gap_sum(in + r * in_stride, P, C, c);
}

// Depthwise convolution stage (MobileNetV2): output channel c at (oy, ox) is the fp32
// FMA chain over its filter taps (ky, kx ascending, from +0) on input channel c, then
// + b; the pre-activation goes to z (channel-major) when requested, act1 to y.  One
// thread per (row, position, channel): consecutive threads read and write
// consecutive channels, and the weights are read as Wt [tap][c].
__global__ void __launch_bounds__(256) k_dwconv(const StageParams p)
{
    const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const int64_t per_row = (int64_t)p.oh * p.ow * p.oc;
    if (i >= (int64_t)p.R * per_row) return;
    const int64_t row = i / per_row;
    const int rem = (int)(i - row * per_row);
    const int c = rem % p.oc, pos = rem / p.oc, oy = pos / p.ow, ox = pos - (pos / p.ow) * p.ow;
    const float *xrow = p.x + (p.x_per_input ? p.t0 + logical_row(p.lrow, row) % p.T : row) * p.x_stride;
    float acc = 0.f;
    for (int ky = 0; ky < p.kh; ++ky) {
        const int iy = oy * p.stride - p.pad + ky;
        for (int kx = 0; kx < p.kw; ++kx) {
            const int ix = ox * p.stride - p.pad + kx;
            if ((unsigned)iy < (unsigned)p.ih && (unsigned)ix < (unsigned)p.iw)
                acc = fmaf(__ldg(p.Wt + (int64_t)(ky * p.kw + kx) * p.oc + c),
                           __ldg(xrow + ((int64_t)iy * p.iw + ix) * p.ic + c), acc);
        }
    }
    const float z = acc + __ldg(p.b + c);
    if (p.z) p.z[row * p.z_stride + (int64_t)c * (p.oh * p.ow) + pos] = z;
    p.y[row * p.y_stride + (int64_t)pos * p.oc + c] = act_apply(p.act1, z);
}

int launch_stage_simt(const Stage &S, Src x, RowMap rm, float *z_out, int64_t z_stride, Src skip, float *y_out,
                      int64_t y_stride, float *gap_tmp, cudaStream_t s)
{
    if (rm.R <= 0) return 0;
    if (S.tc) return launch_tc(S, x, rm, z_out, z_stride, skip, y_out, y_stride, gap_tmp, s);
    if (S.kind == MURE_NODE_EMBED) return launch_embed(S, x, rm, z_out, z_stride, y_out, y_stride, s);
    if (S.kind == MURE_NODE_LSTM) return launch_lstm(S, x, rm, z_out, z_stride, y_out, y_stride, nullptr, s);
    if (S.kind == MURE_NODE_DWCONV) {
        StageParams p{};
        p.x = x.p; p.x_stride = x.stride; p.x_per_input = x.per_input;
        p.t0 = rm.t0; p.T = rm.T; p.R = rm.R; p.lrow = rm.lrow;
        p.ih = S.ih; p.iw = S.iw; p.ic = S.ic; p.kh = S.kh; p.kw = S.kw; p.stride = S.stride; p.pad = S.pad;
        p.oh = S.oh; p.ow = S.ow; p.oc = S.oc; p.K = S.K;
        p.Wt = S.Wt; p.b = S.b; p.act1 = S.act1;
        p.z = z_out; p.z_stride = z_stride;
        p.y = y_out; p.y_stride = y_stride;
        const int64_t n = (int64_t)rm.R * S.oh * S.ow * S.oc;
        k_dwconv<<<(unsigned)((n + 255) / 256), 256, 0, s>>>(p);
        return 1;
    }
    if (S.variant > 0) return launch_conv_small(S, x, rm, z_out, z_stride, y_out, y_stride, s);
    StageParams p{};
    p.x = x.p; p.x_stride = x.stride; p.x_per_input = x.per_input;
    p.t0 = rm.t0; p.T = rm.T; p.R = rm.R; p.lrow = rm.lrow;
    p.ih = S.ih; p.iw = S.iw; p.ic = S.ic; p.kh = S.kh; p.kw = S.kw; p.stride = S.stride; p.pad = S.pad;
    p.oh = S.oh; p.ow = S.ow; p.oc = S.oc; p.K = S.K;
    p.Wt = S.Wt; p.b = S.b;
    p.act1 = S.act1; p.has_add = S.has_add; p.act2 = S.act2; p.pool = S.pool;
    p.skip = skip.p; p.skip_stride = skip.stride; p.skip_per_input = skip.per_input;
    p.sk_w = S.sk_w; p.sk_c = S.sc_c; p.sk_stride = S.sc_stride;
    p.z = z_out; p.z_stride = z_stride;
    // with global average pooling the post-op map goes to gap_tmp first
    const int mh = S.pool ? S.oh / 2 : S.oh, mw = S.pool ? S.ow / 2 : S.ow;
    const int64_t map_stride = round4((int64_t)mh * mw * S.oc);
    p.y = S.gap ? gap_tmp : y_out;
    p.y_stride = S.gap ? map_stride : y_stride;
    p.pw = S.ow / 2;
    p.P = S.pool ? 4 * (S.oh / 2) * (S.ow / 2) : S.oh * S.ow;
    const int64_t M = (int64_t)rm.R * p.P;
    int launches = 1;
    if (S.oc <= 16) {
        dim3 g((unsigned)((M + 255) / 256), (unsigned)((S.oc + 15) / 16));
        k_stage_simt<16><<<g, 256, 0, s>>>(p);
    } else if (S.oc <= 32) {
        dim3 g((unsigned)((M + 127) / 128), (unsigned)((S.oc + 31) / 32));
        k_stage_simt<32><<<g, 256, 0, s>>>(p);
    } else {
        dim3 g((unsigned)((M + 63) / 64), (unsigned)((S.oc + 63) / 64));
        k_stage_simt<64><<<g, 256, 0, s>>>(p);
    }
    if (S.gap) {
        const int64_t n = (int64_t)rm.R * S.oc;
        k_gap<<<(unsigned)((n + 255) / 256), 256, 0, s>>>(gap_tmp, map_stride, mh * mw, S.oc, rm.R, y_out, y_stride);
        ++launches;
    }
    return launches;
}

// ------------------------------------------------------ output layer + epilogue --

struct FinalParams {
    const float *x; int64_t x_stride; int x_per_input;
    int64_t t0; int T; int R;
    const int32_t *lrow;   // compacted batch: logical rows (per-input reads, overlay), else null
    int F, C, act;
    const float *W;  // [C][F]
    const float *Wt; // [F][C] (the same weights, input-major)
    const float *b;
    FinalArgs fa;
    Overlay ov;      // mutated channels of the input rows (ov.patch null: none)
};

// Kill bits of one warp of rows (32 consecutive inputs of one mutant) and the
// near-tie count.  v = the row's logits.
__device__ __forceinline__ void epilogue_row(const FinalArgs &fa, int64_t t0, int T, int64_t row, bool in_range,
                                             const float *v, int C)
{
    const int64_t lr = in_range ? logical_row(fa.lrow, row) : row;
    const int g = (int)(lr / T);
    const int64_t t = t0 + lr % T;
    const bool valid = in_range && t < fa.n_in;
    int arg = 0;
    bool near = false;
    if (valid) {
        arg = argmax_first(v, C);
        near = near_tie(v, C, arg);
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
        for (int c = 0; c < C; ++c) o[c] = v[c];
    }
}

// CP: the class count rounded up to a multiple of 4 (the accumulators kept per row).
template <int CP>
__global__ void __launch_bounds__(128) k_final_dense(const FinalParams p)
{
    constexpr int RB = 128, FC = 32;
    __shared__ float xs[RB][FC + 1];
    __shared__ __align__(16) float ws[FC][CP];
    const int tid = threadIdx.x;
    const int64_t row0 = (int64_t)blockIdx.x * RB;
    const int64_t row = row0 + tid;
    const bool in_range = row < p.R;
    // this row's mutated input channels (overlay), as (slot count, id pointer)
    int ov_k = 0;
    const int32_t *ov_ids = nullptr;
    const int64_t lrow = in_range ? logical_row(p.lrow, row) : row;
    if (p.ov.patch && in_range) {
        const int g = (int)(lrow / p.T);
        ov_k = p.ov.n_neurons[g];
        ov_ids = p.ov.ids + p.ov.neuron_off[g];
    }
    __shared__ const float *xrow_of[RB];
    float acc[CP];
#pragma unroll
    for (int c = 0; c < CP; ++c) acc[c] = 0.f;
    {
        const int64_t r = row0 + tid;
        xrow_of[tid] = r < p.R ? p.x + (p.x_per_input ? (p.t0 + logical_row(p.lrow, r) % p.T) : r) * p.x_stride
                               : nullptr;
    }
    __syncthreads();
    for (int f0 = 0; f0 < p.F; f0 += FC) {
#pragma unroll 8
        for (int i = tid; i < RB * FC; i += RB) {
            const int rl = i / FC, fl = i % FC;
            const float *xr = xrow_of[rl];
            xs[rl][fl] = (xr && f0 + fl < p.F) ? __ldg(xr + f0 + fl) : 0.f;
        }
        for (int i = tid; i < FC * CP; i += RB) {
            const int fl = i / CP, c = i % CP;
            ws[fl][c] = (c < p.C && f0 + fl < p.F) ? __ldg(p.W + (int64_t)c * p.F + f0 + fl) : 0.f;
        }
        __syncthreads();
        const int fe = min(FC, p.F - f0);
        // overlay on this thread's own row (no other thread reads it)
        for (int q = 0; q < ov_k; ++q) {
            const int j = ov_ids[q];
            const int cfirst = f0 - j <= 0 ? 0 : (f0 - j + p.ov.ch - 1) / p.ov.ch;
            for (int c = cfirst; c < p.ov.cells && c * p.ov.ch + j < f0 + fe; ++c)
                xs[tid][c * p.ov.ch + j - f0] = p.ov.patch[lrow * p.ov.row_stride + q * p.ov.cells + c];
        }
        for (int fl = 0; fl < fe; ++fl) {
            const float xv = xs[tid][fl];
#pragma unroll
            for (int c4 = 0; c4 < CP; c4 += 4) {
                const float4 w4 = *reinterpret_cast<const float4 *>(&ws[fl][c4]);
                acc[c4] = fmaf(xv, w4.x, acc[c4]);
                acc[c4 + 1] = fmaf(xv, w4.y, acc[c4 + 1]);
                acc[c4 + 2] = fmaf(xv, w4.z, acc[c4 + 2]);
                acc[c4 + 3] = fmaf(xv, w4.w, acc[c4 + 3]);
            }
        }
        __syncthreads();
    }
    float v[CP];
#pragma unroll
    for (int c = 0; c < CP; ++c) {
        const float z = c < p.C ? acc[c] + __ldg(p.b + c) : 0.f;
        if (in_range && c < p.C && p.fa.z_out) p.fa.z_out[row * p.fa.z_stride + c] = z;
        v[c] = act_apply(p.act, z);
    }
    if (p.fa.mode == 1) {  // cache build: logits rows and original predictions
        if (in_range) {
#pragma unroll
            for (int c = 0; c < CP; ++c)
                if (c < p.C) p.fa.x_out[row * p.fa.x_stride + c] = v[c];
            p.fa.pred_out[row] = argmax_reg<CP>(v, p.C);
        }
        return;
    }
    if (p.fa.mode == 2) {  // per-row logits for a following delta + epilogue
        if (in_range) {
#pragma unroll
            for (int c = 0; c < CP; ++c)
                if (c < p.C) p.fa.logits_rows[row * p.fa.x_stride + c] = v[c];
        }
        return;
    }
    epilogue_reg<CP>(p.fa, p.t0, p.T, row, in_range, v, p.C);
}

// The same output layer with each warp on its own 32 rows (lane = row) and no block-wide
// barrier after the weights are staged: the warp copies its rows' next 32 inputs (16-byte
// loads, eight per lane) while it runs the FMAs of the current 32, through a per-warp
// shared-memory tile.  Each row's sums are the same fp32 chain as k_final_dense's (f
// ascending from +0, fmaf(x, w, acc), then + b), so both kernels give the same bits.
// (One launch of k_final_dense on 6,144 rows of 512 inputs waited 256 us on its loads.)
// Needs F a multiple of 4 and 16-byte aligned rows; the weights [F][CP] in dynamic shared
// memory.
template <int CP>
__global__ void __launch_bounds__(128) k_final_dense_w(const FinalParams p)
{
    extern __shared__ __align__(16) float wsm[];   // [F][CP]
    __shared__ float xs[4][32][33];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    for (int i = threadIdx.x; i < p.F * CP; i += blockDim.x) {
        const int f = i / CP, c = i - f * CP;
        wsm[i] = c < p.C ? __ldg(p.W + (int64_t)c * p.F + f) : 0.f;
    }
    __syncthreads();
    const int64_t row0 = (int64_t)blockIdx.x * 128 + warp * 32;
    const int64_t row = row0 + lane;
    const bool in_range = row < p.R;
    int ov_k = 0;
    const int32_t *ov_ids = nullptr;
    const int64_t lrow = in_range ? logical_row(p.lrow, row) : row;
    if (p.ov.patch && in_range) {
        const int g = (int)(lrow / p.T);
        ov_k = p.ov.n_neurons[g];
        ov_ids = p.ov.ids + p.ov.neuron_off[g];
    }
    // this lane copies 16 bytes (inputs 4 (lane mod 8) .. +3) of rows 4i + lane / 8
    const int fq = 4 * (lane & 7);
    const float *src[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) {
        const int64_t r = row0 + 4 * i + (lane >> 3);
        src[i] = r < p.R ? p.x + (p.x_per_input ? (p.t0 + logical_row(p.lrow, r) % p.T) : r) * p.x_stride : nullptr;
    }
    auto load = [&](int f0, float4 (&v)[8]) {
#pragma unroll
        for (int i = 0; i < 8; ++i)
            v[i] = (src[i] && f0 + fq < p.F) ? __ldg(reinterpret_cast<const float4 *>(src[i] + f0 + fq))
                                             : make_float4(0.f, 0.f, 0.f, 0.f);
    };
    float acc[CP];
#pragma unroll
    for (int c = 0; c < CP; ++c) acc[c] = 0.f;
    float4 cur[8];
    load(0, cur);
    for (int f0 = 0; f0 < p.F; f0 += 32) {
        __syncwarp();
#pragma unroll
        for (int i = 0; i < 8; ++i) {
            float *d = &xs[warp][4 * i + (lane >> 3)][fq];
            d[0] = cur[i].x; d[1] = cur[i].y; d[2] = cur[i].z; d[3] = cur[i].w;
        }
        if (f0 + 32 < p.F) load(f0 + 32, cur);
        __syncwarp();
        const int fe = min(32, p.F - f0);
        // overlay on this lane's own row (no other lane reads it)
        for (int q = 0; q < ov_k; ++q) {
            const int j = ov_ids[q];
            const int cfirst = f0 - j <= 0 ? 0 : (f0 - j + p.ov.ch - 1) / p.ov.ch;
            for (int c = cfirst; c < p.ov.cells && c * p.ov.ch + j < f0 + fe; ++c)
                xs[warp][lane][c * p.ov.ch + j - f0] = p.ov.patch[lrow * p.ov.row_stride + q * p.ov.cells + c];
        }
        for (int fl = 0; fl < fe; ++fl) {
            const float xv = xs[warp][lane][fl];
            const float *wr = wsm + (f0 + fl) * CP;
#pragma unroll
            for (int c4 = 0; c4 < CP; c4 += 4) {
                const float4 w4 = *reinterpret_cast<const float4 *>(wr + c4);
                acc[c4] = fmaf(xv, w4.x, acc[c4]);
                acc[c4 + 1] = fmaf(xv, w4.y, acc[c4 + 1]);
                acc[c4 + 2] = fmaf(xv, w4.z, acc[c4 + 2]);
                acc[c4 + 3] = fmaf(xv, w4.w, acc[c4 + 3]);
            }
        }
    }
    float v[CP];
#pragma unroll
    for (int c = 0; c < CP; ++c) {
        const float z = c < p.C ? acc[c] + __ldg(p.b + c) : 0.f;
        if (in_range && c < p.C && p.fa.z_out) p.fa.z_out[row * p.fa.z_stride + c] = z;
        v[c] = act_apply(p.act, z);
    }
    if (p.fa.mode == 1) {  // cache build: logits rows and original predictions
        if (in_range) {
#pragma unroll
            for (int c = 0; c < CP; ++c)
                if (c < p.C) p.fa.x_out[row * p.fa.x_stride + c] = v[c];
            p.fa.pred_out[row] = argmax_reg<CP>(v, p.C);
        }
        return;
    }
    if (p.fa.mode == 2) {  // per-row logits for a following delta + epilogue
        if (in_range) {
#pragma unroll
            for (int c = 0; c < CP; ++c)
                if (c < p.C) p.fa.logits_rows[row * p.fa.x_stride + c] = v[c];
        }
        return;
    }
    epilogue_reg<CP>(p.fa, p.t0, p.T, row, in_range, v, p.C);
}

// The output layer of 9 to 12 classes with a block's 32 rows shared by its four warps:
// warp w keeps classes w, w+4 and w+8 of every row (lane = row), so a warp's serial
// instruction stream is a quarter of k_final_dense_w's (which keeps all classes of its
// rows in one warp: ncu showed each of its blocks issue-bound at one warp per scheduler,
// about 32 us per block whatever the grid, a third of it spent on a strided weight
// fill).  A class's sum is the same fp32 chain as k_final_dense's (f ascending from +0,
// fmaf(x, w, acc), then + b), so the bits equal those of the other output-layer kernels.
// The weights come from the input-major copy Wt [F][C] with 16-byte loads all in flight;
// each warp copies the rows' next 32 inputs (16-byte loads) into its own tile of 36-float
// lines (16-byte stores and loads without bank conflicts) while it runs the FMAs of the
// current 32; the warps' sums meet in shared memory and warp 0 runs the epilogue.  Needs
// F a multiple of 4 and 16-byte aligned rows; dynamic shared memory [F][4][4] (class c at
// [f][c mod 4][c / 4]).
constexpr int kSplitLine = 36;

__global__ void __launch_bounds__(128) k_final_dense_split(const FinalParams p)
{
    extern __shared__ __align__(16) float wsm[];   // [F][4][4]
    __shared__ __align__(16) float xs[4][32][kSplitLine];
    __shared__ float sums[32][13];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    for (int i = threadIdx.x; i < p.F * 16; i += 128) wsm[i] = 0.f;
    const int64_t row0 = (int64_t)blockIdx.x * 32;
    const int64_t row = row0 + lane;
    const bool in_range = row < p.R;
    int ov_k = 0;
    const int32_t *ov_ids = nullptr;
    const int64_t lrow = in_range ? logical_row(p.lrow, row) : row;
    if (p.ov.patch && in_range) {
        const int g = (int)(lrow / p.T);
        ov_k = p.ov.n_neurons[g];
        ov_ids = p.ov.ids + p.ov.neuron_off[g];
    }
    // this lane copies 16 bytes (inputs 4 (lane mod 8) .. +3) of rows 4i + lane / 8
    const int fq = 4 * (lane & 7);
    const float *src[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) {
        const int64_t r = row0 + 4 * i + (lane >> 3);
        src[i] = r < p.R ? p.x + (p.x_per_input ? (p.t0 + logical_row(p.lrow, r) % p.T) : r) * p.x_stride : nullptr;
    }
    auto load = [&](int f0, float4 (&v)[8]) {
#pragma unroll
        for (int i = 0; i < 8; ++i)
            v[i] = (src[i] && f0 + fq < p.F) ? __ldg(reinterpret_cast<const float4 *>(src[i] + f0 + fq))
                                             : make_float4(0.f, 0.f, 0.f, 0.f);
    };
    float4 cur[8];
    load(0, cur);
    __syncthreads();   // padding zeroed before the weights are placed
    {
        const int n4 = p.F * p.C / 4;
        const float4 *w4p = reinterpret_cast<const float4 *>(p.Wt);
        for (int i0 = threadIdx.x; i0 < n4; i0 += 8 * 128) {
            float4 v[8];
#pragma unroll
            for (int u = 0; u < 8; ++u) {
                const int i = i0 + u * 128;
                v[u] = i < n4 ? __ldg(w4p + i) : make_float4(0.f, 0.f, 0.f, 0.f);
            }
#pragma unroll
            for (int u = 0; u < 8; ++u) {
                const int i = i0 + u * 128;
                if (i >= n4) continue;
                int f = 4 * i / p.C, c = 4 * i - f * p.C;
                const float e[4] = {v[u].x, v[u].y, v[u].z, v[u].w};
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                    wsm[f * 16 + (c & 3) * 4 + (c >> 2)] = e[k];
                    if (++c == p.C) { c = 0; ++f; }
                }
            }
        }
    }
    __syncthreads();   // the weights
    float a0 = 0.f, a1 = 0.f, a2 = 0.f;
    const float *wq = wsm + 4 * warp;
    const float *xr = &xs[warp][lane][0];
    for (int f0 = 0; f0 < p.F; f0 += 32) {
        __syncwarp();
#pragma unroll
        for (int i = 0; i < 8; ++i) *reinterpret_cast<float4 *>(&xs[warp][4 * i + (lane >> 3)][fq]) = cur[i];
        if (f0 + 32 < p.F) load(f0 + 32, cur);
        __syncwarp();
        const int fe = min(32, p.F - f0);
        // overlay on this lane's own row (no other lane reads it)
        for (int q = 0; q < ov_k; ++q) {
            const int j = ov_ids[q];
            const int cfirst = f0 - j <= 0 ? 0 : (f0 - j + p.ov.ch - 1) / p.ov.ch;
            for (int c = cfirst; c < p.ov.cells && c * p.ov.ch + j < f0 + fe; ++c)
                xs[warp][lane][c * p.ov.ch + j - f0] = p.ov.patch[lrow * p.ov.row_stride + q * p.ov.cells + c];
        }
        if (fe == 32) {
#pragma unroll
            for (int f4 = 0; f4 < 32; f4 += 4) {
                const float4 x4 = *reinterpret_cast<const float4 *>(xr + f4);
                const float xq[4] = {x4.x, x4.y, x4.z, x4.w};
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const float4 w4 = *reinterpret_cast<const float4 *>(wq + (f0 + f4 + e) * 16);
                    a0 = fmaf(xq[e], w4.x, a0);
                    a1 = fmaf(xq[e], w4.y, a1);
                    a2 = fmaf(xq[e], w4.z, a2);
                }
            }
        } else {
            for (int fl = 0; fl < fe; ++fl) {
                const float xv = xr[fl];
                const float4 w4 = *reinterpret_cast<const float4 *>(wq + (f0 + fl) * 16);
                a0 = fmaf(xv, w4.x, a0);
                a1 = fmaf(xv, w4.y, a1);
                a2 = fmaf(xv, w4.z, a2);
            }
        }
    }
    sums[lane][warp] = a0;
    sums[lane][warp + 4] = a1;
    sums[lane][warp + 8] = a2;
    __syncthreads();
    if (warp != 0) return;
    float v[12];
#pragma unroll
    for (int c = 0; c < 12; ++c) {
        const float z = c < p.C ? sums[lane][c] + __ldg(p.b + c) : 0.f;
        if (in_range && c < p.C && p.fa.z_out) p.fa.z_out[row * p.fa.z_stride + c] = z;
        v[c] = act_apply(p.act, z);
    }
    if (p.fa.mode == 1) {  // cache build: logits rows and original predictions
        if (in_range) {
#pragma unroll
            for (int c = 0; c < 12; ++c)
                if (c < p.C) p.fa.x_out[row * p.fa.x_stride + c] = v[c];
            p.fa.pred_out[row] = argmax_reg<12>(v, p.C);
        }
        return;
    }
    if (p.fa.mode == 2) {  // per-row logits for a following delta + epilogue
        if (in_range) {
#pragma unroll
            for (int c = 0; c < 12; ++c)
                if (c < p.C) p.fa.logits_rows[row * p.fa.x_stride + c] = v[c];
        }
        return;
    }
    epilogue_reg<12>(p.fa, p.t0, p.T, row, in_range, v, p.C);
}

__global__ void __launch_bounds__(128) k_epilogue(const float *__restrict__ lg, int64_t stride, int per_input, int C,
                                                  int64_t t0, int T, int R, const FinalArgs fa, const Overlay ov)
{
    const int64_t row = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const bool in_range = row < R;
    float v[kMaxClasses];
    const float *src = lg + (per_input ? t0 + row % T : row) * stride;
#pragma unroll
    for (int c = 0; c < kMaxClasses; ++c) v[c] = (in_range && c < C) ? src[c] : 0.f;
    if (ov.patch && in_range) {
        const int g = (int)(row / T);
        const int32_t *ids = ov.ids + ov.neuron_off[g];
        for (int q = 0; q < ov.n_neurons[g]; ++q) {
            const float val = ov.patch[row * ov.row_stride + q * ov.cells];
#pragma unroll
            for (int c = 0; c < kMaxClasses; ++c)
                if (c == ids[q]) v[c] = val;
        }
    }
    epilogue_row(fa, t0, T, row, in_range, v, C);
}

// The output layer for rows (per input or per row) with a dense overlay: each
// thread copies its own input row (16-byte loads, all in flight at once) into its own
// shared-memory row, writes the mutated channels there and runs the same fp32 chain as
// k_final_dense (f ascending, fmaf(x, w, acc)), so both kernels give the same bits.
// No block-wide barrier sits between the loads and the FMAs.
constexpr int kRowsF = 100;   // floats per staged row (F <= 96), a multiple of 4

template <int CP, int UF>
__global__ void __launch_bounds__(128) k_final_dense_rows(const FinalParams p)
{
    extern __shared__ __align__(16) float fsm[];
    float *ws = fsm;                              // [F][CP]
    float *xr = fsm + p.F * CP + threadIdx.x * kRowsF;
    const int tid = threadIdx.x;
    const int64_t row = (int64_t)blockIdx.x * 128 + tid;
    const bool in_range = row < p.R;
    for (int i = tid; i < p.F * CP; i += 128) {
        const int fl = i / CP, c = i % CP;
        ws[i] = c < p.C ? __ldg(p.W + (int64_t)c * p.F + fl) : 0.f;
    }
    if (in_range) {
        const int64_t lrow = logical_row(p.lrow, row);
        const float4 *src = reinterpret_cast<const float4 *>(p.x + (p.x_per_input ? p.t0 + lrow % p.T : row) * p.x_stride);
        float4 v[kRowsF / 4];
#pragma unroll
        for (int i = 0; i < kRowsF / 4; ++i)
            if (4 * i < p.F) v[i] = __ldg(src + i);
#pragma unroll
        for (int i = 0; i < kRowsF / 4; ++i)
            if (4 * i < p.F) *reinterpret_cast<float4 *>(xr + 4 * i) = v[i];
        if (p.ov.patch) {
            const int g = (int)(lrow / p.T);
            const int k = p.ov.n_neurons[g];
            const int32_t *ids = p.ov.ids + p.ov.neuron_off[g];
            for (int q = 0; q < k; ++q) xr[ids[q]] = p.ov.patch[lrow * p.ov.row_stride + q];
        }
    }
    __syncthreads();   // the weights
    float acc[CP];
#pragma unroll
    for (int c = 0; c < CP; ++c) acc[c] = 0.f;
    if (in_range) {
        // four inputs per 16-byte load (rows 400 bytes apart: no bank conflicts)
#pragma unroll UF
        for (int f4 = 0; f4 < p.F; f4 += 4) {
            const float4 x4 = *reinterpret_cast<const float4 *>(xr + f4);
            const float xq[4] = {x4.x, x4.y, x4.z, x4.w};
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const float xv = xq[e];
#pragma unroll
                for (int c4 = 0; c4 < CP; c4 += 4) {
                    const float4 w4 = *reinterpret_cast<const float4 *>(ws + (f4 + e) * CP + c4);
                    acc[c4] = fmaf(xv, w4.x, acc[c4]);
                    acc[c4 + 1] = fmaf(xv, w4.y, acc[c4 + 1]);
                    acc[c4 + 2] = fmaf(xv, w4.z, acc[c4 + 2]);
                    acc[c4 + 3] = fmaf(xv, w4.w, acc[c4 + 3]);
                }
            }
        }
    }
    float v[CP];
#pragma unroll
    for (int c = 0; c < CP; ++c) {
        const float z = c < p.C ? acc[c] + __ldg(p.b + c) : 0.f;
        v[c] = act_apply(p.act, z);
    }
    epilogue_reg<CP>(p.fa, p.t0, p.T, row, in_range, v, p.C);
}

int launch_gap(const float *in, int64_t in_stride, int P, int C, int R, float *y, int64_t y_stride, cudaStream_t s)
{
    const int64_t n = (int64_t)R * C;
    if (n <= 0) return 0;
    k_gap<<<(unsigned)((n + 255) / 256), 256, 0, s>>>(in, in_stride, P, C, R, y, y_stride);
    return 1;
}

int launch_final_dense(const Stage &S, Src x, RowMap rm, const FinalArgs &fa, cudaStream_t s, const Overlay *ov)
{
    if (rm.R <= 0) return 0;
    FinalParams p{};
    if (ov) p.ov = *ov;
    p.x = x.p; p.x_stride = x.stride; p.x_per_input = x.per_input;
    p.t0 = rm.t0; p.T = rm.T; p.R = rm.R; p.lrow = rm.lrow;
    p.F = S.K; p.C = S.oc; p.act = S.act1;
    p.W = S.W; p.Wt = S.Wt; p.b = S.b;
    p.fa = fa;
    const unsigned blocks = (unsigned)((rm.R + 127) / 128);
    const int cp = (p.C + 3) & ~3;
    // per-input rows with a small dense overlay, mutants' kill epilogue only: each
    // thread stages its own row (measured on the LeNet-5 workload, FC 84-10 of the FC
    // 120-84 mutants: 0.68 -> 0.56 ms per step; on row-per-row inputs it was slower)
    if (x.per_input && fa.mode == 0 && !fa.z_out && p.F <= kRowsF - 4 && p.F % 4 == 0 && cp == 12 &&
        (x.stride & 3) == 0 && (reinterpret_cast<uintptr_t>(x.p) & 15) == 0 && (!ov || (ov->cells == 1 && ov->kmax <= 4))) {
        const size_t smem = ((size_t)p.F * 12 + 128 * kRowsF) * sizeof(float);
        cudaFuncSetAttribute(k_final_dense_rows<12, 3>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        k_final_dense_rows<12, 3><<<blocks, 128, smem, s>>>(p);
        return 1;
    }
    // aligned rows of whole 16-byte pieces, weights that fit in shared memory: per-warp rows
    // with the next inputs in flight
    const size_t wbytes = (size_t)p.F * cp * sizeof(float);
    if (p.F % 4 == 0 && (x.stride & 3) == 0 && (reinterpret_cast<uintptr_t>(x.p) & 15) == 0 && cp <= 12 &&
        wbytes <= 96 * 1024) {
        auto go = [&](auto kern) {
            cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)wbytes);
            kern<<<blocks, 128, wbytes, s>>>(p);
        };
        if (cp <= 4) go(k_final_dense_w<4>);
        else if (cp <= 8) go(k_final_dense_w<8>);
        else {
            // 9 to 12 classes: a block's 32 rows shared by four warps
            const size_t sbytes = (size_t)p.F * 16 * sizeof(float);
            cudaFuncSetAttribute(k_final_dense_split, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sbytes);
            k_final_dense_split<<<(unsigned)((rm.R + 31) / 32), 128, sbytes, s>>>(p);
        }
        return 1;
    }
    if (cp <= 4) k_final_dense<4><<<blocks, 128, 0, s>>>(p);
    else if (cp <= 8) k_final_dense<8><<<blocks, 128, 0, s>>>(p);
    else if (cp <= 12) k_final_dense<12><<<blocks, 128, 0, s>>>(p);
    else if (cp <= 16) k_final_dense<16><<<blocks, 128, 0, s>>>(p);
    else if (cp <= 32) k_final_dense<32><<<blocks, 128, 0, s>>>(p);
    else k_final_dense<96><<<blocks, 128, 0, s>>>(p);
    return 1;
}

int launch_epilogue(Src logits, int C, RowMap rm, const FinalArgs &fa, cudaStream_t s, const Overlay *ov)
{
    if (rm.R <= 0) return 0;
    Overlay o;
    if (ov) o = *ov;
    k_epilogue<<<(unsigned)((rm.R + 127) / 128), 128, 0, s>>>(logits.p, logits.stride, logits.per_input, C, rm.t0,
                                                              rm.T, rm.R, fa, o);
    return 1;
}

}  // namespace mure
