// The recurrent family (the paper's RNN models, Sec. 5.3 / Table 1): an embedding of
// token ids and LSTM layers.  Sequences are rows of 1 x T x C values (NHWC with
// H = 1); the ids are integers held in floats.
//
// An LSTM neuron is a unit: its fan-in is the four gate rows of input and recurrent
// weights, W[j][gate][0 .. cin + H), and its biases b[j][gate].  A mutant of an LSTM
// layer changes that layer's whole output from the first step on (the recurrence feeds
// every unit's h to every unit), so there is no channel patch: the layer is recomputed
// for every row of the mutant from its cached input, with the mutated units' rows
// rewritten on the fly (GF / WS: W + e, NAI: -W and -b, NS: the partner's rows and
// biases, NEB: h_j held at 0), and the suffix runs from its output.
#include "common.cuh"
#include "device_util.cuh"

namespace mure {

namespace {

// --------------------------------------------------------------- embedding --

struct EmbedParams {
    const float *x; int64_t x_stride; int x_per_input;   // ids [row][T]
    int64_t t0; int T; int R;
    const int32_t *lrow;
    int steps, dim, vocab;
    const float *W;       // [dim][vocab]
    float *z; int64_t z_stride;   // channel-major [dim][steps] (nullable)
    float *y; int64_t y_stride;   // [steps][dim]
    int *err;
};

// Position t, channel j of a row: W[j][id_t].  An id outside [0, vocab) records
// INVALID_ARG in the context's error word and reads entry 0 (no access outside the
// table).
__global__ void __launch_bounds__(256) k_embed(const EmbedParams p)
{
    const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const int64_t per_row = (int64_t)p.steps * p.dim;
    if (i >= (int64_t)p.R * per_row) return;
    const int64_t row = i / per_row;
    const int rem = (int)(i - row * per_row), t = rem / p.dim, j = rem - t * p.dim;
    const float *xr = p.x + (p.x_per_input ? p.t0 + logical_row(p.lrow, row) % p.T : row) * p.x_stride;
    const float idf = __ldg(xr + t);
    int id = (int)idf;
    if (!(idf >= 0.f && idf < (float)p.vocab) || (float)id != idf) {
        atomicExch(p.err, MURE_ERR_INVALID_ARG);
        id = 0;
    }
    const float v = __ldg(p.W + (int64_t)j * p.vocab + id);
    if (p.z) p.z[row * p.z_stride + (int64_t)j * p.steps + t] = v;
    p.y[row * p.y_stride + (int64_t)t * p.dim + j] = v;
}

// --------------------------------------------------------------------- LSTM --

constexpr int kRows = 32;       // rows per block (one per lane)
constexpr int kWarps = 8;       // warps per block; warp w takes units w, w + 8, ...
constexpr int kMaxUnits = 64;   // units per layer (8 per warp)
constexpr int kUPW = kMaxUnits / kWarps;
constexpr int kMaxIn = 128;     // input width

struct LstmParams {
    const float *x; int64_t x_stride; int x_per_input;
    int64_t t0; int T; int R;
    const int32_t *lrow;
    int steps, cin, H, seq;
    const float *W;       // [H][4][cin + H]
    const float *b;       // [H][4]
    float *z; int64_t z_stride;   // the output again (nullable)
    float *y; int64_t y_stride;   // [steps][H] (seq) or [H]
    PatchArgs pa;         // the batch's mutants (pa.op null: none)
    int mutated;          // 1: rows carry mutants of this layer
};

__device__ __forceinline__ float sigmoid_f(float v) { return 1.f / (1.f + expf(-v)); }

// A block runs kRows rows through every step; lane r of each warp is row r, warp w
// holds units w, w + kWarps, ... with their four gate sums and cell states in
// registers.  Per step the rows' inputs x_t and previous outputs h sit in shared
// memory; every weight load is the same address across the warp.  A gate's
// pre-activation is the fp32 FMA chain over its input weights then its recurrent
// weights in ascending order from +0, then + b.
__global__ void __launch_bounds__(kRows * kWarps) k_lstm(const LstmParams p)
{
    __shared__ float xh[kRows][kMaxIn + kMaxUnits + 1];   // [row][x_t | h_{t-1}]
    __shared__ float hn[kRows][kMaxUnits + 1];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int U = p.cin + p.H;
    const int64_t row0 = (int64_t)blockIdx.x * kRows;
    const int64_t row = row0 + lane;
    const bool ok = row < p.R;
    const float *xr = nullptr;
    if (ok) xr = p.x + (p.x_per_input ? p.t0 + logical_row(p.lrow, row) % p.T : row) * p.x_stride;
    // the mutation of each of this warp's units, uniform over the block's rows (a block
    // of 32 rows lies inside one mutant's rows: input tiles are multiples of 64)
    const float *wp[kUPW], *ep[kUPW], *bp[kUPW];
    float sgn[kUPW];
    bool blocked[kUPW];
    int g = 0;
    if (p.mutated) g = (int)(logical_row(p.lrow, row0) / p.T);
#pragma unroll
    for (int k = 0; k < kUPW; ++k) {
        const int u = warp + k * kWarps;
        wp[k] = p.W + (int64_t)(u < p.H ? u : 0) * 4 * U;
        bp[k] = p.b + 4 * (u < p.H ? u : 0);
        ep[k] = nullptr;
        sgn[k] = 1.f;
        blocked[k] = false;
        if (p.mutated && u < p.H) {
            const int op = p.pa.op[g], n = p.pa.n_neurons[g];
            const int32_t *ids = p.pa.ids + p.pa.neuron_off[g];
            for (int q = 0; q < n; ++q) {
                if (ids[q] != u) continue;
                if (op == MURE_OP_GF || op == MURE_OP_WS) ep[k] = p.pa.patch + p.pa.patch_off[g] + (int64_t)q * 4 * U;
                else if (op == MURE_OP_NAI) sgn[k] = -1.f;
                else if (op == MURE_OP_NEB) blocked[k] = true;
                else if (op == MURE_OP_NS) {
                    const int m = ids[q ^ 1];
                    wp[k] = p.W + (int64_t)m * 4 * U;
                    bp[k] = p.b + 4 * m;
                }
            }
        }
    }
    float cst[kUPW];
#pragma unroll
    for (int k = 0; k < kUPW; ++k) cst[k] = 0.f;
    for (int i = threadIdx.x; i < kRows * p.H; i += blockDim.x) xh[i / p.H][p.cin + i % p.H] = 0.f;
    for (int t = 0; t < p.steps; ++t) {
        for (int i = threadIdx.x; i < kRows * p.cin; i += blockDim.x) {
            const int r = i / p.cin, f = i - r * p.cin;
            const int64_t rr = row0 + r;
            float v = 0.f;
            if (rr < p.R) {
                const float *xrr = p.x + (p.x_per_input ? p.t0 + logical_row(p.lrow, rr) % p.T : rr) * p.x_stride;
                v = __ldg(xrr + (int64_t)t * p.cin + f);
            }
            xh[r][f] = v;
        }
        __syncthreads();
        float acc[kUPW][4];
#pragma unroll
        for (int k = 0; k < kUPW; ++k)
#pragma unroll
            for (int gt = 0; gt < 4; ++gt) acc[k][gt] = 0.f;
        for (int f = 0; f < U; ++f) {
            const float v = xh[lane][f];
#pragma unroll
            for (int k = 0; k < kUPW; ++k) {
                if (warp + k * kWarps >= p.H) break;
#pragma unroll
                for (int gt = 0; gt < 4; ++gt) {
                    float w = __ldg(wp[k] + gt * U + f);
                    if (ep[k]) w = w + __ldg(ep[k] + gt * U + f);
                    acc[k][gt] = fmaf(sgn[k] * w, v, acc[k][gt]);
                }
            }
        }
#pragma unroll
        for (int k = 0; k < kUPW; ++k) {
            const int u = warp + k * kWarps;
            if (u >= p.H) break;
            const float pi = acc[k][0] + sgn[k] * __ldg(bp[k] + 0), pf = acc[k][1] + sgn[k] * __ldg(bp[k] + 1);
            const float pg = acc[k][2] + sgn[k] * __ldg(bp[k] + 2), po = acc[k][3] + sgn[k] * __ldg(bp[k] + 3);
            const float ig = sigmoid_f(pi), fg = sigmoid_f(pf), gg = tanhf(pg), og = sigmoid_f(po);
            cst[k] = fg * cst[k] + ig * gg;
            const float h = blocked[k] ? 0.f : og * tanhf(cst[k]);
            hn[lane][u] = h;
            if (ok && p.seq) {
                p.y[row * p.y_stride + (int64_t)t * p.H + u] = h;
                if (p.z) p.z[row * p.z_stride + (int64_t)t * p.H + u] = h;
            }
        }
        __syncthreads();
        for (int i = threadIdx.x; i < kRows * p.H; i += blockDim.x) xh[i / p.H][p.cin + i % p.H] = hn[i / p.H][i % p.H];
        // the next step's loads of x_t write other columns; the barrier at its top
        // orders them after these reads of hn
    }
    if (ok && !p.seq) {
        for (int k = 0; k < kUPW; ++k) {
            const int u = warp + k * kWarps;
            if (u >= p.H) break;
            p.y[row * p.y_stride + u] = hn[lane][u];
            if (p.z) p.z[row * p.z_stride + u] = hn[lane][u];
        }
    }
}

}  // namespace

int recurrent_supported(const Stage &S)
{
    if (S.kind == MURE_NODE_LSTM) return S.oc <= kMaxUnits && S.ic <= kMaxIn;
    return S.kind == MURE_NODE_EMBED;
}

int launch_embed(const Stage &S, Src x, RowMap rm, float *z_out, int64_t z_stride, float *y_out, int64_t y_stride,
                 cudaStream_t s)
{
    if (rm.R <= 0) return 0;
    EmbedParams p{};
    p.x = x.p; p.x_stride = x.stride; p.x_per_input = x.per_input;
    p.t0 = rm.t0; p.T = rm.T; p.R = rm.R; p.lrow = rm.lrow;
    p.steps = S.iw; p.dim = S.oc; p.vocab = S.vocab;
    p.W = S.W;
    p.z = z_out; p.z_stride = z_stride;
    p.y = y_out; p.y_stride = y_stride;
    p.err = S.err;
    const int64_t n = (int64_t)rm.R * S.iw * S.oc;
    k_embed<<<(unsigned)((n + 255) / 256), 256, 0, s>>>(p);
    return 1;
}

int launch_lstm(const Stage &S, Src x, RowMap rm, float *z_out, int64_t z_stride, float *y_out, int64_t y_stride,
                const PatchArgs *pa, cudaStream_t s)
{
    if (rm.R <= 0) return 0;
    LstmParams p{};
    p.x = x.p; p.x_stride = x.stride; p.x_per_input = x.per_input;
    p.t0 = rm.t0; p.T = rm.T; p.R = rm.R; p.lrow = rm.lrow;
    p.steps = S.iw; p.cin = S.ic; p.H = S.oc; p.seq = S.kh;
    p.W = S.W; p.b = S.b;
    p.z = z_out; p.z_stride = z_stride;
    p.y = y_out; p.y_stride = y_stride;
    if (pa) {
        p.pa = *pa;
        p.mutated = 1;
    }
    k_lstm<<<(unsigned)((rm.R + kRows - 1) / kRows), kRows * kWarps, 0, s>>>(p);
    return 1;
}

}  // namespace mure
