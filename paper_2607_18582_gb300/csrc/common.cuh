// Internal declarations of the GB300 mutation-testing library (not part of the ABI).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include <string>
#include <vector>

#include "../../include/mure.h"

namespace mure {

constexpr int kMaxClasses = 96;   // final-layer kernel keeps one accumulator per class (Reuters: 90)
constexpr int kLabelWords = kMaxClasses / 32;   // 32-bit words of a label set
constexpr int kInputAlign = 64;   // inputs are padded to a multiple of 64 (one kill word)

// A weighted layer together with the unweighted nodes that turn its output into the
// next weighted layer's input ("stage").  Post-ops in order: act1, + skip, act2,
// 2x2/2 max pool, global average pool.
struct Stage {
    int kind;                 // MURE_NODE_CONV2D or MURE_NODE_DENSE
    int ih, iw, ic;           // input x_v (dense: 1 x 1 x fan-in)
    int kh, kw, stride, pad;
    int oh, ow, oc;           // pre-activation z_v
    int K;                    // fan-in kh*kw*ic
    int act1;
    int has_add, skip_src;    // skip tensor = x_{skip_src} (stage-input index)
    int vocab = 0;            // embedding: table entries (ids 0 .. vocab - 1)
    int in_src = -1;          // stage input the layer reads (x_v; an earlier x_s for a
                              // projection in a skip branch, whose add then takes x_v)
    int sc_stride, sc_c;      // shortcut subsampling stride and source channels
    int sk_w;                 // width of the skip source tensor
    int act2;
    int pool, gap;
    int yh, yw, yc;           // output x_{v+1}
    int64_t macs;             // multiply-accumulates per row
    int variant = 0;          // 0: implicit-GEMM kernel; > 0: a shared-memory direct conv
    int geo = 0;              // > 0: a compiled small geometry (the delta's dot-product kernel)
    int tc = 0;               // tensor-core kernel: 1 = 3xTF32, 2 = one TF32 MMA (variant)
    int tc_small = 0;         // tc: the small-image convolution mode
    int tc_conv = 0;          // tc: the staged convolution mode (input rows staged per tile)
    int tc_wide = 0;          // tc_conv: all 256 outputs in one CTA (one N = 256 MMA per K8 step)
    int tc_win = 0;           // tc_conv: a GEMM row per 2x2 output window (16-channel 3x3 layers:
                              // N = 4 positions x 16 outputs over a 4x4 field of 16 channels)
    float *Wtc = nullptr;     // tc: TF32 halves of W in the tensor-core operand layout
    int *err = nullptr;       // device error word of the context (bounded waits)
    const int64_t *wait_limit = nullptr;   // host: the context's wait limit (0 = default)
    float *W = nullptr;       // device [oc][K]
    float *Wt = nullptr;      // device [K][oc] (the same weights, K-major rows)
    float *b = nullptr;       // device [oc]
    float sigma_std = 0.f;    // population std of W (host copy, fp32-rounded for info)
};

// Stage inputs x_s, s = 0..L (x_0 network input, x_L logits): shape and row stride.
struct TensorDim {
    int h, w, c;
    int64_t size, stride;     // elements; stride = size rounded up to a multiple of 4
};

__host__ __device__ inline int round_up16(int n) { return (n + 15) & ~15; }
__host__ __device__ inline int round_up32(int n) { return (n + 31) & ~31; }

}  // namespace mure

struct mure_ctx {
    int device = 0;
    cudaStream_t stream = nullptr;
    mure_allocator alloc{};
    bool has_alloc = false;
    std::string err;
    cudaEvent_t ev[8]{};
    std::vector<cudaEvent_t> evpool;  // per-launch timing events, reused across calls
    int n_sms = 0;
    int64_t launches = 0;             // kernels launched since creation
    int *err_dev = nullptr;           // device error word written by bounded waits
    int64_t wait_limit = 0;           // limit of the device-side waits in SM cycles (0 = default)
};

struct mure_model {
    mure_ctx *ctx = nullptr;
    int precision = MURE_PREC_FP32;
    int L = 0;
    int n_classes = 0;
    std::vector<mure::Stage> st;      // L stages
    std::vector<mure::TensorDim> xd;  // L + 1 stage inputs
    std::vector<mure::TensorDim> zd;  // L pre-activations
    double *sigma_dev = nullptr;      // device [L] population std of each layer's W (fp64)
    std::vector<double> sigma_host;
};

struct mure_cache {
    mure_model *model = nullptr;
    int64_t n_in = 0, n_pad = 0;
    std::vector<float *> x;           // x[s], s = 0..L: [n_pad][xd[s].stride]
    std::vector<float *> z;           // z[v], v = 0..L-1: [n_pad][zd[v].stride]
    int32_t *pred0 = nullptr;         // [n_pad]
    int32_t *label = nullptr;         // [n_pad]
    int n_label_values = 0;           // |L|: distinct labels among the inputs
    bool full = true;                 // false: only x[0] / pred0 / label (vanilla)
};

namespace mure {

// ------------------------------------------------------------ kernel launchers --
// All launchers queue on `s` and return the number of kernels launched.

// Where a batch row reads a tensor: per row (row r at p + r*stride) or per input
// (row r at p + (t0 + r % T)*stride, shared by the batch's mutants).
struct Src {
    const float *p;
    int64_t stride;
    int per_input;
};

struct RowMap {
    int64_t t0;   // first input of the tile
    int T;        // inputs per tile (multiple of 64)
    int R;        // rows = mutants in the batch x T (or the rows left after compaction)
    // compacted batch (unchanged rows removed): physical row r is logical row lrow[r]
    // = g * T + input offset; null: physical = logical
    const int32_t *lrow = nullptr;
};

// The logical row (mutant g = lr / T, input t0 + lr % T) of physical row r.  Per-input
// sources (cached rows), the patch rows, the group tables and the kill bits are
// indexed by it; the batch's own row buffers by r.
__host__ __device__ __forceinline__ int64_t logical_row(const int32_t *lrow, int64_t r)
{
#ifdef __CUDA_ARCH__
    return lrow ? (int64_t)__ldg(lrow + r) : r;
#else
    return lrow ? (int64_t)lrow[r] : r;
#endif
}

// The mutated channels of a batch's rows of x_{l+1}, applied on top of the unmutated
// row by the first suffix kernel: for batch mutant g = r / T and slot q < n_neurons[g],
// channel ids[neuron_off[g] + q] of cell c is patch[r * row_stride + q * cells + c];
// the row's element for (cell c, channel j) is at c * ch + j.
struct Overlay {
    const float *patch = nullptr;   // null: no overlay
    int64_t row_stride = 0;
    int kmax = 0, cells = 0, ch = 0;
    const int32_t *n_neurons = nullptr;
    const int64_t *neuron_off = nullptr;
    const int32_t *ids = nullptr;
    // non-null (window GEMM only): per-group operator codes; NEB rows get their mutated
    // channels zeroed and NS rows their channel pairs swapped in the staged maps, and
    // the patch values of those rows are not read (the delta need not write them)
    const int32_t *op = nullptr;
};

// Stage v over R rows: z (optional) and y = post(act1(conv(x) + b)).
int launch_stage_simt(const Stage &S, Src x, RowMap rm, float *z_out, int64_t z_stride, Src skip,
                      float *y_out, int64_t y_stride, float *gap_tmp, cudaStream_t s);

// The shared-memory direct convolution for small inputs (variant of a stage, 0 when
// the geometry is not one it compiles) and its launcher.
int conv_small_variant(const Stage &S);
int launch_conv_small(const Stage &S, Src x, RowMap rm, float *z_out, int64_t z_stride, float *y_out,
                      int64_t y_stride, cudaStream_t s, const Overlay *ov = nullptr);

// Tensor-core layers (tcgen05; 3xTF32, or one TF32 MMA in the reduced-precision
// mode): which layers the kernel takes, the weight split done at model load, and the
// launcher (arguments as for the stage kernel, plus the overlay).
int tc_supported(const Stage &S);
int64_t tc_weight_floats(const Stage &S);
int tc_overlay_inline(const Stage &S, const Overlay &ov, int64_t groups);
int tc_small_geometry(const Stage &S);
int tc_conv_geometry(const Stage &S);
int tc_wide_geometry(const Stage &S);
int tc_win_geometry(const Stage &S);
int launch_swizzle_weights(const Stage &S, float *out, float *tmp, cudaStream_t s);
int64_t tc_swizzle_tmp_floats(const Stage &S);
int64_t tc_macs_per_row(const Stage &S);
// The output layer (dense, C <= 12 classes) computed in the epilogue of the
// tensor-core dense layer that feeds it, with the kill epilogue: W [C][F], bias b,
// activation act.  The rows of the layer in between are then never stored.
struct FinalFuse;
// Output of the tensor-core delta: column n < n of the GEMM is slot (g[n], q[n]) of the
// batch, channel j[n] of the layer; the GEMM's sum is added to the pre-activation
// z[row][j][position] before the post-ops, and the value for output cell c of input
// row r goes to out[(g * T + r) * stride + q * cells + c].
struct SlotStore {
    float *out = nullptr;
    int64_t stride = 0;
    const int32_t *g = nullptr, *q = nullptr, *j = nullptr;
    int n = 0, cells = 0, T = 0;
    const float *z = nullptr;
    int64_t z_stride = 0;
    int z_per_input = 0;
};
int launch_tc(const Stage &S, Src x, RowMap rm, float *z_out, int64_t z_stride, Src skip, float *y_out,
              int64_t y_stride, float *gap_tmp, cudaStream_t s, const Overlay *ov = nullptr,
              const FinalFuse *ff = nullptr, const SlotStore *ss = nullptr);
// Whether stage S (feeding the output layer SL) can take SL into its epilogue.
int tc_final_fusable(const Stage &S, const Stage &SL);

// The recurrent family: embedding lookups and LSTM layers over R rows of sequences
// (iw = steps).  launch_lstm with pa non-null recomputes a mutated LSTM layer: every row
// of batch mutant g takes its mutated units' rewritten rows (GF / WS: W + e of the
// patch, NAI: negated, NS: the partner's, NEB: h held at 0).
int recurrent_supported(const Stage &S);
int launch_embed(const Stage &S, Src x, RowMap rm, float *z_out, int64_t z_stride, float *y_out, int64_t y_stride,
                 cudaStream_t s);
struct PatchArgs;
int launch_lstm(const Stage &S, Src x, RowMap rm, float *z_out, int64_t z_stride, float *y_out, int64_t y_stride,
                const PatchArgs *pa, cudaStream_t s);

// Global average pooling of R rows of a [P][C] map.
int launch_gap(const float *in, int64_t in_stride, int P, int C, int R, float *y, int64_t y_stride, cudaStream_t s);

// Final dense layer (F -> C, C <= 32) over R rows, with the fused epilogue.
struct FinalArgs {
    const int32_t *mutant_id;   // [G] original mutant index of batch mutant g
    const int32_t *label;       // [n_pad]
    const int32_t *pred0;       // [n_pad]
    int64_t n_in;
    uint32_t *kill32;           // [n_mut][words32] (kill mode)
    int64_t words32;
    float *logits_rows;         // optional per-row logits [R][C] (pre-epilogue mode)
    float *logits_out;          // optional [n_mut][n_in][C]
    float *z_out;               // cache mode: z[L-1] rows; nullable
    int64_t z_stride;
    float *x_out;               // cache mode: logits rows x[L]; nullable
    int64_t x_stride;
    int32_t *pred_out;          // cache mode: pred0 [n_pad]
    unsigned long long *near_ties;
    int mode;                   // 0 = kill, 1 = cache build, 2 = write per-row logits only
    int compact;                // kill mode on a compacted batch: kill bits OR-ed into a zeroed matrix
    const int32_t *lrow;        // compacted batch: logical row of each physical row (else null)
};
int launch_final_dense(const Stage &S, Src x, RowMap rm, const FinalArgs &fa, cudaStream_t s,
                       const Overlay *ov = nullptr);
struct FinalFuse {
    const float *W;   // [C][F]
    const float *b;   // [C]
    int C, F, act;
    FinalArgs fa;     // kill mode
};

// Kill epilogue on logits rows (mutants of the output layer), with an optional overlay.
int launch_epilogue(Src logits, int C, RowMap rm, const FinalArgs &fa, cudaStream_t s, const Overlay *ov = nullptr);


// Per-mutant patch data of a batch, in device memory.
struct PatchArgs {
    const int32_t *op;          // [G]
    const int32_t *n_neurons;   // [G]
    const int64_t *neuron_off;  // [G] into ids
    const int32_t *ids;         // neuron pool
    const int64_t *patch_off;   // [G] offset of slot 0 into patch (-1: none)
    const float *patch;         // GF: sigma * n, WS: W[j][perm f] - W[j][f]; F per slot
    const int32_t *dslot = nullptr;   // the batch's GF / WS slots: (global group, slot q) pairs
    int64_t n_dslot = 0;
    int32_t dslot_g0 = 0;             // global index of the batch's first group
    const int4 *vslot = nullptr;      // the batch's other slots: (global group, q, source channel, op)
    int64_t n_vslot = 0;
};

// Delta of layer l: values of the mutated neurons' channels of x_{l+1}, from z_l
// (channel-major; x_l for GF / WS), the layer's post-ops and skip, into
// out[r][q][c] (slot q < kmax, output cell c of layer l).
int launch_patch_vals(const Stage &S, Src z, Src x, Src skip, RowMap rm, const PatchArgs &pa, int kmax, float *out,
                      int64_t out_stride, cudaStream_t s, bool skip_dot_ops = false, bool skip_copy_ops = false);

// GF / WS delta values on the tensor cores (convolution layers, tensor-core precision
// modes): one implicit GEMM over the batch's inputs whose output channels are the
// weight deltas e of every GF / WS slot of the batch (128 per N slice, so a slot's
// arithmetic never depends on the batch); the epilogue adds the cached pre-activation
// z of the slot's channel (e = 0 gives z exactly), applies the layer's post-ops and
// stores into the patch rows.  Scratch: filters, their swizzled halves and per-column tables
// for up to n_max slots of fan-in up to k_max.
struct TcDeltaWs {
    float *filt = nullptr, *swz = nullptr, *colb = nullptr;
    int32_t *colg = nullptr, *colq = nullptr, *colj = nullptr;
    int n_max = 0, k_max = 0;
};
int tc_delta_supported(const Stage &S, int precision);
void tc_delta_ws_size(int n_slots, int k_max, int64_t &floats, int64_t &ints);
int launch_tc_delta(const Stage &S, int precision, Src z, Src x, Src skip, RowMap rm_inputs, const PatchArgs &pa, float *out,
                    int64_t out_stride, const TcDeltaWs &dw, cudaStream_t s);

// GF / WS delta values of the small-layer geometries (stage variant > 0): the same
// values as launch_patch_vals for those operators; launch_patch_vals then skips them.
int patch_dot_supported(const Stage &S, int kmax);
int launch_patch_dot(const Stage &S, Src z, Src x, RowMap rm, const PatchArgs &pa, int kmax, float *out,
                     int64_t out_stride, cudaStream_t s);

// Materialise rows: out = base rows with the overlay applied.
int launch_rows_overlay(Src base, int64_t n_floats, RowMap rm, const Overlay &ov, float *out, int64_t out_stride,
                        cudaStream_t s);

// The descriptor checks of mure_eval_mutants (status and last-error text), for entry
// points outside the scheduler.
mure_status check_table_status(mure_ctx *c, const mure_model *m, const mure_mutant *t, int64_t n, const int32_t *pool,
                               int64_t pool_len);

// Expand GF / WS descriptors into patches (see mure_expand_patches): one job per
// (mutant, neuron slot).
struct SlotJob {
    int32_t layer, op, F, j, q, reserved;
    float param, reserved2;
    uint64_t seed;
    int64_t out_off;   // F values at patch + out_off
    int64_t perm_off;  // WS: F ints of permutation scratch
};
struct ExpandArgs {
    const SlotJob *jobs;
    int64_t n_jobs;
    const double *sigma;        // [L] population std of each layer's weights
    const float *const *W;      // [L] device weight pointers ([oc][K])
    float *patch;
    int32_t *perm;              // WS permutation scratch
    int ws_as_weights;          // 1: WS patch holds the permuted weights (inspection)
};
int launch_expand(const ExpandArgs &ea, cudaStream_t s);

// Population std of each layer's weights in fp64.
int launch_layer_std(const float *const *W, const int64_t *n, int L, double *out, cudaStream_t s);

// Exact unchanged-row elimination (memoized mode).  Row r of a batch (mutant g =
// r / T, input t0 + r % T) is unchanged when every mutated channel of its patch equals
// the cached original x_{l+1} of its input bit for bit: its suffix then equals the
// original forward pass, so its kill bit is 0 and its logits are the cached original
// logits (written to logits_out when requested; its near tie is counted from them).
// flags[r] = 1 for the rows still to run; lrow receives them in ascending order and
// count their number.  Scratch: block_cnt of ceil(R / 256) ints.
struct UnchangedArgs {
    const float *patch;          // [R][kmax][cells] the delta's values
    int64_t row_stride;
    int cells, ch;               // cells of x_{l+1}; channels (layer l's outputs)
    const int32_t *n_neurons;    // [G] of the batch
    const int64_t *neuron_off;
    const int32_t *ids;
    const float *base;           // cached x_{l+1} rows (per input)
    int64_t base_stride;
    const float *logits;         // cached original logits rows (per input)
    int64_t logits_stride;
    int C;
    FinalArgs fa;                // logits_out, near_ties, mutant ids, n_in
};
int launch_unchanged(const UnchangedArgs &ua, RowMap rm, int32_t *flags, int32_t *block_cnt, int32_t *lrow,
                     int32_t *count, cudaStream_t s);

// Score reduction: per mutant killed flag and |killingLabels|, summed.
int launch_scores(const uint32_t *kill32, int64_t n_mut, int64_t words32, const int32_t *label, int n_classes,
                  unsigned long long *totals /* [2]: killed, sum of label counts */, cudaStream_t s);

// Distinct labels among n inputs (bitset of kLabelWords words; mask zeroed by the caller).
int launch_label_set(const int32_t *label, int64_t n, uint32_t *mask, cudaStream_t s);

}  // namespace mure
