/*
 * mure.h -- C ABI of the GB300 (sm_103a) library for memoized DNN mutation testing.
 *
 * The library evaluates weight-level mutants of one feed-forward network on a test
 * input set and fills the mutants x inputs kill matrix and the mutation score
 * (Ghanbari et al., "Provably Lossless Acceleration of DNN Mutation Testing via
 * Memoization", PACMSE/ISSTA 2026; Algorithm 1, Sec. 3 and Sec. 5.2).
 *
 * Memoized mode follows Algorithm 1: the original network's activations are computed
 * once and kept in device memory (the memo table of Algorithm 3, extended to every
 * layer), mutants are grouped by their first mutated layer (the clusters of
 * Algorithm 1, lines 3-9), and each mutant runs only from its mutated layer onward
 * on memo rows (the chopped mutant of Algorithm 4).  Vanilla mode runs every mutant
 * end to end from the inputs (the paper's exhaustive baseline, Sec. 5.1).
 *
 * Conventions for every call
 *   - Tensors are fp32, NHWC, densely packed, row-major.
 *   - A status other than MURE_OK leaves every output buffer untouched unless the
 *     call says otherwise; mure_last_error() then holds a one-line reason.
 *   - All argument validation happens before any device work is queued.
 *   - Calls on one context are not thread-safe; use one context per host thread.
 *   - Every call is synchronous with respect to the host: when it returns, its
 *     results are in the caller's buffers.  Device work runs on the context's stream.
 *   - Pointers documented as "host" must be host memory; "device" ones must be memory
 *     of the context's device.  The caller keeps ownership of everything it passes.
 */
#ifndef MURE_H
#define MURE_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    MURE_OK = 0,
    MURE_ERR_INVALID_ARG = 1, /* a bad pointer, size, index, graph or descriptor */
    MURE_ERR_UNSUPPORTED = 2, /* valid but outside what the kernels implement */
    MURE_ERR_OOM = 3,         /* device allocation failed (nothing was launched) */
    MURE_ERR_CUDA = 4,        /* a CUDA runtime call failed */
    MURE_ERR_TIMEOUT = 5      /* a device-side bounded wait gave up */
} mure_status;

/* Network node kinds (Sec. 4: a network is a DAG of layer functions). */
enum {
    MURE_NODE_CONV2D = 0,   /* zero-padded 2-D convolution + bias + activation */
    MURE_NODE_DENSE = 1,    /* fully connected + bias + activation */
    MURE_NODE_MAXPOOL2D = 2,/* max pooling, window kh x kw, stride `stride` (floor) */
    MURE_NODE_FLATTEN = 3,  /* reshape to a vector (no data movement in NHWC) */
    MURE_NODE_ADD = 4,      /* element-wise sum of in0 and in1 + activation */
    MURE_NODE_GAP = 5,      /* global average pooling over H and W */
    MURE_NODE_SHORTCUT = 6, /* parameter-free residual shortcut: subsample by
                               `stride`, zero channels appended up to `cout` */
    MURE_NODE_DWCONV = 7,   /* depthwise 2-D convolution (MobileNetV2, Table 1): channel
                               c of the output is a kh x kw filter over channel c of the
                               input, + bias + activation; cin = cout = the input's
                               channels, W [c][kh][kw]; neuron j = channel j, whose fan-in
                               is its kh*kw filter */
    MURE_NODE_EMBED = 8,    /* embedding (the recurrent family of Table 1): the input is
                               1 x T x 1 token ids held in floats (integers in [0, cin));
                               output 1 x T x cout, position t channel j = W[j][id_t];
                               W [cout][cin] (channel-major), b may be NULL (no bias);
                               neuron j = channel j, whose fan-in is its cin table entries */
    MURE_NODE_LSTM = 9      /* LSTM over the 1 x T x cin input sequence, cout units, zero
                               initial state, gates i, f, g, o: pre = b + Wx x_t + Wh h,
                               i, f, o = sigmoid, g = tanh, c = f c + i g, h = o tanh(c);
                               W [cout][4][cin + cout] (a unit's gate rows: input weights,
                               then recurrent weights), b [cout][4]; kh = 1: output every
                               step (1 x T x cout), kh = 0: the last step (1 x 1 x cout);
                               neuron j = unit j, whose fan-in is its 4 (cin + cout)
                               weights (NEB holds h_j at 0 at every step) */
};
enum { MURE_ACT_NONE = 0, MURE_ACT_RELU = 1, MURE_ACT_RELU6 = 2 /* min(max(v, 0), 6) */ };

/* Mutation operators (Sec. 3.1; DeepMutation's weight-level mutators).  Neuron j of
 * a weighted layer is its output channel / output unit j (Sec. 2.1).
 *   GF  Gaussian fuzzing: w[j][f] += sigma * n, n ~ N(0,1), sigma = param x the
 *       population standard deviation of the layer's weights (bias excluded).
 *   NEB neuron effect blocking: the output of neuron j is 0.
 *   NAI neuron activation inverse: the pre-activation of neuron j is negated.
 *   NS  neuron switch: neurons j0, j1 (consecutive pool entries) exchange filters
 *       and biases; n_neurons must be even.
 *   WS  weight shuffling: the fan-in weights of neuron j are permuted.
 *   IDENTITY no change (neurons ignored).
 * GF noise and WS permutations come from the counter-based SplitMix64 generator
 * (Steele, Lea, Flood, OOPSLA 2014): the stream of neuron slot q of a mutant with
 * seed s is seeded with draw q of a generator seeded with s; GF's standard normals
 * come from the Box-Muller transform of draw pairs (2p, 2p+1) in fp64 (cosine for
 * even, sine for odd index), rounded to fp32 after scaling by sigma; WS uses
 * Fisher-Yates from the last index down, j = floor(u (i+1)) with u the top 53 bits. */
enum { MURE_OP_GF = 0, MURE_OP_NEB = 1, MURE_OP_NAI = 2, MURE_OP_NS = 3, MURE_OP_WS = 4, MURE_OP_IDENTITY = 5 };

/* Arithmetic of the layer kernels.  FP32: fp32 FMA chains on the CUDA cores.
 * TF32X3: dense layers and convolutions of >= 16 outputs on the tensor cores
 * (tcgen05), fp32 operands split into two TF32 halves, three products per pair
 * (fp32-level accuracy); small LeNet-size convolutions stay on the CUDA cores.
 * TF32: the same layer selection with one TF32 product (the reduced-precision
 * variant; its kill verdicts are compared with the fp32 oracle's, not bit-matched).  BF16:
 * reserved.  The output layer always uses the fp32 CUDA-core kernel.  One model uses
 * one arithmetic for every layer computation (cache build, vanilla prefix and
 * suffix), so memoized and vanilla results stay bit-identical under every mode. */
enum { MURE_PREC_FP32 = 0, MURE_PREC_TF32X3 = 1, MURE_PREC_BF16 = 2, MURE_PREC_TF32 = 3 };

/* One node.  in0/in1 are node ids (< this node's id) or -1 for the network input.
 * Weighted nodes (CONV2D, DENSE) are numbered 0..L-1 in node order: these numbers
 * are the "layers" of mutant descriptors.  W: conv [cout][kh][kw][cin], dense
 * [cout][cin]; b: [cout].  W and b are host pointers, copied by mure_model_load. */
typedef struct {
    int32_t kind, act, in0, in1;
    int32_t kh, kw, stride, pad;
    int32_t cin, cout;
    const float *W;
    const float *b;
} mure_node;

/* Network description.  Nodes in topological order; the last node is the output
 * (the logits), of size n_classes.  The supported shape of the graph: each
 * weighted node is followed, before the next weighted node reads it, by at most one
 * ADD (its other input a network input, a block input or a SHORTCUT of one), then
 * optional MAXPOOL2D (2x2, stride 2), FLATTEN and GAP nodes; the output node is
 * the last weighted node.  Other graphs return MURE_ERR_UNSUPPORTED. */
typedef struct {
    int32_t in_h, in_w, in_c, n_classes;
    int32_t n_nodes;
    int32_t precision; /* MURE_PREC_* */
    const mure_node *nodes;
} mure_model_desc;

/* One mutant descriptor (the mutant map of Algorithm 1).  Untagged (tagged = 0):
 * mu(M') = {layer}, the pool entries are neuron ids of that layer.  Tagged
 * (tagged = 1): the mutant's set mu(M') may hold several layers (the paper's general
 * case, Sec. 3.2; DeepMutation's model-wide selection ratio); each pool entry is
 * (layer << 20) | neuron and `layer` must be the smallest listed layer (mmi).  The
 * operator applies to every listed neuron in its own layer: GF's sigma comes from that
 * layer's weights, pool slot q keeps random stream q whatever its layer, and NS pairs
 * (consecutive entries) lie in one layer. */
typedef struct {
    int32_t layer;      /* first mutated weighted layer (mmi), 0..L-1 */
    int32_t op;         /* MURE_OP_* */
    int32_t n_neurons;  /* pool entries at neuron_pool[neuron_off .. +n_neurons) */
    int32_t tagged;     /* 0: entries are neurons of `layer`; 1: (layer << 20) | neuron */
    int64_t neuron_off;
    float param;        /* GF: sigma multiplier (e.g. 0.1); ignored otherwise */
    float reserved2;    /* must be 0 */
    uint64_t seed;      /* GF / WS random stream */
} mure_mutant;

/* Device allocator.  When given to mure_create, every device allocation of the
 * library goes through it (for instance a framework's caching allocator); when
 * NULL, the library uses cudaMallocAsync / cudaFreeAsync on the context stream.
 * alloc returns NULL on failure. */
typedef struct {
    void *(*alloc)(size_t bytes, void *stream, void *user);
    void (*free)(void *ptr, void *stream, void *user);
    void *user;
} mure_allocator;

typedef struct {
    int32_t outputs_on_device; /* kill_bits / logits_out are device pointers */
    int32_t kernel_timing;     /* 1: time every kernel launch with CUDA events on the
                                  context stream and report per-layer times in stats */
    int64_t workspace_bytes;   /* cap on per-batch scratch (0: 8 GiB) */
    float *logits_out;         /* nullable; [n_mutants][n_inputs][n_classes]: every
                                  mutant's logits (for parity checks; slows the run) */
    int32_t skip_unchanged;    /* mure_eval_mutants, 1: exact unchanged-row elimination.
                                  A single-layer mutant's row whose input to the first
                                  suffix layer (x_{l+1}: the mutated layer's output after
                                  its activation, residual add and pooling) equals the
                                  original bit for bit is not run: its suffix would repeat
                                  the original forward pass, so its kill bit is 0 and its
                                  logits are the original logits.  Results are identical
                                  to 0 (the default); stats.n_rows_unchanged counts the
                                  rows dropped.  Ignored by mure_eval_vanilla. */
    int32_t reserved;          /* 0 */
} mure_eval_opts;

typedef struct {
    double ms_total;        /* device time of the whole call (CUDA events) */
    double ms_expand;       /* descriptor expansion (GF noise, WS shuffles) */
    double ms_suffix;       /* delta + suffix + epilogue kernels */
    double ms_score;        /* score reduction */
    int64_t n_rows;         /* (mutant, input) pairs evaluated */
    int64_t n_near_ties;    /* rows whose top-2 logit margin < 1e-4 |max logit| */
    int64_t n_groups;       /* first-mutated-layer groups with >= 1 mutant */
    int64_t n_batches;      /* (group, mutant chunk, input tile) batches */
    int64_t kernel_launches;/* library kernels launched by the call */
    int64_t flops;          /* analytic FLOPs of the layer kernels that ran */
    /* with kernel_timing: device time and analytic FLOPs of the kernels of each
       weighted layer (index = layer, up to MURE_MAX_TIMED_LAYERS), of the delta
       kernels (which also copy the cached rows a group starts from), and of the
       stand-alone kill epilogue.  Where the mutated layer's fan-in sums (GF / WS)
       run in a kernel of their own, the delta's value kernels (NEB / NAI / NS: the
       cached pre-activations read, the patch values written) are timed apart in
       ms_delta_values; otherwise they are part of ms_delta */
    double ms_layer[64];
    int64_t flops_layer[64];
    int64_t launches_layer[64];
    double ms_delta, ms_delta_values, ms_epilogue;
    int64_t bytes_gather;   /* row bytes the delta kernel copies (read + write) */
    int64_t launches_delta;
    int64_t bytes_rows;     /* activation rows the stage kernels write and the next stage
                               reads back (2 x rows x row bytes): the device-memory traffic
                               of the batched suffix beyond the algorithmic bytes */
    int64_t n_rows_unchanged; /* rows not run by the unchanged-row elimination */
    int64_t launches_delta_values; /* with kernel_timing: launches timed in ms_delta_values */
    int64_t bytes_delta_values;    /* algorithmic bytes of those value kernels: the patch
                                      values they write and the cached pre-activation row
                                      of each input of a batch, read once for all its
                                      mutants (memoized), or each row's own (vanilla) */
} mure_eval_stats;

#define MURE_MAX_TIMED_LAYERS 64

typedef struct mure_ctx mure_ctx;
typedef struct mure_model mure_model;
typedef struct mure_cache mure_cache;

/* Create a context on CUDA device `device` that queues all work on `cuda_stream`
 * (a cudaStream_t; NULL = the legacy default stream).  alloc may be NULL.
 * Errors: INVALID_ARG (out == NULL, bad device), CUDA. */
mure_status mure_create(int device, void *cuda_stream, const mure_allocator *alloc, mure_ctx **out);

/* Destroy a context.  Models and caches made from it must be freed first. */
void mure_destroy(mure_ctx *ctx);

/* The reason for the last failed call on this context ("" if none).  Valid until
 * the next call on the context. */
const char *mure_last_error(const mure_ctx *ctx);

/* Copy a network to the device and compile it into stages (Algorithm 2: the
 * dependence graph is read from the nodes' inputs).  Errors: INVALID_ARG
 * (inconsistent shapes, bad ids, NULL weights), UNSUPPORTED (graph outside the
 * supported shape, n_classes > 96, unknown precision), OOM, CUDA. */
mure_status mure_model_load(mure_ctx *ctx, const mure_model_desc *desc, mure_model **out);
void mure_model_free(mure_model *model);

/* Validate a network description and a mutant table on the host, without a context
 * or a device: the checks mure_model_load runs on `desc` (its compilation into
 * stages included) and those mure_eval_mutants / mure_eval_vanilla run on the table
 * before any launch (Algorithm 1's inputs: every mutant's layer, operator, neuron
 * range, NS pairing, repeated neurons, and for tagged descriptors each entry's
 * layer and the smallest-layer rule).  n_mutants = 0 checks the description alone.
 * Every pointer is the caller's and is only read.  Returns OK, INVALID_ARG or
 * UNSUPPORTED; when msg != NULL the one-line reason ("" on success) is written there,
 * NUL-terminated and cut to msg_len bytes. */
mure_status mure_check_descriptors(const mure_model_desc *desc, const mure_mutant *table, int64_t n_mutants,
                                   const int32_t *neuron_pool, int64_t pool_len, char *msg, size_t msg_len);

/* Kernels this context has launched since it was created (all calls). */
int64_t mure_kernel_launches(const mure_ctx *ctx);

/* Limit of the device-side waits of this context's tensor-core kernels, in SM clock
 * cycles (0, the initial value, restores the default of 2e9 cycles, about a second at
 * the SM clock).  The paper has no counterpart: this is failure detection.  Every
 * wait of a role of those kernels (for operand copies, MMAs, tensor-memory stages or
 * accumulators) gives up after the limit; the kernel then stops all its roles, lets
 * its own copies and MMAs in flight land (those teardown waits keep the default limit
 * whatever this setting), frees its tensor memory and returns, and the call that
 * launched it returns TIMEOUT with the context still usable (that call's output
 * buffers are then undefined).  A limit far below the
 * kernels' normal waits makes calls fail on purpose (a test of that path).  Applies
 * to launches queued after this call.  Errors: INVALID_ARG (NULL context, negative
 * limit). */
mure_status mure_set_wait_limit(mure_ctx *ctx, int64_t cycles);

/* Number of weighted layers L of a loaded model (or -1 for NULL). */
int32_t mure_model_n_layers(const mure_model *model);

/* Which kernel computes weighted layer `layer` of a loaded model (the choice is fixed
 * when the model is loaded, so every computation of a layer uses one kernel), and the
 * multiply-accumulates that kernel executes per batch row.  Kernel codes:
 *   MURE_KERNEL_SIMT_GEMM    CUDA-core implicit GEMM (fp32 chains)
 *   MURE_KERNEL_SIMT_SMALL   CUDA-core direct convolution for LeNet-size layers
 *   MURE_KERNEL_TC_GEMM      tensor-core GEMM / implicit-GEMM convolution
 *   MURE_KERNEL_TC_WINDOW    tensor-core GEMM over 2x2 pooling windows
 *   MURE_KERNEL_OUTPUT       output layer with the fused argmax / kill epilogue
 *   MURE_KERNEL_TC_CONV      tensor-core convolution over input rows staged in shared
 *                            memory (stride 1, input channels a multiple of 32)
 * macs_per_row counts the GEMM as executed (padding and, for the window form, the
 * zero taps included; one product per MAC, whatever the precision mode).  Either
 * output pointer may be NULL.  Errors: INVALID_ARG (NULL model, layer out of range). */
typedef enum {
    MURE_KERNEL_SIMT_GEMM = 0,
    MURE_KERNEL_SIMT_SMALL = 1,
    MURE_KERNEL_TC_GEMM = 2,
    MURE_KERNEL_TC_WINDOW = 3,
    MURE_KERNEL_OUTPUT = 4,
    MURE_KERNEL_TC_CONV = 5
} mure_kernel;
mure_status mure_model_layer_kernel(const mure_model *model, int32_t layer, int32_t *kernel, int64_t *macs_per_row);

/* Build the prefix-activation cache (the memo table, Algorithm 3 and Algorithm 1
 * lines 11-12, kept for every layer so every cluster shares one table): one forward
 * pass of the original network over X [n_inputs][in_h][in_w][in_c] storing, per
 * input, every weighted layer's input and pre-activation output, plus the original
 * logits, predictions and labels.  labels [n_inputs] in [0, n_classes) or NULL (then
 * label = original prediction, and kill reduces to "prediction changed").  X and
 * labels are device pointers when x_on_device != 0, else host pointers.  n_inputs
 * may be 0.  Errors: INVALID_ARG (NULL X with n_inputs > 0, label out of range),
 * OOM, CUDA. */
mure_status mure_build_prefix_cache(mure_model *model, const float *X, int64_t n_inputs, const int32_t *labels,
                                    int x_on_device, mure_cache **out);
void mure_cache_free(mure_cache *cache);

/* Original logits [n_inputs][n_classes] and predictions [n_inputs] held by a cache,
 * copied to host buffers (either may be NULL). */
mure_status mure_cache_outputs(mure_cache *cache, float *logits, int32_t *pred);

/* Memoized mutation testing (Algorithm 1).  table [n_mutants] and neuron_pool
 * [pool_len] are host arrays.  kill_bits [n_mutants][ceil(n_inputs/64)] receives
 * bit t of row i = kill(mutant i, input t) (Sec. 5.2: the original predicts
 * label(t) and the mutant does not), least significant bit first; padding bits are
 * 0.  score_killed_frac = killed mutants / n_mutants; score_deepmutation =
 * sum_i |killingLabels(i)| / (n_mutants |L|), L the labels present in the inputs
 * (Sec. 5.2).  Either score pointer may be NULL; stats may be NULL; opts may be
 * NULL (host outputs, defaults).  n_mutants may be 0.  Errors: INVALID_ARG (bad
 * descriptor: layer, op, neuron id out of range or repeated, odd NS count,
 * non-zero reserved fields, pool range), OOM, CUDA, TIMEOUT. */
mure_status mure_eval_mutants(mure_cache *cache, const mure_mutant *table, int64_t n_mutants,
                              const int32_t *neuron_pool, int64_t pool_len, const mure_eval_opts *opts,
                              uint64_t *kill_bits, double *score_killed_frac, double *score_deepmutation,
                              mure_eval_stats *stats);

/* Vanilla mutation testing (the paper's exhaustive baseline): every mutant is run
 * end to end from X with no activation reuse across mutants, through the same layer
 * kernels, so its outputs equal mure_eval_mutants' bit for bit (Theorem 1).
 * Arguments as in mure_build_prefix_cache followed by mure_eval_mutants. */
mure_status mure_eval_vanilla(mure_model *model, const float *X, int64_t n_inputs, const int32_t *labels,
                              int x_on_device, const mure_mutant *table, int64_t n_mutants,
                              const int32_t *neuron_pool, int64_t pool_len, const mure_eval_opts *opts,
                              uint64_t *kill_bits, double *score_killed_frac, double *score_deepmutation,
                              mure_eval_stats *stats);

/* The expanded per-neuron patch of each GF / WS mutant, for checking the random
 * number streams: for mutant i and neuron slot q, F_l fp32 values at out +
 * offset[i] + q * F_l, where offset is returned in offsets [n_mutants] (-1 for other
 * operators).  GF: the noise added to each fan-in weight, fl32(sigma * n_f).  WS:
 * the permuted weights W[j][perm[f]].  out_len is the capacity of out (host);
 * Errors: INVALID_ARG (descriptors, or out too small), UNSUPPORTED (a tagged
 * descriptor), OOM, CUDA. */
mure_status mure_expand_patches(mure_model *model, const mure_mutant *table, int64_t n_mutants,
                                const int32_t *neuron_pool, int64_t pool_len, float *out, int64_t out_len,
                                int64_t *offsets);

/* mure_expand_patches without any device allocation.  The paper has no counterpart:
 * this entry point exists for callers that cannot allocate device memory, such as an
 * application whose own allocator has reserved the device's memory and cannot lend
 * it, or a latency-critical loop that forbids allocator calls because cudaMalloc and
 * cudaFree can synchronise the device.  It runs the same expansion kernel; the
 * kernel's scratch (job table, per-layer weight pointers, WS permutation buffers)
 * lives in one fixed device array of 8 MiB inside the library, which every GPU that
 * loads the library holds until the process exits.  The call allocates no device
 * memory.
 *   out_dev   device buffer of out_len floats receiving the patches (same layout and
 *             values as mure_expand_patches, i.e. GF noise and WS-permuted weights);
 *   offsets   host [n_mutants]: offset of each mutant's first slot in out_dev, -1 for
 *             operators without a patch.
 * The first call on a device that has work to do looks up the array's device address
 * with that device current (a failed lookup is retried by the next call).  The call
 * copies its job table from pageable host memory and waits for the context's stream,
 * so it must never be issued while that stream, or any stream of the device, is being
 * captured into a CUDA graph; it returns INVALID_ARG when it finds the context's stream
 * capturing.  Every call shares the one array: calls whose device work overlaps (on
 * different streams or host threads) race and must not be issued.  The kernel
 * initialises every scratch entry it reads, so nothing carries over from an earlier
 * call.  The call returns when the patches are in out_dev.  Errors: the descriptor
 * checks of mure_eval_mutants with their status codes; UNSUPPORTED for tagged
 * descriptors (as mure_expand_patches); INVALID_ARG for out_len too small (the needed
 * count in mure_last_error), for descriptors needing more than the 8 MiB of scratch
 * (the needed size in mure_last_error) and for a capturing stream; OOM when a host
 * allocation fails; CUDA. */
mure_status mure_expand_patches_noalloc(mure_model *model, const mure_mutant *table, int64_t n_mutants,
                                        const int32_t *neuron_pool, int64_t pool_len, float *out_dev,
                                        int64_t out_len, int64_t *offsets);

#ifdef __cplusplus
}
#endif
#endif /* MURE_H */
