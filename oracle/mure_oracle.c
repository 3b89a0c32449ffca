/*
 * mure_oracle.c -- plain, slow CPU oracle for memoized DNN mutation testing
 * (Ghanbari, Greenman, Tavakkol, Ahmed, "Provably Lossless Acceleration of DNN
 * Mutation Testing via Memoization", PACMSE/ISSTA 2026).
 *
 * TEST INFRASTRUCTURE ONLY.  The GPU library never includes, links or loads this
 * file; only the tests, the smoke check and the CPU-baseline leg of bench.py call
 * it.  It shares no header, helper or constant with the CUDA path.
 *
 * What it computes
 *   - a_v(x): the original network, node by node in topological order (Sec. 4,
 *     recursive activation definition).
 *   - b_v(x): a mutant M' built from scratch (its mutated layer's weights are
 *     materialised), run end to end: vanilla mutation testing (Sec. 5.1, baseline 1).
 *   - Algorithm 1 with Algorithms 2-4: dependence graph, memoization boundary K,
 *     clusters keyed by K, a memo table per cluster, chopped mutants run on memo
 *     rows.  Theorem 1 says its outputs equal the vanilla ones.
 *   - kill(mu,t), killingLabels and the DeepMutation-style mutation score (Sec. 5.2).
 *
 * Precision (the paper is silent; its models are Keras float32): every tensor is
 * stored in fp32; every dot product, sum and mean is accumulated in fp64 and rounded
 * to fp32 once.  Products of two fp32 values are exact in fp64.
 *
 * Readings of the paper used here:
 *   - neuron j of a weighted layer = output channel j (conv) / output unit j (dense)
 *     (Sec. 2.1: a conv filter's output channel is one neuron).
 *   - mutation operators (delegated by the paper to DeepMutation, Sec. 3.1):
 *       GF  : w[j][f] <- fl32(w[j][f] + fl32(sigma * n[j][f])), n ~ N(0,1),
 *             sigma = param * population std of the layer's weights (bias excluded)
 *       WS  : w[j][f] <- w[j][perm_j[f]], perm_j a Fisher-Yates shuffle
 *       NAI : w[j] <- -w[j], b[j] <- -b[j]   (negates the pre-activation exactly)
 *       NS  : swap (w[j0], b[j0]) with (w[j1], b[j1]) for each listed pair
 *       NEB : the output of neuron j is forced to 0 (after the layer's activation)
 *       IDENTITY : no change
 *   - recurrent models (Sec. 5.3: an embedding, two LSTM layers, a dense output): a
 *     neuron of an embedding is one output channel (a column of the table, no bias);
 *     a neuron of an LSTM layer is one unit, whose fan-in is the four gates' input and
 *     recurrent weights (4 (cin + units) values) and whose biases are the four gate
 *     biases.  The operators above act on these: NAI negates all of the unit's weights
 *     and biases, NS swaps two units' weights and biases, WS shuffles the unit's whole
 *     fan-in list, and NEB holds the unit's output h at 0 at every step (the
 *     recurrence sees the 0 too).
 *   - mutants over several layers (the paper's set mu(M') of mutated layers, Sec. 3.2;
 *     DeepMutation's model-wide selection): a "tagged" descriptor lists
 *     (layer << 20 | neuron) entries; the operator is applied to each listed neuron in
 *     its own layer (GF's sigma from that layer's weights, slot q of the list keeping
 *     its random stream), NS pairs lie in one layer, and the descriptor's layer is the
 *     smallest listed one (mmi).
 *   - random numbers: SplitMix64 (Steele, Lea, Flood, OOPSLA 2014) used as a
 *     counter-based generator; Gaussians by the Box-Muller transform in fp64.
 *   - argmax: lowest index wins ties; a NaN counts as the maximum.
 *
 * parity: every exported function is pinned by tests/test_oracle_*.py (closed forms,
 * library routines, brute force on tiny networks, published SplitMix64 outputs,
 * Theorem 1, identity mutants, score bounds).  Nothing here is "parity unpinned".
 */
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

/* ------------------------------------------------------------------ types -- */

enum { OR_CONV = 0, OR_DENSE = 1, OR_MAXPOOL = 2, OR_FLATTEN = 3, OR_ADD = 4,
       OR_GAP = 5, OR_SHORTCUT = 6, OR_DWCONV = 7, OR_EMBED = 8, OR_LSTM = 9 };
enum { OR_ACT_NONE = 0, OR_ACT_RELU = 1, OR_ACT_RELU6 = 2 };
enum { OR_OP_GF = 0, OR_OP_NEB = 1, OR_OP_NAI = 2, OR_OP_NS = 3, OR_OP_WS = 4,
       OR_OP_IDENTITY = 5 };
enum { OR_OK = 0, OR_EINVAL = 1, OR_EUNSUP = 2, OR_ENOMEM = 3 };

/* One node of the network DAG.  Inputs are node ids; -1 is the model input. */
typedef struct {
    int32_t kind, act, in0, in1;
    int32_t kh, kw, stride, pad; /* conv window / pool window / shortcut stride; LSTM: kh = 1 returns
                                    every step's output, kh = 0 only the last one */
    int32_t cin, cout;           /* conv & dense fan-in channels / outputs; shortcut channels;
                                    embedding: vocabulary size / width; LSTM: input features / units */
    const float *W;              /* conv [cout][kh][kw][cin], dense [cout][cin], depthwise conv [c][kh][kw],
                                    embedding [cout][cin] (neuron j = column j of the table),
                                    LSTM [cout][4][cin + cout] (unit j, gates i, f, g, o; input then
                                    recurrent weights) */
    const float *b;              /* [cout]; LSTM [cout][4]; embedding none */
} or_node;

typedef struct {
    int32_t in_h, in_w, in_c, n_classes, n_nodes;
    const or_node *nodes;
} or_model;

/* One mutant: first (and only) mutated weighted layer, operator, neuron ids. */
typedef struct {
    int32_t layer, op, n_neurons, tagged;   /* tagged: pool entries are (layer << 20 | neuron) */
    int64_t neuron_off; /* index into the neuron pool */
    float param;        /* GF: sigma multiplier */
    float reserved2;
    uint64_t seed;
} or_mutant;

typedef struct { int32_t h, w, c; } shape3;

/* ------------------------------------------------------- random numbers -- */

/* SplitMix64 output function (Steele, Lea, Flood 2014). */
static uint64_t sm64_mix(uint64_t z)
{
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
    return z ^ (z >> 31);
}

/* The i-th (0-based) output of a SplitMix64 generator whose state starts at seed:
 * the state advances by the golden-ratio increment before each output. */
uint64_t or_sm64(uint64_t seed, uint64_t i)
{
    return sm64_mix(seed + (i + 1) * 0x9E3779B97F4A7C15ULL);
}

/* Uniform double in (0, 1] from the top 53 bits of a draw. */
static double u01_open0(uint64_t x) { return (double)((x >> 11) + 1) * (1.0 / 9007199254740992.0); }

/* Stream of neuron slot q of a mutant: its own SplitMix64 seed. */
static uint64_t slot_seed(uint64_t mutant_seed, int q) { return or_sm64(mutant_seed, (uint64_t)q); }

/* Standard normal number f of a stream (Box-Muller, fp64): the pair (2p, 2p+1)
 * of uniforms gives r*cos(theta) for even f and r*sin(theta) for odd f. */
double or_gauss(uint64_t stream_seed, int64_t f)
{
    int64_t p = f >> 1;
    double u1 = u01_open0(or_sm64(stream_seed, (uint64_t)(2 * p)));
    double u2 = u01_open0(or_sm64(stream_seed, (uint64_t)(2 * p + 1)));
    double r = sqrt(-2.0 * log(u1));
    double th = 6.283185307179586476925286766559 * u2;
    return (f & 1) ? r * sin(th) : r * cos(th);
}

/* Fisher-Yates shuffle of 0..n-1 from a stream: for i = n-1 down to 1, draw
 * number (n-1-i) picks j = floor(u * (i+1)) with u in [0,1), clamped to i. */
void or_fisher_yates(uint64_t stream_seed, int32_t n, int32_t *perm)
{
    for (int32_t i = 0; i < n; ++i) perm[i] = i;
    for (int32_t i = n - 1; i >= 1; --i) {
        uint64_t x = or_sm64(stream_seed, (uint64_t)(n - 1 - i));
        double u = (double)(x >> 11) * (1.0 / 9007199254740992.0);
        int32_t j = (int32_t)(u * (double)(i + 1));
        if (j > i) j = i;
        int32_t t = perm[i]; perm[i] = perm[j]; perm[j] = t;
    }
}

/* ------------------------------------------------------------- shapes -- */

static int is_weighted(int kind)
{
    return kind == OR_CONV || kind == OR_DENSE || kind == OR_DWCONV || kind == OR_EMBED || kind == OR_LSTM;
}

/* Biases a neuron owns: an LSTM unit one per gate, an embedding none. */
static int n_bias(const or_node *nd) { return nd->kind == OR_LSTM ? 4 : nd->kind == OR_EMBED ? 0 : 1; }

/* Output shape of every node; returns OR_EINVAL for an inconsistent graph. */
int or_shapes(const or_model *m, int32_t *out_hwc /* [n_nodes][3] */)
{
    shape3 *s = (shape3 *)malloc(sizeof(shape3) * (size_t)(m->n_nodes > 0 ? m->n_nodes : 1));
    if (!s) return OR_ENOMEM;
    int rc = OR_OK;
    for (int v = 0; v < m->n_nodes && rc == OR_OK; ++v) {
        const or_node *nd = &m->nodes[v];
        if (nd->in0 < -1 || nd->in0 >= v) { rc = OR_EINVAL; break; }
        shape3 a = nd->in0 < 0 ? (shape3){m->in_h, m->in_w, m->in_c} : s[nd->in0];
        shape3 o = a;
        switch (nd->kind) {
        case OR_CONV:
            if (nd->cin != a.c || nd->stride < 1 || nd->kh < 1 || nd->kw < 1 || nd->pad < 0) { rc = OR_EINVAL; break; }
            o.h = (a.h + 2 * nd->pad - nd->kh) / nd->stride + 1;
            o.w = (a.w + 2 * nd->pad - nd->kw) / nd->stride + 1;
            o.c = nd->cout;
            if (o.h < 1 || o.w < 1) rc = OR_EINVAL;
            break;
        case OR_DWCONV:
            /* depthwise: one kh x kw filter per channel (MobileNetV2, Table 1) */
            if (nd->cin != a.c || nd->cout != a.c || nd->stride < 1 || nd->kh < 1 || nd->kw < 1 || nd->pad < 0) {
                rc = OR_EINVAL;
                break;
            }
            o.h = (a.h + 2 * nd->pad - nd->kh) / nd->stride + 1;
            o.w = (a.w + 2 * nd->pad - nd->kw) / nd->stride + 1;
            if (o.h < 1 || o.w < 1) rc = OR_EINVAL;
            break;
        case OR_DENSE:
            if (nd->cin != a.h * a.w * a.c) { rc = OR_EINVAL; break; }
            o.h = 1; o.w = 1; o.c = nd->cout;
            break;
        case OR_MAXPOOL:
            if (nd->kh < 1 || nd->kw < 1 || nd->stride < 1) { rc = OR_EINVAL; break; }
            o.h = (a.h - nd->kh) / nd->stride + 1;
            o.w = (a.w - nd->kw) / nd->stride + 1;
            if (o.h < 1 || o.w < 1) rc = OR_EINVAL;
            break;
        case OR_FLATTEN:
            o.h = 1; o.w = 1; o.c = a.h * a.w * a.c;
            break;
        case OR_ADD: {
            if (nd->in1 < -1 || nd->in1 >= v) { rc = OR_EINVAL; break; }
            shape3 b = nd->in1 < 0 ? (shape3){m->in_h, m->in_w, m->in_c} : s[nd->in1];
            if (a.h != b.h || a.w != b.w || a.c != b.c) rc = OR_EINVAL;
            break;
        }
        case OR_GAP:
            o.h = 1; o.w = 1; o.c = a.c;
            break;
        case OR_SHORTCUT:
            if (nd->stride < 1 || nd->cout < a.c) { rc = OR_EINVAL; break; }
            o.h = (a.h - 1) / nd->stride + 1;
            o.w = (a.w - 1) / nd->stride + 1;
            o.c = nd->cout;
            break;
        case OR_EMBED:
            /* token ids (one per position) from the model input to vectors of width cout */
            if (nd->in0 != -1 || a.c != 1 || nd->cin < 1 || nd->cout < 1 || nd->act != OR_ACT_NONE) {
                rc = OR_EINVAL;
                break;
            }
            o.c = nd->cout;
            break;
        case OR_LSTM:
            /* a sequence of a.w steps of a.c features */
            if (a.h != 1 || nd->cin != a.c || nd->cout < 1 || nd->cout > 4096 || (nd->kh != 0 && nd->kh != 1) ||
                nd->act != OR_ACT_NONE) {
                rc = OR_EINVAL;
                break;
            }
            o.w = nd->kh ? a.w : 1;
            o.c = nd->cout;
            break;
        default:
            rc = OR_EUNSUP;
        }
        s[v] = o;
    }
    if (rc == OR_OK && out_hwc)
        for (int v = 0; v < m->n_nodes; ++v) {
            out_hwc[3 * v] = s[v].h; out_hwc[3 * v + 1] = s[v].w; out_hwc[3 * v + 2] = s[v].c;
        }
    free(s);
    return rc;
}

/* --------------------------------------------------------- layer math -- */

static float act_f(int act, float v)
{
    if (act == OR_ACT_RELU) return v > 0.0f ? v : 0.0f;
    if (act == OR_ACT_RELU6) return v > 0.0f ? (v < 6.0f ? v : 6.0f) : 0.0f;
    return v;
}

/* Conv2d, NHWC, zero padding, fp64 accumulation, then the activation. */
static void conv_fwd(const or_node *nd, shape3 a, const float *x, shape3 o, const float *W,
                     const float *b, float *y)
{
    for (int oy = 0; oy < o.h; ++oy)
        for (int ox = 0; ox < o.w; ++ox)
            for (int co = 0; co < o.c; ++co) {
                double acc = (double)b[co];
                for (int ky = 0; ky < nd->kh; ++ky) {
                    int iy = oy * nd->stride - nd->pad + ky;
                    if (iy < 0 || iy >= a.h) continue;
                    for (int kx = 0; kx < nd->kw; ++kx) {
                        int ix = ox * nd->stride - nd->pad + kx;
                        if (ix < 0 || ix >= a.w) continue;
                        const float *xp = x + ((size_t)iy * a.w + ix) * a.c;
                        const float *wp = W + (((size_t)co * nd->kh + ky) * nd->kw + kx) * a.c;
                        for (int ci = 0; ci < a.c; ++ci) acc += (double)wp[ci] * (double)xp[ci];
                    }
                }
                y[((size_t)oy * o.w + ox) * o.c + co] = act_f(nd->act, (float)acc);
            }
}

/* Depthwise conv2d, NHWC: channel c is convolved with its own kh x kw filter. */
static void dwconv_fwd(const or_node *nd, shape3 a, const float *x, shape3 o, const float *W,
                       const float *b, float *y)
{
    for (int oy = 0; oy < o.h; ++oy)
        for (int ox = 0; ox < o.w; ++ox)
            for (int c = 0; c < o.c; ++c) {
                double acc = (double)b[c];
                for (int ky = 0; ky < nd->kh; ++ky) {
                    int iy = oy * nd->stride - nd->pad + ky;
                    if (iy < 0 || iy >= a.h) continue;
                    for (int kx = 0; kx < nd->kw; ++kx) {
                        int ix = ox * nd->stride - nd->pad + kx;
                        if (ix < 0 || ix >= a.w) continue;
                        acc += (double)W[((size_t)c * nd->kh + ky) * nd->kw + kx] *
                               (double)x[((size_t)iy * a.w + ix) * a.c + c];
                    }
                }
                y[((size_t)oy * o.w + ox) * o.c + c] = act_f(nd->act, (float)acc);
            }
}

/* Embedding lookup: position p holds token id x[p] (checked on entry), its output
 * channel j is W[j][x[p]]. */
static void embed_fwd(const or_node *nd, shape3 a, const float *x, const float *W, float *y)
{
    for (int p = 0; p < a.h * a.w; ++p) {
        int32_t tok = (int32_t)x[p];
        for (int j = 0; j < nd->cout; ++j) y[(size_t)p * nd->cout + j] = W[(size_t)j * nd->cin + tok];
    }
}

static double sigmoid64(double v) { return 1.0 / (1.0 + exp(-v)); }

/* LSTM with the Keras defaults (recurrent activation sigmoid, activation tanh), zero
 * initial state.  Per step t and unit j, with u = [x_t, h_{t-1}]:
 *   a_g = b[j][g] + sum_f W[j][g][f] u[f]   for the gates g = i, f, g, o
 *   i = sigma(a_i), f = sigma(a_f), g = tanh(a_g), o = sigma(a_o)
 *   c_t = f c_{t-1} + i g,   h_t = o tanh(c_t)
 * Every stored value (a, the gates, c, h) is fp32; each sum and product is formed in
 * fp64 and rounded once.  A blocked unit outputs h = 0 at every step, so the next
 * step's gates see 0 too. */
static void lstm_fwd(const or_node *nd, shape3 a, const float *x, const float *W, const float *b,
                     const uint8_t *blocked, float *y)
{
    const int T = a.w, F = nd->cin, H = nd->cout, U = F + H;
    float c[H], h[H], c2[H], h2[H];
    for (int j = 0; j < H; ++j) { c[j] = 0.0f; h[j] = 0.0f; }
    for (int t = 0; t < T; ++t) {
        const float *xt = x + (size_t)t * F;
        for (int j = 0; j < H; ++j) {
            float gate[4];
            for (int g = 0; g < 4; ++g) {
                const float *wp = W + ((size_t)j * 4 + g) * U;
                double acc = (double)b[4 * j + g];
                for (int f = 0; f < F; ++f) acc += (double)wp[f] * (double)xt[f];
                for (int k = 0; k < H; ++k) acc += (double)wp[F + k] * (double)h[k];
                float pre = (float)acc;
                gate[g] = g == 2 ? (float)tanh((double)pre) : (float)sigmoid64((double)pre);
            }
            c2[j] = (float)((double)gate[1] * (double)c[j] + (double)gate[0] * (double)gate[2]);
            h2[j] = blocked && blocked[j] ? 0.0f : (float)((double)gate[3] * tanh((double)c2[j]));
        }
        for (int j = 0; j < H; ++j) { c[j] = c2[j]; h[j] = h2[j]; }
        if (nd->kh) memcpy(y + (size_t)t * H, h, sizeof(float) * (size_t)H);
    }
    if (!nd->kh) memcpy(y, h, sizeof(float) * (size_t)H);
}

static void dense_fwd(const or_node *nd, const float *x, const float *W, const float *b, float *y)
{
    for (int o = 0; o < nd->cout; ++o) {
        double acc = (double)b[o];
        const float *wp = W + (size_t)o * nd->cin;
        for (int f = 0; f < nd->cin; ++f) acc += (double)wp[f] * (double)x[f];
        y[o] = act_f(nd->act, (float)acc);
    }
}

static void maxpool_fwd(const or_node *nd, shape3 a, const float *x, shape3 o, float *y)
{
    for (int oy = 0; oy < o.h; ++oy)
        for (int ox = 0; ox < o.w; ++ox)
            for (int c = 0; c < o.c; ++c) {
                float mx = x[((size_t)(oy * nd->stride) * a.w + ox * nd->stride) * a.c + c];
                for (int ky = 0; ky < nd->kh; ++ky)
                    for (int kx = 0; kx < nd->kw; ++kx) {
                        float v = x[((size_t)(oy * nd->stride + ky) * a.w + ox * nd->stride + kx) * a.c + c];
                        if (v > mx) mx = v;
                    }
                y[((size_t)oy * o.w + ox) * o.c + c] = mx;
            }
}

static void gap_fwd(shape3 a, const float *x, float *y)
{
    for (int c = 0; c < a.c; ++c) {
        double acc = 0.0;
        for (int p = 0; p < a.h * a.w; ++p) acc += (double)x[(size_t)p * a.c + c];
        y[c] = (float)(acc / (double)(a.h * a.w));
    }
}

/* Option-A shortcut: spatial subsampling by `stride`, zero channels appended. */
static void shortcut_fwd(const or_node *nd, shape3 a, const float *x, shape3 o, float *y)
{
    for (int oy = 0; oy < o.h; ++oy)
        for (int ox = 0; ox < o.w; ++ox)
            for (int c = 0; c < o.c; ++c)
                y[((size_t)oy * o.w + ox) * o.c + c] =
                    c < a.c ? x[((size_t)(oy * nd->stride) * a.w + ox * nd->stride) * a.c + c] : 0.0f;
}

/* Layer function Phi(v) (or Phi'(v) when W/b/blocked describe a mutated layer). */
static void node_fwd(const or_model *m, const shape3 *shp, int v, const float *in0, const float *in1,
                     const float *W, const float *b, const uint8_t *blocked, float *out)
{
    const or_node *nd = &m->nodes[v];
    shape3 a = nd->in0 < 0 ? (shape3){m->in_h, m->in_w, m->in_c} : shp[nd->in0];
    shape3 o = shp[v];
    size_t n = (size_t)o.h * o.w * o.c;
    switch (nd->kind) {
    case OR_CONV: conv_fwd(nd, a, in0, o, W, b, out); break;
    case OR_DWCONV: dwconv_fwd(nd, a, in0, o, W, b, out); break;
    case OR_DENSE: dense_fwd(nd, in0, W, b, out); break;
    case OR_MAXPOOL: maxpool_fwd(nd, a, in0, o, out); break;
    case OR_FLATTEN: memcpy(out, in0, n * sizeof(float)); break;
    case OR_ADD:
        for (size_t i = 0; i < n; ++i) out[i] = act_f(nd->act, (float)((double)in0[i] + (double)in1[i]));
        break;
    case OR_GAP: gap_fwd(a, in0, out); break;
    case OR_SHORTCUT: shortcut_fwd(nd, a, in0, o, out); break;
    case OR_EMBED: embed_fwd(nd, a, in0, W, out); break;
    case OR_LSTM: lstm_fwd(nd, a, in0, W, b, blocked, out); break;
    }
    if (blocked && is_weighted(nd->kind))
        for (size_t p = 0; p < (size_t)o.h * o.w; ++p)
            for (int c = 0; c < o.c; ++c)
                if (blocked[c]) out[p * o.c + c] = 0.0f;
}

/* Token ids fed to embedding node v: every value an integer in [0, vocabulary). */
static int check_tokens(const or_node *nd, const float *x, int64_t n)
{
    for (int64_t i = 0; i < n; ++i)
        if (!(x[i] >= 0.0f && x[i] < (float)nd->cin && x[i] == floorf(x[i]))) return OR_EINVAL;
    return OR_OK;
}

/* The model input checked against every embedding that reads it. */
static int check_input(const or_model *m, const float *X, int64_t n)
{
    int64_t per = (int64_t)m->in_h * m->in_w * m->in_c;
    for (int v = 0; v < m->n_nodes; ++v)
        if (m->nodes[v].kind == OR_EMBED && n > 0 && check_tokens(&m->nodes[v], X, n * per)) return OR_EINVAL;
    return OR_OK;
}

/* One node on one input, for pinning the layer functions against library routines. */
int or_node_forward(const or_model *m, int32_t v, const float *in0, const float *in1, float *out)
{
    if (!m || v < 0 || v >= m->n_nodes) return OR_EINVAL;
    shape3 *shp = (shape3 *)malloc(sizeof(shape3) * (size_t)m->n_nodes);
    if (!shp) return OR_ENOMEM;
    int rc = or_shapes(m, (int32_t *)shp);
    if (rc == OR_OK && m->nodes[v].kind == OR_EMBED)
        rc = check_tokens(&m->nodes[v], in0, (int64_t)m->in_h * m->in_w * m->in_c);
    if (rc == OR_OK) node_fwd(m, shp, v, in0, in1, m->nodes[v].W, m->nodes[v].b, NULL, out);
    free(shp);
    return rc;
}

/* ------------------------------------------------------------- mutants -- */

/* Node id of weighted layer `layer` (layers are the weighted nodes in node order). */
static int layer_node(const or_model *m, int layer)
{
    int l = 0;
    for (int v = 0; v < m->n_nodes; ++v)
        if (is_weighted(m->nodes[v].kind)) { if (l == layer) return v; ++l; }
    return -1;
}

int32_t or_n_layers(const or_model *m)
{
    int l = 0;
    for (int v = 0; v < m->n_nodes; ++v) l += is_weighted(m->nodes[v].kind);
    return l;
}

static int64_t fan_in(const or_node *nd)
{
    if (nd->kind == OR_CONV) return (int64_t)nd->kh * nd->kw * nd->cin;
    if (nd->kind == OR_DWCONV) return (int64_t)nd->kh * nd->kw;   /* a channel sees its own input channel */
    if (nd->kind == OR_LSTM) return 4 * ((int64_t)nd->cin + nd->cout);  /* four gates over [x_t, h_{t-1}] */
    return nd->cin;   /* dense; embedding: the neuron's column of the table */
}

/* Population standard deviation (ddof 0) of a layer's weights, two passes in fp64. */
double or_layer_std(const or_model *m, int32_t layer)
{
    int v = layer_node(m, layer);
    if (v < 0) return NAN;
    const or_node *nd = &m->nodes[v];
    int64_t n = fan_in(nd) * nd->cout;
    double mean = 0.0;
    for (int64_t i = 0; i < n; ++i) mean += (double)nd->W[i];
    mean /= (double)n;
    double ss = 0.0;
    for (int64_t i = 0; i < n; ++i) { double d = (double)nd->W[i] - mean; ss += d * d; }
    return sqrt(ss / (double)n);
}

/* Layer and neuron of pool entry e of a mutant. */
static int32_t entry_layer(const or_mutant *mu, int32_t e) { return mu->tagged ? (e >> 20) : mu->layer; }
static int32_t entry_neuron(const or_mutant *mu, int32_t e) { return mu->tagged ? (e & 0xFFFFF) : e; }

static int check_mutant(const or_model *m, const or_mutant *mu, const int32_t *pool, int64_t pool_len)
{
    int L = or_n_layers(m);
    if (mu->layer < 0 || mu->layer >= L) return OR_EINVAL;
    if (mu->op < OR_OP_GF || mu->op > OR_OP_IDENTITY) return OR_EINVAL;
    if (mu->tagged != 0 && mu->tagged != 1) return OR_EINVAL;
    if (mu->n_neurons < 0 || mu->neuron_off < 0 || mu->neuron_off + mu->n_neurons > pool_len) return OR_EINVAL;
    if (mu->op == OR_OP_NS && (mu->n_neurons & 1)) return OR_EINVAL;
    int32_t lmin = L;
    for (int q = 0; q < mu->n_neurons; ++q) {
        int32_t e = pool[mu->neuron_off + q];
        if (e < 0) return OR_EINVAL;
        int32_t l = entry_layer(mu, e), j = entry_neuron(mu, e);
        if (l < 0 || l >= L) return OR_EINVAL;
        if (j >= m->nodes[layer_node(m, l)].cout) return OR_EINVAL;
        if (l < lmin) lmin = l;
        for (int r = 0; r < q; ++r)
            if (pool[mu->neuron_off + r] == e) return OR_EINVAL;
        if (mu->op == OR_OP_NS && (q & 1) && entry_layer(mu, pool[mu->neuron_off + q - 1]) != l) return OR_EINVAL;
    }
    if (mu->tagged && mu->n_neurons > 0 && lmin != mu->layer) return OR_EINVAL;
    return OR_OK;
}

/* Whether mutant mu changes weighted layer `layer`. */
static int touches_layer(const or_mutant *mu, const int32_t *pool, int32_t layer)
{
    if (mu->op == OR_OP_IDENTITY) return 0;
    if (!mu->tagged) return layer == mu->layer;
    for (int q = 0; q < mu->n_neurons; ++q)
        if (entry_layer(mu, pool[mu->neuron_off + q]) == layer) return 1;
    return 0;
}

/* Materialise weighted layer `layer` of M': W_out/b_out receive a full copy of the
 * layer's parameters with the operator applied to the mutant's neurons in that
 * layer (slot q of the neuron list keeps random stream q); blocked_out[c] = 1 for
 * NEB neurons. */
int or_mutant_layer_at(const or_model *m, const or_mutant *mu, const int32_t *pool, int64_t pool_len,
                       int32_t layer, float *W_out, float *b_out, uint8_t *blocked_out)
{
    if (!m || !mu) return OR_EINVAL;
    int rc = check_mutant(m, mu, pool, pool_len);
    if (rc) return rc;
    if (layer < 0 || layer >= or_n_layers(m)) return OR_EINVAL;
    const or_node *nd = &m->nodes[layer_node(m, layer)];
    int64_t F = fan_in(nd);
    int nb = n_bias(nd);
    memcpy(W_out, nd->W, sizeof(float) * (size_t)(F * nd->cout));
    if (nb) memcpy(b_out, nd->b, sizeof(float) * (size_t)nb * nd->cout);
    memset(blocked_out, 0, (size_t)nd->cout);
    const int32_t *ent = pool + mu->neuron_off;
    /* slot q is in this layer: its neuron id, else -1 */
#define SLOT_J(q) (entry_layer(mu, ent[q]) == layer ? entry_neuron(mu, ent[q]) : -1)
    switch (mu->op) {
    case OR_OP_GF: {
        double sigma = (double)mu->param * or_layer_std(m, layer);
        for (int q = 0; q < mu->n_neurons; ++q) {
            if (SLOT_J(q) < 0) continue;
            uint64_t s = slot_seed(mu->seed, q);
            float *w = W_out + (size_t)SLOT_J(q) * F;
            for (int64_t f = 0; f < F; ++f) {
                float e = (float)(sigma * or_gauss(s, f));
                w[f] = w[f] + e;
            }
        }
        break;
    }
    case OR_OP_WS: {
        int32_t *perm = (int32_t *)malloc(sizeof(int32_t) * (size_t)F);
        if (!perm) return OR_ENOMEM;
        for (int q = 0; q < mu->n_neurons; ++q) {
            if (SLOT_J(q) < 0) continue;
            or_fisher_yates(slot_seed(mu->seed, q), (int32_t)F, perm);
            const float *src = nd->W + (size_t)SLOT_J(q) * F;
            float *w = W_out + (size_t)SLOT_J(q) * F;
            for (int64_t f = 0; f < F; ++f) w[f] = src[perm[f]];
        }
        free(perm);
        break;
    }
    case OR_OP_NAI:
        for (int q = 0; q < mu->n_neurons; ++q) {
            if (SLOT_J(q) < 0) continue;
            float *w = W_out + (size_t)SLOT_J(q) * F;
            for (int64_t f = 0; f < F; ++f) w[f] = -w[f];
            for (int g = 0; g < nb; ++g) b_out[nb * SLOT_J(q) + g] = -b_out[nb * SLOT_J(q) + g];
        }
        break;
    case OR_OP_NS:
        for (int q = 0; q + 1 < mu->n_neurons; q += 2) {
            if (SLOT_J(q) < 0) continue;   /* a pair lies in one layer */
            int j0 = SLOT_J(q), j1 = SLOT_J(q + 1);
            memcpy(W_out + (size_t)j0 * F, nd->W + (size_t)j1 * F, sizeof(float) * (size_t)F);
            memcpy(W_out + (size_t)j1 * F, nd->W + (size_t)j0 * F, sizeof(float) * (size_t)F);
            for (int g = 0; g < nb; ++g) {
                b_out[nb * j0 + g] = nd->b[nb * j1 + g];
                b_out[nb * j1 + g] = nd->b[nb * j0 + g];
            }
        }
        break;
    case OR_OP_NEB:
        for (int q = 0; q < mu->n_neurons; ++q)
            if (SLOT_J(q) >= 0) blocked_out[SLOT_J(q)] = 1;
        break;
    case OR_OP_IDENTITY:
        break;
    }
#undef SLOT_J
    return OR_OK;
}

/* The mutant's first mutated layer (mmi), materialised. */
int or_mutant_layer(const or_model *m, const or_mutant *mu, const int32_t *pool, int64_t pool_len,
                    float *W_out, float *b_out, uint8_t *blocked_out)
{
    if (!mu) return OR_EINVAL;
    return or_mutant_layer_at(m, mu, pool, pool_len, mu->layer, W_out, b_out, blocked_out);
}

/* ------------------------------------------------------------- forward -- */

typedef struct {
    const or_model *m;
    shape3 *shp;
    size_t *size;   /* elements per node output */
    float **buf;    /* per-node output buffers for one input */
    int n_layers;
    int *node_of_layer;
} fwd_ws;

static void ws_free(fwd_ws *w)
{
    if (w->buf) for (int v = 0; v < w->m->n_nodes; ++v) free(w->buf[v]);
    free(w->buf); free(w->shp); free(w->size); free(w->node_of_layer);
    memset(w, 0, sizeof(*w));
}

static int ws_init(fwd_ws *w, const or_model *m)
{
    memset(w, 0, sizeof(*w));
    w->m = m;
    int V = m->n_nodes;
    w->shp = (shape3 *)calloc((size_t)V, sizeof(shape3));
    w->size = (size_t *)calloc((size_t)V, sizeof(size_t));
    w->buf = (float **)calloc((size_t)V, sizeof(float *));
    w->node_of_layer = (int *)calloc((size_t)V + 1, sizeof(int));
    if (!w->shp || !w->size || !w->buf || !w->node_of_layer) { ws_free(w); return OR_ENOMEM; }
    int rc = or_shapes(m, (int32_t *)w->shp);
    if (rc) { ws_free(w); return rc; }
    for (int v = 0; v < V; ++v) {
        w->size[v] = (size_t)w->shp[v].h * w->shp[v].w * w->shp[v].c;
        w->buf[v] = (float *)malloc(sizeof(float) * w->size[v]);
        if (!w->buf[v]) { ws_free(w); return OR_ENOMEM; }
        if (is_weighted(m->nodes[v].kind)) w->node_of_layer[w->n_layers++] = v;
    }
    return OR_OK;
}

static const float *node_in(const fwd_ws *w, int id, const float *x) { return id < 0 ? x : w->buf[id]; }

/* Forward of the whole network on one input; node `mv` (or -1) uses the mutated
 * parameters (W, b, blocked).  Returns a pointer to the output node's buffer. */
static const float *forward_one(fwd_ws *w, const float *x, int mv, const float *W, const float *b,
                                const uint8_t *blocked)
{
    const or_model *m = w->m;
    for (int v = 0; v < m->n_nodes; ++v) {
        const or_node *nd = &m->nodes[v];
        const float *i0 = node_in(w, nd->in0, x);
        const float *i1 = nd->kind == OR_ADD ? node_in(w, nd->in1, x) : NULL;
        if (v == mv) node_fwd(m, w->shp, v, i0, i1, W, b, blocked, w->buf[v]);
        else node_fwd(m, w->shp, v, i0, i1, nd->W, nd->b, NULL, w->buf[v]);
    }
    return w->buf[m->n_nodes - 1];
}

/* The layers one mutant changes, materialised (buffers per weighted node, allocated
 * on first use and kept for the worker's later mutants). */
typedef struct {
    int V;
    float **W, **b;
    uint8_t **blk;
    uint8_t *on;    /* [V]: node v runs with the mutated parameters */
} mut_params;

static void mp_free(mut_params *p)
{
    if (p->W) for (int v = 0; v < p->V; ++v) { free(p->W[v]); free(p->b[v]); free(p->blk[v]); }
    free(p->W); free(p->b); free(p->blk); free(p->on);
    memset(p, 0, sizeof(*p));
}

static int mp_init(mut_params *p, const or_model *m)
{
    memset(p, 0, sizeof(*p));
    p->V = m->n_nodes;
    p->W = (float **)calloc((size_t)p->V, sizeof(float *));
    p->b = (float **)calloc((size_t)p->V, sizeof(float *));
    p->blk = (uint8_t **)calloc((size_t)p->V, sizeof(uint8_t *));
    p->on = (uint8_t *)calloc((size_t)p->V, 1);
    if (!p->W || !p->b || !p->blk || !p->on) { mp_free(p); return OR_ENOMEM; }
    return OR_OK;
}

static int mp_load(mut_params *p, const or_model *m, const or_mutant *mu, const int32_t *pool, int64_t pool_len)
{
    memset(p->on, 0, (size_t)p->V);
    int L = or_n_layers(m);
    for (int l = 0; l < L; ++l) {
        /* the first mutated layer is always materialised (an identity copy where the
         * operator changes nothing there) */
        if (l != mu->layer && !touches_layer(mu, pool, l)) continue;
        int v = layer_node(m, l);
        const or_node *nd = &m->nodes[v];
        if (!p->W[v]) {
            p->W[v] = (float *)malloc(sizeof(float) * (size_t)(fan_in(nd) * nd->cout));
            p->b[v] = (float *)malloc(sizeof(float) * (size_t)(n_bias(nd) ? n_bias(nd) : 1) * nd->cout);
            p->blk[v] = (uint8_t *)malloc((size_t)nd->cout);
            if (!p->W[v] || !p->b[v] || !p->blk[v]) return OR_ENOMEM;
        }
        int rc = or_mutant_layer_at(m, mu, pool, pool_len, l, p->W[v], p->b[v], p->blk[v]);
        if (rc) return rc;
        p->on[v] = 1;
    }
    return OR_OK;
}

/* Forward of the whole network on one input with the mutant's layers. */
static const float *forward_mut(fwd_ws *w, const float *x, const mut_params *p)
{
    const or_model *m = w->m;
    for (int v = 0; v < m->n_nodes; ++v) {
        const or_node *nd = &m->nodes[v];
        const float *i0 = node_in(w, nd->in0, x);
        const float *i1 = nd->kind == OR_ADD ? node_in(w, nd->in1, x) : NULL;
        if (p->on[v]) node_fwd(m, w->shp, v, i0, i1, p->W[v], p->b[v], p->blk[v], w->buf[v]);
        else node_fwd(m, w->shp, v, i0, i1, nd->W, nd->b, NULL, w->buf[v]);
    }
    return w->buf[m->n_nodes - 1];
}

static int argmax_f(const float *v, int n)
{
    int best = 0;
    for (int c = 1; c < n; ++c) {
        if (isnan(v[best])) break;
        if (isnan(v[c]) || v[c] > v[best]) best = c;
    }
    return best;
}

static int check_model(const or_model *m)
{
    if (!m || m->n_nodes < 1 || !m->nodes || m->n_classes < 1) return OR_EINVAL;
    int32_t *tmp = (int32_t *)malloc(sizeof(int32_t) * 3 * (size_t)m->n_nodes);
    if (!tmp) return OR_ENOMEM;
    int rc = or_shapes(m, tmp);
    int V = m->n_nodes;
    if (rc == OR_OK && tmp[3 * (V - 1)] * tmp[3 * (V - 1) + 1] * tmp[3 * (V - 1) + 2] != m->n_classes) rc = OR_EINVAL;
    free(tmp);
    return rc;
}

/* Original network on n inputs: logits [n][C] and predictions [n]. */
int or_forward(const or_model *m, const float *X, int64_t n, float *logits, int32_t *pred)
{
    int rc = check_model(m);
    if (rc) return rc;
    if (n > 0 && (rc = check_input(m, X, n))) return rc;
    fwd_ws w;
    if ((rc = ws_init(&w, m))) return rc;
    size_t in_sz = (size_t)m->in_h * m->in_w * m->in_c;
    for (int64_t t = 0; t < n; ++t) {
        const float *y = forward_one(&w, X + (size_t)t * in_sz, -1, NULL, NULL, NULL);
        if (logits) memcpy(logits + (size_t)t * m->n_classes, y, sizeof(float) * (size_t)m->n_classes);
        if (pred) pred[t] = argmax_f(y, m->n_classes);
    }
    ws_free(&w);
    return OR_OK;
}

/* Output of every node for one input, concatenated in node order (for pins). */
int or_forward_nodes(const or_model *m, const float *x, float *all_out)
{
    int rc = check_model(m);
    if (rc) return rc;
    if ((rc = check_input(m, x, 1))) return rc;
    fwd_ws w;
    if ((rc = ws_init(&w, m))) return rc;
    forward_one(&w, x, -1, NULL, NULL, NULL);
    size_t off = 0;
    for (int v = 0; v < m->n_nodes; ++v) { memcpy(all_out + off, w.buf[v], sizeof(float) * w.size[v]); off += w.size[v]; }
    ws_free(&w);
    return OR_OK;
}

/* ------------------------------------------------------ kill and score -- */

typedef struct {
    int64_t n_in, n_mut;
    int C;
    const int32_t *label;   /* [n_in] */
    const int32_t *pred0;   /* [n_in] */
} kill_ctx;

static void set_kill(uint64_t *row, int64_t t) { row[t >> 6] |= (uint64_t)1 << (t & 63); }

/* Sec. 5.2: kill(mu,t) <=> argmax m(t) = label(t) and argmax mu(t) != label(t). */
static int kill_pred(const kill_ctx *k, int64_t t, int pred) { return k->pred0[t] == k->label[t] && pred != k->label[t]; }

/* Mutation scores from a kill matrix: scoreA = killed fraction, scoreB = the
 * DeepMutation score sum_mu |killingLabels(mu)| / (|M| |L|). */
int or_scores(const uint64_t *kill_bits, int64_t n_mut, int64_t n_in, const int32_t *label, int32_t n_label_values,
              double *scoreA, double *scoreB, int64_t *killed_out /* nullable [n_mut] */)
{
    int64_t W = (n_in + 63) / 64;
    uint8_t *seen = (uint8_t *)calloc((size_t)(n_label_values > 0 ? n_label_values : 1), 1);
    uint8_t *lab = (uint8_t *)calloc((size_t)(n_label_values > 0 ? n_label_values : 1), 1);
    if (!seen || !lab) { free(seen); free(lab); return OR_ENOMEM; }
    int64_t nL = 0;
    for (int64_t t = 0; t < n_in; ++t) {
        if (label[t] < 0 || label[t] >= n_label_values) { free(seen); free(lab); return OR_EINVAL; }
        if (!lab[label[t]]) { lab[label[t]] = 1; ++nL; }
    }
    int64_t n_killed = 0, sum_labels = 0;
    for (int64_t i = 0; i < n_mut; ++i) {
        memset(seen, 0, (size_t)n_label_values);
        int64_t nk = 0, killed = 0;
        for (int64_t t = 0; t < n_in; ++t)
            if ((kill_bits[i * W + (t >> 6)] >> (t & 63)) & 1) {
                killed = 1;
                if (!seen[label[t]]) { seen[label[t]] = 1; ++nk; }
            }
        n_killed += killed;
        sum_labels += nk;
        if (killed_out) killed_out[i] = killed;
    }
    *scoreA = n_mut > 0 ? (double)n_killed / (double)n_mut : 0.0;
    *scoreB = (n_mut > 0 && nL > 0) ? (double)sum_labels / ((double)n_mut * (double)nL) : 0.0;
    free(seen); free(lab);
    return OR_OK;
}

/* --------------------------------------------------- vanilla (baseline) -- */

typedef struct {
    const or_model *m;
    const float *X;
    const or_mutant *mut;
    const int32_t *pool;
    int64_t pool_len;
    kill_ctx kc;
    float *logits;       /* nullable [n_mut][n_in][C] */
    uint64_t *kill_bits; /* [n_mut][W] */
    int64_t i0, i1;      /* mutant range of this worker */
    int rc;
} van_job;

static void *vanilla_worker(void *arg)
{
    van_job *j = (van_job *)arg;
    const or_model *m = j->m;
    fwd_ws w;
    mut_params mp;
    if ((j->rc = ws_init(&w, m))) return NULL;
    if ((j->rc = mp_init(&mp, m))) { ws_free(&w); return NULL; }
    size_t in_sz = (size_t)m->in_h * m->in_w * m->in_c;
    int64_t W64 = (j->kc.n_in + 63) / 64;
    for (int64_t i = j->i0; i < j->i1; ++i) {
        const or_mutant *mu = &j->mut[i];
        /* Build M' from scratch: its mutated layers' parameters are materialised. */
        if ((j->rc = mp_load(&mp, m, mu, j->pool, j->pool_len))) goto out;
        uint64_t *row = j->kill_bits + i * W64;
        memset(row, 0, sizeof(uint64_t) * (size_t)W64);
        for (int64_t t = 0; t < j->kc.n_in; ++t) {
            const float *y = forward_mut(&w, j->X + (size_t)t * in_sz, &mp);
            if (j->logits) memcpy(j->logits + ((size_t)i * j->kc.n_in + t) * m->n_classes, y, sizeof(float) * (size_t)m->n_classes);
            if (kill_pred(&j->kc, t, argmax_f(y, m->n_classes))) set_kill(row, t);
        }
    }
out:
    mp_free(&mp);
    ws_free(&w);
    return NULL;
}

static int run_workers(void *(*fn)(void *), void *jobs, size_t job_sz, int n_threads)
{
    pthread_t *th = (pthread_t *)malloc(sizeof(pthread_t) * (size_t)n_threads);
    uint8_t *ok = (uint8_t *)calloc((size_t)n_threads, 1);
    if (!th || !ok) { free(th); free(ok); return OR_ENOMEM; }
    for (int k = 1; k < n_threads; ++k)
        ok[k] = pthread_create(&th[k], NULL, fn, (char *)jobs + (size_t)k * job_sz) == 0;
    fn(jobs); /* worker 0 on the calling thread */
    /* a worker whose thread could not start runs here, serially */
    for (int k = 1; k < n_threads; ++k)
        if (!ok[k]) fn((char *)jobs + (size_t)k * job_sz);
    for (int k = 1; k < n_threads; ++k)
        if (ok[k]) pthread_join(th[k], NULL);
    free(th); free(ok);
    return OR_OK;
}

static int prepare_labels(const or_model *m, const float *X, int64_t n_in, const int32_t *labels,
                          int32_t **pred0_out, int32_t **label_out, float *orig_logits)
{
    int32_t *pred0 = (int32_t *)malloc(sizeof(int32_t) * (size_t)(n_in > 0 ? n_in : 1));
    int32_t *lab = (int32_t *)malloc(sizeof(int32_t) * (size_t)(n_in > 0 ? n_in : 1));
    if (!pred0 || !lab) { free(pred0); free(lab); return OR_ENOMEM; }
    int rc = or_forward(m, X, n_in, orig_logits, pred0);
    if (rc) { free(pred0); free(lab); return rc; }
    for (int64_t t = 0; t < n_in; ++t) {
        lab[t] = labels ? labels[t] : pred0[t];
        if (lab[t] < 0 || lab[t] >= m->n_classes) { free(pred0); free(lab); return OR_EINVAL; }
    }
    *pred0_out = pred0; *label_out = lab;
    return OR_OK;
}

/* Vanilla mutation testing: every mutant built from scratch and run end to end on
 * every input.  labels == NULL means label(t) = the original prediction.
 * Outputs: kill_bits [n_mut][ceil(n_in/64)] (bit t of row i = kill(mu_i, t), LSB
 * first), the two scores, and optionally all logits / the original logits. */
int or_vanilla(const or_model *m, const float *X, int64_t n_in, const int32_t *labels,
               const or_mutant *mut, int64_t n_mut, const int32_t *pool, int64_t pool_len, int32_t n_threads,
               float *logits, float *orig_logits, uint64_t *kill_bits, double *scoreA, double *scoreB)
{
    int rc = check_model(m);
    if (rc) return rc;
    if (n_in < 0 || n_mut < 0 || (n_mut > 0 && !mut) || !kill_bits || !scoreA || !scoreB) return OR_EINVAL;
    for (int64_t i = 0; i < n_mut; ++i)
        if ((rc = check_mutant(m, &mut[i], pool, pool_len))) return rc;
    int32_t *pred0 = NULL, *lab = NULL;
    if ((rc = prepare_labels(m, X, n_in, labels, &pred0, &lab, orig_logits))) return rc;
    if (n_threads < 1) n_threads = 1;
    if (n_threads > n_mut) n_threads = n_mut > 0 ? (int32_t)n_mut : 1;
    van_job *jobs = (van_job *)calloc((size_t)n_threads, sizeof(van_job));
    if (!jobs) { free(pred0); free(lab); return OR_ENOMEM; }
    for (int k = 0; k < n_threads; ++k) {
        jobs[k] = (van_job){m, X, mut, pool, pool_len, {n_in, n_mut, m->n_classes, lab, pred0}, logits, kill_bits,
                            n_mut * k / n_threads, n_mut * (k + 1) / n_threads, OR_OK};
    }
    rc = n_mut > 0 ? run_workers(vanilla_worker, jobs, sizeof(van_job), n_threads) : OR_OK;
    for (int k = 0; rc == OR_OK && k < n_threads; ++k) if (jobs[k].rc) rc = jobs[k].rc;
    if (rc == OR_OK) rc = or_scores(kill_bits, n_mut, n_in, lab, m->n_classes, scoreA, scoreB, NULL);
    free(jobs); free(pred0); free(lab);
    return rc;
}

/* --------------------------------------------------- unchanged rows -- */

/* Exact unchanged-row test (a reference for eliminating rows before their suffix): bit
 * (i, t) is set when, on input t, the output of every node that mutant i changes equals
 * the original network's output of that node bit for bit.  Then every later node, the
 * logits and the prediction are the original's too, so kill(i, t) = 0 without running
 * the suffix.  Bits as in the kill matrix: [n_mut][ceil(n_in/64)], LSB first. */
typedef struct {
    const or_model *m;
    const float *X;
    int64_t n_in;
    const or_mutant *mut;
    const int32_t *pool;
    int64_t pool_len;
    uint64_t *bits;
    int64_t i0, i1;
    int rc;
} unch_job;

static void *unchanged_worker(void *arg)
{
    unch_job *j = (unch_job *)arg;
    const or_model *m = j->m;
    fwd_ws w0, w1;
    mut_params mp;
    if ((j->rc = ws_init(&w0, m))) return NULL;
    if ((j->rc = ws_init(&w1, m))) { ws_free(&w0); return NULL; }
    if ((j->rc = mp_init(&mp, m))) { ws_free(&w0); ws_free(&w1); return NULL; }
    size_t in_sz = (size_t)m->in_h * m->in_w * m->in_c;
    int64_t W64 = (j->n_in + 63) / 64;
    for (int64_t i = j->i0; i < j->i1; ++i) {
        if ((j->rc = mp_load(&mp, m, &j->mut[i], j->pool, j->pool_len))) goto out;
        uint64_t *row = j->bits + i * W64;
        memset(row, 0, sizeof(uint64_t) * (size_t)W64);
        for (int64_t t = 0; t < j->n_in; ++t) {
            const float *x = j->X + (size_t)t * in_sz;
            forward_one(&w0, x, -1, NULL, NULL, NULL);
            forward_mut(&w1, x, &mp);
            int same = 1;
            for (int v = 0; v < m->n_nodes && same; ++v)
                if (mp.on[v] && memcmp(w0.buf[v], w1.buf[v], sizeof(float) * w0.size[v]) != 0) same = 0;
            if (same) set_kill(row, t);
        }
    }
out:
    mp_free(&mp);
    ws_free(&w0);
    ws_free(&w1);
    return NULL;
}

int or_unchanged_rows(const or_model *m, const float *X, int64_t n_in, const or_mutant *mut, int64_t n_mut,
                      const int32_t *pool, int64_t pool_len, int32_t n_threads, uint64_t *bits)
{
    int rc = check_model(m);
    if (rc) return rc;
    if (n_in < 0 || n_mut < 0 || (n_mut > 0 && !mut) || !bits) return OR_EINVAL;
    if (n_in > 0 && (rc = check_input(m, X, n_in))) return rc;
    for (int64_t i = 0; i < n_mut; ++i)
        if ((rc = check_mutant(m, &mut[i], pool, pool_len))) return rc;
    if (n_mut == 0) return OR_OK;
    if (n_threads < 1) n_threads = 1;
    if (n_threads > n_mut) n_threads = (int32_t)n_mut;
    unch_job *jobs = (unch_job *)calloc((size_t)n_threads, sizeof(unch_job));
    if (!jobs) return OR_ENOMEM;
    for (int k = 0; k < n_threads; ++k)
        jobs[k] = (unch_job){m, X, n_in, mut, pool, pool_len, bits, n_mut * k / n_threads,
                             n_mut * (k + 1) / n_threads, OR_OK};
    rc = run_workers(unchanged_worker, jobs, sizeof(unch_job), n_threads);
    for (int k = 0; rc == OR_OK && k < n_threads; ++k) if (jobs[k].rc) rc = jobs[k].rc;
    free(jobs);
    return rc;
}

/* ------------------------------------------- memoized (Algorithms 1-4) -- */

/* Algorithm 2: dg[v] = set of nodes v reads from (node ids; -1 = model input).
 * Stored as up to two entries per node (dg_n[v] of them). */
static void dep_graph(const or_model *m, int *dg, int *dg_n)
{
    for (int v = 0; v < m->n_nodes; ++v) {
        const or_node *nd = &m->nodes[v];
        dg_n[v] = 0;
        dg[2 * v + dg_n[v]++] = nd->in0;
        if (nd->kind == OR_ADD && nd->in1 != nd->in0) dg[2 * v + dg_n[v]++] = nd->in1;
    }
}

/* Memoization boundary of a mutant whose earliest mutated node is mmi (Alg. 1,
 * line 6; Sec. 4): the nodes p < mmi that some node v >= mmi reads.  Encoded as a
 * membership vector over ids -1..V-1 (index p+1). */
static void boundary(const or_model *m, const int *dg, const int *dg_n, int mmi, uint8_t *inK)
{
    memset(inK, 0, (size_t)m->n_nodes + 1);
    for (int v = mmi; v < m->n_nodes; ++v)
        for (int e = 0; e < dg_n[v]; ++e)
            if (dg[2 * v + e] < mmi) inK[dg[2 * v + e] + 1] = 1;
}

typedef struct {
    const or_model *m;
    const float *X;
    const or_mutant *mut;
    const int32_t *pool;
    int64_t pool_len;
    kill_ctx kc;
    const int *dg, *dg_n;
    const int64_t *ids;   /* mutant ids of this cluster */
    int64_t n_ids;
    const uint8_t *inK;
    float **MT;           /* memo table: MT[p+1] = [n_in][size(p)] for p in K */
    float *logits;
    uint64_t *kill_bits;
    int64_t k0, k1;
    int rc;
} memo_job;

/* Algorithm 4 + prediction on memo rows for the mutants ids[k0..k1). */
static void *memo_worker(void *arg)
{
    memo_job *j = (memo_job *)arg;
    const or_model *m = j->m;
    fwd_ws w;
    mut_params mp;
    if ((j->rc = ws_init(&w, m))) return NULL;
    if ((j->rc = mp_init(&mp, m))) { ws_free(&w); return NULL; }
    int64_t W64 = (j->kc.n_in + 63) / 64;
    size_t in_sz = (size_t)m->in_h * m->in_w * m->in_c;
    for (int64_t k = j->k0; k < j->k1; ++k) {
        int64_t id = j->ids[k];
        const or_mutant *mu = &j->mut[id];
        if ((j->rc = mp_load(&mp, m, mu, j->pool, j->pool_len))) goto out;
        int mmi = layer_node(m, mu->layer);
        uint64_t *row = j->kill_bits + id * W64;
        memset(row, 0, sizeof(uint64_t) * (size_t)W64);
        for (int64_t t = 0; t < j->kc.n_in; ++t) {
            /* chopped mutant: nodes mmi..V-1 (every mutated node is >= mmi), inputs
             * p < mmi from the memo table (the fresh input layers u_k), p >= mmi from
             * `past` (w.buf). */
            for (int v = mmi; v < m->n_nodes; ++v) {
                const or_node *nd = &m->nodes[v];
                const float *in[2] = {NULL, NULL};
                int srcs[2] = {nd->in0, nd->kind == OR_ADD ? nd->in1 : nd->in0};
                for (int e = 0; e < (nd->kind == OR_ADD ? 2 : 1); ++e) {
                    int p = srcs[e];
                    if (p < mmi) {
                        size_t sz = p < 0 ? in_sz : w.size[p];
                        in[e] = j->MT[p + 1] + (size_t)t * sz;
                    } else {
                        in[e] = w.buf[p];
                    }
                }
                if (mp.on[v]) node_fwd(m, w.shp, v, in[0], in[1], mp.W[v], mp.b[v], mp.blk[v], w.buf[v]);
                else node_fwd(m, w.shp, v, in[0], in[1], nd->W, nd->b, NULL, w.buf[v]);
            }
            const float *y = w.buf[m->n_nodes - 1];
            if (j->logits) memcpy(j->logits + ((size_t)id * j->kc.n_in + t) * m->n_classes, y, sizeof(float) * (size_t)m->n_classes);
            if (kill_pred(&j->kc, t, argmax_f(y, m->n_classes))) set_kill(row, t);
        }
    }
out:
    mp_free(&mp);
    ws_free(&w);
    return NULL;
}

/* Memoized mutation testing, Algorithm 1: clusters keyed by the boundary K, one
 * memo table per cluster (Algorithm 3: the original network's activations at K),
 * each mutant chopped at its earliest mutated node (Algorithm 4) and run on the
 * memo rows.  Same outputs as or_vanilla (Theorem 1).  n_clusters_out receives the
 * number of distinct K. */
int or_memo(const or_model *m, const float *X, int64_t n_in, const int32_t *labels,
            const or_mutant *mut, int64_t n_mut, const int32_t *pool, int64_t pool_len, int32_t n_threads,
            float *logits, uint64_t *kill_bits, double *scoreA, double *scoreB, int32_t *n_clusters_out)
{
    int rc = check_model(m);
    if (rc) return rc;
    if (n_in < 0 || n_mut < 0 || (n_mut > 0 && !mut) || !kill_bits || !scoreA || !scoreB) return OR_EINVAL;
    for (int64_t i = 0; i < n_mut; ++i)
        if ((rc = check_mutant(m, &mut[i], pool, pool_len))) return rc;
    int32_t *pred0 = NULL, *lab = NULL;
    if ((rc = prepare_labels(m, X, n_in, labels, &pred0, &lab, NULL))) return rc;
    int V = m->n_nodes;
    int *dg = (int *)malloc(sizeof(int) * 2 * (size_t)V), *dg_n = (int *)malloc(sizeof(int) * (size_t)V);
    uint8_t *keys = (uint8_t *)calloc((size_t)(n_mut > 0 ? n_mut : 1) * ((size_t)V + 1), 1);
    int64_t *cl_of = (int64_t *)malloc(sizeof(int64_t) * (size_t)(n_mut > 0 ? n_mut : 1));
    int64_t *ids = (int64_t *)malloc(sizeof(int64_t) * (size_t)(n_mut > 0 ? n_mut : 1));
    float **MT = (float **)calloc((size_t)V + 1, sizeof(float *));
    fwd_ws w;
    int have_ws = 0;
    if (!dg || !dg_n || !keys || !cl_of || !ids || !MT) { rc = OR_ENOMEM; goto done; }
    if ((rc = ws_init(&w, m))) goto done;
    have_ws = 1;
    dep_graph(m, dg, dg_n);                                   /* Alg. 1 line 2 */
    /* Alg. 1 lines 3-9: cluster ids by K. */
    int64_t n_cl = 0;
    for (int64_t i = 0; i < n_mut; ++i) {
        uint8_t *k = keys + (size_t)i * ((size_t)V + 1);
        boundary(m, dg, dg_n, layer_node(m, mut[i].layer), k);
        int64_t c = -1;
        for (int64_t i2 = 0; i2 < i && c < 0; ++i2)
            if (memcmp(keys + (size_t)i2 * ((size_t)V + 1), k, (size_t)V + 1) == 0) c = cl_of[i2];
        cl_of[i] = c >= 0 ? c : n_cl++;
    }
    if (n_clusters_out) *n_clusters_out = (int32_t)n_cl;
    size_t in_sz = (size_t)m->in_h * m->in_w * m->in_c;
    if (n_threads < 1) n_threads = 1;
    for (int64_t c = 0; c < n_cl && rc == OR_OK; ++c) {
        int64_t n_ids = 0;
        for (int64_t i = 0; i < n_mut; ++i) if (cl_of[i] == c) ids[n_ids++] = i;
        const uint8_t *inK = keys + (size_t)ids[0] * ((size_t)V + 1);
        /* Alg. 3 + Alg. 1 lines 11-12: instrument at K, predict on X -> memo table. */
        for (int p = -1; p < V; ++p) {
            if (!inK[p + 1]) continue;
            size_t sz = p < 0 ? in_sz : w.size[p];
            MT[p + 1] = (float *)malloc(sizeof(float) * sz * (size_t)(n_in > 0 ? n_in : 1));
            if (!MT[p + 1]) { rc = OR_ENOMEM; break; }
        }
        for (int64_t t = 0; rc == OR_OK && t < n_in; ++t) {
            const float *x = X + (size_t)t * in_sz;
            forward_one(&w, x, -1, NULL, NULL, NULL);
            for (int p = -1; p < V; ++p)
                if (inK[p + 1]) {
                    size_t sz = p < 0 ? in_sz : w.size[p];
                    memcpy(MT[p + 1] + (size_t)t * sz, p < 0 ? x : w.buf[p], sizeof(float) * sz);
                }
        }
        /* Alg. 1 lines 13-17: chop and predict every mutant of the cluster. */
        if (rc == OR_OK && n_ids > 0) {
            int nt = n_threads > n_ids ? (int)n_ids : n_threads;
            memo_job *jobs = (memo_job *)calloc((size_t)nt, sizeof(memo_job));
            if (!jobs) rc = OR_ENOMEM;
            for (int k = 0; rc == OR_OK && k < nt; ++k)
                jobs[k] = (memo_job){m, X, mut, pool, pool_len, {n_in, n_mut, m->n_classes, lab, pred0}, dg, dg_n,
                                     ids, n_ids, inK, MT, logits, kill_bits, n_ids * k / nt, n_ids * (k + 1) / nt, OR_OK};
            if (rc == OR_OK) rc = run_workers(memo_worker, jobs, sizeof(memo_job), nt);
            for (int k = 0; rc == OR_OK && k < nt; ++k) if (jobs[k].rc) rc = jobs[k].rc;
            free(jobs);
        }
        for (int p = 0; p <= V; ++p) { free(MT[p]); MT[p] = NULL; }
    }
    if (rc == OR_OK) rc = or_scores(kill_bits, n_mut, n_in, lab, m->n_classes, scoreA, scoreB, NULL);
done:
    if (have_ws) ws_free(&w);
    if (MT) for (int p = 0; p <= V; ++p) free(MT[p]);
    free(MT); free(dg); free(dg_n); free(keys); free(cl_of); free(ids); free(pred0); free(lab);
    return rc;
}

/* Analytic multiply-accumulate count of one node on one input (cost model,
 * axioms C1-C3 of Sec. 4.2): conv/dense MACs; every other node costs 0. */
int64_t or_node_macs(const or_model *m, int32_t v)
{
    int32_t *s = (int32_t *)malloc(sizeof(int32_t) * 3 * (size_t)m->n_nodes);
    if (!s || or_shapes(m, s)) { free(s); return -1; }
    const or_node *nd = &m->nodes[v];
    int64_t r = 0;
    if (nd->kind == OR_CONV) r = (int64_t)s[3 * v] * s[3 * v + 1] * nd->cout * nd->kh * nd->kw * nd->cin;
    else if (nd->kind == OR_DWCONV) r = (int64_t)s[3 * v] * s[3 * v + 1] * nd->cout * nd->kh * nd->kw;
    else if (nd->kind == OR_DENSE) r = (int64_t)nd->cin * nd->cout;
    else if (nd->kind == OR_LSTM)   /* steps x units x four gates x [x_t, h_{t-1}] */
        r = (int64_t)(nd->in0 < 0 ? m->in_w : s[3 * nd->in0 + 1]) * nd->cout * 4 * (nd->cin + nd->cout);
    free(s);
    return r;
}

/* Boundary K of a mutant at weighted layer `layer` as a 0/1 vector over node ids
 * -1..V-1 (entry p+1), for the structural checks of Alg. 1 line 6. */
int or_boundary(const or_model *m, int32_t layer, uint8_t *inK)
{
    int mmi = layer_node(m, layer);
    if (mmi < 0) return OR_EINVAL;
    int *dg = (int *)malloc(sizeof(int) * 2 * (size_t)m->n_nodes), *dg_n = (int *)malloc(sizeof(int) * (size_t)m->n_nodes);
    if (!dg || !dg_n) { free(dg); free(dg_n); return OR_ENOMEM; }
    dep_graph(m, dg, dg_n);
    boundary(m, dg, dg_n, mmi, inK);
    free(dg); free(dg_n);
    return OR_OK;
}
