// C ABI of the library: contexts, model compilation (graph -> stages), the prefix
// activation cache, and the memoized / vanilla mutation-testing schedulers.
#include <algorithm>
#include <cstdarg>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <numeric>

#include "common.cuh"
#include "device_util.cuh"

using namespace mure;

namespace {

// Mutants per batch the input tile is sized for (MURE_BATCH_MUTANTS overrides; at least 1).
int64_t batch_mutants()
{
    static int64_t v = 0;
    if (!v) {
        const char *e = getenv("MURE_BATCH_MUTANTS");
        v = e && atoi(e) > 0 ? atoi(e) : 16;
    }
    return v;
}

// MURE_TC_CONV: in the tensor-core modes the LeNet-size convolution runs in the
// small-image mode (a GEMM row per pooling window); "0" keeps its CUDA-core kernel,
// "generic" runs it through the implicit-GEMM producers (one row per position).
// Stride-1 convolutions with input channels a multiple of 32 take the staged mode
// (each tile's input rows staged in shared memory by tensor-map copies); "gather"
// keeps them on the producers' per-row gathers from device memory.
std::string tc_conv_env()
{
    const char *e = getenv("MURE_TC_CONV");
    return e ? e : "";
}

// ------------------------------------------------------------------ plumbing --

struct Fail {
    mure_status st;
};

void set_err(mure_ctx *c, const char *fmt, ...) __attribute__((format(printf, 2, 3)));
void set_err(mure_ctx *c, const char *fmt, ...)
{
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    if (c) c->err = buf;
}

#define FAILIF(cond, ctx, status, ...)        \
    do {                                      \
        if (cond) {                           \
            set_err(ctx, __VA_ARGS__);        \
            throw Fail{status};               \
        }                                     \
    } while (0)

#define CK(ctx, call)                                                                              \
    do {                                                                                           \
        cudaError_t e_ = (call);                                                                   \
        FAILIF(e_ != cudaSuccess, ctx, MURE_ERR_CUDA, "%s: %s", #call, cudaGetErrorString(e_));    \
    } while (0)

void *dalloc(mure_ctx *c, size_t bytes)
{
    if (bytes == 0) bytes = 16;
    void *p = nullptr;
    if (c->has_alloc) {
        p = c->alloc.alloc(bytes, (void *)c->stream, c->alloc.user);
    } else {
        if (cudaMallocAsync(&p, bytes, c->stream) != cudaSuccess) {
            cudaGetLastError();
            p = nullptr;
        }
    }
    FAILIF(!p, c, MURE_ERR_OOM, "device allocation of %zu bytes failed", bytes);
    return p;
}

void dfree(mure_ctx *c, void *p)
{
    if (!p) return;
    if (c->has_alloc) c->alloc.free(p, (void *)c->stream, c->alloc.user);
    else cudaFreeAsync(p, c->stream);
}

// Device allocations owned by one call (freed on every exit path).
struct Scratch {
    mure_ctx *c;
    std::vector<void *> ptrs;
    explicit Scratch(mure_ctx *ctx) : c(ctx) {}
    template <class T>
    T *get(size_t n)
    {
        void *p = dalloc(c, n * sizeof(T));
        ptrs.push_back(p);
        return static_cast<T *>(p);
    }
    ~Scratch()
    {
        for (void *p : ptrs) dfree(c, p);
    }
};

int64_t round_up(int64_t n, int64_t a) { return (n + a - 1) / a * a; }

template <class F>
mure_status run(mure_ctx *c, F &&fn)
{
    if (c) c->err.clear();
    try {
        fn();
    } catch (const Fail &f) {
        return f.st;
    } catch (const std::bad_alloc &) {
        set_err(c, "host allocation failed");
        return MURE_ERR_OOM;
    }
    return MURE_OK;
}

void check_launch(mure_ctx *c)
{
    cudaError_t e = cudaGetLastError();
    FAILIF(e != cudaSuccess, c, MURE_ERR_CUDA, "kernel launch: %s", cudaGetErrorString(e));
}

// Optional per-launch device timing: a pair of events around each launch, summed
// per class (a layer's kernels, delta, gather, epilogue) once the stream is idle.
struct KTimer {
    mure_ctx *c;
    bool on;
    struct Rec {
        int cls;
        cudaEvent_t a, b;
    };
    std::vector<Rec> recs;
    KTimer(mure_ctx *ctx, bool enabled) : c(ctx), on(enabled) {}
    cudaEvent_t ev(size_t i)
    {
        while (c->evpool.size() <= i) {
            cudaEvent_t e;
            CK(c, cudaEventCreate(&e));
            c->evpool.push_back(e);
        }
        return c->evpool[i];
    }
    void begin(int cls)
    {
        if (!on) return;
        Rec r{cls, ev(2 * recs.size()), ev(2 * recs.size() + 1)};
        CK(c, cudaEventRecord(r.a, c->stream));
        recs.push_back(r);
    }
    void end()
    {
        if (on) CK(c, cudaEventRecord(recs.back().b, c->stream));
    }
    // after the stream is idle
    void collect(std::vector<double> &ms)
    {
        for (const Rec &r : recs) {
            float t = 0;
            CK(c, cudaEventElapsedTime(&t, r.a, r.b));
            if (r.cls >= 0 && r.cls < (int)ms.size()) ms[r.cls] += t;
        }
    }
};

// ---------------------------------------------------------- model compilation --

struct Shape {
    int h, w, c;
};

bool weighted(int k)
{
    return k == MURE_NODE_CONV2D || k == MURE_NODE_DENSE || k == MURE_NODE_DWCONV || k == MURE_NODE_EMBED ||
           k == MURE_NODE_LSTM;
}

// Output shapes of all nodes (same rules as the network definition in the header).
std::vector<Shape> node_shapes(mure_ctx *c, const mure_model_desc *d)
{
    std::vector<Shape> s(d->n_nodes);
    const Shape in{d->in_h, d->in_w, d->in_c};
    for (int v = 0; v < d->n_nodes; ++v) {
        const mure_node &n = d->nodes[v];
        FAILIF(n.in0 < -1 || n.in0 >= v, c, MURE_ERR_INVALID_ARG, "node %d: input %d is not an earlier node", v, n.in0);
        const Shape a = n.in0 < 0 ? in : s[n.in0];
        Shape o = a;
        switch (n.kind) {
        case MURE_NODE_CONV2D:
            FAILIF(n.cin != a.c || n.stride < 1 || n.kh < 1 || n.kw < 1 || n.pad < 0 || n.cout < 1, c,
                   MURE_ERR_INVALID_ARG, "node %d: bad conv geometry", v);
            o = {(a.h + 2 * n.pad - n.kh) / n.stride + 1, (a.w + 2 * n.pad - n.kw) / n.stride + 1, n.cout};
            FAILIF(o.h < 1 || o.w < 1, c, MURE_ERR_INVALID_ARG, "node %d: empty conv output", v);
            FAILIF(!n.W || !n.b, c, MURE_ERR_INVALID_ARG, "node %d: NULL weights", v);
            break;
        case MURE_NODE_DWCONV:
            FAILIF(n.cin != a.c || n.cout != a.c || n.stride < 1 || n.kh < 1 || n.kw < 1 || n.pad < 0, c,
                   MURE_ERR_INVALID_ARG, "node %d: bad depthwise geometry", v);
            o = {(a.h + 2 * n.pad - n.kh) / n.stride + 1, (a.w + 2 * n.pad - n.kw) / n.stride + 1, a.c};
            FAILIF(o.h < 1 || o.w < 1, c, MURE_ERR_INVALID_ARG, "node %d: empty depthwise output", v);
            FAILIF(!n.W || !n.b, c, MURE_ERR_INVALID_ARG, "node %d: NULL weights", v);
            break;
        case MURE_NODE_EMBED:
            FAILIF(a.h != 1 || a.c != 1 || n.cin < 1 || n.cout < 1, c, MURE_ERR_INVALID_ARG,
                   "node %d: an embedding reads a 1 x T x 1 sequence of ids", v);
            FAILIF(!n.W, c, MURE_ERR_INVALID_ARG, "node %d: NULL weights", v);
            o = {1, a.w, n.cout};
            break;
        case MURE_NODE_LSTM:
            FAILIF(a.h != 1 || n.cin != a.c || n.cout < 1 || (n.kh != 0 && n.kh != 1), c, MURE_ERR_INVALID_ARG,
                   "node %d: bad LSTM geometry", v);
            FAILIF(!n.W || !n.b, c, MURE_ERR_INVALID_ARG, "node %d: NULL weights", v);
            o = {1, n.kh ? a.w : 1, n.cout};
            break;
        case MURE_NODE_DENSE:
            FAILIF(n.cin != a.h * a.w * a.c || n.cout < 1, c, MURE_ERR_INVALID_ARG, "node %d: dense fan-in mismatch", v);
            FAILIF(!n.W || !n.b, c, MURE_ERR_INVALID_ARG, "node %d: NULL weights", v);
            o = {1, 1, n.cout};
            break;
        case MURE_NODE_MAXPOOL2D:
            FAILIF(n.kh < 1 || n.kw < 1 || n.stride < 1, c, MURE_ERR_INVALID_ARG, "node %d: bad pool", v);
            o = {(a.h - n.kh) / n.stride + 1, (a.w - n.kw) / n.stride + 1, a.c};
            FAILIF(o.h < 1 || o.w < 1, c, MURE_ERR_INVALID_ARG, "node %d: empty pool output", v);
            break;
        case MURE_NODE_FLATTEN:
            o = {1, 1, a.h * a.w * a.c};
            break;
        case MURE_NODE_ADD: {
            FAILIF(n.in1 < -1 || n.in1 >= v, c, MURE_ERR_INVALID_ARG, "node %d: bad second input", v);
            const Shape b = n.in1 < 0 ? in : s[n.in1];
            FAILIF(a.h != b.h || a.w != b.w || a.c != b.c, c, MURE_ERR_INVALID_ARG, "node %d: add shape mismatch", v);
            break;
        }
        case MURE_NODE_GAP:
            o = {1, 1, a.c};
            break;
        case MURE_NODE_SHORTCUT:
            FAILIF(n.stride < 1 || n.cout < a.c, c, MURE_ERR_INVALID_ARG, "node %d: bad shortcut", v);
            o = {(a.h - 1) / n.stride + 1, (a.w - 1) / n.stride + 1, n.cout};
            break;
        default:
            FAILIF(true, c, MURE_ERR_INVALID_ARG, "node %d: unknown kind %d", v, n.kind);
        }
        FAILIF(n.act != MURE_ACT_NONE && n.act != MURE_ACT_RELU && n.act != MURE_ACT_RELU6, c, MURE_ERR_INVALID_ARG,
               "node %d: bad activation", v);
        s[v] = o;
    }
    return s;
}

TensorDim tdim(Shape s)
{
    TensorDim t{s.h, s.w, s.c, (int64_t)s.h * s.w * s.c, 0};
    t.stride = round4(t.size);
    return t;
}

// Group the graph into stages: weighted node + its tail of ADD / MAXPOOL / FLATTEN
// / GAP up to the next weighted node (the dependence graph of Algorithm 2 read off
// the nodes' inputs).
void compile(mure_ctx *c, const mure_model_desc *d, mure_model *m)
{
    const std::vector<Shape> shp = node_shapes(c, d);
    const Shape in{d->in_h, d->in_w, d->in_c};
    auto shape_of = [&](int id) { return id < 0 ? in : shp[id]; };
    std::vector<int> wn;
    for (int v = 0; v < d->n_nodes; ++v)
        if (weighted(d->nodes[v].kind)) wn.push_back(v);
    FAILIF(wn.empty(), c, MURE_ERR_INVALID_ARG, "the network has no weighted node");
    FAILIF(wn.back() != d->n_nodes - 1, c, MURE_ERR_UNSUPPORTED, "the output node must be the last weighted node");
    const int L = (int)wn.size();
    const Shape outs = shp[d->n_nodes - 1];
    FAILIF(outs.h * outs.w * outs.c != d->n_classes, c, MURE_ERR_INVALID_ARG, "output size %d != n_classes %d",
           outs.h * outs.w * outs.c, d->n_classes);
    FAILIF(d->n_classes > kMaxClasses || d->n_classes < 1, c, MURE_ERR_UNSUPPORTED, "n_classes must be 1..%d",
           kMaxClasses);
    // stage_in[s] = node whose output is x_s (-1 = the network input)
    std::vector<int> stage_in(L + 1, -2);
    stage_in[0] = -1;
    std::vector<char> used(d->n_nodes, 0);
    m->st.resize(L);
    m->xd.resize(L + 1);
    m->zd.resize(L);
    m->xd[0] = tdim(in);
    for (int v = 0; v < L; ++v) {
        const int nid = wn[v];
        const mure_node &n = d->nodes[nid];
        // a weighted node reads the previous stage's output x_v, or an earlier stage input
        // x_s: a projection in a residual block's skip branch (Algorithm 2's graph is
        // then not a chain), whose add must take x_v (checked below)
        int in_src = -1;
        for (int s2 = 0; s2 <= v; ++s2)
            if (stage_in[s2] == n.in0) in_src = s2;
        FAILIF(in_src < 0, c, MURE_ERR_UNSUPPORTED, "weighted node %d does not read a stage input", nid);
        used[nid] = 1;
        Stage &S = m->st[v];
        S = Stage{};
        S.kind = n.kind;
        S.in_src = in_src;
        const Shape a = shape_of(n.in0), z = shp[nid];
        if (n.kind == MURE_NODE_CONV2D || n.kind == MURE_NODE_DWCONV) {
            S.ih = a.h; S.iw = a.w; S.ic = a.c; S.kh = n.kh; S.kw = n.kw; S.stride = n.stride; S.pad = n.pad;
        } else if (n.kind == MURE_NODE_EMBED || n.kind == MURE_NODE_LSTM) {
            // sequences: iw = T steps, ic = the input width (1 for the ids); kh = the
            // LSTM's every-step flag
            S.ih = 1; S.iw = a.w; S.ic = a.c; S.kh = n.kh; S.kw = 1; S.stride = 1; S.pad = 0;
        } else {
            S.ih = 1; S.iw = 1; S.ic = n.cin; S.kh = 1; S.kw = 1; S.stride = 1; S.pad = 0;
        }
        S.oh = z.h; S.ow = z.w; S.oc = z.c;
        // a depthwise neuron's fan-in is its own channel's filter; an embedding channel's
        // its table entries; an LSTM unit's its four gates' input and recurrent weights
        S.K = n.kind == MURE_NODE_DWCONV ? S.kh * S.kw
              : n.kind == MURE_NODE_EMBED ? n.cin
              : n.kind == MURE_NODE_LSTM  ? 4 * (S.ic + S.oc)
                                          : S.kh * S.kw * S.ic;
        S.vocab = n.kind == MURE_NODE_EMBED ? n.cin : 0;
        S.act1 = n.act;
        S.skip_src = -1; S.sc_stride = 1; S.sc_c = 0; S.sk_w = 0;
        S.macs = n.kind == MURE_NODE_EMBED ? 0
                 : n.kind == MURE_NODE_LSTM  ? (int64_t)S.iw * S.oc * S.K
                                             : (int64_t)S.oh * S.ow * S.oc * S.K;
        m->zd[v] = tdim(z);
        int cur = nid;
        const int end = v + 1 < L ? wn[v + 1] : d->n_nodes;
        int phase = 0;  // 0: before ADD, 1: after ADD, 2: after pool, 3: after gap
        for (int u = nid + 1; u < end; ++u) {
            const mure_node &t = d->nodes[u];
            if (t.kind == MURE_NODE_SHORTCUT) continue;  // a side branch, checked by its ADD
            FAILIF(v + 1 == L, c, MURE_ERR_UNSUPPORTED, "nodes after the output layer");
            used[u] = 1;
            if (t.kind == MURE_NODE_ADD) {
                FAILIF(phase != 0 || (t.in0 != cur && t.in1 != cur), c, MURE_ERR_UNSUPPORTED,
                       "node %d: unsupported add placement", u);
                int other = t.in0 == cur ? t.in1 : t.in0;
                int sc_stride = 1;
                if (other >= 0 && d->nodes[other].kind == MURE_NODE_SHORTCUT) {
                    used[other] = 1;
                    sc_stride = d->nodes[other].stride;
                    other = d->nodes[other].in0;
                }
                int src = -1;
                for (int s2 = 0; s2 <= v; ++s2)
                    if (stage_in[s2] == other) src = s2;
                FAILIF(src < 0, c, MURE_ERR_UNSUPPORTED, "node %d: skip input is not a stage input", u);
                S.has_add = 1; S.skip_src = src; S.sc_stride = sc_stride;
                S.sc_c = m->xd[src].c; S.sk_w = m->xd[src].w;
                S.act2 = t.act;
                phase = 1;
            } else if (t.kind == MURE_NODE_MAXPOOL2D) {
                FAILIF(t.in0 != cur || phase > 1 || t.kh != 2 || t.kw != 2 || t.stride != 2, c, MURE_ERR_UNSUPPORTED,
                       "node %d: only one 2x2 stride-2 max pool per stage", u);
                FAILIF(t.act != MURE_ACT_NONE, c, MURE_ERR_UNSUPPORTED, "node %d: activation on a pool", u);
                S.pool = 1;
                phase = 2;
            } else if (t.kind == MURE_NODE_FLATTEN) {
                FAILIF(t.in0 != cur, c, MURE_ERR_UNSUPPORTED, "node %d: flatten off the chain", u);
            } else if (t.kind == MURE_NODE_GAP) {
                FAILIF(t.in0 != cur || phase > 2, c, MURE_ERR_UNSUPPORTED, "node %d: unsupported gap", u);
                FAILIF(t.act != MURE_ACT_NONE, c, MURE_ERR_UNSUPPORTED, "node %d: activation on a gap", u);
                S.gap = 1;
                phase = 3;
            } else {
                FAILIF(true, c, MURE_ERR_UNSUPPORTED, "node %d: unsupported node in a stage tail", u);
            }
            cur = u;
        }
        FAILIF(S.kind == MURE_NODE_DWCONV && (S.has_add || S.pool || S.gap), c, MURE_ERR_UNSUPPORTED,
               "depthwise node %d: only an activation may follow it in its stage", nid);
        FAILIF((S.kind == MURE_NODE_EMBED || S.kind == MURE_NODE_LSTM) && (S.has_add || S.pool || S.gap || n.act), c,
               MURE_ERR_UNSUPPORTED, "recurrent node %d: no activation, add or pooling in its stage", nid);
        FAILIF(S.kind == MURE_NODE_EMBED && v != 0, c, MURE_ERR_UNSUPPORTED, "embedding node %d: only as the first layer",
               nid);
        FAILIF((S.kind == MURE_NODE_EMBED || S.kind == MURE_NODE_LSTM) && !recurrent_supported(S), c,
               MURE_ERR_UNSUPPORTED, "LSTM node %d: at most 64 units and 128 inputs", nid);
        FAILIF(S.in_src != v && !(S.has_add && S.skip_src == v && S.sc_stride == 1), c, MURE_ERR_UNSUPPORTED,
               "weighted node %d reads an earlier stage input but its add does not take the previous stage", nid);
        const Shape y = shp[cur];
        S.yh = y.h; S.yw = y.w; S.yc = y.c;
        stage_in[v + 1] = cur;
        m->xd[v + 1] = tdim(y);
        FAILIF(S.yc != S.oc && !S.gap && !(S.yh == 1 && S.yw == 1), c, MURE_ERR_UNSUPPORTED, "stage %d channels", v);
    }
    for (int u = 0; u < d->n_nodes; ++u)
        FAILIF(!used[u], c, MURE_ERR_UNSUPPORTED, "node %d is not part of a supported stage", u);
    m->L = L;
    m->n_classes = d->n_classes;
}

// --------------------------------------------------------------- descriptors --

struct Groups {
    std::vector<int32_t> order;       // mutant ids grouped by layer (stable)
    std::vector<int64_t> begin;       // [L+1] group boundaries in `order`
};

void check_table(mure_ctx *c, const mure_model *m, const mure_mutant *t, int64_t n, const int32_t *pool,
                 int64_t pool_len)
{
    FAILIF(n < 0 || pool_len < 0, c, MURE_ERR_INVALID_ARG, "negative sizes");
    FAILIF(n > 0 && !t, c, MURE_ERR_INVALID_ARG, "NULL mutant table");
    FAILIF(pool_len > 0 && !pool, c, MURE_ERR_INVALID_ARG, "NULL neuron pool");
    FAILIF(n > INT32_MAX, c, MURE_ERR_UNSUPPORTED, "more than 2^31 mutants");
    bool recurrent = false;
    for (int v = 0; v < m->L; ++v) recurrent |= m->st[v].kind == MURE_NODE_EMBED || m->st[v].kind == MURE_NODE_LSTM;
    std::vector<int64_t> seen;
    for (int64_t i = 0; i < n; ++i) {
        const mure_mutant &u = t[i];
        FAILIF(u.layer < 0 || u.layer >= m->L, c, MURE_ERR_INVALID_ARG, "mutant %lld: layer %d out of range",
               (long long)i, u.layer);
        FAILIF(u.op < MURE_OP_GF || u.op > MURE_OP_IDENTITY, c, MURE_ERR_INVALID_ARG, "mutant %lld: bad op", (long long)i);
        FAILIF((u.tagged != 0 && u.tagged != 1) || u.reserved2 != 0.f, c, MURE_ERR_INVALID_ARG,
               "mutant %lld: reserved fields", (long long)i);
        FAILIF(u.n_neurons < 0 || u.neuron_off < 0 || u.neuron_off + u.n_neurons > pool_len, c, MURE_ERR_INVALID_ARG,
               "mutant %lld: neuron range outside the pool", (long long)i);
        FAILIF(u.op == MURE_OP_NS && (u.n_neurons & 1), c, MURE_ERR_INVALID_ARG, "mutant %lld: odd NS neuron count",
               (long long)i);
        seen.assign(pool + u.neuron_off, pool + u.neuron_off + u.n_neurons);
        int lmin = m->L;
        for (int64_t q = 0; q < u.n_neurons; ++q) {
            const int32_t e = seen[q];
            const int l = u.tagged ? (e < 0 ? -1 : e >> 20) : u.layer, j = u.tagged ? (e & 0xFFFFF) : e;
            FAILIF(e < 0 || l < 0 || l >= m->L || j >= m->st[l].oc, c, MURE_ERR_INVALID_ARG,
                   "mutant %lld: neuron entry %lld out of range", (long long)i, (long long)e);
            FAILIF(u.op == MURE_OP_NS && (q & 1) && (u.tagged ? seen[q - 1] >> 20 : u.layer) != l, c,
                   MURE_ERR_INVALID_ARG, "mutant %lld: an NS pair across two layers", (long long)i);
            lmin = std::min(lmin, l);
        }
        FAILIF(u.tagged && recurrent, c, MURE_ERR_UNSUPPORTED,
               "mutant %lld: mutants over several layers of a recurrent network", (long long)i);
        FAILIF(u.tagged && u.n_neurons > 0 && lmin != u.layer, c, MURE_ERR_INVALID_ARG,
               "mutant %lld: layer %d is not its smallest listed layer %d", (long long)i, u.layer, lmin);
        std::sort(seen.begin(), seen.end());
        FAILIF(std::adjacent_find(seen.begin(), seen.end()) != seen.end(), c, MURE_ERR_INVALID_ARG,
               "mutant %lld: repeated neuron", (long long)i);
    }
}

Groups group_by_layer(const mure_model *m, const mure_mutant *t, int64_t n, const int32_t *pool)
{
    Groups g;
    g.begin.assign(m->L + 1, 0);
    for (int64_t i = 0; i < n; ++i) g.begin[t[i].layer + 1]++;
    for (int l = 0; l < m->L; ++l) g.begin[l + 1] += g.begin[l];
    std::vector<int64_t> pos(g.begin.begin(), g.begin.end() - 1);
    g.order.resize(n);
    for (int64_t i = 0; i < n; ++i) g.order[pos[t[i].layer]++] = (int32_t)i;
    // inside a group, tagged mutants by the set of later layers they change (stable):
    // batches then share their later mutated layers, single-layer mutants keep the
    // fused paths, and a batch without mutated tail layers keeps the fused output layer
    // (a mutant's bits never depend on its batch)
    std::vector<uint64_t> key(n, 0);
    bool any = false;
    for (int64_t i = 0; i < n; ++i) {
        const mure_mutant &u = t[i];
        if (!u.tagged || u.op == MURE_OP_IDENTITY) continue;
        for (int q = 0; q < u.n_neurons; ++q) {
            const int v = pool[u.neuron_off + q] >> 20;
            if (v > u.layer && v < 64) key[i] |= 1ull << v;
        }
        any |= key[i] != 0;
    }
    if (any)
        for (int l = 0; l < m->L; ++l)
            std::stable_sort(g.order.begin() + g.begin[l], g.order.begin() + g.begin[l + 1],
                             [&](int32_t a, int32_t b) { return key[a] < key[b]; });
    return g;
}

// Descriptor arrays in group order, uploaded to the device in one copy.
struct DevTable {
    int32_t *op, *nn, *ids, *mid;
    int64_t *noff, *poff;
    float *patch;
    int64_t n_jobs, patch_len;
    std::vector<int> kmax_layer;
    std::vector<int64_t> dot_prefix;   // [n+1] prefix sums of GF/WS neuron slots (group order)
    int32_t *dslot = nullptr;          // [dot_prefix[n]] GF/WS slots in group order: (group, slot q)
    std::vector<int64_t> val_prefix;   // [n+1] prefix sums of NEB/NAI/NS neuron slots (group order)
    std::vector<int64_t> copy_prefix;  // [n+1] the same for NEB/NS alone
    int4 *vslot = nullptr;             // [val_prefix[n]] those slots: (group, q, source channel, op)
    int expand_launches = 0;
    // tagged mutants with neurons in layers after their first: per layer v, per
    // mutant (group order) the count, the offset into ids and the GF / WS patch offset
    // of its neurons in v (0 / -1 where it has none)
    bool has_later = false;
    int64_t n = 0;
    std::vector<std::vector<int32_t>> nn_at_host;   // [L][n]
    int32_t *nn_at = nullptr;                       // [L][n]
    int64_t *noff_at = nullptr, *poff_at = nullptr; // [L][n]
};

DevTable upload_table(mure_ctx *c, Scratch &sc, const mure_model *m, const mure_mutant *t, int64_t n,
                      const int32_t *pool, int64_t pool_len, const Groups &g, int ws_as_weights, float *patch_out,
                      int64_t *ids_from_group)
{
    DevTable dt{};
    const int L = m->L;
    dt.n = n;
    std::vector<int32_t> op(n), nn(n), mid(n);
    std::vector<int64_t> noff(n), poff(n, -1);
    std::vector<SlotJob> jobs;
    // the neuron ids of each mutant, decoded and grouped by layer: its first layer's
    // segment, then one segment per later layer (tagged descriptors), each in pool order
    std::vector<int32_t> ids;
    ids.reserve((size_t)pool_len);
    std::vector<std::vector<int64_t>> noff_at, poff_at;
    int64_t plen = 0, perm_len = 0;
    for (int64_t k = 0; k < n; ++k) {
        const int32_t i = g.order[k];
        const mure_mutant &u = t[i];
        op[k] = u.op;
        mid[k] = i;
        const bool patched = u.op == MURE_OP_GF || u.op == MURE_OP_WS;
        auto layer_of = [&](int q) { return u.tagged ? pool[u.neuron_off + q] >> 20 : u.layer; };
        auto neuron_of = [&](int q) { return u.tagged ? pool[u.neuron_off + q] & 0xFFFFF : pool[u.neuron_off + q]; };
        // segment of layer v: ids, and the patches of GF / WS (slot q keeps stream q)
        auto segment = [&](int v, int64_t &seg_off, int64_t &seg_poff) {
            seg_off = (int64_t)ids.size();
            const int F = m->st[v].K;
            int cnt = 0;
            for (int q = 0; q < u.n_neurons; ++q) {
                if (layer_of(q) != v) continue;
                ids.push_back(neuron_of(q));
                if (patched) {
                    SlotJob jb{};
                    jb.layer = v; jb.op = u.op; jb.F = F; jb.j = neuron_of(q); jb.q = q;
                    jb.param = u.param; jb.seed = u.seed;
                    jb.out_off = plen + (int64_t)cnt * F;
                    jb.perm_off = perm_len;
                    if (u.op == MURE_OP_WS) perm_len += F;
                    jobs.push_back(jb);
                }
                ++cnt;
            }
            seg_poff = patched && cnt > 0 ? plen : -1;
            if (patched) plen += (int64_t)cnt * F;
            return cnt;
        };
        int64_t so = 0, sp = -1;
        const int c0 = segment(u.layer, so, sp);
        nn[k] = u.op == MURE_OP_IDENTITY ? 0 : c0;
        noff[k] = so;
        poff[k] = sp;
        if (u.tagged) {
            for (int v = u.layer + 1; v < L; ++v) {
                int64_t vo = 0, vp = -1;
                const int cv = segment(v, vo, vp);
                if (cv == 0 || u.op == MURE_OP_IDENTITY) continue;
                if (!dt.has_later) {
                    dt.has_later = true;
                    dt.nn_at_host.assign(L, std::vector<int32_t>(n, 0));
                    noff_at.assign(L, std::vector<int64_t>(n, 0));
                    poff_at.assign(L, std::vector<int64_t>(n, -1));
                }
                dt.nn_at_host[v][k] = cv;
                noff_at[v][k] = vo;
                poff_at[v][k] = vp;
            }
        }
        if (ids_from_group) ids_from_group[i] = poff[k];
    }
    dt.n_jobs = (int64_t)jobs.size();
    dt.patch_len = plen;
    dt.dot_prefix.assign(n + 1, 0);
    for (int64_t k = 0; k < n; ++k)
        dt.dot_prefix[k + 1] = dt.dot_prefix[k] + ((op[k] == MURE_OP_GF || op[k] == MURE_OP_WS) ? nn[k] : 0);
    std::vector<int32_t> dslot;
    dslot.reserve(2 * dt.dot_prefix[n]);
    for (int64_t k = 0; k < n; ++k)
        if (op[k] == MURE_OP_GF || op[k] == MURE_OP_WS)
            for (int q = 0; q < nn[k]; ++q) { dslot.push_back((int32_t)k); dslot.push_back(q); }
    // the operators without a fan-in sum: NS reads its partner neuron's channel
    dt.val_prefix.assign(n + 1, 0);
    dt.copy_prefix.assign(n + 1, 0);
    std::vector<int4> vslot;
    for (int64_t k = 0; k < n; ++k) {
        const bool val = op[k] == MURE_OP_NEB || op[k] == MURE_OP_NAI || op[k] == MURE_OP_NS;
        dt.val_prefix[k + 1] = dt.val_prefix[k] + (val ? nn[k] : 0);
        dt.copy_prefix[k + 1] = dt.copy_prefix[k] + ((op[k] == MURE_OP_NEB || op[k] == MURE_OP_NS) ? nn[k] : 0);
        if (val)
            for (int q = 0; q < nn[k]; ++q)
                vslot.push_back(make_int4((int)k, q, ids[noff[k] + (op[k] == MURE_OP_NS ? (q ^ 1) : q)], op[k]));
    }
    // one staging buffer, one H2D copy
    const size_t b_op = n * 4, b_nn = n * 4, b_mid = n * 4, b_noff = n * 8, b_poff = n * 8;
    const size_t b_dslot = std::max<size_t>(dslot.size(), 1) * 4, b_vslot = std::max<size_t>(vslot.size(), 1) * 16;
    const size_t b_ids = std::max<size_t>(ids.size(), 1) * 4, b_jobs = jobs.size() * sizeof(SlotJob);
    const size_t b_later = dt.has_later ? (size_t)L * n : 0;
    size_t off = 0;
    auto place = [&](size_t b) { size_t o = off; off = round_up(off + b, 256); return o; };
    const size_t o_op = place(b_op), o_nn = place(b_nn), o_mid = place(b_mid), o_noff = place(b_noff),
                 o_poff = place(b_poff), o_ids = place(b_ids), o_jobs = place(b_jobs), o_dslot = place(b_dslot),
                 o_vslot = place(b_vslot), o_nnat = place(b_later * 4), o_noffat = place(b_later * 8),
                 o_poffat = place(b_later * 8);
    std::vector<char> host(off);
    memcpy(host.data() + o_op, op.data(), b_op);
    memcpy(host.data() + o_nn, nn.data(), b_nn);
    memcpy(host.data() + o_mid, mid.data(), b_mid);
    memcpy(host.data() + o_noff, noff.data(), b_noff);
    memcpy(host.data() + o_poff, poff.data(), b_poff);
    if (!ids.empty()) memcpy(host.data() + o_ids, ids.data(), ids.size() * 4);
    if (dt.has_later)
        for (int v = 0; v < L; ++v) {
            memcpy(host.data() + o_nnat + (size_t)v * n * 4, dt.nn_at_host[v].data(), (size_t)n * 4);
            memcpy(host.data() + o_noffat + (size_t)v * n * 8, noff_at[v].data(), (size_t)n * 8);
            memcpy(host.data() + o_poffat + (size_t)v * n * 8, poff_at[v].data(), (size_t)n * 8);
        }
    if (!jobs.empty()) memcpy(host.data() + o_jobs, jobs.data(), b_jobs);
    if (!dslot.empty()) memcpy(host.data() + o_dslot, dslot.data(), dslot.size() * 4);
    if (!vslot.empty()) memcpy(host.data() + o_vslot, vslot.data(), vslot.size() * 16);
    char *dev = sc.get<char>(off);
    CK(c, cudaMemcpyAsync(dev, host.data(), off, cudaMemcpyHostToDevice, c->stream));
    dt.op = (int32_t *)(dev + o_op);
    dt.nn = (int32_t *)(dev + o_nn);
    dt.mid = (int32_t *)(dev + o_mid);
    dt.noff = (int64_t *)(dev + o_noff);
    dt.poff = (int64_t *)(dev + o_poff);
    dt.ids = (int32_t *)(dev + o_ids);
    dt.dslot = (int32_t *)(dev + o_dslot);
    dt.vslot = (int4 *)(dev + o_vslot);
    if (dt.has_later) {
        dt.nn_at = (int32_t *)(dev + o_nnat);
        dt.noff_at = (int64_t *)(dev + o_noffat);
        dt.poff_at = (int64_t *)(dev + o_poffat);
    }
    dt.patch = plen ? sc.get<float>(plen) : nullptr;
    if (!jobs.empty()) {
        std::vector<const float *> Wp(m->L);
        for (int l = 0; l < m->L; ++l) Wp[l] = m->st[l].W;
        const float **Wd = sc.get<const float *>(m->L);
        CK(c, cudaMemcpyAsync(Wd, Wp.data(), m->L * sizeof(float *), cudaMemcpyHostToDevice, c->stream));
        ExpandArgs ea{};
        ea.jobs = (const SlotJob *)(dev + o_jobs);
        ea.n_jobs = dt.n_jobs;
        ea.sigma = m->sigma_dev;
        ea.W = Wd;
        ea.patch = dt.patch;
        ea.perm = perm_len ? sc.get<int32_t>(perm_len) : nullptr;
        ea.ws_as_weights = ws_as_weights;
        dt.expand_launches = launch_expand(ea, c->stream);
        check_launch(c);
        if (patch_out) CK(c, cudaMemcpyAsync(patch_out, dt.patch, plen * 4, cudaMemcpyDeviceToHost, c->stream));
    }
    // the largest neuron count per layer bounds the delta kernel's warps per row
    dt.kmax_layer.assign(m->L, 0);
    for (int l = 0; l < m->L; ++l) {
        int km = 0;
        for (int64_t k = g.begin[l]; k < g.begin[l + 1]; ++k) km = std::max(km, nn[k]);
        dt.kmax_layer[l] = km;
    }
    return dt;
}

// ---------------------------------------------------------------- evaluation --

struct EvalCfg {
    int64_t words32;
    uint32_t *kill32;
    unsigned long long *counters;   // [3]: killed, label-count sum, near ties
    float *logits_out;              // device or null
    bool skip_unchanged = false;    // memoized: drop rows whose x_{l+1} equals the original
};

// Per-row buffers of one batch: x_s for s in [s_lo, L], plus z (vanilla) and the
// global-average-pooling map.
struct Workspace {
    std::vector<float *> xb;   // [L+1]
    float *patch = nullptr;    // [rows][kmax * cells] mutated-channel values
    float *zb = nullptr;
    int64_t z_stride = 0;
    float *gap_tmp = nullptr;
    int64_t rows = 0;
    TcDeltaWs dw;              // tensor-core delta scratch (GF / WS slots of a batch)
    // unchanged-row elimination: per-row flags, per-block counts, the compacted row
    // list and its length
    int32_t *uflags = nullptr, *ublk = nullptr, *lrow = nullptr, *ucount = nullptr;
};

int64_t gap_map_stride(const Stage &S)
{
    const int mh = S.pool ? S.oh / 2 : S.oh, mw = S.pool ? S.ow / 2 : S.ow;
    return round4((int64_t)mh * mw * S.oc);
}

// Bytes per batch row for a group at layer l (vanilla: every stage input from 1,
// plus z_l).
int64_t row_bytes(const mure_model *m, int l, bool vanilla, bool z_rows = false)
{
    int64_t b = 0;
    for (int s = vanilla ? 1 : l + 1; s <= m->L; ++s) b += m->xd[s].stride;
    if (z_rows) {
        int64_t zs = 0;
        for (int v = 0; v < m->L; ++v) zs = std::max(zs, m->zd[v].stride);
        b += zs;
    } else if (vanilla) {
        b += m->zd[l].stride;
    }
    const Stage &S = m->st[l];
    b += (int64_t)S.oc * (S.gap ? 1 : (S.pool ? (S.oh / 2) * (S.ow / 2) : S.oh * S.ow));  // patch values (bound)
    int64_t g = 0;
    for (int v = vanilla ? 0 : l + 1; v < m->L; ++v)
        if (m->st[v].gap) g = std::max(g, gap_map_stride(m->st[v]));
    return (b + g) * 4;
}

void alloc_workspace(mure_ctx *c, Scratch &sc, const mure_model *m, int64_t rows, bool vanilla, int lmin,
                     int64_t patch_floats, int delta_slots, int delta_k, Workspace &ws, bool z_rows = false)
{
    ws.rows = rows;
    if (delta_slots > 0) {
        int64_t nf = 0, ni = 0;
        tc_delta_ws_size(delta_slots, delta_k, nf, ni);
        const int64_t Np = (delta_slots + 127) / 128 * 128;
        float *f = sc.get<float>(nf);
        ws.dw.filt = f;
        ws.dw.swz = f + Np * delta_k;
        ws.dw.colb = ws.dw.swz + 2 * Np * round_up32(delta_k);
        int32_t *ip = sc.get<int32_t>(ni);
        ws.dw.colg = ip;
        ws.dw.colq = ip + Np;
        ws.dw.colj = ip + 2 * Np;
        ws.dw.n_max = delta_slots;
        ws.dw.k_max = delta_k;
    }
    ws.patch = sc.get<float>(rows * std::max<int64_t>(patch_floats, 1));
    ws.xb.assign(m->L + 1, nullptr);
    for (int s = vanilla ? 1 : lmin + 1; s <= m->L; ++s) ws.xb[s] = sc.get<float>(rows * m->xd[s].stride);
    if (vanilla || z_rows) {
        int64_t zs = 0;
        for (int l = 0; l < m->L; ++l) zs = std::max(zs, m->zd[l].stride);
        ws.z_stride = zs;
        ws.zb = sc.get<float>(rows * zs);
    }
    int64_t g = 0;
    for (int v = 0; v < m->L; ++v)
        if (m->st[v].gap) g = std::max(g, gap_map_stride(m->st[v]));
    if (g) ws.gap_tmp = sc.get<float>(rows * g);
}

// One batch: G mutants of group l (starting at group position g0) x an input tile.
struct Acct {
    int64_t flops = 0;
    std::vector<int64_t> flops_cls, launches_cls;   // [L + 3]
    int64_t bytes_gather = 0;
    int64_t bytes_rows = 0;
    int64_t bytes_values = 0;
    int64_t rows_unchanged = 0;
};

int run_batch(mure_ctx *c, const mure_model *m, const mure_cache *ca, const DevTable &dt, const EvalCfg &ec,
              const Workspace &ws, int l, int64_t g0, RowMap rm, bool vanilla, Acct &acct, KTimer &tm)
{
    cudaStream_t s = c->stream;
    const int L = m->L;
    const int C_DELTA = L, C_VALS = L + 1, C_EPI = L + 2;
    int launches = 0;
    auto timed = [&](int cls, int64_t fl, auto &&launch) {
        tm.begin(cls);
        const int n = launch();
        tm.end();
        launches += n;
        acct.launches_cls[cls] += n;
        acct.flops_cls[cls] += fl;
        acct.flops += fl;
    };
    PatchArgs pa{dt.op + g0, dt.nn + g0, dt.noff + g0, dt.ids, dt.poff + g0, dt.patch};
    pa.dslot = dt.dslot + 2 * dt.dot_prefix[g0];
    pa.n_dslot = dt.dot_prefix[g0 + rm.R / rm.T] - dt.dot_prefix[g0];
    pa.dslot_g0 = (int32_t)g0;
    pa.vslot = dt.vslot + dt.val_prefix[g0];
    pa.n_vslot = dt.val_prefix[g0 + rm.R / rm.T] - dt.val_prefix[g0];
    FinalArgs fa{};
    fa.mutant_id = dt.mid + g0;
    fa.label = ca->label;
    fa.pred0 = ca->pred0;
    fa.n_in = ca->n_in;
    fa.kill32 = ec.kill32;
    fa.words32 = ec.words32;
    fa.logits_out = ec.logits_out;
    fa.near_ties = ec.counters + 2;
    fa.mode = 0;
    const Src net_in{ca->x[0], m->xd[0].stride, 1};
    // where row r finds stage input x_s: memo reads unmutated tensors (s <= l) from
    // the cache; vanilla recomputes everything except the network input.
    auto xsrc = [&](int s2) -> Src {
        if (s2 == 0) return net_in;
        if (!vanilla && s2 <= l) return Src{ca->x[s2], m->xd[s2].stride, 1};
        return Src{ws.xb[s2], m->xd[s2].stride, 0};
    };
    auto skip_of = [&](const Stage &S) -> Src { return S.has_add ? xsrc(S.skip_src) : Src{nullptr, 0, 0}; };
    auto stage = [&](int v, float *z_out, int64_t z_stride) {
        const Stage &S = m->st[v];
        acct.bytes_rows += 2 * (int64_t)rm.R * m->xd[v + 1].size * 4;
        timed(v, 2 * S.macs * rm.R, [&] {
            return launch_stage_simt(S, xsrc(S.in_src), rm, z_out, z_stride, skip_of(S), ws.xb[v + 1], m->xd[v + 1].stride,
                                     ws.gap_tmp, s);
        });
    };
    const Stage &Sl = m->st[l];
    // GF / WS recompute k channels' dot products; the other operators are copies
    const int64_t G = rm.R / rm.T;
    const int64_t delta_flops =
        (dt.dot_prefix[g0 + G] - dt.dot_prefix[g0]) * rm.T * 2 * (int64_t)Sl.oh * Sl.ow * Sl.K;
    if (Sl.kind == MURE_NODE_LSTM) {
        // a mutated LSTM layer: its recurrence spreads one unit's change to every unit
        // from the first step on, so the layer itself is recomputed for every row from
        // its input (cached in memoized mode, recomputed in vanilla mode) with the mutated
        // units' rows rewritten, then the suffix runs from its output
        if (vanilla)
            for (int v = 0; v < l; ++v) stage(v, nullptr, 0);
        acct.bytes_rows += 2 * (int64_t)rm.R * m->xd[l + 1].size * 4;
        timed(l, 2 * Sl.macs * rm.R, [&] {
            return launch_lstm(Sl, xsrc(Sl.in_src), rm, nullptr, 0, ws.xb[l + 1], m->xd[l + 1].stride, &pa, s);
        });
        for (int v = l + 1; v < L - 1; ++v) stage(v, nullptr, 0);
        const Stage &SLr = m->st[L - 1];
        timed(L - 1, 2 * SLr.macs * rm.R, [&] { return launch_final_dense(SLr, xsrc(SLr.in_src), rm, fa, s); });
        return launches;
    }
    if (vanilla) {
        // the prefix, then layer l itself, from the inputs, row by row
        for (int v = 0; v < l; ++v) stage(v, nullptr, 0);
        if (l < L - 1) {
            stage(l, ws.zb, ws.z_stride);
        } else {
            FinalArgs f2 = fa;
            f2.mode = 2;
            f2.z_out = ws.zb;
            f2.z_stride = ws.z_stride;
            f2.logits_rows = ws.xb[L];
            f2.x_stride = m->xd[L].stride;
            timed(l, 2 * Sl.macs * rm.R, [&] { return launch_final_dense(Sl, xsrc(Sl.in_src), rm, f2, s); });
        }
    }
    // the delta: values of the mutated channels of x_{l+1} (from the cached z_l in
    // memoized mode, from the row's own z_l in vanilla mode)
    const int cells_l = Sl.gap ? 1 : (Sl.pool ? (Sl.oh / 2) * (Sl.ow / 2) : Sl.oh * Sl.ow);
    const int kmax = dt.kmax_layer[l];
    const int64_t pstride = (int64_t)std::max(kmax, 1) * cells_l;
    const Src zsrc = vanilla ? Src{ws.zb, ws.z_stride, 0} : Src{ca->z[l], m->zd[l].stride, 1};
    // GF / WS: on the tensor cores (one GEMM over the batch's inputs with every slot's
    // mutated filter as an output channel), else the CUDA-core dot-product kernels
    const bool tc_delta = tc_delta_supported(Sl, m->precision) && ws.dw.n_max > 0;
    const bool dot_kernel = !tc_delta && patch_dot_supported(Sl, kmax);
    const bool has_dot = dt.dot_prefix[g0 + G] > dt.dot_prefix[g0];
    Overlay ov;
    ov.patch = ws.patch;
    ov.row_stride = pstride;
    ov.kmax = kmax;
    ov.cells = cells_l;
    ov.ch = Sl.oc;
    ov.n_neurons = pa.n_neurons;
    ov.neuron_off = pa.neuron_off;
    ov.ids = pa.ids;
    // x_{l+1} read other than as the first suffix stage's GEMM input (a later residual
    // add, the add of a projection that reads an earlier input, or a later projection
    // reading x_{l+1} itself): its rows are materialised with the patch
    bool skip_reader = l + 1 < L && m->st[l + 1].in_src != l + 1;
    for (int v = l + 2; v < L; ++v)
        skip_reader |= (m->st[v].has_add && m->st[v].skip_src == l + 1) || m->st[v].in_src == l + 1;
    // the window GEMM as first suffix stage applies NEB (zeros) and NS (a swap of the
    // two channels, which is the operator itself: the swapped neurons' channels are
    // computed independently) on its staged maps, so the delta writes no values for
    // them; x_{l+1} must come from the small-convolution kernel, whose pooled values
    // the other operators' patches reproduce bit for bit
    // tagged mutants of the batch with neurons in later layers: the largest count per
    // later layer (their rows then take the materialised path below)
    std::vector<int> kv(L, 0);
    bool later = false;
    if (dt.has_later)
        for (int v = l + 1; v < L; ++v) {
            for (int64_t k = g0; k < g0 + G; ++k) kv[v] = std::max(kv[v], dt.nn_at_host[v][k]);
            later |= kv[v] > 0;
        }
    const bool win_ops = !later && l + 2 < L && m->st[l + 1].tc && m->st[l + 1].tc_small && !skip_reader && !Sl.tc &&
                         Sl.variant > 0 && tc_overlay_inline(m->st[l + 1], ov, G) &&
                         !(l + 1 == L - 2 && tc_final_fusable(m->st[L - 2], m->st[L - 1]));
    if (win_ops) ov.op = pa.op;
    // the delta's algorithmic bytes: the patch values it writes (every mutated channel
    // of every row, but those the window GEMM applies itself) and the rows it reads,
    // z_l (and x_l for GF / WS) once per input of the batch (memoized) or per row
    const int64_t slots = (dt.dot_prefix[g0 + G] - dt.dot_prefix[g0]) + (dt.val_prefix[g0 + G] - dt.val_prefix[g0]) -
                          (win_ops ? dt.copy_prefix[g0 + G] - dt.copy_prefix[g0] : 0);
    acct.bytes_gather += slots * rm.T * cells_l * 4;
    acct.bytes_gather += (vanilla ? rm.R : (int64_t)rm.T) * (m->zd[l].size + (has_dot ? m->xd[Sl.in_src].size : 0)) * 4;
    // where the fan-in sums (GF / WS) run in a kernel of their own, the value kernels
    // (NEB / NAI / NS: the cached pre-activations read, the patch values written) are
    // timed and counted apart: they are the memory-bound part of the delta
    const bool values_only = dot_kernel || tc_delta;
    if (values_only) {
        const int64_t vslots = (dt.val_prefix[g0 + G] - dt.val_prefix[g0]) -
                               (win_ops ? dt.copy_prefix[g0 + G] - dt.copy_prefix[g0] : 0);
        if (vslots > 0)
            acct.bytes_values += vslots * rm.T * cells_l * 4 + (vanilla ? rm.R : (int64_t)rm.T) * m->zd[l].size * 4;
    }
    timed(values_only ? C_VALS : C_DELTA, values_only ? 0 : delta_flops, [&] {
        return launch_patch_vals(Sl, zsrc, xsrc(Sl.in_src), skip_of(Sl), rm, pa, kmax, ws.patch, pstride, s, values_only,
                                 win_ops);
    });
    int delta_err = 0;
    if (tc_delta && has_dot) {
        // the inputs' x_l and z_l: cached rows (memoized) or the batch's first
        // mutant's recomputed rows (vanilla; the prefix up to layer l is unmutated)
        timed(C_DELTA, delta_flops, [&] {
            const int d = launch_tc_delta(Sl, m->precision, zsrc, xsrc(Sl.in_src), skip_of(Sl), rm, pa, ws.patch, pstride,
                                          ws.dw, s);
            if (d < 0) delta_err = 1;
            return std::max(d, 0);
        });
    } else if (dot_kernel && has_dot) {
        timed(C_DELTA, delta_flops,
              [&] { return launch_patch_dot(Sl, zsrc, xsrc(Sl.in_src), rm, pa, kmax, ws.patch, pstride, s); });
    }
    if (delta_err) return -1;
    // the unmutated rows of x_{l+1}: cached (memoized) or just computed (vanilla)
    const Src base = vanilla ? Src{ws.xb[l + 1], m->xd[l + 1].stride, 0} : Src{ca->x[l + 1], m->xd[l + 1].stride, 1};
    if (later) {
        // mu(M') holds later layers too: the rows of x_{l+1} are materialised with layer
        // l's patch, and after every later mutated layer v its own delta (computed from
        // the rows' x_v and z_v) is written over the rows of x_{v+1}; the output layer's
        // delta goes through the kill epilogue.  Memoized and vanilla rows take this
        // same path, and its arithmetic equals the fused paths' (same kernels on the
        // same values), so a mutant's bits do not depend on its batch.
        // an unmutated first suffix stage reads the cached rows with the overlay, as on
        // the single-layer path; otherwise the rows of x_{l+1} are materialised
        int vstart = l + 1;
        if (kv[l + 1] == 0 && l + 2 < L) {
            const Stage &Sn = m->st[l + 1];
            if (Sn.tc && !skip_reader && tc_overlay_inline(Sn, ov, G)) {
                acct.bytes_rows += 2 * (int64_t)rm.R * m->xd[l + 2].size * 4;
                timed(l + 1, 2 * Sn.macs * rm.R, [&] {
                    return launch_tc(Sn, base, rm, nullptr, 0, skip_of(Sn), ws.xb[l + 2], m->xd[l + 2].stride,
                                     ws.gap_tmp, s, &ov);
                });
                vstart = l + 2;
            } else if (Sn.variant > 0 && !skip_reader) {
                acct.bytes_rows += 2 * (int64_t)rm.R * m->xd[l + 2].size * 4;
                timed(l + 1, 2 * Sn.macs * rm.R, [&] {
                    return launch_conv_small(Sn, base, rm, nullptr, 0, ws.xb[l + 2], m->xd[l + 2].stride, s, &ov);
                });
                vstart = l + 2;
            }
        }
        if (vstart == l + 1)
            timed(C_DELTA, 0, [&] {
                return launch_rows_overlay(base, m->xd[l + 1].size, rm, ov, ws.xb[l + 1], m->xd[l + 1].stride, s);
            });
        const bool fuse_tail = L >= 2 && tc_final_fusable(m->st[L - 2], m->st[L - 1]) && kv[L - 2] == 0 &&
                               kv[L - 1] == 0 && !m->st[L - 2].has_add;
        for (int v = vstart; v < L; ++v) {
            const Stage &Sv = m->st[v];
            const bool mut = kv[v] > 0;
            // z_v rows at the layer's own stride (the buffer holds the largest)
            const int64_t zst = m->zd[v].stride;
            const Src zrows{ws.zb, zst, 0};
            if (fuse_tail && v == L - 2) {
                // no mutated neuron from here on: the output layer in the epilogue of the
                // layer before it, as on the single-layer path
                const Stage &SLast = m->st[L - 1];
                const FinalFuse ff{SLast.W, SLast.b, SLast.oc, SLast.K, SLast.act1, fa};
                timed(L - 2, 2 * (Sv.macs + SLast.macs) * rm.R, [&] {
                    return launch_tc(Sv, xsrc(Sv.in_src), rm, nullptr, 0, skip_of(Sv), ws.xb[L - 1], m->xd[L - 1].stride,
                                     ws.gap_tmp, s, nullptr, &ff);
                });
                break;
            }
            const int cells_v = Sv.gap ? 1 : (Sv.pool ? (Sv.oh / 2) * (Sv.ow / 2) : Sv.oh * Sv.ow);
            const int64_t pstride_v = (int64_t)std::max(kv[v], 1) * cells_v;
            PatchArgs pv{dt.op + g0, dt.nn_at ? dt.nn_at + (size_t)v * dt.n + g0 : nullptr,
                         dt.noff_at ? dt.noff_at + (size_t)v * dt.n + g0 : nullptr, dt.ids,
                         dt.poff_at ? dt.poff_at + (size_t)v * dt.n + g0 : nullptr, dt.patch};
            Overlay ovv;
            ovv.patch = ws.patch;
            ovv.row_stride = pstride_v;
            ovv.kmax = kv[v];
            ovv.cells = cells_v;
            ovv.ch = Sv.oc;
            ovv.n_neurons = pv.n_neurons;
            ovv.neuron_off = pv.neuron_off;
            ovv.ids = pv.ids;
            const int64_t dfl = mut ? 2 * (int64_t)kv[v] * rm.R * Sv.oh * Sv.ow * Sv.K : 0;
            if (v < L - 1) {
                stage(v, mut ? ws.zb : nullptr, zst);
                if (!mut) continue;
                acct.bytes_gather += rm.R * ((int64_t)kv[v] * cells_v + m->zd[v].size + m->xd[v].size) * 4;
                timed(C_DELTA, dfl, [&] {
                    return launch_patch_vals(Sv, zrows, xsrc(Sv.in_src), skip_of(Sv), rm, pv, kv[v], ws.patch, pstride_v, s);
                });
                const Src xr{ws.xb[v + 1], m->xd[v + 1].stride, 0};
                timed(C_DELTA, 0, [&] {
                    return launch_rows_overlay(xr, m->xd[v + 1].size, rm, ovv, ws.xb[v + 1], m->xd[v + 1].stride, s);
                });
            } else if (mut) {
                FinalArgs f2 = fa;
                f2.mode = 2;
                f2.z_out = ws.zb;
                f2.z_stride = zst;
                f2.logits_rows = ws.xb[L];
                f2.x_stride = m->xd[L].stride;
                timed(v, 2 * Sv.macs * rm.R, [&] { return launch_final_dense(Sv, xsrc(Sv.in_src), rm, f2, s); });
                acct.bytes_gather += rm.R * ((int64_t)kv[v] + m->zd[v].size + m->xd[v].size) * 4;
                timed(C_DELTA, dfl, [&] {
                    return launch_patch_vals(Sv, zrows, xsrc(Sv.in_src), skip_of(Sv), rm, pv, kv[v], ws.patch, pstride_v, s);
                });
                timed(C_EPI, 0, [&] {
                    return launch_epilogue(Src{ws.xb[L], m->xd[L].stride, 0}, m->n_classes, rm, fa, s, &ovv);
                });
            } else {
                timed(v, 2 * Sv.macs * rm.R, [&] { return launch_final_dense(Sv, xsrc(Sv.in_src), rm, fa, s); });
            }
        }
        return launches;
    }
    // exact unchanged-row elimination (memoized mode): rows whose x_{l+1} equals the
    // original bit for bit keep kill 0 and the original logits; the suffix runs on the
    // others only, as a compacted batch (physical row r = logical row lrow[r]).  The
    // first suffix stage must read its rows through the row map: not the window GEMM
    // or the CUDA-core small convolution, which stage whole consecutive rows.
    {
        const Stage &S1 = m->st[std::min(l + 1, L - 1)];
        const bool first_ok = l + 1 == L - 1 || !(S1.tc_small || (S1.variant > 0 && !S1.tc));
        if (ec.skip_unchanged && l < L - 1 && first_ok) {
            UnchangedArgs ua{ws.patch, pstride, cells_l, Sl.oc, pa.n_neurons, pa.neuron_off, pa.ids,
                             ca->x[l + 1], m->xd[l + 1].stride, ca->x[L], m->xd[L].stride, m->n_classes, fa};
            timed(C_DELTA, 0, [&] { return launch_unchanged(ua, rm, ws.uflags, ws.ublk, ws.lrow, ws.ucount, s); });
            int32_t n_run = 0;
            CK(c, cudaMemcpyAsync(&n_run, ws.ucount, sizeof n_run, cudaMemcpyDeviceToHost, s));
            CK(c, cudaStreamSynchronize(s));
            const int64_t valid = G * std::max<int64_t>(0, std::min<int64_t>(rm.T, ca->n_in - rm.t0));
            acct.rows_unchanged += valid - n_run;
            if (n_run == 0) return launches;
            rm.R = n_run;
            rm.lrow = ws.lrow;
            fa.compact = 1;
            fa.lrow = ws.lrow;
        }
    }
    if (l == L - 1) {
        // mutants of the output layer: the epilogue reads the logits with the overlay
        timed(C_EPI, 0, [&] { return launch_epilogue(base, m->n_classes, rm, fa, s, &ov); });
        return launches;
    }
    if (l + 1 == L - 1) {
        const Stage &SL = m->st[L - 1];
        timed(L - 1, 2 * SL.macs * rm.R, [&] { return launch_final_dense(SL, base, rm, fa, s, &ov); });
        return launches;
    }
    // first suffix stage: the overlay is applied while its input tile is staged, or
    // the rows are materialised for kernels that read plain rows and whenever a later
    // residual add reads x_{l+1} as its skip input
    const Stage &Sn = m->st[l + 1];
    // a tensor-core dense stage L-2 takes the output layer and the kill epilogue into
    // its own epilogue (the rows of x_{L-1} are then never stored)
    const Stage &SLast = m->st[L - 1];
    const FinalFuse ff{SLast.W, SLast.b, SLast.oc, SLast.K, SLast.act1, fa};
    auto fused_last = [&](Src x, const Overlay *ovp) {
        const Stage &S = m->st[L - 2];
        timed(L - 2, 2 * (S.macs + SLast.macs) * rm.R, [&] {
            return launch_tc(S, x, rm, nullptr, 0, skip_of(S), ws.xb[L - 1], m->xd[L - 1].stride, ws.gap_tmp, s, ovp, &ff);
        });
    };
    const bool fuse = L >= 2 && tc_final_fusable(m->st[L - 2], SLast);
    if (Sn.tc && !skip_reader && tc_overlay_inline(Sn, ov, rm.R / rm.T)) {
        if (fuse && l + 1 == L - 2) {
            fused_last(base, &ov);
            return launches;
        }
        acct.bytes_rows += 2 * (int64_t)rm.R * m->xd[l + 2].size * 4;
        timed(l + 1, 2 * Sn.macs * rm.R, [&] {
            return launch_tc(Sn, base, rm, nullptr, 0, skip_of(Sn), ws.xb[l + 2], m->xd[l + 2].stride, ws.gap_tmp, s,
                             &ov);
        });
    } else if (Sn.variant > 0 && !skip_reader) {
        acct.bytes_rows += 2 * (int64_t)rm.R * m->xd[l + 2].size * 4;
        timed(l + 1, 2 * Sn.macs * rm.R, [&] {
            return launch_conv_small(Sn, base, rm, nullptr, 0, ws.xb[l + 2], m->xd[l + 2].stride, s, &ov);
        });
    } else {
        acct.bytes_gather += 2 * (int64_t)rm.R * m->xd[l + 1].size * 4;
        timed(C_DELTA, 0, [&] {
            return launch_rows_overlay(base, m->xd[l + 1].size, rm, ov, ws.xb[l + 1], m->xd[l + 1].stride, s);
        });
        stage(l + 1, nullptr, 0);
    }
    // the rest of the suffix (Algorithm 4) and the fused kill epilogue
    if (fuse && l + 2 <= L - 2) {
        for (int v = l + 2; v < L - 2; ++v) stage(v, nullptr, 0);
        fused_last(xsrc(m->st[L - 2].in_src), nullptr);
        return launches;
    }
    for (int v = l + 2; v < L - 1; ++v) stage(v, nullptr, 0);
    const Stage &SL = m->st[L - 1];
    timed(L - 1, 2 * SL.macs * rm.R, [&] { return launch_final_dense(SL, xsrc(SL.in_src), rm, fa, s); });
    return launches;
}

struct Outputs {
    uint64_t *kill_bits;
    double *sA, *sB;
    mure_eval_stats *stats;
    const mure_eval_opts *opts;
};

void evaluate(mure_ctx *c, const mure_model *m, const mure_cache *ca, const mure_mutant *t, int64_t n,
              const int32_t *pool, int64_t pool_len, bool vanilla, const Outputs &out)
{
    const mure_eval_opts dflt{};
    const mure_eval_opts *o = out.opts ? out.opts : &dflt;
    FAILIF(n > 0 && ca->n_in > 0 && !out.kill_bits, c, MURE_ERR_INVALID_ARG, "NULL kill_bits");
    cudaStream_t s = c->stream;
    Scratch sc(c);
    CK(c, cudaEventRecord(c->ev[0], s));
    const Groups g = group_by_layer(m, t, n, pool);
    const int64_t words32 = ca->n_pad / 32;
    mure_eval_stats st{};
    st.n_rows = n * ca->n_in;
    double sA = 0, sB = 0;
    if (n > 0 && ca->n_in > 0) {
        const DevTable dt = upload_table(c, sc, m, t, n, pool, pool_len, g, 0, nullptr, nullptr);
        CK(c, cudaEventRecord(c->ev[1], s));
        EvalCfg ec{};
        ec.words32 = words32;
        ec.kill32 = o->outputs_on_device ? reinterpret_cast<uint32_t *>(out.kill_bits)
                                         : sc.get<uint32_t>((size_t)n * words32);
        ec.counters = sc.get<unsigned long long>(4);
        CK(c, cudaMemsetAsync(ec.counters, 0, 4 * sizeof(unsigned long long), s));
        float *lg_dev = nullptr;
        if (o->logits_out) {
            lg_dev = o->outputs_on_device ? o->logits_out : sc.get<float>((size_t)n * ca->n_in * m->n_classes);
        }
        ec.logits_out = lg_dev;
        // batch geometry: rows = mutants x input tile, bounded by the workspace cap
        const int64_t cap = o->workspace_bytes > 0 ? o->workspace_bytes : (int64_t)8 << 30;
        int lmin = m->L;
        int64_t rb = 0;
        for (int l = 0; l < m->L; ++l)
            if (g.begin[l + 1] > g.begin[l]) {
                lmin = std::min(lmin, l);
                rb = std::max(rb, row_bytes(m, l, vanilla, dt.has_later));
            }
        int64_t rows = std::max<int64_t>(cap / std::max<int64_t>(rb, 1), 64);
        rows = std::min<int64_t>(rows, (int64_t)1 << 24);
        // the input tile leaves room for batch_mutants() mutants per batch: the delta's
        // tensor-core GEMM is as wide as a batch's mutated channels, and each cached input
        // row staged by the delta kernels serves every mutant of the batch (rows per
        // batch, and so the suffix's work per launch, stay the same)
        int64_t T = std::min<int64_t>(ca->n_pad, std::max<int64_t>(64, rows / batch_mutants() / 64 * 64));
        const int64_t Gmax = std::max<int64_t>(1, rows / T);
        // never more rows than the largest group needs
        int64_t gbig = 0;
        for (int l = 0; l < m->L; ++l) gbig = std::max(gbig, g.begin[l + 1] - g.begin[l]);
        rows = std::min(Gmax, gbig) * T;
        int64_t patch_floats = 1;
        for (int l = 0; l < m->L; ++l) {
            if (g.begin[l + 1] == g.begin[l]) continue;
            const Stage &S = m->st[l];
            const int64_t cl = S.gap ? 1 : (S.pool ? (S.oh / 2) * (S.ow / 2) : S.oh * S.ow);
            patch_floats = std::max<int64_t>(patch_floats, (int64_t)std::max(dt.kmax_layer[l], 1) * cl);
        }
        if (dt.has_later)   // later mutated layers of tagged mutants: their patches too
            for (int v = 0; v < m->L; ++v) {
                const Stage &S = m->st[v];
                const int64_t cl = S.gap ? 1 : (S.pool ? (S.oh / 2) * (S.ow / 2) : S.oh * S.ow);
                int km = 0;
                for (int64_t k = 0; k < n; ++k) km = std::max(km, dt.nn_at_host[v][k]);
                patch_floats = std::max<int64_t>(patch_floats, (int64_t)km * cl);
            }
        // the tensor-core delta: slots of a batch at most G x kmax of its layer
        int delta_slots = 0, delta_k = 0;
        for (int l = 0; l < m->L; ++l) {
            if (g.begin[l + 1] == g.begin[l] || !tc_delta_supported(m->st[l], m->precision)) continue;
            const int64_t gb = std::min<int64_t>(Gmax, g.begin[l + 1] - g.begin[l]);
            delta_slots = (int)std::max<int64_t>(delta_slots, gb * std::max(dt.kmax_layer[l], 1));
            delta_k = std::max(delta_k, m->st[l].K);
        }
        Workspace ws;
        alloc_workspace(c, sc, m, rows, vanilla, lmin, patch_floats, delta_slots, delta_k, ws, dt.has_later);
        FAILIF(o->skip_unchanged != 0 && o->skip_unchanged != 1, c, MURE_ERR_INVALID_ARG, "skip_unchanged must be 0 or 1");
        if (!vanilla && o->skip_unchanged) {
            ec.skip_unchanged = true;
            ws.uflags = sc.get<int32_t>(rows);
            ws.ublk = sc.get<int32_t>(rows / 256 + 1);
            ws.lrow = sc.get<int32_t>(rows);
            ws.ucount = sc.get<int32_t>(1);
            // compacted batches OR their kill bits in
            CK(c, cudaMemsetAsync(ec.kill32, 0, (size_t)n * words32 * 4, s));
        }
        int64_t launches = 0;
        Acct acct;
        acct.flops_cls.assign(m->L + 3, 0);
        acct.launches_cls.assign(m->L + 3, 0);
        KTimer tm(c, o->kernel_timing != 0);
        for (int l = 0; l < m->L; ++l) {
            const int64_t gs = g.begin[l], ge = g.begin[l + 1];
            if (ge == gs) continue;
            ++st.n_groups;
            for (int64_t t0 = 0; t0 < ca->n_pad; t0 += T) {
                const int Tt = (int)std::min<int64_t>(T, ca->n_pad - t0);
                for (int64_t g0 = gs; g0 < ge; g0 += Gmax) {
                    const int64_t G = std::min<int64_t>(Gmax, ge - g0);
                    RowMap rm{t0, Tt, (int)(G * Tt)};
                    const int nb = run_batch(c, m, ca, dt, ec, ws, l, g0, rm, vanilla, acct, tm);
                    FAILIF(nb < 0, c, MURE_ERR_UNSUPPORTED, "delta scratch too small for layer %d", l);
                    launches += nb;
                    check_launch(c);
                    ++st.n_batches;
                }
            }
        }
        CK(c, cudaEventRecord(c->ev[2], s));
        launches += launch_scores(ec.kill32, n, words32, ca->label, m->n_classes, ec.counters, s);
        check_launch(c);
        CK(c, cudaEventRecord(c->ev[3], s));
        unsigned long long host_cnt[4];
        CK(c, cudaMemcpyAsync(host_cnt, ec.counters, sizeof host_cnt, cudaMemcpyDeviceToHost, s));
        int dev_err = 0;
        CK(c, cudaMemcpyAsync(&dev_err, c->err_dev, sizeof(int), cudaMemcpyDeviceToHost, s));
        if (!o->outputs_on_device) {
            CK(c, cudaMemcpyAsync(out.kill_bits, ec.kill32, (size_t)n * words32 * 4, cudaMemcpyDeviceToHost, s));
            if (o->logits_out)
                CK(c, cudaMemcpyAsync(o->logits_out, lg_dev, (size_t)n * ca->n_in * m->n_classes * 4,
                                      cudaMemcpyDeviceToHost, s));
        }
        CK(c, cudaEventRecord(c->ev[4], s));
        CK(c, cudaStreamSynchronize(s));
        CK(c, cudaGetLastError());
        if (dev_err) {
            CK(c, cudaMemset(c->err_dev, 0, sizeof(int)));
            FAILIF(true, c, dev_err == MURE_ERR_TIMEOUT ? MURE_ERR_TIMEOUT : MURE_ERR_UNSUPPORTED,
                   "a device-side check failed (code %d)", dev_err);
        }
        sA = (double)host_cnt[0] / (double)n;
        sB = ca->n_label_values > 0 ? (double)host_cnt[1] / ((double)n * ca->n_label_values) : 0.0;
        st.n_near_ties = (int64_t)host_cnt[2];
        st.kernel_launches = launches + dt.expand_launches;
        c->launches += st.kernel_launches;
        st.flops = acct.flops;
        if (tm.on) {
            std::vector<double> ms(m->L + 3, 0.0);
            tm.collect(ms);
            for (int v = 0; v < m->L && v < MURE_MAX_TIMED_LAYERS; ++v) {
                st.ms_layer[v] = ms[v];
                st.flops_layer[v] = acct.flops_cls[v];
                st.launches_layer[v] = acct.launches_cls[v];
            }
            st.ms_delta = ms[m->L];
            st.ms_delta_values = ms[m->L + 1];
            st.launches_delta_values = acct.launches_cls[m->L + 1];
            st.ms_epilogue = ms[m->L + 2];
            st.launches_delta = acct.launches_cls[m->L];
        }
        st.bytes_gather = acct.bytes_gather;
        st.bytes_rows = acct.bytes_rows;
        st.bytes_delta_values = acct.bytes_values;
        st.n_rows_unchanged = acct.rows_unchanged;
        float ms = 0;
        cudaEventElapsedTime(&ms, c->ev[0], c->ev[4]); st.ms_total = ms;
        cudaEventElapsedTime(&ms, c->ev[0], c->ev[1]); st.ms_expand = ms;
        cudaEventElapsedTime(&ms, c->ev[1], c->ev[2]); st.ms_suffix = ms;
        cudaEventElapsedTime(&ms, c->ev[2], c->ev[3]); st.ms_score = ms;
    } else if (n > 0 && out.kill_bits && o->outputs_on_device == 0) {
        // no inputs: zero-width kill rows, nothing to write
    }
    if (out.sA) *out.sA = sA;
    if (out.sB) *out.sB = sB;
    if (out.stats) *out.stats = st;
}

// Original forward over X: the prefix cache (full) or, for vanilla, only the
// network input, predictions and labels.
mure_cache *build_cache(mure_model *m, const float *X, int64_t n_in, const int32_t *labels, int on_dev, bool full)
{
    mure_ctx *c = m->ctx;
    FAILIF(n_in < 0, c, MURE_ERR_INVALID_ARG, "n_inputs < 0");
    FAILIF(n_in > 0 && !X, c, MURE_ERR_INVALID_ARG, "NULL X");
    FAILIF(n_in > ((int64_t)1 << 30), c, MURE_ERR_UNSUPPORTED, "more than 2^30 inputs");
    std::vector<int32_t> lab_host;
    if (labels && n_in > 0) {
        lab_host.resize(n_in);
        if (on_dev) CK(c, cudaMemcpy(lab_host.data(), labels, n_in * 4, cudaMemcpyDeviceToHost));
        else memcpy(lab_host.data(), labels, n_in * 4);
        for (int64_t t = 0; t < n_in; ++t)
            FAILIF(lab_host[t] < 0 || lab_host[t] >= m->n_classes, c, MURE_ERR_INVALID_ARG, "label %d of input %lld",
                   lab_host[t], (long long)t);
    }
    cudaStream_t s = c->stream;
    auto *ca = new mure_cache();
    ca->model = m;
    ca->full = full;
    ca->n_in = n_in;
    ca->n_pad = round_up(n_in, kInputAlign);
    const int L = m->L;
    ca->x.assign(L + 1, nullptr);
    ca->z.assign(L, nullptr);
    struct Cleanup {
        mure_cache *ca;
        bool ok = false;
        ~Cleanup()
        {
            if (!ok) mure_cache_free(ca);
        }
    } cl{ca};
    const int64_t np = std::max<int64_t>(ca->n_pad, kInputAlign);
    for (int s2 = 0; s2 <= L; ++s2) {
        ca->x[s2] = (float *)dalloc(c, np * m->xd[s2].stride * 4);
        CK(c, cudaMemsetAsync(ca->x[s2], 0, np * m->xd[s2].stride * 4, s));
    }
    for (int v = 0; v < L; ++v) {
        ca->z[v] = (float *)dalloc(c, np * m->zd[v].stride * 4);
        CK(c, cudaMemsetAsync(ca->z[v], 0, np * m->zd[v].stride * 4, s));
    }
    ca->pred0 = (int32_t *)dalloc(c, np * 4);
    ca->label = (int32_t *)dalloc(c, np * 4);
    CK(c, cudaMemsetAsync(ca->pred0, 0, np * 4, s));
    CK(c, cudaMemsetAsync(ca->label, 0, np * 4, s));
    if (n_in > 0) {
        const int64_t sz = m->xd[0].size, str = m->xd[0].stride;
        CK(c, cudaMemcpy2DAsync(ca->x[0], str * 4, X, sz * 4, sz * 4, n_in,
                                on_dev ? cudaMemcpyDeviceToDevice : cudaMemcpyHostToDevice, s));
        Scratch sc(c);
        int64_t g = 0;
        for (int v = 0; v < L; ++v)
            if (m->st[v].gap) g = std::max(g, gap_map_stride(m->st[v]));
        float *gap_tmp = g ? sc.get<float>(ca->n_pad * g) : nullptr;
        // intermediate activations: in the cache (full) or in scratch rows (vanilla
        // only needs the predictions)
        std::vector<float *> xs(L + 1), zs(L);
        for (int s2 = 0; s2 <= L; ++s2) xs[s2] = ca->x[s2];
        for (int v = 0; v < L; ++v) zs[v] = ca->z[v];
        const RowMap rm{0, (int)ca->n_pad, (int)ca->n_pad};
        for (int v = 0; v < L - 1; ++v) {
            const Stage &S = m->st[v];
            const Src skip = S.has_add ? Src{xs[S.skip_src], m->xd[S.skip_src].stride, 0} : Src{nullptr, 0, 0};
            c->launches += launch_stage_simt(S, Src{xs[S.in_src], m->xd[S.in_src].stride, 0}, rm, zs[v], m->zd[v].stride, skip,
                                             xs[v + 1], m->xd[v + 1].stride, gap_tmp, s);
            check_launch(c);
        }
        FinalArgs fa{};
        fa.mode = 1;
        fa.z_out = zs[L - 1];
        fa.z_stride = m->zd[L - 1].stride;
        fa.x_out = xs[L];
        fa.x_stride = m->xd[L].stride;
        fa.pred_out = ca->pred0;
        c->launches += launch_final_dense(m->st[L - 1], Src{xs[L - 1], m->xd[L - 1].stride, 0}, rm, fa, s);
        check_launch(c);
        if (labels) CK(c, cudaMemcpyAsync(ca->label, lab_host.data(), n_in * 4, cudaMemcpyHostToDevice, s));
        else CK(c, cudaMemcpyAsync(ca->label, ca->pred0, n_in * 4, cudaMemcpyDeviceToDevice, s));
        uint32_t *mask = sc.get<uint32_t>(kLabelWords);
        CK(c, cudaMemsetAsync(mask, 0, 4 * kLabelWords, s));
        c->launches += launch_label_set(ca->label, n_in, mask, s);
        check_launch(c);
        uint32_t hm[kLabelWords] = {};
        CK(c, cudaMemcpyAsync(hm, mask, 4 * kLabelWords, cudaMemcpyDeviceToHost, s));
        int dev_err = 0;
        CK(c, cudaMemcpyAsync(&dev_err, c->err_dev, sizeof(int), cudaMemcpyDeviceToHost, s));
        CK(c, cudaStreamSynchronize(s));
        ca->n_label_values = 0;
        for (int k = 0; k < kLabelWords; ++k) ca->n_label_values += __builtin_popcount(hm[k]);
        if (dev_err) {
            // a token id outside an embedding's table, a bounded wait that gave up, or a
            // layer geometry a launch refused
            CK(c, cudaMemset(c->err_dev, 0, sizeof(int)));
            FAILIF(true, c,
                   dev_err == MURE_ERR_TIMEOUT || dev_err == MURE_ERR_UNSUPPORTED ? (mure_status)dev_err : MURE_ERR_INVALID_ARG,
                   "a device-side check failed while building the cache (code %d: %s)", dev_err,
                   dev_err == MURE_ERR_INVALID_ARG   ? "an input id outside the embedding's table"
                   : dev_err == MURE_ERR_UNSUPPORTED ? "a layer geometry the kernels refused"
                                                     : "wait limit");
        }
    }
    CK(c, cudaStreamSynchronize(s));
    cl.ok = true;
    return ca;
}

}  // namespace

// ====================================================================== ABI ==

namespace mure {

mure_status check_table_status(mure_ctx *c, const mure_model *m, const mure_mutant *t, int64_t n, const int32_t *pool,
                               int64_t pool_len)
{
    return run(c, [&] { check_table(c, m, t, n, pool, pool_len); });
}

}  // namespace mure

extern "C" {

mure_status mure_create(int device, void *cuda_stream, const mure_allocator *alloc, mure_ctx **out)
{
    if (!out) return MURE_ERR_INVALID_ARG;
    *out = nullptr;
    int n = 0;
    if (cudaGetDeviceCount(&n) != cudaSuccess) {
        cudaGetLastError();
        return MURE_ERR_CUDA;
    }
    if (device < 0 || device >= n) return MURE_ERR_INVALID_ARG;
    if (alloc && (!alloc->alloc || !alloc->free)) return MURE_ERR_INVALID_ARG;
    auto *c = new mure_ctx();
    c->device = device;
    c->stream = (cudaStream_t)cuda_stream;
    if (alloc) { c->alloc = *alloc; c->has_alloc = true; }
    mure_status st = run(c, [&] {
        CK(c, cudaSetDevice(device));
        CK(c, cudaDeviceGetAttribute(&c->n_sms, cudaDevAttrMultiProcessorCount, device));
        for (auto &e : c->ev) CK(c, cudaEventCreate(&e));
        CK(c, cudaMalloc(&c->err_dev, sizeof(int)));
        CK(c, cudaMemset(c->err_dev, 0, sizeof(int)));
    });
    if (st != MURE_OK) {
        mure_destroy(c);
        return st;
    }
    *out = c;
    return MURE_OK;
}

void mure_destroy(mure_ctx *ctx)
{
    if (!ctx) return;
    for (auto &e : ctx->ev)
        if (e) cudaEventDestroy(e);
    for (auto &e : ctx->evpool) cudaEventDestroy(e);
    if (ctx->err_dev) cudaFree(ctx->err_dev);
    delete ctx;
}

const char *mure_last_error(const mure_ctx *ctx) { return ctx ? ctx->err.c_str() : "NULL context"; }

namespace {

// The checks of a network description's header (before its nodes are compiled).
void check_desc(mure_ctx *c, const mure_model_desc *d)
{
    FAILIF(!d || !d->nodes || d->n_nodes < 1, c, MURE_ERR_INVALID_ARG, "NULL model description");
    FAILIF(d->in_h < 1 || d->in_w < 1 || d->in_c < 1, c, MURE_ERR_INVALID_ARG, "bad input shape");
    FAILIF(d->precision != MURE_PREC_FP32 && d->precision != MURE_PREC_TF32X3 && d->precision != MURE_PREC_TF32,
           c, MURE_ERR_UNSUPPORTED, "precision %d is not available", d->precision);
}

}  // namespace

mure_status mure_model_load(mure_ctx *c, const mure_model_desc *d, mure_model **out)
{
    if (!c) return MURE_ERR_INVALID_ARG;
    return run(c, [&] {
        FAILIF(!out, c, MURE_ERR_INVALID_ARG, "NULL output handle");
        *out = nullptr;
        check_desc(c, d);
        CK(c, cudaSetDevice(c->device));
        auto *m = new mure_model();
        m->ctx = c;
        m->precision = d->precision;
        struct Cleanup {
            mure_model *m;
            bool ok = false;
            ~Cleanup()
            {
                if (!ok) mure_model_free(m);
            }
        } cl{m};
        compile(c, d, m);
        // kernel selection per layer (fixed for the model's lifetime, so every
        // computation of a layer uses one kernel); MURE_FORCE_GENERIC=1 keeps the
        // implicit-GEMM kernel everywhere (the kernels agree bit for bit)
        const char *force = getenv("MURE_FORCE_GENERIC");
        for (Stage &S : m->st) {
            S.variant = (force && force[0] == '1') ? 0 : conv_small_variant(S);
            S.geo = S.variant;
            S.err = c->err_dev;
            S.wait_limit = &c->wait_limit;
        }
        // tensor-core modes: layers before the output layer with >= 16 outputs run on
        // the tensor cores (3xTF32, or one TF32 MMA in the reduced-precision variant);
        // the LeNet-size convolution takes the small-image mode (MURE_TC_CONV above)
        for (int l = 0; l + 1 < m->L; ++l) {
            Stage &S = m->st[l];
            const std::string env = tc_conv_env();
            const bool small = tc_small_geometry(S) && env != "0";
            const bool take = tc_supported(S) && (S.kind == MURE_NODE_DENSE || S.variant == 0 || small);
            if (take && d->precision == MURE_PREC_TF32X3) S.tc = 1;
            else if (take && d->precision == MURE_PREC_TF32) S.tc = 2;
            if (S.tc) {
                S.variant = 0;
                S.tc_small = small && env != "generic";
                S.tc_conv = !S.tc_small && env != "gather" && tc_conv_geometry(S);
                S.tc_wide = S.tc_conv && getenv("MURE_TC_NARROW") == nullptr && tc_wide_geometry(S);
                // 16-channel 3x3 layers: a GEMM row per 2x2 output window (MURE_TC_NOWINDOW
                // keeps a row per position)
                S.tc_win = S.tc_conv && getenv("MURE_TC_NOWINDOW") == nullptr && tc_win_geometry(S);
            }
        }
        std::vector<int> wn;
        for (int v = 0; v < d->n_nodes; ++v)
            if (weighted(d->nodes[v].kind)) wn.push_back(v);
        std::vector<float> Wt;
        for (int l = 0; l < m->L; ++l) {
            Stage &S = m->st[l];
            const mure_node &n = d->nodes[wn[l]];
            const int64_t nw = (int64_t)S.oc * S.K;
            S.W = (float *)dalloc(c, nw * 4);
            S.Wt = (float *)dalloc(c, nw * 4);
            // an LSTM unit has four gate biases; an embedding has none (zeros)
            const int64_t nb = S.kind == MURE_NODE_LSTM ? 4 * (int64_t)S.oc : S.oc;
            S.b = (float *)dalloc(c, nb * 4);
            Wt.resize(nw);
            for (int o = 0; o < S.oc; ++o)
                for (int k = 0; k < S.K; ++k) Wt[(int64_t)k * S.oc + o] = n.W[(int64_t)o * S.K + k];
            CK(c, cudaMemcpyAsync(S.W, n.W, nw * 4, cudaMemcpyHostToDevice, c->stream));
            CK(c, cudaMemcpyAsync(S.Wt, Wt.data(), nw * 4, cudaMemcpyHostToDevice, c->stream));
            if (n.b) CK(c, cudaMemcpyAsync(S.b, n.b, nb * 4, cudaMemcpyHostToDevice, c->stream));
            else CK(c, cudaMemsetAsync(S.b, 0, nb * 4, c->stream));
            CK(c, cudaStreamSynchronize(c->stream));  // Wt is reused
            if (S.tc) {
                S.Wtc = (float *)dalloc(c, tc_weight_floats(S) * 4);
                const int64_t ntmp = tc_swizzle_tmp_floats(S);
                float *tmp = ntmp ? (float *)dalloc(c, ntmp * 4) : nullptr;
                c->launches += launch_swizzle_weights(S, S.Wtc, tmp, c->stream);
                if (tmp) {
                    CK(c, cudaStreamSynchronize(c->stream));
                    dfree(c, tmp);
                }
                check_launch(c);
            }
        }
        // population std of every layer's weights (GF's sigma), fp64 on the device
        {
            Scratch sc(c);
            std::vector<const float *> Wp(m->L);
            std::vector<int64_t> cnt(m->L);
            for (int l = 0; l < m->L; ++l) { Wp[l] = m->st[l].W; cnt[l] = (int64_t)m->st[l].oc * m->st[l].K; }
            const float **Wd = sc.get<const float *>(m->L);
            int64_t *nd = sc.get<int64_t>(m->L);
            m->sigma_dev = (double *)dalloc(c, m->L * 8);
            CK(c, cudaMemcpyAsync(Wd, Wp.data(), m->L * sizeof(float *), cudaMemcpyHostToDevice, c->stream));
            CK(c, cudaMemcpyAsync(nd, cnt.data(), m->L * 8, cudaMemcpyHostToDevice, c->stream));
            c->launches += launch_layer_std(Wd, nd, m->L, m->sigma_dev, c->stream);
            check_launch(c);
            m->sigma_host.resize(m->L);
            CK(c, cudaMemcpyAsync(m->sigma_host.data(), m->sigma_dev, m->L * 8, cudaMemcpyDeviceToHost, c->stream));
            CK(c, cudaStreamSynchronize(c->stream));
            for (int l = 0; l < m->L; ++l) m->st[l].sigma_std = (float)m->sigma_host[l];
        }
        cl.ok = true;
        *out = m;
    });
}

void mure_model_free(mure_model *m)
{
    if (!m) return;
    for (auto &S : m->st) {
        dfree(m->ctx, S.W);
        dfree(m->ctx, S.Wt);
        dfree(m->ctx, S.b);
        dfree(m->ctx, S.Wtc);
    }
    dfree(m->ctx, m->sigma_dev);
    cudaStreamSynchronize(m->ctx->stream);
    delete m;
}

int32_t mure_model_n_layers(const mure_model *m) { return m ? m->L : -1; }

mure_status mure_model_layer_kernel(const mure_model *m, int32_t layer, int32_t *kernel, int64_t *macs_per_row)
{
    if (!m || layer < 0 || layer >= m->L) return MURE_ERR_INVALID_ARG;
    const Stage &S = m->st[layer];
    int32_t k = MURE_KERNEL_SIMT_GEMM;
    int64_t macs = S.macs;
    if (layer == m->L - 1) {
        k = MURE_KERNEL_OUTPUT;
    } else if (S.tc) {
        k = S.tc_small ? MURE_KERNEL_TC_WINDOW : S.tc_conv ? MURE_KERNEL_TC_CONV : MURE_KERNEL_TC_GEMM;
        macs = tc_macs_per_row(S);
    } else if (S.variant > 0) {
        k = MURE_KERNEL_SIMT_SMALL;
    }
    if (kernel) *kernel = k;
    if (macs_per_row) *macs_per_row = macs;
    return MURE_OK;
}

int64_t mure_kernel_launches(const mure_ctx *ctx) { return ctx ? ctx->launches : -1; }

mure_status mure_set_wait_limit(mure_ctx *ctx, int64_t cycles)
{
    if (!ctx) return MURE_ERR_INVALID_ARG;
    ctx->err.clear();
    if (cycles < 0) {
        ctx->err = "negative wait limit";
        return MURE_ERR_INVALID_ARG;
    }
    ctx->wait_limit = cycles;
    return MURE_OK;
}

mure_status mure_build_prefix_cache(mure_model *m, const float *X, int64_t n_inputs, const int32_t *labels,
                                    int x_on_device, mure_cache **out)
{
    if (!m) return MURE_ERR_INVALID_ARG;
    mure_ctx *c = m->ctx;
    return run(c, [&] {
        FAILIF(!out, c, MURE_ERR_INVALID_ARG, "NULL out");
        *out = nullptr;
        CK(c, cudaSetDevice(c->device));
        *out = build_cache(m, X, n_inputs, labels, x_on_device, true);
    });
}

void mure_cache_free(mure_cache *ca)
{
    if (!ca) return;
    mure_ctx *c = ca->model->ctx;
    for (float *p : ca->x) dfree(c, p);
    for (float *p : ca->z) dfree(c, p);
    dfree(c, ca->pred0);
    dfree(c, ca->label);
    cudaStreamSynchronize(c->stream);
    delete ca;
}

mure_status mure_cache_outputs(mure_cache *ca, float *logits, int32_t *pred)
{
    if (!ca) return MURE_ERR_INVALID_ARG;
    mure_ctx *c = ca->model->ctx;
    return run(c, [&] {
        const mure_model *m = ca->model;
        if (ca->n_in == 0) return;
        if (logits)
            CK(c, cudaMemcpy2DAsync(logits, m->n_classes * 4, ca->x[m->L], m->xd[m->L].stride * 4, m->n_classes * 4,
                                    ca->n_in, cudaMemcpyDeviceToHost, c->stream));
        if (pred) CK(c, cudaMemcpyAsync(pred, ca->pred0, ca->n_in * 4, cudaMemcpyDeviceToHost, c->stream));
        CK(c, cudaStreamSynchronize(c->stream));
    });
}

mure_status mure_eval_mutants(mure_cache *ca, const mure_mutant *table, int64_t n_mutants, const int32_t *neuron_pool,
                              int64_t pool_len, const mure_eval_opts *opts, uint64_t *kill_bits,
                              double *score_killed_frac, double *score_deepmutation, mure_eval_stats *stats)
{
    if (!ca) return MURE_ERR_INVALID_ARG;
    mure_ctx *c = ca->model->ctx;
    return run(c, [&] {
        CK(c, cudaSetDevice(c->device));
        FAILIF(!ca->full, c, MURE_ERR_INVALID_ARG, "cache holds no activations");
        check_table(c, ca->model, table, n_mutants, neuron_pool, pool_len);
        evaluate(c, ca->model, ca, table, n_mutants, neuron_pool, pool_len, false,
                 Outputs{kill_bits, score_killed_frac, score_deepmutation, stats, opts});
    });
}

mure_status mure_eval_vanilla(mure_model *m, const float *X, int64_t n_inputs, const int32_t *labels, int x_on_device,
                              const mure_mutant *table, int64_t n_mutants, const int32_t *neuron_pool,
                              int64_t pool_len, const mure_eval_opts *opts, uint64_t *kill_bits,
                              double *score_killed_frac, double *score_deepmutation, mure_eval_stats *stats)
{
    if (!m) return MURE_ERR_INVALID_ARG;
    mure_ctx *c = m->ctx;
    return run(c, [&] {
        CK(c, cudaSetDevice(c->device));
        check_table(c, m, table, n_mutants, neuron_pool, pool_len);
        mure_cache *ca = build_cache(m, X, n_inputs, labels, x_on_device, false);
        struct Free {
            mure_cache *ca;
            ~Free() { mure_cache_free(ca); }
        } fr{ca};
        evaluate(c, m, ca, table, n_mutants, neuron_pool, pool_len, true,
                 Outputs{kill_bits, score_killed_frac, score_deepmutation, stats, opts});
    });
}

mure_status mure_check_descriptors(const mure_model_desc *d, const mure_mutant *table, int64_t n_mutants,
                                   const int32_t *neuron_pool, int64_t pool_len, char *msg, size_t msg_len)
{
    // host state only: the error text and the compiled stages (no device is touched)
    mure_ctx c;
    mure_model m;
    const mure_status st = run(&c, [&] {
        check_desc(&c, d);
        compile(&c, d, &m);
        check_table(&c, &m, table, n_mutants, neuron_pool, pool_len);
    });
    if (msg && msg_len > 0) snprintf(msg, msg_len, "%s", c.err.c_str());
    return st;
}

mure_status mure_expand_patches(mure_model *m, const mure_mutant *table, int64_t n_mutants, const int32_t *neuron_pool,
                                int64_t pool_len, float *out, int64_t out_len, int64_t *offsets)
{
    if (!m) return MURE_ERR_INVALID_ARG;
    mure_ctx *c = m->ctx;
    return run(c, [&] {
        CK(c, cudaSetDevice(c->device));
        check_table(c, m, table, n_mutants, neuron_pool, pool_len);
        for (int64_t i = 0; i < n_mutants; ++i)
            FAILIF(table[i].tagged, c, MURE_ERR_UNSUPPORTED, "mutant %lld: tagged descriptors have no flat patch layout",
                   (long long)i);
        FAILIF(!offsets && n_mutants > 0, c, MURE_ERR_INVALID_ARG, "NULL offsets");
        int64_t need = 0;
        for (int64_t i = 0; i < n_mutants; ++i)
            if (table[i].op == MURE_OP_GF || table[i].op == MURE_OP_WS)
                need += (int64_t)table[i].n_neurons * m->st[table[i].layer].K;
        FAILIF(need > out_len || (need > 0 && !out), c, MURE_ERR_INVALID_ARG, "out holds %lld values, %lld needed",
               (long long)out_len, (long long)need);
        // identity order so that offsets follow the table
        Groups g;
        g.order.resize(n_mutants);
        std::iota(g.order.begin(), g.order.end(), 0);
        g.begin.assign(m->L + 1, n_mutants);
        g.begin[0] = 0;
        Scratch sc(c);
        const DevTable dt = upload_table(c, sc, m, table, n_mutants, neuron_pool, pool_len, g, 1, out, offsets);
        c->launches += dt.expand_launches;
        CK(c, cudaStreamSynchronize(c->stream));
    });
}

}  // extern "C"
