// Allocation-free variant of the GF / WS patch expansion (mure_expand_patches).
//
// Some callers cannot allocate device memory: an application whose own allocator
// has reserved the device's memory and cannot lend it, or a latency-critical loop
// that forbids allocator calls because cudaMalloc / cudaFree can synchronise the
// device.  This entry point serves them: it runs the same expansion kernel, with the
// kernel's scratch (its job table, the per-layer weight pointers and the Fisher-Yates
// permutation buffers) in one file-scope device array of fixed size, and writes the
// patches into a device buffer the caller provides.
#include <algorithm>
#include <cstring>
#include <mutex>
#include <new>
#include <vector>

#include "common.cuh"

namespace {

// The scratch.  Every GPU that loads this library holds it until the process exits.
constexpr size_t kNoallocScratchBytes = size_t(8) << 20;  // 8 MiB
static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoallocScratchBytes];

// Host code cannot use &g_noalloc_scratch as a device address (it names a host-side
// stand-in), so each device's address is looked up with that device current and kept
// once the lookup has succeeded; a failed lookup is retried by the next call.
constexpr int kMaxDevices = 256;
std::mutex g_scratch_mu;
unsigned char *g_scratch_ptr[kMaxDevices] = {};

size_t align256(size_t n) { return (n + 255) & ~size_t(255); }

mure_status fail(mure_ctx *c, mure_status st, const std::string &msg)
{
    c->err = msg;
    return st;
}

mure_status expand_noalloc(mure_ctx *c, mure_model *m, const mure_mutant *table, int64_t n_mutants,
                           const int32_t *neuron_pool, int64_t pool_len, float *out_dev, int64_t out_len,
                           int64_t *offsets)
{
    // the descriptor checks of mure_eval_mutants, then the flat-layout rule of
    // mure_expand_patches: the same status codes as the allocating entry point
    const mure_status st = mure::check_table_status(c, m, table, n_mutants, neuron_pool, pool_len);
    if (st != MURE_OK) return st;
    for (int64_t i = 0; i < n_mutants; ++i)
        if (table[i].tagged)
            return fail(c, MURE_ERR_UNSUPPORTED,
                        "mutant " + std::to_string(i) + ": tagged descriptors have no flat patch layout");
    if (n_mutants > 0 && !offsets) return fail(c, MURE_ERR_INVALID_ARG, "NULL offsets");
    if (c->device < 0 || c->device >= kMaxDevices) return fail(c, MURE_ERR_UNSUPPORTED, "device id out of range");

    // one expansion job per (mutant, neuron slot) of the GF / WS descriptors
    std::vector<mure::SlotJob> jobs;
    int64_t patch_len = 0, perm_len = 0;
    std::vector<int64_t> offs(n_mutants, -1);
    for (int64_t i = 0; i < n_mutants; ++i) {
        const mure_mutant &u = table[i];
        if ((u.op != MURE_OP_GF && u.op != MURE_OP_WS) || u.n_neurons == 0) continue;
        const int F = m->st[u.layer].K;
        offs[i] = patch_len;
        for (int q = 0; q < u.n_neurons; ++q) {
            mure::SlotJob jb{};
            jb.layer = u.layer; jb.op = u.op; jb.F = F; jb.j = neuron_pool[u.neuron_off + q]; jb.q = q;
            jb.param = u.param; jb.seed = u.seed;
            jb.out_off = patch_len + (int64_t)q * F;
            jb.perm_off = perm_len;
            if (u.op == MURE_OP_WS) perm_len += F;
            jobs.push_back(jb);
        }
        patch_len += (int64_t)u.n_neurons * F;
    }
    if (patch_len > out_len || (patch_len > 0 && !out_dev))
        return fail(c, MURE_ERR_INVALID_ARG, "out holds " + std::to_string(out_len) + " values, " +
                                                 std::to_string(patch_len) + " needed");
    // scratch layout: [L weight pointers][jobs][WS permutations]
    const size_t o_w = 0, o_jobs = align256(m->L * sizeof(float *));
    const size_t o_perm = o_jobs + align256(jobs.size() * sizeof(mure::SlotJob));
    const size_t need = o_perm + (size_t)perm_len * sizeof(int32_t);
    if (need > kNoallocScratchBytes)
        return fail(c, MURE_ERR_INVALID_ARG, "the descriptors need " + std::to_string(need) +
                                                 " bytes of scratch; the allocation-free entry point holds at most " +
                                                 std::to_string(kNoallocScratchBytes));
    if (jobs.empty()) {
        std::copy(offs.begin(), offs.end(), offsets);
        return MURE_OK;
    }

    // the call copies from pageable host memory and waits for its stream: neither is
    // allowed while the stream is being captured into a graph
    cudaStreamCaptureStatus cap = cudaStreamCaptureStatusNone;
    cudaError_t e = cudaStreamIsCapturing(c->stream, &cap);
    if (e != cudaSuccess) return fail(c, MURE_ERR_CUDA, std::string("cudaStreamIsCapturing: ") + cudaGetErrorString(e));
    if (cap != cudaStreamCaptureStatusNone)
        return fail(c, MURE_ERR_INVALID_ARG, "the context's stream is being captured");
    e = cudaSetDevice(c->device);
    if (e != cudaSuccess) return fail(c, MURE_ERR_CUDA, std::string("cudaSetDevice: ") + cudaGetErrorString(e));
    unsigned char *scratch = nullptr;
    {
        std::lock_guard<std::mutex> lk(g_scratch_mu);
        if (!g_scratch_ptr[c->device]) {
            void *p = nullptr;
            e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
            if (e != cudaSuccess || !p) {
                cudaGetLastError();
                return fail(c, MURE_ERR_CUDA, std::string("cudaGetSymbolAddress: ") + cudaGetErrorString(e));
            }
            g_scratch_ptr[c->device] = static_cast<unsigned char *>(p);
        }
        scratch = g_scratch_ptr[c->device];
    }

    // one host staging copy of the job table and weight pointers into the scratch
    std::vector<unsigned char> host(o_perm);
    std::vector<const float *> Wp(m->L);
    for (int l = 0; l < m->L; ++l) Wp[l] = m->st[l].W;
    memcpy(host.data() + o_w, Wp.data(), m->L * sizeof(float *));
    memcpy(host.data() + o_jobs, jobs.data(), jobs.size() * sizeof(mure::SlotJob));
    e = cudaMemcpyAsync(scratch, host.data(), o_perm, cudaMemcpyHostToDevice, c->stream);
    if (e != cudaSuccess) return fail(c, MURE_ERR_CUDA, std::string("cudaMemcpyAsync: ") + cudaGetErrorString(e));
    mure::ExpandArgs ea{};
    ea.jobs = reinterpret_cast<const mure::SlotJob *>(scratch + o_jobs);
    ea.n_jobs = (int64_t)jobs.size();
    ea.sigma = m->sigma_dev;
    ea.W = reinterpret_cast<const float *const *>(scratch + o_w);
    ea.patch = out_dev;
    // the kernel initialises every permutation entry it reads, so nothing in the
    // scratch has to start at zero or survives from an earlier call
    ea.perm = reinterpret_cast<int32_t *>(scratch + o_perm);
    ea.ws_as_weights = 1;
    c->launches += mure::launch_expand(ea, c->stream);
    e = cudaGetLastError();
    if (e == cudaSuccess) e = cudaStreamSynchronize(c->stream);
    if (e != cudaSuccess) return fail(c, MURE_ERR_CUDA, std::string("expansion: ") + cudaGetErrorString(e));
    std::copy(offs.begin(), offs.end(), offsets);
    return MURE_OK;
}

}  // namespace

extern "C" mure_status mure_expand_patches_noalloc(mure_model *m, const mure_mutant *table, int64_t n_mutants,
                                                   const int32_t *neuron_pool, int64_t pool_len, float *out_dev,
                                                   int64_t out_len, int64_t *offsets)
{
    if (!m) return MURE_ERR_INVALID_ARG;
    mure_ctx *c = m->ctx;
    c->err.clear();
    // host containers sized by the caller's table: a failed host allocation is a
    // status, never an exception across the C ABI
    try {
        return expand_noalloc(c, m, table, n_mutants, neuron_pool, pool_len, out_dev, out_len, offsets);
    } catch (const std::bad_alloc &) {
        c->err = "host allocation failed";
        return MURE_ERR_OOM;
    }
}
