// Dense layers on the 5th-generation tensor cores (tcgen05) with fp32-level accuracy:
// every fp32 operand a is split into two TF32 halves, a = a_hi + a_lo (a_hi = a
// rounded to TF32, a_lo = the rounded remainder), and each product uses three MMAs,
// a_hi*b_hi + a_hi*b_lo + a_lo*b_hi, accumulated in fp32 in tensor memory.
//
// One CTA of 4 warps computes a 128-row x N tile (N <= 256, a multiple of 16):
//   - all 128 threads stage the K-tile (32 values per row) of A (batch rows, with the
//     first suffix stage's mutated channels written over the cached rows) and of the
//     pre-split weights, split A, and store both halves in the 128-byte-swizzled
//     K-major layout the MMA reads;
//   - thread 0 issues 4 K-steps x 3 MMAs (kind::tf32, M=128, K=8) per K-tile and
//     commits them to the stage's mbarrier; two stages alternate, so staging tile
//     k+1 overlaps the MMAs of tile k;
//   - the epilogue reads the accumulator back with tcgen05.ld (thread = row = TMEM
//     lane), adds the bias, applies the activation and writes z and y rows.
// The K order of the accumulation is fixed and independent of the row's position in
// the tile, so a row gives the same bits in every batch (memoized == vanilla).
// Every mbarrier wait is bounded; on expiry the kernel records an error code, waits
// (bounded) for its outstanding MMAs, frees its tensor memory and returns.
#include <algorithm>

#include "common.cuh"
#include "device_util.cuh"

namespace mure {

namespace {

constexpr int kTileM = 128;
constexpr int kTileK = 32;                  // fp32 / tf32 values per 128-byte row
constexpr int kStages = 2;

__device__ __forceinline__ uint32_t smem_u32(const void *p)
{
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ float tf32_rna(float x)
{
    uint32_t r;
    asm("cvt.rna.tf32.f32 %0, %1;" : "=r"(r) : "f"(x));
    return __uint_as_float(r);
}

// Shared-memory matrix descriptor: K-major operand, 128-byte swizzle, 8-row groups
// 1024 bytes apart.
__device__ __forceinline__ uint64_t sw128_desc(uint32_t saddr)
{
    uint64_t d = 0;
    d |= (uint64_t)((saddr >> 4) & 0x3FFF);          // start address
    d |= (uint64_t)1 << 16;                          // leading byte offset (unused for swizzled K-major)
    d |= (uint64_t)(1024 >> 4) << 32;                // stride byte offset: next 8-row group
    d |= (uint64_t)1 << 46;                          // descriptor version
    d |= (uint64_t)2 << 61;                          // 128-byte swizzle
    return d;
}

// Instruction descriptor, kind::tf32: D fp32, A and B tf32, both K-major, M x N.
__host__ __device__ constexpr uint32_t idesc_tf32(int M, int N)
{
    return (1u << 4) | (2u << 7) | (2u << 10) | ((uint32_t)(N >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
}

// Byte offset of element (r, k), k < 32, in a 128-byte-swizzled K-major tile.
__device__ __forceinline__ uint32_t sw128_off(int r, int chunk)
{
    return (uint32_t)((r >> 3) * 1024 + (r & 7) * 128 + ((chunk ^ (r & 7)) << 4));
}

__device__ __forceinline__ void mbar_init(uint32_t a, uint32_t count)
{
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(a), "r"(count));
}

__device__ __forceinline__ bool mbar_try(uint32_t a, uint32_t parity)
{
    uint32_t ok;
    asm volatile(
        "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}\n"
        : "=r"(ok)
        : "r"(a), "r"(parity)
        : "memory");
    return ok != 0;
}

// Bounded wait: about a second of GPU time at most.
__device__ __forceinline__ bool mbar_wait(uint32_t a, uint32_t parity)
{
    const long long t0 = clock64();
    for (;;) {
        if (mbar_try(a, parity)) return true;
        if (clock64() - t0 > 2000000000LL) return false;
    }
}

__device__ __forceinline__ void mma_tf32(uint32_t d_tmem, uint64_t a, uint64_t b, uint32_t idesc, uint32_t acc)
{
    asm volatile(
        "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
        " tcgen05.mma.cta_group::1.kind::tf32 [%0], %1, %2, %3, p;\n}\n" ::"r"(d_tmem),
        "l"(a), "l"(b), "r"(idesc), "r"(acc));
}

__device__ __forceinline__ void mma_commit(uint32_t mbar)
{
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(mbar)
                 : "memory");
}

__device__ __forceinline__ void tmem_ld16(uint32_t taddr, float *v)
{
    uint32_t r[16];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
        : "r"(taddr));
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
    for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}

}  // namespace

struct TcDenseParams {
    const float *x; int64_t x_stride; int x_per_input;
    int64_t t0; int T; int R;
    int K, Kp, N, Np;            // fan-in (padded to 32), outputs (padded to 16)
    const float *Whi, *Wlo;      // [Np][Kp] TF32 halves of the weights
    const float *b;
    int act;
    float *z; int64_t z_stride;
    float *y; int64_t y_stride;
    Overlay ov;
    int *err;
};

// ncols: the power of two >= max(32, Np) tensor-memory columns this CTA allocates.
__global__ void __launch_bounds__(128, 1) k_tc_dense(const TcDenseParams p, int ncols)
{
    extern __shared__ __align__(1024) unsigned char smraw[];
    // 1024-byte aligned operand stages: [stage][A_hi, A_lo, B_hi, B_lo]
    unsigned char *sm = (unsigned char *)(((uintptr_t)smraw + 1023) & ~(uintptr_t)1023);
    const int n_base = blockIdx.y * 256;            // this CTA's output columns
    const int Nt = min(256, p.Np - n_base);        // a multiple of 16
    const int a_bytes = kTileM * 128, b_bytes = Nt * 128;
    const int stage_bytes = 2 * a_bytes + 2 * b_bytes;
    __shared__ __align__(8) uint64_t mbar[kStages];
    __shared__ uint32_t tmem_base_sh;
    __shared__ int wait_ok;   // thread 0's wait result, so every decision is CTA-uniform
    const int tid = threadIdx.x, warp = tid >> 5;
    const int64_t m0 = (int64_t)blockIdx.x * kTileM;

    if (warp == 0) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(&tmem_base_sh)),
                     "r"(ncols));
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
    }
    if (tid == 0) {
        for (int s = 0; s < kStages; ++s) mbar_init(smem_u32(&mbar[s]), 1);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    const uint32_t tmem = tmem_base_sh;

    // this thread's A row and its overlay
    const int64_t row = m0 + tid;
    const bool row_ok = row < p.R;
    const float *arow = nullptr;
    int ov_k = 0;
    const int32_t *ov_ids = nullptr;
    if (row_ok) {
        arow = p.x + (p.x_per_input ? p.t0 + row % p.T : row) * p.x_stride;
        if (p.ov.patch) {
            const int g = (int)(row / p.T);
            ov_k = p.ov.n_neurons[g];
            ov_ids = p.ov.ids + p.ov.neuron_off[g];
        }
    }
    const int nK = p.Kp / kTileK;
    uint32_t phase[kStages] = {0, 0};
    bool ok = true;
    // registers of the next K-tile, loaded one tile ahead so that their latency
    // overlaps the staging and MMAs of the current one
    float a[kTileK];
    float4 bh[kTileK / 4], bl[kTileK / 4];
    auto load_tile = [&](int k0) {
#pragma unroll
        for (int c = 0; c < kTileK / 4; ++c) {
            float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
            if (row_ok) {
                const int kk = k0 + 4 * c;
                if (kk + 3 < p.K) v = __ldg(reinterpret_cast<const float4 *>(arow + kk));
                else {
                    v.x = kk < p.K ? arow[kk] : 0.f;
                    v.y = kk + 1 < p.K ? arow[kk + 1] : 0.f;
                    v.z = kk + 2 < p.K ? arow[kk + 2] : 0.f;
                    v.w = kk + 3 < p.K ? arow[kk + 3] : 0.f;
                }
            }
            a[4 * c] = v.x; a[4 * c + 1] = v.y; a[4 * c + 2] = v.z; a[4 * c + 3] = v.w;
        }
        if (tid < Nt) {
            const float4 *h = reinterpret_cast<const float4 *>(p.Whi + (int64_t)(n_base + tid) * p.Kp + k0);
            const float4 *l = reinterpret_cast<const float4 *>(p.Wlo + (int64_t)(n_base + tid) * p.Kp + k0);
#pragma unroll
            for (int c = 0; c < kTileK / 4; ++c) { bh[c] = __ldg(h + c); bl[c] = __ldg(l + c); }
        }
    };
    load_tile(0);
    for (int kt = 0; kt < nK; ++kt) {
        const int s = kt % kStages;
        unsigned char *st = sm + s * stage_bytes;
        const int k0 = kt * kTileK;
        float ac[kTileK];
        float4 bhc[kTileK / 4], blc[kTileK / 4];
#pragma unroll
        for (int i = 0; i < kTileK; ++i) ac[i] = a[i];
#pragma unroll
        for (int c = 0; c < kTileK / 4; ++c) { bhc[c] = bh[c]; blc[c] = bl[c]; }
        if (kt + 1 < nK) load_tile(k0 + kTileK);
        if (kt >= kStages) {
            // the MMAs that read this stage two tiles ago must be done
            if (tid == 0) wait_ok = mbar_wait(smem_u32(&mbar[s]), phase[s]);
            __syncthreads();
            if (!wait_ok) { ok = false; break; }
            phase[s] ^= 1;
        }
        for (int q = 0; q < ov_k; ++q) {
            // mutated channels: elements k = c * ch + j of this K-tile
            const int j = ov_ids[q];
            const int cfirst = k0 - j <= 0 ? 0 : (k0 - j + p.ov.ch - 1) / p.ov.ch;
            for (int c = cfirst; c < p.ov.cells && c * p.ov.ch + j < k0 + kTileK; ++c) {
                const float pv = p.ov.patch[row * p.ov.row_stride + q * p.ov.cells + c];
#pragma unroll
                for (int i = 0; i < kTileK; ++i)
                    if (k0 + i == c * p.ov.ch + j) ac[i] = pv;
            }
        }
#pragma unroll
        for (int c = 0; c < kTileK / 4; ++c) {
            float4 hi, lo;
            hi.x = tf32_rna(ac[4 * c]);     lo.x = tf32_rna(ac[4 * c] - hi.x);
            hi.y = tf32_rna(ac[4 * c + 1]); lo.y = tf32_rna(ac[4 * c + 1] - hi.y);
            hi.z = tf32_rna(ac[4 * c + 2]); lo.z = tf32_rna(ac[4 * c + 2] - hi.z);
            hi.w = tf32_rna(ac[4 * c + 3]); lo.w = tf32_rna(ac[4 * c + 3] - hi.w);
            const uint32_t off = sw128_off(tid, c);
            *reinterpret_cast<float4 *>(st + off) = hi;
            *reinterpret_cast<float4 *>(st + a_bytes + off) = lo;
        }
        if (tid < Nt) {
#pragma unroll
            for (int c = 0; c < kTileK / 4; ++c) {
                const uint32_t off = sw128_off(tid, c);
                *reinterpret_cast<float4 *>(st + 2 * a_bytes + off) = bhc[c];
                *reinterpret_cast<float4 *>(st + 2 * a_bytes + b_bytes + off) = blc[c];
            }
        }
        // rows 128..255 of a 256-wide B tile
        for (int n = tid + kTileM; n < Nt; n += kTileM) {
            const float4 *h = reinterpret_cast<const float4 *>(p.Whi + (int64_t)(n_base + n) * p.Kp + k0);
            const float4 *l = reinterpret_cast<const float4 *>(p.Wlo + (int64_t)(n_base + n) * p.Kp + k0);
#pragma unroll
            for (int c = 0; c < kTileK / 4; ++c) {
                const uint32_t off = sw128_off(n, c);
                *reinterpret_cast<float4 *>(st + 2 * a_bytes + off) = __ldg(h + c);
                *reinterpret_cast<float4 *>(st + 2 * a_bytes + b_bytes + off) = __ldg(l + c);
            }
        }
        // make the generic-proxy stores visible to the tensor core, then issue
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        __syncthreads();
        if (tid == 0) {
            asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
            const uint32_t sa = smem_u32(st), sal = sa + a_bytes, sb = sa + 2 * a_bytes, sbl = sb + b_bytes;
            const uint32_t id = idesc_tf32(kTileM, Nt);
#pragma unroll
            for (int ks = 0; ks < kTileK / 8; ++ks) {
                const uint32_t adv = ks * 32;   // 8 TF32 values = 32 bytes along K
                const uint32_t acc0 = (kt > 0 || ks > 0) ? 1u : 0u;
                mma_tf32(tmem, sw128_desc(sal + adv), sw128_desc(sb + adv), id, acc0);   // a_lo * b_hi
                mma_tf32(tmem, sw128_desc(sa + adv), sw128_desc(sbl + adv), id, 1u);     // a_hi * b_lo
                mma_tf32(tmem, sw128_desc(sa + adv), sw128_desc(sb + adv), id, 1u);      // a_hi * b_hi
            }
            mma_commit(smem_u32(&mbar[s]));
        }
    }
    // wait for the outstanding commits (the last one covers every MMA issued)
    if (ok) {
        if (tid == 0) {
            int good = 1;
            for (int kt = max(0, nK - kStages); kt < nK && good; ++kt) {
                const int s = kt % kStages;
                good = mbar_wait(smem_u32(&mbar[s]), phase[s]);
            }
            wait_ok = good;
        }
        __syncthreads();
        ok = wait_ok != 0;
    }
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    if (!ok) {
        if (tid == 0) {
            atomicExch(p.err, MURE_ERR_TIMEOUT);
            // a bounded chance for the tensor core to finish before the memory goes
            const int last = nK - 1;
            if (last >= 0) mbar_wait(smem_u32(&mbar[last % kStages]), phase[last % kStages]);
        }
    } else {
        // epilogue: thread = row = TMEM lane (warp w holds lanes 32w .. 32w+31)
        const uint32_t lane_base = tmem + ((uint32_t)(warp * 32) << 16);
        for (int n0 = 0; n0 < Nt; n0 += 16) {
            float v[16];
            tmem_ld16(lane_base + n0, v);
            if (row_ok) {
#pragma unroll
                for (int c = 0; c < 4; ++c) {
                    const int n = n_base + n0 + 4 * c;
                    float zz[4], yy[4];
#pragma unroll
                    for (int i = 0; i < 4; ++i) {
                        zz[i] = n + i < p.N ? v[4 * c + i] + __ldg(p.b + n + i) : 0.f;
                        yy[i] = act_apply(p.act, zz[i]);
                    }
                    if (n + 3 < p.N) {
                        if (p.z) *reinterpret_cast<float4 *>(p.z + row * p.z_stride + n) = make_float4(zz[0], zz[1], zz[2], zz[3]);
                        *reinterpret_cast<float4 *>(p.y + row * p.y_stride + n) = make_float4(yy[0], yy[1], yy[2], yy[3]);
                    } else {
                        for (int i = 0; i < 4 && n + i < p.N; ++i) {
                            if (p.z) p.z[row * p.z_stride + n + i] = zz[i];
                            p.y[row * p.y_stride + n + i] = yy[i];
                        }
                    }
                }
            }
        }
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    if (warp == 0) asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(ncols));
}

// Split fp32 weights [N][K] into zero-padded TF32 halves [Np][Kp].
__global__ void k_split_weights(const float *__restrict__ W, int N, int K, int Np, int Kp, float *hi, float *lo)
{
    const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= (int64_t)Np * Kp) return;
    const int n = (int)(i / Kp), k = (int)(i % Kp);
    const float w = (n < N && k < K) ? W[(int64_t)n * K + k] : 0.f;
    const float h = tf32_rna(w);
    hi[i] = h;
    lo[i] = tf32_rna(w - h);
}

int tc_dense_supported(const Stage &S)
{
    return S.kind == MURE_NODE_DENSE && S.oc >= 16 && !S.has_add && !S.pool && !S.gap;
}

int launch_split_weights(const Stage &S, float *hi, float *lo, cudaStream_t s)
{
    const int Np = round_up16(S.oc), Kp = round_up32(S.K);
    const int64_t n = (int64_t)Np * Kp;
    k_split_weights<<<(unsigned)((n + 255) / 256), 256, 0, s>>>(S.W, S.oc, S.K, Np, Kp, hi, lo);
    return 1;
}

int launch_tc_dense(const Stage &S, Src x, RowMap rm, float *z_out, int64_t z_stride, float *y_out, int64_t y_stride,
                    cudaStream_t s, const Overlay *ov)
{
    if (rm.R <= 0) return 0;
    TcDenseParams p{};
    p.x = x.p; p.x_stride = x.stride; p.x_per_input = x.per_input;
    p.t0 = rm.t0; p.T = rm.T; p.R = rm.R;
    p.K = S.K; p.Kp = round_up32(S.K); p.N = S.oc; p.Np = round_up16(S.oc);
    p.Whi = S.Wtc_hi; p.Wlo = S.Wtc_lo; p.b = S.b; p.act = S.act1;
    p.z = z_out; p.z_stride = z_stride;
    p.y = y_out; p.y_stride = y_stride;
    if (ov) p.ov = *ov;
    p.err = S.err;
    const int nt = std::min(256, p.Np);
    int ncols = 32;
    while (ncols < nt) ncols <<= 1;
    const size_t smem = 1024 + (size_t)kStages * (2 * kTileM * 128 + 2 * nt * 128);
    cudaFuncSetAttribute(k_tc_dense, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    const dim3 grid((unsigned)((rm.R + kTileM - 1) / kTileM), (unsigned)((p.Np + 255) / 256));
    k_tc_dense<<<grid, kTileM, smem, s>>>(p, ncols);
    return 1;
}

}  // namespace mure
