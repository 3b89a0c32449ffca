// Dense and convolution layers on the 5th-generation tensor cores (tcgen05) with
// fp32-level accuracy: every fp32 operand a is split into two TF32 halves, a = a_hi +
// a_lo (a_hi = a rounded to TF32, a_lo = the rounded remainder), and each product
// uses three MMAs, a_hi*b_hi + a_hi*b_lo + a_lo*b_hi, accumulated in fp32 in tensor
// memory.  (The reduced-precision variant uses a_hi*b_hi alone.)
//
// The GEMM: M = (batch row, output position) pairs, K = the fan-in (ky, kx, ci), N =
// output channels.  A convolution is an implicit GEMM: the producer threads gather
// the im2col rows from the NHWC input.  One CTA of 4 warps computes a 128 x N tile
// (N <= 256, a multiple of 16):
//   - all 128 threads stage the K-tile (32 values per GEMM row) of A (batch rows, with
//     the first suffix stage's mutated channels written over the cached rows) and of
//     the pre-split weights, split A, and store the halves in the 128-byte-swizzled
//     K-major layout the MMA reads;
//   - thread 0 issues 4 K-steps x 3 MMAs (kind::tf32, M=128, K=8) per K-tile and
//     commits them to the stage's mbarrier; two stages alternate, so staging tile
//     k+1 overlaps the MMAs of tile k;
//   - the epilogue reads the accumulator back with tcgen05.ld (thread = GEMM row =
//     TMEM lane), adds the bias and applies activation, residual add and 2x2 max pool
//     (the four positions of a window are four consecutive lanes).
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

struct TcParams {
    const float *x; int64_t x_stride; int x_per_input;
    int64_t t0; int T; int R;
    int dense;                   // 1: a dense layer (one GEMM row per batch row)
    int ih, iw, ic, kh, kw, stride, pad, oh, ow;
    int P, pool, pw;             // GEMM rows per batch row (ordered as k_stage_simt)
    int K, Kp, N, Np;            // fan-in (padded to 32), outputs (padded to 16)
    const float *Whi, *Wlo;      // [Np][Kp] TF32 halves of the weights
    const float *b;
    int act1, has_add, act2;
    const float *skip; int64_t skip_stride; int skip_per_input; int sk_w, sk_c, sk_stride;
    float *z; int64_t z_stride;
    float *y; int64_t y_stride;
    int three;                   // 1: 3xTF32, 0: one TF32 MMA (reduced precision)
    Overlay ov;
    int *err;
};

__device__ __forceinline__ void cp_async16(uint32_t dst, const void *src, int src_bytes)
{
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(src_bytes) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory"); }

// One thread's GEMM row of an M-tile: batch row, output position, input row, overlay.
struct RowInfo {
    int64_t row;
    int oy, ox, py, px;
    const float *xrow;
    int ov_k;
    const int32_t *ov_ids;
    bool ok;
};

__device__ __forceinline__ RowInfo row_info(const TcParams &p, int64_t m)
{
    RowInfo ri{};
    ri.ok = m < (int64_t)p.R * p.P;
    if (!ri.ok) return ri;
    ri.row = m / p.P;
    const int q = (int)(m - ri.row * p.P);
    if (p.pool) {
        const int w = q >> 2, sub = q & 3;
        ri.py = w / p.pw; ri.px = w % p.pw;
        ri.oy = 2 * ri.py + (sub >> 1);
        ri.ox = 2 * ri.px + (sub & 1);
    } else {
        ri.oy = q / p.ow;
        ri.ox = q % p.ow;
    }
    ri.xrow = p.x + (p.x_per_input ? p.t0 + ri.row % p.T : ri.row) * p.x_stride;
    if (p.ov.patch) {
        const int g = (int)(ri.row / p.T);
        ri.ov_k = p.ov.n_neurons[g];
        ri.ov_ids = p.ov.ids + p.ov.neuron_off[g];
    }
    return ri;
}

// ncols: the power of two >= max(32, N tile) tensor-memory columns this CTA allocates.
// DENSE: one GEMM row per batch row; THREE: 3xTF32 (else one TF32 product).
// The CTA is persistent: it loops over M-tiles (blockIdx.x, += gridDim.x) with the
// operand pipeline running D = S-1 K-steps ahead across tile boundaries.
template <bool DENSE, bool THREE>
__global__ void __launch_bounds__(128, 1) k_tc_gemm(const TcParams p, int ncols, int S)
{
    extern __shared__ __align__(1024) unsigned char smraw[];
    // 1024-byte aligned operand stages: [stage][A_hi, A_lo, B_hi, B_lo]
    unsigned char *sm = (unsigned char *)(((uintptr_t)smraw + 1023) & ~(uintptr_t)1023);
    const int n_base = blockIdx.y * 256;            // this CTA's output columns
    const int Nt = min(256, p.Np - n_base);        // a multiple of 16
    const int a_bytes = kTileM * 128, b_bytes = Nt * 128;
    const int stage_bytes = THREE ? 2 * a_bytes + 2 * b_bytes : a_bytes + b_bytes;
    const int b_off = THREE ? 2 * a_bytes : a_bytes;
    constexpr int kMaxStages = 6;
    __shared__ __align__(8) uint64_t mbar[kMaxStages];
    __shared__ uint32_t tmem_base_sh;
    __shared__ int wait_ok;   // thread 0's wait result, so every decision is CTA-uniform
    const int tid = threadIdx.x, warp = tid >> 5;
    const int D = S - 1;
    const int64_t M = (int64_t)p.R * p.P;
    const int64_t n_tiles = (M + kTileM - 1) / kTileM;
    const int nK = p.Kp / kTileK;
    // this CTA's tiles: blockIdx.x, blockIdx.x + gridDim.x, ...
    const int64_t my_tiles = blockIdx.x < n_tiles ? (n_tiles - 1 - blockIdx.x) / gridDim.x + 1 : 0;
    const int64_t total = my_tiles * nK;

    if (warp == 0) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(&tmem_base_sh)),
                     "r"(ncols));
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
    }
    if (tid == 0) {
        for (int s = 0; s < S; ++s) mbar_init(smem_u32(&mbar[s]), 1);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    const uint32_t tmem = tmem_base_sh;
    // thread 0's bookkeeping of each stage's MMA commits (issued, waited for)
    uint32_t issued[kMaxStages] = {0, 0, 0, 0, 0, 0}, waited[kMaxStages] = {0, 0, 0, 0, 0, 0};
    auto wait_stage = [&](int s) -> bool {
        while (waited[s] < issued[s]) {
            if (!mbar_wait(smem_u32(&mbar[s]), waited[s] & 1)) return false;
            ++waited[s];
        }
        return true;
    };

    // queue the copies of K-step j (tile j / nK, K-tile j % nK) into its stage
    int64_t pf_tile = -1;
    RowInfo pf{};
    auto issue = [&](int64_t j) {
        const int64_t tile = blockIdx.x + (j / nK) * gridDim.x;
        const int kt = (int)(j % nK), s = (int)(j % S), k0 = kt * kTileK;
        if (tile != pf_tile) { pf = row_info(p, tile * kTileM + tid); pf_tile = tile; }
        const uint32_t st = smem_u32(sm + s * stage_bytes);
        if (DENSE) {
#pragma unroll
            for (int c = 0; c < kTileK / 4; ++c) {
                const int kk = k0 + 4 * c;
                const int nb = pf.ok ? max(0, min(16, (p.K - kk) * 4)) : 0;
                cp_async16(st + sw128_off(tid, c), nb ? (const void *)(pf.xrow + kk) : (const void *)p.b, nb);
            }
        } else if ((p.ic & 3) == 0) {
#pragma unroll
            for (int c = 0; c < kTileK / 4; ++c) {
                const int kk = k0 + 4 * c;
                const float *src = p.b;
                int nb = 0;
                if (pf.ok && kk < p.K) {
                    const int ci = kk % p.ic, t = kk / p.ic, kx = t % p.kw, ky = t / p.kw;
                    const int iy = pf.oy * p.stride - p.pad + ky, ix = pf.ox * p.stride - p.pad + kx;
                    if ((unsigned)iy < (unsigned)p.ih && (unsigned)ix < (unsigned)p.iw) {
                        src = pf.xrow + ((int64_t)iy * p.iw + ix) * p.ic + ci;
                        nb = 16;
                    }
                }
                cp_async16(st + sw128_off(tid, c), src, nb);
            }
        } else {
            // channels not a multiple of 4: plain loads, fp32 stored in place
            int ci = k0 % p.ic, t = k0 / p.ic, kx = t % p.kw, ky = t / p.kw;
            float v[kTileK];
#pragma unroll
            for (int i = 0; i < kTileK; ++i) {
                v[i] = 0.f;
                if (pf.ok && k0 + i < p.K) {
                    const int iy = pf.oy * p.stride - p.pad + ky, ix = pf.ox * p.stride - p.pad + kx;
                    if ((unsigned)iy < (unsigned)p.ih && (unsigned)ix < (unsigned)p.iw)
                        v[i] = __ldg(pf.xrow + ((int64_t)iy * p.iw + ix) * p.ic + ci);
                }
                if (++ci == p.ic) { ci = 0; if (++kx == p.kw) { kx = 0; ++ky; } }
            }
#pragma unroll
            for (int c = 0; c < kTileK / 4; ++c)
                *reinterpret_cast<float4 *>(sm + s * stage_bytes + sw128_off(tid, c)) =
                    make_float4(v[4 * c], v[4 * c + 1], v[4 * c + 2], v[4 * c + 3]);
        }
        for (int n = tid; n < Nt; n += kTileM) {
            const float *h = p.Whi + (int64_t)(n_base + n) * p.Kp + k0;
            const float *l = p.Wlo + (int64_t)(n_base + n) * p.Kp + k0;
#pragma unroll
            for (int c = 0; c < kTileK / 4; ++c) {
                cp_async16(st + b_off + sw128_off(n, c), h + 4 * c, 16);
                if (THREE) cp_async16(st + b_off + b_bytes + sw128_off(n, c), l + 4 * c, 16);
            }
        }
    };

    bool ok = true;
    for (int64_t j = 0; j < D; ++j) {
        if (j < total) issue(j);
        cp_async_commit();
    }
    int64_t cur_tile = -1;
    RowInfo ri{};
    for (int64_t it = 0; it < total; ++it) {
        const int64_t tile = blockIdx.x + (it / nK) * gridDim.x;
        const int kt = (int)(it % nK), s = (int)(it % S), k0 = kt * kTileK;
        if (tile != cur_tile) { ri = row_info(p, tile * kTileM + tid); cur_tile = tile; }
        unsigned char *st = sm + s * stage_bytes;
        // copies of this K-step have landed (each thread waits for its own, the
        // barrier makes everybody's visible)
        switch (D) {   // all but the D-1 most recent groups complete
        case 1: cp_async_wait<0>(); break;
        case 2: cp_async_wait<1>(); break;
        case 3: cp_async_wait<2>(); break;
        case 4: cp_async_wait<3>(); break;
        default: cp_async_wait<4>(); break;
        }
        __syncthreads();
        // split this row's 32 values into TF32 halves (the mutated channels first)
        {
            float ac[kTileK];
#pragma unroll
            for (int c = 0; c < kTileK / 4; ++c) {
                const float4 v = *reinterpret_cast<const float4 *>(st + sw128_off(tid, c));
                ac[4 * c] = v.x; ac[4 * c + 1] = v.y; ac[4 * c + 2] = v.z; ac[4 * c + 3] = v.w;
            }
            for (int q = 0; q < ri.ov_k; ++q) {
                const int jn = ri.ov_ids[q];
                if (DENSE) {
                    const int cfirst = k0 - jn <= 0 ? 0 : (k0 - jn + p.ov.ch - 1) / p.ov.ch;
                    for (int c = cfirst; c < p.ov.cells && c * p.ov.ch + jn < k0 + kTileK; ++c) {
                        const float pv = p.ov.patch[ri.row * p.ov.row_stride + q * p.ov.cells + c];
#pragma unroll
                        for (int i = 0; i < kTileK; ++i)
                            if (k0 + i == c * p.ov.ch + jn) ac[i] = pv;
                    }
                } else {
                    int ci = k0 % p.ic, t = k0 / p.ic, kx = t % p.kw, ky = t / p.kw;
#pragma unroll
                    for (int i = 0; i < kTileK; ++i) {
                        if (ci == jn && k0 + i < p.K) {
                            const int iy = ri.oy * p.stride - p.pad + ky, ix = ri.ox * p.stride - p.pad + kx;
                            if ((unsigned)iy < (unsigned)p.ih && (unsigned)ix < (unsigned)p.iw)
                                ac[i] = p.ov.patch[ri.row * p.ov.row_stride + q * p.ov.cells + iy * p.iw + ix];
                        }
                        if (++ci == p.ic) { ci = 0; if (++kx == p.kw) { kx = 0; ++ky; } }
                    }
                }
            }
#pragma unroll
            for (int c = 0; c < kTileK / 4; ++c) {
                float4 hi;
                hi.x = tf32_rna(ac[4 * c]);
                hi.y = tf32_rna(ac[4 * c + 1]);
                hi.z = tf32_rna(ac[4 * c + 2]);
                hi.w = tf32_rna(ac[4 * c + 3]);
                const uint32_t off = sw128_off(tid, c);
                *reinterpret_cast<float4 *>(st + off) = hi;
                if (THREE) {
                    const float4 lo = make_float4(tf32_rna(ac[4 * c] - hi.x), tf32_rna(ac[4 * c + 1] - hi.y),
                                                  tf32_rna(ac[4 * c + 2] - hi.z), tf32_rna(ac[4 * c + 3] - hi.w));
                    *reinterpret_cast<float4 *>(st + a_bytes + off) = lo;
                }
            }
        }
        // make the generic-proxy stores visible to the tensor core, then issue
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        __syncthreads();
        if (tid == 0) {
            asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
            const uint32_t sa = smem_u32(st), sal = sa + a_bytes, sb = sa + b_off, sbl = sb + b_bytes;
            const uint32_t id = idesc_tf32(kTileM, Nt);
#pragma unroll
            for (int ks = 0; ks < kTileK / 8; ++ks) {
                const uint32_t adv = ks * 32;   // 8 TF32 values = 32 bytes along K
                const uint32_t first = (kt > 0 || ks > 0) ? 1u : 0u;
                if (THREE) {
                    mma_tf32(tmem, sw128_desc(sal + adv), sw128_desc(sb + adv), id, first);   // a_lo * b_hi
                    mma_tf32(tmem, sw128_desc(sa + adv), sw128_desc(sbl + adv), id, 1u);      // a_hi * b_lo
                    mma_tf32(tmem, sw128_desc(sa + adv), sw128_desc(sb + adv), id, 1u);       // a_hi * b_hi
                } else {
                    mma_tf32(tmem, sw128_desc(sa + adv), sw128_desc(sb + adv), id, first);    // a_hi * b_hi
                }
            }
            mma_commit(smem_u32(&mbar[s]));
            ++issued[s];
        }
        // refill the stage the previous K-step's MMAs read, D steps ahead
        if (it + D < total) {
            if (tid == 0) wait_ok = wait_stage((int)((it + D) % S));
            __syncthreads();
            if (!wait_ok) { ok = false; break; }
            issue(it + D);
        }
        cp_async_commit();
        if (kt == nK - 1) {
            // the tile's accumulator is complete once its last commit has arrived
            if (tid == 0) wait_ok = wait_stage(s);
            __syncthreads();
            if (!wait_ok) { ok = false; break; }
            asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
            // epilogue: thread = GEMM row = TMEM lane (warp w holds lanes 32w .. 32w+31)
            const uint32_t lane_base = tmem + ((uint32_t)(warp * 32) << 16);
            const float *srow = nullptr;
            if (p.has_add && ri.ok) srow = p.skip + (p.skip_per_input ? p.t0 + ri.row % p.T : ri.row) * p.skip_stride;
            float *yrow = ri.ok ? p.y + ri.row * p.y_stride : nullptr;
            for (int n0 = 0; n0 < Nt; n0 += 16) {
                float v[16];
                tmem_ld16(lane_base + n0, v);
#pragma unroll
                for (int i = 0; i < 16; ++i) {
                    const int n = n_base + n0 + i;
                    const float zz = (ri.ok && n < p.N) ? v[i] + __ldg(p.b + n) : 0.f;
                    if (p.z && ri.ok && n < p.N) {
                        if (DENSE) p.z[ri.row * p.z_stride + n] = zz;
                        else p.z[ri.row * p.z_stride + (int64_t)n * (p.oh * p.ow) + ri.oy * p.ow + ri.ox] = zz;
                    }
                    float val = act_apply(p.act1, zz);
                    if (!DENSE && p.has_add && ri.ok && n < p.N) {
                        const float sv = n < p.sk_c
                            ? srow[((int64_t)ri.oy * p.sk_stride * p.sk_w + ri.ox * p.sk_stride) * p.sk_c + n]
                            : 0.f;
                        val = act_apply(p.act2, val + sv);
                    }
                    v[i] = val;
                }
                if (!DENSE && p.pool) {
                    // lanes 4w .. 4w+3 hold the four positions of one pooling window
                    const int lane = tid & 31;
#pragma unroll
                    for (int i = 0; i < 16; ++i) {
                        const float w1 = __shfl_down_sync(0xffffffffu, v[i], 1);
                        const float w2 = __shfl_down_sync(0xffffffffu, v[i], 2);
                        const float w3 = __shfl_down_sync(0xffffffffu, v[i], 3);
                        if ((lane & 3) == 0) v[i] = max4_first(v[i], w1, w2, w3);
                    }
                    if (ri.ok && (lane & 3) == 0) {
                        float *yo = yrow + ((int64_t)ri.py * p.pw + ri.px) * p.N;
#pragma unroll
                        for (int i = 0; i < 16; ++i)
                            if (n_base + n0 + i < p.N) yo[n_base + n0 + i] = v[i];
                    }
                } else if (ri.ok) {
                    float *yo = yrow + (DENSE ? 0 : ((int64_t)ri.oy * p.ow + ri.ox) * p.N);
                    const int nb = n_base + n0;
                    if (nb + 15 < p.N && ((p.N & 3) == 0)) {
#pragma unroll
                        for (int c = 0; c < 4; ++c)
                            *reinterpret_cast<float4 *>(yo + nb + 4 * c) =
                                make_float4(v[4 * c], v[4 * c + 1], v[4 * c + 2], v[4 * c + 3]);
                    } else {
#pragma unroll
                        for (int i = 0; i < 16; ++i)
                            if (nb + i < p.N) yo[nb + i] = v[i];
                    }
                }
            }
            // the next tile's first MMA overwrites the accumulator only after every
            // thread's reads (the barrier at the top of the next K-step)
            asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
        }
    }
    cp_async_wait<0>();
    if (!ok) {
        if (tid == 0) {
            atomicExch(p.err, MURE_ERR_TIMEOUT);
            // a bounded chance for the tensor core to finish before the memory goes
            for (int s = 0; s < S; ++s) wait_stage(s);
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

int tc_supported(const Stage &S)
{
    if (S.oc < 16) return 0;
    if (S.kind == MURE_NODE_DENSE) return !S.has_add && !S.pool && !S.gap;
    // implicit-GEMM convolution: pooled maps need whole windows per warp (always true:
    // a window is 4 consecutive GEMM rows and tiles start at multiples of 128)
    return S.kind == MURE_NODE_CONV2D;
}

int launch_split_weights(const Stage &S, float *hi, float *lo, cudaStream_t s)
{
    const int Np = round_up16(S.oc), Kp = round_up32(S.K);
    const int64_t n = (int64_t)Np * Kp;
    k_split_weights<<<(unsigned)((n + 255) / 256), 256, 0, s>>>(S.W, S.oc, S.K, Np, Kp, hi, lo);
    return 1;
}

int launch_tc(const Stage &S, Src x, RowMap rm, float *z_out, int64_t z_stride, Src skip, float *y_out,
              int64_t y_stride, float *gap_tmp, cudaStream_t s, const Overlay *ov)
{
    if (rm.R <= 0) return 0;
    TcParams p{};
    p.x = x.p; p.x_stride = x.stride; p.x_per_input = x.per_input;
    p.t0 = rm.t0; p.T = rm.T; p.R = rm.R;
    p.dense = S.kind == MURE_NODE_DENSE;
    p.ih = S.ih; p.iw = S.iw; p.ic = S.ic; p.kh = S.kh; p.kw = S.kw; p.stride = S.stride; p.pad = S.pad;
    p.oh = S.oh; p.ow = S.ow;
    p.pool = S.pool; p.pw = S.ow / 2;
    p.P = p.dense ? 1 : (S.pool ? 4 * (S.oh / 2) * (S.ow / 2) : S.oh * S.ow);
    p.K = S.K; p.Kp = round_up32(S.K); p.N = S.oc; p.Np = round_up16(S.oc);
    p.Whi = S.Wtc_hi; p.Wlo = S.Wtc_lo; p.b = S.b;
    p.act1 = S.act1; p.has_add = S.has_add; p.act2 = S.act2;
    p.skip = skip.p; p.skip_stride = skip.stride; p.skip_per_input = skip.per_input;
    p.sk_w = S.sk_w; p.sk_c = S.sc_c; p.sk_stride = S.sc_stride;
    p.z = z_out; p.z_stride = z_stride;
    // with global average pooling the post-op map goes to gap_tmp first
    const int mh = S.pool ? S.oh / 2 : S.oh, mw = S.pool ? S.ow / 2 : S.ow;
    const int64_t map_stride = round4((int64_t)mh * mw * S.oc);
    p.y = S.gap ? gap_tmp : y_out;
    p.y_stride = S.gap ? map_stride : y_stride;
    p.three = S.tc == 1;
    if (ov) p.ov = *ov;
    p.err = S.err;
    const int nt = std::min(256, p.Np);
    int ncols = 32;
    while (ncols < nt) ncols <<= 1;
    const size_t stage = p.three ? (2 * kTileM * 128 + 2 * nt * 128) : (kTileM * 128 + nt * 128);
    const int n_stages = (int)std::min<size_t>(6, (220 * 1024 - 1024) / stage);   // 2 .. 6 stages
    const size_t smem = 1024 + (size_t)n_stages * stage;
    const int64_t M = (int64_t)rm.R * p.P;
    const int64_t tiles = (M + kTileM - 1) / kTileM;
    // persistent CTAs: one per SM (per N slice), each looping over M-tiles
    const int n_sm = 152;
    const int ny = (p.Np + 255) / 256;
    const dim3 grid((unsigned)std::max<int64_t>(1, std::min<int64_t>(tiles, std::max(1, n_sm / ny))), (unsigned)ny);
    auto go = [&](auto kern) {
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        kern<<<grid, kTileM, smem, s>>>(p, ncols, n_stages);
    };
    if (p.dense) { if (p.three) go(k_tc_gemm<true, true>); else go(k_tc_gemm<true, false>); }
    else { if (p.three) go(k_tc_gemm<false, true>); else go(k_tc_gemm<false, false>); }
    int launches = 1;
    if (S.gap) launches += launch_gap(gap_tmp, map_stride, mh * mw, S.oc, rm.R, y_out, y_stride, s);
    return launches;
}

}  // namespace mure
