// Dense and convolution layers on the 5th-generation tensor cores (tcgen05) with
// fp32-level accuracy: every fp32 operand a is split into two TF32 halves, a = a_hi +
// a_lo (a_hi = a rounded to TF32, a_lo = the rounded remainder), and each product
// uses three MMAs, a_lo*b_hi + a_hi*b_lo + a_hi*b_hi, accumulated in fp32 in tensor
// memory.  (The reduced-precision variant uses a_hi*b_hi alone.)
//
// The GEMM: M = (batch row, output position) pairs, K = the fan-in (ky, kx, ci), N =
// output channels (a CTA takes a slice of <= 128).  A convolution is an implicit
// GEMM: the producers gather the im2col rows from the NHWC input.  The CTA is
// persistent (one per SM) and warp-specialised:
//   warps 0-3  producers: thread = GEMM row = tensor-memory lane.  Each streams its
//              row's 32-value K-steps into a private shared-memory ring with
//              cp.async, several steps ahead (the first suffix stage's mutated
//              channels are fetched from the patch buffer instead of the cached row),
//              splits them into TF32 halves and stores the halves into a tensor-memory
//              A stage (tcgen05.st); the MMA reads A from tensor memory, so the
//              operand never goes through shared memory a second time;
//   warps 8-10 MMA issue (kind::tf32, M=128, K=8): one thread issues an MMA only about
//              every 120 cycles, whatever N is, so where tensor memory allows, a
//              K-step's MMAs are dealt to up to three warps, each accumulating into its
//              own partial accumulator; the epilogue adds the partials in a fixed order;
//   warp 11    one thread moves the weights: pre-split, pre-swizzled K-step chunks
//              (one bulk copy each), or the whole slice once when it fits;
//   warps 4-7  epilogue: two accumulator sets alternate, so the bias / activation /
//              residual / 2x2 pool / store of tile i overlaps the MMAs of tile i+1;
//              unpooled rows go out through shared memory in coalesced stores.
// The K order of the accumulation is fixed and independent of the row's position in
// the tile, so a row gives the same bits in every batch (memoized == vanilla).
// Every wait is bounded; on expiry the kernel records an error code, stops every
// role, lets its own copies and MMAs drain (bounded), frees its tensor memory and
// returns.
#include <algorithm>
#include <cuda.h>
#include <cudaTypedefs.h>

#include "common.cuh"
#include "device_util.cuh"
#include "epilogue.cuh"

namespace mure {

namespace {

constexpr int kTileM = 128;
constexpr int kTileK = 32;             // fp32 / tf32 values per 128-byte row
constexpr int kNA = 4;                 // producer cp.async ring depth (K-steps)
constexpr int kNB = 3;                 // streamed weight stages
constexpr int kSlice = 128;            // output channels per CTA (the default N slice)
constexpr int kSliceMax = 256;         // wide slice: one N = 256 MMA per K8 step (staged convolutions)
constexpr int kFuseClasses = 12;       // classes of an output layer fused into a dense epilogue
constexpr int kThreads = 384;          // 4 producer + 4 epilogue + 3 MMA + weight warps
constexpr int kEpiStride = 36;         // floats per row of an epilogue staging chunk (32 + pad)
constexpr int kMaxNT = 8;              // tensor-memory A stages, at most
constexpr int kNBufMax = 4;            // staging buffers (small-image and staged-convolution modes)
constexpr uint32_t kStageA = kTileM * 128;   // bytes of one producer ring slot
constexpr long long kSpin = 2000000000LL;    // default wait limit: about a second at the SM clock

// The CTA's abort state: set by the role whose wait ran out (after `limit` cycles), seen
// by every other role's waits.
struct WaitCtl {
    int abort;
    long long limit;
};

__device__ __forceinline__ uint32_t smem_u32(const void *p)
{
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

// The high TF32 half of a finite fp32 value on the integer pipes: add half a unit in
// the last TF32 place to the magnitude bits and clear the 13 low bits (round to
// nearest, ties away from zero).  The remainder x - hi is exact in fp32; the MMA reads
// only its top 19 bits.  (The conversion instruction runs on a slow pipe and was the
// producers' bottleneck.)
__device__ __forceinline__ float tf32_hi(float x)
{
    return __uint_as_float((__float_as_uint(x) + 0x1000u) & 0xFFFFE000u);
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

// Byte offset of 16-byte chunk `chunk` of row r in a 128-byte-swizzled K-major tile.
__host__ __device__ __forceinline__ uint32_t sw128_off(int r, int chunk)
{
    return (uint32_t)(r * 128 + ((chunk ^ (r & 7)) << 4));
}

__device__ __forceinline__ void mbar_init(uint32_t a, uint32_t count)
{
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(a), "r"(count));
}

__device__ __forceinline__ void mbar_arrive(uint32_t a)
{
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(a) : "memory");
}

__device__ __forceinline__ void mbar_expect_tx(uint32_t a, uint32_t bytes)
{
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(a), "r"(bytes) : "memory");
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

// Wait for the phase of parity `parity`, polling every ~NS nanoseconds (a sleeping
// warp leaves the issue slots of its SM sub-partition to the producers); false when
// another role has aborted or the wait limit has passed (then this role aborts the
// CTA).
template <int NS = 0>
__device__ __forceinline__ bool wait_phase(uint32_t a, uint32_t parity, volatile WaitCtl *abort_flag)
{
    if (mbar_try(a, parity)) return true;
    const long long t0 = clock64();
    for (;;) {
        if (NS > 0) __nanosleep(NS);
        if (mbar_try(a, parity)) return true;
        if (abort_flag->abort) return false;
        if (clock64() - t0 > abort_flag->limit) { abort_flag->abort = 1; return false; }
    }
}

// The same for a whole warp: every lane polls, the verdict is the warp's AND, so the
// .sync.aligned tensor-memory instructions that follow see a converged warp.
template <int NS = 0>
__device__ __forceinline__ bool warp_wait_phase(uint32_t a, uint32_t parity, volatile WaitCtl *abort_flag)
{
    const bool ok = wait_phase<NS>(a, parity, abort_flag);
    return __all_sync(0xffffffffu, ok);
}

// Teardown wait: bounded by the default limit whatever the CTA's limit, ignores the
// abort flag, so that copies and MMAs in flight land before shared and tensor memory
// are released.
__device__ __forceinline__ void wait_phase_drain(uint32_t a, uint32_t parity)
{
    const long long t0 = clock64();
    while (!mbar_try(a, parity))
        if (clock64() - t0 > kSpin) return;
}

// A from tensor memory, B from shared memory.
__device__ __forceinline__ void mma_tf32_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t b, uint32_t idesc, uint32_t acc)
{
    asm volatile(
        "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
        " tcgen05.mma.cta_group::1.kind::tf32 [%0], [%1], %2, %3, p;\n}\n" ::"r"(d_tmem),
        "r"(a_tmem), "l"(b), "r"(idesc), "r"(acc));
}

// MMAs q = LO .. HI-1 of a K-step, q = ks * kTerms + term (3xTF32: a_lo*b_hi,
// a_hi*b_lo, a_hi*b_hi for K8 step ks), into accumulator d; the first one overwrites
// unless acc0.  Fully unrolled: scalar work between two MMAs adds its latency to the
// issuing thread's MMA rate.
template <bool THREE, int LO, int HI>
__device__ __forceinline__ void mma_block(uint32_t d, uint32_t ta, uint64_t dh, uint64_t dl, uint32_t id, uint32_t acc0)
{
    constexpr int kTerms = THREE ? 3 : 1;
#pragma unroll
    for (int q = LO; q < HI; ++q) {
        const int ks = q / kTerms, term = q % kTerms;
        const uint32_t acc = q > LO ? 1u : acc0;
        // K8 step ks starts 32 bytes further along the swizzled rows: +2 in the
        // descriptor's 16-byte address field
        if (!THREE || term == 2) mma_tf32_ts(d, ta + ks * 8, dh + 2 * ks, id, acc);    // a_hi * b_hi
        else if (term == 0) mma_tf32_ts(d, ta + 32 + ks * 8, dh + 2 * ks, id, acc);   // a_lo * b_hi
        else mma_tf32_ts(d, ta + ks * 8, dl + 2 * ks, id, acc);                       // a_hi * b_lo
    }
}

// The same three products per K8 step in two MMAs (merge_lo): a_hi * [b_hi | b_lo] with
// instruction descriptor id2 (N = 2 Nt), then a_lo * b_hi with id1 (N = Nt).  A narrow MMA
// occupies the tensor pipe about as long as one of twice its width, so two instructions
// per K8 step instead of three.
__device__ __forceinline__ void mma_block_merged(uint32_t d, uint32_t ta, uint64_t dh, uint32_t id2, uint32_t id1,
                                                 uint32_t acc0)
{
#pragma unroll
    for (int ks = 0; ks < 4; ++ks) {
        mma_tf32_ts(d, ta + ks * 8, dh + 2 * ks, id2, ks > 0 ? 1u : acc0);   // a_hi * [b_hi | b_lo]
        mma_tf32_ts(d, ta + 32 + ks * 8, dh + 2 * ks, id1, 1u);              // a_lo * b_hi
    }
}

__device__ __forceinline__ void mma_commit(uint32_t mbar)
{
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(mbar)
                 : "memory");
}

__device__ __forceinline__ void bulk_g2s(uint32_t dst, const void *src, uint32_t bytes, uint32_t mbar)
{
    asm volatile("cp.async.bulk.shared::cta.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
                 "l"(src), "r"(bytes), "r"(mbar)
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

// Thread t's 32 values go to lane (warp quadrant) t, columns taddr .. taddr+31.
__device__ __forceinline__ void tmem_st32(uint32_t taddr, const float *v)
{
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,"
        "%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};" ::"r"(taddr),
        "r"(__float_as_uint(v[0])), "r"(__float_as_uint(v[1])), "r"(__float_as_uint(v[2])),
        "r"(__float_as_uint(v[3])), "r"(__float_as_uint(v[4])), "r"(__float_as_uint(v[5])),
        "r"(__float_as_uint(v[6])), "r"(__float_as_uint(v[7])), "r"(__float_as_uint(v[8])),
        "r"(__float_as_uint(v[9])), "r"(__float_as_uint(v[10])), "r"(__float_as_uint(v[11])),
        "r"(__float_as_uint(v[12])), "r"(__float_as_uint(v[13])), "r"(__float_as_uint(v[14])),
        "r"(__float_as_uint(v[15])), "r"(__float_as_uint(v[16])), "r"(__float_as_uint(v[17])),
        "r"(__float_as_uint(v[18])), "r"(__float_as_uint(v[19])), "r"(__float_as_uint(v[20])),
        "r"(__float_as_uint(v[21])), "r"(__float_as_uint(v[22])), "r"(__float_as_uint(v[23])),
        "r"(__float_as_uint(v[24])), "r"(__float_as_uint(v[25])), "r"(__float_as_uint(v[26])),
        "r"(__float_as_uint(v[27])), "r"(__float_as_uint(v[28])), "r"(__float_as_uint(v[29])),
        "r"(__float_as_uint(v[30])), "r"(__float_as_uint(v[31]))
        : "memory");
}

__device__ __forceinline__ void cp_async16(uint32_t dst, const void *src, int src_bytes)
{
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(src_bytes) : "memory");
}
__device__ __forceinline__ void cp_async4(uint32_t dst, const void *src, int src_bytes)
{
    asm volatile("cp.async.ca.shared.global [%0], [%1], 4, %2;" ::"r"(dst), "l"(src), "r"(src_bytes) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory"); }

}  // namespace

struct TcParams {
    const float *x; int64_t x_stride; int x_per_input;
    int64_t t0; int T; int R;
    const int32_t *lrow;         // compacted batch: logical row of each physical row, else null
    int ih, iw, ic, kh, kw, stride, pad, oh, ow;
    int P, pool, pw;             // GEMM rows per batch row (pooled maps: window-major)
    int K, Kp, N, Np;            // fan-in (padded to 32), outputs (padded to 16)
    const float *Wsw;            // pre-split, pre-swizzled weight chunks (see k_swizzle_weights)
    int64_t w_slice_floats;      // distance between the N slices' chunk sequences
    int b_resident;              // 1: the CTA's whole weight slice sits in shared memory
    const float *b;
    int act1, has_add, act2;
    const float *skip; int64_t skip_stride; int skip_per_input; int sk_w, sk_c, sk_stride;
    float *z; int64_t z_stride;
    float *y; int64_t y_stride;
    Overlay ov;                  // mutated channels of the input rows (ov.patch null: none)
    int n_mma;                   // MMA-issuing warps
    int n_part;                  // partial accumulators per set: n_mma, or 1 when the warps
                                 // take turns (mma_chain)
    int mma_chain;               // 1: the issuing warps take the K-steps in turn, in K-step
                                 // order, into one accumulator (handed over by barrier arrivals)
    int cv_win;                  // MODE 3: a GEMM row per 2x2 output window (rows: windows
                                 // (py, px), origin (2 py, 2 px); N = 4 positions x N outputs;
                                 // taps of a 4x4 field)
    int cv_fw, cv_ntap;          // MODE 3: the taps' field width (kw, or 4) and count
    int cv_pair;                 // MODE 3: units of two 128-row tiles (rows r and 128 + r per
                                 // producer thread; MMA warp w issues tile w; one weight stage
                                 // serves both)
    int merge_lo;                // 3xTF32 with narrow slices (Nt <= 64): a_hi * [b_hi | b_lo] as
                                 // one MMA of width 2 Nt (the lo weight panel follows the hi
                                 // panel) plus a_lo * b_hi; the accumulator's columns Nt .. 2 Nt
                                 // hold the a_hi * b_lo sums, added to columns 0 .. Nt last
    int acc_cols;                // tensor-memory columns of one partial accumulator
    int n_acc;                   // accumulator sets (tiles in flight): 1 or 2
    int n_stages;                // tensor-memory A stages (<= kMaxNT), from column a_col
    int slice_w;                 // output channels per CTA: kSlice, or kSliceMax for a wide slice
    int nb;                      // streamed weight stages (<= kNB)
    int a_col;
    int *err;
    long long spin;              // wait limit in SM cycles (0: the default, about a second)
    FinalFuse ff;                // the output layer computed in the epilogue (FCP > 0)
    SlotStore slot;              // slot.out: the tensor-core delta's scattered store
    // dense layers: A tiles (128 rows x one K-step) by tensor-map copies from warp 10
    // instead of the producers' 16-byte copies; tile m0 starts at row coordinate m0
    int a_tma;
    CUtensorMap tmap_a;
    // MODE 3 (staged convolution): each tile's input rows with their zero border, 32
    // channels at a time, land by tensor-map copies in a ring of cv_nbuf buffers; the
    // producers gather every tap's 32 values from there.  K order: (chunk, tap, channel)
    int cv_cw;                   // channels per chunk: 32, or 16 (a K-step then holds two taps;
                                 // the copies still stage 32-channel lines, the upper 16 zero-filled)
    int cv_taps;                 // K-steps per chunk
    int cv_nchunk;               // chunks of cv_cw input channels
    int cv_imgs, cv_rows;        // batch rows per tile; output rows per tile and batch row
    int cv_hw, cv_hh;            // staged width and height (input pixels, border included)
    uint32_t cv_img_bytes;       // one batch row's staged chunk in shared memory
    int cv_nbuf;
    CUtensorMap tmap_x;          // the input rows as [row][ih][iw][ic]: boxes {32, cv_hw, cv_hh, 1}
};

// Per producer ring slot, the overlay values of a row's K-step: up to kOvMax
// (position, value) entries, the values fetched by cp.async into ov_val.
constexpr int kOvMax = 8;
constexpr uint32_t kOvSlotBytes = kTileM * (kOvMax * 4 + kOvMax + 4);   // values, positions, count

// One GEMM row of an M-tile: batch row, output position, input row, overlay.
struct RowInfo {
    int64_t row;
    int oy, ox, py, px;
    const float *xrow;
    int ov_k;
    const int32_t *ov_ids;
    const float *ov_patch;
    int ov_pos[4], ov_c[4];   // dense overlay walk: next position j + c * ch of slots 0..3
    bool ok;
};

template <bool DENSE, bool OVERLAY = true>
__device__ __forceinline__ RowInfo row_info(const TcParams &p, int64_t m)
{
    RowInfo ri{};
    ri.ok = m < (int64_t)p.R * p.P;
    if (!ri.ok) return ri;
    if (DENSE) {
        ri.row = m;
    } else {
        ri.row = m / p.P;
        const int q = (int)(m - ri.row * p.P);
        if (p.pool) {
            const int w = q >> 2, sub = q & 3;
            ri.py = w / p.pw; ri.px = w % p.pw;
            ri.oy = 2 * ri.py + (sub >> 1);
            ri.ox = 2 * ri.px + (sub & 1);
        } else if (p.cv_win) {
            // a 2x2 output window: its top-left position
            ri.py = q / p.pw; ri.px = q % p.pw;
            ri.oy = 2 * ri.py;
            ri.ox = 2 * ri.px;
        } else {
            ri.oy = q / p.ow;
            ri.ox = q % p.ow;
        }
    }
    // per-input sources, the overlay and its group by the logical row; the batch's own
    // row buffers by the physical row
    const int64_t lr = logical_row(p.lrow, ri.row);
    ri.xrow = p.x + (p.x_per_input ? p.t0 + lr % p.T : ri.row) * p.x_stride;
    if (OVERLAY && p.ov.patch) {
        const int g = (int)(lr / p.T);
        ri.ov_k = p.ov.n_neurons[g];
        ri.ov_ids = p.ov.ids + p.ov.neuron_off[g];
        ri.ov_patch = p.ov.patch + lr * p.ov.row_stride;
        if (DENSE) {
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                ri.ov_c[q] = 0;
                ri.ov_pos[q] = q < ri.ov_k ? ri.ov_ids[q] : 0;
            }
        }
    }
    return ri;
}

// The rows a producer lane copies for its warp: lane l copies 16-byte chunk l & 7 of
// rows 4c + (l >> 3), c = 0..7, of the warp's 32 GEMM rows, so that one copy
// instruction covers four whole 128-byte row segments (a thread copying its own row
// would touch 32 rows per instruction and saturate the load/store unit).
struct LoadRows {
    const float *xrow[8];   // null: row past the end
    int oy[8], ox[8];
    int ci, kx, ky;         // convolution: (ky, kx, ci) of this lane's 4-value chunk at the next K-step
};

template <bool DENSE>
__device__ __forceinline__ void load_rows(const RowInfo &pf, LoadRows &lr)
{
    const int lane = threadIdx.x & 31;
#pragma unroll
    for (int c = 0; c < 8; ++c) {
        const int src = 4 * c + (lane >> 3);
        const unsigned long long xp =
            __shfl_sync(0xffffffffu, (unsigned long long)(uintptr_t)(pf.ok ? pf.xrow : nullptr), src);
        lr.xrow[c] = reinterpret_cast<const float *>((uintptr_t)xp);
        if (!DENSE) {
            lr.oy[c] = __shfl_sync(0xffffffffu, pf.oy, src);
            lr.ox[c] = __shfl_sync(0xffffffffu, pf.ox, src);
        }
    }
}

// The chunk cursor of a convolution's first K-step: k = 4 * (lane mod 8).
__device__ __forceinline__ void chunk_cursor(const TcParams &p, LoadRows &lr)
{
    const int kk = 4 * ((threadIdx.x & 31) & 7);
    const int t = kk / p.ic;
    lr.ci = kk - t * p.ic;
    lr.kx = t % p.kw;
    lr.ky = t / p.kw;
}

// Queue the cp.async copies of K-step k0 .. k0+31 of the warp's 32 GEMM rows into
// their 128-byte rows of `slot` (swizzled like the MMA operand layout, so that each
// thread's read-back of its own row is free of bank conflicts).  Values past the
// fan-in, outside the image (zero padding) or of rows past the end are zero-filled.
// The mutated channels of the first suffix stage: the row owner (thread r) fetches
// their patch values into the slot's overlay entries (ov), written over its row once
// the copies have landed.
template <bool DENSE>
__device__ __forceinline__ void produce_issue(const TcParams &p, RowInfo &pf, LoadRows &lr, int r, uint32_t slot,
                                              uint32_t ov, int k0)
{
    const float *dummy = p.b;   // a valid address for zero-byte copies
    const int lane = r & 31, wbase = r & ~31, ch = lane & 7;
    int cnt = 0;
    auto entry = [&](int pos, const float *src) {
        if (cnt < kOvMax) {
            cp_async4(ov + (uint32_t)(cnt * kTileM + r) * 4, src, 4);
            asm volatile("st.shared.u8 [%0], %1;" ::"r"(ov + kTileM * kOvMax * 4 + cnt * kTileM + r), "r"(pos));
        } else {
            atomicExch(p.err, MURE_ERR_UNSUPPORTED);   // the host keeps the entry count in range
        }
        ++cnt;
    };
    if (DENSE) {
        const int kk = k0 + 4 * ch;
        const int nbk = max(0, min(16, (p.K - kk) * 4));
#pragma unroll
        for (int c = 0; c < 8; ++c) {
            const int row = wbase + 4 * c + (lane >> 3);
            const int nb = lr.xrow[c] ? nbk : 0;
            cp_async16(slot + sw128_off(row, ch), nb ? (const void *)(lr.xrow[c] + kk) : (const void *)dummy, nb);
        }
        // overlay positions are c * ch + j (cell c of mutated channel j); the K-steps of a
        // row come in ascending k, so each slot keeps a cursor
        const int nq = min(pf.ov_k, 4);
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            if (q >= nq) break;
            while (pf.ov_c[q] < p.ov.cells && pf.ov_pos[q] < k0 + kTileK) {
                entry(pf.ov_pos[q] - k0, pf.ov_patch + q * p.ov.cells + pf.ov_c[q]);
                pf.ov_pos[q] += p.ov.ch;
                ++pf.ov_c[q];
            }
        }
    } else if ((p.ic & 3) == 0) {
        // 16-byte chunks: 4 channels of one input pixel; this lane's chunk has the same
        // (ky, kx, ci) in all its rows
        const int kk = k0 + 4 * ch;
        const int ci = lr.ci, kx = lr.kx, ky = lr.ky;
        // the cursor of the next K-step, 32 values on (no divisions per K-step)
        lr.ci += kTileK;
        while (lr.ci >= p.ic) {
            lr.ci -= p.ic;
            if (++lr.kx == p.kw) { lr.kx = 0; ++lr.ky; }
        }
#pragma unroll
        for (int c = 0; c < 8; ++c) {
            const int row = wbase + 4 * c + (lane >> 3);
            const int iy = lr.oy[c] * p.stride - p.pad + ky, ix = lr.ox[c] * p.stride - p.pad + kx;
            const bool in = lr.xrow[c] && kk < p.K && (unsigned)iy < (unsigned)p.ih && (unsigned)ix < (unsigned)p.iw;
            cp_async16(slot + sw128_off(row, ch), in ? lr.xrow[c] + ((int64_t)iy * p.iw + ix) * p.ic + ci : dummy,
                       in ? 16 : 0);
        }
        if (pf.ov_k > 0) {
            // the owner's mutated channels in its own row
            int ci2 = k0 % p.ic, t2 = k0 / p.ic, kx2 = t2 % p.kw, ky2 = t2 / p.kw;
            for (int c = 0; c < kTileK / 4; ++c) {
                const int iy = pf.oy * p.stride - p.pad + ky2, ix = pf.ox * p.stride - p.pad + kx2;
                const bool in = k0 + 4 * c < p.K && (unsigned)iy < (unsigned)p.ih && (unsigned)ix < (unsigned)p.iw;
                if (in)
                    for (int q = 0; q < pf.ov_k; ++q) {
                        const int jn = pf.ov_ids[q];
                        if (jn >= ci2 && jn < ci2 + 4)
                            entry(4 * c + jn - ci2, pf.ov_patch + q * p.ov.cells + iy * p.iw + ix);
                    }
                ci2 += 4;
                if (ci2 == p.ic) { ci2 = 0; if (++kx2 == p.kw) { kx2 = 0; ++ky2; } }
            }
        }
    } else {
        // channel counts that are not a multiple of 4: 4-byte copies of the thread's own
        // row, the patch value taken directly for a mutated channel
        int ci = k0 % p.ic, t = k0 / p.ic, kx = t % p.kw, ky = t / p.kw;
        for (int i = 0; i < kTileK; ++i) {
            const int k = k0 + i;
            const int iy = pf.oy * p.stride - p.pad + ky, ix = pf.ox * p.stride - p.pad + kx;
            const bool in = pf.ok && k < p.K && (unsigned)iy < (unsigned)p.ih && (unsigned)ix < (unsigned)p.iw;
            const float *src = in ? pf.xrow + ((int64_t)iy * p.iw + ix) * p.ic + ci : dummy;
            if (in)
                for (int q = 0; q < pf.ov_k; ++q)
                    if (pf.ov_ids[q] == ci) src = pf.ov_patch + q * p.ov.cells + iy * p.iw + ix;
            cp_async4(slot + sw128_off(r, i >> 2) + 4 * (i & 3), src, in ? 4 : 0);
            if (++ci == p.ic) { ci = 0; if (++kx == p.kw) { kx = 0; ++ky; } }
        }
    }
    if (p.ov.patch) asm volatile("st.shared.u8 [%0], %1;" ::"r"(ov + kTileM * kOvMax * 5 + r), "r"(min(cnt, kOvMax)));
}

// The small-image convolution mode: 5x5 filters over a 14 x 14 x 6 map, stride 1, no
// padding, 16 output channels, 2x2 max pool (LeNet-5's second convolution).  A GEMM
// row is a pooling window rather than an output position: K is the window's 6 x 6 x 6
// receptive field (216) and N = 4 positions x 16 channels = 64, with the weights
// expanded once (zeros where a tap is outside a position's 5 x 5 filter).  With only
// 16 output channels a per-position GEMM would have N = 16, where the MMA issue rate,
// not the tensor core, is the limit; per window the layer takes a third of the MMA
// instructions and of the gathers, and the epilogue pools inside each row.  The
// loader warp stages a tile's whole input maps in shared memory (one bulk copy per
// map) and the producers gather each row's receptive field from there with
// compile-time offsets, 16 bytes per load (a receptive-field row is 36 consecutive,
// 16-byte-aligned values).  A tile holds the windows of MAPS whole maps (125 of its
// 128 rows; the other 3 are computed and dropped), so that three staging buffers fit
// beside the resident weights and the loader runs two tiles ahead of the producers.
// Each tile's maps are bulk copies (with per-input maps, from L2), and so are the
// patch values of the tile's rows, which are consecutive in memory.
struct SmallConv {
    static constexpr int IH = 14, IW = 14, IC = 6, KH = 5, KW = 5, OH = 10, OW = 10, PW = 5, OC = 16;
    static constexpr int KU = KH + 1;                         // receptive field of a window: KU x KU
    static constexpr int P = (OH / 2) * (OW / 2);             // GEMM rows (windows) per map
    static constexpr int K = KU * KU * IC, NKT = (K + kTileK - 1) / kTileK;
    static constexpr int N = 4 * OC;                          // GEMM columns: (window position, channel)
    static constexpr int CELLS = IH * IW;                     // overlay cells of a mutated channel
    static constexpr uint32_t IMG_B = IH * IW * IC * 4;       // bytes of one staged map
    static constexpr int MAXQ = 2;                            // mutated channels per row (overlay)
    static constexpr int MAXG = 256;                          // mutants per batch (overlay table)
    static constexpr int MAPS = kTileM / P;                   // maps per tile
    static constexpr int ROWS = MAPS * P;                     // live rows of a tile
    static constexpr int NBUF = 3;                            // staging buffers
    static constexpr uint32_t BUF_B = MAPS * IMG_B;           // one buffer of staged maps
    static constexpr uint32_t OVST_B = MAPS * MAXQ * CELLS * 4;   // one buffer of staged patch values
    static constexpr uint32_t TAB_B = MAXG * (1 + MAXQ) * 4;      // [g][count, channel ids]
    static constexpr uint32_t BYTES = NBUF * (BUF_B + OVST_B) + TAB_B;
};
static_assert(SmallConv::IMG_B % 16 == 0, "maps are bulk copies of whole 16-byte chunks");
static_assert(SmallConv::NBUF <= kNBufMax, "staging barriers");

// Tiles of the small-image mode over R rows: tile i holds rows MAPS*i .. MAPS*i+MAPS-1.
__host__ __device__ __forceinline__ int64_t small_tiles(int64_t R) { return (R + SmallConv::MAPS - 1) / SmallConv::MAPS; }
static_assert(2 * SmallConv::N * 128 * SmallConv::NKT <= 112 * 1024,
              "the small-image mode keeps its weights resident (its loader warp stages the maps)");
static_assert((SmallConv::CELLS * 4) % 16 == 0, "patch values are bulk copies of whole 16-byte chunks");
static_assert((SmallConv::KU * SmallConv::IC) % 4 == 0 && (SmallConv::IW * SmallConv::IC * 4) % 16 == 0,
              "receptive-field rows are 16-byte aligned runs of whole 4-value chunks");

// K-step KT of a window row: 8 chunks of 4 values at compile-time offsets from the
// window's receptive-field origin `base`, k = (wy, wx, ci).
template <int KT>
__device__ __forceinline__ void small_gather(uint32_t base, float (&v)[kTileK])
{
    using G = SmallConv;
    constexpr int RUN = G::KU * G::IC;   // values per receptive-field row
#pragma unroll
    for (int c = 0; c < kTileK / 4; ++c) {
        const int k = KT * kTileK + 4 * c;
        if (k < G::K) {
            const uint32_t off = (uint32_t)((k / RUN) * G::IW * G::IC + k % RUN) * 4;
            asm volatile("ld.shared.v4.f32 {%0,%1,%2,%3}, [%4];"
                         : "=f"(v[4 * c]), "=f"(v[4 * c + 1]), "=f"(v[4 * c + 2]), "=f"(v[4 * c + 3])
                         : "r"(base + off));
        } else {
            v[4 * c] = v[4 * c + 1] = v[4 * c + 2] = v[4 * c + 3] = 0.f;
        }
    }
}

// The K-steps KT .. NKT-1 of a small-image row, each handed to `push`.
template <int KT>
struct SmallSteps {
    template <class Push>
    __device__ __forceinline__ static void run(uint32_t base, Push &push, bool &ok)
    {
        if constexpr (KT < SmallConv::NKT) {
            float v[kTileK];
            small_gather<KT>(base, v);
            if (ok) ok = push(v);
            SmallSteps<KT + 1>::run(base, push, ok);
        }
    }
};

// MODE 0: dense layer (one GEMM row per batch row); 1: implicit-GEMM convolution; 2:
// the small-image convolution; 3: the staged convolution (see TcParams).  THREE: 3xTF32 (else one TF32 product).  FCP > 0
// (dense, one N slice): the output layer, with up to FCP classes, is computed from
// each row's outputs in the epilogue, followed by the kill epilogue, and the rows
// themselves are not stored.
template <int MODE, bool THREE, int FCP = 0>
__global__ void __launch_bounds__(kThreads, 1) k_tc_gemm(const __grid_constant__ TcParams p)
{
    static_assert(FCP == 0 || (MODE == 0 && FCP % 4 == 0) || (MODE == 3 && FCP == -1),
                  "the output layer is fused into dense layers only; -1: the staged mode's slot GEMM with a residual add");
    constexpr bool DENSE = MODE == 0;
    constexpr int kNT = kMaxNT;                    // barrier slots; p.n_stages are used
    constexpr int kAColsPerStage = THREE ? 64 : 32;
    extern __shared__ __align__(1024) unsigned char smraw[];
    __shared__ __align__(8) uint64_t bar_afull[kNT], bar_aempty[kNT], bar_bfull[kNB], bar_bempty[kNB];
    __shared__ __align__(8) uint64_t bar_accfull[2], bar_accempty[2], bar_drain;
    // small-image and staged-convolution modes, per staging buffer: copies landed,
    // overlay applied, producers done
    __shared__ __align__(8) uint64_t bar_landed[kNBufMax], bar_ready[kNBufMax], bar_released[kNBufMax];
    // dense A tiles by tensor-map copies: slot landed, slot read by the producers
    __shared__ __align__(8) uint64_t bar_alanded[kNA], bar_afree[kNA];
    __shared__ uint32_t tmem_sh;
    // mma_chain: warp w's turn comes with an arrival on bar_turn[w] from the other warp
    __shared__ __align__(8) uint64_t bar_turn[2];
    __shared__ WaitCtl abort_sh;
    __shared__ float bias_sh[kSliceMax];
    __shared__ __align__(16) float epi_stage[4][32 * kEpiStride];   // per epilogue warp: 32 rows x 32 values
    __shared__ float *epi_ptr[4][32];                               // per epilogue warp: each row's output
    volatile WaitCtl *abort_flag = &abort_sh;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t sbase = (smem_u32(smraw) + 1023u) & ~1023u;
    const int n_base = blockIdx.y * p.slice_w;
    const int Nt = min(p.slice_w, p.Np - n_base);           // a multiple of 16
    constexpr int planes = THREE ? 2 : 1;
    const uint32_t b_step = (uint32_t)(planes * Nt * 128);  // one K-step of the weight slice
    const int nK = p.Kp / kTileK;
    const uint32_t b_region = sbase;
    const uint32_t a_region = sbase + (p.b_resident ? (uint32_t)nK * b_step : (uint32_t)p.nb * b_step);
    const uint32_t ov_region = a_region + kNA * kStageA;    // kNA overlay slots (with an overlay)
    const uint32_t cv_region = a_region;                    // MODE 3: the staging ring
    const uint32_t cv_buf_bytes = MODE == 3 ? (uint32_t)p.cv_imgs * p.cv_img_bytes : 0u;
    // FCP > 0: the output layer's weights as [F][FCP] (zeros beyond its C classes)
    const uint32_t fw_region = (ov_region + (p.ov.patch ? kNA * kOvSlotBytes : 0) + 15u) & ~15u;
    const float4 *fw4 = reinterpret_cast<const float4 *>(smraw + (fw_region - smem_u32(smraw)));
    const int64_t M = (int64_t)p.R * p.P;
    // MODE 3 with cv_pair: a unit of two tiles (rows m0 .. m0 + 255) per iteration
    const bool pair = MODE == 3 && p.cv_pair;
    const int64_t TM = pair ? 2 * kTileM : kTileM;
    const int64_t n_tiles = MODE == 2 ? small_tiles(p.R) : (M + TM - 1) / TM;
    const int64_t my_tiles = blockIdx.x < n_tiles ? (n_tiles - 1 - blockIdx.x) / gridDim.x + 1 : 0;
    const int64_t total = my_tiles * nK;
    const float *wslice = p.Wsw + (int64_t)blockIdx.y * p.w_slice_floats;

    if (warp == 0) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(&tmem_sh)),
                     "r"(512));
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
    }
    if constexpr (FCP > 0) {
        for (int i = threadIdx.x; i < p.ff.F * FCP; i += kThreads) {
            const int f = i / FCP, c = i % FCP;
            const float wv = c < p.ff.C ? p.ff.W[(int64_t)c * p.ff.F + f] : 0.f;
            asm volatile("st.shared.f32 [%0], %1;" ::"r"(fw_region + 4 * i), "f"(wv) : "memory");
        }
    }
    for (int n = threadIdx.x; n < kSliceMax; n += kThreads) {
        if (MODE == 2) bias_sh[n] = n < SmallConv::N ? p.b[n % SmallConv::OC] : 0.f;
        else bias_sh[n] = n_base + n < p.N ? p.b[n_base + n] : 0.f;
    }
    // small-image mode: staged maps, staged patch values, the batch's mutated-channel table
    const uint32_t img_region = a_region;
    const uint32_t ovst_region = img_region + SmallConv::NBUF * SmallConv::BUF_B;
    const uint32_t ovtab_region = ovst_region + SmallConv::NBUF * SmallConv::OVST_B;
    if (MODE == 2 && p.ov.patch) {
        const int G = p.R / p.T;
        for (int g = threadIdx.x; g < G; g += kThreads) {
            const int n = p.ov.n_neurons[g];
            const uint32_t tab = ovtab_region + (uint32_t)g * (1 + SmallConv::MAXQ) * 4;
            // count, and in bits 16+ how the finisher writes the channels: 0 from the
            // patch, 1 zeros (NEB), 2 swapped in pairs (NS)
            const int op = p.ov.op ? p.ov.op[g] : -1;
            const uint32_t how = op == MURE_OP_NEB ? 1u : op == MURE_OP_NS ? 2u : 0u;
            asm volatile("st.shared.u32 [%0], %1;" ::"r"(tab), "r"((uint32_t)n | (how << 16)));
            for (int q = 0; q < SmallConv::MAXQ; ++q)
                asm volatile("st.shared.u32 [%0], %1;" ::"r"(tab + 4 + 4 * q), "r"(q < n ? p.ov.ids[p.ov.neuron_off[g] + q] : 0));
        }
    }
    if (threadIdx.x == 32) {
        for (int s = 0; s < kNT; ++s) {
            mbar_init(smem_u32(&bar_afull[s]), 4);
            // each K-step has one issuing warp (two with tile pairs, one per tile)
            mbar_init(smem_u32(&bar_aempty[s]), pair ? 2 : 1);
        }
        for (int s = 0; s < kNB; ++s) {
            mbar_init(smem_u32(&bar_bfull[s]), 1);
            mbar_init(smem_u32(&bar_bempty[s]), pair ? 2 : 1);
        }
        for (int s = 0; s < 2; ++s) {
            mbar_init(smem_u32(&bar_accfull[s]), p.n_mma);
            mbar_init(smem_u32(&bar_accempty[s]), 4);
        }
        mbar_init(smem_u32(&bar_drain), p.n_mma);
        for (int s = 0; s < kNA; ++s) {
            mbar_init(smem_u32(&bar_alanded[s]), 1);
            mbar_init(smem_u32(&bar_afree[s]), 4);
        }
        for (int s = 0; s < kNBufMax; ++s) {
            mbar_init(smem_u32(&bar_landed[s]), 1);
            mbar_init(smem_u32(&bar_ready[s]), 1);
            mbar_init(smem_u32(&bar_released[s]), 4);
        }
        abort_sh.abort = 0;
        mbar_init(smem_u32(&bar_turn[0]), 1);
        mbar_init(smem_u32(&bar_turn[1]), 1);
        abort_sh.limit = p.spin > 0 ? p.spin : kSpin;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    const uint32_t tmem = tmem_sh;

    // small-image mode staging (warps 10 and 11).  A map's mutant g = row / T and input
    // t0 + row % T (rows fit 32 bits).
    using G2 = SmallConv;
    auto tab_of = [&](uint32_t row) { return ovtab_region + (row / (uint32_t)p.T) * (1 + G2::MAXQ) * 4; };
    // tile i's first row and its number of rows
    auto tile_rows = [&](int64_t i, uint32_t &row0) {
        row0 = (uint32_t)((blockIdx.x + i * gridDim.x) * G2::MAPS);
        return (int)min((uint32_t)G2::MAPS, (uint32_t)p.R - row0);
    };
    // bulk copies of tile i into buffer b: a map per row and, in one piece, the rows'
    // patch values, each from its own lane of the calling warp (one thread's bulk copies
    // complete one after another)
    auto issue_tile = [&](int64_t i, int b) {
        uint32_t row0;
        const int nimg = tile_rows(i, row0);
        const uint32_t buf = img_region + (uint32_t)b * G2::BUF_B;
        const uint32_t bar = smem_u32(&bar_landed[b]);
        // the rows' patch values, unless every row of the tile is NEB / NS (or has no
        // mutated channel): the finisher then reads none
        bool need = false;
        if (p.ov.patch)
            for (int im = 0; im < nimg; ++im) {
                uint32_t k;
                asm volatile("ld.shared.u32 %0, [%1];" : "=r"(k) : "r"(tab_of(row0 + im)));
                need |= (k >> 16) == 0 && (k & 0xffffu) != 0;
            }
        const uint32_t pbytes = need ? (uint32_t)(nimg * p.ov.row_stride * 4) : 0u;
        if (lane == 0) mbar_expect_tx(bar, nimg * G2::IMG_B + pbytes);
        __syncwarp();
        // the buffer was last read and written by generic loads and stores
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        if (lane < nimg) {
            const uint32_t row = row0 + lane;
            const int64_t xr = p.x_per_input ? p.t0 + row % (uint32_t)p.T : row;
            bulk_g2s(buf + lane * G2::IMG_B, p.x + xr * p.x_stride, G2::IMG_B, bar);
        }
        if (pbytes && lane == nimg)
            bulk_g2s(ovst_region + (uint32_t)b * G2::OVST_B, p.ov.patch + (int64_t)row0 * p.ov.row_stride, pbytes, bar);
    };

    if (warp < 4) {
        // ------------------------------------------------------------ producers --
        const int r = threadIdx.x;                        // GEMM row in the tile = TMEM lane
        const uint32_t lane_off = (uint32_t)(warp * 32) << 16;
        int t = 0;
        uint32_t wraps = 0;                               // completed rounds of the A-stage ring
        // split one K-step of this row into TF32 halves and hand it to the MMA warps
        auto push = [&](float (&hi)[kTileK]) -> bool {
            float lo[kTileK];
#pragma unroll
            for (int i = 0; i < kTileK; ++i) {
                const float h = tf32_hi(hi[i]);
                if (THREE) lo[i] = hi[i] - h;
                hi[i] = h;
            }
            if (wraps >= 1 && !warp_wait_phase<32>(smem_u32(&bar_aempty[t]), (wraps - 1) & 1, abort_flag)) return false;
            asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
            const uint32_t ta = tmem + lane_off + p.a_col + t * kAColsPerStage;
            tmem_st32(ta, hi);
            if (THREE) tmem_st32(ta + 32, lo);
            asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
            asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
            __syncwarp();
            if (lane == 0) mbar_arrive(smem_u32(&bar_afull[t]));
            if (++t == p.n_stages) { t = 0; ++wraps; }
            return true;
        };
        // tile pairs: the K-step of row r (part 0), then of row 128 + r (part 1), into one
        // stage of 2 kAColsPerStage columns; the stage goes to the MMA warps after part 1
        auto push_part = [&](float (&hi)[kTileK], int part) -> bool {
            float lo[kTileK];
#pragma unroll
            for (int i = 0; i < kTileK; ++i) {
                const float h = tf32_hi(hi[i]);
                if (THREE) lo[i] = hi[i] - h;
                hi[i] = h;
            }
            if (part == 0) {
                if (wraps >= 1 && !warp_wait_phase<32>(smem_u32(&bar_aempty[t]), (wraps - 1) & 1, abort_flag))
                    return false;
                asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
            }
            const uint32_t ta = tmem + lane_off + p.a_col + (uint32_t)(t * 2 + part) * kAColsPerStage;
            tmem_st32(ta, hi);
            if (THREE) tmem_st32(ta + 32, lo);
            asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");   // the registers are reused
            if (part == 1) {
                asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
                __syncwarp();
                if (lane == 0) mbar_arrive(smem_u32(&bar_afull[t]));
                if (++t == p.n_stages) { t = 0; ++wraps; }
            }
            return true;
        };
        if constexpr (MODE == 2) {
            // warps 10 and 11 stage each tile's maps (mutated channels written in) in
            // buffer i mod NBUF; the producers only gather from them
            using G = SmallConv;
            // this thread's GEMM row: map r / P of the tile and its pooling window (the
            // padding rows gather from map 0, which is always staged)
            const int im = r < G::ROWS ? r / G::P : 0, w = r < G::ROWS ? r % G::P : 0;
            const uint32_t off = (uint32_t)im * G::IMG_B + (uint32_t)((2 * (w / G::PW) * G::IW + 2 * (w % G::PW)) * G::IC) * 4;
            bool ok = true;
            int b = 0;
            uint32_t uses = 0;                            // completed rounds of the buffer ring
            for (int64_t i = 0; ok && i < my_tiles; ++i) {
                if (!warp_wait_phase<32>(smem_u32(&bar_ready[b]), uses & 1, abort_flag)) break;
                SmallSteps<0>::run(img_region + (uint32_t)b * G::BUF_B + off, push, ok);
                // every gather of the tile has been consumed by push: the buffer is free
                __syncwarp();
                if (lane == 0) mbar_arrive(smem_u32(&bar_released[b]));
                if (++b == G::NBUF) { b = 0; ++uses; }
            }
        } else if constexpr (MODE == 3) {
            // the tile's staged input rows, one chunk of channels at a time (zero border
            // included, overlay written in by warp 10), one 128-byte line per pixel:
            // this thread gathers its GEMM row's values of each filter tap from the
            // chunk, 16 bytes per load, in the 128-byte swizzle of the copies (byte b of
            // the buffer sits at b ^ ((b >> 3) & 0x70)); a K-step is one tap of 32
            // channels or two taps of 16
            const bool fin = p.ov.patch != nullptr;
            bool ok = true;
            int64_t job = 0;
            for (int64_t i = 0; ok && i < my_tiles; ++i) {
                const int64_t m0 = (blockIdx.x + i * gridDim.x) * TM;
                const int64_t row0 = m0 / p.P;
                const int oy0 = p.cv_imgs > 1 ? 0 : (int)((m0 - row0 * p.P) / TM) * p.cv_rows;
                // rows past the end gather from the unit's first staged row (dropped later)
                const RowInfo ri = row_info<false, false>(p, m0 + r);
                const uint32_t im = ri.ok ? (uint32_t)(ri.row - row0) : 0u;
                const int line0 = ri.ok ? (ri.oy - oy0) * p.cv_hw + ri.ox : 0;
                // tile pairs: this thread's row of the second tile too
                uint32_t im1 = 0;
                int line1 = 0;
                if (pair) {
                    const RowInfo r1 = row_info<false, false>(p, m0 + kTileM + r);
                    im1 = r1.ok ? (uint32_t)(r1.row - row0) : 0u;
                    line1 = r1.ok ? (r1.oy - oy0) * p.cv_hw + r1.ox : 0;
                }
                for (int c = 0; c < p.cv_nchunk; ++c, ++job) {
                    const int b = (int)(job % p.cv_nbuf);
                    const uint32_t use = (uint32_t)(job / p.cv_nbuf);
                    if (!warp_wait_phase<32>(smem_u32(fin ? &bar_ready[b] : &bar_landed[b]), use & 1, abort_flag)) {
                        ok = false;
                        break;
                    }
                    const uint32_t buf = cv_region + (uint32_t)b * cv_buf_bytes;
                    const uint32_t base = buf + im * p.cv_img_bytes, base1 = buf + im1 * p.cv_img_bytes;
                    const int ntap = p.cv_ntap;
                    // the current tap and its line relative to a row's line0 (ky * cv_hw + kx),
                    // over the filter (or a window's 4x4 field)
                    int tap = 0, kx = 0, off = 0;
                    auto next_tap = [&]() {
                        ++tap;
                        if (++kx == p.cv_fw) {
                            kx = 0;
                            off += p.cv_hw - p.cv_fw + 1;
                        } else {
                            ++off;
                        }
                    };
                    // chunk cc of line l sits at l * 128 + (cc ^ (l mod 8)) * 16
                    auto gather = [&](float *v, int nc, uint32_t bse, int line) {
                        const uint32_t l = (uint32_t)line;
                        const uint32_t a = bse + l * 128u, sw = l & 7u;
#pragma unroll
                        for (int cc = 0; cc < 8; ++cc) {
                            if (cc >= nc) break;
                            asm volatile("ld.shared.v4.f32 {%0,%1,%2,%3}, [%4];"
                                         : "=f"(v[4 * cc]), "=f"(v[4 * cc + 1]), "=f"(v[4 * cc + 2]), "=f"(v[4 * cc + 3])
                                         : "r"(a + (((uint32_t)cc ^ sw) << 4)));
                        }
                    };
                    for (int ks = 0; ks < p.cv_taps; ++ks) {
                        // this K-step's taps: one of 32 channels, or two of 16 (the first
                        // half of their lines; past the last tap the second half is zero)
                        const int offa = off;
                        next_tap();
                        int offb = -1;
                        if (p.cv_cw != kTileK) {
                            if (tap < ntap) offb = off;
                            next_tap();
                        }
                        auto gather_k = [&](float (&v)[kTileK], uint32_t bse, int l0) {
                            if (p.cv_cw == kTileK) {
                                gather(v, 8, bse, l0 + offa);
                            } else {
                                gather(v, 4, bse, l0 + offa);
                                if (offb >= 0) {
                                    gather(v + 16, 4, bse, l0 + offb);
                                } else {
#pragma unroll
                                    for (int e = 16; e < kTileK; ++e) v[e] = 0.f;
                                }
                            }
                        };
                        float v[kTileK];
                        gather_k(v, base, line0);
                        if (pair) {
                            if (!push_part(v, 0)) { ok = false; break; }
                            gather_k(v, base1, line1);
                            if (!push_part(v, 1)) { ok = false; break; }
                        } else if (!push(v)) {
                            ok = false;
                            break;
                        }
                    }
                    // every gather of the chunk has been consumed by push: the buffer is free
                    __syncwarp();
                    if (lane == 0) mbar_arrive(smem_u32(&bar_released[b]));
                    if (!ok) break;
                }
            }
        } else if (DENSE && p.a_tma) {
            // A tiles land by tensor-map copies (warp 10); each thread reads its row
            bool ok = true;
            int slot_i = 0;
            uint32_t slot_wraps = 0;
            for (int64_t j = 0; ok && j < total; ++j) {
                if (!warp_wait_phase<32>(smem_u32(&bar_alanded[slot_i]), slot_wraps & 1, abort_flag)) break;
                const uint32_t slot = a_region + (uint32_t)slot_i * kStageA;
                float v[kTileK];
#pragma unroll
                for (int c = 0; c < kTileK / 4; ++c) {
                    asm volatile("ld.shared.v4.f32 {%0,%1,%2,%3}, [%4];"
                                 : "=f"(v[4 * c]), "=f"(v[4 * c + 1]), "=f"(v[4 * c + 2]), "=f"(v[4 * c + 3])
                                 : "r"(slot + sw128_off(r, c)));
                }
                __syncwarp();
                if (lane == 0) mbar_arrive(smem_u32(&bar_afree[slot_i]));
                if (++slot_i == kNA) { slot_i = 0; ++slot_wraps; }
                ok = push(v);
            }
        } else {
            // issue cursor (tile i, K-tile kt, ring slot) runs kNA - 1 steps ahead
            RowInfo pf{};
            LoadRows lr{};
            int64_t iss_i = 0, issued = 0;
            int iss_kt = 0, iss_slot = 0;
            auto issue_next = [&]() {
                if (iss_kt == 0) {
                    pf = row_info<DENSE>(p, (blockIdx.x + iss_i * gridDim.x) * kTileM + r);
                    if (DENSE || (p.ic & 3) == 0) load_rows<DENSE>(pf, lr);
                    if (!DENSE && (p.ic & 3) == 0) chunk_cursor(p, lr);
                }
                produce_issue<DENSE>(p, pf, lr, r, a_region + (uint32_t)iss_slot * kStageA,
                                     ov_region + (uint32_t)iss_slot * kOvSlotBytes, iss_kt * kTileK);
                if (++iss_kt == nK) { iss_kt = 0; ++iss_i; }
                if (++iss_slot == kNA) iss_slot = 0;
                ++issued;
            };
            for (int s0 = 0; s0 < kNA - 1; ++s0) {
                if (issued < total) issue_next();
                cp_async_commit();
            }
            int slot_i = 0;
            for (int64_t j = 0; j < total; ++j) {
                if (issued < total) issue_next();
                cp_async_commit();
                cp_async_wait<kNA - 1>();                 // this thread's copies of step j
                __syncwarp();                             // ... and those of the warp's other lanes
                const uint32_t slot = a_region + (uint32_t)slot_i * kStageA;
                if (p.ov.patch) {
                    // the row's overlay entries of this K-step, written over the landed copy
                    const uint32_t ov = ov_region + (uint32_t)slot_i * kOvSlotBytes;
                    uint32_t n;
                    asm volatile("ld.shared.u8 %0, [%1];" : "=r"(n) : "r"(ov + kTileM * kOvMax * 5 + r));
                    for (uint32_t e = 0; e < n; ++e) {
                        uint32_t pos, val;
                        asm volatile("ld.shared.u8 %0, [%1];" : "=r"(pos) : "r"(ov + kTileM * kOvMax * 4 + e * kTileM + r));
                        asm volatile("ld.shared.u32 %0, [%1];" : "=r"(val) : "r"(ov + (e * kTileM + r) * 4));
                        asm volatile("st.shared.u32 [%0], %1;" ::"r"(slot + sw128_off(r, pos >> 2) + 4 * (pos & 3)),
                                     "r"(val)
                                     : "memory");
                    }
                }
                if (++slot_i == kNA) slot_i = 0;
                float v[kTileK];
#pragma unroll
                for (int c = 0; c < kTileK / 4; ++c) {
                    asm volatile("ld.shared.v4.f32 {%0,%1,%2,%3}, [%4];"
                                 : "=f"(v[4 * c]), "=f"(v[4 * c + 1]), "=f"(v[4 * c + 2]), "=f"(v[4 * c + 3])
                                 : "r"(slot + sw128_off(r, c)));
                }
                if (!push(v)) break;
            }
            cp_async_wait<0>();
        }
    } else if (warp < 8) {
        // ------------------------------------------------------------- epilogue --
        const int qd = warp & 3;
        const uint32_t lane_off = (uint32_t)(qd * 32) << 16;
        for (int64_t i = 0; i < my_tiles; ++i) {
            const int a = p.n_acc == 2 ? (int)(i & 1) : 0;
            const int64_t use = p.n_acc == 2 ? (i >> 1) : i;
            if (!warp_wait_phase<64>(smem_u32(&bar_accfull[a]), (uint32_t)(use & 1), abort_flag)) break;
            asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
            const int64_t tile = blockIdx.x + i * gridDim.x;
            if constexpr (MODE == 2) {
                // a pooling window: columns n = s * OC + c for its position s = 2 dy + dx
                using G = SmallConv;
                const int rr = qd * 32 + lane;
                const int64_t row = tile * G::MAPS + rr / G::P;
                const bool ok = rr < G::ROWS && row < p.R;
                const int w = rr % G::P;
                const int py = w / G::PW, px = w % G::PW;
                const uint32_t acc = tmem + lane_off + (uint32_t)(a * p.n_part * p.acc_cols);
                float v[G::N];
#pragma unroll
                for (int n0 = 0; n0 < G::N; n0 += 16) {
                    tmem_ld16(acc + n0, v + n0);
                    for (int w2 = 1; w2 < p.n_part; ++w2) {
                        float u[16];
                        tmem_ld16(acc + (uint32_t)(w2 * p.acc_cols) + n0, u);
#pragma unroll
                        for (int e = 0; e < 16; ++e) v[n0 + e] += u[e];
                    }
                    if (p.merge_lo) {
                        float u[16];
                        tmem_ld16(acc + (uint32_t)G::N + n0, u);
#pragma unroll
                        for (int e = 0; e < 16; ++e) v[n0 + e] += u[e];
                    }
                }
                float o[G::OC];
#pragma unroll
                for (int c = 0; c < G::OC; ++c) {
                    float v4[4];
#pragma unroll
                    for (int s4 = 0; s4 < 4; ++s4) {
                        const float zz = v[s4 * G::OC + c] + bias_sh[c];
                        if (p.z && ok)
                            p.z[row * p.z_stride + (int64_t)c * (G::OH * G::OW) + (2 * py + (s4 >> 1)) * G::OW + 2 * px + (s4 & 1)] = zz;
                        v4[s4] = act_apply(p.act1, zz);
                    }
                    o[c] = max4_first(v4[0], v4[1], v4[2], v4[3]);
                }
                if (ok) {
                    float *yo = p.y + row * p.y_stride + (int64_t)w * G::OC;
#pragma unroll
                    for (int c = 0; c < G::OC; c += 4)
                        *reinterpret_cast<float4 *>(yo + c) = make_float4(o[c], o[c + 1], o[c + 2], o[c + 3]);
                }
                asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
                __syncwarp();
                if (lane == 0) mbar_arrive(smem_u32(&bar_accempty[a]));
                continue;
            }
            if (MODE == 3 && p.cv_win) {
                // a 2x2 output window per row: columns s * N + c for position s = 2 dy + dx
                const RowInfo ri = row_info<false, false>(p, tile * kTileM + qd * 32 + lane);
                const uint32_t acc = tmem + lane_off + (uint32_t)(a * p.n_part * p.acc_cols);
                const float *srow = nullptr;
                if (p.has_add && ri.ok)
                    srow = p.skip + (p.skip_per_input ? p.t0 + logical_row(p.lrow, ri.row) % p.T : ri.row) * p.skip_stride;
#pragma unroll 1
                for (int sp = 0; sp < 4; ++sp) {
                    const int oy = ri.oy + (sp >> 1), ox = ri.ox + (sp & 1);
                    float v[16];   // N == 16 outputs per position
                    tmem_ld16(acc + (uint32_t)(sp * 16), v);
                    for (int w2 = 1; w2 < p.n_part; ++w2) {
                        float u[16];
                        tmem_ld16(acc + (uint32_t)(w2 * p.acc_cols + sp * 16), u);
#pragma unroll
                        for (int e = 0; e < 16; ++e) v[e] += u[e];
                    }
                    if (p.merge_lo) {
                        float u[16];
                        tmem_ld16(acc + (uint32_t)(Nt + sp * 16), u);
#pragma unroll
                        for (int e = 0; e < 16; ++e) v[e] += u[e];
                    }
#pragma unroll
                    for (int e = 0; e < 16; ++e) v[e] += bias_sh[e];
                    if (p.z && ri.ok)
                        for (int e = 0; e < 16; ++e)
                            p.z[ri.row * p.z_stride + (int64_t)e * (p.oh * p.ow) + oy * p.ow + ox] = v[e];
                    if (p.act1 != MURE_ACT_NONE) {
#pragma unroll
                        for (int e = 0; e < 16; ++e) v[e] = act_apply(p.act1, v[e]);
                    }
                    if (p.has_add && ri.ok) {
                        const float *skp = srow + ((int64_t)oy * p.sk_stride * p.sk_w + ox * p.sk_stride) * p.sk_c;
#pragma unroll
                        for (int e = 0; e < 16; ++e) v[e] = act_apply(p.act2, v[e] + (e < p.sk_c ? skp[e] : 0.f));
                    }
                    if (ri.ok) {
                        float *yo = p.y + ri.row * p.y_stride + ((int64_t)oy * p.ow + ox) * 16;
#pragma unroll
                        for (int c = 0; c < 4; ++c)
                            *reinterpret_cast<float4 *>(yo + 4 * c) = make_float4(v[4 * c], v[4 * c + 1], v[4 * c + 2], v[4 * c + 3]);
                    }
                }
                asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
                __syncwarp();
                if (lane == 0) mbar_arrive(smem_u32(&bar_accempty[a]));
                continue;
            }
            // tile pairs: the unit's two tiles one after the other, each from its own
            // accumulator; the accumulator set is released after the second
            const int nsub = pair ? 2 : 1;
            for (int sub = 0; sub < nsub; ++sub) {
            const uint32_t abase = pair ? (uint32_t)((a * 2 + sub) * p.acc_cols) : (uint32_t)(a * p.n_part * p.acc_cols);
            const RowInfo ri = row_info<DENSE, false>(p, (tile * nsub + sub) * kTileM + qd * 32 + lane);
            const float *srow = nullptr;
            if (p.has_add && ri.ok)
                srow = p.skip + (p.skip_per_input ? p.t0 + logical_row(p.lrow, ri.row) % p.T : ri.row) * p.skip_stride;
            float *yrow = ri.ok ? p.y + ri.row * p.y_stride : nullptr;
            // unpooled outputs go through shared memory: one store instruction then
            // covers 4 rows x 128 bytes instead of 32 rows x 16 bytes
            float *stage = epi_stage[qd];
            const bool vec = DENSE || (p.N & 3) == 0;
            if (!(!DENSE && p.pool))
                epi_ptr[qd][lane] = ri.ok ? yrow + (DENSE ? 0 : ((int64_t)ri.oy * p.ow + ri.ox) * p.N) : nullptr;
            float facc[FCP > 0 ? FCP : 1];
#pragma unroll
            for (int c = 0; c < (FCP > 0 ? FCP : 1); ++c) facc[c] = 0.f;
            for (int n0 = 0; n0 < Nt; n0 += 32) {
                const int nc = min(32, Nt - n0);
                float v[32];
#pragma unroll
                for (int h = 0; h < 32; h += 16) {
                    if (h >= nc) break;
                    float *vh = v + h;
                    // the accumulator: the n_part partials added in a fixed order
                    const uint32_t acc = tmem + lane_off + abase + n0 + h;
                    tmem_ld16(acc, vh);
                    for (int w = 1; w < p.n_part; ++w) {
                        float u[16];
                        tmem_ld16(acc + (uint32_t)(w * p.acc_cols), u);
#pragma unroll
                        for (int e = 0; e < 16; ++e) vh[e] += u[e];
                    }
                    if (MODE == 3 && p.merge_lo) {
                        float u[16];
                        tmem_ld16(acc + (uint32_t)Nt, u);
#pragma unroll
                        for (int e = 0; e < 16; ++e) vh[e] += u[e];
                    }
#pragma unroll
                    for (int e = 0; e < 16; ++e) vh[e] += bias_sh[n0 + h + e];   // padding channels hold 0
                    if (p.z && ri.ok) {
                        for (int e = 0; e < 16 && n_base + n0 + h + e < p.N; ++e) {
                            const int n = n_base + n0 + h + e;
                            if (DENSE) p.z[ri.row * p.z_stride + n] = vh[e];
                            else p.z[ri.row * p.z_stride + (int64_t)n * (p.oh * p.ow) + ri.oy * p.ow + ri.ox] = vh[e];
                        }
                    }
                    if (!DENSE && p.slot.out && ri.ok) {
                        // the delta GEMM's sum on top of the slot channel's pre-activation
                        const float *zr = p.slot.z + (p.slot.z_per_input ? p.t0 + ri.row : ri.row) * p.slot.z_stride +
                                          ri.oy * p.ow + ri.ox;
#pragma unroll
                        for (int e = 0; e < 16; ++e) {
                            const int n = n_base + n0 + h + e;
                            if (n < p.slot.n) vh[e] = __ldg(zr + (int64_t)__ldg(p.slot.j + n) * (p.oh * p.ow)) + vh[e];
                        }
                    }
                    if (p.act1 != MURE_ACT_NONE) {
#pragma unroll
                        for (int e = 0; e < 16; ++e) vh[e] = act_apply(p.act1, vh[e]);
                    }
                    if constexpr (FCP > 0) {
                        // the output layer: fp32 FMAs over the inputs f in ascending
                        // order, as the output-layer kernel does
#pragma unroll
                        for (int e = 0; e < 16; ++e) {
                            const int f = n0 + h + e;
                            if (f < p.N) {
#pragma unroll
                                for (int c4 = 0; c4 < FCP; c4 += 4) {
                                    const float4 w4 = fw4[(f * FCP + c4) >> 2];
                                    facc[c4] = fmaf(vh[e], w4.x, facc[c4]);
                                    facc[c4 + 1] = fmaf(vh[e], w4.y, facc[c4 + 1]);
                                    facc[c4 + 2] = fmaf(vh[e], w4.z, facc[c4 + 2]);
                                    facc[c4 + 3] = fmaf(vh[e], w4.w, facc[c4 + 3]);
                                }
                            }
                        }
                    }
                    if (!DENSE && p.has_add && ri.ok) {
                        const float *sp = srow + ((int64_t)ri.oy * p.sk_stride * p.sk_w + ri.ox * p.sk_stride) * p.sk_c;
#pragma unroll
                        for (int e = 0; e < 16; ++e) {
                            const int n = n_base + n0 + h + e;
                            // the delta GEMM of a residual-add layer (FCP < 0): column n is a
                            // slot, its skip value that of the slot's channel
                            const int ch = FCP < 0 ? (n < p.slot.n ? __ldg(p.slot.j + n) : p.sk_c) : n;
                            const float sv = ch < p.sk_c ? sp[ch] : 0.f;
                            vh[e] = act_apply(p.act2, vh[e] + sv);
                        }
                    }
                    if (!DENSE && !p.pool && p.slot.out && ri.ok) {
                        const int cell = ri.oy * p.ow + ri.ox;
#pragma unroll
                        for (int e = 0; e < 16; ++e) {
                            const int n = n_base + n0 + h + e;
                            if (n < p.slot.n)
                                p.slot.out[((int64_t)__ldg(p.slot.g + n) * p.slot.T + ri.row) * p.slot.stride +
                                           (int64_t)__ldg(p.slot.q + n) * p.slot.cells + cell] = vh[e];
                        }
                    }
                    if (MODE == 3 && p.pool && !p.slot.out && n_base + n0 + h + 15 < p.N && (p.N & 3) == 0) {
                        // lanes 4w .. 4w+3 hold the four positions (a, b, c, d) of one
                        // pooling window; two exchanges leave lane q with all four values
                        // of channels (q & 1) * 8 + (q >> 1) * 4 + 0..3, pooled in the
                        // order a, b, c, d, and stored as one 16-byte piece
                        const int q = lane & 3;
                        float P[8], Q[8];   // positions a / c (P) and b / d (Q) of 8 channels
#pragma unroll
                        for (int i = 0; i < 8; ++i) {
                            const float send = (q & 1) ? vh[i] : vh[8 + i];
                            const float recv = __shfl_xor_sync(0xffffffffu, send, 1);
                            const float own = (q & 1) ? vh[8 + i] : vh[i];
                            P[i] = (q & 1) ? recv : own;
                            Q[i] = (q & 1) ? own : recv;
                        }
                        float o4[4];
#pragma unroll
                        for (int i = 0; i < 4; ++i) {
                            const float sp = (q & 2) ? P[i] : P[4 + i], sq = (q & 2) ? Q[i] : Q[4 + i];
                            const float rp = __shfl_xor_sync(0xffffffffu, sp, 2), rq = __shfl_xor_sync(0xffffffffu, sq, 2);
                            o4[i] = (q & 2) ? max4_first(rp, rq, P[4 + i], Q[4 + i]) : max4_first(P[i], Q[i], rp, rq);
                        }
                        if (ri.ok) {
                            float *yo = yrow + ((int64_t)ri.py * p.pw + ri.px) * p.N + n_base + n0 + h + (q & 1) * 8 +
                                        (q >> 1) * 4;
                            *reinterpret_cast<float4 *>(yo) = make_float4(o4[0], o4[1], o4[2], o4[3]);
                        }
                    } else if (!DENSE && p.pool) {
                        // lanes 4w .. 4w+3 hold the four positions of one pooling window
#pragma unroll
                        for (int e = 0; e < 16; ++e) {
                            const float w1 = __shfl_down_sync(0xffffffffu, vh[e], 1);
                            const float w2 = __shfl_down_sync(0xffffffffu, vh[e], 2);
                            const float w3 = __shfl_down_sync(0xffffffffu, vh[e], 3);
                            if ((lane & 3) == 0) vh[e] = max4_first(vh[e], w1, w2, w3);
                        }
                        if (p.slot.out) {
                            if (ri.ok && (lane & 3) == 0) {
                                const int cell = ri.py * p.pw + ri.px;
#pragma unroll
                                for (int e = 0; e < 16; ++e) {
                                    const int n = n_base + n0 + h + e;
                                    if (n < p.slot.n)
                                        p.slot.out[((int64_t)__ldg(p.slot.g + n) * p.slot.T + ri.row) * p.slot.stride +
                                                   (int64_t)__ldg(p.slot.q + n) * p.slot.cells + cell] = vh[e];
                                }
                            }
                        } else if (ri.ok && (lane & 3) == 0) {
                            float *yo = yrow + ((int64_t)ri.py * p.pw + ri.px) * p.N + n_base + n0 + h;
                            if (n_base + n0 + h + 15 < p.N && (p.N & 3) == 0) {
#pragma unroll
                                for (int c = 0; c < 4; ++c)
                                    *reinterpret_cast<float4 *>(yo + 4 * c) =
                                        make_float4(vh[4 * c], vh[4 * c + 1], vh[4 * c + 2], vh[4 * c + 3]);
                            } else {
#pragma unroll
                                for (int e = 0; e < 16; ++e)
                                    if (n_base + n0 + h + e < p.N) yo[e] = vh[e];
                            }
                        }
                    }
                }
                if ((!DENSE && p.pool) || FCP > 0 || p.slot.out) continue;
#pragma unroll
                for (int c = 0; c < 8; ++c)
                    *reinterpret_cast<float4 *>(stage + lane * kEpiStride + 4 * c) =
                        make_float4(v[4 * c], v[4 * c + 1], v[4 * c + 2], v[4 * c + 3]);
                __syncwarp();
#pragma unroll
                for (int k = 0; k < 8; ++k) {
                    const int rr = 4 * k + (lane >> 3), c4 = lane & 7;
                    float *dst = epi_ptr[qd][rr];
                    const int n = n_base + n0 + 4 * c4;
                    if (dst && 4 * c4 < nc && n < p.N) {
                        const float4 val = *reinterpret_cast<const float4 *>(stage + rr * kEpiStride + 4 * c4);
                        if (vec && n + 3 < p.N) {
                            *reinterpret_cast<float4 *>(dst + n) = val;
                        } else {
                            dst[n] = val.x;
                            if (n + 1 < p.N) dst[n + 1] = val.y;
                            if (n + 2 < p.N) dst[n + 2] = val.z;
                            if (n + 3 < p.N) dst[n + 3] = val.w;
                        }
                    }
                }
                __syncwarp();
            }
            if (sub == nsub - 1) {
                asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
                __syncwarp();
                if (lane == 0) mbar_arrive(smem_u32(&bar_accempty[a]));
            }
            if constexpr (FCP > 0) {
                // logits = act(acc + b), then argmax / kill as the output-layer kernel
                float lv[FCP];
#pragma unroll
                for (int c = 0; c < FCP; ++c) lv[c] = c < p.ff.C ? act_apply(p.ff.act, facc[c] + __ldg(p.ff.b + c)) : 0.f;
                epilogue_reg<FCP>(p.ff.fa, p.t0, p.T, ri.row, ri.ok, lv, p.ff.C);
            }
            }
        }
    } else if (DENSE && warp == 10 && p.a_tma) {
        // ------------------------------------------------------ A tiles by TMA --
        if (lane == 0) {
            const uint64_t tmap = reinterpret_cast<uint64_t>(&p.tmap_a);
            int slot_i = 0, kt = 0;
            uint32_t slot_wraps = 0;
            int64_t i = 0, j = 0;
            for (; j < total; ++j) {
                if (slot_wraps >= 1 &&
                    !wait_phase<32>(smem_u32(&bar_afree[slot_i]), (slot_wraps - 1) & 1, abort_flag))
                    break;
                // the producers' reads of the slot (generic proxy) before this copy's writes
                asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
                const int64_t m0 = (blockIdx.x + i * gridDim.x) * kTileM;
                const int row = (int)m0;
                const uint32_t bar = smem_u32(&bar_alanded[slot_i]);
                mbar_expect_tx(bar, (uint32_t)kStageA);
                asm volatile(
                    "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];"
                    ::"r"(a_region + (uint32_t)slot_i * kStageA), "l"(tmap), "r"(kt * kTileK), "r"(row), "r"(bar)
                    : "memory");
                if (++slot_i == kNA) { slot_i = 0; ++slot_wraps; }
                if (++kt == nK) { kt = 0; ++i; }
            }
            // copies still in flight land before the shared memory is released
            for (int64_t jj = j > kNA ? j - kNA : 0; jj < j; ++jj)
                wait_phase_drain(smem_u32(&bar_alanded[jj % kNA]), (uint32_t)((jj / kNA) & 1));
        }
    } else if (MODE == 2 && warp == 10) {
        // ------------------------------------------------ map staging: finish --
        // Tile i once landed: each row's mutated channels are written over its map, and
        // the buffer goes to the producers.
        using G = SmallConv;
        int b = 0;
        uint32_t uses = 0;
        for (int64_t i = 0; i < my_tiles; ++i) {
            if (!warp_wait_phase<32>(smem_u32(&bar_landed[b]), uses & 1, abort_flag)) break;
            if (p.ov.patch) {
                uint32_t row0;
                const int nimg = tile_rows(i, row0);
                const uint32_t buf = img_region + (uint32_t)b * G::BUF_B;
                const uint32_t ovb = ovst_region + (uint32_t)b * G::OVST_B;
                constexpr int U = (G::CELLS + 31) / 32;
                for (int im = 0; im < nimg; ++im) {
                    const uint32_t tab = tab_of(row0 + im);
                    uint32_t k;
                    asm volatile("ld.shared.u32 %0, [%1];" : "=r"(k) : "r"(tab));
                    const uint32_t how = k >> 16;
                    k &= 0xffffu;
                    const uint32_t map = buf + im * G::IMG_B;
                    if (how == 1) {
                        // NEB: the channels' post-activation values are +0
                        for (uint32_t q = 0; q < k; ++q) {
                            uint32_t jn;
                            asm volatile("ld.shared.u32 %0, [%1];" : "=r"(jn) : "r"(tab + 4 + q * 4));
#pragma unroll
                            for (int u = 0; u < U; ++u)
                                if (lane + 32 * u < G::CELLS)
                                    asm volatile("st.shared.u32 [%0], %1;" ::"r"(map + ((lane + 32 * u) * G::IC + jn) * 4), "r"(0u)
                                                 : "memory");
                        }
                        continue;
                    }
                    if (how == 2) {
                        // NS: channels q and q + 1 trade places (each lane its own cells)
                        for (uint32_t q = 0; q + 1 < k; q += 2) {
                            uint32_t ja, jb;
                            asm volatile("ld.shared.u32 %0, [%1];" : "=r"(ja) : "r"(tab + 4 + q * 4));
                            asm volatile("ld.shared.u32 %0, [%1];" : "=r"(jb) : "r"(tab + 8 + q * 4));
#pragma unroll
                            for (int u = 0; u < U; ++u)
                                if (lane + 32 * u < G::CELLS) {
                                    const uint32_t cell = map + (lane + 32 * u) * G::IC * 4;
                                    uint32_t va, vb;
                                    asm volatile("ld.shared.u32 %0, [%1];" : "=r"(va) : "r"(cell + ja * 4));
                                    asm volatile("ld.shared.u32 %0, [%1];" : "=r"(vb) : "r"(cell + jb * 4));
                                    asm volatile("st.shared.u32 [%0], %1;" ::"r"(cell + ja * 4), "r"(vb) : "memory");
                                    asm volatile("st.shared.u32 [%0], %1;" ::"r"(cell + jb * 4), "r"(va) : "memory");
                                }
                        }
                        continue;
                    }
                    for (uint32_t q = 0; q < k; ++q) {
                        uint32_t jn, val[U];
                        asm volatile("ld.shared.u32 %0, [%1];" : "=r"(jn) : "r"(tab + 4 + q * 4));
                        const uint32_t src = ovb + (uint32_t)(im * p.ov.row_stride + q * G::CELLS) * 4;
                        const uint32_t dst = buf + im * G::IMG_B + jn * 4;
#pragma unroll
                        for (int u = 0; u < U; ++u)
                            if (lane + 32 * u < G::CELLS)
                                asm volatile("ld.shared.u32 %0, [%1];" : "=r"(val[u]) : "r"(src + (lane + 32 * u) * 4));
#pragma unroll
                        for (int u = 0; u < U; ++u)
                            if (lane + 32 * u < G::CELLS)
                                asm volatile("st.shared.u32 [%0], %1;" ::"r"(dst + (lane + 32 * u) * (G::IC * 4)), "r"(val[u])
                                             : "memory");
                    }
                }
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(smem_u32(&bar_ready[b]));
            if (++b == G::NBUF) { b = 0; ++uses; }
        }
    } else if (MODE == 3 && warp == 10) {
        // ------------------------------------- staged convolution: input staging --
        // Lane 0 copies each job's input rows (tile i, chunk c: 32 channels of the rows
        // with their zero border) into buffer job mod cv_nbuf as soon as the producers
        // have released it.  With an overlay (the first suffix stage) the warp then
        // writes the mutated channels of its batch rows over each landed chunk, at every
        // staged pixel inside the image, before the producers read it.  (A thread's bulk
        // copies complete one after another, so the weight ring has a thread of its own.)
        const bool fin = p.ov.patch != nullptr;
        const int64_t n_jobs = my_tiles * p.cv_nchunk;
        const uint32_t box_bytes = (uint32_t)p.cv_hw * p.cv_hh * 128u;
        const uint64_t tmap = reinterpret_cast<uint64_t>(&p.tmap_x);
        // tile i's first batch row, its first staged output row and its rows
        auto tile_geo = [&](int64_t i, int64_t &row0, int &oy0) {
            const int64_t m0 = (blockIdx.x + i * gridDim.x) * TM;
            row0 = m0 / p.P;
            oy0 = p.cv_imgs > 1 ? 0 : (int)((m0 - row0 * p.P) / TM) * p.cv_rows;
            return (int)min((int64_t)p.cv_imgs, (int64_t)p.R - row0);
        };
        auto issue = [&](int64_t jc) {
            const int b = (int)(jc % p.cv_nbuf);
            const int64_t i = jc / p.cv_nchunk;
            const int c = (int)(jc - i * p.cv_nchunk);
            int64_t row0;
            int oy0;
            const int nimg = tile_geo(i, row0, oy0);
            const uint32_t bar = smem_u32(&bar_landed[b]);
            // the buffer was last read (and written) through the generic proxy
            asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
            mbar_expect_tx(bar, (uint32_t)max(nimg, 0) * box_bytes);
            for (int im = 0; im < nimg; ++im) {
                const int64_t row = row0 + im;
                const int src = (int)(p.x_per_input ? p.t0 + logical_row(p.lrow, row) % p.T : row);
                asm volatile(
                    "cp.async.bulk.tensor.4d.shared::cluster.global.mbarrier::complete_tx::bytes "
                    "[%0], [%1, {%2, %3, %4, %5}], [%6];" ::"r"(cv_region + (uint32_t)b * cv_buf_bytes +
                                                                  (uint32_t)im * p.cv_img_bytes),
                    "l"(tmap), "r"(c * p.cv_cw), "r"(-p.pad), "r"(oy0 - p.pad), "r"(src), "r"(bar)
                    : "memory");
            }
        };
        int64_t issued = 0;
        bool ok = true;
        // the job's buffer once the producers released its previous use (blocking or not)
        auto try_issue = [&](bool block) -> bool {
            const int b = (int)(issued % p.cv_nbuf);
            const int64_t use = issued / p.cv_nbuf;
            if (use >= 1) {
                const uint32_t a = smem_u32(&bar_released[b]), par = (uint32_t)((use - 1) & 1);
                if (block) {
                    if (!warp_wait_phase<32>(a, par, abort_flag)) { ok = false; return false; }
                } else if (!__all_sync(0xffffffffu, mbar_try(a, par))) {
                    return false;
                }
            }
            if (lane == 0) issue(issued);
            __syncwarp();
            ++issued;
            return true;
        };
        for (int64_t job = 0; ok && job < n_jobs; ++job) {
            while (ok && issued <= job) try_issue(true);
            if (!ok) break;
            if (fin) {
                const int b = (int)(job % p.cv_nbuf);
                if (!warp_wait_phase<32>(smem_u32(&bar_landed[b]), (uint32_t)(job / p.cv_nbuf) & 1, abort_flag)) {
                    ok = false;
                    break;
                }
                const int64_t i = job / p.cv_nchunk;
                const int c = (int)(job - i * p.cv_nchunk);
                int64_t row0;
                int oy0;
                const int nimg = tile_geo(i, row0, oy0);
                const int ncell = p.cv_hw * p.cv_hh;
                for (int im = 0; im < nimg; ++im) {
                    const int64_t row = logical_row(p.lrow, row0 + im);
                    const int g = (int)(row / p.T);
                    const int k = p.ov.n_neurons[g];
                    const int32_t *ids = p.ov.ids + p.ov.neuron_off[g];
                    const float *prow = p.ov.patch + row * p.ov.row_stride;
                    const uint32_t base = cv_region + (uint32_t)b * cv_buf_bytes + (uint32_t)im * p.cv_img_bytes;
                    for (int q = 0; q < k; ++q) {
                        const int jl = ids[q] - c * p.cv_cw;
                        if (jl < 0 || jl >= p.cv_cw) continue;
                        const float *pq = prow + (int64_t)q * p.ov.cells;
                        for (int cell = lane; cell < ncell; cell += 32) {
                            const int hy = cell / p.cv_hw, hx = cell - hy * p.cv_hw;
                            const int iy = oy0 - p.pad + hy, ix = hx - p.pad;
                            if ((unsigned)iy >= (unsigned)p.ih || (unsigned)ix >= (unsigned)p.iw) continue;
                            const uint32_t lin = (uint32_t)cell * 128u + (uint32_t)jl * 4u;
                            asm volatile("st.shared.f32 [%0], %1;" ::"r"(base + (lin ^ ((lin >> 3) & 0x70u))),
                                         "f"(__ldg(pq + iy * p.iw + ix))
                                         : "memory");
                        }
                    }
                }
                __syncwarp();
                if (lane == 0) mbar_arrive(smem_u32(&bar_ready[b]));
            }
            // run ahead while buffers are free, without holding up the next job's overlay
            while (ok && issued < n_jobs && issued < job + p.cv_nbuf && try_issue(!fin)) {
            }
        }
        // the copies still in flight land before the shared memory is released
        if (lane == 0)
            for (int64_t jj = issued > p.cv_nbuf ? issued - p.cv_nbuf : 0; jj < issued; ++jj)
                wait_phase_drain(smem_u32(&bar_landed[jj % p.cv_nbuf]), (uint32_t)((jj / p.cv_nbuf) & 1));
    } else if (warp < 11) {
        // ------------------------------------------------------------------ MMA --
        // The K-steps of a tile are dealt to the n_mma issuing warps by their index
        // (kt mod n_mma = w), each warp into its own partial accumulator.  One thread
        // issues an MMA only about every 60 cycles and then waits for its next stage,
        // so while one warp waits the others keep the tensor pipe busy.  The split
        // depends on kt alone: a row's partial sums never depend on its place in the
        // batch.  With mma_chain the warps share one accumulator and take the K-steps
        // in turn: a warp issues K-step g only once the warp before it has issued g - 1
        // (an arrival on the turn barrier), so the MMAs reach the tensor pipe in K-step
        // order, as from one warp, while each warp's barrier waits and commits overlap
        // the other's issue.  (A barrier is never two phases ahead of its waiter: the
        // other warp's next turn waits for this warp's arrival.)
        const int w = warp - 8;
        if (pair) {
            // tile pairs: warp w issues tile w of each unit into its own accumulator, both
            // warps side by side from the same A and weight stages (each stage is released
            // by the commits of both)
            if (lane == 0 && w < 2) {
                constexpr int Q = THREE ? 12 : 4;
                const uint32_t id = idesc_tf32(kTileM, Nt), id2 = idesc_tf32(kTileM, 2 * Nt);
                const bool merged = THREE && p.merge_lo;
                bool ok = true;
                if (p.b_resident) ok = wait_phase<32>(smem_u32(&bar_bfull[0]), 0, abort_flag);
                const uint64_t desc_b0 = sw128_desc(b_region);
                const uint32_t b_step16 = b_step >> 4, lo16 = (uint32_t)Nt * 128 >> 4;
                int t = 0, sb = 0;
                uint32_t t_wraps = 0, b_wraps = 0;
                for (int64_t i = 0; ok && i < my_tiles; ++i) {
                    const int a = p.n_acc == 2 ? (int)(i & 1) : 0;
                    const int64_t use = p.n_acc == 2 ? (i >> 1) : i;
                    if (use >= 1 && !wait_phase<32>(smem_u32(&bar_accempty[a]), (uint32_t)((use - 1) & 1), abort_flag)) break;
                    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
                    const uint32_t d = tmem + (uint32_t)((a * 2 + w) * p.acc_cols);
                    for (int kt = 0; kt < nK; ++kt) {
                        if (!wait_phase<32>(smem_u32(&bar_afull[t]), t_wraps & 1, abort_flag)) { ok = false; break; }
                        if (!p.b_resident &&
                            !wait_phase<32>(smem_u32(&bar_bfull[sb]), b_wraps & 1, abort_flag)) { ok = false; break; }
                        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
                        const uint64_t dh = desc_b0 + (uint64_t)((p.b_resident ? kt : sb) * b_step16), dl = dh + lo16;
                        const uint32_t ta = tmem + p.a_col + (uint32_t)(t * 2 + w) * kAColsPerStage;
                        const uint32_t acc0 = kt > 0 ? 1u : 0u;   // K-step 0 of the tile overwrites
                        if (merged) mma_block_merged(d, ta, dh, id2, id, acc0);
                        else mma_block<THREE, 0, Q>(d, ta, dh, dl, id, acc0);
                        mma_commit(smem_u32(&bar_aempty[t]));
                        if (!p.b_resident) mma_commit(smem_u32(&bar_bempty[sb]));
                        if (++t == p.n_stages) { t = 0; ++t_wraps; }
                        if (!p.b_resident && ++sb == p.nb) { sb = 0; ++b_wraps; }
                    }
                    if (!ok) break;
                    mma_commit(smem_u32(&bar_accfull[a]));
                }
                // every MMA of both issuing warps has finished before the teardown
                mma_commit(smem_u32(&bar_drain));
                wait_phase_drain(smem_u32(&bar_drain), 0);
            }
        } else if (lane == 0 && w < p.n_mma) {
            const int nmma = p.n_mma, nacc = p.n_acc;
            constexpr int Q = THREE ? 12 : 4;
            const uint32_t id = idesc_tf32(kTileM, Nt), id2 = idesc_tf32(kTileM, 2 * Nt);
            // (the window GEMM never takes these paths: compiled out of its latency-bound
            // issuing loop)
            const bool merged = MODE == 3 && THREE && p.merge_lo;
            bool ok = true;
            if (p.b_resident) ok = wait_phase<32>(smem_u32(&bar_bfull[0]), 0, abort_flag);
            const uint64_t desc_b0 = sw128_desc(b_region);
            const uint32_t b_step16 = b_step >> 4, lo16 = (uint32_t)Nt * 128 >> 4;
            int t = 0, sb = 0;                  // ring slots of K-step kt (every warp tracks every step)
            uint32_t t_wraps = 0, b_wraps = 0;
            for (int64_t i = 0; ok && i < my_tiles; ++i) {
                const int a = nacc == 2 ? (int)(i & 1) : 0;
                const int64_t use = nacc == 2 ? (i >> 1) : i;
                if (use >= 1 && !wait_phase<32>(smem_u32(&bar_accempty[a]), (uint32_t)((use - 1) & 1), abort_flag)) break;
                asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
                const bool chain = MODE != 2 && p.mma_chain != 0;
                const uint32_t d = tmem + (uint32_t)((a * p.n_part + (chain ? 0 : w)) * p.acc_cols);
                // two warps keep dealing across tiles (an odd nK alternates which warp
                // takes the extra K-step); the epilogue's p0 + p1 is commutative, so a
                // row's sum does not depend on which partial holds which K-steps
                int own = nmma == 2 ? (int)((i * nK) & 1) : 0;
                bool first = true;              // the warp's first K-step of the tile overwrites
                for (int kt = 0; kt < nK; ++kt) {
                    if (own == w) {
                        if (!wait_phase<32>(smem_u32(&bar_afull[t]), t_wraps & 1, abort_flag)) { ok = false; break; }
                        if (!p.b_resident &&
                            !wait_phase<32>(smem_u32(&bar_bfull[sb]), b_wraps & 1, abort_flag)) { ok = false; break; }
                        const uint32_t g = (uint32_t)(i * nK + kt);
                        // K-step g goes to warp g mod 2; it waits for the other warp's
                        // arrival after K-step g - 1, the ((g + w) / 2)-th on its barrier
                        if (chain && g > 0 &&
                            !wait_phase<0>(smem_u32(&bar_turn[w]), (((g + (uint32_t)w) >> 1) + 1) & 1, abort_flag)) {
                            ok = false;
                            break;
                        }
                        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
                        const uint64_t dh = desc_b0 + (uint64_t)((p.b_resident ? kt : sb) * b_step16), dl = dh + lo16;
                        // shared accumulator: K-step 0 of the tile overwrites
                        const uint32_t acc0 = chain ? (kt > 0 ? 1u : 0u) : (first ? 0u : 1u);
                        if (merged) mma_block_merged(d, tmem + p.a_col + t * kAColsPerStage, dh, id2, id, acc0);
                        else mma_block<THREE, 0, Q>(d, tmem + p.a_col + t * kAColsPerStage, dh, dl, id, acc0);
                        first = false;
                        if (chain) {
                            asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
                            mbar_arrive(smem_u32(&bar_turn[1 - w]));
                        }
                        mma_commit(smem_u32(&bar_aempty[t]));
                        if (!p.b_resident) mma_commit(smem_u32(&bar_bempty[sb]));
                    }
                    if (++own == nmma) own = 0;
                    if (++t == p.n_stages) { t = 0; ++t_wraps; }
                    if (!p.b_resident && ++sb == p.nb) { sb = 0; ++b_wraps; }
                }
                if (!ok) break;
                mma_commit(smem_u32(&bar_accfull[a]));
            }
            // every MMA of every issuing warp has finished before the teardown
            mma_commit(smem_u32(&bar_drain));
            wait_phase_drain(smem_u32(&bar_drain), 0);
        }
    } else {
        // -------------------------------------------------------------- weights --
        if (MODE == 3 && lane == 0) {
            // the weight K-steps, each copy as soon as the MMAs have released its slot (the
            // staged input rows come from warp 10)
            const int64_t n_b = p.b_resident ? 0 : total;
            if (p.b_resident) {
                const uint32_t bytes = (uint32_t)nK * b_step;
                mbar_expect_tx(smem_u32(&bar_bfull[0]), bytes);
                for (uint32_t o = 0; o < bytes; o += 32768u)
                    bulk_g2s(b_region + o, (const unsigned char *)wslice + o, min(32768u, bytes - o),
                             smem_u32(&bar_bfull[0]));
            }
            int64_t jb = 0;
            for (; jb < n_b; ++jb) {
                const int sb = (int)(jb % p.nb);
                const int64_t use = jb / p.nb;
                if (use >= 1 && !wait_phase<32>(smem_u32(&bar_bempty[sb]), (uint32_t)((use - 1) & 1), abort_flag)) break;
                mbar_expect_tx(smem_u32(&bar_bfull[sb]), b_step);
                bulk_g2s(b_region + (uint32_t)sb * b_step, (const unsigned char *)wslice + (size_t)(jb % nK) * b_step,
                         b_step, smem_u32(&bar_bfull[sb]));
            }
            // the copies still in flight land before the shared memory is released
            for (int64_t jj = jb > p.nb ? jb - p.nb : 0; jj < jb; ++jj)
                wait_phase_drain(smem_u32(&bar_bfull[(int)(jj % p.nb)]), (uint32_t)((jj / p.nb) & 1));
        } else if (lane == 0) {
            if (p.b_resident) {
                const uint32_t bytes = (uint32_t)nK * b_step;
                mbar_expect_tx(smem_u32(&bar_bfull[0]), bytes);
                for (uint32_t o = 0; o < bytes; o += 32768u)
                    bulk_g2s(b_region + o, (const unsigned char *)wslice + o, min(32768u, bytes - o),
                             smem_u32(&bar_bfull[0]));
            } else {
                int64_t j = 0;
                int sb = 0, kt = 0;
                uint32_t wraps = 0;
                for (; j < total; ++j) {
                    if (wraps >= 1 && !wait_phase<64>(smem_u32(&bar_bempty[sb]), (wraps - 1) & 1, abort_flag)) break;
                    mbar_expect_tx(smem_u32(&bar_bfull[sb]), b_step);
                    bulk_g2s(b_region + (uint32_t)sb * b_step, (const unsigned char *)wslice + (size_t)kt * b_step,
                             b_step, smem_u32(&bar_bfull[sb]));
                    if (++kt == nK) kt = 0;
                    if (++sb == p.nb) { sb = 0; ++wraps; }
                }
                // the copies still in flight land before the shared memory is released
                for (int64_t jj = std::max<int64_t>(0, j - p.nb); jj < j; ++jj)
                    wait_phase_drain(smem_u32(&bar_bfull[(int)(jj % p.nb)]), (uint32_t)((jj / p.nb) & 1));
            }
        }
        if constexpr (MODE == 2) {
            // ------------------------------------------------ map staging: copies --
            // tile j goes to buffer j mod NBUF once the producers have released the
            // tile that held it (a bulk copy issue can stall for hundreds of cycles, so
            // this warp does nothing else)
            using G = SmallConv;
            int64_t issued = 0;
            int b = 0;
            uint32_t uses = 0;
            for (; issued < my_tiles; ++issued) {
                if (issued >= G::NBUF && !warp_wait_phase<32>(smem_u32(&bar_released[b]), (uses - 1) & 1, abort_flag)) break;
                issue_tile(issued, b);
                __syncwarp();
                if (++b == G::NBUF) { b = 0; ++uses; }
            }
            // the copies of the last tiles (the only ones that can still be in flight)
            // land before the shared memory is released
            if (lane == 0)
                for (int64_t j = issued > G::NBUF ? issued - G::NBUF : 0; j < issued; ++j)
                    wait_phase_drain(smem_u32(&bar_landed[j % G::NBUF]), (uint32_t)((j / G::NBUF) & 1));
        }
        if (lane == 0 && p.b_resident) wait_phase_drain(smem_u32(&bar_bfull[0]), 0);
    }

    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    if (threadIdx.x == 0 && abort_sh.abort) atomicExch(p.err, MURE_ERR_TIMEOUT);
    if (warp == 0) {
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(512));
    }
}

// Split fp32 weights [N][K] into TF32 halves laid out as the kernel's shared-memory
// operand: for each 128-channel slice s and K-step kc, the hi plane then (3xTF32)
// the lo plane, each Nt rows of 32 values in 128-byte-swizzled order.
// perm_ic > 0 (the staged convolution): K-step kc holds channels 32 (kc / taps) .. +31
// of filter tap kc mod taps, i.e. the K order (chunk, tap, channel) of its producers.
__global__ void k_swizzle_weights(const float *__restrict__ W, int N, int K, int Np, int Kp, int planes,
                                  int64_t slice_floats, float *out, int perm_ic, int taps, int slice_w)
{
    const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= (int64_t)Np * Kp) return;
    const int n = (int)(i / Kp), k = (int)(i % Kp);
    int ks = k;
    if (perm_ic > 0) {
        const int kc = k / kTileK;
        ks = (kc % taps) * perm_ic + (kc / taps) * kTileK + k % kTileK;
    }
    const float w = (n < N && k < K) ? W[(int64_t)n * K + ks] : 0.f;
    const float h = tf32_rna(w);
    const int s = n / slice_w, nl = n % slice_w, Nt = min(slice_w, Np - s * slice_w);
    const int kc = k / kTileK, kk = k % kTileK;
    const int64_t chunk = (int64_t)s * slice_floats + (int64_t)kc * planes * Nt * kTileK;
    const int64_t off = (sw128_off(nl, kk >> 2) >> 2) + (kk & 3);
    out[chunk + off] = h;
    if (planes == 2) out[chunk + (int64_t)Nt * kTileK + off] = tf32_rna(w - h);
}

int tc_supported(const Stage &S)
{
    if (S.oc < 16) return 0;
    if (S.kind == MURE_NODE_DENSE) return !S.has_add && !S.pool && !S.gap;
    // implicit-GEMM convolution: pooled maps need whole windows per warp (always true:
    // a window is 4 consecutive GEMM rows and tiles start at multiples of 128)
    return S.kind == MURE_NODE_CONV2D;
}

// Whether a convolution has the small-image mode's geometry.
int tc_small_geometry(const Stage &S)
{
    using G = SmallConv;
    return S.kind == MURE_NODE_CONV2D && S.ih == G::IH && S.iw == G::IW && S.ic == G::IC && S.kh == G::KH &&
           S.kw == G::KW && S.stride == 1 && S.pad == 0 && S.pool && !S.has_add && !S.gap && S.oc == G::OC;
}

// The staged convolution's tile: 128 GEMM rows are whole output rows of one batch row
// (maps of >= 128 positions) or whole maps of several batch rows; the staged input is
// the rows they read, zero border included, one 32-channel chunk per buffer.
struct ConvTile {
    int imgs, rows, hw, hh, cw;
    uint32_t img_bytes;
};

// The staged geometry of units of tm GEMM rows (one tile, or a pair of tiles), with at most
// max_bytes of staged rows per buffer.
static bool conv_tile(const Stage &S, ConvTile &t, int tm = kTileM, size_t max_bytes = 48 * 1024, bool win = false)
{
    if (S.kind != MURE_NODE_CONV2D || S.stride != 1 || (S.ic % kTileK != 0 && S.ic != 16)) return false;
    t.cw = S.ic == 16 ? 16 : kTileK;
    if ((S.pool || win) && ((S.oh & 1) || (S.ow & 1))) return false;
    const int P = S.pool ? 4 * (S.oh / 2) * (S.ow / 2) : S.oh * S.ow;
    if (win) {
        // whole rows of 2x2 windows: tm windows are 2 tm / (ow / 2) output rows
        const int pw = S.ow / 2, Pw = (S.oh / 2) * pw;
        if (S.pool || S.kh != 3 || S.kw != 3 || S.pad != 1 || Pw % tm != 0 || tm % pw != 0) return false;
        t.imgs = 1;
        t.rows = 2 * (tm / pw);
    } else if (P >= tm) {
        // whole output rows per tile; pooled tiles hold whole rows of pooling windows
        if (P % tm != 0 || tm % S.ow != 0) return false;
        t.imgs = 1;
        t.rows = tm / S.ow;
        if (S.pool && (t.rows & 1)) return false;
    } else {
        if (tm % P != 0) return false;
        t.imgs = tm / P;
        t.rows = S.oh;
    }
    // staged width: the kw - 1 border columns, then padded (zero-filled columns past the
    // image) to 4 mod 8 lines, so that the 8 lanes of a quarter warp reading a pooling
    // window pair (lines b, b+1, b+hw, b+hw+1, b+2, ...) hit 8 different 16-byte bank
    // groups of the 128-byte swizzle (line l's chunk c sits at c ^ (l mod 8))
    t.hw = S.ow + S.kw - 1;
    t.hw += (4 - t.hw % 8 + 8) % 8;
    t.hh = t.rows + S.kh - 1;
    if (t.hw > 256 || t.hh > 256) return false;
    t.img_bytes = (uint32_t)((t.hw * t.hh * 128 + 1023) & ~1023);
    // at least two buffers beside the streamed weights (three K-steps of 128 channels)
    return (size_t)t.imgs * t.img_bytes <= max_bytes;
}

// The window form of the staged mode: 16-channel 3x3 convolutions with 16 outputs,
// stride 1, pad 1, no pooling, whose windows fill whole 128-row tiles.
int tc_win_geometry(const Stage &S)
{
    ConvTile t;
    return S.ic == 16 && S.oc == 16 && conv_tile(S, t, kTileM, 96 * 1024, true) ? 1 : 0;
}

int tc_conv_geometry(const Stage &S)
{
    ConvTile t;
    return conv_tile(S, t) ? 1 : 0;
}

// Whether the tensor-core kernel can fetch a first-suffix overlay itself: at most
// kOvMax patch values per row and K-step (dense: at most 4 mutated channels).
int tc_overlay_inline(const Stage &S, const Overlay &ov, int64_t groups)
{
    if (S.tc_conv) return 1;   // warp 10 writes any number of mutated channels
    if (S.tc_small)
        return ov.kmax <= SmallConv::MAXQ && groups <= SmallConv::MAXG && ov.cells == SmallConv::CELLS;
    if (S.kind == MURE_NODE_DENSE) {
        if (ov.kmax > 4) return 0;
        const int per_slot = std::min(ov.cells, (kTileK + ov.ch - 1) / ov.ch + 1);
        return ov.kmax * per_slot <= kOvMax;
    }
    if ((S.ic & 3) != 0) return 1;   // 4-byte copies take the patch value directly
    const int pixels = (S.ic % kTileK == 0 || kTileK % S.ic == 0) ? std::max(1, kTileK / S.ic) : kTileK / S.ic + 2;
    return ov.kmax * pixels <= kOvMax;
}

// The GEMM's N and K: the small-image mode multiplies by the window-expanded weights.
static int gemm_n(const Stage &S) { return S.tc_small ? SmallConv::N : S.tc_win ? 4 * S.oc : S.oc; }
static int gemm_k(const Stage &S) { return S.tc_small ? SmallConv::K : S.tc_win ? 16 * S.ic : S.K; }

// W [OC][(ky, kx, ci)] -> W' [(s, c)][(wy, wx, ci)]: the filter of window position
// s = 2 dy + dx placed at offset (dy, dx) in the window's receptive field.
__global__ void k_expand_window_weights(const float *__restrict__ W, float *out)
{
    using G = SmallConv;
    const int i = blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= G::N * G::K) return;
    const int n = i / G::K, k = i % G::K;
    const int sidx = n / G::OC, c = n % G::OC, dy = sidx >> 1, dx = sidx & 1;
    const int wy = k / (G::KU * G::IC), wx = (k / G::IC) % G::KU, ci = k % G::IC;
    const int ky = wy - dy, kx = wx - dx;
    out[i] = ((unsigned)ky < (unsigned)G::KH && (unsigned)kx < (unsigned)G::KW)
                 ? W[(int64_t)c * (G::KH * G::KW * G::IC) + (ky * G::KW + kx) * G::IC + ci]
                 : 0.f;
}

// The staged mode's windows: W [OC][(ky, kx, ci)] of a 3x3 filter -> W' [(s, c)][(wy, wx,
// ci)] over the 4x4 field of a 2x2 output window, position s = 2 dy + dx's filter at
// offset (dy, dx), zeros elsewhere.
__global__ void k_expand_field_weights(const float *__restrict__ W, int oc, int ic, float *out)
{
    const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const int N = 4 * oc, K = 16 * ic;
    if (i >= (int64_t)N * K) return;
    const int n = (int)(i / K), k = (int)(i % K);
    const int sidx = n / oc, c = n % oc, dy = sidx >> 1, dx = sidx & 1;
    const int wy = k / (4 * ic), wx = (k / ic) % 4, ci = k % ic;
    const int ky = wy - dy, kx = wx - dx;
    out[i] = ((unsigned)ky < 3u && (unsigned)kx < 3u) ? W[(int64_t)c * (9 * ic) + (ky * 3 + kx) * ic + ci] : 0.f;
}

// Output channels per CTA: one wide N = 256 slice for staged convolutions of exactly
// 256 outputs (the MMA's tensor work per K-step then exceeds its issue cost), else
// slices of 128.
static int slice_width(const Stage &S) { return S.tc_wide ? kSliceMax : kSlice; }

int64_t tc_weight_floats(const Stage &S)
{
    const int Np = round_up16(gemm_n(S)), Kp = round_up32(gemm_k(S)), planes = S.tc == 1 ? 2 : 1;
    const int sw = slice_width(S);
    const int64_t slice = (int64_t)planes * sw * Kp;
    return slice * ((Np + sw - 1) / sw);
}

int tc_wide_geometry(const Stage &S) { return S.tc_conv && round_up16(S.oc) == kSliceMax; }

// tmp: scratch of SmallConv::N * SmallConv::K floats for the small-image mode (else unused).
int launch_swizzle_weights(const Stage &S, float *out, float *tmp, cudaStream_t s)
{
    const int N = gemm_n(S), K = gemm_k(S);
    const int Np = round_up16(N), Kp = round_up32(K), planes = S.tc == 1 ? 2 : 1;
    const int64_t n = (int64_t)Np * Kp;
    int launches = 1;
    const float *W = S.W;
    if (S.tc_small) {
        k_expand_window_weights<<<(N * K + 255) / 256, 256, 0, s>>>(S.W, tmp);
        W = tmp;
        ++launches;
    } else if (S.tc_win) {
        k_expand_field_weights<<<(N * K + 255) / 256, 256, 0, s>>>(S.W, S.oc, S.ic, tmp);
        W = tmp;
        ++launches;
    }
    cudaMemsetAsync(out, 0, tc_weight_floats(S) * sizeof(float), s);
    k_swizzle_weights<<<(unsigned)((n + 255) / 256), 256, 0, s>>>(W, N, K, Np, Kp, planes,
                                                                   (int64_t)planes * slice_width(S) * Kp, out,
                                                                   S.tc_conv && S.ic > kTileK ? S.ic : 0, S.kh * S.kw,
                                                                   slice_width(S));
    return launches;
}

// Multiply-accumulates one batch row costs the tensor-core kernel, padding included.
int64_t tc_macs_per_row(const Stage &S)
{
    const int64_t Np = round_up16(gemm_n(S)), Kp = round_up32(gemm_k(S));
    if (S.kind == MURE_NODE_DENSE) return Np * Kp;
    // the small-image mode runs a 128-row tile per SmallConv::MAPS maps
    if (S.tc_small) return (kTileM * Np * Kp + SmallConv::MAPS / 2) / SmallConv::MAPS;
    if (S.tc_win) return (int64_t)(S.oh / 2) * (S.ow / 2) * Np * Kp;
    const int64_t P = S.pool ? 4 * (S.oh / 2) * (S.ow / 2) : (int64_t)S.oh * S.ow;
    return P * Np * Kp;
}

int64_t tc_swizzle_tmp_floats(const Stage &S)
{
    return S.tc_small ? (int64_t)SmallConv::N * SmallConv::K : S.tc_win ? (int64_t)gemm_n(S) * gemm_k(S) : 0;
}

// The longest run of the K-step sequence (tile after tile, nK steps each) between two
// consecutive K-steps of one issuing warp, when K-step kt goes to warp kt mod m.
static int mma_gap(int nK, int m)
{
    int g = nK > m ? m : 0;
    for (int w = 0; w < m; ++w) g = std::max(g, nK - (w + m * ((nK - 1 - w) / m)) + w);
    return g;
}

// Tensor-memory layout (512 columns): n_acc sets of n_part partial accumulators, then
// n_stages A stages.  A function of the layer alone, so a row's arithmetic never
// depends on the batch.
static void tc_config(TcParams &p, int nt_max, bool three, bool chain)
{
    p.acc_cols = round_up32(p.merge_lo ? 2 * nt_max : nt_max);
    // a wide slice's accumulator takes half of tensor memory: one set
    p.n_acc = p.acc_cols > 128 ? 1 : 2;
    p.a_col = 256;
    p.n_stages = three ? 4 : 8;
    // An issuing warp waits on a ring slot's barrier by the parity of the slot's use
    // count, which names the right phase only while the warp's consecutive K-steps are
    // at most a ring's depth apart; every warp also has a K-step in every tile.
    const int nK = p.Kp / kTileK, depth = p.b_resident ? p.n_stages : std::min(p.n_stages, p.nb);
    int m = std::max(1, std::min({3, 256 / (p.n_acc * p.acc_cols), nK}));
    while (m > 1 && mma_gap(nK, m) > depth) --m;
    p.n_mma = m;
    p.n_part = m;
    p.mma_chain = 0;
    if (chain && nK >= 2 && mma_gap(nK, 2) <= depth) {
        // two issuing warps in turn on one accumulator per set: two sets up to 128
        // columns, one wide set
        p.n_mma = 2;
        p.n_part = 1;
        p.mma_chain = 1;
    }
}

// cuTensorMapEncodeTiled through the runtime's driver entry point (no link to libcuda).
static PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder()
{
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    static bool tried = false;
    if (!tried) {
        tried = true;
        void *f = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(f);
    }
    return fn;
}

// The A operand of a dense layer as a 2-D tensor [rows][K] with 128-byte swizzled
// boxes of 128 rows x 32 values (the producers' shared-memory layout): false for
// per-input rows, unaligned rows or without the encoder.
static bool dense_a_tensor_map(const Stage &S, Src x, RowMap rm, CUtensorMap &map)
{
    // rows of per-input tensors always carry a patch (the first suffix stage), so only
    // row-per-row tensors take this path
    if (x.per_input) return false;
    if ((x.stride * 4) % 16 != 0 || (reinterpret_cast<uintptr_t>(x.p) & 15) != 0) return false;
    PFN_cuTensorMapEncodeTiled_v12000 enc = tensor_map_encoder();
    if (!enc) return false;
    const float *base = x.p;
    const cuuint64_t dims[2] = {(cuuint64_t)S.K, (cuuint64_t)rm.R};
    const cuuint64_t strides[1] = {(cuuint64_t)x.stride * 4};
    const cuuint32_t box[2] = {(cuuint32_t)kTileK, (cuuint32_t)kTileM};
    const cuuint32_t estr[2] = {1, 1};
    return enc(&map, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, const_cast<float *>(base), dims, strides, box, estr,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_128B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// The input rows of a staged convolution as a 4-D tensor [row][ih][iw][ic] with boxes
// {32 channels, hw, hh, 1 row}, 128-byte swizzled, zero-filled outside the image.
static bool conv_x_tensor_map(const Stage &S, Src x, RowMap rm, const ConvTile &t, CUtensorMap &map)
{
    if ((x.stride * 4) % 16 != 0 || (reinterpret_cast<uintptr_t>(x.p) & 15) != 0) return false;
    PFN_cuTensorMapEncodeTiled_v12000 enc = tensor_map_encoder();
    if (!enc) return false;
    const int64_t rows = x.per_input ? rm.t0 + rm.T : rm.R;
    const cuuint64_t dims[4] = {(cuuint64_t)S.ic, (cuuint64_t)S.iw, (cuuint64_t)S.ih, (cuuint64_t)rows};
    const cuuint64_t strides[3] = {(cuuint64_t)S.ic * 4, (cuuint64_t)S.iw * S.ic * 4, (cuuint64_t)x.stride * 4};
    // 32 channels per line whatever the chunk: a 16-channel tensor's lines get 16 zeros
    const cuuint32_t box[4] = {(cuuint32_t)kTileK, (cuuint32_t)t.hw, (cuuint32_t)t.hh, 1};
    const cuuint32_t estr[4] = {1, 1, 1, 1};
    return enc(&map, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 4, const_cast<float *>(x.p), dims, strides, box, estr,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_128B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Dynamic shared memory a k_tc_gemm instance may use: the device's opt-in maximum less
// the kernel's static shared memory.
template <class Kern>
static size_t tc_dyn_smem_max(Kern kern)
{
    static size_t cached = 0;
    if (!cached) {
        int dev = 0, optin = 0;
        cudaGetDevice(&dev);
        cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
        cudaFuncAttributes fa{};
        cudaFuncGetAttributes(&fa, kern);
        cached = optin > (int)fa.sharedSizeBytes ? (size_t)optin - fa.sharedSizeBytes : 0;
    }
    return cached;
}

int tc_final_fusable(const Stage &S, const Stage &SL)
{
    return S.tc && S.kind == MURE_NODE_DENSE && tc_supported(S) && round_up16(S.oc) <= kSlice &&
           SL.kind == MURE_NODE_DENSE && SL.K == S.oc && SL.oc >= 1 && SL.oc <= kFuseClasses && !SL.has_add &&
           !SL.gap && !SL.pool;
}

int launch_tc(const Stage &S, Src x, RowMap rm, float *z_out, int64_t z_stride, Src skip, float *y_out,
              int64_t y_stride, float *gap_tmp, cudaStream_t s, const Overlay *ov, const FinalFuse *ff,
              const SlotStore *ss)
{
    if (rm.R <= 0) return 0;
    TcParams p{};
    const bool dense = S.kind == MURE_NODE_DENSE;
    p.x = x.p; p.x_stride = x.stride; p.x_per_input = x.per_input;
    p.t0 = rm.t0; p.T = rm.T; p.R = rm.R; p.lrow = rm.lrow;
    p.ih = S.ih; p.iw = S.iw; p.ic = S.ic; p.kh = S.kh; p.kw = S.kw; p.stride = S.stride; p.pad = S.pad;
    p.oh = S.oh; p.ow = S.ow;
    p.pool = S.pool; p.pw = S.ow / 2;
    p.P = dense ? 1 : (S.pool ? 4 * (S.oh / 2) * (S.ow / 2) : S.oh * S.ow);
    p.K = S.K; p.Kp = round_up32(S.K); p.N = S.oc; p.Np = round_up16(S.oc);
    if (S.tc_small) {
        p.P = SmallConv::P;
        p.K = SmallConv::K; p.Kp = round_up32(SmallConv::K); p.Np = SmallConv::N;
    }
    p.cv_fw = S.kw;
    p.cv_ntap = S.kh * S.kw;
    if (S.tc_win) {
        // GEMM rows = 2x2 windows, columns = (position, output), K = the 4x4 field
        p.P = (S.oh / 2) * (S.ow / 2);
        p.K = p.Kp = gemm_k(S);
        p.Np = gemm_n(S);
        p.cv_win = 1;
        p.cv_fw = 4;
        p.cv_ntap = 16;
    }
    const bool three = S.tc == 1;
    const int planes = three ? 2 : 1;
    p.Wsw = S.Wtc;
    p.slice_w = slice_width(S);
    p.w_slice_floats = (int64_t)planes * p.slice_w * p.Kp;
    p.b = S.b;
    p.act1 = S.act1; p.has_add = S.has_add; p.act2 = S.act2;
    p.skip = skip.p; p.skip_stride = skip.stride; p.skip_per_input = skip.per_input;
    p.sk_w = S.sk_w; p.sk_c = S.sc_c; p.sk_stride = S.sc_stride;
    p.z = z_out; p.z_stride = z_stride;
    // with global average pooling the post-op map goes to gap_tmp first
    const int mh = S.pool ? S.oh / 2 : S.oh, mw = S.pool ? S.ow / 2 : S.ow;
    const int64_t map_stride = round4((int64_t)mh * mw * S.oc);
    p.y = S.gap ? gap_tmp : y_out;
    p.y_stride = S.gap ? map_stride : y_stride;
    if (ov) p.ov = *ov;
    p.err = S.err;
    p.spin = S.wait_limit ? *S.wait_limit : 0;
    // shared memory: the weights (whole slice, or kNB K-steps), then the producer ring
    const int nt_max = std::min(p.slice_w, p.Np);
    const size_t b_step = (size_t)planes * nt_max * 128;
    const size_t slice_bytes = b_step * (p.Kp / kTileK);
    p.b_resident = slice_bytes <= (S.tc_small ? 112 : 96) * 1024;
    // a wide slice streams 64 KiB per K-step: two stages in flight
    // (the windows' staged rows leave room for two weight stages)
    p.nb = p.slice_w > kSlice || S.tc_win ? 2 : kNB;
    size_t b_bytes = p.b_resident ? slice_bytes : p.nb * b_step;
    // at least 116 KiB so that one CTA (holding all 512 tensor-memory columns) runs per SM
    size_t a_bytes = S.tc_small ? (size_t)SmallConv::BYTES
                                : (size_t)kNA * kStageA + (p.ov.patch ? (size_t)kNA * kOvSlotBytes : 0);
    ConvTile ct{};
    if (S.tc_conv) {
        // the staged convolution: as many staging buffers (up to 4) as fit beside the
        // weights; the weights' K order was fixed for it at model load.  Slices of up to
        // 64 outputs (not the delta GEMM) take units of two tiles where two buffers of
        // their staged rows fit (measured: conv 64->64 -14%, ResNet-20's 16- to 64-channel
        // convolutions -9..-10%; at 128 outputs the pair's single accumulator set, which
        // no longer overlaps the epilogue, made it 4-20% slower)
        const size_t room = three ? tc_dyn_smem_max(k_tc_gemm<3, true>) : tc_dyn_smem_max(k_tc_gemm<3, false>);
        bool ok = false;
        if (!ss && !S.tc_win && nt_max <= 64 && conv_tile(S, ct, 2 * kTileM, 64 * 1024) &&
            room >= 1024 + b_bytes + 2 * (size_t)ct.imgs * ct.img_bytes)
            ok = p.cv_pair = conv_x_tensor_map(S, x, rm, ct, p.tmap_x) ? 1 : 0;
        if (!ok) {
            p.cv_pair = 0;
            ok = conv_tile(S, ct, kTileM, S.tc_win ? 96 * 1024 : 48 * 1024, S.tc_win != 0) &&
                 conv_x_tensor_map(S, x, rm, ct, p.tmap_x);
        }
        const size_t buf = (size_t)ct.imgs * ct.img_bytes;
        if (p.b_resident && room < 1024 + b_bytes + 2 * buf) {
            // resident weights would leave room for fewer than two staging buffers: stream them
            p.b_resident = 0;
            b_bytes = (size_t)p.nb * b_step;
        }
        const int nbuf = ok && room > 1024 + b_bytes ? (int)std::min<size_t>(kNBufMax, (room - 1024 - b_bytes) / buf) : 0;
        if (nbuf < 2) {
            static const int unsupported = MURE_ERR_UNSUPPORTED;
            cudaMemcpyAsync(S.err, &unsupported, sizeof(int), cudaMemcpyHostToDevice, s);
            return 0;
        }
        p.cv_cw = ct.cw;
        p.cv_taps = (p.cv_ntap * ct.cw + kTileK - 1) / kTileK;
        p.cv_nchunk = S.ic / ct.cw;
        p.cv_imgs = ct.imgs;
        p.cv_rows = ct.rows;
        p.cv_hw = ct.hw;
        p.cv_hh = ct.hh;
        p.cv_img_bytes = ct.img_bytes;
        p.cv_nbuf = nbuf;
        a_bytes = (size_t)nbuf * buf;
    }
    if (ff) p.ff = *ff;
    if (ss) p.slot = *ss;
    const size_t f_bytes = ff ? 16 + (size_t)ff->F * kFuseClasses * 4 : 0;
    const size_t smem = std::max<size_t>(1024 + b_bytes + a_bytes + f_bytes, 116 * 1024);
    // partial accumulators: n_acc sets of n_part in columns 0..255; a function of the layer
    // alone, so a row's arithmetic never depends on the batch
    // (the window GEMM keeps two partial accumulators: measured as fast, no merged MMAs)
    // (not in the delta GEMM, whose slice width depends on the slots of its batch)
    // (with tile pairs only up to 32 outputs, where two accumulator sets of the merged
    // width still fit)
    p.merge_lo = S.tc_conv && three && !ss && nt_max <= (p.cv_pair ? 32 : 64) ? 1 : 0;
    tc_config(p, nt_max, three, !S.tc_small);
    // the delta GEMM: one issuing warp (or two in turn, which is the same sum), so that a
    // column's sum never depends on how many slots share its batch
    if (ss && !p.mma_chain) p.n_mma = p.n_part = 1;
    // dense rows without an overlay: A tiles by tensor-map copies from warp 10
    p.a_tma = dense && !p.ov.patch && p.n_mma <= 2 && dense_a_tensor_map(S, x, rm, p.tmap_a) ? 1 : 0;
    if (S.tc_small || S.tc_conv) {
        // warp 10 stages maps in those modes
        p.n_mma = std::min(p.n_mma, 2);
        if (!p.mma_chain) p.n_part = p.n_mma;
    }
    if (p.cv_pair) {
        // units of two tiles: MMA warp w issues tile w of a unit into its own accumulator,
        // the two warps side by side; an A stage holds the K-step of both tiles
        p.n_mma = 2;
        p.n_part = 1;
        p.mma_chain = 0;
        p.n_acc = 4 * p.acc_cols <= 256 ? 2 : 1;
        p.n_stages = three ? 2 : 4;
    }
    const int64_t M = (int64_t)rm.R * p.P;
    const int64_t unit = p.cv_pair ? 2 * kTileM : kTileM;
    const int64_t tiles = S.tc_small ? small_tiles(rm.R) : (M + unit - 1) / unit;
    static int n_sm = 0;
    if (!n_sm) {
        int dev = 0;
        cudaGetDevice(&dev);
        cudaDeviceGetAttribute(&n_sm, cudaDevAttrMultiProcessorCount, dev);
        if (n_sm <= 0) n_sm = 148;
    }
    const int ny = (p.Np + p.slice_w - 1) / p.slice_w;
    const dim3 grid((unsigned)std::max<int64_t>(1, std::min<int64_t>(tiles, std::max(1, n_sm / ny))), (unsigned)ny);
    auto go = [&](auto kern) {
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        kern<<<grid, kThreads, smem, s>>>(p);
    };
    if (dense && ff) { if (three) go(k_tc_gemm<0, true, kFuseClasses>); else go(k_tc_gemm<0, false, kFuseClasses>); }
    else if (dense) { if (three) go(k_tc_gemm<0, true>); else go(k_tc_gemm<0, false>); }
    else if (S.tc_small) { if (three) go(k_tc_gemm<2, true>); else go(k_tc_gemm<2, false>); }
    else if (S.tc_conv && ss && S.has_add) { if (three) go(k_tc_gemm<3, true, -1>); else go(k_tc_gemm<3, false, -1>); }
    else if (S.tc_conv) { if (three) go(k_tc_gemm<3, true>); else go(k_tc_gemm<3, false>); }
    else { if (three) go(k_tc_gemm<1, true>); else go(k_tc_gemm<1, false>); }
    int launches = 1;
    if (S.gap) launches += launch_gap(gap_tmp, map_stride, mh * mw, S.oc, rm.R, y_out, y_stride, s);
    return launches;
}

// ------------------------------------------------ tensor-core delta (GF / WS) --

// Column n of the batch's delta GEMM: slot n (its pair (group, q) listed by the host)
// takes the weight delta e of its neuron j (GF: the noise; WS: W[j][perm f] - W[j][f]);
// columns past the slots are zero.  The column bias is 0: the epilogue adds the cached
// pre-activation of channel j instead.  One thread per (column, k).
__global__ void k_slot_filters(int K, const PatchArgs pa, int n_slot, int Np, float *filt, float *colb, int32_t *colg,
                               int32_t *colq, int32_t *colj)
{
    const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= (int64_t)Np * K) return;
    const int n = (int)(i / K), k = (int)(i - (int64_t)n * K);
    if (n >= n_slot) {
        filt[i] = 0.f;
        if (k == 0) { colb[n] = 0.f; colg[n] = 0; colq[n] = 0; colj[n] = 0; }
        return;
    }
    const int g = pa.dslot[2 * n] - pa.dslot_g0, q = pa.dslot[2 * n + 1];
    filt[i] = pa.patch[pa.patch_off[g] + (int64_t)q * K + k];
    if (k == 0) { colb[n] = 0.f; colg[n] = g; colq[n] = q; colj[n] = pa.ids[pa.neuron_off[g] + q]; }
}

// Layers with a compiled small geometry keep the CUDA-core dot-product kernel, which
// stages each input once for all slots; the GEMM's gathers want channel counts that
// are multiples of 4 (16-byte copies).
int tc_delta_supported(const Stage &S, int precision)
{
    // (a residual add: the staged mode's slot instantiation adds each slot's own skip channel)
    return precision != MURE_PREC_FP32 && S.kind == MURE_NODE_CONV2D && !S.gap && S.geo == 0 && S.ic % 4 == 0 &&
           (!S.has_add || S.tc_conv);
}

void tc_delta_ws_size(int n_slots, int k_max, int64_t &floats, int64_t &ints)
{
    const int64_t Np = (int64_t)(n_slots + kSlice - 1) / kSlice * kSlice, Kp = round_up32(k_max);
    floats = Np * k_max + 2 * Np * Kp + Np;   // filters, swizzled halves, biases
    ints = 3 * Np;
}

int launch_tc_delta(const Stage &S, int precision, Src z, Src x, Src skip, RowMap rm_inputs, const PatchArgs &pa, float *out,
                    int64_t out_stride, const TcDeltaWs &dw, cudaStream_t s)
{
    const int n = (int)pa.n_dslot;
    if (n <= 0 || rm_inputs.R <= 0) return 0;
    const int Np = round_up16(n), K = S.K, Kp = round_up32(K);
    if (n > dw.n_max || K > dw.k_max) return -1;
    const int planes = precision == MURE_PREC_TF32X3 ? 2 : 1;
    k_slot_filters<<<(unsigned)(((int64_t)Np * K + 255) / 256), 256, 0, s>>>(K, pa, n, Np, dw.filt, dw.colb, dw.colg,
                                                                         dw.colq, dw.colj);
    k_swizzle_weights<<<(unsigned)(((int64_t)Np * Kp + 255) / 256), 256, 0, s>>>(dw.filt, Np, K, Np, Kp, planes,
                                                                               (int64_t)planes * kSlice * Kp, dw.swz,
                                                                               S.tc_conv && S.ic > kTileK ? S.ic : 0,
                                                                               S.kh * S.kw, kSlice);
    Stage D = S;
    D.oc = Np;
    D.tc_wide = 0;   // the slot filters are laid out in slices of 128
    D.tc = precision == MURE_PREC_TF32X3 ? 1 : 2;
    D.tc_small = 0;
    D.tc_win = 0;   // the slot GEMM runs per output position
    D.Wtc = dw.swz;
    D.b = dw.colb;
    SlotStore ss;
    ss.out = out;
    ss.stride = out_stride;
    ss.g = dw.colg;
    ss.q = dw.colq;
    ss.j = dw.colj;
    ss.z = z.p;
    ss.z_stride = z.stride;
    ss.z_per_input = z.per_input;
    ss.n = n;
    ss.cells = S.pool ? (S.oh / 2) * (S.ow / 2) : S.oh * S.ow;
    ss.T = rm_inputs.T;
    const RowMap rmT{rm_inputs.t0, rm_inputs.T, rm_inputs.T};
    // a residual add: the skip rows of the batch's inputs (per input, or the first
    // mutant's rows), added to each slot's own channel
    return 2 + launch_tc(D, x, rmT, nullptr, 0, skip, nullptr, 0, nullptr, s, nullptr, nullptr, &ss);
}

}  // namespace mure
