// Convolution as implicit GEMM on the 5th-generation tensor cores (tcgen05),
// operands staged by TMA, accumulators in tensor memory (TMEM).
//
// GEMM view (NHWC activations, KRSC weights, fp16/bf16 in, fp32 accumulate):
//   D[m, k] = sum_{r, s, c} A[m, (r, s, c)] * B[k, (r, s, c)]
//   m = output pixel (n, p, q), k = output channel.
// A tile of D is 128 pixels x BN channels.  The K loop runs over filter taps
// (r, s) and 64-channel blocks; every step stages
//   A: the 128 output pixels' input pixels for that tap, 64 channels
//      (one TMA box of a 4-D [N, H, W, C] tensor map: the tile is a
//      BNI x BH x BW block of output pixels, so for stride 1 the tap's input
//      pixels form a box too; zero padding comes from TMA's out-of-bounds
//      fill; stride 2 uses four tensor maps over the even/odd row and column
//      sub-lattices), or for 1x1 stride-1 layers a plain 2-D [N*H*W, C] box;
//   B: BN output channels x 64 channels of the tap (3-D [K, R*S, C] map).
// Both land in shared memory in the 128-byte-swizzled K-major layout that
// tcgen05.mma reads directly.
//
// The kernel is persistent: one CTA per SM walks the work units (a tile, or
// one K-range of a tile when the layer is split along K because it has too
// few tiles to fill the GPU), A-sharing tiles adjacent, with two TMEM
// accumulators so that draining one overlaps the main loop of the next.
// Warp roles (320 threads): warp 0 = TMA producer (+ TMEM allocation),
// warp 1 = MMA issuer (one thread), warps 2-9 = epilogue in two groups of
// four, group g draining accumulator g (alternate work units): TMEM ->
// registers -> bias + activation -> fp16/bf16 -> 128-byte-swizzled staging
// in shared memory -> one TMA tensor store per 32 rows x 64 channels
// (clipped at the tensor edges), or fp32 partial sums for a K split, summed
// by splitk_reduce_kernel.  Every mbarrier wait is bounded;
// on expiry the kernel records an error code in the library's error word,
// waits (bounded) for its own copies and MMAs, frees TMEM and exits.
#include <cuda.h>

#include <algorithm>
#include <cstdio>
#include <mutex>
#include <type_traits>
#include <vector>

#include "kern_common.cuh"

namespace sn {
namespace k {

namespace tc {

constexpr int BM = 128;
constexpr int BK = 64;
constexpr int THREADS = 320;
constexpr int EPI_WARPS = 8;
constexpr int MAX_K = 65536;
constexpr uint32_t STG_BYTES = 32 * 64 * 2;      // one epilogue staging block: 32 rows x 64 channels
constexpr long long WAIT_LIMIT = 4000000000LL;  // SM cycles (~2 s)
enum : int { ERR_TMA_WAIT = 0x10, ERR_MMA_WAIT = 0x20, ERR_ACC_WAIT = 0x40, ERR_EPI_WAIT = 0x80 };

struct Params {
    int32_t N, H, W, C, K, P, Q, R, S;
    int32_t stride, ph, pw, dh, dw;
    int32_t cblocks, kiters, ksplit;
    int32_t BW, BH, BNI, tq, tp;   // pixel-tile geometry (implicit mode)
    int32_t mtiles, ntiles;
    int64_t M;                     // plain mode: input rows (= output pixels)
    int64_t Mout;                  // output pixels N * P * Q
    int32_t act;
    const float *bias;
    void *y;                       // output, NHWC, fp16/bf16
    float *part;                   // K split: fp32 partial sums [ksplit][Mout][K]
    int *err;                      // the library's device error word
};

// ---------------------------------------------------------------- PTX helpers
__device__ __forceinline__ uint32_t su32(const void *p) { return (uint32_t)__cvta_generic_to_shared(p); }

__device__ __forceinline__ void mbar_init(uint64_t *b, uint32_t cnt) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(su32(b)), "r"(cnt) : "memory");
}
__device__ __forceinline__ void fence_mbar_init() {
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint64_t *b, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(su32(b)), "r"(bytes) : "memory");
}
__device__ __forceinline__ bool mbar_try(uint64_t *b, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(su32(b)), "r"(parity)
        : "memory");
    return ok != 0;
}
// bounded wait for the phase with the given parity; false on expiry
__device__ __forceinline__ bool mbar_wait(uint64_t *b, uint32_t parity) {
    if (mbar_try(b, parity)) return true;
    const long long t0 = clock64();
    while (!mbar_try(b, parity))
        if (clock64() - t0 > WAIT_LIMIT) return false;
    return true;
}

__device__ __forceinline__ void tma_2d(void *dst, const CUtensorMap *m, uint64_t *bar, int c0, int c1) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%3, %4}], [%2];"
        ::"r"(su32(dst)), "l"(reinterpret_cast<uint64_t>(m)), "r"(su32(bar)), "r"(c0), "r"(c1)
        : "memory");
}
__device__ __forceinline__ void tma_3d(void *dst, const CUtensorMap *m, uint64_t *bar, int c0, int c1, int c2) {
    asm volatile(
        "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%3, %4, %5}], [%2];"
        ::"r"(su32(dst)), "l"(reinterpret_cast<uint64_t>(m)), "r"(su32(bar)), "r"(c0), "r"(c1), "r"(c2)
        : "memory");
}
__device__ __forceinline__ void tma_4d(void *dst, const CUtensorMap *m, uint64_t *bar, int c0, int c1, int c2,
                                       int c3) {
    asm volatile(
        "cp.async.bulk.tensor.4d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%3, %4, %5, %6}], [%2];"
        ::"r"(su32(dst)), "l"(reinterpret_cast<uint64_t>(m)), "r"(su32(bar)), "r"(c0), "r"(c1), "r"(c2), "r"(c3)
        : "memory");
}

__device__ __forceinline__ void tmem_alloc(uint32_t *dst, uint32_t ncols) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(su32(dst)), "r"(ncols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}
__device__ __forceinline__ void tc_fence_before() {
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

// D[tmem] (+)= A[smem] * B[smem]^T, both K-major, fp32 accumulate
__device__ __forceinline__ void umma(uint32_t d, uint64_t a, uint64_t b, uint32_t idesc, uint32_t acc) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}"
        ::"r"(d), "l"(a), "l"(b), "r"(idesc), "r"(acc)
        : "memory");
}
// arrive on `bar` once every previously issued MMA of this thread has completed
__device__ __forceinline__ void umma_commit(uint64_t *bar) {
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(su32(bar))
                 : "memory");
}

__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&v)[32]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
        "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
        "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
        : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]), "=r"(v[7]),
          "=r"(v[8]), "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]), "=r"(v[13]), "=r"(v[14]), "=r"(v[15]),
          "=r"(v[16]), "=r"(v[17]), "=r"(v[18]), "=r"(v[19]), "=r"(v[20]), "=r"(v[21]), "=r"(v[22]), "=r"(v[23]),
          "=r"(v[24]), "=r"(v[25]), "=r"(v[26]), "=r"(v[27]), "=r"(v[28]), "=r"(v[29]), "=r"(v[30]), "=r"(v[31])
        : "r"(taddr));
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

// shared-memory matrix descriptor: K-major, 128-byte swizzle, rows of 128 B,
// 8-row groups 1024 B apart (SBO); LBO unused for this layout
__device__ __forceinline__ uint64_t sdesc_sw128(uint32_t saddr) {
    uint64_t d = 0;
    d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);
    d |= (uint64_t)1 << 16;
    d |= (uint64_t)(1024 >> 4) << 32;
    d |= (uint64_t)1 << 46;  // descriptor version for tcgen05
    d |= (uint64_t)2 << 61;  // 128-byte swizzle
    return d;
}

// instruction descriptor, kind::f16: fp32 accumulate, A/B fp16 (0) or bf16 (1), K-major
template <typename T>
__device__ __forceinline__ uint32_t idesc_f16(int M, int N) {
    const uint32_t fmt = std::is_same<T, __half>::value ? 0u : 1u;
    return (1u << 4) | (fmt << 7) | (fmt << 10) | ((uint32_t)(N >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
}

template <typename T>
__device__ __forceinline__ uint32_t pack2(float a, float b);
template <>
__device__ __forceinline__ uint32_t pack2<__half>(float a, float b) {
    __half2 h = __floats2half2_rn(a, b);
    return *reinterpret_cast<uint32_t *>(&h);
}
template <>
__device__ __forceinline__ uint32_t pack2<__nv_bfloat16>(float a, float b) {
    __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
    return *reinterpret_cast<uint32_t *>(&h);
}



__device__ __forceinline__ void mbar_arrive(uint64_t *b) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(su32(b)) : "memory");
}
__device__ __forceinline__ void fence_proxy_async_smem() {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
__device__ __forceinline__ void tma_store_2d(const CUtensorMap *m, const void *src, int c0, int c1) {
    asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.tile.bulk_group [%0, {%2, %3}], [%1];"
                 ::"l"(reinterpret_cast<uint64_t>(m)), "r"(su32(src)), "r"(c0), "r"(c1)
                 : "memory");
}
__device__ __forceinline__ void tma_store_4d(const CUtensorMap *m, const void *src, int c0, int c1, int c2, int c3) {
    asm volatile("cp.async.bulk.tensor.4d.global.shared::cta.tile.bulk_group [%0, {%2, %3, %4, %5}], [%1];"
                 ::"l"(reinterpret_cast<uint64_t>(m)), "r"(su32(src)), "r"(c0), "r"(c1), "r"(c2), "r"(c3)
                 : "memory");
}
__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
// at most one store group may still be reading shared memory
__device__ __forceinline__ void bulk_wait_read_0() { asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory"); }
__device__ __forceinline__ void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }

// one unit of work: a 128 x BN tile and the K-range [it0, it1) it accumulates
struct Work {
    int n0;          // first output channel
    int64_t m0;      // plain mode: first pixel row
    int q0, p0, i0;  // implicit mode: box origin (q, p, image)
    int sp, it0, it1;
};

__device__ __forceinline__ Work work_of(const Params &p, int u, int bn, bool implicit) {
    Work w;
    w.sp = u % p.ksplit;
    const int t = u / p.ksplit;
    const int mt = t / p.ntiles, nt = t - mt * p.ntiles;  // A-sharing tiles are adjacent
    w.n0 = nt * bn;
    w.m0 = 0;
    w.q0 = w.p0 = w.i0 = 0;
    if (implicit) {
        int bx = mt;
        const int bq = bx % p.tq;
        bx /= p.tq;
        const int bp = bx % p.tp;
        bx /= p.tp;
        w.q0 = bq * p.BW;
        w.p0 = bp * p.BH;
        w.i0 = bx * p.BNI;
    } else {
        w.m0 = (int64_t)mt * BM;
    }
    w.it0 = (int)((int64_t)w.sp * p.kiters / p.ksplit);
    w.it1 = (int)((int64_t)(w.sp + 1) * p.kiters / p.ksplit);
    return w;
}

// --------------------------------------------------------------------- kernel
template <typename T, int BN, int STAGES, bool IMPLICIT>
__global__ void __launch_bounds__(THREADS, 1)
    conv_tc_kernel(const __grid_constant__ CUtensorMap mA0, const __grid_constant__ CUtensorMap mA1,
                   const __grid_constant__ CUtensorMap mA2, const __grid_constant__ CUtensorMap mA3,
                   const __grid_constant__ CUtensorMap mB, const __grid_constant__ CUtensorMap mY,
                   const Params p) {
    constexpr uint32_t A_BYTES = BM * BK * 2;
    constexpr uint32_t B_BYTES = BN * BK * 2;
    constexpr uint32_t STAGE_BYTES = A_BYTES + B_BYTES;
    constexpr uint32_t TMEM_COLS = 2 * BN;  // two accumulators
    extern __shared__ uint8_t smem_raw[];
    __shared__ __align__(8) uint64_t full_bar[STAGES];
    __shared__ __align__(8) uint64_t empty_bar[STAGES];
    __shared__ __align__(8) uint64_t accf_bar[2];  // MMA -> epilogue: accumulator ready
    __shared__ __align__(8) uint64_t acce_bar[2];  // epilogue -> MMA: accumulator drained
    __shared__ uint32_t tmem_sh;
    __shared__ volatile int abort_sh;
    __shared__ int issued_sh, consumed_sh;

    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t *stg = smem + STAGES * STAGE_BYTES;  // epilogue staging: 8 warps x 2 buffers, 1024-B aligned
    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    const int total = p.mtiles * p.ntiles * p.ksplit;

    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(&full_bar[s], 1);
            mbar_init(&empty_bar[s], 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(&accf_bar[b], 1);
            mbar_init(&acce_bar[b], EPI_WARPS / 2);  // one arrival per warp of the group draining it
        }
        abort_sh = 0;
        issued_sh = 0;
        consumed_sh = 0;
        fence_mbar_init();
    }
    if (warp == 0) tmem_alloc(&tmem_sh, TMEM_COLS);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_sh;

    if (warp == 0) {
        if (lane == 0) {  // ---------------- TMA producer
            int g = 0;
            bool stop = false;
            for (int u = blockIdx.x; u < total && !stop; u += gridDim.x) {
                const Work w = work_of(p, u, BN, IMPLICIT);
                for (int it = w.it0; it < w.it1; ++it, ++g) {
                    const int s = g % STAGES;
                    const uint32_t ph = (uint32_t)(g / STAGES) & 1u;
                    if (!mbar_wait(&empty_bar[s], ph ^ 1u)) {
                        atomicOr(p.err, ERR_TMA_WAIT);
                        abort_sh = 1;
                    }
                    if (abort_sh) {
                        stop = true;
                        break;
                    }
                    uint8_t *sa = smem + s * STAGE_BYTES;
                    uint8_t *sb = sa + A_BYTES;
                    const int tap = it / p.cblocks, cb = it - tap * p.cblocks;
                    const int r = tap / p.S, ss = tap - r * p.S;
                    const int c0 = cb * BK;
                    mbar_expect_tx(&full_bar[s], STAGE_BYTES);
                    if (IMPLICIT) {
                        const int oh = r * p.dh - p.ph, ow = ss * p.dw - p.pw;
                        if (p.stride == 1) {
                            tma_4d(sa, &mA0, &full_bar[s], c0, w.q0 + ow, w.p0 + oh, w.i0);
                        } else {  // stride 2: even/odd sub-lattice maps
                            const int bh = oh & 1, bw = ow & 1;
                            const int ah = (oh - bh) / 2, aw = (ow - bw) / 2;
                            const CUtensorMap *m = bh ? (bw ? &mA3 : &mA2) : (bw ? &mA1 : &mA0);
                            tma_4d(sa, m, &full_bar[s], c0, w.q0 + aw, w.p0 + ah, w.i0);
                        }
                    } else {
                        tma_2d(sa, &mA0, &full_bar[s], c0, (int)w.m0);
                    }
                    tma_3d(sb, &mB, &full_bar[s], c0, tap, w.n0);
                }
            }
            issued_sh = g;
        }
    } else if (warp == 1) {
        if (lane == 0) {  // ---------------- MMA issuer
            const uint32_t idesc = idesc_f16<T>(BM, BN);
            int g = 0, lt = 0;
            bool stop = false;
            for (int u = blockIdx.x; u < total && !stop; u += gridDim.x, ++lt) {
                const Work w = work_of(p, u, BN, IMPLICIT);
                const int b = lt & 1;
                const uint32_t aph = (uint32_t)(lt >> 1) & 1u;
                if (!mbar_wait(&acce_bar[b], aph ^ 1u)) {
                    atomicOr(p.err, ERR_EPI_WAIT);
                    abort_sh = 1;
                    break;
                }
                tc_fence_after();
                const uint32_t d = tmem + (uint32_t)(b * BN);
                for (int it = w.it0; it < w.it1; ++it, ++g) {
                    const int s = g % STAGES;
                    const uint32_t ph = (uint32_t)(g / STAGES) & 1u;
                    if (!mbar_wait(&full_bar[s], ph)) {
                        atomicOr(p.err, ERR_MMA_WAIT);
                        abort_sh = 1;
                        stop = true;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t sa = su32(smem + s * STAGE_BYTES), sb = sa + A_BYTES;
#pragma unroll
                    for (int k = 0; k < BK / 16; ++k)
                        umma(d, sdesc_sw128(sa + k * 32), sdesc_sw128(sb + k * 32), idesc,
                             (it > w.it0 || k > 0) ? 1u : 0u);
                    umma_commit(&empty_bar[s]);  // frees the stage once these MMAs have read it
                }
                if (!stop) umma_commit(&accf_bar[b]);
            }
            consumed_sh = g;
        }
    } else {  // ---------------- epilogue: warps 2..9
        // two groups of four warps; group eg drains accumulator eg, i.e. the
        // work units with lt % 2 == eg; within a group warp w reads TMEM lanes
        // 32*(w%4) .. +31 (tile rows) and walks all channels in 64-wide chunks
        const int eg = (warp - 2) >> 2;
        const int g4 = warp & 3;
        const int row = g4 * 32 + lane;
        uint8_t *buf = stg + (warp - 2) * STG_BYTES;  // one 32 x 64 staging block per warp
        const int r0 = g4 * 32;
        const int wq0 = IMPLICIT ? r0 % p.BW : 0;
        const int hp0 = IMPLICIT ? (r0 / p.BW) % p.BH : 0;
        const int ni0 = IMPLICIT ? r0 / (p.BW * p.BH) : 0;
        constexpr int NCH = BN / 64 > 0 ? BN / 64 : 1;  // 64-channel chunks per tile
        int lt = eg;
        for (int u = blockIdx.x + eg * gridDim.x; u < total; u += 2 * gridDim.x, lt += 2) {
            const uint32_t aph = (uint32_t)(lt >> 1) & 1u;
            const Work w = work_of(p, u, BN, IMPLICIT);
            // bias of channels chunk + lane and chunk + 32 + lane, loaded before
            // the accumulator wait so the latency is hidden
            float bias_r[NCH][2];
#pragma unroll
            for (int i = 0; i < NCH; ++i)
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    const int kb = w.n0 + 64 * i + 32 * h + lane;
                    bias_r[i][h] = (p.ksplit == 1 && kb < p.K) ? __ldg(p.bias + kb) : 0.f;
                }
            if (!mbar_wait(&accf_bar[eg], aph)) {
                if (lane == 0) atomicOr(p.err, ERR_ACC_WAIT);
                abort_sh = 1;
                break;
            }
            tc_fence_after();
            bool valid;
            int64_t pix;
            if (IMPLICIT) {
                const int wq = row % p.BW, hp = (row / p.BW) % p.BH, ni = row / (p.BW * p.BH);
                const int q = w.q0 + wq, pp = w.p0 + hp, n = w.i0 + ni;
                valid = q < p.Q && pp < p.P && n < p.N;
                pix = ((int64_t)n * p.P + pp) * p.Q + q;
            } else {
                pix = w.m0 + row;
                valid = pix < p.Mout;
            }
#pragma unroll
            for (int ci = 0; ci < NCH; ++ci) {
                const int k0 = w.n0 + 64 * ci;
                if (k0 >= p.K) break;
                const uint32_t taddr = tmem + ((uint32_t)(g4 * 32) << 16) + (uint32_t)(eg * BN + 64 * ci);
                if (p.ksplit == 1) {
                    // bias + activation -> 16-bit, staged with the 128-byte swizzle
                    // (row = lane, 16-byte chunk j at j ^ (row & 7)), then one TMA
                    // tensor store of the warp's 32 x 64 block, clipped at the edges
                    uint32_t wv[32];
#pragma unroll
                    for (int h = 0; h < 2; ++h) {
                        uint32_t v[32];
                        __syncwarp();
                        tmem_ld32(taddr + 32 * h, v);
#pragma unroll
                        for (int j = 0; j < 16; ++j) {
                            const float f0 = act_apply(
                                __uint_as_float(v[2 * j]) + __shfl_sync(0xffffffffu, bias_r[ci][h], 2 * j), p.act);
                            const float f1 = act_apply(
                                __uint_as_float(v[2 * j + 1]) + __shfl_sync(0xffffffffu, bias_r[ci][h], 2 * j + 1),
                                p.act);
                            wv[16 * h + j] = pack2<T>(f0, f1);
                        }
                    }
                    if (lane == 0) bulk_wait_read_0();  // the previous store has read the staging block
                    __syncwarp();
#pragma unroll
                    for (int j = 0; j < 8; ++j)
                        *reinterpret_cast<uint4 *>(buf + lane * 128 + ((j ^ (lane & 7)) << 4)) =
                            make_uint4(wv[4 * j], wv[4 * j + 1], wv[4 * j + 2], wv[4 * j + 3]);
                    fence_proxy_async_smem();
                    __syncwarp();
                    if (lane == 0) {
                        if (IMPLICIT)
                            tma_store_4d(&mY, buf, k0, w.q0 + wq0, w.p0 + hp0, w.i0 + ni0);
                        else
                            tma_store_2d(&mY, buf, k0, (int)(w.m0 + r0));
                        bulk_commit();
                    }
                } else {
#pragma unroll
                    for (int h = 0; h < 2; ++h) {
                        uint32_t v[32];
                        __syncwarp();
                        tmem_ld32(taddr + 32 * h, v);
                        const int kh = k0 + 32 * h;
                        if (!valid || kh >= p.K) continue;
                        float *dst = p.part + ((int64_t)w.sp * p.Mout + pix) * p.K + kh;
                        if (kh + 32 <= p.K) {
#pragma unroll
                            for (int q4 = 0; q4 < 8; ++q4)
                                reinterpret_cast<uint4 *>(dst)[q4] =
                                    make_uint4(v[4 * q4], v[4 * q4 + 1], v[4 * q4 + 2], v[4 * q4 + 3]);
                        } else {
#pragma unroll
                            for (int j = 0; j < 32; ++j)
                                if (kh + j < p.K) dst[j] = __uint_as_float(v[j]);
                        }
                    }
                }
            }
            // every TMEM read of accumulator eg by this warp is done: hand it back
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&acce_bar[eg]);
        }
        if (lane == 0) bulk_wait_all();  // stores done before the CTA's shared memory is released
        __syncwarp();
    }

    tc_fence_before();
    __syncthreads();
    if (warp == 0) {
        if (abort_sh && lane == 0) {
            // let this CTA's own copies and MMAs land before its memory goes away
            for (int g = consumed_sh; g < issued_sh; ++g)
                mbar_wait(&full_bar[g % STAGES], (uint32_t)(g / STAGES) & 1u);
            if (consumed_sh > 0) {
                const int g = consumed_sh - 1;
                mbar_wait(&empty_bar[g % STAGES], (uint32_t)(g / STAGES) & 1u);
            }
        }
        __syncwarp();
        tc_fence_after();
        tmem_dealloc(tmem, TMEM_COLS);
    }
}

// y[m][k] = act(bias[k] + sum_s part[s][m][k]), four channels per thread
template <typename T>
__global__ void splitk_reduce_kernel(const float *__restrict__ part, const float *__restrict__ bias,
                                     T *__restrict__ y, int64_t M, int K, int ks, int act) {
    const int K4 = K / 4;
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < M * K4;
         i += (int64_t)gridDim.x * blockDim.x) {
        const int64_t m = i / K4;
        const int k = (int)(i - m * K4) * 4;
        float4 acc = make_float4(bias[k], bias[k + 1], bias[k + 2], bias[k + 3]);
        for (int s = 0; s < ks; ++s) {
            const float4 v = *reinterpret_cast<const float4 *>(part + ((int64_t)s * M + m) * K + k);
            acc.x += v.x;
            acc.y += v.y;
            acc.z += v.z;
            acc.w += v.w;
        }
        uint2 o;
        o.x = pack2<T>(act_apply(acc.x, act), act_apply(acc.y, act));
        o.y = pack2<T>(act_apply(acc.z, act), act_apply(acc.w, act));
        *reinterpret_cast<uint2 *>(y + m * K + k) = o;
    }
}

// ------------------------------------------------------------------ host side
typedef CUresult (*EncodeTiled)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *, const cuuint64_t *,
                                const cuuint64_t *, const cuuint32_t *, const cuuint32_t *, CUtensorMapInterleave,
                                CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

static EncodeTiled encoder() {
    static EncodeTiled fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiled>(p);
    });
    return fn;
}

static bool encode(CUtensorMap *m, int dt, int rank, const void *base, const uint64_t *dims,
                   const uint64_t *strides_bytes, const uint32_t *box,
                   CUtensorMapSwizzle sw = CU_TENSOR_MAP_SWIZZLE_128B) {
    EncodeTiled fn = encoder();
    if (!fn) return false;
    cuuint64_t gd[5], gs[4];
    cuuint32_t bx[5], es[5];
    for (int i = 0; i < rank; ++i) {
        gd[i] = dims[i];
        bx[i] = box[i];
        es[i] = 1;
        if (i < rank - 1) gs[i] = strides_bytes[i];
    }
    const CUtensorMapDataType t = dt == SN_F16 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT16 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16;
    return fn(m, t, (cuuint32_t)rank, const_cast<void *>(base), gd, gs, bx, es, CU_TENSOR_MAP_INTERLEAVE_NONE, sw,
              CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}


struct Config {
    bool implicit;
    int BN;
    int BW, BH, BNI;
    int ksplit;
};

constexpr int kSmCount = 152;  // GB300; only used to decide which K splits to offer

// deterministic list of routine-parameter combinations for a layer
static std::vector<Config> configs(const Layer &l, const Shape &in, sn_schema s) {
    std::vector<Config> out;
    const sn_conv_params &c = l.conv;
    if (l.type != SN_L_CONV2 || c.groups != 1) return out;
    if (s.dtype == SN_F32 || s.layout != SN_NHWC) return out;
    if (c.c_in % 8 || c.c_out % 8 || c.c_out > MAX_K) return out;
    if (c.sh != c.sw || (c.sh != 1 && c.sh != 2)) return out;
    if (c.sh == 2 && (in.h % 2 || in.w % 2 || in.h < 2 || in.w < 2)) return out;
    const int K = c.c_out;
    const int kiters = c.kh * c.kw * ((c.c_in + BK - 1) / BK);
    std::vector<int> bns;
    if (K <= 64) bns = {64};
    else if (K <= 128) bns = {64, 128};
    else bns = {64, 128, 256};
    const bool plain = c.kh == 1 && c.kw == 1 && c.sh == 1 && c.ph == 0 && c.pw == 0;
    const int64_t N = l.out.n, P = l.out.h, Q = l.out.w;
    auto push_splits = [&](Config cf, int64_t mtiles) {
        cf.ksplit = 1;
        out.push_back(cf);
        const int64_t tiles = mtiles * ((K + cf.BN - 1) / cf.BN);
        for (int ks : {2, 4})
            if (tiles * ks <= 2 * kSmCount && kiters >= 4 * ks) {
                cf.ksplit = ks;
                out.push_back(cf);
            }
    };
    if (plain) {
        for (int bn : bns) push_splits({false, bn, 0, 0, 0, 1}, (N * P * Q + BM - 1) / BM);
        return out;
    }
    struct G {
        double waste;
        int bw, bh, bni;
    };
    std::vector<G> gs;
    for (int bw = 1; bw <= 128; bw *= 2)
        for (int bh = 1; bw * bh <= 128; bh *= 2) {
            const int bni = 128 / (bw * bh);
            const double cover = (double)((Q + bw - 1) / bw * bw) * ((P + bh - 1) / bh * bh) * ((N + bni - 1) / bni * bni);
            gs.push_back({cover / (double)(N * P * Q), bw, bh, bni});
        }
    std::sort(gs.begin(), gs.end(), [](const G &a, const G &b) {
        if (a.waste != b.waste) return a.waste < b.waste;
        if (a.bw != b.bw) return a.bw > b.bw;
        return a.bh > b.bh;
    });
    const int keep = std::min<int>(2, (int)gs.size());
    for (int gi = 0; gi < keep; ++gi) {
        const G &gg = gs[gi];
        const int64_t mtiles = ((Q + gg.bw - 1) / gg.bw) * ((P + gg.bh - 1) / gg.bh) * ((N + gg.bni - 1) / gg.bni);
        for (int bn : bns) push_splits({true, bn, gg.bw, gg.bh, gg.bni, 1}, mtiles);
    }
    return out;
}

static int num_sms() {
    static int n = 0;
    if (!n) {
        int dev = 0;
        cudaGetDevice(&dev);
        if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) n = 1;
    }
    return n;
}

template <typename T, int BN, bool IMPLICIT>
static cudaError_t launch(const CUtensorMap *mA, const CUtensorMap &mB, const CUtensorMap &mY, const Params &p,
                          cudaStream_t st) {
    constexpr int STAGES = BN == 256 ? 4 : (BN == 128 ? 6 : 8);
    constexpr size_t smem = (size_t)STAGES * (BM * BK * 2 + BN * BK * 2) + EPI_WARPS * STG_BYTES + 1024;
    auto kern = conv_tc_kernel<T, BN, STAGES, IMPLICIT>;
    static bool attr = false;
    if (!attr) {
        cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
        attr = true;
    }
    const int total = p.mtiles * p.ntiles * p.ksplit;
    const unsigned grid = (unsigned)std::min(total, num_sms());
    kern<<<grid, THREADS, smem, st>>>(mA[0], mA[1], mA[2], mA[3], mB, mY, p);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess || p.ksplit == 1) return e;
    const int64_t n4 = p.Mout * (p.K / 4);
    splitk_reduce_kernel<T><<<grid_for(n4, 256), 256, 0, st>>>(p.part, p.bias, static_cast<T *>(p.y), p.Mout, p.K,
                                                               p.ksplit, p.act);
    return cudaGetLastError();
}

}  // namespace tc

int32_t conv_tc_variants(const Layer &l, const Shape &in, sn_schema s) {
    return (int32_t)tc::configs(l, in, s).size();
}

size_t conv_tc_ws(const Layer &l, const Shape &in, sn_schema s, int32_t v) {
    const std::vector<tc::Config> cfgs = tc::configs(l, in, s);
    if (v < 0 || v >= (int)cfgs.size() || cfgs[v].ksplit == 1) return 0;
    return (size_t)cfgs[v].ksplit * l.out.n * l.out.h * l.out.w * l.conv.c_out * sizeof(float);
}

const char *conv_tc_variant_name(int32_t v) {
    static thread_local char buf[32];
    snprintf(buf, sizeof(buf), "cfg%d", v);
    return buf;
}

cudaError_t conv_tc(const LaunchArgs &a) {
    using namespace tc;
    const Layer &l = *a.layer;
    const Shape &in = a.in_shapes[0];
    const std::vector<Config> cfgs = configs(l, in, a.schema);
    if (a.variant < 0 || a.variant >= (int)cfgs.size()) return cudaErrorInvalidValue;
    const Config cf = cfgs[a.variant];
    const sn_conv_params &c = l.conv;
    Params p{};
    p.N = (int)in.n, p.H = (int)in.h, p.W = (int)in.w, p.C = (int)in.c;
    p.K = c.c_out, p.P = (int)l.out.h, p.Q = (int)l.out.w, p.R = c.kh, p.S = c.kw;
    p.stride = c.sh, p.ph = c.ph, p.pw = c.pw, p.dh = c.dh, p.dw = c.dw;
    p.cblocks = (p.C + BK - 1) / BK;
    p.kiters = p.R * p.S * p.cblocks;
    p.ksplit = cf.ksplit;
    p.act = c.act;
    p.bias = a.bias;
    p.y = a.out;
    p.err = device_error_word();
    p.M = in.n * (int64_t)in.h * in.w;
    p.Mout = (int64_t)p.N * p.P * p.Q;
    p.ntiles = (p.K + cf.BN - 1) / cf.BN;
    if (cf.ksplit > 1) {
        const size_t need = (size_t)cf.ksplit * p.Mout * p.K * sizeof(float);
        if (!a.ws || a.ws_bytes < need || (uintptr_t)a.ws % 16) return cudaErrorInvalidValue;
        p.part = static_cast<float *>(a.ws);
    }
    const int dt = a.schema.dtype;
    const uint64_t es = 2;
    CUtensorMap mA[4], mB, mY;
    {  // B: weights [K][R*S][C]
        const uint64_t dims[3] = {(uint64_t)p.C, (uint64_t)(p.R * p.S), (uint64_t)p.K};
        const uint64_t str[2] = {p.C * es, (uint64_t)p.R * p.S * p.C * es};
        const uint32_t box[3] = {BK, 1, (uint32_t)cf.BN};
        if (!encode(&mB, dt, 3, a.wt, dims, str, box)) return cudaErrorInvalidValue;
    }
    if (!cf.implicit) {
        const uint64_t dims[2] = {(uint64_t)p.C, (uint64_t)p.M};
        const uint64_t str[1] = {p.C * es};
        const uint32_t box[2] = {BK, BM};
        if (!encode(&mA[0], dt, 2, a.in[0], dims, str, box)) return cudaErrorInvalidValue;
        mA[1] = mA[2] = mA[3] = mA[0];
        p.mtiles = (int)((p.M + BM - 1) / BM);
        // output [Mout][K], one 32-row x 64-channel box per epilogue-warp chunk
        const uint64_t ydims[2] = {(uint64_t)p.K, (uint64_t)p.Mout};
        const uint64_t ystr[1] = {p.K * es};
        const uint32_t ybox[2] = {64, 32};
        if (!encode(&mY, dt, 2, a.out, ydims, ystr, ybox, CU_TENSOR_MAP_SWIZZLE_128B)) return cudaErrorInvalidValue;
    } else {
        p.BW = cf.BW, p.BH = cf.BH, p.BNI = cf.BNI;
        p.tq = (p.Q + cf.BW - 1) / cf.BW;
        p.tp = (p.P + cf.BH - 1) / cf.BH;
        const int tn = (p.N + cf.BNI - 1) / cf.BNI;
        const uint32_t box[4] = {BK, (uint32_t)cf.BW, (uint32_t)cf.BH, (uint32_t)cf.BNI};
        if (p.stride == 1) {
            const uint64_t dims[4] = {(uint64_t)p.C, (uint64_t)p.W, (uint64_t)p.H, (uint64_t)p.N};
            const uint64_t str[3] = {p.C * es, (uint64_t)p.W * p.C * es, (uint64_t)p.H * p.W * p.C * es};
            if (!encode(&mA[0], dt, 4, a.in[0], dims, str, box)) return cudaErrorInvalidValue;
            mA[1] = mA[2] = mA[3] = mA[0];
        } else {
            for (int bh = 0; bh < 2; ++bh)
                for (int bw = 0; bw < 2; ++bw) {
                    const char *base = static_cast<const char *>(a.in[0]) + ((int64_t)bh * p.W + bw) * p.C * es;
                    const uint64_t dims[4] = {(uint64_t)p.C, (uint64_t)(p.W / 2), (uint64_t)(p.H / 2), (uint64_t)p.N};
                    const uint64_t str[3] = {2 * p.C * es, 2 * (uint64_t)p.W * p.C * es,
                                             (uint64_t)p.H * p.W * p.C * es};
                    if (!encode(&mA[bh * 2 + bw], dt, 4, base, dims, str, box)) return cudaErrorInvalidValue;
                }
        }
        p.mtiles = p.tq * p.tp * tn;
        // output [N][P][Q][K]; an epilogue warp's 32 tile rows form a sub-box
        // of sbw x sbh x sbn pixels (all dimensions powers of two)
        const uint32_t sbw = (uint32_t)std::min(cf.BW, 32);
        const uint32_t sbh = (uint32_t)std::min<int>(cf.BH, 32 / sbw);
        const uint32_t sbn = 32 / (sbw * sbh);
        const uint64_t ydims[4] = {(uint64_t)p.K, (uint64_t)p.Q, (uint64_t)p.P, (uint64_t)p.N};
        const uint64_t ystr[3] = {p.K * es, (uint64_t)p.Q * p.K * es, (uint64_t)p.P * p.Q * p.K * es};
        const uint32_t ybox[4] = {64, sbw, sbh, sbn};
        if (!encode(&mY, dt, 4, a.out, ydims, ystr, ybox, CU_TENSOR_MAP_SWIZZLE_128B)) return cudaErrorInvalidValue;
    }
    if (p.mtiles <= 0 || (int64_t)p.mtiles * p.ntiles * p.ksplit > INT32_MAX) return cudaErrorInvalidValue;
    const bool bf = dt == SN_BF16;
#define SN_TC_LAUNCH(TT, BNV)                                                                     \
    return cf.implicit ? launch<TT, BNV, true>(mA, mB, mY, p, a.stream)                            \
                       : launch<TT, BNV, false>(mA, mB, mY, p, a.stream)
    if (bf) {
        if (cf.BN == 64) SN_TC_LAUNCH(__nv_bfloat16, 64);
        if (cf.BN == 128) SN_TC_LAUNCH(__nv_bfloat16, 128);
        SN_TC_LAUNCH(__nv_bfloat16, 256);
    } else {
        if (cf.BN == 64) SN_TC_LAUNCH(__half, 64);
        if (cf.BN == 128) SN_TC_LAUNCH(__half, 128);
        SN_TC_LAUNCH(__half, 256);
    }
#undef SN_TC_LAUNCH
}

// ---------------------------------------------------------------------------
// childnet routines built on the tensor-core GEMM (section III-D)
// ---------------------------------------------------------------------------

// 1x1 stride-1 conv2 of c_in -> c_out channels: the plain GEMM path of conv_tc
static Layer gemm_layer(int c_in, int c_out, int act, Shape out) {
    Layer g;
    g.type = SN_L_CONV2;
    g.conv = sn_conv_params{c_in, c_out, 1, 1, 1, 1, 0, 0, 1, 1, 1, act};
    g.act = act;
    g.out = out;
    return g;
}

static int64_t im2col_kpad(const Layer &l) {
    return ((int64_t)l.conv.c_in / l.conv.groups * l.conv.kh * l.conv.kw + 63) / 64 * 64;
}

// im2col -> GEMM: for layers the implicit routine cannot take (few input
// channels such as an RGB stem, odd sizes with stride 2)
int32_t conv_im2col_tc_variants(const Layer &l, const Shape &in, sn_schema s) {
    const sn_conv_params &c = l.conv;
    if (l.type != SN_L_CONV2 || c.groups != 1 || s.dtype == SN_F32 || s.layout != SN_NHWC) return 0;
    if (c.c_out % 8) return 0;
    if (!tc::configs(l, in, s).empty()) return 0;  // the implicit routine serves this layer
    const Layer gl = gemm_layer((int)im2col_kpad(l), c.c_out, c.act, l.out);
    const Shape gin{l.out.n, im2col_kpad(l), l.out.h, l.out.w};
    return (int32_t)tc::configs(gl, gin, s).size();
}

static size_t im2col_bytes(const Layer &l, sn_schema s) {
    return ((size_t)l.out.n * l.out.h * l.out.w * im2col_kpad(l) * dtype_size(s.dtype) + 255) & ~size_t(255);
}

size_t conv_im2col_tc_ws(const Layer &l, const Shape &in, sn_schema s, int32_t v) {
    (void)in;
    const Layer gl = gemm_layer((int)im2col_kpad(l), l.conv.c_out, l.conv.act, l.out);
    const Shape gin{l.out.n, im2col_kpad(l), l.out.h, l.out.w};
    return im2col_bytes(l, s) + conv_tc_ws(gl, gin, s, v);
}

// A[m][kk] = x[n, p*sh - ph + r*dh, q*sw - pw + s*dw, c], kk = (r*S + s)*C + c,
// zero outside the image and for kk >= C*R*S; 8 taps (16 bytes) per thread
template <typename T>
__global__ void im2col_nhwc_kernel(const T *__restrict__ x, T *__restrict__ A, ConvDims d, int kpad, int64_t M) {
    const int g8 = kpad / 8;
    const int crs = d.C * d.R * d.S;
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < M * g8;
         i += (int64_t)gridDim.x * blockDim.x) {
        const int64_t m = i / g8;
        const int k0 = (int)(i % g8) * 8;
        const int q = (int)(m % d.Q), p = (int)((m / d.Q) % d.P);
        const int64_t n = m / ((int64_t)d.Q * d.P);
        uint4 o;
        T *po = reinterpret_cast<T *>(&o);
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            const int kk = k0 + e;
            float v = 0.f;
            if (kk < crs) {
                const int c = kk % d.C, rs = kk / d.C, r = rs / d.S, s = rs % d.S;
                const int h = p * d.sh - d.ph + r * d.dh, w = q * d.sw - d.pw + s * d.dw;
                if (h >= 0 && h < d.H && w >= 0 && w < d.W) v = ldf<T>(x + ((n * d.H + h) * d.W + w) * d.C + c);
            }
            po[e] = cvt<T>(v);  // exact: v is a stored value or zero
        }
        reinterpret_cast<uint4 *>(A)[i] = o;
    }
}

// One block per output row (n, p): the R input rows it reads (W x C each,
// zeros outside the image) are staged in shared memory with coalesced loads,
// then the block writes its Q rows of A as 16-byte stores.
template <typename T>
__global__ void __launch_bounds__(256) im2col_rows_kernel(const T *__restrict__ x, T *__restrict__ A, ConvDims d,
                                                          int kpad) {
    extern __shared__ uint8_t im2col_smem[];
    // per tap kk: (offset of (r, w = -pw + s*dw, c) in the staged rows, w) --
    // the divisions by C and S happen once per block, not per element
    int2 *tab = reinterpret_cast<int2 *>(im2col_smem);
    T *rows = reinterpret_cast<T *>(im2col_smem + (size_t)kpad * sizeof(int2));
    const int p = blockIdx.x;
    const int64_t n = blockIdx.y;
    const int WC = d.W * d.C;
    const int crs = d.C * d.R * d.S;
    for (int kk = threadIdx.x; kk < kpad; kk += blockDim.x) {
        if (kk < crs) {
            const int c = kk % d.C, rs = kk / d.C, r = rs / d.S, s = rs - r * d.S;
            const int w = s * d.dw - d.pw;
            tab[kk] = make_int2(r * WC + w * d.C + c, w);
        } else {
            tab[kk] = make_int2(0, -(1 << 29));  // padding tap: always zero
        }
    }
    for (int i = threadIdx.x; i < d.R * WC; i += blockDim.x) {
        const int r = i / WC, rem = i - r * WC;
        const int h = p * d.sh - d.ph + r * d.dh;
        rows[i] = (h >= 0 && h < d.H) ? x[((n * d.H + h) * d.W) * d.C + rem] : cvt<T>(0.f);
    }
    __syncthreads();
    const int g8 = kpad / 8;
    uint4 *out = reinterpret_cast<uint4 *>(A + ((n * d.P + p) * (int64_t)d.Q) * kpad);
    for (int i = threadIdx.x; i < d.Q * g8; i += blockDim.x) {
        const int q = i / g8, k0 = (i - q * g8) * 8;
        const int qs = q * d.sw;
        uint4 o;
        T *po = reinterpret_cast<T *>(&o);
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            const int2 t = tab[k0 + e];
            const int w = t.y + qs;
            po[e] = (w >= 0 && w < d.W) ? rows[t.x + qs * d.C] : cvt<T>(0.f);
        }
        out[i] = o;
    }
}

cudaError_t conv_im2col_tc(const LaunchArgs &a) {
    const Layer &l = *a.layer;
    const ConvDims d = conv_dims(a);
    const int64_t kpad = im2col_kpad(l);
    const int64_t M = (int64_t)d.N * d.P * d.Q;
    const size_t need = im2col_bytes(l, a.schema);
    if (!a.ws || a.ws_bytes < need || (uintptr_t)a.ws % 16) return cudaErrorInvalidValue;
    const size_t rows_bytes = (size_t)kpad * sizeof(int2) + (size_t)d.R * d.W * d.C * dtype_size(a.schema.dtype);
    if (rows_bytes <= 48 * 1024 && d.N <= 65535) {
        SN_DT_SWITCH(a.schema.dtype, T,
                     im2col_rows_kernel<T><<<dim3((unsigned)d.P, (unsigned)d.N), 256, rows_bytes, a.stream>>>(
                         (const T *)a.in[0], (T *)a.ws, d, (int)kpad));
    } else {
        SN_DT_SWITCH(a.schema.dtype, T,
                     im2col_nhwc_kernel<T><<<grid_for(M * (kpad / 8), 256), 256, 0, a.stream>>>(
                         (const T *)a.in[0], (T *)a.ws, d, (int)kpad, M));
    }
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    const Layer gl = gemm_layer((int)kpad, d.K, d.act, l.out);
    LaunchArgs g = a;
    g.layer = &gl;
    g.routine = R_CONV_TC;
    g.in_shapes = {Shape{l.out.n, kpad, l.out.h, l.out.w}};
    g.in[0] = a.ws;
    g.ws = static_cast<uint8_t *>(a.ws) + im2col_bytes(l, a.schema);
    g.ws_bytes = a.ws_bytes - im2col_bytes(l, a.schema);
    return conv_tc(g);
}

// dense = reshape -> 1x1 conv2 -> reshape on an N x C x 1 x 1 blob (identical
// bytes in NCHW and NHWC), run as the tensor-core GEMM
int32_t dense_tc_variants(const Layer &l, const Shape &in, sn_schema s) {
    if (l.type != SN_L_DENSE || s.dtype == SN_F32) return 0;
    const sn_schema nhwc{s.dtype, SN_NHWC};
    const Layer gl = gemm_layer(l.dense_in, l.dense_out, l.act, l.out);
    return (int32_t)tc::configs(gl, in, nhwc).size();
}

size_t dense_tc_ws(const Layer &l, const Shape &in, sn_schema s, int32_t v) {
    const Layer gl = gemm_layer(l.dense_in, l.dense_out, l.act, l.out);
    return conv_tc_ws(gl, in, sn_schema{s.dtype, SN_NHWC}, v);
}

cudaError_t dense_tc(const LaunchArgs &a) {
    const Layer &l = *a.layer;
    const Layer gl = gemm_layer(l.dense_in, l.dense_out, l.act, l.out);
    LaunchArgs g = a;
    g.layer = &gl;
    g.routine = R_CONV_TC;
    g.schema = sn_schema{a.schema.dtype, SN_NHWC};
    return conv_tc(g);
}

}  // namespace k
}  // namespace sn
