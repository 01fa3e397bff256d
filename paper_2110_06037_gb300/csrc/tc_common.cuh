// Shared pieces of the tcgen05 convolution kernels: launch parameters,
// inline-PTX wrappers (mbarrier, TMA, TMEM, MMA) and the work-unit map.
#pragma once
#include <cuda.h>

#include <type_traits>

#include "kern_common.cuh"

namespace sn {
namespace k {
namespace tc {

constexpr int BM = 128;
constexpr int BK = 64;
// 12 warps: producer 0, MMA, 8 epilogue, producers 1-2.  Three warps per SM
// sub-partition leave the epilogue up to 168 registers a thread.
constexpr int THREADS = 384;
// TMA producer threads for a ring of `stages` stages: one issuing thread
// walks the stages s with s % n == its index, so n must divide the depth.
// Two for an even depth; the third producer warp then waits on the MMA
// issuer's barriers for it (see waits_for_mma).
constexpr int producers_for(int stages) { return stages % 2 == 0 ? 2 : 3; }
// A shared-memory access by the MMA-issuing thread (an mbarrier wait included)
// queues behind the tensor core's operand reads and costs ~250 cycles, as much
// as four MMAs: with an even ring depth, warp 11 waits on the stage-full and
// accumulator-drained barriers instead and hands each result to the MMA warp
// through a hardware named barrier (bar.red.or: both warps pass it together,
// and the OR of their predicates tells both whether to stop).
constexpr bool waits_for_mma(int stages) { return producers_for(stages) == 2; }
constexpr uint32_t BAR_MMA = 1;  // named barrier of the MMA warp and its waiter (0 is __syncthreads)
// pipeline depth: as many stages of KB 64-channel blocks as fit beside the
// epilogue staging (227 KB - 32 KB staging - 1 KB alignment slack)
constexpr int stages_for(int bn, int g, int kb, int ms = 1, int extra = 0) {
    return (198656 - extra) / (kb * (16384 * ms + bn / g * 128)) < 8
               ? (198656 - extra) / (kb * (16384 * ms + bn / g * 128))
               : 8;
}
// halo tiles (3x3, stride 1): 8 x 16 output pixels of one image; a stage
// holds the 10 x 16 input pixels one tap row reads (all three column taps)
constexpr int HALO_BW = 8, HALO_BH = 16, HALO_W = HALO_BW + 2, HALO_ROWS = HALO_W * HALO_BH;
constexpr int halo_stages(int bn) {
    return 198656 / (HALO_ROWS * 128 + 3 * bn * 128) < 8 ? 198656 / (HALO_ROWS * 128 + 3 * bn * 128) : 8;
}
// weight-stationary tiles: the layer's whole B (K steps x BN rows x 128 B) is
// loaded once per CTA and stays in shared memory beside this many A stages
constexpr int BST_STAGES = 4;
constexpr int EPI_WARPS = 8;
constexpr int MAX_K = 65536;
constexpr uint32_t STG_BYTES = 32 * 64 * 2;      // one epilogue staging block: 32 rows x 64 channels
constexpr uint32_t XBLK_BYTES = 32 * 64 * 4;     // cluster K split: one warp's fp32 partial block
constexpr long long WAIT_LIMIT = 4000000000LL;  // SM cycles (~2 s)
enum : int { ERR_TMA_WAIT = 0x10, ERR_MMA_WAIT = 0x20, ERR_ACC_WAIT = 0x40, ERR_EPI_WAIT = 0x80 };

struct Params {
    int32_t N, H, W, C, K, P, Q, R, S;
    int32_t stride, ph, pw, dh, dw;
    int32_t cblocks, kiters, ksplit;  // 64-channel blocks; K steps (of KB blocks) per tile; K split
    int32_t BW, BH, BNI, tq, tp;   // pixel-tile geometry (implicit mode)
    int32_t mtiles, ntiles;
    FastDiv fd_ksplit, fd_ntiles, fd_tq, fd_tp, fd_spt, fd_S;  // spt: K steps per filter tap
    int32_t lbw, lbwh;             // log2 BW, log2 (BW * BH): the tile geometry is powers of two
    int64_t M;                     // plain mode: input rows (= output pixels)
    int64_t Mout;                  // output pixels N * P * Q
    int32_t act;
    int32_t bst_bytes;             // weight-stationary: bytes of the resident B (0 otherwise)
    const float *bias;             // fp32 [K], zero-padded to a multiple of 256 entries
    void *y;                       // output, NHWC, fp16/bf16
    const void *res;               // residual added before the activation (output's layout), or null
    float *part;                   // K split: fp32 partial sums [ksplit][Mout][K]
    int *err;                      // the library's device error word
    long long wait_limit;          // SM cycles a pipeline wait may take before the kernel gives up
    int32_t y_nchw;                // 1: the output is written in NCHW (same dtype)
    // stream-K (one-CTA tiles): the tiles' K steps laid end to end, sk_steps =
    // mtiles * ntiles * kiters in all, CTA c taking [c sk_len, (c + 1) sk_len)
    int32_t sk_len, sk_steps;      // 0: off
    int *sk_count;                 // per (tile, epilogue warp): parts arrived; zero between launches
    float *sk_part;                // fp32 partial tiles, two slots of 128 x BN per CTA
    // the layer's weights (not written by the previous kernel): each CTA asks
    // L2 for its slice of them before the dependency wait
    const void *wt;
    int64_t wt_bytes;
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
// non-suspending test of the phase with the given parity
__device__ __forceinline__ bool mbar_test(uint64_t *b, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(su32(b)), "r"(parity)
        : "memory");
    return ok != 0;
}
// bounded wait for the phase with the given parity (limit in SM cycles);
// false on expiry.  try_wait may suspend the thread inside the hardware for
// a while, so a limit shorter than the default polls with test_wait instead,
// which lets even a limit of a few cycles be honoured.
__device__ __forceinline__ bool mbar_wait(uint64_t *b, uint32_t parity, long long limit = WAIT_LIMIT) {
    if (limit < WAIT_LIMIT) {
        if (mbar_test(b, parity)) return true;
        const long long t0 = clock64();
        while (!mbar_test(b, parity))
            if (clock64() - t0 > limit) return false;
        return true;
    }
    if (mbar_try(b, parity)) return true;
    const long long t0 = clock64();
    while (!mbar_try(b, parity))
        if (clock64() - t0 > limit) return false;
    return true;
}

// TMA tiled loads into this CTA's shared memory at `dst`, completing on the
// mbarrier at shared::cluster address `bar`.  G = 2 (CTA pair): the barrier
// may live in the peer CTA (the pair's leader counts both CTAs' bytes).
#define SN_TMA_LOAD(DIM, COORDS, ...)                                                                      \
    if constexpr (G == 2)                                                                                 \
        asm volatile("cp.async.bulk.tensor." DIM                                                         \
                     ".shared::cluster.global.tile.mbarrier::complete_tx::bytes.cta_group::2 [%0], [%1, " \
                     COORDS "], [%2];" ::"r"(dst), "l"(reinterpret_cast<uint64_t>(m)), "r"(bar), __VA_ARGS__ \
                     : "memory");                                                                         \
    else                                                                                                  \
        asm volatile("cp.async.bulk.tensor." DIM                                                         \
                     ".shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, " COORDS       \
                     "], [%2];" ::"r"(dst), "l"(reinterpret_cast<uint64_t>(m)), "r"(bar), __VA_ARGS__     \
                     : "memory")

template <int G>
__device__ __forceinline__ void tma_2d(uint32_t dst, const CUtensorMap *m, uint32_t bar, int c0, int c1) {
    SN_TMA_LOAD("2d", "{%3, %4}", "r"(c0), "r"(c1));
}
template <int G>
__device__ __forceinline__ void tma_3d(uint32_t dst, const CUtensorMap *m, uint32_t bar, int c0, int c1, int c2) {
    SN_TMA_LOAD("3d", "{%3, %4, %5}", "r"(c0), "r"(c1), "r"(c2));
}
template <int G>
__device__ __forceinline__ void tma_4d(uint32_t dst, const CUtensorMap *m, uint32_t bar, int c0, int c1, int c2,
                                       int c3) {
    SN_TMA_LOAD("4d", "{%3, %4, %5, %6}", "r"(c0), "r"(c1), "r"(c2), "r"(c3));
}
template <int G>
__device__ __forceinline__ void tma_5d(uint32_t dst, const CUtensorMap *m, uint32_t bar, int c0, int c1, int c2,
                                       int c3, int c4) {
    SN_TMA_LOAD("5d", "{%3, %4, %5, %6, %7}", "r"(c0), "r"(c1), "r"(c2), "r"(c3), "r"(c4));
}
#undef SN_TMA_LOAD

// bring [p, p + bytes) into L2 (no data is returned; p and bytes multiples of 16)
__device__ __forceinline__ void prefetch_l2(const void *p, uint32_t bytes) {
    asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(reinterpret_cast<uint64_t>(p)), "r"(bytes)
                 : "memory");
}

// TMEM allocation; G = 2 allocates the same columns in both CTAs of the pair
// (one warp of each CTA executes it)
template <int G>
__device__ __forceinline__ void tmem_alloc(uint32_t *dst, uint32_t ncols) {
    if constexpr (G == 2) {
        asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(su32(dst)),
                     "r"(ncols)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
    } else {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(su32(dst)),
                     "r"(ncols)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
}
template <int G>
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
    if constexpr (G == 2)
        asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
    else
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}
__device__ __forceinline__ void tc_fence_before() {
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

// D[tmem] (+)= A[smem] * B[smem]^T, both K-major, fp32 accumulate.  G = 2:
// A's rows 0-127 come from the leader's shared memory and 128-255 from the
// peer's, B's first and second N/2 rows likewise; D rows land in the TMEM of
// the CTA that holds the A rows.
template <int G>
__device__ __forceinline__ void umma(uint32_t d, uint64_t a, uint64_t b, uint32_t idesc, uint32_t acc) {
    if constexpr (G == 2)
        asm volatile(
            "{\n\t.reg .pred p;\n\t"
            "setp.ne.b32 p, %4, 0;\n\t"
            "tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n\t}"
            ::"r"(d), "l"(a), "l"(b), "r"(idesc), "r"(acc)
            : "memory");
    else
        asm volatile(
            "{\n\t.reg .pred p;\n\t"
            "setp.ne.b32 p, %4, 0;\n\t"
            "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}"
            ::"r"(d), "l"(a), "l"(b), "r"(idesc), "r"(acc)
            : "memory");
}
// arrive on `bar` once every previously issued MMA of this thread has
// completed; G = 2 arrives on the barrier at the same offset in both CTAs
template <int G>
__device__ __forceinline__ void umma_commit(uint64_t *bar) {
    if constexpr (G == 2)
        asm volatile(
            "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64 [%0], %1;" ::"r"(
                su32(bar)),
            "h"((uint16_t)3)
            : "memory");
    else
        asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(su32(bar))
                     : "memory");
}

// ----------------------------------------------------------- cluster helpers
__device__ __forceinline__ uint32_t cluster_rank() {
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
    return r;
}
// every thread of both CTAs; orders shared-memory writes before it (release)
// with reads after it (acquire) across the cluster
__device__ __forceinline__ void cluster_sync_all() {
    asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}
// shared::cluster address of the same variable in CTA `rank` of the cluster
__device__ __forceinline__ uint32_t mapa(uint32_t saddr, uint32_t rank) {
    uint32_t r;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(saddr), "r"(rank));
    return r;
}
__device__ __forceinline__ void mbar_arrive_cluster(uint32_t caddr) {
    asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(caddr) : "memory");
}
__device__ __forceinline__ bool mbar_try_cluster(uint64_t *b, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(su32(b)), "r"(parity)
        : "memory");
    return ok != 0;
}
__device__ __forceinline__ bool mbar_test_cluster(uint64_t *b, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.test_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(su32(b)), "r"(parity)
        : "memory");
    return ok != 0;
}
__device__ __forceinline__ bool mbar_wait_cluster(uint64_t *b, uint32_t parity, long long limit = WAIT_LIMIT) {
    if (limit < WAIT_LIMIT) {
        if (mbar_test_cluster(b, parity)) return true;
        const long long t0 = clock64();
        while (!mbar_test_cluster(b, parity))
            if (clock64() - t0 > limit) return false;
        return true;
    }
    if (mbar_try_cluster(b, parity)) return true;
    const long long t0 = clock64();
    while (!mbar_try_cluster(b, parity))
        if (clock64() - t0 > limit) return false;
    return true;
}
__device__ __forceinline__ void st_cluster_v4(uint32_t caddr, uint32_t a, uint32_t b, uint32_t c, uint32_t d) {
    asm volatile("st.shared::cluster.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(caddr), "r"(a), "r"(b), "r"(c), "r"(d)
                 : "memory");
}
__device__ __forceinline__ void st_cluster_u32(uint32_t caddr, uint32_t v) {
    asm volatile("st.shared::cluster.u32 [%0], %1;" ::"r"(caddr), "r"(v) : "memory");
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
// 64 consecutive columns of the warp's 32 lanes, one wait for both halves
__device__ __forceinline__ void tmem_ld64(uint32_t taddr, uint32_t (&v)[64]) {
#define SN_LD32(OFF, B)                                                                                        \
    asm volatile(                                                                                              \
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 "                                                              \
        "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "                              \
        "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"              \
        : "=r"(v[B + 0]), "=r"(v[B + 1]), "=r"(v[B + 2]), "=r"(v[B + 3]), "=r"(v[B + 4]), "=r"(v[B + 5]),      \
          "=r"(v[B + 6]), "=r"(v[B + 7]), "=r"(v[B + 8]), "=r"(v[B + 9]), "=r"(v[B + 10]), "=r"(v[B + 11]),    \
          "=r"(v[B + 12]), "=r"(v[B + 13]), "=r"(v[B + 14]), "=r"(v[B + 15]), "=r"(v[B + 16]), "=r"(v[B + 17]), \
          "=r"(v[B + 18]), "=r"(v[B + 19]), "=r"(v[B + 20]), "=r"(v[B + 21]), "=r"(v[B + 22]), "=r"(v[B + 23]), \
          "=r"(v[B + 24]), "=r"(v[B + 25]), "=r"(v[B + 26]), "=r"(v[B + 27]), "=r"(v[B + 28]), "=r"(v[B + 29]), \
          "=r"(v[B + 30]), "=r"(v[B + 31])                                                                     \
        : "r"(taddr + OFF))
    SN_LD32(0, 0);
    SN_LD32(32, 32);
#undef SN_LD32
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

// the same with 8-row groups sbo bytes apart (a multiple of 128 B): the
// 128-byte swizzle is a function of the absolute shared-memory address, so a
// matrix may start at any row of a box TMA wrote and step by any whole number
// of rows per group
__device__ __forceinline__ uint64_t sdesc_sw128_sbo(uint32_t saddr, uint32_t sbo) {
    uint64_t d = 0;
    d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);
    d |= (uint64_t)1 << 16;
    d |= (uint64_t)((sbo >> 4) & 0x3FFFu) << 32;
    d |= (uint64_t)1 << 46;
    d |= (uint64_t)2 << 61;
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
// the two 16-bit values of a packed pair, widened exactly
template <typename T>
__device__ __forceinline__ float2 unpack2(uint32_t v);
template <>
__device__ __forceinline__ float2 unpack2<__half>(uint32_t v) {
    return __half22float2(*reinterpret_cast<const __half2 *>(&v));
}
template <>
__device__ __forceinline__ float2 unpack2<__nv_bfloat16>(uint32_t v) {
    return __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162 *>(&v));
}



// named barrier `id` over `count` threads (whole warps) that also ORs a
// predicate across them; every participant gets the result
__device__ __forceinline__ bool bar_red_or(uint32_t id, uint32_t count, bool pred) {
    uint32_t r;
    asm volatile(
        "{\n\t.reg .pred pi, po;\n\t"
        "setp.ne.u32 pi, %1, 0;\n\t"
        "bar.red.or.pred po, %2, %3, pi;\n\t"
        "selp.u32 %0, 1, 0, po;\n\t}"
        : "=r"(r)
        : "r"((uint32_t)pred), "r"(id), "r"(count)
        : "memory");
    return r != 0;
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
    int mt;          // pixel tile index (>= mtiles: the idle half of a CTA pair)
    // stream-K: the tile, its number of parts (CTAs that take some of its K
    // steps; 1 = this CTA takes all), the first of those CTAs, and this
    // CTA's partial slot for it (0 when the tile is the first of the CTA's range)
    int sk_t, sk_n, sk_c0, sk_slot;
};

// work unit u: K-split part sp of output-channel tile nt of pixel-tile group
// mg; a group is `ctas` consecutive pixel tiles (one per CTA of a pair), and
// units sharing a group are adjacent so that their A tiles are reused in L2
__device__ __forceinline__ Work work_of(const Params &p, int u, int bn, bool implicit, int ctas, int ms,
                                        int rank = 0) {
    Work w;
    const int t = (int)fdiv((uint32_t)u, p.fd_ksplit);
    w.sp = u - t * p.ksplit;
    const int mg = (int)fdiv((uint32_t)t, p.fd_ntiles), nt = t - mg * p.ntiles;
    const int mt = mg * ctas + rank;
    w.mt = mt;
    w.sk_t = t, w.sk_n = 1, w.sk_c0 = 0, w.sk_slot = 0;
    w.n0 = nt * bn;
    w.m0 = 0;
    w.q0 = w.p0 = w.i0 = 0;
    if (implicit) {
        int bx = mt;
        int nb = (int)fdiv((uint32_t)bx, p.fd_tq);
        const int bq = bx - nb * p.tq;
        bx = nb;
        nb = (int)fdiv((uint32_t)bx, p.fd_tp);
        const int bp = bx - nb * p.tp;
        bx = nb;
        w.q0 = bq * p.BW;
        w.p0 = bp * p.BH;
        w.i0 = bx * p.BNI;
    } else {
        w.m0 = (int64_t)mt * BM * ms;
    }
    w.it0 = (int)fdiv((uint32_t)(w.sp * p.kiters), p.fd_ksplit);
    w.it1 = (int)fdiv((uint32_t)((w.sp + 1) * p.kiters), p.fd_ksplit);
    return w;
}

// host: encode a tiled tensor map over an f16/bf16 tensor (dims innermost
// first, byte strides of the outer dims); false if the driver refuses it
bool tma_encode(CUtensorMap *m, int dt, int rank, const void *base, const uint64_t *dims,
                const uint64_t *strides_bytes, const uint32_t *box, CUtensorMapSwizzle sw);

}  // namespace tc
}  // namespace k
}  // namespace sn
