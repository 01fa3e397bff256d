// Convolution as implicit GEMM on the 5th-generation tensor cores (tcgen05),
// operands staged by TMA, accumulators in tensor memory (TMEM).
//
// GEMM view (NHWC activations, KRSC weights, fp16/bf16 in, fp32 accumulate):
//   D[m, k] = sum_{r, s, c} A[m, (r, s, c)] * B[k, (r, s, c)]
//   m = output pixel (n, p, q), k = output channel.
// One CTA computes a 128 x BN tile of D.  The K loop runs over filter taps
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
// Warp roles (192 threads): warp 0 = TMA producer (+ TMEM allocation),
// warp 1 = MMA issuer (one thread), warps 2-5 = epilogue (TMEM -> registers
// -> bias + activation -> fp16/bf16 -> global).  Every mbarrier wait is
// bounded; on expiry the kernel records an error code in the library's error
// word, waits (bounded) for its own copies and MMAs, frees TMEM and exits.
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
constexpr int THREADS = 192;
constexpr long long WAIT_LIMIT = 4000000000LL;  // SM cycles (~2 s)
enum : int { ERR_TMA_WAIT = 0x10, ERR_MMA_WAIT = 0x20, ERR_ACC_WAIT = 0x40 };

struct Params {
    int32_t N, H, W, C, K, P, Q, R, S;
    int32_t stride, ph, pw, dh, dw;
    int32_t cblocks, kiters;
    int32_t BW, BH, BNI, tq, tp;
    int64_t M;
    int32_t act;
    const float *bias;
    void *y;
    int *err;  // the library's device error word
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

// --------------------------------------------------------------------- kernel
template <typename T, int BN, int STAGES, bool IMPLICIT>
__global__ void __launch_bounds__(THREADS, 1)
    conv_tc_kernel(const __grid_constant__ CUtensorMap mA0, const __grid_constant__ CUtensorMap mA1,
                   const __grid_constant__ CUtensorMap mA2, const __grid_constant__ CUtensorMap mA3,
                   const __grid_constant__ CUtensorMap mB, const Params p) {
    constexpr uint32_t A_BYTES = BM * BK * 2;
    constexpr uint32_t B_BYTES = BN * BK * 2;
    constexpr uint32_t STAGE_BYTES = A_BYTES + B_BYTES;
    constexpr uint32_t TMEM_COLS = BN;
    extern __shared__ uint8_t smem_raw[];
    __shared__ __align__(8) uint64_t full_bar[STAGES];
    __shared__ __align__(8) uint64_t empty_bar[STAGES];
    __shared__ __align__(8) uint64_t acc_bar;
    __shared__ uint32_t tmem_sh;
    __shared__ volatile int abort_sh;
    __shared__ int issued_sh, consumed_sh;
    __shared__ float bias_sh[BN];

    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    const int n0 = blockIdx.y * BN;
    int64_t m0 = 0;
    int q0 = 0, p0 = 0, i0 = 0;
    if (IMPLICIT) {
        int bx = blockIdx.x;
        const int bq = bx % p.tq;
        bx /= p.tq;
        const int bp = bx % p.tp;
        bx /= p.tp;
        q0 = bq * p.BW;
        p0 = bp * p.BH;
        i0 = bx * p.BNI;
    } else {
        m0 = (int64_t)blockIdx.x * BM;
    }

    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(&full_bar[s], 1);
            mbar_init(&empty_bar[s], 1);
        }
        mbar_init(&acc_bar, 1);
        abort_sh = 0;
        issued_sh = 0;
        consumed_sh = 0;
        fence_mbar_init();
    }
    if (warp == 0) tmem_alloc(&tmem_sh, TMEM_COLS);
    for (int j = threadIdx.x; j < BN; j += THREADS) bias_sh[j] = (n0 + j < p.K) ? p.bias[n0 + j] : 0.f;
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_sh;

    if (warp == 0) {
        if (lane == 0) {  // ---------------- TMA producer
            int it = 0;
            for (; it < p.kiters; ++it) {
                const int s = it % STAGES;
                const uint32_t ph = (uint32_t)(it / STAGES) & 1u;
                if (!mbar_wait(&empty_bar[s], ph ^ 1u)) {
                    atomicOr(p.err, ERR_TMA_WAIT);
                    abort_sh = 1;
                    break;
                }
                if (abort_sh) break;
                uint8_t *sa = smem + s * STAGE_BYTES;
                uint8_t *sb = sa + A_BYTES;
                const int tap = it / p.cblocks, cb = it - tap * p.cblocks;
                const int r = tap / p.S, ss = tap - r * p.S;
                const int c0 = cb * BK;
                mbar_expect_tx(&full_bar[s], STAGE_BYTES);
                if (IMPLICIT) {
                    const int oh = r * p.dh - p.ph, ow = ss * p.dw - p.pw;
                    if (p.stride == 1) {
                        tma_4d(sa, &mA0, &full_bar[s], c0, q0 + ow, p0 + oh, i0);
                    } else {  // stride 2: even/odd sub-lattice maps
                        const int bh = oh & 1, bw = ow & 1;
                        const int ah = (oh - bh) / 2, aw = (ow - bw) / 2;
                        const CUtensorMap *m = bh ? (bw ? &mA3 : &mA2) : (bw ? &mA1 : &mA0);
                        tma_4d(sa, m, &full_bar[s], c0, q0 + aw, p0 + ah, i0);
                    }
                } else {
                    tma_2d(sa, &mA0, &full_bar[s], c0, (int)m0);
                }
                tma_3d(sb, &mB, &full_bar[s], c0, tap, n0);
            }
            issued_sh = it;
        }
    } else if (warp == 1) {
        if (lane == 0) {  // ---------------- MMA issuer
            const uint32_t idesc = idesc_f16<T>(BM, BN);
            int it = 0;
            for (; it < p.kiters; ++it) {
                const int s = it % STAGES;
                const uint32_t ph = (uint32_t)(it / STAGES) & 1u;
                if (!mbar_wait(&full_bar[s], ph)) {
                    atomicOr(p.err, ERR_MMA_WAIT);
                    abort_sh = 1;
                    break;
                }
                tc_fence_after();
                const uint32_t sa = su32(smem + s * STAGE_BYTES), sb = sa + A_BYTES;
#pragma unroll
                for (int k = 0; k < BK / 16; ++k)
                    umma(tmem, sdesc_sw128(sa + k * 32), sdesc_sw128(sb + k * 32), idesc, (it | k) ? 1u : 0u);
                umma_commit(&empty_bar[s]);  // frees the stage once these MMAs have read it
            }
            consumed_sh = it;
            if (it == p.kiters) umma_commit(&acc_bar);
        }
    } else {  // ---------------- epilogue: warps 2..5
        const int g = warp & 3;  // TMEM lanes 32g..32g+31 belong to this warp
        const int row = g * 32 + lane;
        const bool ok = mbar_wait(&acc_bar, 0);
        if (!ok) {
            if (lane == 0) atomicOr(p.err, ERR_ACC_WAIT);
            abort_sh = 1;
        } else {
            tc_fence_after();
            bool valid;
            int64_t off;
            if (IMPLICIT) {
                const int wq = row % p.BW, hp = (row / p.BW) % p.BH, ni = row / (p.BW * p.BH);
                const int q = q0 + wq, pp = p0 + hp, n = i0 + ni;
                valid = q < p.Q && pp < p.P && n < p.N;
                off = (((int64_t)n * p.P + pp) * p.Q + q) * p.K;
            } else {
                const int64_t m = m0 + row;
                valid = m < p.M;
                off = m * p.K;
            }
            T *yrow = static_cast<T *>(p.y) + off + n0;
#pragma unroll 1
            for (int c = 0; c < BN; c += 32) {
                uint32_t v[32];
                __syncwarp();
                tmem_ld32(tmem + ((uint32_t)(g * 32) << 16) + (uint32_t)c, v);
                if (valid && n0 + c < p.K) {
                float f[32];
#pragma unroll
                for (int j = 0; j < 32; ++j) f[j] = act_apply(__uint_as_float(v[j]) + bias_sh[c + j], p.act);
                if (n0 + c + 32 <= p.K) {
                    uint4 *dst = reinterpret_cast<uint4 *>(yrow + c);
#pragma unroll
                    for (int q4 = 0; q4 < 4; ++q4) {
                        uint4 w;
                        w.x = pack2<T>(f[8 * q4 + 0], f[8 * q4 + 1]);
                        w.y = pack2<T>(f[8 * q4 + 2], f[8 * q4 + 3]);
                        w.z = pack2<T>(f[8 * q4 + 4], f[8 * q4 + 5]);
                        w.w = pack2<T>(f[8 * q4 + 6], f[8 * q4 + 7]);
                        dst[q4] = w;
                    }
                } else {
                    for (int j = 0; j < 32 && n0 + c + j < p.K; ++j) stf<T>(yrow + c + j, f[j]);
                }
                }
            }
        }
    }

    tc_fence_before();
    __syncthreads();
    if (warp == 0) {
        if (abort_sh && lane == 0) {
            // let this CTA's own copies and MMAs land before its memory goes away
            for (int it = consumed_sh; it < issued_sh; ++it)
                mbar_wait(&full_bar[it % STAGES], (uint32_t)(it / STAGES) & 1u);
            if (consumed_sh > 0) {
                const int it = consumed_sh - 1;
                mbar_wait(&empty_bar[it % STAGES], (uint32_t)(it / STAGES) & 1u);
            }
        }
        __syncwarp();
        tc_fence_after();
        tmem_dealloc(tmem, TMEM_COLS);
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
                   const uint64_t *strides_bytes, const uint32_t *box) {
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
    return fn(m, t, (cuuint32_t)rank, const_cast<void *>(base), gd, gs, bx, es, CU_TENSOR_MAP_INTERLEAVE_NONE,
              CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

struct Config {
    bool implicit;
    int BN;
    int BW, BH, BNI;
};

// deterministic list of routine-parameter combinations for a layer
static std::vector<Config> configs(const Layer &l, const Shape &in, sn_schema s) {
    std::vector<Config> out;
    const sn_conv_params &c = l.conv;
    if (l.type != SN_L_CONV2 || c.groups != 1) return out;
    if (s.dtype == SN_F32 || s.layout != SN_NHWC) return out;
    if (c.c_in % 8 || c.c_out % 8) return out;
    if (c.sh != c.sw || (c.sh != 1 && c.sh != 2)) return out;
    if (c.sh == 2 && (in.h % 2 || in.w % 2 || in.h < 2 || in.w < 2)) return out;
    const int K = c.c_out;
    std::vector<int> bns;
    if (K <= 64) bns = {64};
    else if (K <= 128) bns = {64, 128};
    else bns = {128, 256};
    const bool plain = c.kh == 1 && c.kw == 1 && c.sh == 1 && c.ph == 0 && c.pw == 0;
    if (plain) {
        for (int bn : bns) out.push_back({false, bn, 0, 0, 0});
        return out;
    }
    struct G {
        double waste;
        int bw, bh, bni;
    };
    std::vector<G> gs;
    const int64_t N = l.out.n, P = l.out.h, Q = l.out.w;
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
    for (int gi = 0; gi < keep; ++gi)
        for (int bn : bns) out.push_back({true, bn, gs[gi].bw, gs[gi].bh, gs[gi].bni});
    return out;
}

template <typename T, int BN, bool IMPLICIT>
static cudaError_t launch(const CUtensorMap *mA, const CUtensorMap &mB, const Params &p, dim3 grid,
                          cudaStream_t st) {
    constexpr int STAGES = BN == 256 ? 4 : (BN == 128 ? 6 : 8);
    constexpr size_t smem = (size_t)STAGES * (BM * BK * 2 + BN * BK * 2) + 1024;
    auto kern = conv_tc_kernel<T, BN, STAGES, IMPLICIT>;
    static bool attr = false;
    if (!attr) {
        cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
        attr = true;
    }
    kern<<<grid, THREADS, smem, st>>>(mA[0], mA[1], mA[2], mA[3], mB, p);
    return cudaGetLastError();
}

}  // namespace tc

int32_t conv_tc_variants(const Layer &l, const Shape &in, sn_schema s) {
    return (int32_t)tc::configs(l, in, s).size();
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
    p.act = c.act;
    p.bias = a.bias;
    p.y = a.out;
    p.err = device_error_word();
    p.M = in.n * (int64_t)in.h * in.w;
    const int dt = a.schema.dtype;
    const uint64_t es = 2;
    CUtensorMap mA[4], mB;
    // B: weights [K][R*S][C]
    {
        const uint64_t dims[3] = {(uint64_t)p.C, (uint64_t)(p.R * p.S), (uint64_t)p.K};
        const uint64_t str[2] = {p.C * es, (uint64_t)p.R * p.S * p.C * es};
        const uint32_t box[3] = {BK, 1, (uint32_t)cf.BN};
        if (!encode(&mB, dt, 3, a.wt, dims, str, box)) return cudaErrorInvalidValue;
    }
    dim3 grid;
    grid.y = (unsigned)((p.K + cf.BN - 1) / cf.BN);
    if (!cf.implicit) {
        const uint64_t dims[2] = {(uint64_t)p.C, (uint64_t)p.M};
        const uint64_t str[1] = {p.C * es};
        const uint32_t box[2] = {BK, BM};
        if (!encode(&mA[0], dt, 2, a.in[0], dims, str, box)) return cudaErrorInvalidValue;
        mA[1] = mA[2] = mA[3] = mA[0];
        grid.x = (unsigned)((p.M + BM - 1) / BM);
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
        grid.x = (unsigned)((int64_t)p.tq * p.tp * tn);
    }
    if (grid.y > 65535 || grid.x == 0) return cudaErrorInvalidValue;
    const bool bf = dt == SN_BF16;
#define SN_TC_LAUNCH(TT, BNV)                                                                     \
    return cf.implicit ? launch<TT, BNV, true>(mA, mB, p, grid, a.stream)                          \
                       : launch<TT, BNV, false>(mA, mB, p, grid, a.stream)
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

}  // namespace k
}  // namespace sn
