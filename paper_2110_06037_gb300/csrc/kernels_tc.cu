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
// Warp roles (384 threads): warps 0, 10 and 11 = TMA producers, each filling
// every NPROD-th stage (warp 0 also allocates TMEM), warp 1 = MMA issuer (one
// thread), warps 2-9 = epilogue, all eight draining each accumulator (four
// row quarters x two column halves): TMEM ->
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
#include <string>
#include <type_traits>
#include <vector>

#include "tc_common.cuh"

namespace sn {
namespace k {

namespace tc {

// --------------------------------------------------------------------- kernel
// G = 1: one CTA per tile of 128 pixels x BN channels.
// G = 2: a CTA pair (cluster of two on one TPC) shares a 256 x BN tile: each
// CTA stages its own 128 pixel rows and half of the BN weight rows, the
// leader (cluster rank 0) issues cta_group::2 MMAs that read both CTAs'
// shared memory, and each CTA's TMEM receives its own 128 rows, drained by
// its own epilogue.  Per SM this halves the weight bytes staged and read per
// MMA, the shared-memory bandwidth that limits a one-CTA tile.
template <typename T, int BN, int STAGES, bool IMPLICIT, int G, int KB, bool BST, int MS, int CSK>
__global__ void __launch_bounds__(THREADS, 1)
    conv_tc_kernel(const __grid_constant__ CUtensorMap mA0, const __grid_constant__ CUtensorMap mA1,
                   const __grid_constant__ CUtensorMap mA2, const __grid_constant__ CUtensorMap mA3,
                   const __grid_constant__ CUtensorMap mB, const __grid_constant__ CUtensorMap mY,
                   const __grid_constant__ CUtensorMap mR, const Params p) {
    // a stage holds KB 64-channel blocks of one filter tap; a block of A is
    // 128 rows x 128 B, of B (BN / G) rows x 128 B (this CTA's share)
    // MS = 2: a one-CTA tile of 256 rows, one TMA box of A for both 128-row
    // halves and two MMAs (one per half, one TMEM accumulator each) sharing B
    constexpr uint32_t A_SUB = BM * BK * 2;  // one 128-row half
    constexpr uint32_t A_BLK = MS * A_SUB;
    constexpr uint32_t B_BLK = (BN / G) * BK * 2;
    constexpr uint32_t A_BYTES = KB * A_BLK;
    constexpr uint32_t B_BYTES = KB * B_BLK;
    // BST (weight-stationary, G = 1, one N tile, no K split): a stage holds A
    // only; B of every K step sits after the stages for the whole kernel
    constexpr uint32_t STAGE_BYTES = BST ? A_BYTES : A_BYTES + B_BYTES;
    constexpr uint32_t TMEM_COLS = 2 * MS * BN;  // two accumulators (of MS halves each)
    extern __shared__ uint8_t smem_raw[];
    __shared__ __align__(8) uint64_t full_bar[STAGES];
    __shared__ __align__(8) uint64_t empty_bar[STAGES];
    __shared__ __align__(8) uint64_t accf_bar[2];  // MMA -> epilogue: accumulator ready
    __shared__ __align__(8) uint64_t acce_bar[2];  // epilogue -> MMA: accumulator drained
    __shared__ __align__(8) uint64_t res_bar[EPI_WARPS];  // residual tile landed in a warp's staging block
    __shared__ __align__(8) uint64_t bst_bar;              // weight-stationary B landed
    // CSK = 2 (cluster K split): the two CTAs of a cluster take the two halves
    // of a tile's K steps; CTA 1's epilogue warps write their fp32 partial
    // rows into CTA 0's exchange blocks (distributed shared memory), each
    // block handed to CTA 1 once CTA 0's stages are done with (xfree)
    __shared__ __align__(8) uint64_t xfull_bar[EPI_WARPS];  // CTA 0: a partial block landed
    __shared__ __align__(8) uint64_t xfree_bar[EPI_WARPS];  // CTA 1: CTA 0 has read the block
    __shared__ uint32_t tmem_sh;
    __shared__ volatile int abort_sh;
    __shared__ int issued_sh[4], consumed_sh;

    griddep_launch();
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t *bst = smem + STAGES * STAGE_BYTES;  // weight-stationary B (BST), 1024-B aligned
    uint8_t *stg = bst + (BST ? p.bst_bytes : 0);  // epilogue staging: one block per warp, 1024-B aligned
    // CSK: the exchange blocks (32 x 64 fp32 per warp) reuse the pipeline
    // stages, free once this CTA's only unit has been accumulated (the host
    // launches the split only when every cluster gets one unit)
    uint8_t *xbuf = smem;
    constexpr bool CLUSTER = G == 2 || CSK == 2;
    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    const uint32_t crank = CLUSTER ? cluster_rank() : 0u;
    const uint32_t rank = G == 2 ? crank : 0u;    // rank within a CTA pair (B rows, MMA issue)
    const uint32_t krank = CSK == 2 ? crank : 0u;  // half of the K steps (cluster K split)
    const bool leader = rank == 0;
    const int cid = CLUSTER ? (int)(blockIdx.x / 2) : (int)blockIdx.x;  // pair / cluster (or CTA) index
    const int ncl = CLUSTER ? (int)(gridDim.x / 2) : (int)gridDim.x;
    const int total = (p.mtiles + G - 1) / G * p.ntiles * p.ksplit;
    // this CTA's K steps of a unit: all, or one half under the cluster split
    auto krange = [&](Work &w) {
        if (CSK == 2) {
            const int mid = p.kiters >> 1;
            w.it0 = krank ? mid : 0;
            w.it1 = krank ? p.kiters : mid;
        }
    };
    // stop this CTA's loops, and the peer's
    auto set_abort = [&]() {
        abort_sh = 1;
        if (CLUSTER) st_cluster_u32(mapa(su32((const void *)&abort_sh), crank ^ 1u), 1u);
    };

    if (threadIdx.x == 0) {
        // the tensor maps are kernel parameters, not data of the previous kernel
        const CUtensorMap *maps[7] = {&mA0, &mA1, &mA2, &mA3, &mB, &mY, &mR};
        for (int i = 0; i < 7; ++i) asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(maps[i])) : "memory");
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(&full_bar[s], 1);  // the (leader's) producer of the stage
            mbar_init(&empty_bar[s], 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(&accf_bar[b], 1);
            // one arrival per epilogue warp draining it, in both CTAs of a pair
            mbar_init(&acce_bar[b], G * (BN >= 128 || MS == 2 ? EPI_WARPS : EPI_WARPS / 2));
        }
        for (int i = 0; i < EPI_WARPS; ++i) {
            mbar_init(&res_bar[i], 1);
        }
        mbar_init(&bst_bar, 1);
        for (int i = 0; i < EPI_WARPS; ++i) {
            mbar_init(&xfull_bar[i], 32);  // every lane of the peer warp arrives after its stores
            mbar_init(&xfree_bar[i], 32);
        }
        abort_sh = 0;
        issued_sh[0] = issued_sh[1] = issued_sh[2] = issued_sh[3] = 0;
        consumed_sh = 0;
        fence_mbar_init();
    }
    if (CLUSTER) cluster_sync_all();  // both CTAs' barriers exist before either signals the other
    if (warp == 0) tmem_alloc<G>(&tmem_sh, TMEM_COLS);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_sh;
    // Everything up to each role's griddep_wait() overlaps the previous
    // kernel's tail: the producers wait before their first TMA load, the
    // epilogue warps before their first residual load or store (the MMA warp
    // touches no global memory); kernel parameters, bias and weights are not
    // written by the previous kernel.

    constexpr int NPROD = producers_for(STAGES);
    constexpr bool WAITER = waits_for_mma(STAGES);
    const int prod = warp == 0 ? 0 : (warp >= 10 ? warp - 9 : -1);  // producer index of this warp
    if (WAITER && warp == 11) {
        if (leader) {  // ---------------- the MMA warp's barrier waits (whole warp)
            // the same sequence as the MMA warp: per unit, accumulator b
            // drained, then every K step's stage full; one bar_red_or each
            int lt = 0, s = 0;
            uint32_t par = 0;
            bool stop = false;
            for (int u = cid; u < total && !stop; u += ncl, ++lt) {
                Work w = work_of(p, u, BN, IMPLICIT, G, MS, 0);
                krange(w);
                const int b = lt & 1;
                const uint32_t aph = (uint32_t)(lt >> 1) & 1u;
                bool ok = G == 2 ? mbar_wait_cluster(&acce_bar[b], aph ^ 1u, p.wait_limit) : mbar_wait(&acce_bar[b], aph ^ 1u, p.wait_limit);
                if (!ok) {
                    if (lane == 0) atomicOr(p.err, ERR_EPI_WAIT);
                    set_abort();
                }
                __syncwarp();  // bar.red is warp-aligned: reconverge after the polling loops
                if (bar_red_or(BAR_MMA, 64, !ok || abort_sh)) break;
                for (int it = w.it0; it < w.it1; ++it) {
                    ok = mbar_wait(&full_bar[s], par, p.wait_limit);
                    if (!ok) {
                        if (lane == 0) atomicOr(p.err, ERR_MMA_WAIT);
                        set_abort();
                    }
                    __syncwarp();
                    if (bar_red_or(BAR_MMA, 64, !ok || abort_sh)) {
                        stop = true;
                        break;
                    }
                    if (++s == STAGES) {
                        s = 0;
                        par ^= 1u;
                    }
                }
            }
        }
    } else if (prod >= 0) {
        if (lane == 0 && prod < NPROD) {  // ---------------- TMA producers
            // Producer `prod` fills the stages s with s % NPROD == prod (A and B
            // of every CTA's own rows); several issuing threads, because one
            // thread's issue loop is slower than the MMAs of a stage.  The
            // tap / channel-block position advances incrementally for every
            // K step, with no division per step.
            const int cblocks = p.cblocks, S = p.S, dh = p.dh, dw = p.dw, ph0 = p.ph, pw0 = p.pw;
            const int brow = (int)rank * (BN / G);
            int g = 0, s = prod, issued = 0;
            uint32_t par = 0;
            bool stop = false, waited = false;
            if (BST && prod == 0) {
                // the weights are not written by the previous kernel: loaded
                // before the dependency wait, one box per K step
                mbar_expect_tx(&bst_bar, (uint32_t)p.bst_bytes);
                int tap = 0, cb = 0;
                for (int it = 0; it < p.kiters; ++it) {
                    tma_3d<1>(su32(bst + it * B_BYTES), &mB, su32(&bst_bar), cb * BK, tap, 0);
                    if (++cb == cblocks) {
                        cb = 0;
                        ++tap;
                    }
                }
            }
            for (int u = cid; u < total && !stop; u += ncl) {
                Work w = work_of(p, u, BN, IMPLICIT, G, MS, (int)rank);
                krange(w);
                int tap = (int)fdiv((uint32_t)w.it0, p.fd_spt);
                int cb = (w.it0 - tap * p.fd_spt.d) * KB;
                int r = (int)fdiv((uint32_t)tap, p.fd_S), ss = tap - r * S;
                for (int it = w.it0; it < w.it1; ++it, ++g) {
                    if (g % NPROD == prod) {
                        if (!mbar_wait(&empty_bar[s], par ^ 1u, p.wait_limit)) {
                            atomicOr(p.err, ERR_TMA_WAIT);
                            set_abort();
                        }
                        if (abort_sh) {
                            stop = true;
                            break;
                        }
                        if (!waited) {
                            griddep_wait();
                            waited = true;
                        }
                        const uint32_t sa = su32(smem + s * STAGE_BYTES);
                        // KB = 1: channel coordinate cb * 64 on the innermost axis;
                        // KB > 1: the maps carry a block axis (stride 128 B) and one
                        // box spans KB blocks
                        const int c0 = cb * BK;
                        // the leader's barrier counts the bytes of both CTAs
                        if (leader) mbar_expect_tx(&full_bar[s], G * STAGE_BYTES);  // A only when BST
                        const uint32_t bar = G == 2 ? mapa(su32(&full_bar[s]), 0u) : su32(&full_bar[s]);
                        if (IMPLICIT) {
                            const int oh = r * dh - ph0, ow = ss * dw - pw0;
                            const CUtensorMap *m = &mA0;
                            int qa = w.q0 + ow, pa = w.p0 + oh;
                            if (p.stride != 1) {  // stride 2: even/odd sub-lattice maps
                                const int bh = oh & 1, bw = ow & 1;
                                m = bh ? (bw ? &mA3 : &mA2) : (bw ? &mA1 : &mA0);
                                qa = w.q0 + ((ow - bw) >> 1);
                                pa = w.p0 + ((oh - bh) >> 1);
                            }
                            if (KB == 1)
                                tma_4d<G>(sa, m, bar, c0, qa, pa, w.i0);
                            else
                                tma_5d<G>(sa, m, bar, 0, qa, pa, w.i0, cb);
                        } else {
                            if (KB == 1)
                                tma_2d<G>(sa, &mA0, bar, c0, (int)w.m0);
                            else
                                tma_3d<G>(sa, &mA0, bar, 0, (int)w.m0, cb);
                        }
                        if (!BST) {  // weight-stationary B is already resident
                            if (KB == 1)
                                tma_3d<G>(sa + A_BYTES, &mB, bar, c0, tap, w.n0 + brow);
                            else
                                tma_4d<G>(sa + A_BYTES, &mB, bar, 0, tap, w.n0 + brow, cb);
                        }
                        issued = g + 1;
                        s += NPROD;
                        if (s >= STAGES) {
                            s -= STAGES;
                            par ^= 1u;
                        }
                    }
                    if ((cb += KB) == cblocks) {
                        cb = 0;
                        ++tap;
                        if (++ss == S) {
                            ss = 0;
                            ++r;
                        }
                    }
                }
            }
            issued_sh[prod] = issued;
        }
    } else if (warp == 1 && WAITER) {
        if (leader) {  // ---------------- MMA issuer (lane 0; the whole warp meets the waiter)
            const uint32_t idesc = idesc_f16<T>(BM * G, BN);
            const uint64_t desc0 = sdesc_sw128(su32(smem));  // stage 0, A; offsets add to the address field
            const uint64_t descb = sdesc_sw128(su32(bst));   // weight-stationary B, K step 0
            int g = 0, lt = 0, s = 0;
            bool stop = false;
            if (BST && lane == 0 && !mbar_wait(&bst_bar, 0u, p.wait_limit)) {
                atomicOr(p.err, ERR_MMA_WAIT);
                set_abort();
            }
            __syncwarp();
            for (int u = cid; u < total && !stop; u += ncl, ++lt) {
                Work w = work_of(p, u, BN, IMPLICIT, G, MS, 0);
                krange(w);
                const int b = lt & 1;
                if (bar_red_or(BAR_MMA, 64, false)) break;  // accumulator b drained
                tc_fence_after();
                const uint32_t d = tmem + (uint32_t)(b * MS * BN);
                for (int it = w.it0; it < w.it1; ++it, ++g) {
                    if (bar_red_or(BAR_MMA, 64, false)) {  // stage s full
                        stop = true;
                        break;
                    }
                    tc_fence_after();
                    if (lane == 0) {
                        // descriptors of this stage; a K step of 16 is 32 bytes (2 units)
                        const uint64_t da = desc0 + (uint64_t)((s * STAGE_BYTES) >> 4);
                        const uint64_t db =
                            BST ? descb + (uint64_t)(((uint32_t)it * B_BYTES) >> 4) : da + (A_BYTES >> 4);
#pragma unroll
                        for (int j = 0; j < KB; ++j)
#pragma unroll
                            for (int k = 0; k < BK / 16; ++k)
#pragma unroll
                                for (int m = 0; m < MS; ++m)
                                    umma<G>(d + (uint32_t)(m * BN), da + j * (A_BLK >> 4) + m * (A_SUB >> 4) + 2 * k,
                                            db + j * (B_BLK >> 4) + 2 * k, idesc,
                                            (it > w.it0 || j > 0 || k > 0) ? 1u : 0u);
                        umma_commit<G>(&empty_bar[s]);  // frees the stage (in both CTAs) once read
                    }
                    __syncwarp();
                    if (++s == STAGES) s = 0;
                }
                if (!stop && lane == 0) umma_commit<G>(&accf_bar[b]);
                __syncwarp();
            }
            if (lane == 0) consumed_sh = g;
        }
    } else if (warp == 1) {
        if (lane == 0 && leader) {  // ---------------- MMA issuer (the pair's leader)
            const uint32_t idesc = idesc_f16<T>(BM * G, BN);
            const uint64_t desc0 = sdesc_sw128(su32(smem));  // stage 0, A; offsets add to the address field
            const uint64_t descb = sdesc_sw128(su32(bst));   // weight-stationary B, K step 0
            int g = 0, lt = 0, s = 0;
            uint32_t par = 0;
            bool stop = false;
            if (BST && !mbar_wait(&bst_bar, 0u, p.wait_limit)) {
                atomicOr(p.err, ERR_MMA_WAIT);
                set_abort();
                stop = true;
            }
            for (int u = cid; u < total && !stop; u += ncl, ++lt) {
                Work w = work_of(p, u, BN, IMPLICIT, G, MS, 0);
                krange(w);
                const int b = lt & 1;
                const uint32_t aph = (uint32_t)(lt >> 1) & 1u;
                const bool drained = G == 2 ? mbar_wait_cluster(&acce_bar[b], aph ^ 1u, p.wait_limit) : mbar_wait(&acce_bar[b], aph ^ 1u, p.wait_limit);
                if (!drained) {
                    atomicOr(p.err, ERR_EPI_WAIT);
                    set_abort();
                    break;
                }
                tc_fence_after();
                const uint32_t d = tmem + (uint32_t)(b * MS * BN);
                for (int it = w.it0; it < w.it1; ++it, ++g) {
                    if (!mbar_wait(&full_bar[s], par, p.wait_limit)) {
                        atomicOr(p.err, ERR_MMA_WAIT);
                        set_abort();
                        stop = true;
                        break;
                    }
                    tc_fence_after();
                    // descriptors of this stage; a K step of 16 is 32 bytes (2 units)
                    const uint64_t da = desc0 + (uint64_t)((s * STAGE_BYTES) >> 4);
                    const uint64_t db = BST ? descb + (uint64_t)(((uint32_t)it * B_BYTES) >> 4) : da + (A_BYTES >> 4);
#pragma unroll
                    for (int j = 0; j < KB; ++j)
#pragma unroll
                        for (int k = 0; k < BK / 16; ++k)
#pragma unroll
                            for (int m = 0; m < MS; ++m)
                                umma<G>(d + (uint32_t)(m * BN), da + j * (A_BLK >> 4) + m * (A_SUB >> 4) + 2 * k,
                                        db + j * (B_BLK >> 4) + 2 * k, idesc,
                                        (it > w.it0 || j > 0 || k > 0) ? 1u : 0u);
                    umma_commit<G>(&empty_bar[s]);  // frees the stage (in both CTAs) once read
                    if (++s == STAGES) {
                        s = 0;
                        par ^= 1u;
                    }
                }
                if (!stop) umma_commit<G>(&accf_bar[b]);
            }
            consumed_sh = g;
        }
    } else if (CSK == 2 && krank == 1) {  // ---------------- cluster K split, CTA 1: send partials
        // the same units and chunks as CTA 0's warp of the same index; each
        // lane's row of 64 fp32 goes to the peer's exchange block, 16-byte
        // piece j at slot j ^ (lane & 15) (fewer bank conflicts there)
        constexpr int NCH = BN / 64;
        constexpr int CPH = NCH / 2;
        const int half = (warp - 2) >> 2;
        const int g4 = warp & 3;
        const int cbase = half * CPH;
        const uint32_t peer_row = mapa(su32(xbuf + (warp - 2) * XBLK_BYTES + lane * 256), 0u);
        const uint32_t peer_full = mapa(su32(&xfull_bar[warp - 2]), 0u);
        uint32_t xph = 0;
        int lt = 0;
        bool stop = false;
        for (int u = cid; u < total && !stop; u += ncl, ++lt) {
            const int b = lt & 1;
            const uint32_t aph = (uint32_t)(lt >> 1) & 1u;
            const Work w = work_of(p, u, BN, IMPLICIT, G, MS, 0);
            const bool tile_live = w.mt < p.mtiles;
            if (!mbar_wait(&accf_bar[b], aph, p.wait_limit)) {
                if (lane == 0) atomicOr(p.err, ERR_ACC_WAIT);
                set_abort();
                break;
            }
            tc_fence_after();
#pragma unroll
            for (int cj = 0; cj < CPH; ++cj) {
                const int k0 = w.n0 + 64 * (cbase + cj);
                if (k0 >= p.K || !tile_live) break;
                const uint32_t taddr = tmem + ((uint32_t)(g4 * 32) << 16) + (uint32_t)(b * BN + 64 * (cbase + cj));
                uint32_t v[64];
                __syncwarp();
                tmem_ld64(taddr, v);
                if (!mbar_wait_cluster(&xfree_bar[warp - 2], xph, p.wait_limit)) {
                    if (lane == 0) atomicOr(p.err, ERR_EPI_WAIT);
                    set_abort();
                    stop = true;
                    break;
                }
#pragma unroll
                for (int j = 0; j < 16; ++j)
                    st_cluster_v4(peer_row + ((uint32_t)(j ^ (lane & 15)) << 4), v[4 * j], v[4 * j + 1], v[4 * j + 2],
                                  v[4 * j + 3]);
                mbar_arrive_cluster(peer_full);
                xph ^= 1u;
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&acce_bar[b]);
        }
    } else {  // ---------------- epilogue: warps 2..9
        // Warp w reads TMEM lanes 32*(w%4) .. +31 (tile rows).  Tiles of two or
        // more 64-channel chunks: all eight warps drain every unit, warp w the
        // chunks of column half (w-2)/4.  One-chunk tiles (BN = 64): the two
        // groups of four take alternate units, i.e. one accumulator each.
        // Two-half tiles (MS = 2): group (w-2)/4 drains half (w-2)/4, all chunks.
        const int half = (warp - 2) >> 2;
        const int g4 = warp & 3;
        const int msub = MS == 2 ? half : 0;          // the 128-row half this warp drains
        const int row = msub * BM + g4 * 32 + lane;    // row within the unit's tile
        uint8_t *buf = stg + (warp - 2) * STG_BYTES;  // one 32 x 64 staging block per warp
        const int r0 = msub * BM + g4 * 32;
        const int wq0 = IMPLICIT ? r0 & (p.BW - 1) : 0;
        const int hp0 = IMPLICIT ? (r0 >> p.lbw) & (p.BH - 1) : 0;
        const int ni0 = IMPLICIT ? r0 >> p.lbwh : 0;
        constexpr int NCH = BN / 64 > 0 ? BN / 64 : 1;  // 64-channel chunks per tile
        constexpr int CPH = MS == 2 ? NCH : (NCH >= 2 ? NCH / 2 : 1);  // chunks this warp drains
        constexpr bool ALT = NCH == 1 && MS == 1;        // alternate units between the groups
        const int cbase = (ALT || MS == 2) ? 0 : half * CPH;  // first chunk of this warp
        int lt = ALT ? half : 0;
        uint32_t rpar = 0;  // phase parity of this warp's residual barrier
        int res_issued = 0, res_landed = 0;  // residual loads issued / waited for (warp-uniform)
        uint32_t xph = 0;   // cluster K split: phase parity of this warp's exchange block
        bool waited = false;
        for (int u = cid + (ALT ? half * ncl : 0); u < total; u += (ALT ? 2 : 1) * ncl, lt += ALT ? 2 : 1) {
            const int b = lt & 1;
            const uint32_t aph = (uint32_t)(lt >> 1) & 1u;
            const Work w = work_of(p, u, BN, IMPLICIT, G, MS, (int)rank);
            // bias of this warp's channels (lane j holds channel chunk + 32h + j;
            // the buffer is zero-padded to a multiple of 256 channels), loaded
            // before the accumulator wait so that the latency is hidden
            float bias_r[CPH][2];
#pragma unroll
            for (int cj = 0; cj < CPH; ++cj)
#pragma unroll
                for (int h = 0; h < 2; ++h)
                    bias_r[cj][h] = (p.ksplit == 1 && cbase + cj < NCH)
                                        ? __ldg(p.bias + w.n0 + 64 * (cbase + cj) + 32 * h + lane)
                                        : 0.f;
            bool valid;
            int64_t pix;
            if (IMPLICIT) {
                const int wq = row & (p.BW - 1), hp = (row >> p.lbw) & (p.BH - 1), ni = row >> p.lbwh;
                const int q = w.q0 + wq, pp = w.p0 + hp, n = w.i0 + ni;
                valid = q < p.Q && pp < p.P && n < p.N;
                pix = ((int64_t)n * p.P + pp) * p.Q + q;
            } else {
                pix = w.m0 + row;
                valid = pix < p.Mout;
            }
            // NCHW output (a routine that writes the next layer's layout): this
            // row's first element of output channel k0 sits at
            // ((n K + k0) P + p) Q + q; channel c adds c P Q
            T *ynchw = nullptr;
            if (p.y_nchw && valid) {
                const int64_t PQ = (int64_t)p.P * p.Q;
                const int64_t n_img = pix / PQ;
                ynchw = static_cast<T *>(p.y) + n_img * p.K * PQ + (pix - n_img * PQ);
            }
            // the idle CTA of a pair whose group has one tile stores nothing
            const bool tile_live = w.mt < p.mtiles;
            // residual (fused add): the warp's 32 x 64 block of it is loaded by
            // TMA into the warp's staging block (the box and coordinates of the
            // output store; zero outside the tensor) once the previous store has
            // read that block; the first chunk's load is issued before the
            // accumulator wait, the next one's after the current chunk's store
            if (!waited) {
                griddep_wait();
                waited = true;
            }
            const bool has_res = p.res != nullptr && p.ksplit == 1;
            auto issue_res = [&](int k0) {
                // no new copies once the kernel is stopping
                if (!has_res || !tile_live || k0 >= p.K || __shfl_sync(0xffffffffu, (int)abort_sh, 0)) return;
                ++res_issued;
                if (lane == 0) {
                    bulk_wait_read_0();
                    mbar_expect_tx(&res_bar[warp - 2], STG_BYTES);
                    if (IMPLICIT)
                        tma_4d<1>(su32(buf), &mR, su32(&res_bar[warp - 2]), k0, w.q0 + wq0, w.p0 + hp0, w.i0 + ni0);
                    else
                        tma_2d<1>(su32(buf), &mR, su32(&res_bar[warp - 2]), k0, (int)(w.m0 + r0));
                }
            };
            issue_res(w.n0 + 64 * cbase);
            if (!mbar_wait(&accf_bar[b], aph, p.wait_limit)) {
                if (lane == 0) atomicOr(p.err, ERR_ACC_WAIT);
                set_abort();
                break;
            }
            tc_fence_after();
            // cluster K split: this CTA's MMAs have read their last stage, so
            // the stage memory may now take CTA 1's partials
            if (CSK == 2) mbar_arrive_cluster(mapa(su32(&xfree_bar[warp - 2]), 1u));
#pragma unroll
            for (int cj = 0; cj < CPH; ++cj) {
                const int ci = cbase + cj;
                const int k0 = w.n0 + 64 * ci;
                if (k0 >= p.K || !tile_live) break;
                const uint32_t taddr = tmem + ((uint32_t)(g4 * 32) << 16) + (uint32_t)((b * MS + msub) * BN + 64 * ci);
                if (p.ksplit == 1) {
                    // bias + activation -> 16-bit, staged with the 128-byte swizzle
                    // (row = lane, 16-byte chunk j at j ^ (row & 7)), then one TMA
                    // tensor store of the warp's 32 x 64 block, clipped at the edges
                    // this row's residual: 16-byte piece j of the row at j ^ (row & 7)
                    uint32_t rv[2][16];
#pragma unroll
                    for (int h = 0; h < 2; ++h)
#pragma unroll
                        for (int j = 0; j < 16; ++j) rv[h][j] = 0u;
                    if (!has_res && lane == 0) bulk_wait_read_0();  // the previous store has read the block
                    if (has_res) {
                        const bool landed = mbar_wait(&res_bar[warp - 2], rpar, p.wait_limit);
                        rpar ^= 1u;
                        if (!__all_sync(0xffffffffu, landed)) {
                            if (lane == 0) atomicOr(p.err, ERR_EPI_WAIT);
                            set_abort();
                            break;
                        }
                        ++res_landed;
#pragma unroll
                        for (int j = 0; j < 8; ++j) {
                            const uint4 u = *reinterpret_cast<const uint4 *>(buf + lane * 128 + ((j ^ (lane & 7)) << 4));
                            rv[j >> 2][4 * (j & 3)] = u.x;
                            rv[j >> 2][4 * (j & 3) + 1] = u.y;
                            rv[j >> 2][4 * (j & 3) + 2] = u.z;
                            rv[j >> 2][4 * (j & 3) + 3] = u.w;
                        }
                    }
                    uint32_t v[64];
                    __syncwarp();
                    tmem_ld64(taddr, v);
                    if (CSK == 2) {
                        // add CTA 1's partial of the same rows and channels, then
                        // hand its exchange block back
                        if (!mbar_wait_cluster(&xfull_bar[warp - 2], xph, p.wait_limit)) {
                            if (lane == 0) atomicOr(p.err, ERR_EPI_WAIT);
                            set_abort();
                        }
                        const uint8_t *xr = xbuf + (warp - 2) * XBLK_BYTES + lane * 256;
#pragma unroll
                        for (int j = 0; j < 16; ++j) {
                            const uint4 x = *reinterpret_cast<const uint4 *>(xr + ((j ^ (lane & 15)) << 4));
                            v[4 * j] = __float_as_uint(__uint_as_float(v[4 * j]) + __uint_as_float(x.x));
                            v[4 * j + 1] = __float_as_uint(__uint_as_float(v[4 * j + 1]) + __uint_as_float(x.y));
                            v[4 * j + 2] = __float_as_uint(__uint_as_float(v[4 * j + 2]) + __uint_as_float(x.z));
                            v[4 * j + 3] = __float_as_uint(__uint_as_float(v[4 * j + 3]) + __uint_as_float(x.w));
                        }
                        mbar_arrive_cluster(mapa(su32(&xfree_bar[warp - 2]), 1u));
                        xph ^= 1u;
                    }
                    // every 4 packed pairs (8 channels) go to their 16-byte piece
                    // of the row as soon as they are computed; the activation is
                    // chosen once per chunk, so the unrolled body carries only its own
                    auto stage_rows = [&](auto act) {
#pragma unroll
                        for (int q = 0; q < 8; ++q) {
                            const int h = q >> 2;
                            uint32_t wq[4];
#pragma unroll
                            for (int e = 0; e < 4; ++e) {
                                const int j = 4 * (q & 3) + e;  // pair index within the half
                                const float2 r2 = unpack2<T>(rv[h][j]);
                                const float f0 = act(__uint_as_float(v[32 * h + 2 * j]) +
                                                     __shfl_sync(0xffffffffu, bias_r[cj][h], 2 * j) + r2.x);
                                const float f1 = act(__uint_as_float(v[32 * h + 2 * j + 1]) +
                                                     __shfl_sync(0xffffffffu, bias_r[cj][h], 2 * j + 1) + r2.y);
                                wq[e] = pack2<T>(f0, f1);
                            }
                            *reinterpret_cast<uint4 *>(buf + lane * 128 + ((q ^ (lane & 7)) << 4)) =
                                make_uint4(wq[0], wq[1], wq[2], wq[3]);
                        }
                    };
                    if (p.act == SN_ACT_RELU)
                        stage_rows([](float x) { return fmaxf(x, 0.0f); });
                    else if (p.act == SN_ACT_NONE)
                        stage_rows([](float x) { return x; });
                    else
                        stage_rows([act = p.act](float x) { return act_apply(x, act); });
                    fence_proxy_async_smem();
                    __syncwarp();
                    if (!p.y_nchw) {
                        if (lane == 0) {
                            if (IMPLICIT)
                                tma_store_4d(&mY, buf, k0, w.q0 + wq0, w.p0 + hp0, w.i0 + ni0);
                            else
                                tma_store_2d(&mY, buf, k0, (int)(w.m0 + r0));
                            bulk_commit();
                        }
                    } else if (ynchw) {
                        // NCHW output: each lane reads its own row of the staged
                        // block back, channel by channel (the same rounded values),
                        // and stores it at its pixel of that channel's plane; a
                        // warp's rows are consecutive pixels, so each store
                        // instruction writes neighbouring elements
                        const int64_t pq = (int64_t)p.P * p.Q;
                        T *yc = ynchw + (int64_t)k0 * pq;
                        const int kmax = min(64, p.K - k0);
                        for (int j = 0; j < kmax; ++j) {
                            const T val = *reinterpret_cast<const T *>(buf + lane * 128 + (((j >> 3) ^ (lane & 7)) << 4) +
                                                                       (j & 7) * 2);
                            yc[(int64_t)j * pq] = val;
                        }
                        fence_proxy_async_smem();  // these reads before TMA writes the block again
                    }
                    __syncwarp();
                    if (cj + 1 < CPH) issue_res(k0 + 64);
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
            // every TMEM read of accumulator b by this warp is done: hand it back
            tc_fence_before();
            __syncwarp();
            if (lane == 0) {
                if (G == 2)
                    mbar_arrive_cluster(mapa(su32(&acce_bar[b]), 0u));
                else
                    mbar_arrive(&acce_bar[b]);
            }
        }
        // the last stores have read their staging blocks before the CTA's shared
        // memory is released (their global writes complete with the grid), and
        // after an abort the residual loads still in flight have landed
        if (lane == 0) {
            bulk_wait_read_0();
            const long long t0 = clock64();
            for (int i = res_landed; i < res_issued; ++i)
                while (!mbar_try(&res_bar[warp - 2], (uint32_t)i & 1u) && clock64() - t0 < WAIT_LIMIT) {
                }
        }
        __syncwarp();
    }

    tc_fence_before();
    __syncthreads();
    if (warp == 0) {
        if (abort_sh && lane == 0 && leader) {
            // let the copies and MMAs this CTA waited for land before its
            // memory goes away (one deadline for the whole drain)
            const long long t0 = clock64();
            int issued = 0;
            for (int i = 0; i < 3; ++i) issued = issued_sh[i] > issued ? issued_sh[i] : issued;
            for (int g = consumed_sh; g < issued; ++g)
                while (!mbar_try(&full_bar[g % STAGES], (uint32_t)(g / STAGES) & 1u) && clock64() - t0 < WAIT_LIMIT) {
                }
            if (consumed_sh > 0) {
                const int g = consumed_sh - 1;
                while (!mbar_try(&empty_bar[g % STAGES], (uint32_t)(g / STAGES) & 1u) && clock64() - t0 < WAIT_LIMIT) {
                }
            }
            if (BST)
                while (!mbar_try(&bst_bar, 0u) && clock64() - t0 < WAIT_LIMIT) {
                }
        }
        __syncwarp();
    }
    // neither CTA of a pair leaves while the other may still signal its
    // barriers or the leader's MMAs may still write its TMEM
    if (CLUSTER) cluster_sync_all();
    if (warp == 0) {
        tc_fence_after();
        tmem_dealloc<G>(tmem, TMEM_COLS);
    }
}

// y[m][k] = act(bias[k] + sum_s part[s][m][k] (+ res[m][k])), four channels per thread
template <typename T>
__global__ void splitk_reduce_kernel(const float *__restrict__ part, const float *__restrict__ bias,
                                     const T *__restrict__ res, T *__restrict__ y, int64_t M, int K, int ks,
                                     int act) {
    griddep_launch();
    griddep_wait();
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
        if (res) {
            const uint2 r = *reinterpret_cast<const uint2 *>(res + m * K + k);
            const float2 r0 = unpack2<T>(r.x), r1 = unpack2<T>(r.y);
            acc.x += r0.x;
            acc.y += r0.y;
            acc.z += r1.x;
            acc.w += r1.y;
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

bool tma_encode(CUtensorMap *m, int dt, int rank, const void *base, const uint64_t *dims,
                const uint64_t *strides_bytes, const uint32_t *box, CUtensorMapSwizzle sw) {
    return encode(m, dt, rank, base, dims, strides_bytes, box, sw);
}

struct Config {
    bool implicit;
    int BN;
    int BW, BH, BNI;
    int ksplit;
    int G;   // CTAs per tile: 1, or 2 (CTA pair, 256-pixel tile)
    int KB;  // 64-channel blocks per pipeline stage (one TMA box spans them)
    bool bst = false;  // weight-stationary: B loaded once per CTA (one N tile, G = 1, no split)
    int ms = 1;        // 128-row halves per one-CTA tile (2: 256 x BN, one A box, B shared)
    int csk = 1;       // 2: a cluster of two CTAs splits each tile's K steps, reducing on chip
};

constexpr int kSmCount = 152;  // GB300; only used to decide which K splits to offer

// deterministic list of routine-parameter combinations for a layer
// a_blocks > 0: the space-to-depth formulation (a 1x1 layer of a_blocks x 64
// "channels" over a caller-laid-out A): implicit tiles only, BN = 64, one
// CTA per tile, all a_blocks blocks in one stage
static std::vector<Config> configs(const Layer &l, const Shape &in, sn_schema s, int a_blocks = 0) {
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
    // one-CTA tiles (128 x BN) with K splits of {1, 2, 4}; CTA-pair tiles
    // (256 x BN) with K splits of {1, 2, 3, 4}; a split is offered
    // while the units stay within two waves of the GPU and each part keeps
    // at least four K steps
    auto push_splits = [&](Config cf, int64_t mtiles) {
        const int64_t units = (mtiles + cf.G - 1) / cf.G * ((K + cf.BN - 1) / cf.BN);
        const int64_t slots = 2 * kSmCount / cf.G;
        cf.ksplit = 1;
        out.push_back(cf);
        for (int ks : {2, 3, 4}) {
            if (ks == 3 && cf.G == 1) continue;
            if (units * ks <= slots && kiters >= 4 * ks) {
                cf.ksplit = ks;
                out.push_back(cf);
            }
        }
    };
    auto push_all = [&](Config cf, int64_t mtiles) {
        for (int bn : bns) {
            cf.BN = bn;
            cf.G = 1;
            push_splits(cf, mtiles);
            // two channel blocks per box: a TMA box costs the SM ~400 cycles
            // whatever its size (up to 32 KB), so fewer, larger boxes
            if (bn <= 128 && c.c_in % 128 == 0) {
                cf.KB = 2;
                push_splits(cf, mtiles);
                cf.KB = 1;
            }
        }
        for (int bn : bns) {
            // a pair issues one MMA for both SMs: twice the work per issued
            // instruction, half the B rows staged per SM
            cf.BN = bn;
            cf.G = 2;
            // two channel blocks per stage when the channels split evenly
            cf.KB = c.c_in % 128 == 0 ? 2 : 1;
            push_splits(cf, mtiles);
            cf.KB = 1;
        }
    };
    // weight-stationary variant: the whole B of a one-N-tile layer fits in
    // shared memory beside BST_STAGES A stages and the epilogue staging
    auto push_bst = [&](Config cf) {
        for (int bn : bns)
            if (K <= bn) {
                const int64_t bytes = (int64_t)kiters * bn * BK * 2;
                // 227 KB less the alignment slack, the static barriers and the A stages and staging
                const int64_t room = 227 * 1024 - 2048 - (int64_t)BST_STAGES * BM * BK * 2 - EPI_WARPS * STG_BYTES;
                if (bytes <= room) {
                    cf.BN = bn, cf.G = 1, cf.KB = 1, cf.ksplit = 1, cf.bst = true;
                    out.push_back(cf);
                }
                break;
            }
    };
    // 256-row one-CTA tiles for 64- and 128-channel N tiles: one 32 KB A box
    // per stage for two MMAs that share B (the SM's TMA issue, not bytes, is
    // what small tiles run out of)
    auto push_ms2 = [&](Config cf, int64_t mtiles256) {
        for (int bn : bns)
            if (bn <= 128) {
                cf.BN = bn, cf.G = 1, cf.KB = 1, cf.ms = 2;
                push_splits(cf, mtiles256);
            }
    };
    // cluster K split for layers whose tiles do not fill the GPU: two CTAs per
    // tile, each half the K steps, partials summed through distributed
    // shared memory (no fp32 round trip through HBM, no reduction kernel)
    auto push_csk = [&](Config cf, int64_t mtiles) {
        for (int bn : bns)
            if (bn >= 128 && kiters >= 4 && 2 * mtiles * ((K + bn - 1) / bn) <= kSmCount) {  // one wave of pairs
                cf.BN = bn, cf.G = 1, cf.KB = 1, cf.ksplit = 1, cf.csk = 2;
                out.push_back(cf);
            }
    };
    if (plain && a_blocks == 0) {
        push_all({false, 0, 0, 0, 0, 1, 1, 1}, (N * P * Q + BM - 1) / BM);
        push_bst({false, 0, 0, 0, 0, 1, 1, 1});
        push_ms2({false, 0, 0, 0, 0, 1, 1, 1}, (N * P * Q + 2 * BM - 1) / (2 * BM));
        push_csk({false, 0, 0, 0, 0, 1, 1, 1}, (N * P * Q + BM - 1) / BM);
        return out;
    }
    struct Geo {
        double waste;
        int bw, bh, bni;
    };
    // box geometries of `tm` pixels (powers of two), least padding first
    auto geos = [&](int tm) {
        std::vector<Geo> gs;
        for (int bw = 1; bw <= tm && bw <= 256; bw *= 2)
            for (int bh = 1; bw * bh <= tm && bh <= 256; bh *= 2) {
                const int bni = tm / (bw * bh);
                if (bni > 256) continue;
                const double cover =
                    (double)((Q + bw - 1) / bw * bw) * ((P + bh - 1) / bh * bh) * ((N + bni - 1) / bni * bni);
                gs.push_back({cover / (double)(N * P * Q), bw, bh, bni});
            }
        std::sort(gs.begin(), gs.end(), [](const Geo &a, const Geo &b) {
            if (a.waste != b.waste) return a.waste < b.waste;
            if (a.bw != b.bw) return a.bw > b.bw;
            return a.bh > b.bh;
        });
        if (gs.size() > 2) gs.resize(2);
        return gs;
    };
    auto tiles_of = [&](const Geo &gg) {
        return ((Q + gg.bw - 1) / gg.bw) * ((P + gg.bh - 1) / gg.bh) * ((N + gg.bni - 1) / gg.bni);
    };
    for (const Geo &gg : geos(BM)) {
        if (a_blocks > 0) {
            out.push_back({true, 64, gg.bw, gg.bh, gg.bni, 1, 1, a_blocks});
        } else {
            push_all({true, 0, gg.bw, gg.bh, gg.bni, 1, 1, 1}, tiles_of(gg));
            push_bst({true, 0, gg.bw, gg.bh, gg.bni, 1, 1, 1});
            push_csk({true, 0, gg.bw, gg.bh, gg.bni, 1, 1, 1}, tiles_of(gg));
        }
    }
    if (a_blocks == 0)
        for (const Geo &gg : geos(2 * BM)) push_ms2({true, 0, gg.bw, gg.bh, gg.bni, 1, 1, 1}, tiles_of(gg));
    return out;
}

template <typename T, int BN, bool IMPLICIT, int G, int KB, bool BST = false, int MS = 1, int CSK = 1>
static cudaError_t launch(const CUtensorMap *mA, const CUtensorMap &mB, const CUtensorMap &mY, const CUtensorMap &mR,
                          const Params &p,
                          cudaStream_t st) {
    constexpr int STAGES = BST ? BST_STAGES : stages_for(BN, G, KB, MS);
    static_assert(CSK == 1 || (size_t)STAGES * KB * (BM * BK * 2 + BN * BK * 2) >= EPI_WARPS * XBLK_BYTES,
                  "cluster K split: the exchange blocks live in the stage memory");
    constexpr size_t smem_max = 227 * 1024;
    const size_t smem = BST ? (size_t)STAGES * BM * BK * 2 + p.bst_bytes + EPI_WARPS * STG_BYTES + 1024
                            : (size_t)STAGES * KB * (MS * BM * BK * 2 + (BN / G) * BK * 2) + EPI_WARPS * STG_BYTES + 1024;
    static_assert(BST ||
                      (size_t)STAGES * KB * (MS * BM * BK * 2 + (BN / G) * BK * 2) + EPI_WARPS * STG_BYTES + 1024 <=
                          smem_max,
                  "shared memory per CTA");
    static_assert(!BST || (G == 1 && KB == 1 && MS == 1), "weight-stationary tiles are one-CTA, one block per stage");
    static_assert(MS == 1 || (G == 1 && KB == 1 && !BST && 2 * MS * BN <= 512), "two-half tiles: one CTA, TMEM");
    static_assert(CSK == 1 || (G == 1 && MS == 1 && !BST && BN >= 128), "cluster K split: one-CTA tiles of >= 2 chunks");
    static_assert(STAGES >= 2, "pipeline depth");
    if (smem > smem_max) return cudaErrorInvalidValue;
    auto kern = conv_tc_kernel<T, BN, STAGES, IMPLICIT, G, KB, BST, MS, CSK>;
    constexpr bool CLUSTER = G == 2 || CSK == 2;
    static int max_groups = 0;  // co-resident CTAs (G = 1) or clusters of two (pairs, K split)
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr[2];
    cfg.blockDim = dim3(THREADS);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cfg.attrs = attr;
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;  // see launch_pdl
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.numAttrs = 1;
    if (CLUSTER) {
        attr[1].id = cudaLaunchAttributeClusterDimension;
        attr[1].val.clusterDim.x = 2;
        attr[1].val.clusterDim.y = 1;
        attr[1].val.clusterDim.z = 1;
        cfg.numAttrs = 2;
    }
    static size_t smem_set = 0;  // dynamic shared memory the kernel is currently allowed
    if (smem > smem_set) {
        cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
        smem_set = smem;
    }
    if (!max_groups) {
        cudaError_t e = cudaSuccess;
        if (CLUSTER) {
            cudaLaunchConfig_t q = cfg;  // the cluster shape alone
            q.gridDim = dim3(2);
            q.attrs = attr + 1;
            q.numAttrs = 1;
            int n = 0;
            e = cudaOccupancyMaxActiveClusters(&n, kern, &q);
            if (e != cudaSuccess) return e;
            if (n <= 0) return cudaErrorInvalidConfiguration;
            max_groups = n;
        } else {
            max_groups = num_sms();
        }
    }
    const int total = (p.mtiles + G - 1) / G * p.ntiles * p.ksplit;
    // the cluster K split reuses stage memory for its exchange: one unit per cluster
    if (CSK == 2 && total > max_groups) return cudaErrorNotSupported;
    cfg.gridDim = dim3((unsigned)((CLUSTER ? 2 : 1) * std::min(total, max_groups)));
    cudaError_t e = cudaLaunchKernelEx(&cfg, kern, mA[0], mA[1], mA[2], mA[3], mB, mY, mR, p);
    if (e != cudaSuccess || p.ksplit == 1) return e;
    const int64_t n4 = p.Mout * (p.K / 4);
    launch_pdl(splitk_reduce_kernel<T>, grid_for(n4, 256), 256, 0, st, p.part, p.bias, static_cast<const T *>(p.res),
               static_cast<T *>(p.y), p.Mout, p.K,
                                                               p.ksplit, p.act);
    return cudaGetLastError();
}

}  // namespace tc

int32_t conv_tc_variants(const Layer &l, const Shape &in, sn_schema s) {
    return (int32_t)tc::configs(l, in, s).size();
}

// The tile shape a layer takes inside a chained launch (one CTA per tile of
// 128 pixels, no K split): the selected variant's pixel formulation (plain or
// implicit, and its tile geometry; a 256-row geometry is halved along its
// outermost axis), the widest output-channel tile the layer fills, and two
// channel blocks per stage only for 64-channel tiles (the chain's stage holds
// 48 KB).  False when the variant is not a conv2/igemm_tc one.
bool conv_tc_chain_shape(const Layer &l, const Shape &in, sn_schema s, int32_t v, bool *implicit, int *bn, int *kb,
                         int *bw, int *bh, int *bni) {
    const std::vector<tc::Config> cfgs = tc::configs(l, in, s);
    if (v < 0 || v >= (int)cfgs.size()) return false;
    const tc::Config &cf = cfgs[v];
    *implicit = cf.implicit;
    // the widest output-channel tile the layer fills: a stage costs its TMA
    // boxes (about the same per box whatever its size), so a 256-wide tile
    // does twice the MMA work of a 128-wide one for the same two boxes, and
    // wide tiles mean fewer units to drain and fewer dependency checks
    *bn = l.conv.c_out <= 64 ? 64 : l.conv.c_out <= 128 ? 128 : 256;
    *kb = (*bn == 64 && l.conv.c_in % 128 == 0) ? 2 : 1;
    int w = cf.BW, h = cf.BH, n = cf.BNI;
    if (cf.implicit && cf.ms == 2) {
        if (n >= 2) n /= 2;
        else if (h >= 2) h /= 2;
        else w /= 2;
    }
    *bw = w, *bh = h, *bni = n;
    return !cf.implicit || w * h * n == tc::BM;
}

// the routine parameters of variant v for a layer, spelled out: output-channel
// tile, CTAs per tile, channel blocks per stage, 128-row halves per tile, K
// split, weight-stationary B, cluster K split, and the pixel tiling
std::string conv_tc_config_desc(const Layer &l, const Shape &in, sn_schema s, int32_t v, int32_t a_blocks) {
    const std::vector<tc::Config> cfgs = tc::configs(l, in, s, a_blocks);
    if (v < 0 || v >= (int)cfgs.size()) return "?";
    const tc::Config &c = cfgs[v];
    char b[160];
    if (c.implicit)
        snprintf(b, sizeof(b), "bn=%d cta=%d kb=%d rows=%d ksplit=%d bst=%d csk=%d tile=%dx%dx%d", c.BN, c.G, c.KB,
                 128 * c.ms * c.G, c.ksplit, c.bst ? 1 : 0, c.csk, c.BW, c.BH, c.BNI);
    else
        snprintf(b, sizeof(b), "bn=%d cta=%d kb=%d rows=%d ksplit=%d bst=%d csk=%d plain", c.BN, c.G, c.KB,
                 128 * c.ms * c.G, c.ksplit, c.bst ? 1 : 0, c.csk);
    return b;
}

int32_t conv_tc_ksplit(const Layer &l, const Shape &in, sn_schema s, int32_t v) {
    const std::vector<tc::Config> cfgs = tc::configs(l, in, s);
    return v >= 0 && v < (int)cfgs.size() ? cfgs[v].ksplit : 0;
}

size_t conv_tc_ws(const Layer &l, const Shape &in, sn_schema s, int32_t v, int32_t a_blocks) {
    const std::vector<tc::Config> cfgs = tc::configs(l, in, s, a_blocks);
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
    const std::vector<Config> cfgs = configs(l, in, a.schema, a.a_blocks);
    if (a.variant < 0 || a.variant >= (int)cfgs.size()) return cudaErrorInvalidValue;
    const Config cf = cfgs[a.variant];
    const sn_conv_params &c = l.conv;
    Params p{};
    p.N = (int)in.n, p.H = (int)in.h, p.W = (int)in.w, p.C = (int)in.c;
    p.K = c.c_out, p.P = (int)l.out.h, p.Q = (int)l.out.w, p.R = c.kh, p.S = c.kw;
    p.stride = c.sh, p.ph = c.ph, p.pw = c.pw, p.dh = c.dh, p.dw = c.dw;
    p.cblocks = (p.C + BK - 1) / BK;
    if (p.cblocks % cf.KB) return cudaErrorInvalidValue;
    p.kiters = p.R * p.S * p.cblocks / cf.KB;  // K steps of KB channel blocks
    p.ksplit = cf.ksplit;
    p.act = c.act;
    p.bias = a.bias;
    p.y = a.out;
    p.res = a.in[1];  // residual input of a fused add (null when the layer has one input)
    if (p.res && (uintptr_t)p.res % 16) return cudaErrorInvalidValue;  // read as 16-byte vectors
    p.err = device_error_word();
    p.wait_limit = a.wait_limit > 0 ? a.wait_limit : WAIT_LIMIT;
    // a routine that writes the next layer's layout: the same dtype in NCHW
    // (one CTA's epilogue per tile, so no K split through fp32 partials)
    p.y_nchw = 0;
    if (a.out_schema.dtype >= 0 && !schema_eq(a.out_schema, a.schema)) {
        if (a.out_schema.dtype != a.schema.dtype || a.out_schema.layout != SN_NCHW || cf.ksplit != 1 ||
            a.a_blocks > 0)
            return cudaErrorInvalidValue;
        p.y_nchw = 1;
    }
    p.M = in.n * (int64_t)in.h * in.w;
    p.Mout = (int64_t)p.N * p.P * p.Q;
    p.ntiles = (p.K + cf.BN - 1) / cf.BN;
    if (cf.bst) {
        if (p.ntiles != 1 || cf.ksplit != 1 || cf.G != 1 || cf.KB != 1) return cudaErrorInvalidValue;
        p.bst_bytes = p.kiters * cf.BN * BK * 2;
    }
    if (cf.ksplit > 1) {
        const size_t need = (size_t)cf.ksplit * p.Mout * p.K * sizeof(float);
        if (!a.ws || a.ws_bytes < need || (uintptr_t)a.ws % 16) return cudaErrorInvalidValue;
        p.part = static_cast<float *>(a.ws);
    }
    const int dt = a.schema.dtype;
    const uint64_t es = 2;
    CUtensorMap mA[4], mB, mY, mR;
    // KB > 1 (channels a multiple of 128): every map gets an outermost
    // channel-block axis of stride 128 B over the 64-channel inner axis, so that
    // one box lands KB consecutive 128-B-row blocks in shared memory
    const bool blk = cf.KB > 1;
    const uint64_t CB = (uint64_t)p.cblocks;
    {  // B: weights [K][R*S][C]
        const uint64_t dims[4] = {blk ? 64 : (uint64_t)p.C, (uint64_t)(p.R * p.S), (uint64_t)p.K, CB};
        const uint64_t str[3] = {p.C * es, (uint64_t)p.R * p.S * p.C * es, 128};
        const uint32_t box[4] = {BK, 1, (uint32_t)(cf.BN / cf.G), (uint32_t)cf.KB};  // a CTA's share of the BN rows
        if (!encode(&mB, dt, blk ? 4 : 3, a.wt, dims, str, box)) return cudaErrorInvalidValue;
    }
    if (!cf.implicit) {
        const uint64_t dims[3] = {blk ? 64 : (uint64_t)p.C, (uint64_t)p.M, CB};
        const uint64_t str[2] = {p.C * es, 128};
        const uint32_t box[3] = {BK, (uint32_t)(BM * cf.ms), (uint32_t)cf.KB};
        if (!encode(&mA[0], dt, blk ? 3 : 2, a.in[0], dims, str, box)) return cudaErrorInvalidValue;
        mA[1] = mA[2] = mA[3] = mA[0];
        p.mtiles = (int)((p.M + BM * cf.ms - 1) / (BM * cf.ms));
        // output [Mout][K], one 32-row x 64-channel box per epilogue-warp chunk
        const uint64_t ydims[2] = {(uint64_t)p.K, (uint64_t)p.Mout};
        const uint64_t ystr[1] = {p.K * es};
        const uint32_t ybox[2] = {64, 32};
        if (!encode(&mY, dt, 2, a.out, ydims, ystr, ybox, CU_TENSOR_MAP_SWIZZLE_128B)) return cudaErrorInvalidValue;
        mR = mY;  // the residual has the output's layout
        if (p.res && !encode(&mR, dt, 2, p.res, ydims, ystr, ybox, CU_TENSOR_MAP_SWIZZLE_128B))
            return cudaErrorInvalidValue;
    } else {
        p.BW = cf.BW, p.BH = cf.BH, p.BNI = cf.BNI;
        p.tq = (p.Q + cf.BW - 1) / cf.BW;
        p.tp = (p.P + cf.BH - 1) / cf.BH;
        const int tn = (p.N + cf.BNI - 1) / cf.BNI;
        const uint32_t box[5] = {BK, (uint32_t)cf.BW, (uint32_t)cf.BH, (uint32_t)cf.BNI, (uint32_t)cf.KB};
        const uint64_t c0dim = blk ? 64 : (uint64_t)p.C;
        if (p.stride == 1) {
            const uint64_t dims[5] = {c0dim, (uint64_t)p.W, (uint64_t)p.H, (uint64_t)p.N, CB};
            uint64_t str[4] = {p.C * es, (uint64_t)p.W * p.C * es, (uint64_t)p.H * p.W * p.C * es, 128};
            if (a.a_strides[0] > 0)  // a caller-laid-out A (overlapping pixel rows)
                for (int i = 0; i < 4; ++i) str[i] = (uint64_t)a.a_strides[i];
            if (!encode(&mA[0], dt, blk ? 5 : 4, a.in[0], dims, str, box)) return cudaErrorInvalidValue;
            mA[1] = mA[2] = mA[3] = mA[0];
        } else {
            for (int bh = 0; bh < 2; ++bh)
                for (int bw = 0; bw < 2; ++bw) {
                    const char *base = static_cast<const char *>(a.in[0]) + ((int64_t)bh * p.W + bw) * p.C * es;
                    const uint64_t dims[5] = {c0dim, (uint64_t)(p.W / 2), (uint64_t)(p.H / 2), (uint64_t)p.N, CB};
                    const uint64_t str[4] = {2 * p.C * es, 2 * (uint64_t)p.W * p.C * es,
                                             (uint64_t)p.H * p.W * p.C * es, 128};
                    if (!encode(&mA[bh * 2 + bw], dt, blk ? 5 : 4, base, dims, str, box))
                        return cudaErrorInvalidValue;
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
        mR = mY;
        if (p.res && !encode(&mR, dt, 4, p.res, ydims, ystr, ybox, CU_TENSOR_MAP_SWIZZLE_128B))
            return cudaErrorInvalidValue;
    }
    if (p.mtiles <= 0 || (int64_t)p.mtiles * p.ntiles * p.ksplit > INT32_MAX) return cudaErrorInvalidValue;
    if ((int64_t)(p.ksplit + 1) * p.kiters > INT32_MAX) return cudaErrorInvalidValue;
    p.fd_ksplit = make_fastdiv((uint32_t)p.ksplit);
    p.fd_ntiles = make_fastdiv((uint32_t)p.ntiles);
    p.fd_tq = make_fastdiv((uint32_t)std::max(p.tq, 1));
    p.fd_tp = make_fastdiv((uint32_t)std::max(p.tp, 1));
    p.fd_spt = make_fastdiv((uint32_t)(p.cblocks / cf.KB));
    p.fd_S = make_fastdiv((uint32_t)p.S);
    p.lbw = p.lbwh = 0;
    if (cf.implicit) {
        while ((1 << p.lbw) < cf.BW) ++p.lbw;
        while ((1 << p.lbwh) < cf.BW * cf.BH) ++p.lbwh;
    }
    const bool bf = dt == SN_BF16;
#define SN_TC_LAUNCH(TT, BNV, GV, KBV)                                                            \
    return cf.implicit ? launch<TT, BNV, true, GV, KBV>(mA, mB, mY, mR, p, a.stream)               \
                       : launch<TT, BNV, false, GV, KBV>(mA, mB, mY, mR, p, a.stream)
#define SN_TC_LAUNCH_T(TT)                                                                          \
    if (cf.csk == 2) {                                                                              \
        if (cf.G != 1 || cf.KB != 1 || cf.ms != 1 || cf.bst || cf.ksplit != 1) return cudaErrorInvalidValue; \
        if (cf.implicit) {                                                                          \
            if (cf.BN == 128) return launch<TT, 128, true, 1, 1, false, 1, 2>(mA, mB, mY, mR, p, a.stream); \
            if (cf.BN == 256) return launch<TT, 256, true, 1, 1, false, 1, 2>(mA, mB, mY, mR, p, a.stream); \
            return cudaErrorInvalidValue;                                                           \
        }                                                                                           \
        if (cf.BN == 128) return launch<TT, 128, false, 1, 1, false, 1, 2>(mA, mB, mY, mR, p, a.stream); \
        if (cf.BN == 256) return launch<TT, 256, false, 1, 1, false, 1, 2>(mA, mB, mY, mR, p, a.stream); \
        return cudaErrorInvalidValue;                                                               \
    }                                                                                               \
    if (cf.ms == 2) {                                                                               \
        if (cf.G != 1 || cf.KB != 1 || cf.bst) return cudaErrorInvalidValue;                        \
        if (cf.implicit) {                                                                          \
            if (cf.BN == 64) return launch<TT, 64, true, 1, 1, false, 2>(mA, mB, mY, mR, p, a.stream); \
            if (cf.BN == 128) return launch<TT, 128, true, 1, 1, false, 2>(mA, mB, mY, mR, p, a.stream); \
            return cudaErrorInvalidValue;                                                           \
        }                                                                                           \
        if (cf.BN == 64) return launch<TT, 64, false, 1, 1, false, 2>(mA, mB, mY, mR, p, a.stream); \
        if (cf.BN == 128) return launch<TT, 128, false, 1, 1, false, 2>(mA, mB, mY, mR, p, a.stream); \
        return cudaErrorInvalidValue;                                                               \
    }                                                                                               \
    if (cf.bst) {                                                                                   \
        if (cf.implicit) {                                                                          \
            if (cf.BN == 64) return launch<TT, 64, true, 1, 1, true>(mA, mB, mY, mR, p, a.stream);  \
            if (cf.BN == 128) return launch<TT, 128, true, 1, 1, true>(mA, mB, mY, mR, p, a.stream);\
            return launch<TT, 256, true, 1, 1, true>(mA, mB, mY, mR, p, a.stream);                  \
        }                                                                                           \
        if (cf.BN == 64) return launch<TT, 64, false, 1, 1, true>(mA, mB, mY, mR, p, a.stream);     \
        if (cf.BN == 128) return launch<TT, 128, false, 1, 1, true>(mA, mB, mY, mR, p, a.stream);   \
        return launch<TT, 256, false, 1, 1, true>(mA, mB, mY, mR, p, a.stream);                     \
    }                                                                                               \
    if (cf.G == 1 && cf.KB > 1) {                                                                   \
        if (cf.KB == 4) {                                                                           \
            if (!cf.implicit || cf.BN != 64) return cudaErrorInvalidValue;                          \
            return launch<TT, 64, true, 1, 4>(mA, mB, mY, mR, p, a.stream);                         \
        }                                                                                           \
        if (cf.KB != 2) return cudaErrorInvalidValue;                                               \
        if (cf.BN == 64) SN_TC_LAUNCH(TT, 64, 1, 2);                                                \
        if (cf.BN == 128) SN_TC_LAUNCH(TT, 128, 1, 2);                                              \
        return cudaErrorInvalidValue;                                                               \
    }                                                                                               \
    if (cf.G == 2) {                                                                                \
        if (cf.KB == 2) {                                                                           \
            if (cf.BN == 64) SN_TC_LAUNCH(TT, 64, 2, 2);                                            \
            if (cf.BN == 128) SN_TC_LAUNCH(TT, 128, 2, 2);                                          \
            SN_TC_LAUNCH(TT, 256, 2, 2);                                                            \
        }                                                                                           \
        if (cf.BN == 64) SN_TC_LAUNCH(TT, 64, 2, 1);                                                \
        if (cf.BN == 128) SN_TC_LAUNCH(TT, 128, 2, 1);                                              \
        SN_TC_LAUNCH(TT, 256, 2, 1);                                                                \
    }                                                                                               \
    if (cf.BN == 64) SN_TC_LAUNCH(TT, 64, 1, 1);                                                    \
    if (cf.BN == 128) SN_TC_LAUNCH(TT, 128, 1, 1);                                                  \
    SN_TC_LAUNCH(TT, 256, 1, 1)
    if (bf) {
        SN_TC_LAUNCH_T(__nv_bfloat16);
    } else {
        SN_TC_LAUNCH_T(__half);
    }
#undef SN_TC_LAUNCH_T
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
    griddep_launch();
    griddep_wait();
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
    griddep_launch();
    griddep_wait();
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

cudaError_t conv_im2col_tc(const LaunchArgs &a) { return conv_im2col_tc_stage(a, -1); }

// stage 0: im2col; stage 1: the tensor-core GEMM; -1: both
cudaError_t conv_im2col_tc_stage(const LaunchArgs &a, int stage) {
    const Layer &l = *a.layer;
    const ConvDims d = conv_dims(a);
    const int64_t kpad = im2col_kpad(l);
    const int64_t M = (int64_t)d.N * d.P * d.Q;
    const size_t need = im2col_bytes(l, a.schema);
    if (!a.ws || a.ws_bytes < need || (uintptr_t)a.ws % 16) return cudaErrorInvalidValue;
    const size_t rows_bytes = (size_t)kpad * sizeof(int2) + (size_t)d.R * d.W * d.C * dtype_size(a.schema.dtype);
    if (stage == 1) {
    } else if (rows_bytes <= 48 * 1024 && d.N <= 65535) {
        SN_DT_SWITCH(a.schema.dtype, T,
                     launch_pdl(im2col_rows_kernel<T>, dim3((unsigned)d.P, (unsigned)d.N), 256, rows_bytes, a.stream, 
                         (const T *)a.in[0], (T *)a.ws, d, (int)kpad));
    } else {
        SN_DT_SWITCH(a.schema.dtype, T,
                     launch_pdl(im2col_nhwc_kernel<T>, grid_for(M * (kpad / 8), 256), 256, 0, a.stream, 
                         (const T *)a.in[0], (T *)a.ws, d, (int)kpad, M));
    }
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess || stage == 0) return e;
    const Layer gl = gemm_layer((int)kpad, d.K, d.act, l.out);
    LaunchArgs g = a;
    g.layer = &gl;
    g.routine = R_CONV_TC;
    g.out_schema = g.schema;
    g.in_shapes = {Shape{l.out.n, kpad, l.out.h, l.out.w}};
    g.in[0] = a.ws;
    g.ws = static_cast<uint8_t *>(a.ws) + im2col_bytes(l, a.schema);
    g.ws_bytes = a.ws_bytes - im2col_bytes(l, a.schema);
    return conv_tc(g);
}

// ---------------------------------------------------------------------------
// space-to-depth childnet: stride-2 convolutions of at most 4 input channels
// (the RGB stem) as a stride-1 tensor-core convolution, with no im2col matrix.
//
// With xp the input zero-padded by (ph, pw) and taps r = 2a + i, s = 2b + j,
//   y[p][q] = sum_{a, b, i, j, c} X[p + a][q + b][(2i + j) C + c] * W[a][b][(2i + j) C + c]
//   X[u][v][(2i + j) C + c] = xp[2u + i][2v + j][c],   W[a][b][..] = w[2a + i][2b + j][c]
// (W zero where 2a + i >= kh or 2b + j >= kw): ceil(kh/2) x ceil(kw/2) taps
// over an image of 4C channels.  X stores 16 channels per pixel (4C <= 16,
// the rest zero) and b runs over 4 pixels (kw <= 8), so the 64 values that
// one row of taps a multiplies for output pixel (p, q) are X[p + a][q .. q+3],
// contiguous: the GEMM's A row is one 128-byte window of X whose start moves
// by one 32-byte pixel per output pixel.  The tensor map over X says exactly
// that (pixel stride 32 B, rows of 64 values), with a fifth axis over the
// rows of taps (stride one X row), so one TMA box brings all A = 2 or 4 rows
// of taps of a 128-pixel tile (A x 16 KB) and the implicit-GEMM kernel runs
// one pipeline stage per tile: a TMA box costs about the same whatever its
// size, so few large boxes keep the tensor cores fed.
// ---------------------------------------------------------------------------
namespace {
struct S2dDims {
    int32_t N, H, W, C, ph, pw, Pp, Qp;  // input; X extent Pp x Qp
};
}  // namespace

static bool s2d_applies(const Layer &l, sn_schema s) {
    const sn_conv_params &c = l.conv;
    return l.type == SN_L_CONV2 && c.groups == 1 && c.sh == 2 && c.sw == 2 && c.dh == 1 && c.dw == 1 &&
           4 * c.c_in <= 16 && c.kh >= 3 && c.kh <= 8 && c.kw <= 8 && c.c_out % 8 == 0 && s.dtype != SN_F32 &&
           s.layout == SN_NHWC;
}

// rows of taps A = ceil(kh/2) rounded up to 2 or 4 (zero weights beyond kh);
// all A rows, 64 values each, are one TMA box and one pipeline stage
static int s2d_rows(const Layer &l) { return l.conv.kh <= 4 ? 2 : 4; }

// the GEMM as a 1x1 layer of A x 64 "channels" over the P x Q output pixels:
// "channel" block a of pixel (p, q) is X[p + a][q .. q + 3]
static Layer s2d_gemm_layer(const Layer &l) {
    Layer g;
    g.type = SN_L_CONV2;
    g.conv = sn_conv_params{64 * s2d_rows(l), l.conv.c_out, 1, 1, 1, 1, 0, 0, 1, 1, 1, l.conv.act};
    g.act = l.conv.act;
    g.out = l.out;
    return g;
}
static Shape s2d_gemm_in(const Layer &l) { return Shape{l.out.n, 64 * s2d_rows(l), l.out.h, l.out.w}; }

static size_t s2d_bytes(const Layer &l, sn_schema s) {
    const int64_t Pp = l.out.h + s2d_rows(l) - 1, Qp = l.out.w + 3;
    return ((size_t)l.out.n * Pp * Qp * 16 * dtype_size(s.dtype) + 255) & ~size_t(255);
}

int32_t conv_s2d_tc_variants(const Layer &l, const Shape &in, sn_schema s) {
    (void)in;
    if (!s2d_applies(l, s)) return 0;
    return (int32_t)tc::configs(s2d_gemm_layer(l), s2d_gemm_in(l), s, s2d_rows(l)).size();
}

size_t conv_s2d_tc_ws(const Layer &l, const Shape &in, sn_schema s, int32_t v) {
    (void)in;
    return s2d_bytes(l, s) + conv_tc_ws(s2d_gemm_layer(l), s2d_gemm_in(l), s, v, s2d_rows(l));
}

// X[n][u][v][16]: one thread per X pixel, two 16-byte stores
template <typename T>
__global__ void __launch_bounds__(256) s2d_kernel(const T *__restrict__ x, T *__restrict__ X, S2dDims d) {
    griddep_launch();
    griddep_wait();
    const int64_t total = (int64_t)d.N * d.Pp * d.Qp;
    for (int64_t t = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; t < total; t += (int64_t)gridDim.x * blockDim.x) {
        const int v = (int)(t % d.Qp), u = (int)((t / d.Qp) % d.Pp);
        const int64_t n = t / ((int64_t)d.Qp * d.Pp);
        uint4 o[2] = {make_uint4(0, 0, 0, 0), make_uint4(0, 0, 0, 0)};
        T *po = reinterpret_cast<T *>(o);
#pragma unroll
        for (int ij = 0; ij < 4; ++ij) {
            const int h = 2 * u + (ij >> 1) - d.ph, w = 2 * v + (ij & 1) - d.pw;
            if (h < 0 || h >= d.H || w < 0 || w >= d.W) continue;
            const T *xp = x + ((n * d.H + h) * d.W + w) * d.C;
            for (int c = 0; c < d.C; ++c) po[ij * d.C + c] = xp[c];
        }
        uint4 *dst = reinterpret_cast<uint4 *>(X + t * 16);
        dst[0] = o[0];
        dst[1] = o[1];
    }
}

cudaError_t conv_s2d_tc(const LaunchArgs &a) { return conv_s2d_tc_stage(a, -1); }

// stage 0: space-to-depth re-layout; stage 1: the tensor-core GEMM; -1: both
cudaError_t conv_s2d_tc_stage(const LaunchArgs &a, int stage) {
    const Layer &l = *a.layer;
    if (!s2d_applies(l, a.schema)) return cudaErrorInvalidValue;
    const Shape &in = a.in_shapes[0];
    const Shape gin = s2d_gemm_in(l);
    S2dDims d{(int32_t)in.n, (int32_t)in.h, (int32_t)in.w, (int32_t)in.c, l.conv.ph, l.conv.pw,
              (int32_t)(l.out.h + s2d_rows(l) - 1), (int32_t)(l.out.w + 3)};
    const size_t xb = s2d_bytes(l, a.schema);
    if (!a.ws || a.ws_bytes < xb || (uintptr_t)a.ws % 256) return cudaErrorInvalidValue;
    const int64_t total = (int64_t)d.N * d.Pp * d.Qp;
    if (stage != 1) {
        SN_DT_SWITCH(a.schema.dtype, T,
                     launch_pdl(s2d_kernel<T>, grid_for(total, 256), 256, 0, a.stream, (const T *)a.in[0], (T *)a.ws,
                                d));
        cudaError_t e = cudaGetLastError();
        if (e != cudaSuccess || stage == 0) return e;
    }
    const Layer gl = s2d_gemm_layer(l);
    LaunchArgs g = a;
    g.layer = &gl;
    g.routine = R_CONV_TC;
    g.out_schema = g.schema;
    g.in_shapes = {gin};
    g.in[0] = a.ws;
    const int64_t pix = 16 * (int64_t)dtype_size(a.schema.dtype);  // 32 bytes: one X pixel
    g.a_strides[0] = pix;                   // next output column: next window
    g.a_strides[1] = pix * d.Qp;            // next output row
    g.a_strides[2] = pix * d.Qp * d.Pp;     // next image
    g.a_strides[3] = pix * d.Qp;            // next row of taps: one X row down
    g.a_blocks = s2d_rows(l);
    g.ws = static_cast<uint8_t *>(a.ws) + xb;
    g.ws_bytes = a.ws_bytes - xb;
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
    g.out_schema = g.schema;  // N x C x 1 x 1: the same bytes in either layout
    return conv_tc(g);
}

}  // namespace k
}  // namespace sn
