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
#pragma once

#include <cuda.h>

#include <algorithm>

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
// SK (stream-K, one-CTA tiles of >= 2 chunks): the layer's tiles' K steps,
// laid end to end, are cut into one equal range per CTA (sk_len steps), so
// that every SM gets the same MMA work however the tile count falls against
// the SM count.  A CTA takes the tiles its range touches in order; a tile
// split between CTAs is a part in each: every epilogue warp writes its fp32
// rows of the part to the CTA's slot, and the warp that arrives last at the
// tile's counter (one per epilogue warp) sums the parts in CTA order and
// finishes the tile (bias, residual, activation, store).  No CTA waits for
// another, so the split needs no co-residency.
// HALO (3x3, stride 1, one-CTA tiles of 8 x 16 output pixels of one image):
// a K step is one tap row r of one 64-channel block; its stage holds A = the
// 10 x 16 input pixels the row's three column taps read, as one TMA box, and
// B = the three taps' weight rows.  Tap s reads A from box row s on, with
// 8-row groups 10 rows apart (the swizzle follows the absolute address, so
// any row offset and group stride work): one A box per three taps instead of
// three, and 10/8 of the rows instead of three times them.
template <typename T, int BN, int STAGES, bool IMPLICIT, int G, int KB, bool BST, int MS, int CSK, bool SK,
          bool HALO>
__global__ void __launch_bounds__(THREADS, 1)
    conv_tc_kernel(const __grid_constant__ CUtensorMap mA0, const __grid_constant__ CUtensorMap mA1,
                   const __grid_constant__ CUtensorMap mA2, const __grid_constant__ CUtensorMap mA3,
                   const __grid_constant__ CUtensorMap mB, const __grid_constant__ CUtensorMap mY,
                   const __grid_constant__ CUtensorMap mR, const Params p) {
    // a stage holds KB 64-channel blocks of one filter tap; a block of A is
    // 128 rows x 128 B, of B (BN / G) rows x 128 B (this CTA's share)
    // MS = 2: a one-CTA tile of 256 rows, one TMA box of A for both 128-row
    // halves and two MMAs (one per half, one TMEM accumulator each) sharing B
    constexpr uint32_t A_SUB = HALO ? HALO_ROWS * BK * 2 : BM * BK * 2;  // one 128-row half (or the halo box)
    constexpr uint32_t A_BLK = MS * A_SUB;
    constexpr uint32_t B_TAP = (BN / G) * BK * 2;          // one tap's weight rows
    constexpr uint32_t B_BLK = B_TAP * (HALO ? 3 : 1);
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
    // the units this CTA takes, in order: every ncl-th unit from cid, or
    // (stream-K) the tiles that its range of K steps touches
    const int sk_a = SK ? cid * p.sk_len : 0;
    const int sk_b = SK ? min(sk_a + p.sk_len, p.sk_steps) : 0;
    const int nunits = SK ? (sk_a < sk_b ? (sk_b - 1) / p.kiters - sk_a / p.kiters + 1 : 0)
                          : (cid < total ? (total - 1 - cid) / ncl + 1 : 0);
    auto unit = [&](int j, int r) -> Work {
        if constexpr (SK) {
            const int t = sk_a / p.kiters + j;
            Work w = work_of(p, t, BN, IMPLICIT, 1, 1, r);
            const int t0 = t * p.kiters, t1 = t0 + p.kiters;
            w.it0 = max(sk_a, t0) - t0;
            w.it1 = min(sk_b, t1) - t0;
            w.sk_c0 = t0 / p.sk_len;
            w.sk_n = (t1 - 1) / p.sk_len - w.sk_c0 + 1;
            w.sk_slot = sk_a >= t0 ? 0 : 1;
            return w;
        } else {
            Work w = work_of(p, cid + j * ncl, BN, IMPLICIT, G, MS, r);
            krange(w);
            return w;
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
        // this CTA's slice of the weights into L2 while the previous kernel
        // finishes (after an L2 flush they would otherwise come from HBM
        // on the critical path of the first K steps)
        if (p.wt_bytes > 0) {
            const int64_t slice = ((p.wt_bytes + gridDim.x - 1) / gridDim.x + 15) & ~(int64_t)15;
            const int64_t off = (int64_t)blockIdx.x * slice;
            if (off < p.wt_bytes)
                prefetch_l2(static_cast<const uint8_t *>(p.wt) + off, (uint32_t)min(slice, p.wt_bytes - off));
        }
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
            for (int ui = 0; ui < nunits && !stop; ++ui, ++lt) {
                const Work w = unit(ui, 0);
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
            // (halo tiles: a "tap" is a row of three taps, and the box starts
            // at the row's first column tap)
            const int cblocks = p.cblocks, S = HALO ? 1 : p.S, dh = p.dh, dw = p.dw, ph0 = p.ph, pw0 = p.pw;
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
            for (int ui = 0; ui < nunits && !stop; ++ui) {
                const Work w = unit(ui, (int)rank);
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
                        if (HALO) {  // the three taps of row `tap`: map [C][K][R*S], box 64 x BN x 3
                            tma_3d<G>(sa + A_BYTES, &mB, bar, c0, w.n0 + brow, tap * 3);
                        } else if (!BST) {  // weight-stationary B is already resident
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
            // stage 0, A; offsets add to the address field (halo: 8-row groups one box row apart)
            const uint64_t desc0 = HALO ? sdesc_sw128_sbo(su32(smem), HALO_W * 128u) : sdesc_sw128(su32(smem));
            const uint64_t descb = sdesc_sw128(su32(bst));   // weight-stationary B, K step 0
            const uint64_t deschb = sdesc_sw128(su32(smem) + A_BYTES);  // halo: stage 0, B
            int g = 0, lt = 0, s = 0;
            bool stop = false;
            if (BST && lane == 0 && !mbar_wait(&bst_bar, 0u, p.wait_limit)) {
                atomicOr(p.err, ERR_MMA_WAIT);
                set_abort();
            }
            __syncwarp();
            for (int ui = 0; ui < nunits && !stop; ++ui, ++lt) {
                const Work w = unit(ui, 0);
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
                        if constexpr (HALO) {
                            // tap s_ of the row: A from box row s_ on (128 B = 8 units), B its own rows
                            const uint64_t db = deschb + (uint64_t)((s * STAGE_BYTES) >> 4);
#pragma unroll
                            for (int s_ = 0; s_ < 3; ++s_)
#pragma unroll
                                for (int k = 0; k < BK / 16; ++k)
                                    umma<G>(d, da + 8 * s_ + 2 * k, db + s_ * (B_TAP >> 4) + 2 * k, idesc,
                                            (it > w.it0 || s_ > 0 || k > 0) ? 1u : 0u);
                        } else {
                            const uint64_t db =
                                BST ? descb + (uint64_t)(((uint32_t)it * B_BYTES) >> 4) : da + (A_BYTES >> 4);
#pragma unroll
                            for (int j = 0; j < KB; ++j)
#pragma unroll
                                for (int k = 0; k < BK / 16; ++k)
#pragma unroll
                                    for (int m = 0; m < MS; ++m)
                                        umma<G>(d + (uint32_t)(m * BN),
                                                da + j * (A_BLK >> 4) + m * (A_SUB >> 4) + 2 * k,
                                                db + j * (B_BLK >> 4) + 2 * k, idesc,
                                                (it > w.it0 || j > 0 || k > 0) ? 1u : 0u);
                        }
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
            // stage 0, A; offsets add to the address field (halo: 8-row groups one box row apart)
            const uint64_t desc0 = HALO ? sdesc_sw128_sbo(su32(smem), HALO_W * 128u) : sdesc_sw128(su32(smem));
            const uint64_t descb = sdesc_sw128(su32(bst));   // weight-stationary B, K step 0
            const uint64_t deschb = sdesc_sw128(su32(smem) + A_BYTES);  // halo: stage 0, B
            int g = 0, lt = 0, s = 0;
            uint32_t par = 0;
            bool stop = false;
            if (BST && !mbar_wait(&bst_bar, 0u, p.wait_limit)) {
                atomicOr(p.err, ERR_MMA_WAIT);
                set_abort();
                stop = true;
            }
            for (int ui = 0; ui < nunits && !stop; ++ui, ++lt) {
                const Work w = unit(ui, 0);
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
                    if constexpr (HALO) {
                        const uint64_t db = deschb + (uint64_t)((s * STAGE_BYTES) >> 4);
#pragma unroll
                        for (int s_ = 0; s_ < 3; ++s_)
#pragma unroll
                            for (int k = 0; k < BK / 16; ++k)
                                umma<G>(d, da + 8 * s_ + 2 * k, db + s_ * (B_TAP >> 4) + 2 * k, idesc,
                                        (it > w.it0 || s_ > 0 || k > 0) ? 1u : 0u);
                    } else {
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
                    }
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
        for (int ui = 0; ui < nunits && !stop; ++ui, ++lt) {
            const int b = lt & 1;
            const uint32_t aph = (uint32_t)(lt >> 1) & 1u;
            const Work w = unit(ui, 0);
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
        for (int ui = ALT ? half : 0; ui < nunits; ui += ALT ? 2 : 1, lt += ALT ? 2 : 1) {
            const int b = lt & 1;
            const uint32_t aph = (uint32_t)(lt >> 1) & 1u;
            const Work w = unit(ui, (int)rank);
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
            // (a stream-K part reads the residual only if it finishes the tile)
            const bool has_res = p.res != nullptr && p.ksplit == 1 && (!SK || w.sk_n == 1);
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
            if constexpr (SK) {
                if (w.sk_n > 1 && tile_live) {
                    // a part of a tile split between CTAs: this warp's fp32 rows
                    // go to the CTA's slot, 16-byte piece q of a lane's row of
                    // chunk ci at [ci][row quarter][q][lane], so that a store
                    // instruction writes 512 contiguous bytes
                    constexpr int SLOT4 = BM * BN / 4;          // float4 per slot
                    constexpr int CHUNK4 = EPI_WARPS / 2 * 16 * 32;  // float4 per 64-channel chunk
                    const int wofs = g4 * 16 * 32 + lane;
                    float4 *mine = reinterpret_cast<float4 *>(p.sk_part) + (int64_t)(cid * 2 + w.sk_slot) * SLOT4 + wofs;
#pragma unroll
                    for (int cj = 0; cj < CPH; ++cj) {
                        const int ci = cbase + cj;
                        if (w.n0 + 64 * ci >= p.K) break;
                        uint32_t v[64];
                        __syncwarp();
                        tmem_ld64(tmem + ((uint32_t)(g4 * 32) << 16) + (uint32_t)(b * BN + 64 * ci), v);
                        float4 *dst = mine + ci * CHUNK4;
#pragma unroll
                        for (int q = 0; q < 16; ++q)
                            dst[q * 32] = make_float4(__uint_as_float(v[4 * q]), __uint_as_float(v[4 * q + 1]),
                                                      __uint_as_float(v[4 * q + 2]), __uint_as_float(v[4 * q + 3]));
                    }
                    // the accumulator is free for this CTA's next unit
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0) mbar_arrive(&acce_bar[b]);
                    // publish the part; the warp whose arrival completes the
                    // tile's count finishes the tile and clears the count
                    __threadfence();
                    __syncwarp();
                    int *cnt = p.sk_count + (int64_t)w.sk_t * EPI_WARPS + (warp - 2);
                    int last = 0;
                    if (lane == 0) last = atomicAdd(cnt, 1) == w.sk_n - 1;
                    last = __shfl_sync(0xffffffffu, last, 0);
                    if (!last) continue;
                    if (lane == 0) *cnt = 0;
                    __threadfence();
#pragma unroll
                    for (int cj = 0; cj < CPH; ++cj) {
                        const int ci = cbase + cj;
                        const int k0 = w.n0 + 64 * ci;
                        if (k0 >= p.K) break;
                        // the parts summed in CTA order (read through L2: other SMs wrote them)
                        float acc[64];
#pragma unroll
                        for (int e = 0; e < 64; ++e) acc[e] = 0.0f;
                        for (int c = w.sk_c0; c < w.sk_c0 + w.sk_n; ++c) {
                            const int slot = c * p.sk_len >= w.sk_t * p.kiters ? 0 : 1;
                            const float4 *src = reinterpret_cast<const float4 *>(p.sk_part) +
                                                (int64_t)(c * 2 + slot) * SLOT4 + wofs + ci * CHUNK4;
#pragma unroll
                            for (int q = 0; q < 16; ++q) {
                                const float4 x = __ldcg(src + q * 32);
                                acc[4 * q] += x.x;
                                acc[4 * q + 1] += x.y;
                                acc[4 * q + 2] += x.z;
                                acc[4 * q + 3] += x.w;
                            }
                        }
                        // this row's residual (the output's NHWC layout), 8 channels per piece
                        uint32_t rv[2][16];
#pragma unroll
                        for (int h = 0; h < 2; ++h)
#pragma unroll
                            for (int q = 0; q < 16; ++q) rv[h][q] = 0u;
                        if (p.res && valid) {
                            const uint4 *rr = reinterpret_cast<const uint4 *>(static_cast<const T *>(p.res) + pix * p.K + k0);
#pragma unroll
                            for (int q = 0; q < 8; ++q)
                                if (k0 + 8 * q < p.K) {
                                    const uint4 u = rr[q];
                                    rv[q >> 2][4 * (q & 3)] = u.x;
                                    rv[q >> 2][4 * (q & 3) + 1] = u.y;
                                    rv[q >> 2][4 * (q & 3) + 2] = u.z;
                                    rv[q >> 2][4 * (q & 3) + 3] = u.w;
                                }
                        }
                        if (lane == 0) bulk_wait_read_0();  // the previous store has read the block
                        __syncwarp();
                        auto finish_rows = [&](auto act) {
#pragma unroll
                            for (int q = 0; q < 8; ++q) {
                                const int h = q >> 2;
                                uint32_t wq[4];
#pragma unroll
                                for (int e = 0; e < 4; ++e) {
                                    const int jp = 4 * (q & 3) + e;  // pair index within the half
                                    const float2 r2 = unpack2<T>(rv[h][jp]);
                                    const float f0 = act(acc[32 * h + 2 * jp] +
                                                         __shfl_sync(0xffffffffu, bias_r[cj][h], 2 * jp) + r2.x);
                                    const float f1 = act(acc[32 * h + 2 * jp + 1] +
                                                         __shfl_sync(0xffffffffu, bias_r[cj][h], 2 * jp + 1) + r2.y);
                                    wq[e] = pack2<T>(f0, f1);
                                }
                                *reinterpret_cast<uint4 *>(buf + lane * 128 + ((q ^ (lane & 7)) << 4)) =
                                    make_uint4(wq[0], wq[1], wq[2], wq[3]);
                            }
                        };
                        if (p.act == SN_ACT_RELU)
                            finish_rows([](float x) { return fmaxf(x, 0.0f); });
                        else if (p.act == SN_ACT_NONE)
                            finish_rows([](float x) { return x; });
                        else
                            finish_rows([act = p.act](float x) { return act_apply(x, act); });
                        fence_proxy_async_smem();
                        __syncwarp();
                        if (lane == 0) {
                            if (IMPLICIT)
                                tma_store_4d(&mY, buf, k0, w.q0 + wq0, w.p0 + hp0, w.i0 + ni0);
                            else
                                tma_store_2d(&mY, buf, k0, (int)(w.m0 + r0));
                            bulk_commit();
                        }
                        __syncwarp();
                    }
                    continue;
                }
            }
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

template <typename T, int BN, bool IMPLICIT, int G, int KB, bool BST = false, int MS = 1, int CSK = 1,
          bool SK = false, bool HALO = false>
static cudaError_t launch(const CUtensorMap *mA, const CUtensorMap &mB, const CUtensorMap &mY, const CUtensorMap &mR,
                          const Params &p,
                          cudaStream_t st) {
    constexpr int STAGES = BST ? BST_STAGES : HALO ? halo_stages(BN / G) : stages_for(BN, G, KB, MS);
    // bytes of one pipeline stage (A and this CTA's share of B), as the kernel lays them out
    constexpr size_t STAGE = HALO ? (size_t)HALO_ROWS * BK * 2 + 3 * (size_t)(BN / G) * BK * 2
                                  : (size_t)KB * (MS * BM * BK * 2 + (BN / G) * BK * 2);
    static_assert(CSK == 1 || (size_t)STAGES * KB * (BM * BK * 2 + BN * BK * 2) >= EPI_WARPS * XBLK_BYTES,
                  "cluster K split: the exchange blocks live in the stage memory");
    constexpr size_t smem_max = 227 * 1024;
    const size_t smem = BST ? (size_t)STAGES * BM * BK * 2 + p.bst_bytes + EPI_WARPS * STG_BYTES + 1024
                            : (size_t)STAGES * STAGE + EPI_WARPS * STG_BYTES + 1024;
    static_assert(BST || (size_t)STAGES * STAGE + EPI_WARPS * STG_BYTES + 1024 <= smem_max, "shared memory per CTA");
    static_assert(!HALO || (IMPLICIT && KB == 1 && MS == 1 && !BST && CSK == 1 && !SK),
                  "halo tiles: implicit tiles of one CTA or a pair, one channel block per stage");
    static_assert(!BST || (G == 1 && KB == 1 && MS == 1), "weight-stationary tiles are one-CTA, one block per stage");
    static_assert(MS == 1 || (G == 1 && KB == 1 && !BST && 2 * MS * BN <= 512), "two-half tiles: one CTA, TMEM");
    static_assert(CSK == 1 || (G == 1 && MS == 1 && !BST && BN >= 128), "cluster K split: one-CTA tiles of >= 2 chunks");
    static_assert(!SK || (G == 1 && MS == 1 && !BST && CSK == 1 && BN >= 128), "stream-K: one-CTA tiles of >= 2 chunks");
    static_assert(STAGES >= 2, "pipeline depth");
    if (smem > smem_max) return cudaErrorInvalidValue;
    auto kern = conv_tc_kernel<T, BN, STAGES, IMPLICIT, G, KB, BST, MS, CSK, SK, HALO>;
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
    if (SK) {  // one CTA per range of sk_len K steps
        if (p.sk_len <= 0 || p.ksplit != 1 || !p.sk_count || !p.sk_part) return cudaErrorInvalidValue;
        cfg.gridDim = dim3((unsigned)((p.sk_steps + p.sk_len - 1) / p.sk_len));
    } else {
        cfg.gridDim = dim3((unsigned)((CLUSTER ? 2 : 1) * std::min(total, max_groups)));
    }
    cudaError_t e = cudaLaunchKernelEx(&cfg, kern, mA[0], mA[1], mA[2], mA[3], mB, mY, mR, p);
    if (e != cudaSuccess || p.ksplit == 1) return e;
    const int64_t n4 = p.Mout * (p.K / 4);
    launch_pdl(splitk_reduce_kernel<T>, grid_for(n4, 256), 256, 0, st, p.part, p.bias, static_cast<const T *>(p.res),
               static_cast<T *>(p.y), p.Mout, p.K,
                                                               p.ksplit, p.act);
    return cudaGetLastError();
}

// halo launches (kernels_tc_halo.cu): 3x3 stride-1 tiles of 8 x 16 pixels per
// CTA; one CTA (g = 1, bn in {64, 128}) or a pair sharing B (g = 2, bn in {64, 128, 256})
cudaError_t launch_halo(int dtype, int bn, int g, const CUtensorMap *mA, const CUtensorMap &mB,
                        const CUtensorMap &mY, const CUtensorMap &mR, const Params &p, cudaStream_t st);

// stream-K launches (kernels_tc_sk.cu): one-CTA tiles of bn in {128, 256}
// output channels, kb channel blocks per stage
cudaError_t launch_sk(int dtype, int bn, int kb, bool implicit, const CUtensorMap *mA, const CUtensorMap &mB,
                      const CUtensorMap &mY, const CUtensorMap &mR, const Params &p, cudaStream_t st);

}  // namespace tc
}  // namespace k
}  // namespace sn
