// Chained execution of consecutive tensor-core convolution layers: one
// persistent launch runs every work unit of a run of conv2/igemm_tc layers
// (section III-A: the tuned net is executed layer after layer; here the
// layers' tiles are scheduled by data flow instead of by kernel boundaries).
//
// Each layer of the chain keeps its own implicit-GEMM formulation (the
// per-layer routine of the selected path: tensor maps over its input, its
// weights, its output and its residual; its output-channel tile BN and pixel
// tiling).  The units of all layers form one list, layer after layer, a
// layer's units pixel tile by pixel tile with the output-channel tiles of a
// pixel tile adjacent; CTA c of the grid takes units c, c + grid, ...  Before
// a unit loads its input, its producer warps wait until every pixel tile of
// the layer that writes that input, and that covers the unit's receptive
// field, is complete; the epilogue likewise waits for the residual's tiles.
// A pixel tile is complete when every epilogue warp of every one of its
// output-channel tiles has seen its TMA stores land (bulk wait_group 0) and
// bumped the tile's counter with a release add.  So the next layer's tiles
// start as soon as their inputs exist, the epilogue of one layer overlaps the
// main loop of the next, and there is no launch, prologue or drain between
// layers.
//
// Progress: units are taken in list order and depend only on units of
// earlier layers, i.e. on smaller unit indices; the launch is cooperative
// (every CTA resident), so the smallest unfinished unit always has its
// inputs and its CTA is working on it.  Every wait is still bounded: on
// expiry the kernel records the cause in the library's error word and raises
// the launch's abort flag, every CTA sees the flag and stops, drains its own
// copies and MMAs, frees TMEM and exits.  The last CTA to exit zeroes the
// completion counters and the flag for the next launch.
//
// Roles (384 threads): warp 0 lane 0 and warp 10 lane 0 = TMA producers of
// the even / odd pipeline stages (warp 0 also allocates TMEM; the whole warp
// polls dependencies), warp 1 = MMA issuer, warp 11 = the MMA issuer's
// waiter (it performs the stage-full and accumulator-drained waits and hands
// them over through a named barrier), warps 2-9 = epilogue (four row
// quarters x two column halves; 64-channel tiles alternate between the two
// groups of four).
#include <cuda.h>

#include <algorithm>
#include <cstring>
#include <string>
#include <vector>

#include "tc_common.cuh"

namespace sn {
namespace k {
namespace tc {

constexpr int CH_STAGES = 4;              // pipeline depth
constexpr uint32_t CH_SLOT = 49152;       // one stage: A (KB x 16 KB) + B (KB x BN x 128 B) <= 48 KB
constexpr uint32_t CH_TMEM_COLS = 512;    // two accumulators of up to 256 columns
constexpr uint32_t CH_ACC_STRIDE = 256;
constexpr size_t CH_SMEM = (size_t)CH_STAGES * CH_SLOT + EPI_WARPS * STG_BYTES + 1024;
enum : int { ERR_DEP_WAIT = 0x100 };

// one layer of a chain, as the kernel reads it (global memory, written by the
// host before the launch; the tensor maps are 64-byte aligned)
struct alignas(128) ChainLayer {
    CUtensorMap mA[4];  // input; stride 2: the even/odd row and column sub-lattices
    CUtensorMap mB;     // weights [K][R*S][C] (block axis when KB = 2)
    CUtensorMap mY;     // output
    CUtensorMap mR;     // residual (the output's layout); unused without one
    int32_t N, H, W, C, K, P, Q, R, S, stride, ph, pw, dh, dw;
    int32_t cblocks, kiters, KB, BN, implicit;
    int32_t BW, BH, BNI, tq, tp, lbw, lbh, lbn, lbwh;
    int32_t mtiles, ntiles;
    FastDiv fd_ntiles, fd_tq, fd_tp, fd_spt, fd_S, fd_PQ, fd_Q;
    int32_t Mout;
    int32_t act, has_res;
    int32_t unit_begin, unit_end;
    int32_t done_base, done_target;  // this layer's per-pixel-tile counters; arrivals when complete
    int32_t src, res_src;            // chain index of the layer writing input 0 / the residual; -1: none
    const float *bias;
};

struct ChainArgs {
    const ChainLayer *L;
    int32_t n_layers, total;
    int32_t *done;      // [done_count] completion counters, then the exit counter and the abort flag
    int32_t done_count;
    int *err;           // the library's error word (reporting only)
};

// a unit's tile: output-channel offset and pixel origin
struct CUnit {
    int mt, n0, m0, q0, p0, i0;
};
__device__ __forceinline__ CUnit decode(const ChainLayer &L, int v) {
    CUnit w;
    w.mt = (int)fdiv((uint32_t)v, L.fd_ntiles);
    w.n0 = (v - w.mt * L.ntiles) * L.BN;
    w.m0 = w.q0 = w.p0 = w.i0 = 0;
    if (L.implicit) {
        int bx = w.mt;
        int nb = (int)fdiv((uint32_t)bx, L.fd_tq);
        w.q0 = (bx - nb * L.tq) * L.BW;
        bx = nb;
        nb = (int)fdiv((uint32_t)bx, L.fd_tp);
        w.p0 = (bx - nb * L.tp) * L.BH;
        w.i0 = nb * L.BNI;
    } else {
        w.m0 = w.mt * BM;
    }
    return w;
}

// inclusive pixel box [n0, n1] x [h0, h1] x [w0, w1]
struct PBox {
    int n0, n1, h0, h1, w0, w1;
};
// the output pixels of a unit's tile (clamped to the output)
__device__ __forceinline__ PBox out_box(const ChainLayer &L, const CUnit &w) {
    PBox b;
    if (L.implicit) {
        b.n0 = w.i0, b.n1 = min(w.i0 + L.BNI, L.N) - 1;
        b.h0 = w.p0, b.h1 = min(w.p0 + L.BH, L.P) - 1;
        b.w0 = w.q0, b.w1 = min(w.q0 + L.BW, L.Q) - 1;
    } else {  // rows [m0, m0 + 128) of the N x P x Q pixels, as a covering box
        const int r0 = w.m0, r1 = min(w.m0 + BM, L.Mout) - 1;
        const int na = (int)fdiv((uint32_t)r0, L.fd_PQ), nb = (int)fdiv((uint32_t)r1, L.fd_PQ);
        const int ra = r0 - na * L.P * L.Q, rb = r1 - nb * L.P * L.Q;
        const int ha = (int)fdiv((uint32_t)ra, L.fd_Q), hb = (int)fdiv((uint32_t)rb, L.fd_Q);
        b.n0 = na, b.n1 = nb;
        if (na != nb) {
            b.h0 = 0, b.h1 = L.P - 1, b.w0 = 0, b.w1 = L.Q - 1;
        } else {
            b.h0 = ha, b.h1 = hb;
            if (ha != hb) b.w0 = 0, b.w1 = L.Q - 1;
            else b.w0 = ra - ha * L.Q, b.w1 = rb - hb * L.Q;
        }
    }
    return b;
}
// the input pixels the output box reads (its receptive field, clamped)
__device__ __forceinline__ PBox in_box(const ChainLayer &L, const PBox &o) {
    PBox b;
    b.n0 = o.n0, b.n1 = o.n1;
    b.h0 = max(o.h0 * L.stride - L.ph, 0);
    b.h1 = min(o.h1 * L.stride - L.ph + (L.R - 1) * L.dh, L.H - 1);
    b.w0 = max(o.w0 * L.stride - L.pw, 0);
    b.w1 = min(o.w1 * L.stride - L.pw + (L.S - 1) * L.dw, L.W - 1);
    return b;
}

__device__ __forceinline__ int ld_acquire(const int32_t *p) {
    int v;
    asm volatile("ld.acquire.gpu.global.s32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}
__device__ __forceinline__ void red_release_add(int32_t *p, int v) {
    asm volatile("red.release.gpu.global.add.s32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}
__device__ __forceinline__ void fence_proxy_async_global() { asm volatile("fence.proxy.async.global;" ::: "memory"); }
__device__ __forceinline__ int ld_volatile(const int *p) {
    int v;
    asm volatile("ld.volatile.global.s32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}

// Whole warp: wait until every pixel tile of layer PL that holds a pixel of
// box b (in PL's output) is complete.  Lanes poll disjoint tiles; the warp
// then synchronises (bar.warp.sync orders the lanes' acquires before what
// lane 0 does next).  False on expiry or when another CTA reported an error.
__device__ bool wait_box(const ChainLayer &PL, const int32_t *done, const PBox &b, const int *abort_flag, int lane) {
    const int target = PL.done_target;
    const int32_t *cnt = done + PL.done_base;
    const long long t0 = clock64();
    for (;;) {
        bool mine = true;
        if (PL.implicit) {
            const int bq0 = b.w0 >> PL.lbw, bq1 = b.w1 >> PL.lbw;
            const int bp0 = b.h0 >> PL.lbh, bp1 = b.h1 >> PL.lbh;
            const int bn0 = b.n0 >> PL.lbn, bn1 = b.n1 >> PL.lbn;
            const int nq = bq1 - bq0 + 1, np = bp1 - bp0 + 1;
            const int count = nq * np * (bn1 - bn0 + 1);
            for (int i = lane; i < count; i += 32) {
                const int q = i % nq, rest = i / nq;
                const int pp = rest % np, nn = rest / np;
                const int t = ((bn0 + nn) * PL.tp + bp0 + pp) * PL.tq + bq0 + q;
                if (ld_acquire(cnt + t) < target) mine = false;
            }
        } else {  // 128-row tiles of the flattened pixels: one row range per image
            for (int n = b.n0 + lane; n <= b.n1; n += 32) {
                const int t0r = ((n * PL.P + b.h0) * PL.Q + b.w0) >> 7;
                const int t1r = ((n * PL.P + b.h1) * PL.Q + b.w1) >> 7;
                for (int t = t0r; t <= t1r; ++t)
                    if (ld_acquire(cnt + t) < target) mine = false;
            }
        }
        const bool all = __all_sync(0xffffffffu, mine);
        __syncwarp();
        if (all) return true;
        int stop = 0;
        if (lane == 0) stop = ld_volatile(abort_flag) != 0 || clock64() - t0 > WAIT_LIMIT;
        if (__shfl_sync(0xffffffffu, stop, 0)) return false;
        __nanosleep(128);
    }
}

template <typename T>
__global__ void __launch_bounds__(THREADS, 1) conv_chain_kernel(const ChainArgs a) {
    extern __shared__ uint8_t smem_raw[];
    __shared__ __align__(8) uint64_t full_bar[CH_STAGES];
    __shared__ __align__(8) uint64_t empty_bar[CH_STAGES];
    __shared__ __align__(8) uint64_t accf_bar[2];
    __shared__ __align__(8) uint64_t acce_bar[2];
    __shared__ __align__(8) uint64_t res_bar[EPI_WARPS];
    __shared__ uint32_t tmem_sh;
    __shared__ volatile int abort_sh;
    __shared__ int issued_sh[2], consumed_sh, last_sh;

    griddep_launch();
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t *stg = smem + CH_STAGES * CH_SLOT;  // epilogue staging: one 4 KB block per warp
    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    const int cid = (int)blockIdx.x, ncl = (int)gridDim.x;
    const ChainLayer *__restrict__ Ls = a.L;
    // this launch's abort flag (after the exit counter): set by a CTA that
    // gives up, read by every wait, cleared with the counters
    int32_t *abort_flag = a.done + a.done_count + 1;
    auto set_abort = [&]() {
        abort_sh = 1;
        atomicExch(abort_flag, 1);
    };

    if (threadIdx.x == 0) {
        for (int s = 0; s < CH_STAGES; ++s) {
            mbar_init(&full_bar[s], 1);
            mbar_init(&empty_bar[s], 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(&accf_bar[b], 1);
            mbar_init(&acce_bar[b], EPI_WARPS);  // every epilogue warp arrives once per unit
        }
        for (int i = 0; i < EPI_WARPS; ++i) mbar_init(&res_bar[i], 1);
        abort_sh = 0;
        issued_sh[0] = issued_sh[1] = 0;
        consumed_sh = 0;
        fence_mbar_init();
    }
    if (warp == 0) tmem_alloc<1>(&tmem_sh, CH_TMEM_COLS);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_sh;

    if (warp == 11) {  // ---------------- the MMA issuer's waiter
        int l = 0, lt = 0, s = 0;
        uint32_t par = 0;
        bool stop = false;
        for (int u = cid; u < a.total && !stop; u += ncl, ++lt) {
            while (u >= Ls[l].unit_end) ++l;
            const int kiters = Ls[l].kiters;
            const int b = lt & 1;
            const uint32_t aph = (uint32_t)(lt >> 1) & 1u;
            bool ok = mbar_wait(&acce_bar[b], aph ^ 1u);
            if (!ok) {
                if (lane == 0) atomicOr(a.err, ERR_EPI_WAIT);
                set_abort();
            }
            __syncwarp();
            if (bar_red_or(BAR_MMA, 64, !ok || abort_sh)) break;
            for (int it = 0; it < kiters; ++it) {
                ok = mbar_wait(&full_bar[s], par);
                if (!ok) {
                    if (lane == 0) atomicOr(a.err, ERR_MMA_WAIT);
                    set_abort();
                }
                __syncwarp();
                if (bar_red_or(BAR_MMA, 64, !ok || abort_sh)) {
                    stop = true;
                    break;
                }
                if (++s == CH_STAGES) {
                    s = 0;
                    par ^= 1u;
                }
            }
        }
    } else if (warp == 0 || warp == 10) {  // ---------------- TMA producers (the whole warp polls)
        const int prod = warp == 0 ? 0 : 1;
        int l = -1, g = 0, s = prod, issued = 0;
        uint32_t par = 0;
        bool stop = false, waited = false;
        for (int u = cid; u < a.total && !stop; u += ncl) {
            if (l < 0 || u >= Ls[l].unit_end) {
                do ++l;
                while (u >= Ls[l].unit_end);
                if (lane == 0)
                    for (int i = 0; i < 7; ++i)
                        asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&Ls[l].mA[0] + i))
                                     : "memory");
            }
            const ChainLayer &L = Ls[l];
            const CUnit w = decode(L, u - L.unit_begin);
            if (!waited) {
                griddep_wait();  // the previous kernel's output, and the counters it left zeroed
                waited = true;
            }
            if (L.src >= 0) {
                const PBox ib = in_box(L, out_box(L, w));
                if (!wait_box(Ls[L.src], a.done, ib, abort_flag, lane)) {
                    if (lane == 0) atomicOr(a.err, ERR_DEP_WAIT);
                    set_abort();
                    break;
                }
            }
            if (lane == 0) fence_proxy_async_global();  // the tiles' generic-proxy acquire before our TMA reads
            const int KB = L.KB, BN = L.BN, S = L.S, cblocks = L.cblocks;
            const uint32_t a_bytes = (uint32_t)KB * BM * BK * 2, stage_bytes = a_bytes + (uint32_t)KB * BN * BK * 2;
            int tap = 0, cb = 0, r = 0, ss = 0;
            for (int it = 0; it < L.kiters; ++it, ++g) {
                if ((g & 1) == prod) {
                    bool ok = true;
                    if (lane == 0) ok = mbar_wait(&empty_bar[s], par ^ 1u);
                    ok = __shfl_sync(0xffffffffu, ok, 0);
                    if (!ok) {
                        if (lane == 0) atomicOr(a.err, ERR_TMA_WAIT);
                        set_abort();
                    }
                    if (__shfl_sync(0xffffffffu, (int)abort_sh, 0)) {
                        stop = true;
                        break;
                    }
                    if (lane == 0) {
                        const uint32_t sa = su32(smem + s * CH_SLOT);
                        const uint32_t bar = su32(&full_bar[s]);
                        const int c0 = cb * BK;
                        mbar_expect_tx(&full_bar[s], stage_bytes);
                        if (L.implicit) {
                            const int oh = r * L.dh - L.ph, ow = ss * L.dw - L.pw;
                            const CUtensorMap *m = &L.mA[0];
                            int qa = w.q0 + ow, pa = w.p0 + oh;
                            if (L.stride != 1) {
                                const int bh = oh & 1, bw = ow & 1;
                                m = &L.mA[bh * 2 + bw];
                                qa = w.q0 + ((ow - bw) >> 1);
                                pa = w.p0 + ((oh - bh) >> 1);
                            }
                            if (KB == 1)
                                tma_4d<1>(sa, m, bar, c0, qa, pa, w.i0);
                            else
                                tma_5d<1>(sa, m, bar, 0, qa, pa, w.i0, cb);
                        } else {
                            if (KB == 1)
                                tma_2d<1>(sa, &L.mA[0], bar, c0, w.m0);
                            else
                                tma_3d<1>(sa, &L.mA[0], bar, 0, w.m0, cb);
                        }
                        if (KB == 1)
                            tma_3d<1>(sa + a_bytes, &L.mB, bar, c0, tap, w.n0);
                        else
                            tma_4d<1>(sa + a_bytes, &L.mB, bar, 0, tap, w.n0, cb);
                    }
                    issued = g + 1;
                    s += 2;
                    if (s >= CH_STAGES) {
                        s -= CH_STAGES;
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
        if (lane == 0) issued_sh[prod] = issued;
    } else if (warp == 1) {  // ---------------- MMA issuer (lane 0; the whole warp meets the waiter)
        const uint64_t desc0 = sdesc_sw128(su32(smem));
        int l = 0, g = 0, lt = 0, s = 0;
        bool stop = false;
        for (int u = cid; u < a.total && !stop; u += ncl, ++lt) {
            while (u >= Ls[l].unit_end) ++l;
            const int kiters = Ls[l].kiters, KB = Ls[l].KB, BN = Ls[l].BN;
            const uint32_t idesc = idesc_f16<T>(BM, BN);
            const uint32_t a_units = (uint32_t)(KB * BM * BK * 2) >> 4, b_blk = (uint32_t)(BN * BK * 2) >> 4;
            const int b = lt & 1;
            if (bar_red_or(BAR_MMA, 64, false)) break;  // accumulator b drained
            tc_fence_after();
            const uint32_t d = tmem + (uint32_t)b * CH_ACC_STRIDE;
            for (int it = 0; it < kiters; ++it, ++g) {
                if (bar_red_or(BAR_MMA, 64, false)) {  // stage s full
                    stop = true;
                    break;
                }
                tc_fence_after();
                if (lane == 0) {
                    const uint64_t da = desc0 + (uint64_t)((s * CH_SLOT) >> 4);
                    const uint64_t db = da + a_units;
#pragma unroll
                    for (int k = 0; k < BK / 16; ++k)
                        umma<1>(d, da + 2 * k, db + 2 * k, idesc, (it > 0 || k > 0) ? 1u : 0u);
                    if (KB == 2) {
#pragma unroll
                        for (int k = 0; k < BK / 16; ++k)
                            umma<1>(d, da + ((BM * BK * 2) >> 4) + 2 * k, db + b_blk + 2 * k, idesc, 1u);
                    }
                    umma_commit<1>(&empty_bar[s]);
                }
                __syncwarp();
                if (++s == CH_STAGES) s = 0;
            }
            if (!stop && lane == 0) umma_commit<1>(&accf_bar[b]);
            __syncwarp();
        }
        if (lane == 0) consumed_sh = g;
    } else {  // ---------------- epilogue: warps 2..9
        const int half = (warp - 2) >> 2;
        const int g4 = warp & 3;
        uint8_t *buf = stg + (warp - 2) * STG_BYTES;
        const int r0 = g4 * 32;
        int l = 0, lt = 0;
        uint32_t rpar = 0;
        bool waited = false;
        // Completion of a unit is signalled once its stores have landed, but
        // this warp does not wait for that before draining the next unit: the
        // signal stays pending (one unit at most) and is sent when the next
        // unit's stores have been issued (its bulk groups are younger), or
        // before any wait that could depend on it.
        int32_t *pending = nullptr;
        auto flush = [&]() {
            if (pending && lane == 0) {
                bulk_wait_all();
                fence_proxy_async_global();
                red_release_add(pending, 1);
            }
            pending = nullptr;
            __syncwarp();
        };
        for (int u = cid; u < a.total; u += ncl, ++lt) {
            while (u >= Ls[l].unit_end) ++l;
            const ChainLayer &L = Ls[l];
            const int b = lt & 1;
            const uint32_t aph = (uint32_t)(lt >> 1) & 1u;
            const int nch = L.BN >> 6;
            // 64-channel tiles: the two groups of four take alternate units
            // (group (lt & 1)); the other group only keeps the barrier phases
            if (nch == 1 && half != (lt & 1)) {
                if (!mbar_try(&accf_bar[b], aph)) flush();
                if (!mbar_wait(&accf_bar[b], aph)) {
                    if (lane == 0) atomicOr(a.err, ERR_ACC_WAIT);
                    set_abort();
                    break;
                }
                __syncwarp();
                if (lane == 0) mbar_arrive(&acce_bar[b]);
                continue;
            }
            const int cph = nch == 1 ? 1 : nch >> 1;  // chunks this warp drains
            const int cbase = nch == 1 ? 0 : half * cph;
            const CUnit w = decode(L, u - L.unit_begin);
            const int wq0 = L.implicit ? r0 & (L.BW - 1) : 0;
            const int hp0 = L.implicit ? (r0 >> L.lbw) & (L.BH - 1) : 0;
            const int ni0 = L.implicit ? r0 >> L.lbwh : 0;
            float bias_r[2][2];
#pragma unroll
            for (int cj = 0; cj < 2; ++cj)
#pragma unroll
                for (int h = 0; h < 2; ++h)
                    bias_r[cj][h] = cj < cph ? __ldg(L.bias + w.n0 + 64 * (cbase + cj) + 32 * h + lane) : 0.f;
            if (!waited) {
                griddep_wait();
                waited = true;
            }
            const bool has_res = L.has_res != 0;
            if (has_res && L.res_src >= 0) {
                flush();  // the residual may be a tile whose signal this warp holds
                if (!wait_box(Ls[L.res_src], a.done, out_box(L, w), abort_flag, lane)) {
                    if (lane == 0) atomicOr(a.err, ERR_DEP_WAIT);
                    set_abort();
                    break;
                }
            }
            if (has_res && lane == 0) fence_proxy_async_global();
            auto issue_res = [&](int k0) {
                if (!has_res || k0 >= L.K) return;
                if (lane == 0) {
                    bulk_wait_read_0();
                    mbar_expect_tx(&res_bar[warp - 2], STG_BYTES);
                    if (L.implicit)
                        tma_4d<1>(su32(buf), &L.mR, su32(&res_bar[warp - 2]), k0, w.q0 + wq0, w.p0 + hp0, w.i0 + ni0);
                    else
                        tma_2d<1>(su32(buf), &L.mR, su32(&res_bar[warp - 2]), k0, w.m0 + r0);
                }
            };
            issue_res(w.n0 + 64 * cbase);
            if (!mbar_try(&accf_bar[b], aph)) flush();
            if (!mbar_wait(&accf_bar[b], aph)) {
                if (lane == 0) atomicOr(a.err, ERR_ACC_WAIT);
                set_abort();
                break;
            }
            tc_fence_after();
            const int act = L.act;
            int groups = 0;  // bulk store groups this warp commits for the unit
#pragma unroll
            for (int cj = 0; cj < 2; ++cj) {
                if (cj >= cph) break;
                const int ci = cbase + cj;
                const int k0 = w.n0 + 64 * ci;
                if (k0 >= L.K) break;
                const uint32_t taddr = tmem + ((uint32_t)(g4 * 32) << 16) + (uint32_t)b * CH_ACC_STRIDE + 64 * ci;
                uint32_t rv[2][16];
#pragma unroll
                for (int h = 0; h < 2; ++h)
#pragma unroll
                    for (int j = 0; j < 16; ++j) rv[h][j] = 0u;
                if (!has_res && lane == 0) bulk_wait_read_0();
                if (has_res) {
                    if (!mbar_wait(&res_bar[warp - 2], rpar)) {
                        if (lane == 0) atomicOr(a.err, ERR_EPI_WAIT);
                        set_abort();
                    }
                    rpar ^= 1u;
#pragma unroll
                    for (int j = 0; j < 8; ++j) {
                        const uint4 q = *reinterpret_cast<const uint4 *>(buf + lane * 128 + ((j ^ (lane & 7)) << 4));
                        rv[j >> 2][4 * (j & 3)] = q.x;
                        rv[j >> 2][4 * (j & 3) + 1] = q.y;
                        rv[j >> 2][4 * (j & 3) + 2] = q.z;
                        rv[j >> 2][4 * (j & 3) + 3] = q.w;
                    }
                }
                uint32_t v[64];
                __syncwarp();
                tmem_ld64(taddr, v);
                auto stage_rows = [&](auto actf) {
#pragma unroll
                    for (int q = 0; q < 8; ++q) {
                        const int h = q >> 2;
                        uint32_t wq[4];
#pragma unroll
                        for (int e = 0; e < 4; ++e) {
                            const int j = 4 * (q & 3) + e;
                            const float2 r2 = unpack2<T>(rv[h][j]);
                            const float f0 = actf(__uint_as_float(v[32 * h + 2 * j]) +
                                                  __shfl_sync(0xffffffffu, bias_r[cj][h], 2 * j) + r2.x);
                            const float f1 = actf(__uint_as_float(v[32 * h + 2 * j + 1]) +
                                                  __shfl_sync(0xffffffffu, bias_r[cj][h], 2 * j + 1) + r2.y);
                            wq[e] = pack2<T>(f0, f1);
                        }
                        *reinterpret_cast<uint4 *>(buf + lane * 128 + ((q ^ (lane & 7)) << 4)) =
                            make_uint4(wq[0], wq[1], wq[2], wq[3]);
                    }
                };
                if (act == SN_ACT_RELU)
                    stage_rows([](float x) { return fmaxf(x, 0.0f); });
                else if (act == SN_ACT_NONE)
                    stage_rows([](float x) { return x; });
                else
                    stage_rows([act](float x) { return act_apply(x, act); });
                fence_proxy_async_smem();
                __syncwarp();
                if (lane == 0) {
                    if (L.implicit)
                        tma_store_4d(&L.mY, buf, k0, w.q0 + wq0, w.p0 + hp0, w.i0 + ni0);
                    else
                        tma_store_2d(&L.mY, buf, k0, w.m0 + r0);
                    bulk_commit();
                }
                ++groups;
                if (cj + 1 < cph) issue_res(k0 + 64);
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) {
                mbar_arrive(&acce_bar[b]);
                // the previous unit's stores are older than this unit's
                // `groups` bulk groups: once at most that many remain, the
                // previous unit's part is in global memory and is counted
                if (pending) {
                    if (groups >= 2) asm volatile("cp.async.bulk.wait_group 2;" ::: "memory");
                    else if (groups == 1) asm volatile("cp.async.bulk.wait_group 1;" ::: "memory");
                    else bulk_wait_all();
                    fence_proxy_async_global();
                    red_release_add(pending, 1);
                }
            }
            pending = a.done + L.done_base + w.mt;
            __syncwarp();
            if (__shfl_sync(0xffffffffu, lane == 0 ? ld_volatile(abort_flag) : 0, 0) != 0) break;
        }
        flush();
        if (lane == 0) bulk_wait_all();
        __syncwarp();
    }

    tc_fence_before();
    __syncthreads();
    if (warp == 0) {
        if (abort_sh && lane == 0) {
            // let the copies and MMAs this CTA waited for land before its
            // memory goes away (one deadline for the whole drain)
            const long long t0 = clock64();
            const int issued = max(issued_sh[0], issued_sh[1]);
            for (int g = consumed_sh; g < issued; ++g)
                while (!mbar_try(&full_bar[g % CH_STAGES], (uint32_t)(g / CH_STAGES) & 1u) &&
                       clock64() - t0 < WAIT_LIMIT) {
                }
            if (consumed_sh > 0) {
                const int g = consumed_sh - 1;
                while (!mbar_try(&empty_bar[g % CH_STAGES], (uint32_t)(g / CH_STAGES) & 1u) &&
                       clock64() - t0 < WAIT_LIMIT) {
                }
            }
        }
        __syncwarp();
        tc_fence_after();
        tmem_dealloc<1>(tmem, CH_TMEM_COLS);
    }
    // the last CTA to leave zeroes the completion counters: every other CTA
    // has finished all of its waits by then
    if (threadIdx.x == 0) {
        __threadfence();
        last_sh = atomicAdd(a.done + a.done_count, 1) == (int)gridDim.x - 1;
    }
    __syncthreads();
    if (last_sh) {
        for (int i = threadIdx.x; i < a.done_count; i += blockDim.x) a.done[i] = 0;
        __syncthreads();
        if (threadIdx.x == 0) {
            __threadfence();
            a.done[a.done_count + 1] = 0;  // abort flag
            a.done[a.done_count] = 0;      // exit counter
        }
    }
}

// the chain's tile shape of a layer, derived from its selected routine parameters
struct ChainShape {
    bool implicit;
    int BN, KB, BW, BH, BNI;
};

}  // namespace tc

// ------------------------------------------------------------------ host side
using tc::ChainLayer;

static int ilog2(int v) {
    int l = 0;
    while ((1 << l) < v) ++l;
    return l;
}

size_t chain_desc_bytes(int n_layers) { return (size_t)n_layers * sizeof(ChainLayer); }

cudaError_t chain_encode(const std::vector<ChainOp> &ops, std::vector<uint8_t> &blob, int32_t *total_units,
                         int32_t *done_count) {
    using namespace tc;
    std::vector<ChainLayer> L(ops.size());
    int32_t units = 0, tiles = 0;
    for (size_t i = 0; i < ops.size(); ++i) {
        const ChainOp &o = ops[i];
        ChainShape sh;
        if (!conv_tc_chain_shape(*o.layer, o.in, o.schema, o.variant, &sh.implicit, &sh.BN, &sh.KB, &sh.BW, &sh.BH,
                                 &sh.BNI))
            return cudaErrorInvalidValue;
        ChainLayer &c = L[i];
        std::memset(&c, 0, sizeof(c));
        const sn_conv_params &cp = o.layer->conv;
        c.N = (int)o.in.n, c.H = (int)o.in.h, c.W = (int)o.in.w, c.C = (int)o.in.c;
        c.K = cp.c_out, c.P = (int)o.layer->out.h, c.Q = (int)o.layer->out.w, c.R = cp.kh, c.S = cp.kw;
        c.stride = cp.sh, c.ph = cp.ph, c.pw = cp.pw, c.dh = cp.dh, c.dw = cp.dw;
        c.cblocks = (c.C + BK - 1) / BK;
        c.KB = sh.KB, c.BN = sh.BN, c.implicit = sh.implicit;
        if (c.cblocks % c.KB) return cudaErrorInvalidValue;
        c.kiters = c.R * c.S * c.cblocks / c.KB;
        c.act = cp.act;
        c.has_res = o.res != nullptr;
        c.bias = o.bias;
        c.src = o.src;
        c.res_src = o.res_src;
        const int64_t mout = (int64_t)c.N * c.P * c.Q;
        if (mout >= INT32_MAX - 256 || (int64_t)c.N * c.H * c.W >= INT32_MAX - 256) return cudaErrorInvalidValue;
        if (o.res && (uintptr_t)o.res % 16) return cudaErrorInvalidValue;
        c.Mout = (int32_t)mout;
        c.ntiles = (c.K + c.BN - 1) / c.BN;
        const int dt = o.schema.dtype;
        const uint64_t es = 2;
        const bool blk = c.KB > 1;
        const uint64_t CB = (uint64_t)c.cblocks;
        {  // B: weights [K][R*S][C]
            const uint64_t dims[4] = {blk ? 64 : (uint64_t)c.C, (uint64_t)(c.R * c.S), (uint64_t)c.K, CB};
            const uint64_t str[3] = {c.C * es, (uint64_t)c.R * c.S * c.C * es, 128};
            const uint32_t box[4] = {BK, 1, (uint32_t)c.BN, (uint32_t)c.KB};
            if (!tma_encode(&c.mB, dt, blk ? 4 : 3, o.wt, dims, str, box, CU_TENSOR_MAP_SWIZZLE_128B))
                return cudaErrorInvalidValue;
        }
        if (!c.implicit) {
            const uint64_t M = (uint64_t)c.N * c.H * c.W;
            const uint64_t dims[3] = {blk ? 64 : (uint64_t)c.C, M, CB};
            const uint64_t str[2] = {c.C * es, 128};
            const uint32_t box[3] = {BK, (uint32_t)BM, (uint32_t)c.KB};
            if (!tma_encode(&c.mA[0], dt, blk ? 3 : 2, o.in0, dims, str, box, CU_TENSOR_MAP_SWIZZLE_128B))
                return cudaErrorInvalidValue;
            c.mA[1] = c.mA[2] = c.mA[3] = c.mA[0];
            c.mtiles = (int)((mout + BM - 1) / BM);
            const uint64_t ydims[2] = {(uint64_t)c.K, (uint64_t)mout};
            const uint64_t ystr[1] = {c.K * es};
            const uint32_t ybox[2] = {64, 32};
            if (!tma_encode(&c.mY, dt, 2, o.out, ydims, ystr, ybox, CU_TENSOR_MAP_SWIZZLE_128B))
                return cudaErrorInvalidValue;
            c.mR = c.mY;
            if (o.res && !tma_encode(&c.mR, dt, 2, o.res, ydims, ystr, ybox, CU_TENSOR_MAP_SWIZZLE_128B))
                return cudaErrorInvalidValue;
            c.BW = c.BH = c.BNI = 1;
        } else {
            c.BW = sh.BW, c.BH = sh.BH, c.BNI = sh.BNI;
            if (c.BW * c.BH * c.BNI != BM) return cudaErrorInvalidValue;
            c.tq = (c.Q + c.BW - 1) / c.BW;
            c.tp = (c.P + c.BH - 1) / c.BH;
            const int tn = (c.N + c.BNI - 1) / c.BNI;
            const uint32_t box[5] = {BK, (uint32_t)c.BW, (uint32_t)c.BH, (uint32_t)c.BNI, (uint32_t)c.KB};
            const uint64_t c0dim = blk ? 64 : (uint64_t)c.C;
            if (c.stride == 1) {
                const uint64_t dims[5] = {c0dim, (uint64_t)c.W, (uint64_t)c.H, (uint64_t)c.N, CB};
                const uint64_t str[4] = {c.C * es, (uint64_t)c.W * c.C * es, (uint64_t)c.H * c.W * c.C * es, 128};
                if (!tma_encode(&c.mA[0], dt, blk ? 5 : 4, o.in0, dims, str, box, CU_TENSOR_MAP_SWIZZLE_128B))
                    return cudaErrorInvalidValue;
                c.mA[1] = c.mA[2] = c.mA[3] = c.mA[0];
            } else {
                if (c.stride != 2 || c.H % 2 || c.W % 2) return cudaErrorInvalidValue;
                for (int bh = 0; bh < 2; ++bh)
                    for (int bw = 0; bw < 2; ++bw) {
                        const char *base = static_cast<const char *>(o.in0) + ((int64_t)bh * c.W + bw) * c.C * es;
                        const uint64_t dims[5] = {c0dim, (uint64_t)(c.W / 2), (uint64_t)(c.H / 2), (uint64_t)c.N, CB};
                        const uint64_t str[4] = {2 * c.C * es, 2 * (uint64_t)c.W * c.C * es,
                                                 (uint64_t)c.H * c.W * c.C * es, 128};
                        if (!tma_encode(&c.mA[bh * 2 + bw], dt, blk ? 5 : 4, base, dims, str, box,
                                        CU_TENSOR_MAP_SWIZZLE_128B))
                            return cudaErrorInvalidValue;
                    }
            }
            c.mtiles = c.tq * c.tp * tn;
            const uint32_t sbw = (uint32_t)std::min(c.BW, 32);
            const uint32_t sbh = (uint32_t)std::min<int>(c.BH, 32 / sbw);
            const uint32_t sbn = 32 / (sbw * sbh);
            const uint64_t ydims[4] = {(uint64_t)c.K, (uint64_t)c.Q, (uint64_t)c.P, (uint64_t)c.N};
            const uint64_t ystr[3] = {c.K * es, (uint64_t)c.Q * c.K * es, (uint64_t)c.P * c.Q * c.K * es};
            const uint32_t ybox[4] = {64, sbw, sbh, sbn};
            if (!tma_encode(&c.mY, dt, 4, o.out, ydims, ystr, ybox, CU_TENSOR_MAP_SWIZZLE_128B))
                return cudaErrorInvalidValue;
            c.mR = c.mY;
            if (o.res && !tma_encode(&c.mR, dt, 4, o.res, ydims, ystr, ybox, CU_TENSOR_MAP_SWIZZLE_128B))
                return cudaErrorInvalidValue;
        }
        c.lbw = ilog2(c.BW), c.lbh = ilog2(c.BH), c.lbn = ilog2(c.BNI), c.lbwh = ilog2(c.BW * c.BH);
        if ((1 << c.lbw) != c.BW || (1 << c.lbh) != c.BH || (1 << c.lbn) != c.BNI) return cudaErrorInvalidValue;
        const int64_t lu = (int64_t)c.mtiles * c.ntiles;
        if (c.mtiles <= 0 || lu + units > INT32_MAX / 2 || (int64_t)tiles + c.mtiles > INT32_MAX / 2)
            return cudaErrorInvalidValue;
        c.unit_begin = units;
        c.unit_end = units + (int32_t)lu;
        units = c.unit_end;
        c.done_base = tiles;
        tiles += c.mtiles;
        c.done_target = c.ntiles * (c.BN == 64 ? EPI_WARPS / 2 : EPI_WARPS);
        c.fd_ntiles = make_fastdiv((uint32_t)c.ntiles);
        c.fd_tq = make_fastdiv((uint32_t)std::max(c.tq, 1));
        c.fd_tp = make_fastdiv((uint32_t)std::max(c.tp, 1));
        c.fd_spt = make_fastdiv((uint32_t)(c.cblocks / c.KB));
        c.fd_S = make_fastdiv((uint32_t)c.S);
        c.fd_PQ = make_fastdiv((uint32_t)(c.P * c.Q));
        c.fd_Q = make_fastdiv((uint32_t)c.Q);
        // a dependency must be an earlier layer of the chain
        if (c.src >= (int)i || c.res_src >= (int)i) return cudaErrorInvalidValue;
    }
    // the layers a unit waits on must tile their output the way the
    // dependency walk assumes: their pixel shapes are checked above; their
    // outputs must be what this layer reads
    for (size_t i = 0; i < ops.size(); ++i) {
        const ChainOp &o = ops[i];
        if (o.src >= 0) {
            const ChainLayer &p = L[o.src];
            if (p.N != L[i].N || p.P != L[i].H || p.Q != L[i].W || p.K != L[i].C) return cudaErrorInvalidValue;
        }
        if (o.res_src >= 0) {
            const ChainLayer &p = L[o.res_src];
            if (p.N != L[i].N || p.P != L[i].P || p.Q != L[i].Q || p.K != L[i].K) return cudaErrorInvalidValue;
        }
    }
    blob.resize(L.size() * sizeof(ChainLayer));
    std::memcpy(blob.data(), L.data(), blob.size());
    *total_units = units;
    *done_count = tiles;
    return cudaSuccess;
}

cudaError_t chain_launch(int dtype, const void *desc_dev, int32_t n_layers, int32_t total_units, int32_t *done_dev,
                         int32_t done_count, cudaStream_t st) {
    using namespace tc;
    if (!desc_dev || !done_dev || total_units <= 0 || (uintptr_t)desc_dev % 128) return cudaErrorInvalidValue;
    ChainArgs a;
    a.L = static_cast<const ChainLayer *>(desc_dev);
    a.n_layers = n_layers;
    a.total = total_units;
    a.done = done_dev;
    a.done_count = done_count;
    a.err = device_error_word();
    auto kern = dtype == SN_F16 ? conv_chain_kernel<__half> : conv_chain_kernel<__nv_bfloat16>;
    static bool attr_set[2] = {false, false};
    bool &set = attr_set[dtype == SN_F16 ? 0 : 1];
    if (!set) {
        cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)CH_SMEM);
        if (e != cudaSuccess) return e;
        set = true;
    }
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr[1];
    cfg.gridDim = dim3((unsigned)std::min(total_units, num_sms()));
    cfg.blockDim = dim3(THREADS);
    cfg.dynamicSmemBytes = CH_SMEM;
    cfg.stream = st;
    // every CTA resident at once: the units' waits on one another need it
    attr[0].id = cudaLaunchAttributeCooperative;
    attr[0].val.cooperative = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kern, a);
}

}  // namespace k
}  // namespace sn
