// Depthwise 3x3 convolution, NHWC f16/bf16, with the input rows staged in
// shared memory by TMA: the shared-memory routine parameter of the direct
// depthwise routine (section III-B: a routine's parameters are part of what
// the profiler chooses among).
//
// A persistent CTA owns a contiguous range of output rows in (image, channel
// slice, row) order.  One producer thread walks the input rows that range
// reads, in order, and copies each (all W + halo columns of one channel
// slice, zero-filled outside the image by the TMA unit) into the next slot of
// a ring; fifteen consumer warps take the range's output vectors in rounds of
// one per thread, each warp at its own pace, and release the rows no later
// round needs.  Each input row crosses HBM -> shared memory once per range,
// so the kernel reads the input about once and writes the output once: the
// HBM floor of the operation.
#include <algorithm>
#include <type_traits>

#include "tc_common.cuh"

namespace sn {
namespace k {

namespace {

using tc::mbar_arrive;
using tc::mbar_expect_tx;
using tc::mbar_init;
using tc::mbar_wait;
using tc::su32;

constexpr int DW_CONSUMER_WARPS = 15;  // with the producer warp: 4 warps per SM sub-partition, 128 registers
constexpr int DW_CONSUMERS = 32 * DW_CONSUMER_WARPS;
constexpr int DW_THREADS = 32 + DW_CONSUMERS;
constexpr int ERR_DW_WAIT = 0x100;
constexpr int DW_MAX_SLOTS = 32;

struct DwRing {
    int32_t H, C, P, Q, ph, pw, act;
    int32_t CS, nslices, WB;  // channel slice; input columns per row (box width)
    int32_t QBLK, CVS;        // column blocks; 16-byte channel vectors per slice
    int32_t rows_total, NS;   // output rows N * nslices * P; ring slots
    uint32_t box_bytes;   // one row of one slice: WB * CS elements
    uint32_t slot_bytes;  // slot stride: box_bytes rounded up to the 128-byte alignment of a TMA destination
    FastDiv fd_P, fd_nslices, fd_NS, fd_CVS, fd_row_items;
    const float *bias;
    int *err;
};

// a run of output rows [pA, pB) of image n, channel slice sl, inside one
// CTA's range, and the input rows [hlo, hhi) it reads
struct Seg {
    int n, sl, pA, pB, hlo, hhi;
};

template <int SW>
__device__ __forceinline__ Seg seg_at(const DwRing &p, int f, int f1) {
    Seg s;
    const int ns = (int)fdiv((uint32_t)f, p.fd_P);
    s.pA = f - ns * p.P;
    s.pB = min(p.P, s.pA + (f1 - f));
    s.n = (int)fdiv((uint32_t)ns, p.fd_nslices);
    s.sl = ns - s.n * p.nslices;
    s.hlo = max(s.pA * SW - p.ph, 0);
    s.hhi = min((s.pB - 1) * SW - p.ph + 3, p.H);
    return s;
}

__device__ __forceinline__ uint32_t slot_of(uint32_t i, const DwRing &p) { return i - fdiv(i, p.fd_NS) * p.NS; }

template <typename T, int SW, int QB>
__global__ void __launch_bounds__(DW_THREADS, 1)
    dw3_nhwc_ring(const __grid_constant__ CUtensorMap mx, const T *__restrict__ w, T *__restrict__ y, const DwRing p) {
    extern __shared__ __align__(128) uint8_t smem[];
    uint64_t *full = reinterpret_cast<uint64_t *>(smem);
    uint64_t *empty = full + DW_MAX_SLOTS;
    // ring slots start on a 128-byte boundary (TMA destinations must)
    uint8_t *ring = smem + ((su32(smem) + 2 * DW_MAX_SLOTS * 8 + 127u) & ~127u) - su32(smem);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (threadIdx.x == 0) {
        asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&mx)) : "memory");
        for (int i = 0; i < p.NS; ++i) {
            mbar_init(&full[i], 1);
            mbar_init(&empty[i], DW_CONSUMER_WARPS);
        }
        tc::fence_mbar_init();
    }
    __syncthreads();
    griddep_launch();
    griddep_wait();
    const int f0 = (int)((int64_t)blockIdx.x * p.rows_total / gridDim.x);
    const int f1 = (int)((int64_t)(blockIdx.x + 1) * p.rows_total / gridDim.x);

    if (warp == 0) {
        // ---------------------------------------------------------- producer
        if (lane != 0) return;
        uint32_t L = 0;  // rows issued so far; row i goes to slot i % NS
        bool ok = true;
        for (int f = f0; f < f1 && ok;) {
            const Seg s = seg_at<SW>(p, f, f1);
            for (int h = s.hlo; h < s.hhi; ++h, ++L) {
                const uint32_t use = fdiv(L, p.fd_NS), slot = L - use * p.NS;
                if (use > 0 && !mbar_wait(&empty[slot], (use - 1) & 1)) {
                    ok = false;
                    break;
                }
                mbar_expect_tx(&full[slot], p.box_bytes);
                tc::tma_4d<1>(su32(ring + slot * p.slot_bytes), &mx, su32(&full[slot]), s.sl * p.CS, -p.pw, h, s.n);
            }
            f += s.pB - s.pA;
        }
        if (!ok) atomicOr(p.err, ERR_DW_WAIT);
        // every issued copy has landed before this CTA may exit
        for (uint32_t i = L > (uint32_t)p.NS ? L - p.NS : 0; i < L; ++i) {
            const uint32_t use = fdiv(i, p.fd_NS);
            if (!mbar_wait(&full[i - use * p.NS], use & 1)) {
                atomicOr(p.err, ERR_DW_WAIT);
                break;
            }
        }
        return;
    }

    // -------------------------------------------------------------- consumers
    constexpr int E = 16 / (int)sizeof(T);
    constexpr int WN = (QB - 1) * SW + 3;  // input columns behind QB outputs
    const int ct = threadIdx.x - 32;
    const T *ringT = reinterpret_cast<const T *>(ring);
    const uint32_t slot_elems = p.slot_bytes / (uint32_t)sizeof(T);
    const int row_items = p.QBLK * p.CVS;
    uint32_t L = 0;  // index of the current segment's first input row
    for (int f = f0; f < f1;) {
        const Seg s = seg_at<SW>(p, f, f1);
        const int nl = max(0, s.hhi - s.hlo);
        int waited = 0, released = 0;
        // the segment's items (output row, column block, channel vector),
        // row-major, in rounds of one item per consumer thread; a warp moves
        // to its next round as soon as the rows it needs have landed
        const int total = (s.pB - s.pA) * row_items;
        for (int base = 0; base < total; base += DW_CONSUMERS) {
            const int last = min(total, base + DW_CONSUMERS) - 1;
            const int prow = s.pA + (int)fdiv((uint32_t)last, p.fd_row_items);
            const int need = min(s.hhi, prow * SW - p.ph + 3) - s.hlo;
            for (; waited < need; ++waited) {
                const uint32_t i = L + waited, use = fdiv(i, p.fd_NS);
                if (!mbar_wait(&full[i - use * p.NS], use & 1)) {
                    atomicOr(p.err, ERR_DW_WAIT);
                    return;
                }
            }
            if (base + ct < total) {
                const int it = base + ct;
                const int j = (int)fdiv((uint32_t)it, p.fd_row_items);
                const int rem = it - j * row_items;
                const int qb = (int)fdiv((uint32_t)rem, p.fd_CVS);
                const int cl = (rem - qb * p.CVS) * E;  // channel within the slice
                const int c0 = s.sl * p.CS + cl;
                const int pp = s.pA + j, q0 = qb * QB;
                uint4 wt[9];  // the item's nine taps, fetched together
#pragma unroll
                for (int t = 0; t < 9; ++t) wt[t] = *reinterpret_cast<const uint4 *>(w + t * p.C + c0);
                T *yrow = y + ((int64_t)(s.n * p.P + pp) * p.Q) * p.C + c0;
                if constexpr (std::is_same<T, __half>::value) {
                    // fp16: packed half2 multiply-adds (two channels per
                    // instruction) accumulating in fp16, half the issue slots
                    // of the widening fp32 path
                    const float4 b0 = *reinterpret_cast<const float4 *>(p.bias + c0);
                    const float4 b1 = *reinterpret_cast<const float4 *>(p.bias + c0 + 4);
                    const __half2 hb[4] = {__floats2half2_rn(b0.x, b0.y), __floats2half2_rn(b0.z, b0.w),
                                           __floats2half2_rn(b1.x, b1.y), __floats2half2_rn(b1.z, b1.w)};
                    __half2 hacc[QB][4];
#pragma unroll
                    for (int q = 0; q < QB; ++q)
#pragma unroll
                        for (int k = 0; k < 4; ++k) hacc[q][k] = hb[k];
#pragma unroll
                    for (int r = 0; r < 3; ++r) {
                        const int h = pp * SW - p.ph + r;
                        if (h < s.hlo || h >= s.hhi) continue;  // zero padding
                        const T *row = ringT + slot_of(L + (h - s.hlo), p) * slot_elems + cl;
                        uint4 win[WN];
#pragma unroll
                        for (int t = 0; t < WN; ++t) {
                            const int col = q0 * SW + t;
                            win[t] = col < p.WB ? *reinterpret_cast<const uint4 *>(row + col * p.CS)
                                                : make_uint4(0u, 0u, 0u, 0u);
                        }
#pragma unroll
                        for (int sx = 0; sx < 3; ++sx) {
                            const __half2 *wq = reinterpret_cast<const __half2 *>(&wt[r * 3 + sx]);
#pragma unroll
                            for (int q = 0; q < QB; ++q) {
                                const __half2 *xv = reinterpret_cast<const __half2 *>(&win[q * SW + sx]);
#pragma unroll
                                for (int k = 0; k < 4; ++k) hacc[q][k] = __hfma2(xv[k], wq[k], hacc[q][k]);
                            }
                        }
                    }
                    const __half2 z2 = __float2half2_rn(0.0f), six2 = __float2half2_rn(6.0f);
#pragma unroll
                    for (int q = 0; q < QB; ++q) {
                        if (q0 + q >= p.Q) break;
                        uint4 o;
                        __half2 *oh = reinterpret_cast<__half2 *>(&o);
#pragma unroll
                        for (int k = 0; k < 4; ++k) {
                            __half2 v = hacc[q][k];
                            if (p.act == SN_ACT_RELU) {
                                v = __hmax2(v, z2);
                            } else if (p.act == SN_ACT_RELU6) {
                                v = __hmin2(__hmax2(v, z2), six2);
                            } else if (p.act != SN_ACT_NONE) {
                                const float2 f = __half22float2(v);
                                v = __floats2half2_rn(act_apply(f.x, p.act), act_apply(f.y, p.act));
                            }
                            oh[k] = v;
                        }
                        *reinterpret_cast<uint4 *>(yrow + (int64_t)(q0 + q) * p.C) = o;
                    }
                } else {
                float acc[QB][E];
                {
                    const float4 b0 = *reinterpret_cast<const float4 *>(p.bias + c0);
                    const float4 b1 = *reinterpret_cast<const float4 *>(p.bias + c0 + 4);
                    const float bb[8] = {b0.x, b0.y, b0.z, b0.w, b1.x, b1.y, b1.z, b1.w};
#pragma unroll
                    for (int q = 0; q < QB; ++q)
#pragma unroll
                        for (int e = 0; e < E; ++e) acc[q][e] = bb[e];
                }
#pragma unroll
                for (int r = 0; r < 3; ++r) {
                    const int h = pp * SW - p.ph + r;
                    if (h < s.hlo || h >= s.hhi) continue;  // zero padding
                    const T *row = ringT + slot_of(L + (h - s.hlo), p) * slot_elems + cl;
                    uint4 win[WN];
#pragma unroll
                    for (int t = 0; t < WN; ++t) {
                        const int col = q0 * SW + t;
                        win[t] = col < p.WB ? *reinterpret_cast<const uint4 *>(row + col * p.CS)
                                            : make_uint4(0u, 0u, 0u, 0u);
                    }
#pragma unroll
                    for (int sx = 0; sx < 3; ++sx) {
                        const uint4 wq = wt[r * 3 + sx];
#pragma unroll
                        for (int q = 0; q < QB; ++q) {
                            const uint4 xv = win[q * SW + sx];
                            mac2<T>(acc[q][0], acc[q][1], xv.x, wq.x);
                            mac2<T>(acc[q][2], acc[q][3], xv.y, wq.y);
                            mac2<T>(acc[q][4], acc[q][5], xv.z, wq.z);
                            mac2<T>(acc[q][6], acc[q][7], xv.w, wq.w);
                        }
                    }
                }
#pragma unroll
                for (int q = 0; q < QB; ++q) {
                    if (q0 + q >= p.Q) break;
                    uint4 o;
                    o.x = tc::pack2<T>(act_apply(acc[q][0], p.act), act_apply(acc[q][1], p.act));
                    o.y = tc::pack2<T>(act_apply(acc[q][2], p.act), act_apply(acc[q][3], p.act));
                    o.z = tc::pack2<T>(act_apply(acc[q][4], p.act), act_apply(acc[q][5], p.act));
                    o.w = tc::pack2<T>(act_apply(acc[q][6], p.act), act_apply(acc[q][7], p.act));
                    *reinterpret_cast<uint4 *>(yrow + (int64_t)(q0 + q) * p.C) = o;
                }
                }  // fp32-accumulating path
            }
            // rows below the next round's first input row are done with
            const int nrow = base + DW_CONSUMERS < total
                                 ? s.pA + (int)fdiv((uint32_t)(base + DW_CONSUMERS), p.fd_row_items)
                                 : s.pB;
            const int freed = min(s.hhi, nrow * SW - p.ph) - s.hlo;
            __syncwarp();
            if (lane == 0)
                for (int i = released; i < freed; ++i) mbar_arrive(&empty[slot_of(L + i, p)]);
            released = max(released, freed);
        }
        __syncwarp();
        if (lane == 0)
            for (int i = released; i < nl; ++i) mbar_arrive(&empty[slot_of(L + i, p)]);
        L += nl;
        f += s.pB - s.pA;
    }
}

struct RingPlan {
    int CS, QB, NS;
    double score;
};

// input rows one round of DW_CONSUMERS consecutive items can touch
inline int round_rows(int row_items, int sw) {
    const int span = (DW_CONSUMERS + row_items - 1) / row_items + 1;  // output rows
    return (span - 1) * sw + 3;
}

// routine parameters of one launch: channel slice CS (a divisor of C, at most
// 256 channels: the TMA box limit), QB columns per thread and the ring depth
// (one CTA per SM with a ~200 KB ring).  A round's rows must fit the ring
// with rows to spare for prefetch; whole-channel rows are preferred, since a
// slice reads each pixel's channels in pieces, which costs DRAM efficiency.
RingPlan plan_ring(const ConvDims &d, int es, bool packed) {
    RingPlan best{0, 0, 0, -1.0};
    const int E = 16 / es;
    const int WB = (d.Q - 1) * d.sw + 3;
    const size_t budget = 200 * 1024;
    for (int CS = std::min(d.C, 256) / E * E; CS >= E; CS -= E) {
        if (d.C % CS) continue;
        const size_t slot = ((size_t)WB * CS * es + 127) & ~(size_t)127;
        const int NS = (int)std::min<size_t>(DW_MAX_SLOTS, budget / slot);
        for (int QB : {8, 4, 2, 1}) {
            // the fp32 accumulators of 4 columns at stride 2 (a 9-column window),
            // or of 8 columns, do not fit the register budget; packed half2
            // accumulators (fp16) take half the registers
            if (QB == 8 && !(packed && d.sw == 1)) continue;
            if (QB == 4 && d.sw == 2 && !packed) continue;
            const int QBLK = (d.Q + QB - 1) / QB;
            const double colutil = (double)d.Q / (QBLK * QB);
            const int need = std::min(round_rows(QBLK * (CS / E), d.sw), std::min(d.H, (d.P - 1) * d.sw + 3));
            if (NS < need + 1) continue;
            const double spare = std::min(1.0, 0.5 + 0.125 * (NS - need));  // prefetch depth
            const double score =
                colutil * (QB == 8 ? 1.02 : QB == 4 ? 1.0 : QB == 2 ? 0.96 : 0.9) * spare * (CS == d.C ? 1.0 : 0.85);
            if (score > best.score) best = RingPlan{CS, QB, NS, score};
        }
    }
    return best;
}

template <typename T, int SW, int QB>
cudaError_t launch_ring(const CUtensorMap &mx, const T *w, T *y, const DwRing &p, int grid, size_t smem,
                        cudaStream_t st) {
    static bool attr = false;
    if (!attr) {
        cudaError_t e = cudaFuncSetAttribute(dw3_nhwc_ring<T, SW, QB>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             227 * 1024);
        if (e != cudaSuccess) return e;
        attr = true;
    }
    const cudaError_t e = launch_pdl(dw3_nhwc_ring<T, SW, QB>, (unsigned)grid, DW_THREADS, smem, st, mx, w, y, p);
    return e != cudaSuccess ? e : cudaGetLastError();
}

template <typename T>
cudaError_t dispatch_ring(const CUtensorMap &mx, const LaunchArgs &a, const DwRing &p, int QB, int SW, int grid,
                          size_t smem) {
    const T *w = (const T *)a.wt;
    T *y = (T *)a.out;
    if constexpr (std::is_same<T, __half>::value) {
        if (SW == 1 && QB == 8) return launch_ring<T, 1, 8>(mx, w, y, p, grid, smem, a.stream);
        if (SW == 2 && QB == 4) return launch_ring<T, 2, 4>(mx, w, y, p, grid, smem, a.stream);
    }
    if (SW == 1) {
        if (QB == 4) return launch_ring<T, 1, 4>(mx, w, y, p, grid, smem, a.stream);
        if (QB == 2) return launch_ring<T, 1, 2>(mx, w, y, p, grid, smem, a.stream);
        return launch_ring<T, 1, 1>(mx, w, y, p, grid, smem, a.stream);
    }
    if (QB == 2) return launch_ring<T, 2, 2>(mx, w, y, p, grid, smem, a.stream);
    return launch_ring<T, 2, 1>(mx, w, y, p, grid, smem, a.stream);
}

}  // namespace

bool dw3_ring_applies(const LaunchArgs &a, const ConvDims &d) {
    const int es = dtype_size(a.schema.dtype);
    if (a.schema.dtype == SN_F32 || a.schema.layout != SN_NHWC) return false;
    if (d.R != 3 || d.S != 3 || d.dh != 1 || d.dw != 1 || d.sh != d.sw || (d.sw != 1 && d.sw != 2)) return false;
    if (d.groups != d.C || d.K != d.C || (d.C * es) % 16 != 0) return false;
    if ((uintptr_t)a.in[0] % 16 || (uintptr_t)a.out % 16 || (uintptr_t)a.wt % 16 || (uintptr_t)a.bias % 16)
        return false;
    if ((d.Q - 1) * d.sw + 3 > 256 || d.W > 65535 || d.H > 65535) return false;
    return (int64_t)d.N * d.C / (16 / es) * d.P < ((int64_t)1 << 30);
}

cudaError_t dw3_nhwc_ring(const LaunchArgs &a, const ConvDims &d) {
    if (!dw3_ring_applies(a, d)) return cudaErrorNotSupported;
    const int es = dtype_size(a.schema.dtype);
    const int WB = (d.Q - 1) * d.sw + 3;
    const size_t hdr = 2 * DW_MAX_SLOTS * 8 + 128;  // barriers and alignment slack
    const RingPlan pl = plan_ring(d, es, a.schema.dtype == SN_F16);
    if (pl.score < 0) return cudaErrorNotSupported;
    DwRing p{};
    p.H = d.H;
    p.C = d.C;
    p.P = d.P;
    p.Q = d.Q;
    p.ph = d.ph;
    p.pw = d.pw;
    p.act = d.act;
    p.CS = pl.CS;
    p.nslices = d.C / pl.CS;
    p.WB = WB;
    p.QBLK = (d.Q + pl.QB - 1) / pl.QB;
    p.CVS = pl.CS / (16 / es);
    p.rows_total = d.N * p.nslices * d.P;
    p.NS = pl.NS;
    p.box_bytes = (uint32_t)((size_t)WB * pl.CS * es);
    p.slot_bytes = (p.box_bytes + 127u) & ~127u;
    p.fd_P = make_fastdiv((uint32_t)d.P);
    p.fd_nslices = make_fastdiv((uint32_t)p.nslices);
    p.fd_NS = make_fastdiv((uint32_t)p.NS);
    p.fd_CVS = make_fastdiv((uint32_t)p.CVS);
    p.fd_row_items = make_fastdiv((uint32_t)(p.QBLK * p.CVS));
    p.bias = a.bias;
    p.err = device_error_word();
    // input as a 4-D tensor {C, W, H, N}; one box = one row of one slice with
    // the padding columns (starts at column -pw; rows outside are never asked)
    const uint64_t dims[4] = {(uint64_t)d.C, (uint64_t)d.W, (uint64_t)d.H, (uint64_t)d.N};
    const uint64_t strides[3] = {(uint64_t)d.C * es, (uint64_t)d.W * d.C * es, (uint64_t)d.H * d.W * d.C * es};
    const uint32_t box[4] = {(uint32_t)pl.CS, (uint32_t)WB, 1, 1};
    CUtensorMap mx;
    if (!tc::tma_encode(&mx, a.schema.dtype, 4, a.in[0], dims, strides, box, CU_TENSOR_MAP_SWIZZLE_NONE))
        return cudaErrorNotSupported;
    const int grid = (int)std::min<int64_t>(p.rows_total, (int64_t)num_sms());
    const size_t smem = hdr + (size_t)p.NS * p.slot_bytes;
    if (a.schema.dtype == SN_F16)
        return dispatch_ring<__half>(mx, a, p, pl.QB, d.sw, grid, smem);
    return dispatch_ring<__nv_bfloat16>(mx, a, p, pl.QB, d.sw, grid, smem);
}

}  // namespace k
}  // namespace sn
