// Host side of the tensor-core convolution (implicit GEMM on tcgen05; the
// kernel is in tc_conv.cuh): routine-parameter combinations, tensor maps,
// dispatch, and the childnet routines built on the same GEMM.
#include <cuda.h>

#include <algorithm>
#include <cstdio>
#include <mutex>
#include <string>
#include <type_traits>
#include <vector>

#include "tc_conv.cuh"

namespace sn {
namespace k {

namespace tc {

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
    int sk = 0;        // 1: stream-K, one equal range of the tiles' K steps per SM
    int halo = 0;      // 1: 3x3 stride 1, 8 x 16 pixel tiles, one A box per row of taps
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
    // stream-K for layers whose tile count falls badly against the SM count
    // (fewer than three waves, not a whole number of them): the tiles' K
    // steps are cut into one equal range per SM; appended after every other
    // combination, so that the earlier ones keep their indices
    auto push_sk = [&](Config cf, int64_t mtiles) {
        for (int bn : bns)
            if (bn >= 128)
                for (int kb : {1, 2}) {
                    if (kb == 2 && (bn != 128 || c.c_in % 128)) continue;
                    const int64_t tiles = mtiles * ((K + bn - 1) / bn);
                    if (tiles % kSmCount == 0 || tiles > 3 * kSmCount || kiters / kb < 4) continue;
                    cf.BN = bn, cf.G = 1, cf.KB = kb, cf.ksplit = 1, cf.sk = 1;
                    out.push_back(cf);
                }
    };
    if (plain && a_blocks == 0) {
        push_all({false, 0, 0, 0, 0, 1, 1, 1}, (N * P * Q + BM - 1) / BM);
        push_bst({false, 0, 0, 0, 0, 1, 1, 1});
        push_ms2({false, 0, 0, 0, 0, 1, 1, 1}, (N * P * Q + 2 * BM - 1) / (2 * BM));
        push_csk({false, 0, 0, 0, 0, 1, 1, 1}, (N * P * Q + BM - 1) / BM);
        push_sk({false, 0, 0, 0, 0, 1, 1, 1}, (N * P * Q + BM - 1) / BM);
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
    if (a_blocks == 0) {
        for (const Geo &gg : geos(2 * BM)) push_ms2({true, 0, gg.bw, gg.bh, gg.bni, 1, 1, 1}, tiles_of(gg));
        for (const Geo &gg : geos(BM)) push_sk({true, 0, gg.bw, gg.bh, gg.bni, 1, 1, 1}, tiles_of(gg));
        // halo tiles for 3x3 stride-1 layers (appended last, like stream-K):
        // one CTA per tile (BN <= 128), and CTA pairs that share B
        if (c.kh == 3 && c.kw == 3 && c.sh == 1 && c.dh == 1 && c.dw == 1) {
            for (int bn : bns)
                if (bn <= 128) {
                    Config cf{true, bn, HALO_BW, HALO_BH, 1, 1, 1, 1};
                    cf.halo = 1;
                    out.push_back(cf);
                }
            for (int bn : bns) {
                Config cf{true, bn, HALO_BW, HALO_BH, 1, 1, 2, 1};
                cf.halo = 1;
                out.push_back(cf);
            }
        }
    }
    return out;
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
        snprintf(b, sizeof(b), "bn=%d cta=%d kb=%d rows=%d ksplit=%d bst=%d csk=%d%s tile=%dx%dx%d", c.BN, c.G,
                 c.KB, 128 * c.ms * c.G, c.ksplit, c.bst ? 1 : 0, c.csk,
                 c.sk ? " streamk" : c.halo ? " halo" : "", c.BW, c.BH, c.BNI);
    else
        snprintf(b, sizeof(b), "bn=%d cta=%d kb=%d rows=%d ksplit=%d bst=%d csk=%d%s plain", c.BN, c.G, c.KB,
                 128 * c.ms * c.G, c.ksplit, c.bst ? 1 : 0, c.csk, c.sk ? " streamk" : "");
    return b;
}

bool conv_tc_nchw_ok(const Layer &l, const Shape &in, sn_schema s, int32_t v) {
    const std::vector<tc::Config> cfgs = tc::configs(l, in, s);
    return v >= 0 && v < (int)cfgs.size() && cfgs[v].ksplit == 1 && !cfgs[v].sk;
}

size_t conv_tc_ws(const Layer &l, const Shape &in, sn_schema s, int32_t v, int32_t a_blocks) {
    const std::vector<tc::Config> cfgs = tc::configs(l, in, s, a_blocks);
    if (v < 0 || v >= (int)cfgs.size()) return 0;
    // stream-K: two fp32 partial-tile slots per CTA, at most one CTA per SM
    if (cfgs[v].sk) return (size_t)2 * num_sms() * tc::BM * cfgs[v].BN * sizeof(float);
    if (cfgs[v].ksplit == 1) return 0;
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
    // the prepared weights [K][R*S][C] (16-byte multiple: C is a multiple of
    // 8); none for the space-to-depth form, whose weights have another layout
    p.wt = a.wt;
    p.wt_bytes = (uintptr_t)a.wt % 16 == 0 && a.a_blocks == 0 ? (int64_t)c.c_out * c.kh * c.kw * in.c * 2 : 0;
    if (p.wt_bytes >= ((int64_t)1 << 32) * 64) p.wt_bytes = 0;  // slices stay below 4 GB
    // a routine that writes the next layer's layout: the same dtype in NCHW
    // (one CTA's epilogue per tile, so no K split through fp32 partials)
    p.y_nchw = 0;
    if (a.out_schema.dtype >= 0 && !schema_eq(a.out_schema, a.schema)) {
        if (a.out_schema.dtype != a.schema.dtype || a.out_schema.layout != SN_NCHW || cf.ksplit != 1 || cf.sk)
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
    if (cf.sk) {
        const size_t need = (size_t)2 * num_sms() * BM * cf.BN * sizeof(float);
        if (!a.ws || a.ws_bytes < need || (uintptr_t)a.ws % 16 || !a.tile_counts) return cudaErrorInvalidValue;
        p.sk_part = static_cast<float *>(a.ws);
        p.sk_count = a.tile_counts;
    }
    const int dt = a.schema.dtype;
    const uint64_t es = 2;
    CUtensorMap mA[4], mB, mY, mR;
    // KB > 1 (channels a multiple of 128): every map gets an outermost
    // channel-block axis of stride 128 B over the 64-channel inner axis, so that
    // one box lands KB consecutive 128-B-row blocks in shared memory
    const bool blk = cf.KB > 1;
    const uint64_t CB = (uint64_t)p.cblocks;
    if (cf.halo) {
        // halo tiles: a K step is one row of three taps of one channel block
        if (p.R != 3 || p.S != 3 || p.stride != 1 || p.dh != 1 || p.dw != 1 || cf.KB != 1 || cf.ms != 1)
            return cudaErrorInvalidValue;
        p.kiters = p.R * p.cblocks;
        {  // B: weights [K][R*S][C] read as [R*S][K][C], one box = a row's three taps x BN x 64
            const uint64_t dims[3] = {(uint64_t)p.C, (uint64_t)p.K, (uint64_t)(p.R * p.S)};
            const uint64_t str[2] = {(uint64_t)p.R * p.S * p.C * es, p.C * es};
            const uint32_t box[3] = {BK, (uint32_t)(cf.BN / cf.G), 3};  // a CTA's share of the BN rows
            if (!encode(&mB, dt, 3, a.wt, dims, str, box)) return cudaErrorInvalidValue;
        }
        {  // A: [N][H][W][C], one box = 16 rows x 10 columns of one image
            const uint64_t dims[4] = {(uint64_t)p.C, (uint64_t)p.W, (uint64_t)p.H, (uint64_t)p.N};
            const uint64_t str[3] = {p.C * es, (uint64_t)p.W * p.C * es, (uint64_t)p.H * p.W * p.C * es};
            const uint32_t box[4] = {BK, (uint32_t)HALO_W, (uint32_t)HALO_BH, 1};
            if (!encode(&mA[0], dt, 4, a.in[0], dims, str, box)) return cudaErrorInvalidValue;
            mA[1] = mA[2] = mA[3] = mA[0];
        }
    } else {  // B: weights [K][R*S][C]
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
        if (cf.halo) {
            // A was encoded above (one box per row of taps)
        } else if (p.stride == 1) {
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
    if (cf.sk) {
        // every SM one range of ceil(steps / SMs) K steps; one counter per
        // (tile, epilogue warp) in the caller's zeroed counter array
        const int64_t tiles = (int64_t)p.mtiles * p.ntiles, steps = tiles * p.kiters;
        if (steps + p.kiters > INT32_MAX || tiles * EPI_WARPS > (int64_t)a.tile_counts_n) return cudaErrorNotSupported;
        const int nsm = num_sms();
        p.sk_steps = (int32_t)steps;
        p.sk_len = (int32_t)((steps + nsm - 1) / nsm);
    }
    p.fd_ksplit = make_fastdiv((uint32_t)p.ksplit);
    p.fd_ntiles = make_fastdiv((uint32_t)p.ntiles);
    p.fd_tq = make_fastdiv((uint32_t)std::max(p.tq, 1));
    p.fd_tp = make_fastdiv((uint32_t)std::max(p.tp, 1));
    p.fd_spt = make_fastdiv((uint32_t)(p.cblocks / cf.KB));
    p.fd_S = make_fastdiv((uint32_t)(cf.halo ? 1 : p.S));  // halo: a K step's "tap" is a row of taps
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
    if (cf.halo) return launch_halo(dt, cf.BN, cf.G, mA, mB, mY, mR, p, a.stream);                 \
    if (cf.sk) {                                                                                    \
        if (cf.G != 1 || cf.ms != 1 || cf.bst || cf.ksplit != 1 || cf.csk != 1) return cudaErrorInvalidValue; \
        return launch_sk(dt, cf.BN, cf.KB, cf.implicit, mA, mB, mY, mR, p, a.stream);              \
    }                                                                                               \
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
           s.dtype != SN_QI8;  // input in either layout (the re-layout reads both)
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
    if (!s2d_applies(l, s)) return 0;  // the GEMM on X is NHWC-like whatever the input layout
    return (int32_t)tc::configs(s2d_gemm_layer(l), s2d_gemm_in(l), sn_schema{s.dtype, SN_NHWC}, s2d_rows(l)).size();
}

size_t conv_s2d_tc_ws(const Layer &l, const Shape &in, sn_schema s, int32_t v) {
    (void)in;
    return s2d_bytes(l, s) + conv_tc_ws(s2d_gemm_layer(l), s2d_gemm_in(l), sn_schema{s.dtype, SN_NHWC}, v, s2d_rows(l));
}

// X[n][u][v][16]: one thread per X pixel, two 16-byte stores; the input is
// NHWC, or NCHW (NCHW_IN: the layout change fused into the re-layout, so an
// NCHW net input needs no separate adapt)
template <typename T, bool NCHW_IN>
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
            if (NCHW_IN) {
                const T *xp = x + (n * d.C * d.H + h) * d.W + w;
                for (int c = 0; c < d.C; ++c) po[ij * d.C + c] = xp[(int64_t)c * d.H * d.W];
            } else {
                const T *xp = x + ((n * d.H + h) * d.W + w) * d.C;
                for (int c = 0; c < d.C; ++c) po[ij * d.C + c] = xp[c];
            }
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
        if (a.schema.layout == SN_NCHW) {
            SN_DT_SWITCH(a.schema.dtype, T,
                         launch_pdl(s2d_kernel<T, true>, grid_for(total, 256), 256, 0, a.stream, (const T *)a.in[0],
                                    (T *)a.ws, d));
        } else {
            SN_DT_SWITCH(a.schema.dtype, T,
                         launch_pdl(s2d_kernel<T, false>, grid_for(total, 256), 256, 0, a.stream, (const T *)a.in[0],
                                    (T *)a.ws, d));
        }
        cudaError_t e = cudaGetLastError();
        if (e != cudaSuccess || stage == 0) return e;
    }
    const Layer gl = s2d_gemm_layer(l);
    LaunchArgs g = a;
    g.layer = &gl;
    g.routine = R_CONV_TC;
    // the GEMM reads X (its own layout) and writes the output in the
    // candidate's written schema: NHWC, or NCHW through the NCHW epilogue
    g.schema = sn_schema{a.schema.dtype, SN_NHWC};
    g.out_schema = a.out_schema.dtype >= 0 ? a.out_schema : a.schema;
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
