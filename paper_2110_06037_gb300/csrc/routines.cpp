// Routine registry (section III-C): which routines can serve a layer in a
// schema, their routine-parameter combinations ("variants"), the weight
// format each expects, and dispatch to the kernels.
//
// Every routine reads its inputs and writes its output in its own schema;
// conversions between schemas are separate adapt routines on the edges.
#include <string>

#include "sn_internal.h"

namespace sn {

const char *routine_name(int32_t r) {
    switch (r) {
    case R_IO: return "io";
    case R_CONV_DIRECT: return "conv2/direct";
    case R_CONV_IGEMM: return "conv2/igemm_simt";
    case R_CONV_WINO: return "conv2/wino_f2x2_3x3";
    case R_CONV_WINO4: return "conv2/wino_f4x4_3x3";
    case R_CONV_WINO6: return "conv2/wino_f6x6_3x3";
    case R_CONV_TC: return "conv2/igemm_tc";
    case R_DW_DIRECT: return "dwconv2/direct";
    case R_MAXPOOL: return "maxpool/direct";
    case R_GAP: return "gap/reduce";
    case R_ADD: return "add/eltwise";
    case R_MUL: return "mul/eltwise";
    case R_DENSE: return "dense/simt";
    case R_ADAPT: return "adapt/convert";
    case R_CONV_IM2COL_TC: return "conv2/im2col_tc";
    case R_DENSE_TC: return "dense/gemm_tc";
    case R_CONV_S2D_TC: return "conv2/s2d_tc";
    case R_CONV_DP4A: return "conv2/igemm_dp4a";
    default: return nullptr;
    }
}

const char *variant_name(int32_t r, int32_t v) {
    switch (r) {
    case R_CONV_IGEMM: return v == 0 ? "tile=64x64" : "tile=128x64";
    case R_CONV_WINO: return v == 0 ? "gemm=simt" : "gemm=tc";
    case R_DW_DIRECT: return v == 0 ? "nhwc:window|nchw:rows" : v == 1 ? "nhwc:tma_rows|nchw:plane_tile" : "nhwc:band";
    case R_CONV_TC:
    case R_CONV_IM2COL_TC:
    case R_CONV_S2D_TC:
    case R_DENSE_TC: return k::conv_tc_variant_name(v);
    default: return v == 0 ? "" : "?";
    }
}

std::string candidate_desc(const Graph &g, int32_t cand) {
    const Candidate &c = g.cands[cand];
    const Layer &L = g.layers[c.layer];
    std::string d = routine_name(c.routine) ? routine_name(c.routine) : "?";
    d += " " + schema_str(g.schemas[c.schema]);
    if (cand_out(c) != c.schema) d += "->" + schema_str(g.schemas[cand_out(c)]);
    std::vector<Shape> in;
    for (int32_t j : L.inputs) in.push_back(g.layers[j].out);
    std::string params;
    if (c.routine == R_CONV_TC && !in.empty())
        params = k::conv_tc_config_desc(L, in[0], g.schemas[c.schema], c.variant);
    else
        params = variant_name(c.routine, c.variant);
    if (!params.empty()) d += " [" + params + "]";
    return d;
}

static bool is_conv(const Layer &l) { return l.type == SN_L_CONV2; }

// qint8 schema: the routines that have an int8 kernel (one variant each)
static int32_t q8_variants(int32_t r, const Layer &l, const std::vector<Shape> &in, sn_schema s) {
    switch (r) {
    case R_CONV_DIRECT: return is_conv(l) ? 1 : 0;
    case R_CONV_DP4A: return k::q8_conv_dp4a_applies(l, in[0], s) ? 1 : 0;
    case R_DW_DIRECT: return l.type == SN_L_DWCONV2 ? 1 : 0;
    case R_MAXPOOL: return l.type == SN_L_MAXPOOL ? 1 : 0;
    case R_GAP: return l.type == SN_L_GAP ? 1 : 0;
    case R_ADD: return l.type == SN_L_ADD ? 1 : 0;
    case R_MUL: return l.type == SN_L_MUL ? 1 : 0;
    case R_DENSE: return (l.type == SN_L_DENSE && in[0].h == 1 && in[0].w == 1) ? 1 : 0;
    default: return 0;
    }
}

int32_t routine_variants(int32_t r, const Layer &l, const std::vector<Shape> &in, sn_schema s) {
    if (s.dtype == SN_QI8) return q8_variants(r, l, in, s);
    if (r == R_CONV_DP4A) return 0;
    const sn_conv_params &p = l.conv;
    // a conv2 with a residual input is served by the routines whose epilogue
    // adds it: direct and the tensor-core implicit GEMM
    if (is_conv(l) && in.size() == 2 && r != R_CONV_DIRECT && r != R_CONV_TC) return 0;
    switch (r) {
    case R_CONV_DIRECT:
        return is_conv(l) ? 1 : 0;
    case R_CONV_IGEMM:
        return (is_conv(l) && p.groups == 1) ? 2 : 0;
    case R_CONV_WINO:
    case R_CONV_WINO4:
    case R_CONV_WINO6:
        return (is_conv(l) && p.groups == 1 && p.kh == 3 && p.kw == 3 && p.sh == 1 && p.sw == 1 &&
                p.dh == 1 && p.dw == 1 && p.ph <= 2 && p.pw <= 2)
                   ? 1
                   : 0;
    case R_CONV_TC:
        return is_conv(l) ? k::conv_tc_variants(l, in[0], s) : 0;
    case R_DW_DIRECT:
        if (l.type != SN_L_DWCONV2) return 0;
        // NHWC 3x3 of small maps: a third parameter, the shared-memory band kernel
        return (s.layout == SN_NHWC && k::dw3_band_applies(l, in[0], s)) ? 3 : 2;
    case R_MAXPOOL:
        return l.type == SN_L_MAXPOOL ? 1 : 0;
    case R_GAP:
        return l.type == SN_L_GAP ? 1 : 0;
    case R_ADD:
        return l.type == SN_L_ADD ? 1 : 0;
    case R_MUL:
        return l.type == SN_L_MUL ? 1 : 0;
    case R_DENSE:
        return l.type == SN_L_DENSE ? 1 : 0;
    case R_CONV_IM2COL_TC:
        return is_conv(l) ? k::conv_im2col_tc_variants(l, in[0], s) : 0;
    case R_DENSE_TC:
        return l.type == SN_L_DENSE ? k::dense_tc_variants(l, in[0], s) : 0;
    case R_CONV_S2D_TC:
        return is_conv(l) ? k::conv_s2d_tc_variants(l, in[0], s) : 0;
    default:
        return 0;
    }
}

size_t routine_workspace(int32_t r, int32_t v, const Layer &l, const std::vector<Shape> &in,
                         sn_schema s) {
    if (r == R_CONV_WINO) return k::conv_wino_ws(l, in[0], s);
    if (r == R_CONV_WINO4) return k::conv_wino4_ws(l, in[0], s);
    if (r == R_CONV_WINO6) return k::conv_wino6_ws(l, in[0], s);
    if (r == R_CONV_TC) return k::conv_tc_ws(l, in[0], s, v);
    if (r == R_CONV_IM2COL_TC) return k::conv_im2col_tc_ws(l, in[0], s, v);
    if (r == R_DENSE_TC) return k::dense_tc_ws(l, in[0], s, v);
    if (r == R_CONV_S2D_TC) return k::conv_s2d_tc_ws(l, in[0], s, v);
    return 0;
}

// weight format of (routine, layout)
static int weight_format_of(int32_t r, sn_schema s) {
    if (s.dtype == SN_QI8) {
        switch (r) {
        case R_CONV_DIRECT:
        case R_DW_DIRECT: return s.layout == SN_NCHW ? k::W_KCRS : k::W_RSCK;
        case R_CONV_DP4A: return k::W_KRSC;
        case R_DENSE: return k::W_KCRS;
        default: return -1;
        }
    }
    switch (r) {
    case R_CONV_DIRECT: return s.layout == SN_NCHW ? k::W_KCRS : k::W_RSCK;
    case R_CONV_IGEMM: return s.layout == SN_NCHW ? k::W_KCRS : k::W_KRSC;
    case R_CONV_WINO: return k::W_WINO;
    case R_CONV_WINO4: return k::W_WINO4;
    case R_CONV_WINO6: return k::W_WINO6;
    case R_CONV_TC: return k::W_KRSC;
    case R_DW_DIRECT: return s.layout == SN_NCHW ? k::W_KCRS : k::W_RSCK;
    case R_DENSE: return k::W_KCRS;
    case R_CONV_IM2COL_TC: return k::W_KRSC_PAD64;
    case R_DENSE_TC: return k::W_KRSC;
    case R_CONV_S2D_TC: return k::W_S2D;
    default: return -1;
    }
}

sn_status prepare_weights(Graph *g, int32_t li, int32_t r, int32_t v, sn_schema s,
                          const void **wt, const float **bias, cudaStream_t st) {
    (void)v;
    *wt = nullptr;
    *bias = nullptr;
    const Layer &L = g->layers[li];
    if (L.weight.empty()) return SN_OK;
    const int fmt = weight_format_of(r, s);
    if (fmt < 0) return SN_OK;
    int64_t K, Cg, R, S;
    if (L.type == SN_L_DENSE) {
        K = L.dense_out, Cg = L.dense_in, R = S = 1;
    } else {
        K = L.conv.c_out, Cg = L.conv.c_in / L.conv.groups, R = L.conv.kh, S = L.conv.kw;
    }
    // bias: fp32 on the device, shared by every routine of the layer, zero-
    // padded to a multiple of 256 entries so that a tile's epilogue may read
    // its whole channel range without a bounds check
    auto bit = g->bias_cache.find(li);
    if (bit == g->bias_cache.end()) {
        Buffer b;
        const size_t padded = (L.bias.size() + 255) / 256 * 256;
        sn_status rc = dev_alloc(g, padded * sizeof(float), &b);
        if (rc != SN_OK) return rc;
        SN_CUDA_TRY(cudaMemsetAsync(b.ptr, 0, padded * sizeof(float), st));
        SN_CUDA_TRY(cudaMemcpyAsync(b.ptr, L.bias.data(), L.bias.size() * sizeof(float),
                                    cudaMemcpyHostToDevice, st));
        bit = g->bias_cache.emplace(li, b).first;
    }
    *bias = static_cast<const float *>(bit->second.ptr);

    const std::string key = std::to_string(li) + "/" + std::to_string(fmt) + "/" + std::to_string(s.dtype);
    auto it = g->weight_cache.find(key);
    if (it != g->weight_cache.end()) {
        *wt = it->second.ptr;
        return SN_OK;
    }
    const int64_t elems = (fmt == k::W_WINO)         ? 16 * K * Cg
                          : (fmt == k::W_WINO4)      ? 36 * K * Cg
                          : (fmt == k::W_WINO6)      ? 64 * K * Cg
                          : (fmt == k::W_KRSC_PAD64) ? K * ((Cg * R * S + 63) / 64 * 64)
                          : (fmt == k::W_S2D)        ? K * (R <= 4 ? 2 : 4) * 64
                                                     : K * Cg * R * S;
    Buffer src, dst;
    sn_status rc = dev_alloc(g, (size_t)K * Cg * R * S * sizeof(float), &src);
    if (rc != SN_OK) return rc;
    const size_t dst_bytes = s.dtype == SN_QI8 ? k::q8_weight_bytes(K, elems)  // codes + per-channel scales
                             : (size_t)elems * ((fmt == k::W_WINO4 || fmt == k::W_WINO6) ? sizeof(float) : dtype_size(s.dtype));
    rc = dev_alloc(g, dst_bytes, &dst);
    if (rc != SN_OK) {
        dev_free(g, &src);
        return rc;
    }
    cudaError_t e = cudaMemcpyAsync(src.ptr, L.weight.data(), L.weight.size() * sizeof(float),
                                    cudaMemcpyHostToDevice, st);
    if (e == cudaSuccess)
        e = s.dtype == SN_QI8
                ? k::weight_format_q8(static_cast<const float *>(src.ptr), dst.ptr, fmt, K, Cg, R, S, st)
                : k::weight_format(static_cast<const float *>(src.ptr), dst.ptr, fmt, s.dtype, K, Cg, R, S, st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);  // src is freed next
    dev_free(g, &src);
    if (e != cudaSuccess) {
        dev_free(g, &dst);
        return fail(SN_ECUDA, std::string("weight preparation: ") + cudaGetErrorString(e));
    }
    g->weight_cache.emplace(key, dst);
    *wt = dst.ptr;
    return SN_OK;
}

int32_t kernels_per_launch(int32_t r, int32_t v, const Layer &l, const std::vector<Shape> &in, sn_schema s) {
    if (s.dtype == SN_QI8) return 1;
    // a K-split tensor-core GEMM adds its reduction kernel (it is the only
    // variant with a workspace)
    const int split = (r == R_CONV_TC || r == R_CONV_IM2COL_TC || r == R_DENSE_TC || r == R_CONV_S2D_TC) &&
                      routine_workspace(r, v, l, in, s) >
                          (r == R_CONV_IM2COL_TC ? k::conv_im2col_tc_ws(l, in[0], s, -1)
                           : r == R_CONV_S2D_TC  ? k::conv_s2d_tc_ws(l, in[0], s, -1)
                                                 : 0);
    if (r == R_CONV_WINO || r == R_CONV_WINO4 || r == R_CONV_WINO6) return 3;  // wgenc, wgconv, wgdec
    if (r == R_CONV_IM2COL_TC || r == R_CONV_S2D_TC) return 2 + split;  // re-layout, GEMM (+ reduction)
    return 1 + split;
}

std::vector<sn_schema> fused_outputs(int32_t r, const Layer &l, sn_schema s) {
    // the tensor-core convolution can write its NHWC result straight in the
    // NCHW layout of the same dtype (the permutation fused into its epilogue)
    if (r == R_CONV_TC && l.type == SN_L_CONV2 && s.layout == SN_NHWC && (s.dtype == SN_F16 || s.dtype == SN_BF16))
        return {{s.dtype, SN_NCHW}};
    // the space-to-depth stem reads either layout and its GEMM writes either
    // (NHWC from its TMA store, NCHW from the NCHW epilogue)
    if (r == R_CONV_S2D_TC && l.type == SN_L_CONV2 && (s.dtype == SN_F16 || s.dtype == SN_BF16))
        return {{s.dtype, s.layout == SN_NHWC ? SN_NCHW : SN_NHWC}};
    // qint8 routines can leave their fp32 result in a float schema of the
    // same layout instead of requantising it (dequantisation fused into the
    // epilogue)
    if (s.dtype != SN_QI8) return {};
    switch (r) {
    case R_CONV_DIRECT:
    case R_CONV_DP4A:
    case R_DW_DIRECT:
    case R_MAXPOOL:
    case R_GAP:
    case R_ADD:
    case R_MUL:
    case R_DENSE: return {{SN_F16, s.layout}, {SN_BF16, s.layout}, {SN_F32, s.layout}};
    default: return {};
    }
}

bool fused_variant_ok(int32_t r, const Layer &l, const std::vector<Shape> &in, sn_schema s, int32_t v) {
    if (s.dtype == SN_QI8) return true;
    // the NCHW writer drains each tile in one CTA's epilogue: no K split
    // through fp32 partials, no stream-K parts
    if (r == R_CONV_TC && !in.empty()) return k::conv_tc_nchw_ok(l, in[0], s, v);
    if (r == R_CONV_S2D_TC) return true;  // one-CTA tiles without a K split
    return false;
}

int32_t childnet_stages(int32_t r, sn_schema s) {
    if (s.dtype == SN_QI8) return 1;
    switch (r) {
    case R_CONV_IM2COL_TC:
    case R_CONV_S2D_TC: return 2;  // re-layout, GEMM
    case R_CONV_WINO:
    case R_CONV_WINO4:
    case R_CONV_WINO6: return 3;   // wgenc, wgconv, wgdec
    default: return 1;
    }
}

bool stage_uses_variant(int32_t r, int32_t stage) {
    // the GEMM of the im2col / space-to-depth childnets carries the tile
    // parameters; their re-layout and the Winograd stages have none
    return (r == R_CONV_IM2COL_TC || r == R_CONV_S2D_TC) && stage == 1;
}

sn_status launch_routine_stage(const LaunchArgs &a, int32_t stage) {
    cudaError_t e = cudaSuccess;
    switch (a.routine) {
    case R_CONV_IM2COL_TC: e = k::conv_im2col_tc_stage(a, stage); break;
    case R_CONV_S2D_TC: e = k::conv_s2d_tc_stage(a, stage); break;
    case R_CONV_WINO: e = k::conv_wino_stage(a, stage); break;
    case R_CONV_WINO4: e = k::conv_wino4_stage(a, stage); break;
    case R_CONV_WINO6: e = k::conv_wino6_stage(a, stage); break;
    default: return launch_routine(a);
    }
    if (e == cudaErrorNotSupported)
        return fail(SN_EUNSUPPORTED, std::string(routine_name(a.routine)) + ": not supported here");
    if (e != cudaSuccess)
        return fail(SN_ECUDA, std::string(routine_name(a.routine)) + " (stage): " + cudaGetErrorString(e));
    return SN_OK;
}

static cudaError_t launch_q8(const LaunchArgs &a) {
    switch (a.routine) {
    case R_CONV_DIRECT:
    case R_DW_DIRECT: return k::q8_conv_direct(a);
    case R_CONV_DP4A: return k::q8_conv_dp4a(a);
    case R_MAXPOOL: return k::q8_maxpool(a);
    case R_GAP: return k::q8_gap(a);
    case R_ADD: return k::q8_add(a);
    case R_MUL: return k::q8_mul(a);
    case R_DENSE: return k::q8_dense(a);
    default: return cudaErrorInvalidValue;
    }
}

sn_status launch_routine(const LaunchArgs &a) {
    cudaError_t e = cudaSuccess;
    if (a.schema.dtype == SN_QI8) {
        e = launch_q8(a);
        if (e != cudaSuccess)
            return fail(SN_ECUDA, std::string(routine_name(a.routine)) + " (qi8): " + cudaGetErrorString(e));
        return SN_OK;
    }
    switch (a.routine) {
    case R_CONV_DIRECT: e = k::conv_direct(a); break;
    case R_CONV_IGEMM: e = k::conv_igemm(a); break;
    case R_CONV_WINO: e = k::conv_wino(a); break;
    case R_CONV_WINO4: e = k::conv_wino4(a); break;
    case R_CONV_WINO6: e = k::conv_wino6(a); break;
    case R_CONV_TC: e = k::conv_tc(a); break;
    case R_DW_DIRECT: e = k::dwconv(a); break;
    case R_MAXPOOL: e = k::maxpool(a); break;
    case R_GAP: e = k::gap(a); break;
    case R_ADD: e = k::add(a); break;
    case R_MUL: e = k::mul(a); break;
    case R_DENSE: e = k::dense(a); break;
    case R_CONV_IM2COL_TC: e = k::conv_im2col_tc(a); break;
    case R_DENSE_TC: e = k::dense_tc(a); break;
    case R_CONV_S2D_TC: e = k::conv_s2d_tc(a); break;
    default: return fail(SN_EINVAL, "launch of a non-launchable routine");
    }
    if (e == cudaErrorNotSupported)  // a routine parameter this device cannot run (e.g. too few co-resident clusters)
        return fail(SN_EUNSUPPORTED, std::string(routine_name(a.routine)) + ": not supported here");
    if (e != cudaSuccess)
        return fail(SN_ECUDA, std::string(routine_name(a.routine)) + ": " + cudaGetErrorString(e));
    return SN_OK;
}

}  // namespace sn
