// Internal declarations of the routine-selecting inference core.
#pragma once

#include <cuda_runtime.h>

#include <cstdint>
#include <map>
#include <memory>
#include <string>
#include <vector>

#include "../../include/sn.h"

namespace sn {

constexpr int64_t kInf = INT64_MAX;

inline int64_t sat_add(int64_t a, int64_t b) { return (a == kInf || b == kInf) ? kInf : a + b; }

// -------------------------------------------------------------------------
// error reporting
// -------------------------------------------------------------------------
struct Error {
    sn_status status;
    std::string msg;
};
void set_error(const std::string &msg);
sn_status fail(sn_status s, const std::string &msg);
#define SN_CUDA_TRY(expr)                                                              \
    do {                                                                               \
        cudaError_t _e = (expr);                                                       \
        if (_e != cudaSuccess)                                                         \
            return ::sn::fail(SN_ECUDA, std::string(#expr) + ": " + cudaGetErrorString(_e)); \
    } while (0)

// -------------------------------------------------------------------------
// tensors
// -------------------------------------------------------------------------
struct Shape {
    int64_t n = 0, c = 0, h = 0, w = 0;
    int64_t numel() const { return n * c * h * w; }
    bool operator==(const Shape &o) const { return n == o.n && c == o.c && h == o.h && w == o.w; }
};

inline int dtype_size(int dt) { return dt == SN_F32 ? 4 : dt == SN_QI8 ? 1 : 2; }
inline bool schema_eq(sn_schema a, sn_schema b) { return a.dtype == b.dtype && a.layout == b.layout; }
inline bool schema_valid(sn_schema s) {
    return s.dtype >= SN_F32 && s.dtype <= SN_QI8 && s.layout >= SN_NCHW && s.layout <= SN_NHWC;
}
std::string schema_str(sn_schema s);

// -------------------------------------------------------------------------
// routine registry (section III-C: routines, descriptors, routine parameters)
// -------------------------------------------------------------------------
enum RoutineId : int32_t {
    R_IO = 0,            // auxiliary input/output layer, zero cost (section IV-E)
    R_CONV_DIRECT = 1,   // direct convolution, one output per thread
    R_CONV_IGEMM = 2,    // implicit GEMM on CUDA cores (FFMA), register-tiled
    R_CONV_WINO = 3,     // Winograd F(2x2,3x3) childnet: wgenc -> wgconv -> wgdec
    R_CONV_TC = 4,       // implicit GEMM on tcgen05 tensor cores, TMA-fed (NHWC)
    R_DW_DIRECT = 5,     // depthwise conv
    R_MAXPOOL = 6,
    R_GAP = 7,
    R_ADD = 8,
    R_DENSE = 9,         // dense on CUDA cores
    R_ADAPT = 10,        // adapt layer (cast / layout change)
    R_CONV_IM2COL_TC = 11,  // childnet: im2col -> tensor-core GEMM (any C, stride, dilation)
    R_DENSE_TC = 12,     // childnet: reshape -> 1x1 conv2 on tensor cores -> reshape (section III-D)
    R_CONV_S2D_TC = 13,  // childnet: space-to-depth -> stride-1 tensor-core conv (stride 2, <= 4 channels)
    R_MUL = 14,          // per-channel scale (squeeze-and-excite)
    R_CONV_WINO4 = 15,   // Winograd F(4x4,3x3) childnet (fp32 transformed filters)
    R_CONV_DP4A = 16,    // qint8 implicit GEMM with dp4a (NHWC)
    R_CONV_WINO6 = 17,   // Winograd F(6x6,3x3) childnet (fp32 transformed filters)
    R_COUNT = 18
};

// -------------------------------------------------------------------------
// graph (section III-B)
// -------------------------------------------------------------------------
struct Layer {
    int32_t type = -1;         // sn_layer_type, or -1 = input aux, -2 = output aux
    sn_conv_params conv{};     // CONV2 / DWCONV2
    sn_pool_params pool{};     // MAXPOOL
    int32_t act = SN_ACT_NONE; // ADD / DENSE / CONV
    int32_t dense_in = 0, dense_out = 0;
    std::vector<int32_t> inputs;  // internal layer indices
    Shape out;
    std::vector<float> weight, bias;  // host fp32 copies
    float qscale = 0.0f;              // qint8 scale of the output blob (0 = not set)
};

struct Candidate {
    int32_t routine, variant, schema, layer;  // schema: the one the routine reads
    int64_t cost;
    int32_t out_schema = -1;  // the schema it writes; -1 = the one it reads
};
inline int32_t cand_out(const Candidate &c) { return c.out_schema < 0 ? c.schema : c.out_schema; }

struct Buffer {  // device allocation owned by the graph
    void *ptr = nullptr;
    size_t bytes = 0;
    bool view = false;  // a part of another buffer (the activation arena): not freed on its own
};

struct PlanOp {
    enum Kind { LAYER, ADAPT } kind;
    int32_t layer = -1;    // LAYER: internal layer; ADAPT: consumer layer
    int32_t edge = -1;     // ADAPT: edge index
    int32_t cand = -1;     // LAYER: candidate index
    std::vector<int32_t> in_slots;
    int32_t out_slot = -1;
    const void *wt = nullptr;      // LAYER: prepared weights
    const float *bias = nullptr;   // LAYER: fp32 bias
};

struct Graph;

// One layer of a chained launch (consecutive conv2/igemm_tc layers run as one
// persistent kernel whose tiles wait on the tiles they read): the layer, its
// selected routine parameter and its resolved buffers; src / res_src = index
// within the chain of the layer that writes input 0 / the residual (-1: the
// buffer is written before the chain starts).
struct ChainOp {
    const Layer *layer = nullptr;
    Shape in;
    sn_schema schema{};
    int32_t variant = 0;
    const void *in0 = nullptr, *res = nullptr;
    void *out = nullptr;
    const void *wt = nullptr;
    const float *bias = nullptr;
    int32_t src = -1, res_src = -1;
};

// A chain of the plan: ops [first_op, last_op] run as one launch.
struct ChainPlan {
    int32_t first_op = -1, last_op = -1;
    int32_t n_layers = 0, total_units = 0, done_count = 0;
    int32_t dtype = 0;
    Buffer desc, done;  // layer descriptors; completion counters (+ exit counter, abort flag)
};

// A launchable routine instance: everything a kernel needs, resolved.
struct LaunchArgs {
    const Graph *g;
    const Layer *layer;
    int32_t routine, variant;
    sn_schema schema;
    std::vector<Shape> in_shapes;
    const void *in[2] = {nullptr, nullptr};
    void *out = nullptr;
    sn_schema out_schema{-1, -1};  // schema of `out` when the routine writes another (fused boundary)
    const void *wt = nullptr;   // prepared weights in the routine's format
    const float *bias = nullptr;
    void *ws = nullptr;         // workspace
    size_t ws_bytes = 0;
    // tensor-core implicit GEMM only: byte strides of the A tensor's pixel,
    // row, image and 64-value-block axes when they differ from dense NHWC
    // (0 = dense); a pixel stride below the 128-byte row makes consecutive
    // pixels' rows overlap
    int64_t a_strides[4] = {0, 0, 0, 0};
    // tensor-core implicit GEMM only: > 0 when the layer's "channels" are
    // a_blocks blocks of 64 read as one box (the space-to-depth stem's taps)
    int32_t a_blocks = 0;
    // qint8 routines: scales of the input blobs and of the output blob
    float qs_in[2] = {0.0f, 0.0f};
    float qs_out = 0.0f;
    // tensor-core routines: SM cycles a pipeline wait may take before the
    // kernel gives up and reports SN_ETIMEOUT (0 = the library default)
    int64_t wait_limit = 0;
    // tensor-core stream-K routines: the graph's zeroed counter array (the
    // kernels leave it zeroed) and its length in ints
    int *tile_counts = nullptr;
    int64_t tile_counts_n = 0;
    cudaStream_t stream = nullptr;
};

struct Graph {
    Shape in_shape;
    sn_schema in_schema{}, out_schema{};
    std::vector<sn_schema> schemas;   // universe: Lambda, then in/out if absent
    int32_t n_lambda = 0;             // |Lambda| (first entries of `schemas`)
    int32_t in_schema_idx = 0, out_schema_idx = 0;
    sn_alloc_fn alloc = nullptr;
    sn_free_fn free_fn = nullptr;
    void *alloc_ctx = nullptr;

    float in_qscale = 0.0f;           // qint8 scale of the net input (0 = not set)
    std::vector<Shape> extra_in;      // net inputs 1.. (section IV-E: several input layers)
    std::vector<float> extra_in_qscale;
    std::vector<int32_t> outputs;     // user ids of the net outputs (default: the last layer)
    std::vector<Layer> user;          // as added
    bool finalized = false;
    std::vector<Layer> layers;        // internal: [input, user..., output]
    std::vector<std::pair<int32_t, int32_t>> edges;
    std::vector<Candidate> cands;     // grouped by layer
    std::vector<int32_t> cand_begin;  // [n_layers + 1]
    std::vector<int64_t> adapt_cost;  // [n_edges][ns][ns]

    bool has_path = false;
    std::vector<int32_t> path_cand;   // per layer
    int64_t path_total = kInf;

    // plan (built lazily by sn_run)
    bool plan_valid = false;
    std::vector<PlanOp> plan;
    std::vector<Buffer> slots;        // activation buffers; slot 0 = in, 1 = out (external)
    std::vector<Shape> slot_shape;
    std::vector<sn_schema> slot_schema;
    std::vector<float> slot_qscale;   // qint8 scale of the blob a slot holds
    int32_t n_ext = 2;                // slots [0, n_ext) are the caller's: inputs, then outputs
    std::map<std::string, Buffer> weight_cache;  // key: layer/format/dtype
    std::map<int32_t, Buffer> bias_cache;        // per layer fp32 bias
    Buffer workspace;
    Buffer tile_counts;               // kTileCounts zeroed ints for the stream-K tensor-core routines
    Buffer arena;                     // the plan's activation buffers, placed by liveness
    size_t arena_unshared = 0;        // what the activation buffers would take one allocation each
    Buffer host_in, host_out;         // device staging of sn_run_host
    // sn_run_host's input upload: two landing buffers filled on the graph's
    // own copy stream (so that a call's upload overlaps the previous call's
    // net), each copied into host_in on the caller's stream
    Buffer host_land[2];
    cudaStream_t copy_stream = nullptr;
    cudaEvent_t land_done[2] = {nullptr, nullptr};  // upload into landing buffer b finished
    cudaEvent_t land_free[2] = {nullptr, nullptr};  // landing buffer b copied out (may be refilled)
    bool land_used[2] = {false, false};
    int land_next = 0;
    int opt_graph = 0, opt_check = 0;
    int64_t opt_wait_limit = 0;       // SN_OPT_WAIT_LIMIT (0 = default)
    int opt_share = 1;                // SN_OPT_SHARE_BUFFERS: place activations by liveness
    int opt_chain = 0;                // run runs of tensor-core convolutions as chained launches
    std::vector<ChainPlan> chains;    // built with the plan
    std::vector<int32_t> op_chain;    // per plan op: its chain, or -1
    bool profiling = false;           // plans built while profiling may lack qint8 scales
    cudaGraphExec_t gexec = nullptr;
    std::vector<const void *> gexec_in;
    std::vector<void *> gexec_out;
    cudaStream_t gexec_stream = nullptr;

    ~Graph();
    int32_t n_layers() const { return (int32_t)layers.size(); }
    int32_t n_in() const { return 1 + (int32_t)extra_in.size(); }
    int32_t n_out() const { return outputs.empty() ? 1 : (int32_t)outputs.size(); }
    int32_t n_schemas() const { return (int32_t)schemas.size(); }
    int64_t &adapt(int32_t e, int32_t a, int32_t b) {
        return adapt_cost[((size_t)e * schemas.size() + a) * schemas.size() + b];
    }
    int64_t adapt(int32_t e, int32_t a, int32_t b) const {
        return adapt_cost[((size_t)e * schemas.size() + a) * schemas.size() + b];
    }
};

sn_status graph_finalize(Graph *g);
sn_status fuse_residual(Graph *g, std::vector<int32_t> &new_id, int32_t *n_fused);
sn_status add_input(Graph *g, const int64_t nchw[4], int32_t *id);
sn_status set_outputs(Graph *g, const int32_t *ids, int32_t n);

// the caller's buffers of one run: net inputs in in_schema, outputs in out_schema
struct IoPtrs {
    std::vector<const void *> in;
    std::vector<void *> out;
};
sn_status dev_alloc(Graph *g, size_t bytes, Buffer *b);
// stream-K counters: one int per (tile, epilogue warp), 1024 tiles of 8 warps
constexpr int64_t kTileCounts = 8192;
sn_status ensure_tile_counts(Graph *g, cudaStream_t st);
void dev_free(Graph *g, Buffer *b);
void invalidate_plan(Graph *g);

// routine applicability: variants of `routine` that can serve `layer` in `s`
int32_t routine_variants(int32_t routine, const Layer &layer, const std::vector<Shape> &in,
                         sn_schema s);
const char *routine_name(int32_t routine);
const char *variant_name(int32_t routine, int32_t variant);
// descriptor of one candidate of a graph: routine name, schema and routine parameters
std::string candidate_desc(const Graph &g, int32_t cand);
size_t routine_workspace(int32_t routine, int32_t variant, const Layer &layer,
                         const std::vector<Shape> &in, sn_schema s);
// prepare weights for (layer, routine, variant, schema); returns device pointer
sn_status prepare_weights(Graph *g, int32_t li, int32_t routine, int32_t variant, sn_schema s,
                          const void **wt, const float **bias, cudaStream_t st);
sn_status launch_routine(const LaunchArgs &a);
// childnets (section III-D): routines made of sub-layers that the profiler
// times one by one.  childnet_stages = number of sub-layers (1 = a plain
// routine); stage_uses_variant = whether a sub-layer's time depends on the
// parent routine's parameter (otherwise it is timed once for all of them).
int32_t childnet_stages(int32_t routine, sn_schema s);
bool stage_uses_variant(int32_t routine, int32_t stage);
sn_status launch_routine_stage(const LaunchArgs &a, int32_t stage);
int32_t kernels_per_launch(int32_t routine, int32_t variant, const Layer &layer, const std::vector<Shape> &in,
                           sn_schema s);
// schemas other than `s` that the routine can write its output in, reading
// its inputs in `s` (a fused boundary: dequantisation in a qint8 epilogue)
std::vector<sn_schema> fused_outputs(int32_t routine, const Layer &layer, sn_schema s);
// whether variant v of the routine can write those other schemas
bool fused_variant_ok(int32_t routine, const Layer &layer, const std::vector<Shape> &in, sn_schema s, int32_t v);

// selection (section IV)
sn_status select_dprs(const Graph &g, std::vector<int32_t> &schema_of, int64_t &total);
sn_status select_brute(const Graph &g, std::vector<int32_t> &schema_of, int64_t &total);
// either method on the graph's candidates: when some routine writes a schema
// other than the one it reads, a layer's state is the pair (read, written)
// and an edge costs the adapt from its producer's written schema to its
// consumer's read one.  cand_of[i] = the chosen candidate of layer i.
sn_status select_path(const Graph &g, int32_t method, std::vector<int32_t> &cand_of, int64_t &total);
void fastest_per_schema(const Graph &g, std::vector<int64_t> &F, std::vector<int32_t> &argF);

// plan + run
sn_status build_plan(Graph *g, cudaStream_t st);
sn_status build_chains(Graph *g, cudaStream_t st);
// [first op, last op] of every run of plan ops that a chained launch would run
std::vector<std::pair<int32_t, int32_t>> chain_runs(const Graph *g);
sn_status run_plan(Graph *g, const IoPtrs &io, cudaStream_t st,
                   std::vector<cudaEvent_t> *evs);
// one run of the plan replayed from a CUDA graph with a timing node around
// every op (device time of each op, no host launch cost); op_ms[q] in ms
sn_status run_plan_timed(Graph *g, const IoPtrs &io, cudaStream_t st, std::vector<float> *op_ms);
sn_status profile_graph(Graph *g, const sn_profile_opts &o, cudaStream_t st);
// qint8 calibration: run the fastest float-schema path, set every blob's scale
// to max |x| / 127
sn_status calibrate(Graph *g, const void *in, cudaStream_t st);

// -------------------------------------------------------------------------
// kernels (launchers; all asynchronous on `st`)
// -------------------------------------------------------------------------
namespace k {
cudaError_t convert(const void *x, int dt_in, int lay_in, void *y, int dt_out, int lay_out,
                    Shape s, cudaStream_t st);
cudaError_t fill_pattern(void *y, int dt, int64_t n, uint32_t seed, float scale,
                         cudaStream_t st);
// weight re-layout / cast from fp32 KCRS (device) into a routine format
enum WFormat { W_KCRS = 0, W_RSCK = 1, W_KRSC = 2, W_WINO = 3, W_KRSC_PAD64 = 4, W_S2D = 5, W_WINO4 = 6, W_WINO6 = 7 };
cudaError_t weight_format(const float *w_kcrs, void *out, int fmt, int dt, int64_t K,
                          int64_t Cg, int64_t R, int64_t S, cudaStream_t st);

cudaError_t conv_direct(const LaunchArgs &a);
cudaError_t conv_igemm(const LaunchArgs &a);
cudaError_t conv_wino(const LaunchArgs &a);
size_t conv_wino_ws(const Layer &l, const Shape &in, sn_schema s);
cudaError_t conv_wino4(const LaunchArgs &a);
size_t conv_wino4_ws(const Layer &l, const Shape &in, sn_schema s);
cudaError_t conv_wino6(const LaunchArgs &a);
// childnet stages, launched on their own (stage -1 = the whole routine)
cudaError_t conv_wino_stage(const LaunchArgs &a, int stage);
cudaError_t conv_wino4_stage(const LaunchArgs &a, int stage);
cudaError_t conv_wino6_stage(const LaunchArgs &a, int stage);
cudaError_t conv_im2col_tc_stage(const LaunchArgs &a, int stage);
cudaError_t conv_s2d_tc_stage(const LaunchArgs &a, int stage);
size_t conv_wino6_ws(const Layer &l, const Shape &in, sn_schema s);
cudaError_t conv_tc(const LaunchArgs &a);
int32_t conv_tc_variants(const Layer &l, const Shape &in, sn_schema s);
size_t conv_tc_ws(const Layer &l, const Shape &in, sn_schema s, int32_t v, int32_t a_blocks = 0);  // K-split partials
size_t dense_tc_ws(const Layer &l, const Shape &in, sn_schema s, int32_t v);
const char *conv_tc_variant_name(int32_t v);
bool conv_tc_nchw_ok(const Layer &l, const Shape &in, sn_schema s, int32_t v);  // variant v can write NCHW
std::string conv_tc_config_desc(const Layer &l, const Shape &in, sn_schema s, int32_t v, int32_t a_blocks = 0);
// chained launches of consecutive tensor-core convolutions
bool conv_tc_chain_shape(const Layer &l, const Shape &in, sn_schema s, int32_t v, bool *implicit, int *bn, int *kb,
                         int *bw, int *bh, int *bni);
size_t chain_desc_bytes(int n_layers);
cudaError_t chain_encode(const std::vector<ChainOp> &ops, std::vector<uint8_t> &blob, int32_t *total_units,
                         int32_t *done_count);
cudaError_t chain_launch(int dtype, const void *desc_dev, int32_t n_layers, int32_t total_units, int32_t *done_dev,
                         int32_t done_count, cudaStream_t st);
// im2col childnet and dense childnet on the tensor-core GEMM
int32_t conv_im2col_tc_variants(const Layer &l, const Shape &in, sn_schema s);
size_t conv_im2col_tc_ws(const Layer &l, const Shape &in, sn_schema s, int32_t v);
cudaError_t conv_im2col_tc(const LaunchArgs &a);
int32_t dense_tc_variants(const Layer &l, const Shape &in, sn_schema s);
// space-to-depth childnet for stride-2 convolutions of few input channels
int32_t conv_s2d_tc_variants(const Layer &l, const Shape &in, sn_schema s);
size_t conv_s2d_tc_ws(const Layer &l, const Shape &in, sn_schema s, int32_t v);
cudaError_t conv_s2d_tc(const LaunchArgs &a);
cudaError_t dense_tc(const LaunchArgs &a);
cudaError_t dwconv(const LaunchArgs &a);
bool dw3_band_applies(const Layer &l, const Shape &in, sn_schema s);  // NHWC small-map depthwise kernel
cudaError_t maxpool(const LaunchArgs &a);
cudaError_t gap(const LaunchArgs &a);
cudaError_t add(const LaunchArgs &a);
cudaError_t mul(const LaunchArgs &a);
cudaError_t dense(const LaunchArgs &a);
int *device_error_word();  // device address of the library's error word
// qint8 schema (symmetric codes, one scale per blob, per-channel weight scales)
cudaError_t convert_q8(const void *x, int dt_in, int lay_in, void *y, int dt_out, int lay_out, Shape s,
                       float qscale, cudaStream_t st);
cudaError_t fill_q8(void *y, int64_t n, uint32_t seed, cudaStream_t st);
size_t q8_weight_bytes(int64_t K, int64_t elems);  // codes, then fp32 scales [K]
cudaError_t weight_format_q8(const float *w_kcrs, void *out, int fmt, int64_t K, int64_t Cg, int64_t R,
                             int64_t S, cudaStream_t st);
cudaError_t q8_conv_direct(const LaunchArgs &a);
bool q8_conv_dp4a_applies(const Layer &l, const Shape &in, sn_schema s);
cudaError_t q8_conv_dp4a(const LaunchArgs &a);
cudaError_t q8_dense(const LaunchArgs &a);
cudaError_t q8_maxpool(const LaunchArgs &a);
cudaError_t q8_gap(const LaunchArgs &a);
cudaError_t q8_add(const LaunchArgs &a);
cudaError_t q8_mul(const LaunchArgs &a);
// running max |x| of a float blob into *out (fp32 bits; zero it first)
cudaError_t absmax(const void *x, int dt, int64_t n, unsigned *out, cudaStream_t st);
}  // namespace k

}  // namespace sn
