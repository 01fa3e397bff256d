/*
 * sn.h -- C ABI of the GB300 routine-selecting CNN inference library
 * (SoftNeuro, arXiv 2110.06037, reimplemented for sm_103a).
 *
 * The calls follow the paper's statement of the tuning problem (Alg. 1,
 * "Input: a 1-in-1-out net {L_i}, layer-wise optimal routines {F_i},
 * {F^a_ij}, a routine schema set Lambda; Output: the optimal routine path
 * S*"):
 *   sn_graph_create / sn_add_layer  build the net            (section III-B)
 *   sn_profile                      measures T(r)            (section III-C)
 *   sn_get/set_cost_table           the profiling data T(r), T(r^a)
 *   sn_select_path                  DPRS (Alg. 1) or brute force (Def. 2)
 *   sn_run                          inference with the tuned path
 *
 * Conventions for every call:
 *   - Every function returns sn_status; no C++ exception, abort or CUDA error
 *     crosses this boundary.  On a status other than SN_OK the graph is left
 *     as it was and sn_last_error() gives a message (thread-local, valid until
 *     the next call on the same thread).
 *   - Pointers named *_dev are device pointers on the current CUDA device;
 *     all other pointers are host pointers.  `stream` is a cudaStream_t
 *     (NULL = the legacy default stream).  The library launches only on that
 *     stream and never synchronises the device; calls that must read results
 *     back (profiling, SN_OPT_CHECK) synchronise that stream only.
 *   - Host arrays passed in are copied; the caller keeps ownership.  Device
 *     memory the library needs (weights in each schema, activations,
 *     workspace) comes from the allocator given to sn_graph_create (or
 *     cudaMalloc when none is given) and is released by sn_graph_destroy.
 *   - Tensor extents are always given as logical (N, C, H, W); the schema's
 *     layout says how they are stored (NCHW or NHWC, dense, row-major).
 *   - Costs are int64 nanoseconds; SN_COST_INF (INT64_MAX) = infeasible.
 */
#ifndef SN_H
#define SN_H

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define SN_API __attribute__((visibility("default")))
#else
#define SN_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef struct sn_graph sn_graph; /* opaque, owned by the library */

typedef enum {
    SN_OK = 0,
    SN_EINVAL = 1,        /* bad argument, size or layer parameter            */
    SN_ENOMEM = 2,        /* the allocator returned NULL                      */
    SN_ECUDA = 3,         /* a CUDA runtime/driver call failed                */
    SN_EUNSUPPORTED = 4,  /* valid request this build cannot serve            */
    SN_ESTATE = 5,        /* call out of order (e.g. sn_run before a path)    */
    SN_ETIMEOUT = 6,      /* a device-side bounded wait gave up               */
    SN_EINFEASIBLE = 7    /* no routine path with finite cost exists          */
} sn_status;

#define SN_COST_INF INT64_MAX

/* Routine schema (section III-C): the platform is always this GPU, so a
 * schema is the pair (data type, layout).  Two adjacent layers whose routines
 * have different schemas are joined by an adapt routine that casts and/or
 * permutes the blob.
 *
 * SN_QI8 is the quantised schema of section II-C in its symmetric form
 * (offset 0): a blob holds int8 codes q in [-127, 127] and one fp32 scale s
 * per blob (set by sn_set_qscale or sn_calibrate), standing for the values
 * q * s.  Quantising a float blob gives q = clamp(rint(x * (1/s)), -127, 127)
 * (1/s rounded to fp32; round half to even); dequantising gives the fp32
 * value q * s.  qint8 routines keep one scale per weight output channel,
 * s_w[k] = max |W[k, .]| / 127, sum code products exactly and requantise
 * y = act(float(acc) * (s_x * s_w[k]) + bias[k] (+ residual value)) to the
 * output blob's scale, every fp32 operation rounded on its own. */
typedef enum { SN_F32 = 0, SN_F16 = 1, SN_BF16 = 2, SN_QI8 = 3 } sn_dtype;
typedef enum { SN_NCHW = 0, SN_NHWC = 1 } sn_layout;
typedef struct { int32_t dtype; int32_t layout; } sn_schema;

/* Layer types (section III-B); activations are fused layer attributes (the
 * importer's ReLU fusion, section III-A). */
typedef enum {
    SN_L_CONV2 = 0,   /* 2-D convolution (cross-correlation) + bias + act;
                       * optionally + a residual blob before the act (fused add) */
    SN_L_DWCONV2 = 1, /* depthwise conv2: groups = c_in = c_out                */
    SN_L_MAXPOOL = 2, /* max pooling, -inf padding                             */
    SN_L_GAP = 3,     /* global average pooling -> N x C x 1 x 1               */
    SN_L_ADD = 4,     /* elementwise sum of two blobs + act                    */
    SN_L_DENSE = 5,   /* y = W x + b on an N x C x 1 x 1 blob                  */
    SN_L_MUL = 6      /* y[n,c,h,w] = x[n,c,h,w] * s[n,c] + act: the scale of
                       * a squeeze-and-excite block; inputs (x, s), s is
                       * N x C x 1 x 1; params sn_add_params                   */
} sn_layer_type;

/* Activations: max(0,x); min(max(0,x),6); hard swish x * relu6(x+3) / 6 and
 * hard sigmoid relu6(x+3) / 6 (MobileNetV3's piecewise-linear forms). */
typedef enum {
    SN_ACT_NONE = 0,
    SN_ACT_RELU = 1,
    SN_ACT_RELU6 = 2,
    SN_ACT_HSWISH = 3,
    SN_ACT_HSIGMOID = 4
} sn_act;

/* conv2 / dwconv2 parameters: output extent P = floor((H + 2ph - dh(kh-1) - 1)/sh) + 1. */
typedef struct {
    int32_t c_in, c_out, kh, kw, sh, sw, ph, pw, dh, dw, groups, act;
} sn_conv_params;
typedef struct { int32_t kh, kw, sh, sw, ph, pw; } sn_pool_params;
typedef struct { int32_t act; } sn_add_params;
typedef struct { int32_t in_features, out_features, act; } sn_dense_params;

/* Device allocator hooks (e.g. the PyTorch caching allocator).  alloc returns
 * a device pointer aligned to >= 256 bytes or NULL; free releases it. */
typedef void *(*sn_alloc_fn)(size_t bytes, void *ctx);
typedef void (*sn_free_fn)(void *ptr, void *ctx);

/*
 * Create an empty net with one input blob of logical shape in_nchw, stored in
 * in_schema, whose output will be produced in out_schema.  schemas[0..n) is
 * the schema set Lambda the routines may use (section IV-A).  The input and
 * output are the net's auxiliary layers L_1 and L_n (section IV-E): one
 * zero-cost routine each, in in_schema / out_schema.
 * alloc/free may both be NULL (cudaMalloc/cudaFree are used).
 * Errors: SN_EINVAL (bad shape or schema, n_schemas < 1, only one of alloc/free).
 */
SN_API sn_status sn_graph_create(const int64_t in_nchw[4], sn_schema in_schema, sn_schema out_schema,
                          const sn_schema *schemas, int32_t n_schemas, sn_alloc_fn alloc,
                          sn_free_fn free_fn, void *alloc_ctx, sn_graph **out);

/*
 * Append a layer (section III-B).  params points to the struct for the type
 * (sn_conv_params for CONV2/DWCONV2, sn_pool_params, sn_add_params,
 * sn_dense_params; NULL for GAP).  inputs[0..n_inputs) are ids returned by
 * earlier calls, -1 = the net input, -2, -3, ... = the inputs declared by
 * sn_add_input (ADD takes two, the others one).
 * CONV2 may take a second input, a residual of exactly the output's shape:
 * y = act(conv(x) + bias + residual), the residual add of a ResNet block fused
 * into the convolution that feeds it (the paper's graph optimiser fuses
 * layers before tuning, section III-A); the direct and the tensor-core
 * routines serve such a layer.
 * weights: host fp32, conv [c_out][c_in/groups][kh][kw], dense [out][in];
 * bias: host fp32 [c_out] or NULL (zeros).  Both are copied.  The last layer
 * added is the net output unless sn_set_outputs names others.
 * *out_layer_id receives the new layer's id.
 * Errors: SN_EINVAL (shape mismatch, bad parameter), SN_ESTATE (after the
 * net was finalised by sn_profile/sn_get_cost_table/sn_select_path/...).
 */
SN_API sn_status sn_add_layer(sn_graph *g, int32_t type, const void *params, const int32_t *inputs,
                       int32_t n_inputs, const float *weights, const float *bias,
                       int32_t *out_layer_id);

/* ---------------- several inputs and outputs (section IV-E) ---------------
 * A net may read several input blobs and produce several output blobs; the
 * auxiliary input layer feeds every input layer and the auxiliary output layer
 * merges every output, so the tuning problem stays 1-in-1-out.
 * sn_add_input: declare another net input of logical shape in_nchw, stored in
 *   in_schema; *input_id receives its id for sn_add_layer's inputs (-2 for the
 *   second input, -3 for the third, ...; the first, from sn_graph_create, is
 *   -1).  Every input must be declared before the first sn_add_layer, and
 *   every input must feed some layer.
 * sn_set_outputs: the net outputs, in order (distinct layer ids); each is
 *   delivered in out_schema.  Default: the last layer added.
 * sn_get_io: the number of net inputs and outputs.
 * Errors: SN_EINVAL (bad extent or id), SN_ESTATE (after finalisation, or
 * sn_add_input after a layer). */
SN_API sn_status sn_add_input(sn_graph *g, const int64_t in_nchw[4], int32_t *input_id);
SN_API sn_status sn_set_outputs(sn_graph *g, const int32_t *layer_ids, int32_t n);
/* Residual-add fusion, the graph optimiser pass run before tuning (section
 * III-A: layers are fused ahead of profiling and routine selection): every
 * SN_L_ADD one of whose inputs is an SN_L_CONV2 with SN_ACT_NONE and one
 * input, read by nothing else and not a net output, is replaced by that
 * conv2 with the add's other input as a residual and the add's activation,
 * y = act(conv(x) + bias + residual) (the conv2-with-residual layer of
 * sn_add_layer).  The fused layer takes the add's place and the conv2 is
 * removed, so layer ids change: new_id[old] (n_ids = the number of layers
 * added so far; may be NULL) receives each old id's new id, -1 for a conv2
 * folded into its add; net output ids are remapped.  *n_fused (may be NULL)
 * = the number of adds fused.  Call after the last sn_add_layer /
 * sn_set_outputs and before anything that finalises the net (cost table,
 * profiling, path selection, run).
 * Errors: SN_ESTATE (net already finalised), SN_EINVAL (NULL graph, n_ids
 * not the number of layers). */
SN_API sn_status sn_fuse_residual(sn_graph *g, int32_t *new_id, int32_t n_ids, int32_t *n_fused);
SN_API sn_status sn_get_io(sn_graph *g, int32_t *n_inputs, int32_t *n_outputs);

/* ---------------- the cost table (profiling data, section III-C) ----------
 * After finalisation the net has n_layers = (net inputs) + (layers added) + 1
 * internal layers in topological order: 0 is the auxiliary input layer (it
 * holds the first net input), 1 .. n_inputs-1 hold the other net inputs,
 * layer id u returned by sn_add_layer is internal layer u + n_inputs, and
 * n_layers-1 is the auxiliary output layer.
 * Each layer has candidate routines (routine id, routine-parameter
 * combination "variant", schema index); each edge (src, dst) has an adapt
 * cost for every ordered schema pair (void adapt = 0 on the diagonal).
 * Schema indices run over the graph's schema universe: Lambda in the order
 * given, then in_schema and out_schema if they are not in Lambda. */
typedef struct {
    int32_t routine;    /* routine id, see sn_routine_name()                */
    int32_t variant;    /* routine-parameter combination index              */
    int32_t schema;     /* schema index the routine reads its inputs in     */
    int32_t layer;      /* internal layer index                              */
    int64_t cost_ns;    /* T(r); SN_COST_INF until profiled or set           */
    int32_t out_schema; /* schema index it writes its output in: = schema,
                           except for fused-boundary routines (a qint8
                           routine leaving its result in a float schema).
                           When any candidate has out_schema != schema, the
                           selection runs over (schema, out_schema) pairs and
                           an edge's adapt goes from the producer's
                           out_schema to the consumer's schema. */
} sn_candidate;

typedef struct {
    int32_t n_layers, n_schemas, n_edges, n_candidates;
    sn_candidate *candidates; /* [n_candidates], grouped by layer, ascending  */
    int32_t *edges;           /* [n_edges][2] = (src, dst) internal layers    */
    int64_t *adapt_cost;      /* [n_edges][n_schemas (from)][n_schemas (to)]  */
} sn_cost_table;

/* Finalise the net if needed and report the table.  With t->candidates,
 * t->edges and t->adapt_cost all NULL only the four sizes are written;
 * otherwise the caller provides arrays of those sizes and they are filled. */
SN_API sn_status sn_get_cost_table(sn_graph *g, sn_cost_table *t);
/* Overwrite every candidate cost and adapt cost from t (sizes must match the
 * graph's; the routine/variant/schema/layer fields are checked, not copied).
 * Lets a caller inject or reuse profiling data.  Errors: SN_EINVAL. */
SN_API sn_status sn_set_cost_table(sn_graph *g, const sn_cost_table *t);
/* Schema universe queries. */
SN_API sn_status sn_get_schema(sn_graph *g, int32_t index, sn_schema *out, int32_t *n_schemas);

/* ---------------- profiling (section III-C) --------------------------------
 * Unit profiling times every candidate of every layer, deduplicated by layer
 * signature, on scratch buffers: `warmup` untimed launches, then the median
 * of `iters` launches timed with CUDA events on `stream`, rounded to ns.
 * Every adapt (blob shape, from, to) is timed the same way.  With topk > 0,
 * integrated profiling then re-times the topk best candidates per (layer,
 * schema) inside whole-net passes (one pass per schema and rank, `passes`
 * repetitions, median) and replaces their unit times.  Synchronises stream. */
typedef struct {
    int32_t warmup;   /* default 3  */
    int32_t iters;    /* default 20 */
    int32_t topk;     /* default 2; 0 = unit profiling only */
    int32_t passes;   /* default 5  */
} sn_profile_opts;
SN_API sn_status sn_profile(sn_graph *g, const sn_profile_opts *opts, void *stream);

/* ---------------- path selection (section IV) ------------------------------ */
#define SN_SELECT_DPRS 0  /* Alg. 1                                            */
#define SN_SELECT_BRUTE 1 /* exhaustive argmin of Def. 2 (small nets only)     */

typedef struct {
    int64_t total_ns;   /* T(S*)                                          */
    int32_t n_layers;   /* in: capacity of the arrays; out: n_layers       */
    int32_t *schema;    /* [n_layers] chosen schema index per layer, or NULL */
    int32_t *candidate; /* [n_layers] chosen candidate index (global index
                           into the cost table's candidates), or NULL       */
} sn_path;

/* Select S* from the current cost table and make it the path sn_run uses.
 * Errors: SN_EINFEASIBLE (every path has infinite cost), SN_EUNSUPPORTED
 * (brute force on a net with too many assignments), SN_EINVAL. */
SN_API sn_status sn_select_path(sn_graph *g, int32_t method, sn_path *out);
/* Force a path: candidate[i] is a global candidate index of layer i for
 * every internal layer (tests use this to run one routine in isolation). */
SN_API sn_status sn_set_path(sn_graph *g, const int32_t *candidate, int32_t n_layers);

/* ---------------- inference --------------------------------------------- */
#define SN_OPT_CUDA_GRAPH 0 /* 1 = replay the launch sequence as a CUDA graph    */
#define SN_OPT_CHECK 1      /* 1 = sync stream after sn_run and read the device
                               error word (SN_ETIMEOUT / SN_ECUDA on failure)    */
#define SN_OPT_CHAIN 2      /* 1 (default) = run every run of two or more
                               consecutive conv2/igemm_tc layers of the plan as
                               one persistent launch whose tiles wait on the
                               tiles they read (section III-A executes the tuned
                               net layer by layer; the routine and its
                               parameters per layer are unchanged, the launch
                               boundaries between them go); 0 = one launch per
                               layer.  Profiling and sn_run_timed always run
                               one launch per layer.                             */
#define SN_OPT_SHARE_BUFFERS 4 /* 1 (default) = activation blobs whose live
                               ranges do not overlap share bytes of the plan's
                               arena (sn_plan_memory); 0 = every blob its own
                               bytes.  The outputs are the same either way.   */
#define SN_OPT_WAIT_LIMIT 3 /* SM clock cycles that one pipeline wait of a
                               tensor-core routine (conv2/igemm_tc and the
                               routines built on it) may take before the kernel
                               stops, lets its own copies and MMAs land, frees
                               its tensor memory, records the cause in the
                               library's error word and returns (sn_run then
                               reports SN_ETIMEOUT under SN_OPT_CHECK and
                               clears the word).  0 (default) = about 2 s at
                               the maximum clock.  A small value makes waits
                               that would have completed expire: the run's
                               output is then not valid.                         */
SN_API sn_status sn_set_option(sn_graph *g, int32_t option, int64_t value);

/* Run the net with the selected path: in_dev holds the input in in_schema,
 * out_dev receives the output in out_schema (both caller-owned device
 * buffers of the full tensor size).  The first call after a path change
 * builds the plan (adapt insertion, buffers, weight copies per schema).
 * Errors: SN_ESTATE (no path), SN_ENOMEM, SN_ECUDA, SN_ETIMEOUT. */
SN_API sn_status sn_run(sn_graph *g, const void *in_dev, void *out_dev, void *stream);
/* sn_run from and to host memory: the input is copied from in_host (host
 * memory holding the input in in_schema, the full tensor) into a device
 * buffer the graph owns, the net runs, and the output is copied back to
 * out_host (out_schema, the full tensor), all asynchronously and in order
 * on `stream`: read out_host only after synchronising the stream.  The
 * upload itself runs on a stream the graph owns, into one of two device
 * landing buffers used in turn, so that the upload of one call overlaps the
 * net of the call before it; `stream` waits for it.  Page-locked host
 * buffers (cudaHostAlloc / cudaHostRegister) make the copies asynchronous;
 * pageable ones work but the copies then synchronise with the host.  Both
 * host buffers are the caller's and must stay valid (in_host unchanged)
 * until the stream has passed this call.  Nets with one input and one
 * output only.
 * Errors: as sn_run, plus SN_EINVAL for a net with several inputs or
 * outputs and SN_ENOMEM when the device staging buffers cannot be made. */
SN_API sn_status sn_run_host(sn_graph *g, const void *in_host, void *out_host, void *stream);
/* sn_run for a net with several inputs or outputs: in_devs[0..n_in) in the
 * order of their ids (-1, -2, ...), out_devs[0..n_out) in the order given to
 * sn_set_outputs.  n_in and n_out must match the net (SN_EINVAL otherwise);
 * sn_run is this call with one of each. */
SN_API sn_status sn_run_multi(sn_graph *g, const void *const *in_devs, int32_t n_in, void *const *out_devs,
                              int32_t n_out, void *stream);

/* sn_run with a CUDA event pair around every launch of the plan; after the
 * stream has finished (this call synchronises it) layer_ms[i] holds the time
 * of layer i's routine and edge_ms[e] that of edge e's adapt (0 if void).
 * Either array may be NULL.  Sizes: n_layers and n_edges.  Nets with one
 * input and one output only (SN_EINVAL otherwise). */
SN_API sn_status sn_run_timed(sn_graph *g, const void *in_dev, void *out_dev, void *stream,
                       float *layer_ms, float *edge_ms);

/* Launch statistics of the current plan (built on `stream` if needed): the
 * number of plan operations (layer routines + adapts) and of CUDA kernels
 * that one sn_run launches.  Either output may be NULL.
 * Errors: SN_ESTATE (no path), plus those of plan building. */
SN_API sn_status sn_plan_stats(sn_graph *g, int32_t *n_ops, int32_t *n_kernels, void *stream);
/* Device memory of the current plan's activations (built on `stream` if
 * needed): *arena_bytes = the one allocation that holds every graph-owned
 * blob, placed by liveness (a blob lives from the op that writes it to the
 * last op that reads it; blobs live at the same time never share bytes);
 * *unshared_bytes = what the same blobs take one allocation each.  The
 * caller's input and output buffers, weights and the routines' workspace are
 * not counted.  Either output may be NULL.
 * Errors: SN_ESTATE (no path), plus those of plan building. */
SN_API sn_status sn_plan_memory(sn_graph *g, int64_t *arena_bytes, int64_t *unshared_bytes, void *stream);

/* Logical output shape of internal layer `layer` (N, C, H, W). */
SN_API sn_status sn_layer_shape(sn_graph *g, int32_t layer, int64_t out_nchw[4]);

/* Save / restore the tuned state (cost table + selected path) as JSON.  A
 * loaded file must describe the same net (same layers and candidates). */
SN_API sn_status sn_save_plan(sn_graph *g, const char *path);
SN_API sn_status sn_load_plan(sn_graph *g, const char *path);

SN_API void sn_graph_destroy(sn_graph *g);

/* ---------------- routines and adapts used directly ------------------------ */
/* Routine descriptor "cuda:<dtype>.<layout>/<algorithm>" style name of a
 * routine id (section III-C), or NULL for an unknown id. */
SN_API const char *sn_routine_name(int32_t routine);
/* Human-readable routine parameters of (routine, variant), e.g. "bn=128". */
SN_API const char *sn_variant_name(int32_t routine, int32_t variant);
/* Descriptor of candidate `cand` of a graph (section III-C: a routine is
 * identified by its descriptor and its routine parameters): routine name,
 * the schema it reads (and "->" the one it writes when they differ) and its
 * parameter values, e.g. "conv2/igemm_tc bf16.nhwc [bn=128 cta=2 kb=2 ...]".
 * The string lives in thread-local storage until the next call on the same
 * thread.  NULL for a NULL graph, an unfinalisable graph or a bad index. */
SN_API const char *sn_candidate_desc(sn_graph *g, int32_t cand);

/* Adapt routine on its own (section III-C, jobs (2) and (3)): convert the
 * N x C x H x W blob x_dev stored in `from` into y_dev stored in `to`
 * (layout permutation and/or round-to-nearest-even cast; bit-exact).
 * Errors: SN_EINVAL, SN_ECUDA. */
SN_API sn_status sn_convert(const void *x_dev, sn_schema from, void *y_dev, sn_schema to,
                     const int64_t nchw[4], void *stream);
/* sn_convert where either side may be SN_QI8: qscale > 0 is the blob's
 * scale (quantise: float -> codes; dequantise: codes -> float; codes ->
 * codes: layout permutation only).  Errors: SN_EINVAL (bad schema, no qint8
 * side, qscale not finite and positive), SN_ECUDA. */
SN_API sn_status sn_convert_q(const void *x_dev, sn_schema from, void *y_dev, sn_schema to,
                              const int64_t nchw[4], float qscale, void *stream);

/* ---------------- qint8 scales (section II-C, hybrid tuning of section V-C)
 * Every blob that a selected path keeps in SN_QI8 needs a scale: the net
 * input (layer id -1) and the output of each layer (ids from sn_add_layer).
 * Profiling does not need them (it times on scratch codes); building the plan
 * of a path that quantises a blob without a scale fails with SN_ESTATE.
 * sn_set_qscale: scale finite and > 0.  Invalidates the plan.
 * sn_get_qscale: *scale = the blob's scale, 0 when none is set.
 * Errors: SN_EINVAL (bad id or scale). */
SN_API sn_status sn_set_qscale(sn_graph *g, int32_t layer_id, float scale);
SN_API sn_status sn_get_qscale(sn_graph *g, int32_t layer_id, float *scale);
/* Calibration (post-training, symmetric, per tensor): run the net once on
 * in_dev (in in_schema, caller-owned) along the cheapest path that keeps every
 * layer in a float schema of Lambda (DPRS over the current cost table with the
 * qint8 candidates left out), and set the scale of the net input and of every
 * layer's output to max |x| / 127 of the blob as that path stores it (1 for an
 * all-zero blob).  The selected path, if any, is kept.  Synchronises stream.
 * Errors: SN_ESTATE (costs not profiled or set: no finite float path),
 * SN_EUNSUPPORTED (in_schema or out_schema is SN_QI8, or the net has several
 * inputs: set their scales with sn_set_qscale), SN_ECUDA, SN_ENOMEM.
 * sn_set_qscale / sn_get_qscale take the ids of sn_add_input too. */
SN_API sn_status sn_calibrate(sn_graph *g, const void *in_dev, void *stream);

/* ---------------- allocation-free Winograd convolution --------------------
 * The paper has no counterpart to this call; it exists for callers that
 * cannot allocate device memory at the point where they run a layer: plug-ins
 * inside a host application that owns every device allocation, services
 * whose memory budget is fixed at start-up, or latency-critical loops where a
 * cudaMalloc (and its implicit synchronisation) is not acceptable.
 *
 * It computes the same conv2 as the graph's "conv2/wino_f2x2_3x3" routine
 * (3x3 kernel, stride 1, dilation 1, groups 1, zero padding `pad` on both
 * axes, bias + act), using the same kernels, but its scratch (the transformed
 * filter U and the Winograd buffers V and M) lives in one fixed device array
 * of SN_NOALLOC_SCRATCH_BYTES that is part of the library image.  A GPU
 * takes that memory when the library's device code is loaded on it: no later
 * than this call's first use there (earlier if CUDA loads modules eagerly,
 * e.g. CUDA_MODULE_LOADING=EAGER, or another entry point of the library
 * loaded them), and it keeps it until the process exits; count it in the
 * fixed memory budget of every device the library runs on.  The call itself
 * never allocates: no cudaMalloc, no cudaFree, no allocator hook.
 *
 *   x_dev    input, logical N x C x H x W stored in `schema` (caller-owned)
 *   w_dev    device fp32 weights [c_out][C][3][3] (caller-owned)
 *   bias_dev device fp32 [c_out] (required)
 *   y_dev    output, N x c_out x P x Q in `schema`, P = H + 2 pad - 2
 *   act      sn_act
 *   stream   cudaStream_t the kernels are launched on (asynchronous)
 *
 * The first call on a device resolves the array's device address (one
 * cudaGetSymbolAddress with that device current); make that first call
 * before any stream capture.  All calls share the one array and it keeps the
 * previous call's contents; every element a call reads is first written by
 * the same call, so nothing needs clearing.  Calls that can overlap on the
 * GPU (different streams, or host threads without ordering) race on the
 * array: serialise them.
 * Errors: SN_EINVAL (NULL pointer, bad extent, schema, pad or act),
 * SN_EUNSUPPORTED (schema.dtype is SN_QI8, which this routine has no form
 * for, or the scratch need exceeds SN_NOALLOC_SCRATCH_BYTES; nothing is
 * launched), SN_ECUDA. */
#define SN_NOALLOC_SCRATCH_BYTES (32u * 1024u * 1024u)
SN_API sn_status sn_conv2d_wino_noalloc(const void *x_dev, sn_schema schema, const int64_t in_nchw[4],
                                        int32_t c_out, int32_t pad, int32_t act, const float *w_dev,
                                        const float *bias_dev, void *y_dev, void *stream);

SN_API const char *sn_last_error(void);

#ifdef __cplusplus
}
#endif
#endif /* SN_H */
