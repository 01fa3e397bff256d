// extern "C" boundary of the library (declared in include/sn.h).  Every entry
// point catches C++ exceptions and turns them into a status, so nothing but
// an sn_status crosses the ABI.
#include <cmath>
#include <cstdio>
#include <cstring>
#include <fstream>
#include <sstream>
#include <string>

#include "sn_internal.h"

namespace sn {
const char *last_error();
sn_status add_layer(Graph *g, int32_t type, const void *params, const int32_t *inputs,
                    int32_t n_inputs, const float *weights, const float *bias, int32_t *out_id);
}  // namespace sn

using namespace sn;

#define SN_GUARD(...)                                                    \
    try {                                                                \
        __VA_ARGS__                                                      \
    } catch (const std::bad_alloc &) {                                   \
        return fail(SN_ENOMEM, "host allocation failed");                \
    } catch (const std::exception &ex) {                                 \
        return fail(SN_EINVAL, std::string("internal error: ") + ex.what()); \
    } catch (...) {                                                      \
        return fail(SN_EINVAL, "internal error");                        \
    }

extern "C" {

const char *sn_last_error(void) { return last_error(); }

const char *sn_routine_name(int32_t routine) { return routine_name(routine); }

const char *sn_variant_name(int32_t routine, int32_t variant) {
    if (!routine_name(routine)) return nullptr;
    return variant_name(routine, variant);
}

const char *sn_candidate_desc(sn_graph *gg, int32_t cand) {
    static thread_local std::string buf;
    try {
        if (!gg) return nullptr;
        Graph *g = reinterpret_cast<Graph *>(gg);
        if (graph_finalize(g) != SN_OK || cand < 0 || cand >= (int32_t)g->cands.size()) return nullptr;
        buf = candidate_desc(*g, cand);
        return buf.c_str();
    } catch (...) {
        return nullptr;
    }
}

sn_status sn_graph_create(const int64_t in_nchw[4], sn_schema in_schema, sn_schema out_schema,
                          const sn_schema *schemas, int32_t n_schemas, sn_alloc_fn alloc,
                          sn_free_fn free_fn, void *alloc_ctx, sn_graph **out) {
    SN_GUARD({
        if (!out || !in_nchw || !schemas || n_schemas < 1 || n_schemas > 16)
            return fail(SN_EINVAL, "sn_graph_create: bad arguments");
        *out = nullptr;
        if ((alloc == nullptr) != (free_fn == nullptr))
            return fail(SN_EINVAL, "sn_graph_create: give both alloc and free, or neither");
        for (int k = 0; k < 4; ++k)
            if (in_nchw[k] < 1) return fail(SN_EINVAL, "sn_graph_create: input extents must be >= 1");
        if (!schema_valid(in_schema) || !schema_valid(out_schema))
            return fail(SN_EINVAL, "sn_graph_create: invalid in/out schema");
        auto *g = new Graph();
        g->in_shape = {in_nchw[0], in_nchw[1], in_nchw[2], in_nchw[3]};
        g->in_schema = in_schema;
        g->out_schema = out_schema;
        for (int32_t i = 0; i < n_schemas; ++i) {
            if (!schema_valid(schemas[i])) {
                delete g;
                return fail(SN_EINVAL, "sn_graph_create: invalid schema in Lambda");
            }
            for (auto &s : g->schemas)
                if (schema_eq(s, schemas[i])) {
                    delete g;
                    return fail(SN_EINVAL, "sn_graph_create: duplicate schema in Lambda");
                }
            g->schemas.push_back(schemas[i]);
        }
        g->n_lambda = n_schemas;
        auto find_or_add = [&](sn_schema s) {
            for (size_t i = 0; i < g->schemas.size(); ++i)
                if (schema_eq(g->schemas[i], s)) return (int32_t)i;
            g->schemas.push_back(s);
            return (int32_t)g->schemas.size() - 1;
        };
        g->in_schema_idx = find_or_add(in_schema);
        g->out_schema_idx = find_or_add(out_schema);
        g->alloc = alloc;
        g->free_fn = free_fn;
        g->alloc_ctx = alloc_ctx;
        *out = reinterpret_cast<sn_graph *>(g);
        return SN_OK;
    })
}

static Graph *G(sn_graph *g) { return reinterpret_cast<Graph *>(g); }

sn_status sn_add_layer(sn_graph *g, int32_t type, const void *params, const int32_t *inputs,
                       int32_t n_inputs, const float *weights, const float *bias,
                       int32_t *out_layer_id) {
    SN_GUARD({
        if (!g || !out_layer_id) return fail(SN_EINVAL, "sn_add_layer: NULL argument");
        return add_layer(G(g), type, params, inputs, n_inputs, weights, bias, out_layer_id);
    })
}

sn_status sn_get_cost_table(sn_graph *gg, sn_cost_table *t) {
    SN_GUARD({
        if (!gg || !t) return fail(SN_EINVAL, "sn_get_cost_table: NULL argument");
        Graph *g = G(gg);
        sn_status rc = graph_finalize(g);
        if (rc != SN_OK) return rc;
        const bool sizes_only = !t->candidates && !t->edges && !t->adapt_cost;
        if (!sizes_only) {
            if (t->n_layers != g->n_layers() || t->n_schemas != g->n_schemas() ||
                t->n_edges != (int32_t)g->edges.size() || t->n_candidates != (int32_t)g->cands.size())
                return fail(SN_EINVAL, "sn_get_cost_table: array sizes do not match the graph");
            if (t->candidates)
                for (size_t c = 0; c < g->cands.size(); ++c) {
                    const Candidate &k = g->cands[c];
                    t->candidates[c] = {k.routine, k.variant, k.schema, k.layer, k.cost, cand_out(k)};
                }
            if (t->edges)
                for (size_t e = 0; e < g->edges.size(); ++e) {
                    t->edges[2 * e] = g->edges[e].first;
                    t->edges[2 * e + 1] = g->edges[e].second;
                }
            if (t->adapt_cost)
                std::memcpy(t->adapt_cost, g->adapt_cost.data(), g->adapt_cost.size() * sizeof(int64_t));
        }
        t->n_layers = g->n_layers();
        t->n_schemas = g->n_schemas();
        t->n_edges = (int32_t)g->edges.size();
        t->n_candidates = (int32_t)g->cands.size();
        return SN_OK;
    })
}

sn_status sn_set_cost_table(sn_graph *gg, const sn_cost_table *t) {
    SN_GUARD({
        if (!gg || !t || !t->candidates || !t->adapt_cost)
            return fail(SN_EINVAL, "sn_set_cost_table: NULL argument");
        Graph *g = G(gg);
        sn_status rc = graph_finalize(g);
        if (rc != SN_OK) return rc;
        if (t->n_layers != g->n_layers() || t->n_schemas != g->n_schemas() ||
            t->n_edges != (int32_t)g->edges.size() || t->n_candidates != (int32_t)g->cands.size())
            return fail(SN_EINVAL, "sn_set_cost_table: sizes do not match the graph");
        for (size_t c = 0; c < g->cands.size(); ++c) {
            const Candidate &k = g->cands[c];
            const sn_candidate &x = t->candidates[c];
            if (x.routine != k.routine || x.variant != k.variant || x.schema != k.schema || x.layer != k.layer ||
                x.out_schema != cand_out(k))
                return fail(SN_EINVAL, "sn_set_cost_table: candidate " + std::to_string(c) + " differs");
            if (x.cost_ns < 0) return fail(SN_EINVAL, "sn_set_cost_table: negative cost");
        }
        const int32_t ns = g->n_schemas();
        for (size_t e = 0; e < g->edges.size(); ++e)
            for (int32_t a = 0; a < ns; ++a) {
                if (t->adapt_cost[(e * ns + a) * ns + a] != 0)
                    return fail(SN_EINVAL, "sn_set_cost_table: void adapt must cost 0");
                for (int32_t b = 0; b < ns; ++b)
                    if (t->adapt_cost[(e * ns + a) * ns + b] < 0)
                        return fail(SN_EINVAL, "sn_set_cost_table: negative adapt cost");
            }
        for (size_t c = 0; c < g->cands.size(); ++c) g->cands[c].cost = t->candidates[c].cost_ns;
        std::memcpy(g->adapt_cost.data(), t->adapt_cost, g->adapt_cost.size() * sizeof(int64_t));
        return SN_OK;
    })
}

sn_status sn_get_schema(sn_graph *gg, int32_t index, sn_schema *out, int32_t *n_schemas) {
    SN_GUARD({
        if (!gg) return fail(SN_EINVAL, "sn_get_schema: NULL graph");
        Graph *g = G(gg);
        if (n_schemas) *n_schemas = g->n_schemas();
        if (out) {
            if (index < 0 || index >= g->n_schemas()) return fail(SN_EINVAL, "schema index out of range");
            *out = g->schemas[index];
        }
        return SN_OK;
    })
}

sn_status sn_profile(sn_graph *gg, const sn_profile_opts *opts, void *stream) {
    SN_GUARD({
        if (!gg) return fail(SN_EINVAL, "sn_profile: NULL graph");
        Graph *g = G(gg);
        sn_status rc = graph_finalize(g);
        if (rc != SN_OK) return rc;
        sn_profile_opts o{3, 20, 2, 5};
        if (opts) o = *opts;
        if (o.warmup < 0 || o.iters < 1 || o.topk < 0 || o.passes < 1 || o.iters > 10000)
            return fail(SN_EINVAL, "sn_profile: bad options");
        return profile_graph(g, o, static_cast<cudaStream_t>(stream));
    })
}

static sn_status fill_path(Graph *g, const std::vector<int32_t> &pc, int64_t total, sn_path *out) {
    const int32_t n = g->n_layers();
    std::vector<int32_t> schema_of(n);
    for (int32_t i = 0; i < n; ++i) schema_of[i] = g->cands[pc[i]].schema;
    g->path_cand = pc;
    g->path_total = total;
    g->has_path = true;
    invalidate_plan(g);
    if (out) {
        if ((out->schema || out->candidate) && out->n_layers < n)
            return fail(SN_EINVAL, "sn_path arrays too small");
        out->total_ns = total;
        out->n_layers = n;
        for (int32_t i = 0; i < n; ++i) {
            if (out->schema) out->schema[i] = schema_of[i];
            if (out->candidate) out->candidate[i] = pc[i];
        }
    }
    return SN_OK;
}

sn_status sn_select_path(sn_graph *gg, int32_t method, sn_path *out) {
    SN_GUARD({
        if (!gg) return fail(SN_EINVAL, "sn_select_path: NULL graph");
        Graph *g = G(gg);
        sn_status rc = graph_finalize(g);
        if (rc != SN_OK) return rc;
        if (method != SN_SELECT_DPRS && method != SN_SELECT_BRUTE) return fail(SN_EINVAL, "sn_select_path: unknown method");
        std::vector<int32_t> cand_of;
        int64_t total = kInf;
        rc = select_path(*g, method, cand_of, total);
        if (rc != SN_OK) return rc;
        return fill_path(g, cand_of, total, out);
    })
}

sn_status sn_set_path(sn_graph *gg, const int32_t *candidate, int32_t n_layers) {
    SN_GUARD({
        if (!gg || !candidate) return fail(SN_EINVAL, "sn_set_path: NULL argument");
        Graph *g = G(gg);
        sn_status rc = graph_finalize(g);
        if (rc != SN_OK) return rc;
        const int32_t n = g->n_layers();
        if (n_layers != n) return fail(SN_EINVAL, "sn_set_path: wrong number of layers");
        int64_t total = 0;
        std::vector<int32_t> sch(n);
        for (int32_t i = 0; i < n; ++i) {
            const int32_t c = candidate[i];
            if (c < g->cand_begin[i] || c >= g->cand_begin[i + 1])
                return fail(SN_EINVAL, "sn_set_path: candidate " + std::to_string(c) +
                                           " does not belong to layer " + std::to_string(i));
            sch[i] = g->cands[c].schema;
            total = sat_add(total, g->cands[c].cost);
        }
        for (size_t e = 0; e < g->edges.size(); ++e) {
            auto [u, v] = g->edges[e];
            if (sch[u] != sch[v]) total = sat_add(total, g->adapt((int32_t)e, sch[u], sch[v]));
        }
        g->path_cand.assign(candidate, candidate + n);
        g->path_total = total;
        g->has_path = true;
        invalidate_plan(g);
        return SN_OK;
    })
}

sn_status sn_set_option(sn_graph *gg, int32_t option, int64_t value) {
    SN_GUARD({
        if (!gg) return fail(SN_EINVAL, "sn_set_option: NULL graph");
        Graph *g = G(gg);
        if (option == SN_OPT_CUDA_GRAPH) {
            g->opt_graph = value ? 1 : 0;
            if (g->gexec) {
                cudaGraphExecDestroy(g->gexec);
                g->gexec = nullptr;
            }
        } else if (option == SN_OPT_CHECK) {
            g->opt_check = value ? 1 : 0;
        } else if (option == SN_OPT_WAIT_LIMIT) {
            if (value < 0) return fail(SN_EINVAL, "sn_set_option: the wait limit is a cycle count >= 0");
            if (g->opt_wait_limit != value) {
                g->opt_wait_limit = value;
                if (g->gexec) {  // the limit is a launch argument baked into a captured graph
                    cudaGraphExecDestroy(g->gexec);
                    g->gexec = nullptr;
                }
            }
        } else if (option == SN_OPT_SHARE_BUFFERS) {
            if (g->opt_share != (value ? 1 : 0)) {
                g->opt_share = value ? 1 : 0;
                invalidate_plan(g);
            }
        } else if (option == SN_OPT_CHAIN) {
            if (g->opt_chain != (value ? 1 : 0)) {
                g->opt_chain = value ? 1 : 0;
                invalidate_plan(g);
            }
        } else {
            return fail(SN_EINVAL, "sn_set_option: unknown option");
        }
        return SN_OK;
    })
}

static sn_status check_device(Graph *g, cudaStream_t st) {
    SN_CUDA_TRY(cudaStreamSynchronize(st));
    int word = 0;
    SN_CUDA_TRY(cudaMemcpy(&word, k::device_error_word(), sizeof(int), cudaMemcpyDeviceToHost));
    if (word) {
        const int zero = 0;
        cudaMemcpy(k::device_error_word(), &zero, sizeof(int), cudaMemcpyHostToDevice);
        // a stopped stream-K launch may have left tile counts behind
        if (g->tile_counts.ptr) cudaMemset(g->tile_counts.ptr, 0, g->tile_counts.bytes);
        return fail(SN_ETIMEOUT, "device error word set: " + std::to_string(word) +
                                     " (a bounded wait in a kernel gave up)");
    }
    return SN_OK;
}

static sn_status run_io(Graph *g, const IoPtrs &io, cudaStream_t st) {
    if (!g->has_path) return fail(SN_ESTATE, "sn_run: select or set a routine path first");
    if ((int32_t)io.in.size() != g->n_in() || (int32_t)io.out.size() != g->n_out())
        return fail(SN_EINVAL, "sn_run: the net has " + std::to_string(g->n_in()) + " input(s) and " +
                                   std::to_string(g->n_out()) + " output(s) (sn_run_multi)");
    for (const void *p : io.in)
        if (!p) return fail(SN_EINVAL, "sn_run: NULL input buffer");
    for (void *p : io.out)
        if (!p) return fail(SN_EINVAL, "sn_run: NULL output buffer");
    if (!g->plan_valid) {
        sn_status rc = build_plan(g, st);
        if (rc != SN_OK) return rc;
    }
    sn_status rc = SN_OK;
    if (g->opt_graph && st != nullptr) {
        if (!g->gexec || g->gexec_in != io.in || g->gexec_out != io.out || g->gexec_stream != st) {
            if (g->gexec) {
                cudaGraphExecDestroy(g->gexec);
                g->gexec = nullptr;
            }
            cudaGraph_t graph = nullptr;
            SN_CUDA_TRY(cudaStreamBeginCapture(st, cudaStreamCaptureModeThreadLocal));
            rc = run_plan(g, io, st, nullptr);
            cudaError_t ce = cudaStreamEndCapture(st, &graph);
            if (rc != SN_OK) {
                if (graph) cudaGraphDestroy(graph);
                return rc;
            }
            if (ce != cudaSuccess) return fail(SN_ECUDA, std::string("graph capture: ") + cudaGetErrorString(ce));
            ce = cudaGraphInstantiate(&g->gexec, graph, 0);
            cudaGraphDestroy(graph);
            if (ce != cudaSuccess) {
                g->gexec = nullptr;
                return fail(SN_ECUDA, std::string("graph instantiate: ") + cudaGetErrorString(ce));
            }
            g->gexec_in = io.in;
            g->gexec_out = io.out;
            g->gexec_stream = st;
        }
        SN_CUDA_TRY(cudaGraphLaunch(g->gexec, st));
    } else {
        rc = run_plan(g, io, st, nullptr);
        if (rc != SN_OK) return rc;
    }
    if (g->opt_check) return check_device(g, st);
    return SN_OK;
}

sn_status sn_run(sn_graph *gg, const void *in_dev, void *out_dev, void *stream) {
    SN_GUARD({
        if (!gg || !in_dev || !out_dev) return fail(SN_EINVAL, "sn_run: NULL argument");
        IoPtrs io;
        io.in = {in_dev};
        io.out = {out_dev};
        return run_io(G(gg), io, static_cast<cudaStream_t>(stream));
    })
}

sn_status sn_run_host(sn_graph *gg, const void *in_host, void *out_host, void *stream) {
    SN_GUARD({
        if (!gg || !in_host || !out_host) return fail(SN_EINVAL, "sn_run_host: NULL argument");
        Graph *g = G(gg);
        sn_status rc = graph_finalize(g);
        if (rc != SN_OK) return rc;
        if (g->n_in() != 1 || g->n_out() != 1)
            return fail(SN_EINVAL, "sn_run_host: the net has several inputs or outputs");
        const Shape &os = g->layers[g->layers.back().inputs[0]].out;
        const size_t in_bytes = (size_t)g->in_shape.numel() * dtype_size(g->in_schema.dtype);
        const size_t out_bytes = (size_t)os.numel() * dtype_size(g->out_schema.dtype);
        if (g->host_in.bytes < in_bytes) {
            dev_free(g, &g->host_in);
            if ((rc = dev_alloc(g, in_bytes, &g->host_in)) != SN_OK) return rc;
        }
        if (g->host_out.bytes < out_bytes) {
            dev_free(g, &g->host_out);
            if ((rc = dev_alloc(g, out_bytes, &g->host_out)) != SN_OK) return rc;
        }
        cudaStream_t st = static_cast<cudaStream_t>(stream);
        // the upload runs on the graph's copy stream into one of two landing
        // buffers (alternating per call), after the call two before this one
        // has copied that buffer out; the caller's stream waits for it and
        // copies it into the net's input buffer (the captured CUDA graph keeps
        // one input address).  So the upload of one call overlaps the net of
        // the previous one, and everything stays in order on `stream`.
        if (!g->copy_stream) {
            SN_CUDA_TRY(cudaStreamCreateWithFlags(&g->copy_stream, cudaStreamNonBlocking));
            for (int i = 0; i < 2; ++i) {
                SN_CUDA_TRY(cudaEventCreateWithFlags(&g->land_done[i], cudaEventDisableTiming));
                SN_CUDA_TRY(cudaEventCreateWithFlags(&g->land_free[i], cudaEventDisableTiming));
            }
        }
        const int b = g->land_next;
        if (g->host_land[b].bytes < in_bytes) {
            if (g->land_used[b]) SN_CUDA_TRY(cudaEventSynchronize(g->land_free[b]));
            dev_free(g, &g->host_land[b]);
            g->land_used[b] = false;
            if ((rc = dev_alloc(g, in_bytes, &g->host_land[b])) != SN_OK) return rc;
        }
        if (g->land_used[b]) SN_CUDA_TRY(cudaStreamWaitEvent(g->copy_stream, g->land_free[b], 0));
        SN_CUDA_TRY(cudaMemcpyAsync(g->host_land[b].ptr, in_host, in_bytes, cudaMemcpyHostToDevice, g->copy_stream));
        SN_CUDA_TRY(cudaEventRecord(g->land_done[b], g->copy_stream));
        SN_CUDA_TRY(cudaStreamWaitEvent(st, g->land_done[b], 0));
        SN_CUDA_TRY(cudaMemcpyAsync(g->host_in.ptr, g->host_land[b].ptr, in_bytes, cudaMemcpyDeviceToDevice, st));
        SN_CUDA_TRY(cudaEventRecord(g->land_free[b], st));
        g->land_used[b] = true;
        g->land_next = b ^ 1;
        IoPtrs io;
        io.in = {g->host_in.ptr};
        io.out = {g->host_out.ptr};
        if ((rc = run_io(g, io, st)) != SN_OK) return rc;
        SN_CUDA_TRY(cudaMemcpyAsync(out_host, g->host_out.ptr, out_bytes, cudaMemcpyDeviceToHost, st));
        return SN_OK;
    })
}

sn_status sn_run_multi(sn_graph *gg, const void *const *in_devs, int32_t n_in, void *const *out_devs, int32_t n_out,
                       void *stream) {
    SN_GUARD({
        if (!gg || !in_devs || !out_devs || n_in < 1 || n_out < 1) return fail(SN_EINVAL, "sn_run_multi: bad argument");
        IoPtrs io;
        io.in.assign(in_devs, in_devs + n_in);
        io.out.assign(out_devs, out_devs + n_out);
        return run_io(G(gg), io, static_cast<cudaStream_t>(stream));
    })
}

sn_status sn_fuse_residual(sn_graph *gg, int32_t *new_id, int32_t n_ids, int32_t *n_fused) {
    SN_GUARD({
        if (!gg) return fail(SN_EINVAL, "sn_fuse_residual: NULL graph");
        Graph *g = G(gg);
        if (new_id && n_ids != (int32_t)g->user.size())
            return fail(SN_EINVAL, "sn_fuse_residual: new_id must have one entry per layer added (" +
                                       std::to_string(g->user.size()) + ")");
        std::vector<int32_t> map;
        sn_status rc = fuse_residual(g, map, n_fused);
        if (rc != SN_OK) return rc;
        if (new_id)
            for (size_t i = 0; i < map.size(); ++i) new_id[i] = map[i];
        return SN_OK;
    })
}

sn_status sn_add_input(sn_graph *gg, const int64_t in_nchw[4], int32_t *input_id) {
    SN_GUARD({
        if (!gg || !in_nchw || !input_id) return fail(SN_EINVAL, "sn_add_input: NULL argument");
        return add_input(G(gg), in_nchw, input_id);
    })
}

sn_status sn_set_outputs(sn_graph *gg, const int32_t *layer_ids, int32_t n) {
    SN_GUARD({
        if (!gg) return fail(SN_EINVAL, "sn_set_outputs: NULL graph");
        return set_outputs(G(gg), layer_ids, n);
    })
}

sn_status sn_get_io(sn_graph *gg, int32_t *n_inputs, int32_t *n_outputs) {
    SN_GUARD({
        if (!gg) return fail(SN_EINVAL, "sn_get_io: NULL graph");
        Graph *g = G(gg);
        if (n_inputs) *n_inputs = g->n_in();
        if (n_outputs) *n_outputs = g->n_out();
        return SN_OK;
    })
}

sn_status sn_run_timed(sn_graph *gg, const void *in_dev, void *out_dev, void *stream,
                       float *layer_ms, float *edge_ms) {
    SN_GUARD({
        if (!gg || !in_dev || !out_dev) return fail(SN_EINVAL, "sn_run_timed: NULL argument");
        Graph *g = G(gg);
        if (!g->has_path) return fail(SN_ESTATE, "sn_run_timed: select or set a routine path first");
        cudaStream_t st = static_cast<cudaStream_t>(stream);
        if (!g->plan_valid) {
            sn_status rc = build_plan(g, st);
            if (rc != SN_OK) return rc;
        }
        if (g->n_in() != 1 || g->n_out() != 1)
            return fail(SN_EINVAL, "sn_run_timed: the net has several inputs or outputs");
        IoPtrs io;
        io.in = {in_dev};
        io.out = {out_dev};
        std::vector<float> op_ms;
        sn_status rc = run_plan_timed(g, io, st, &op_ms);
        if (rc != SN_OK) return rc;
        if (layer_ms)
            for (int32_t i = 0; i < g->n_layers(); ++i) layer_ms[i] = 0.f;
        if (edge_ms)
            for (size_t e = 0; e < g->edges.size(); ++e) edge_ms[e] = 0.f;
        for (size_t q = 0; q < g->plan.size(); ++q) {
            const PlanOp &op = g->plan[q];
            if (op.kind == PlanOp::LAYER && layer_ms) layer_ms[op.layer] += op_ms[q];
            if (op.kind == PlanOp::ADAPT && edge_ms && op.edge >= 0) edge_ms[op.edge] += op_ms[q];
        }
        if (g->opt_check) return check_device(g, st);
        return SN_OK;
    })
}

sn_status sn_plan_stats(sn_graph *gg, int32_t *n_ops, int32_t *n_kernels, void *stream) {
    SN_GUARD({
        if (!gg) return fail(SN_EINVAL, "sn_plan_stats: NULL graph");
        Graph *g = G(gg);
        if (!g->has_path) return fail(SN_ESTATE, "sn_plan_stats: select or set a routine path first");
        if (!g->plan_valid) {
            sn_status rc = build_plan(g, static_cast<cudaStream_t>(stream));
            if (rc != SN_OK) return rc;
        }
        int32_t kern = 0;
        for (size_t q = 0; q < g->plan.size(); ++q) {
            const PlanOp &op = g->plan[q];
            if (q < g->op_chain.size() && g->op_chain[q] >= 0) {  // one launch per chain
                kern += g->chains[g->op_chain[q]].first_op == (int32_t)q ? 1 : 0;
            } else if (op.kind == PlanOp::ADAPT) {
                kern += 1;
            } else {
                const Candidate &c = g->cands[op.cand];
                const Layer &L = g->layers[op.layer];
                std::vector<Shape> in;
                for (int32_t j : L.inputs) in.push_back(g->layers[j].out);
                kern += kernels_per_launch(c.routine, c.variant, L, in, g->schemas[c.schema]);
            }
        }
        if (n_ops) *n_ops = (int32_t)g->plan.size();
        if (n_kernels) *n_kernels = kern;
        return SN_OK;
    })
}

sn_status sn_plan_memory(sn_graph *gg, int64_t *arena_bytes, int64_t *unshared_bytes, void *stream) {
    SN_GUARD({
        if (!gg) return fail(SN_EINVAL, "sn_plan_memory: NULL graph");
        Graph *g = G(gg);
        if (!g->has_path) return fail(SN_ESTATE, "sn_plan_memory: select or set a routine path first");
        if (!g->plan_valid) {
            sn_status rc = build_plan(g, static_cast<cudaStream_t>(stream));
            if (rc != SN_OK) return rc;
        }
        if (arena_bytes) *arena_bytes = (int64_t)g->arena.bytes;
        if (unshared_bytes) *unshared_bytes = (int64_t)g->arena_unshared;
        return SN_OK;
    })
}

sn_status sn_layer_shape(sn_graph *gg, int32_t layer, int64_t out_nchw[4]) {
    SN_GUARD({
        if (!gg || !out_nchw) return fail(SN_EINVAL, "sn_layer_shape: NULL argument");
        Graph *g = G(gg);
        sn_status rc = graph_finalize(g);
        if (rc != SN_OK) return rc;
        if (layer < 0 || layer >= g->n_layers()) return fail(SN_EINVAL, "layer out of range");
        const Shape &s = g->layers[layer].out;
        out_nchw[0] = s.n, out_nchw[1] = s.c, out_nchw[2] = s.h, out_nchw[3] = s.w;
        return SN_OK;
    })
}

// ---- plan files: a small JSON document with integer arrays ----
sn_status sn_save_plan(sn_graph *gg, const char *path) {
    SN_GUARD({
        if (!gg || !path) return fail(SN_EINVAL, "sn_save_plan: NULL argument");
        Graph *g = G(gg);
        sn_status rc = graph_finalize(g);
        if (rc != SN_OK) return rc;
        std::ofstream f(path);
        if (!f) return fail(SN_EINVAL, std::string("cannot open ") + path);
        f << "{\n \"format\": \"softneuro-gb300-plan-1\",\n";
        f << " \"n_layers\": " << g->n_layers() << ",\n \"n_schemas\": " << g->n_schemas()
          << ",\n \"n_edges\": " << g->edges.size() << ",\n \"n_candidates\": " << g->cands.size() << ",\n";
        f << " \"candidates\": [";
        for (size_t c = 0; c < g->cands.size(); ++c) {
            const Candidate &k = g->cands[c];
            f << (c ? ", " : "") << "[" << k.routine << ", " << k.variant << ", " << k.schema << ", "
              << k.layer << ", " << k.cost << "]";
        }
        f << "],\n \"adapt_cost\": [";
        for (size_t i = 0; i < g->adapt_cost.size(); ++i) f << (i ? ", " : "") << g->adapt_cost[i];
        f << "],\n \"path\": [";
        if (g->has_path)
            for (size_t i = 0; i < g->path_cand.size(); ++i) f << (i ? ", " : "") << g->path_cand[i];
        f << "],\n \"total_ns\": " << (g->has_path ? g->path_total : -1) << "\n}\n";
        if (!f) return fail(SN_EINVAL, "write failed");
        return SN_OK;
    })
}

static bool read_int_array(const std::string &doc, const std::string &key, std::vector<int64_t> &out) {
    const size_t k = doc.find("\"" + key + "\"");
    if (k == std::string::npos) return false;
    size_t p = doc.find('[', k);
    if (p == std::string::npos) return false;
    int depth = 0;
    std::string num;
    out.clear();
    for (; p < doc.size(); ++p) {
        const char ch = doc[p];
        if (ch == '[') {
            ++depth;
        } else if (ch == ']' || ch == ',') {
            if (!num.empty()) {
                out.push_back(std::stoll(num));
                num.clear();
            }
            if (ch == ']' && --depth == 0) return true;
        } else if ((ch >= '0' && ch <= '9') || ch == '-') {
            num += ch;
        }
    }
    return false;
}

static bool read_int(const std::string &doc, const std::string &key, int64_t &v) {
    const size_t k = doc.find("\"" + key + "\"");
    if (k == std::string::npos) return false;
    size_t p = doc.find(':', k);
    if (p == std::string::npos) return false;
    v = std::stoll(doc.substr(p + 1));
    return true;
}

sn_status sn_load_plan(sn_graph *gg, const char *path) {
    SN_GUARD({
        if (!gg || !path) return fail(SN_EINVAL, "sn_load_plan: NULL argument");
        Graph *g = G(gg);
        sn_status rc = graph_finalize(g);
        if (rc != SN_OK) return rc;
        std::ifstream f(path);
        if (!f) return fail(SN_EINVAL, std::string("cannot open ") + path);
        std::stringstream ss;
        ss << f.rdbuf();
        const std::string doc = ss.str();
        int64_t nl, ns, ne, nc, total;
        std::vector<int64_t> cands, ac, pth;
        if (!read_int(doc, "n_layers", nl) || !read_int(doc, "n_schemas", ns) || !read_int(doc, "n_edges", ne) ||
            !read_int(doc, "n_candidates", nc) || !read_int(doc, "total_ns", total) ||
            !read_int_array(doc, "candidates", cands) || !read_int_array(doc, "adapt_cost", ac) ||
            !read_int_array(doc, "path", pth))
            return fail(SN_EINVAL, "sn_load_plan: malformed plan file");
        if (nl != g->n_layers() || ns != g->n_schemas() || ne != (int64_t)g->edges.size() ||
            nc != (int64_t)g->cands.size() || cands.size() != (size_t)nc * 5 || ac.size() != g->adapt_cost.size())
            return fail(SN_EINVAL, "sn_load_plan: plan describes a different net");
        for (size_t c = 0; c < g->cands.size(); ++c) {
            const Candidate &k = g->cands[c];
            if (cands[5 * c] != k.routine || cands[5 * c + 1] != k.variant || cands[5 * c + 2] != k.schema ||
                cands[5 * c + 3] != k.layer)
                return fail(SN_EINVAL, "sn_load_plan: candidate list differs");
        }
        if (!pth.empty()) {
            if ((int64_t)pth.size() != nl) return fail(SN_EINVAL, "sn_load_plan: bad path length");
            for (int32_t i = 0; i < g->n_layers(); ++i)
                if (pth[i] < g->cand_begin[i] || pth[i] >= g->cand_begin[i + 1])
                    return fail(SN_EINVAL, "sn_load_plan: path candidate out of range");
        }
        for (size_t c = 0; c < g->cands.size(); ++c) g->cands[c].cost = cands[5 * c + 4];
        for (size_t i = 0; i < ac.size(); ++i) g->adapt_cost[i] = ac[i];
        if (!pth.empty()) {
            g->path_cand.assign(pth.begin(), pth.end());
            g->path_total = total;
            g->has_path = true;
        } else {
            g->has_path = false;
        }
        invalidate_plan(g);
        return SN_OK;
    })
}

void sn_graph_destroy(sn_graph *g) {
    try {
        delete G(g);
    } catch (...) {
    }
}

sn_status sn_convert(const void *x_dev, sn_schema from, void *y_dev, sn_schema to,
                     const int64_t nchw[4], void *stream) {
    SN_GUARD({
        if (!x_dev || !y_dev || !nchw) return fail(SN_EINVAL, "sn_convert: NULL argument");
        if (!schema_valid(from) || !schema_valid(to)) return fail(SN_EINVAL, "sn_convert: invalid schema");
        for (int k = 0; k < 4; ++k)
            if (nchw[k] < 0) return fail(SN_EINVAL, "sn_convert: negative extent");
        if (from.dtype == SN_QI8 || to.dtype == SN_QI8)
            return fail(SN_EINVAL, "sn_convert: a qint8 side needs its scale (sn_convert_q)");
        const Shape s{nchw[0], nchw[1], nchw[2], nchw[3]};
        if (s.numel() == 0) return SN_OK;
        SN_CUDA_TRY(k::convert(x_dev, from.dtype, from.layout, y_dev, to.dtype, to.layout, s,
                               static_cast<cudaStream_t>(stream)));
        return SN_OK;
    })
}

sn_status sn_convert_q(const void *x_dev, sn_schema from, void *y_dev, sn_schema to, const int64_t nchw[4],
                       float qscale, void *stream) {
    SN_GUARD({
        if (!x_dev || !y_dev || !nchw) return fail(SN_EINVAL, "sn_convert_q: NULL argument");
        if (!schema_valid(from) || !schema_valid(to)) return fail(SN_EINVAL, "sn_convert_q: invalid schema");
        if (from.dtype != SN_QI8 && to.dtype != SN_QI8) return fail(SN_EINVAL, "sn_convert_q: no qint8 side");
        if (!(qscale > 0.0f) || !std::isfinite(qscale)) return fail(SN_EINVAL, "sn_convert_q: bad scale");
        for (int k = 0; k < 4; ++k)
            if (nchw[k] < 0) return fail(SN_EINVAL, "sn_convert_q: negative extent");
        const Shape s{nchw[0], nchw[1], nchw[2], nchw[3]};
        if (s.numel() == 0) return SN_OK;
        SN_CUDA_TRY(k::convert_q8(x_dev, from.dtype, from.layout, y_dev, to.dtype, to.layout, s, qscale,
                                  static_cast<cudaStream_t>(stream)));
        return SN_OK;
    })
}

static float *qscale_ref(Graph *g, int32_t id, bool internal) {
    const int32_t m_in = g->n_in();
    if (id == -1) return internal ? &g->layers[0].qscale : &g->in_qscale;
    if (id < -1 && id >= -m_in) {  // another net input
        const int32_t k = -1 - id;
        return internal ? &g->layers[k].qscale : &g->extra_in_qscale[k - 1];
    }
    if (id < 0 || id >= (int32_t)g->user.size()) return nullptr;
    return internal ? &g->layers[id + m_in].qscale : &g->user[id].qscale;
}

sn_status sn_set_qscale(sn_graph *gg, int32_t layer_id, float scale) {
    SN_GUARD({
        if (!gg) return fail(SN_EINVAL, "sn_set_qscale: NULL graph");
        Graph *g = G(gg);
        if (!(scale > 0.0f) || !std::isfinite(scale)) return fail(SN_EINVAL, "sn_set_qscale: bad scale");
        float *u = qscale_ref(g, layer_id, false);
        if (!u) return fail(SN_EINVAL, "sn_set_qscale: bad layer id");
        *u = scale;
        if (g->finalized) *qscale_ref(g, layer_id, true) = scale;
        invalidate_plan(g);
        return SN_OK;
    })
}

sn_status sn_get_qscale(sn_graph *gg, int32_t layer_id, float *scale) {
    SN_GUARD({
        if (!gg || !scale) return fail(SN_EINVAL, "sn_get_qscale: NULL argument");
        Graph *g = G(gg);
        const float *u = qscale_ref(g, layer_id, false);
        if (!u) return fail(SN_EINVAL, "sn_get_qscale: bad layer id");
        *scale = *u;
        return SN_OK;
    })
}

sn_status sn_calibrate(sn_graph *gg, const void *in_dev, void *stream) {
    SN_GUARD({
        if (!gg || !in_dev) return fail(SN_EINVAL, "sn_calibrate: NULL argument");
        Graph *g = G(gg);
        sn_status rc = graph_finalize(g);
        if (rc != SN_OK) return rc;
        if (g->in_schema.dtype == SN_QI8 || g->out_schema.dtype == SN_QI8)
            return fail(SN_EUNSUPPORTED, "sn_calibrate: the net input and output must be float");
        if (g->n_in() != 1)
            return fail(SN_EUNSUPPORTED, "sn_calibrate: nets with several inputs take their scales from sn_set_qscale");
        rc = calibrate(g, in_dev, static_cast<cudaStream_t>(stream));
        if (rc != SN_OK) return rc;
        // mirror into the layers as added
        g->in_qscale = g->layers[0].qscale;
        for (size_t u = 0; u < g->user.size(); ++u) g->user[u].qscale = g->layers[u + g->n_in()].qscale;
        return SN_OK;
    })
}

}  // extern "C"
