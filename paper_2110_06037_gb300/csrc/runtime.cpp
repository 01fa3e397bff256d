// Plan construction, execution and profiling.
//
// Plan (inference with the tuned path, section III-A step 3): every layer
// runs its selected routine; an adapt routine is inserted on every edge whose
// endpoint schemas differ (section III-C; one conversion per edge, as Def. 1
// charges one adapt per edge).  Activations live in graph-owned buffers; the
// net input and output are the caller's buffers.
//
// Profiling (section III-C): unit profiling of every candidate, deduplicated
// by layer signature, then integrated profiling of the best candidates per
// (layer, schema) inside whole-net passes.
#include <algorithm>
#include <cstdio>
#include <cstring>
#include <sstream>
#include <string>

#include "sn_internal.h"

namespace sn {

static sn_status schema_slot(Graph *g, Shape s, sn_schema sc, float qscale) {
    g->slots.push_back({});
    g->slot_shape.push_back(s);
    g->slot_schema.push_back(sc);
    g->slot_qscale.push_back(qscale);
    return SN_OK;
}

// an adapt between two schemas; a qint8 side uses the blob's scale
static cudaError_t convert_blob(const void *x, sn_schema a, void *y, sn_schema b, Shape s, float qscale,
                                cudaStream_t st) {
    if (a.dtype == SN_QI8 || b.dtype == SN_QI8)
        return k::convert_q8(x, a.dtype, a.layout, y, b.dtype, b.layout, s, qscale, st);
    return k::convert(x, a.dtype, a.layout, y, b.dtype, b.layout, s, st);
}

// stand-in scale of qint8 blobs while profiling (timing does not depend on it)
constexpr float kProfileQScale = 1.0f / 64.0f;

static bool chain_eligible(const Graph *g, const PlanOp &op);

// Activation buffers by liveness (the plan step of section III-C): every
// graph-owned blob is live from the op that writes it to the last op that
// reads it, in plan order (an op's inputs and its output are live together,
// so no op writes over what it reads); blobs whose live ranges overlap get
// disjoint places in one arena, the others may share bytes.  Ops of a chained
// launch run at once, so what they touch is live across the whole chain.
// Placement: largest blob first, at the lowest offset (256-byte aligned) free
// of every placed blob it is live with.
// The zeroed counters of the stream-K tensor-core routines (one per tile and
// epilogue warp; every launch leaves them zeroed): allocated once per graph.
sn_status ensure_tile_counts(Graph *g, cudaStream_t st) {
    if (g->tile_counts.ptr) return SN_OK;
    sn_status rc = dev_alloc(g, kTileCounts * sizeof(int), &g->tile_counts);
    if (rc != SN_OK) return rc;
    if (cudaMemsetAsync(g->tile_counts.ptr, 0, g->tile_counts.bytes, st) != cudaSuccess)
        return fail(SN_ECUDA, "stream-K counters: memset failed");
    return SN_OK;
}

static sn_status place_slots(Graph *g) {
    const size_t ns = g->slots.size();
    std::vector<int32_t> first(ns, INT32_MAX), last(ns, -1);
    auto touch = [&](int32_t s, int32_t a, int32_t b) {
        if (s < 0) return;
        first[s] = std::min(first[s], a);
        last[s] = std::max(last[s], b);
    };
    for (size_t q = 0; q < g->plan.size(); ++q) {
        const PlanOp &op = g->plan[q];
        for (int32_t s : op.in_slots) touch(s, (int32_t)q, (int32_t)q);
        touch(op.out_slot, (int32_t)q, (int32_t)q);
    }
    if (g->opt_chain && !g->profiling)
        for (const auto &r : chain_runs(g))
            for (int32_t q = r.first; q <= r.second; ++q) {
                for (int32_t s : g->plan[q].in_slots) touch(s, r.first, r.second);
                touch(g->plan[q].out_slot, r.first, r.second);
            }
    struct Item {
        size_t s, bytes, off;
    };
    std::vector<Item> items;
    size_t unshared = 0;
    for (size_t s = g->n_ext; s < ns; ++s) {
        if (last[s] < 0) continue;  // never referenced
        const size_t bytes = ((size_t)g->slot_shape[s].numel() * dtype_size(g->slot_schema[s].dtype) + 255) & ~size_t(255);
        items.push_back({s, bytes, 0});
        unshared += bytes;
    }
    std::sort(items.begin(), items.end(),
              [](const Item &a, const Item &b) { return a.bytes != b.bytes ? a.bytes > b.bytes : a.s < b.s; });
    size_t total = 0;
    for (size_t i = 0; i < items.size(); ++i) {
        Item &it = items[i];
        std::vector<std::pair<size_t, size_t>> busy;  // [off, end) of placed blobs live with this one
        for (size_t j = 0; j < i; ++j) {
            const Item &o = items[j];
            if (!g->opt_share || (first[o.s] <= last[it.s] && first[it.s] <= last[o.s]))
                busy.push_back({o.off, o.off + o.bytes});
        }
        std::sort(busy.begin(), busy.end());
        size_t off = 0;
        for (const auto &b : busy) {
            if (off + it.bytes <= b.first) break;
            off = std::max(off, b.second);
        }
        it.off = off;
        total = std::max(total, off + it.bytes);
    }
    sn_status rc = dev_alloc(g, total, &g->arena);
    if (rc != SN_OK) return rc;
    for (const Item &it : items) {
        g->slots[it.s].ptr = static_cast<uint8_t *>(g->arena.ptr) + it.off;
        g->slots[it.s].bytes = it.bytes;
        g->slots[it.s].view = true;
    }
    g->arena_unshared = unshared;
    return SN_OK;
}

sn_status build_plan(Graph *g, cudaStream_t st) {
    if (!g->has_path) return fail(SN_ESTATE, "no routine path selected");
    invalidate_plan(g);
    for (auto &b : g->slots) dev_free(g, &b);
    dev_free(g, &g->arena);
    g->arena_unshared = 0;
    g->slots.clear();
    g->slot_shape.clear();
    g->slot_schema.clear();
    g->slot_qscale.clear();
    const int32_t n = g->n_layers();
    const int32_t m_in = g->n_in();
    const Layer &OL = g->layers[n - 1];  // auxiliary output layer: its inputs are the net outputs
    const int32_t m_out = (int32_t)OL.inputs.size();
    // the schema each layer's routine reads its inputs in and writes its output in
    std::vector<sn_schema> sch(n), sch_out(n);
    for (int32_t i = 0; i < n; ++i) {
        sch[i] = g->schemas[g->cands[g->path_cand[i]].schema];
        sch_out[i] = g->schemas[cand_out(g->cands[g->path_cand[i]])];
    }
    // external slots: the caller's input buffers 0..m_in-1, then its output
    // buffers m_in..m_in+m_out-1
    for (int32_t k = 0; k < m_in; ++k) schema_slot(g, g->layers[k].out, g->in_schema, g->layers[k].qscale);
    for (int32_t q = 0; q < m_out; ++q) {
        const Layer &src = g->layers[OL.inputs[q]];
        schema_slot(g, src.out, g->out_schema, src.qscale);
    }
    g->n_ext = m_in + m_out;
    std::vector<int32_t> out_slot(n, -1);
    for (int32_t k = 0; k < m_in; ++k) out_slot[k] = k;
    // output index of each layer that is a net output (-1 otherwise)
    std::vector<int32_t> out_index(n, -1);
    for (int32_t q = 0; q < m_out; ++q)
        if (OL.inputs[q] >= m_in) out_index[OL.inputs[q]] = q;
    size_t ws = 0;
    for (int32_t i = m_in; i < n; ++i) {
        const Layer &L = g->layers[i];
        PlanOp op;
        op.kind = PlanOp::LAYER;
        op.layer = i;
        op.cand = g->path_cand[i];
        for (size_t k = 0; k < L.inputs.size(); ++k) {
            const int32_t j = L.inputs[k];
            int32_t e = -1;
            for (size_t q = 0; q < g->edges.size(); ++q)
                if (g->edges[q].first == j && g->edges[q].second == i) {
                    e = (int32_t)q;
                    if (k == 1 && L.inputs[0] == j) {  // second edge of add(x, x)
                        for (size_t q2 = q + 1; q2 < g->edges.size(); ++q2)
                            if (g->edges[q2].first == j && g->edges[q2].second == i) {
                                e = (int32_t)q2;
                                break;
                            }
                    }
                    break;
                }
            int32_t src = out_slot[j];
            const bool same = schema_eq(sch_out[j], sch[i]);
            if (i == n - 1) {
                // output layer: adapt into the caller's buffer unless the
                // producer already wrote there
                if (!same || out_slot[j] != m_in + (int32_t)k) {
                    PlanOp a;
                    a.kind = PlanOp::ADAPT;
                    a.layer = i;
                    a.edge = e;
                    a.in_slots = {src};
                    a.out_slot = m_in + (int32_t)k;
                    g->plan.push_back(a);
                }
                continue;
            }
            if (!same) {
                schema_slot(g, g->layers[j].out, sch[i], g->layers[j].qscale);
                PlanOp a;
                a.kind = PlanOp::ADAPT;
                a.layer = i;
                a.edge = e;
                a.in_slots = {src};
                a.out_slot = (int32_t)g->slots.size() - 1;
                g->plan.push_back(a);
                src = a.out_slot;
            }
            op.in_slots.push_back(src);
        }
        if (i == n - 1) break;
        if (out_index[i] >= 0 && schema_eq(sch_out[i], g->out_schema)) {
            op.out_slot = m_in + out_index[i];  // a net output written in place
        } else {
            schema_slot(g, L.out, sch_out[i], L.qscale);
            op.out_slot = (int32_t)g->slots.size() - 1;
        }
        out_slot[i] = op.out_slot;
        const Candidate &c = g->cands[op.cand];
        std::vector<Shape> in;
        for (int32_t j : L.inputs) in.push_back(g->layers[j].out);
        ws = std::max(ws, routine_workspace(c.routine, c.variant, L, in, sch[i]));
        sn_status rc = prepare_weights(g, i, c.routine, c.variant, sch[i], &op.wt, &op.bias, st);
        if (rc != SN_OK) return rc;
        g->plan.push_back(op);
    }
    // every blob the path keeps in qint8 needs its scale
    for (size_t s = 0; s < g->slots.size(); ++s) {
        if (g->slot_qscale[s] > 0.0f) continue;
        if (g->profiling) {
            g->slot_qscale[s] = kProfileQScale;  // both sides of a timed adapt
        } else if (g->slot_schema[s].dtype == SN_QI8) {
            return fail(SN_ESTATE, "the path keeps a blob in qi8 without a scale (sn_set_qscale or sn_calibrate)");
        }
    }
    {
        sn_status rc = place_slots(g);
        if (rc != SN_OK) return rc;
    }
    if (ws > g->workspace.bytes) {
        dev_free(g, &g->workspace);
        sn_status rc = dev_alloc(g, ws, &g->workspace);
        if (rc != SN_OK) return rc;
    }
    {
        sn_status rc = ensure_tile_counts(g, st);
        if (rc != SN_OK) return rc;
    }
    if (g->opt_chain && !g->profiling) {
        sn_status rc = build_chains(g, st);
        if (rc != SN_OK) return rc;
    }
    g->plan_valid = true;
    return SN_OK;
}

// A plan op that a chained launch can run: a conv2 on the tensor-core
// routine reading and writing graph-owned buffers (the caller's buffers may
// change from run to run; a chain's tensor maps are encoded once).
static bool chain_eligible(const Graph *g, const PlanOp &op) {
    if (op.kind != PlanOp::LAYER) return false;
    const Candidate &c = g->cands[op.cand];
    if (c.routine != R_CONV_TC || cand_out(c) != c.schema) return false;
    if (op.out_slot < g->n_ext) return false;
    for (int32_t s : op.in_slots)
        if (s < g->n_ext) return false;
    const Layer &L = g->layers[op.layer];
    if (L.type != SN_L_CONV2 || L.inputs.empty() || L.inputs.size() > 2) return false;
    bool imp;
    int bn, kb, bw, bh, bni;
    return k::conv_tc_chain_shape(L, g->layers[L.inputs[0]].out, g->schemas[c.schema], c.variant, &imp, &bn, &kb,
                                  &bw, &bh, &bni);
}

// Group maximal runs of two or more consecutive chain-eligible ops of one
// dtype into chains and upload their descriptors.
std::vector<std::pair<int32_t, int32_t>> chain_runs(const Graph *g) {
    std::vector<std::pair<int32_t, int32_t>> runs;
    const size_t n = g->plan.size();
    auto dtype_of = [&](size_t q) { return g->schemas[g->cands[g->plan[q].cand].schema].dtype; };
    size_t i = 0;
    while (i < n) {
        if (!chain_eligible(g, g->plan[i])) {
            ++i;
            continue;
        }
        size_t j = i;
        while (j + 1 < n && chain_eligible(g, g->plan[j + 1]) && dtype_of(j + 1) == dtype_of(i)) ++j;
        if (j > i) runs.push_back({(int32_t)i, (int32_t)j});
        i = j + 1;
    }
    return runs;
}

sn_status build_chains(Graph *g, cudaStream_t st) {
    g->chains.clear();
    g->op_chain.assign(g->plan.size(), -1);
    auto dtype_of = [&](size_t q) { return g->schemas[g->cands[g->plan[q].cand].schema].dtype; };
    for (const auto &run : chain_runs(g)) {
        const size_t i = (size_t)run.first, j = (size_t)run.second;
        {
            std::vector<ChainOp> ops;
            for (size_t q = i; q <= j; ++q) {
                const PlanOp &op = g->plan[q];
                const Candidate &c = g->cands[op.cand];
                const Layer &L = g->layers[op.layer];
                ChainOp co;
                co.layer = &L;
                co.in = g->layers[L.inputs[0]].out;
                co.schema = g->schemas[c.schema];
                co.variant = c.variant;
                co.in0 = g->slots[op.in_slots[0]].ptr;
                co.res = op.in_slots.size() > 1 ? g->slots[op.in_slots[1]].ptr : nullptr;
                co.out = g->slots[op.out_slot].ptr;
                co.wt = op.wt;
                co.bias = op.bias;
                for (size_t p = i; p < q; ++p) {
                    if (g->plan[p].out_slot == op.in_slots[0]) co.src = (int32_t)(p - i);
                    if (op.in_slots.size() > 1 && g->plan[p].out_slot == op.in_slots[1]) co.res_src = (int32_t)(p - i);
                }
                ops.push_back(co);
            }
            ChainPlan cp;
            cp.first_op = (int32_t)i;
            cp.last_op = (int32_t)j;
            cp.n_layers = (int32_t)ops.size();
            cp.dtype = dtype_of(i);
            std::vector<uint8_t> blob;
            cudaError_t e = k::chain_encode(ops, blob, &cp.total_units, &cp.done_count);
            if (e != cudaSuccess) return fail(SN_ECUDA, std::string("chain descriptors: ") + cudaGetErrorString(e));
            sn_status rc = dev_alloc(g, blob.size(), &cp.desc);
            if (rc == SN_OK) rc = dev_alloc(g, ((size_t)cp.done_count + 2) * sizeof(int32_t), &cp.done);
            if (rc != SN_OK) {
                dev_free(g, &cp.desc);
                dev_free(g, &cp.done);
                return rc;
            }
            g->chains.push_back(cp);  // owned by the graph from here on (freed with the plan)
            SN_CUDA_TRY(cudaMemcpyAsync(cp.desc.ptr, blob.data(), blob.size(), cudaMemcpyHostToDevice, st));
            SN_CUDA_TRY(cudaMemsetAsync(cp.done.ptr, 0, cp.done.bytes, st));
            SN_CUDA_TRY(cudaStreamSynchronize(st));  // `blob` is freed on return
            for (size_t q = i; q <= j; ++q) g->op_chain[q] = (int32_t)g->chains.size() - 1;
        }
    }
    return SN_OK;
}

static sn_status launch_op(Graph *g, const PlanOp &op, const IoPtrs &io, cudaStream_t st) {
    const int32_t m_in = (int32_t)io.in.size();
    auto ptr = [&](int32_t s) -> void * {
        if (s < m_in) return const_cast<void *>(io.in[s]);
        if (s < g->n_ext) return io.out[s - m_in];
        return g->slots[s].ptr;
    };
    if (op.kind == PlanOp::ADAPT) {
        const int32_t si = op.in_slots[0], so = op.out_slot;
        const sn_schema a = g->slot_schema[si], b = g->slot_schema[so];
        const float qs = a.dtype == SN_QI8 ? g->slot_qscale[si] : g->slot_qscale[so];  // the qi8 side's
        cudaError_t e = convert_blob(ptr(si), a, ptr(so), b, g->slot_shape[si], qs, st);
        if (e != cudaSuccess) return fail(SN_ECUDA, std::string("adapt: ") + cudaGetErrorString(e));
        return SN_OK;
    }
    const Layer &L = g->layers[op.layer];
    const Candidate &c = g->cands[op.cand];
    LaunchArgs a;
    a.g = g;
    a.layer = &L;
    a.routine = c.routine;
    a.variant = c.variant;
    a.schema = g->schemas[c.schema];
    a.out_schema = g->schemas[cand_out(c)];
    for (size_t k = 0; k < op.in_slots.size(); ++k) {
        a.in[k] = ptr(op.in_slots[k]);
        a.in_shapes.push_back(g->layers[L.inputs[k]].out);
        a.qs_in[k] = g->slot_qscale[op.in_slots[k]];
    }
    a.out = ptr(op.out_slot);
    a.qs_out = g->slot_qscale[op.out_slot];
    a.wt = op.wt;
    a.bias = op.bias;
    a.ws = g->workspace.ptr;
    a.ws_bytes = g->workspace.bytes;
    a.wait_limit = g->opt_wait_limit;
    a.tile_counts = static_cast<int *>(g->tile_counts.ptr);
    a.tile_counts_n = (int64_t)(g->tile_counts.bytes / sizeof(int));
    a.stream = st;
    return launch_routine(a);
}

sn_status run_plan(Graph *g, const IoPtrs &io, cudaStream_t st, std::vector<cudaEvent_t> *evs) {
    if (!g->plan_valid) {
        sn_status rc = build_plan(g, st);
        if (rc != SN_OK) return rc;
    }
    if ((int32_t)(io.in.size() + io.out.size()) != g->n_ext || (int32_t)io.in.size() != g->n_in())
        return fail(SN_EINVAL, "run: wrong number of input or output buffers");
    for (size_t i = 0; i < g->plan.size(); ++i) {
        if (!evs && i < g->op_chain.size() && g->op_chain[i] >= 0) {  // a chained launch runs the whole chain
            const ChainPlan &c = g->chains[g->op_chain[i]];
            if (c.first_op == (int32_t)i) {
                cudaError_t e = k::chain_launch(c.dtype, c.desc.ptr, c.n_layers, c.total_units,
                                                static_cast<int32_t *>(c.done.ptr), c.done_count, st);
                if (e != cudaSuccess) return fail(SN_ECUDA, std::string("chained launch: ") + cudaGetErrorString(e));
            }
            continue;
        }
        // external records: timing nodes when the stream is being captured
        if (evs) SN_CUDA_TRY(cudaEventRecordWithFlags((*evs)[2 * i], st, cudaEventRecordExternal));
        sn_status rc = launch_op(g, g->plan[i], io, st);
        if (rc != SN_OK) return rc;
        if (evs) SN_CUDA_TRY(cudaEventRecordWithFlags((*evs)[2 * i + 1], st, cudaEventRecordExternal));
    }
    return SN_OK;
}

// ---------------------------------------------------------------------------
// profiling
// ---------------------------------------------------------------------------
namespace {

struct Scratch {
    Buffer in0, in1, out;
};

sn_status ensure(Graph *g, Buffer &b, size_t bytes) {
    if (b.bytes >= bytes && b.ptr) return SN_OK;
    dev_free(g, &b);
    return dev_alloc(g, bytes, &b);
}

// Capture the stream work `body` issues into a CUDA graph and instantiate it.
template <class F>
sn_status capture_graph(cudaStream_t st, F body, cudaGraphExec_t *exec) {
    cudaGraph_t graph = nullptr;
    SN_CUDA_TRY(cudaStreamBeginCapture(st, cudaStreamCaptureModeThreadLocal));
    sn_status rc = body();
    cudaError_t ce = cudaStreamEndCapture(st, &graph);
    if (rc != SN_OK) {
        if (graph) cudaGraphDestroy(graph);
        return rc;
    }
    if (ce != cudaSuccess) return fail(SN_ECUDA, std::string("profiling capture: ") + cudaGetErrorString(ce));
    ce = cudaGraphInstantiate(exec, graph, 0);
    cudaGraphDestroy(graph);
    if (ce != cudaSuccess) return fail(SN_ECUDA, std::string("profiling instantiate: ") + cudaGetErrorString(ce));
    return SN_OK;
}

// Device time of one launch: `warm` eager launches (first-use set-up), then
// `iters` back-to-back launches captured into a CUDA graph, replayed three
// times; the median replay over iters.  Timing a replay rather than each
// eager launch keeps the host's launch cost out of the figure (for a small
// kernel it exceeds the kernel) and averages over the ~2 us resolution of
// events; the launches overlap as they do in a replayed net.
template <class F>
sn_status time_median(int warm, int iters, cudaStream_t st, F launch, int64_t *ns_out) {
    for (int i = 0; i < std::max(warm, 1); ++i) {
        sn_status rc = launch();
        if (rc != SN_OK) return rc;
    }
    iters = std::max(iters, 1);
    cudaGraphExec_t exec = nullptr;
    sn_status rc = capture_graph(st, [&]() -> sn_status {
        for (int i = 0; i < iters; ++i) {
            sn_status r = launch();
            if (r != SN_OK) return r;
        }
        return SN_OK;
    }, &exec);
    if (rc != SN_OK) return rc;
    constexpr int REPS = 3;
    cudaEvent_t ev[REPS + 1];
    for (auto &e : ev) SN_CUDA_TRY(cudaEventCreate(&e));
    cudaError_t e = cudaGraphLaunch(exec, st);  // warm replay
    for (int r = 0; r < REPS && e == cudaSuccess; ++r) {
        if (r == 0) e = cudaEventRecord(ev[0], st);
        if (e == cudaSuccess) e = cudaGraphLaunch(exec, st);
        if (e == cudaSuccess) e = cudaEventRecord(ev[r + 1], st);
    }
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
    std::vector<float> ms;
    if (e == cudaSuccess)
        for (int r = 0; r < REPS; ++r) {
            float t = 0;
            cudaEventElapsedTime(&t, ev[r], ev[r + 1]);
            ms.push_back(t);
        }
    for (auto &x : ev) cudaEventDestroy(x);
    cudaGraphExecDestroy(exec);
    if (e != cudaSuccess) return fail(SN_ECUDA, std::string("profiling: ") + cudaGetErrorString(e));
    std::sort(ms.begin(), ms.end());
    *ns_out = std::max<int64_t>(1, (int64_t)(ms[REPS / 2] / iters * 1e6 + 0.5));
    return SN_OK;
}

std::string signature(const Graph *g, int32_t i, const Candidate &c) {
    const Layer &L = g->layers[i];
    std::ostringstream o;
    o << L.type << ':';
    for (int32_t j : L.inputs) {
        const Shape &s = g->layers[j].out;
        o << s.n << 'x' << s.c << 'x' << s.h << 'x' << s.w << ';';
    }
    const sn_conv_params &p = L.conv;
    o << p.c_in << ',' << p.c_out << ',' << p.kh << ',' << p.kw << ',' << p.sh << ',' << p.sw << ','
      << p.ph << ',' << p.pw << ',' << p.dh << ',' << p.dw << ',' << p.groups << ',' << L.act << ','
      << L.pool.kh << ',' << L.pool.sh << ',' << L.pool.ph << ',' << L.dense_in << ',' << L.dense_out
      << '|' << c.routine << '/' << c.variant << '/' << c.schema << '>' << cand_out(c);
    return o.str();
}

}  // namespace

sn_status run_plan_timed(Graph *g, const IoPtrs &io, cudaStream_t user, std::vector<float> *op_ms) {
    if (!g->plan_valid) {
        sn_status rc = build_plan(g, user);
        if (rc != SN_OK) return rc;
    }
    SN_CUDA_TRY(cudaStreamSynchronize(user));
    cudaStream_t st = nullptr;
    SN_CUDA_TRY(cudaStreamCreateWithFlags(&st, cudaStreamNonBlocking));
    std::vector<cudaEvent_t> evs(2 * g->plan.size());
    for (auto &e : evs) cudaEventCreate(&e);
    cudaGraphExec_t exec = nullptr;
    sn_status rc = run_plan(g, io, st, nullptr);  // first-use set-up outside the capture
    if (rc == SN_OK) rc = capture_graph(st, [&]() { return run_plan(g, io, st, &evs); }, &exec);
    if (rc == SN_OK && cudaGraphLaunch(exec, st) != cudaSuccess) rc = fail(SN_ECUDA, "timed run: replay failed");
    if (cudaStreamSynchronize(st) != cudaSuccess && rc == SN_OK) rc = fail(SN_ECUDA, "timed run: stream failed");
    if (rc == SN_OK) {
        op_ms->assign(g->plan.size(), 0.f);
        for (size_t q = 0; q < g->plan.size(); ++q) cudaEventElapsedTime(&(*op_ms)[q], evs[2 * q], evs[2 * q + 1]);
    }
    if (exec) cudaGraphExecDestroy(exec);
    for (auto &e : evs) cudaEventDestroy(e);
    cudaStreamDestroy(st);
    return rc;
}

static sn_status profile_graph_on(Graph *g, const sn_profile_opts &o, cudaStream_t st);

// Profiling runs on a private stream (a CUDA graph cannot be captured on the
// legacy default stream), after the caller's stream has drained.
sn_status profile_graph(Graph *g, const sn_profile_opts &o, cudaStream_t user) {
    SN_CUDA_TRY(cudaStreamSynchronize(user));
    cudaStream_t st = nullptr;
    SN_CUDA_TRY(cudaStreamCreateWithFlags(&st, cudaStreamNonBlocking));
    g->profiling = true;
    const sn_status rc = profile_graph_on(g, o, st);
    g->profiling = false;
    const cudaError_t e = cudaStreamSynchronize(st);
    cudaStreamDestroy(st);
    if (rc == SN_OK && e != cudaSuccess) return fail(SN_ECUDA, std::string("profiling: ") + cudaGetErrorString(e));
    return rc;
}

static sn_status profile_graph_on(Graph *g, const sn_profile_opts &o, cudaStream_t st) {
    const int32_t n = g->n_layers(), ns = g->n_schemas();
    size_t max_bytes = 0;
    for (int32_t i = 0; i < n; ++i)
        max_bytes = std::max(max_bytes, (size_t)g->layers[i].out.numel() * 4);
    Scratch sc;
    sn_status rc = SN_OK;
    auto cleanup = [&]() {
        dev_free(g, &sc.in0);
        dev_free(g, &sc.in1);
        dev_free(g, &sc.out);
    };
    if ((rc = ensure(g, sc.in0, max_bytes)) != SN_OK || (rc = ensure(g, sc.in1, max_bytes)) != SN_OK ||
        (rc = ensure(g, sc.out, max_bytes)) != SN_OK || (rc = ensure_tile_counts(g, st)) != SN_OK) {
        cleanup();
        return rc;
    }
    // scratch inputs: small deterministic values (fp32 patterns reinterpreted
    // per dtype are not needed: fill each dtype's worth of elements)
    std::map<std::string, int64_t> seen, seen_stage;
    // --- unit profiling of layer routines ---
    for (int32_t i = 1; i < n - 1 && rc == SN_OK; ++i) {
        const Layer &L = g->layers[i];
        if (L.type < 0) continue;  // a net input layer: its one routine is the caller's buffer
        std::vector<Shape> in;
        for (int32_t j : L.inputs) in.push_back(g->layers[j].out);
        for (int32_t c = g->cand_begin[i]; c < g->cand_begin[i + 1] && rc == SN_OK; ++c) {
            Candidate &cd = g->cands[c];
            const std::string sig = signature(g, i, cd);
            auto it = seen.find(sig);
            if (it != seen.end()) {
                cd.cost = it->second;
                continue;
            }
            const sn_schema s = g->schemas[cd.schema];
            LaunchArgs a;
            a.g = g;
            a.layer = &L;
            a.routine = cd.routine;
            a.variant = cd.variant;
            a.schema = s;
            a.in_shapes = in;
            a.in[0] = sc.in0.ptr;
            a.in[1] = in.size() > 1 ? sc.in1.ptr : nullptr;  // a residual only where the layer has one
            a.out = sc.out.ptr;
            a.out_schema = g->schemas[cand_out(cd)];
            a.stream = st;
            a.qs_in[0] = a.qs_in[1] = a.qs_out = kProfileQScale;
            if (k::fill_pattern(sc.in0.ptr, s.dtype, in[0].numel(), 1234u + i, 1.0f, st) != cudaSuccess ||
                (in.size() > 1 &&
                 k::fill_pattern(sc.in1.ptr, s.dtype, in[1].numel(), 99u + i, 1.0f, st) != cudaSuccess)) {
                rc = fail(SN_ECUDA, "profiling: fill failed");
                break;
            }
            rc = prepare_weights(g, i, cd.routine, cd.variant, s, &a.wt, &a.bias, st);
            if (rc != SN_OK) break;
            const size_t ws = routine_workspace(cd.routine, cd.variant, L, in, s);
            if (ws > g->workspace.bytes) {
                invalidate_plan(g);
                dev_free(g, &g->workspace);
                if ((rc = dev_alloc(g, ws, &g->workspace)) != SN_OK) break;
            }
            a.ws = g->workspace.ptr;
            a.ws_bytes = g->workspace.bytes;
            a.tile_counts = static_cast<int *>(g->tile_counts.ptr);
            a.tile_counts_n = (int64_t)(g->tile_counts.bytes / sizeof(int));
            int64_t t = kInf;
            const int32_t nst = childnet_stages(cd.routine, s);
            if (nst == 1) {
                rc = time_median(o.warmup, o.iters, st, [&]() { return launch_routine(a); }, &t);
            } else {
                // a childnet (section III-D): each sub-layer is timed on its
                // own, once for every routine parameter it depends on, and
                // the childnet's cost is the sum along its chain (DPRS on a
                // chain whose sub-layer schemas the parent routine fixes)
                t = 0;
                for (int32_t stg = 0; stg < nst && rc == SN_OK && t != kInf; ++stg) {
                    // (the last sub-layer writes the candidate's output schema)
                    Candidate sc_{cd.routine, stage_uses_variant(cd.routine, stg) ? cd.variant : -1, cd.schema,
                                  cd.layer, 0};
                    if (stg == nst - 1) sc_.out_schema = cd.out_schema;
                    std::ostringstream sk;
                    sk << signature(g, i, sc_) << "#stage" << stg;
                    auto hit = seen_stage.find(sk.str());
                    int64_t ts = kInf;
                    if (hit != seen_stage.end()) {
                        ts = hit->second;
                    } else {
                        rc = time_median(o.warmup, o.iters, st, [&]() { return launch_routine_stage(a, stg); }, &ts);
                        if (rc == SN_OK) seen_stage.emplace(sk.str(), ts);
                    }
                    t = sat_add(t, ts);
                }
            }
            if (rc == SN_EUNSUPPORTED) {  // a routine parameter this device cannot run: infeasible
                rc = SN_OK;
                t = kInf;
            }
            if (rc != SN_OK) break;
            cd.cost = t;
            seen.emplace(sig, t);
        }
    }
    // --- unit profiling of adapt routines: every edge, every ordered pair of
    // a schema its producer can write and one its consumer can read ---
    std::vector<int64_t> Fw((size_t)n * ns, kInf), F((size_t)n * ns, kInf);
    for (const Candidate &c : g->cands) {
        int64_t &w = Fw[(size_t)c.layer * ns + cand_out(c)], &r = F[(size_t)c.layer * ns + c.schema];
        w = std::min(w, c.cost);
        r = std::min(r, c.cost);
    }
    std::map<std::string, int64_t> seen_a;
    for (size_t e = 0; e < g->edges.size() && rc == SN_OK; ++e) {
        auto [j, i] = g->edges[e];
        const Shape s = g->layers[j].out;
        for (int32_t a = 0; a < ns && rc == SN_OK; ++a) {
            if (Fw[(size_t)j * ns + a] == kInf) continue;
            for (int32_t b = 0; b < ns && rc == SN_OK; ++b) {
                if (a == b || F[(size_t)i * ns + b] == kInf) continue;
                std::ostringstream key;
                key << s.n << 'x' << s.c << 'x' << s.h << 'x' << s.w << ':' << a << '>' << b;
                auto it = seen_a.find(key.str());
                if (it != seen_a.end()) {
                    g->adapt((int32_t)e, a, b) = it->second;
                    continue;
                }
                const sn_schema A = g->schemas[a], B = g->schemas[b];
                if (k::fill_pattern(sc.in0.ptr, A.dtype, s.numel(), 7u, 1.0f, st) != cudaSuccess) {
                    rc = fail(SN_ECUDA, "profiling: fill failed");
                    break;
                }
                int64_t t = kInf;
                rc = time_median(o.warmup, o.iters, st, [&]() -> sn_status {
                    cudaError_t ce = convert_blob(sc.in0.ptr, A, sc.out.ptr, B, s, kProfileQScale, st);
                    return ce == cudaSuccess ? SN_OK : fail(SN_ECUDA, cudaGetErrorString(ce));
                }, &t);
                if (rc != SN_OK) break;
                g->adapt((int32_t)e, a, b) = t;
                seen_a.emplace(key.str(), t);
            }
        }
    }
    cleanup();
    if (rc != SN_OK) return rc;

    // --- integrated profiling: top-k per (layer, schema) in whole-net passes ---
    if (o.topk <= 0) return SN_OK;
    const bool had_path = g->has_path;
    const std::vector<int32_t> saved_path = g->path_cand;
    const int64_t saved_total = g->path_total;
    // ranked candidates per (layer, schema) by unit time
    std::vector<std::vector<std::vector<int32_t>>> ranked(n, std::vector<std::vector<int32_t>>(ns));
    for (int32_t i = 0; i < n; ++i) {
        for (int32_t c = g->cand_begin[i]; c < g->cand_begin[i + 1]; ++c)
            if (g->cands[c].cost != kInf) ranked[i][g->cands[c].schema].push_back(c);
        for (auto &v : ranked[i])
            std::stable_sort(v.begin(), v.end(), [&](int32_t x, int32_t y) {
                return g->cands[x].cost < g->cands[y].cost;
            });
    }
    // scratch net inputs (filled) and outputs
    std::vector<Buffer> xbufs;
    IoPtrs io;
    auto free_io = [&]() {
        for (auto &b : xbufs) dev_free(g, &b);
    };
    for (int32_t k = 0; k < g->n_in() && rc == SN_OK; ++k) {
        Buffer b;
        const Shape &sh = g->layers[k].out;
        if ((rc = dev_alloc(g, (size_t)sh.numel() * dtype_size(g->in_schema.dtype), &b)) != SN_OK) break;
        xbufs.push_back(b);
        io.in.push_back(b.ptr);
        k::fill_pattern(b.ptr, g->in_schema.dtype, sh.numel(), 5u + k, 1.0f, st);
    }
    for (int32_t j : g->layers[n - 1].inputs) {
        if (rc != SN_OK) break;
        Buffer b;
        if ((rc = dev_alloc(g, (size_t)g->layers[j].out.numel() * dtype_size(g->out_schema.dtype), &b)) != SN_OK)
            break;
        xbufs.push_back(b);
        io.out.push_back(b.ptr);
    }
    if (rc != SN_OK) {
        free_io();
        return rc;
    }
    std::vector<std::vector<float>> insitu(g->cands.size());
    for (int32_t lam = 0; lam < g->n_lambda && rc == SN_OK; ++lam) {
        for (int32_t r = 0; r < o.topk && rc == SN_OK; ++r) {
            std::vector<int32_t> pc(n);
            bool any = false;
            for (int32_t i = 0; i < n; ++i) {
                const auto &v = ranked[i][lam];
                if (i == 0 || i == n - 1) {
                    pc[i] = g->cand_begin[i];
                } else if (!v.empty()) {
                    pc[i] = v[std::min<size_t>(r, v.size() - 1)];
                    any = any || (size_t)r < v.size();
                } else {  // no routine in this schema: best overall
                    int32_t best = g->cand_begin[i];
                    for (int32_t c = g->cand_begin[i]; c < g->cand_begin[i + 1]; ++c)
                        if (g->cands[c].cost < g->cands[best].cost) best = c;
                    pc[i] = best;
                }
            }
            if (!any) continue;
            g->path_cand = pc;
            g->has_path = true;
            if ((rc = build_plan(g, st)) != SN_OK) break;
            std::vector<cudaEvent_t> evs(2 * g->plan.size());
            for (auto &e : evs) cudaEventCreate(&e);
            std::vector<std::vector<float>> per_op(g->plan.size());
            for (int32_t w = 0; w < std::max(o.warmup, 1) && rc == SN_OK; ++w)
                rc = run_plan(g, io, st, nullptr);
            // the whole net with a timing node around every op, replayed
            cudaGraphExec_t exec = nullptr;
            if (rc == SN_OK)
                rc = capture_graph(st, [&]() { return run_plan(g, io, st, &evs); }, &exec);
            for (int32_t p = 0; p < o.passes && rc == SN_OK; ++p) {
                if (cudaGraphLaunch(exec, st) != cudaSuccess) {
                    rc = fail(SN_ECUDA, "integrated profiling: replay failed");
                    break;
                }
                if (cudaStreamSynchronize(st) != cudaSuccess) {
                    rc = fail(SN_ECUDA, "integrated profiling: stream failed");
                    break;
                }
                for (size_t q = 0; q < g->plan.size(); ++q) {
                    float t = 0;
                    cudaEventElapsedTime(&t, evs[2 * q], evs[2 * q + 1]);
                    per_op[q].push_back(t);
                }
            }
            if (exec) cudaGraphExecDestroy(exec);
            for (auto &e : evs) cudaEventDestroy(e);
            if (rc != SN_OK) break;
            for (size_t q = 0; q < g->plan.size(); ++q) {
                const PlanOp &op = g->plan[q];
                if (op.kind != PlanOp::LAYER) continue;
                auto v = per_op[q];
                std::sort(v.begin(), v.end());
                insitu[op.cand].push_back(v[v.size() / 2]);
            }
        }
    }
    free_io();
    // in-situ medians replace the unit times of the re-timed candidates; the
    // candidates of the same (layer, schema) that were not re-timed keep their
    // unit ranking, moved to the in-situ scale by the best candidate's ratio
    // (in-situ times carry the op's whole latency, unit times its share of a
    // back-to-back replay, so mixing the two unscaled would favour the
    // candidates that were not re-timed)
    const std::vector<Candidate> unit = g->cands;
    for (size_t c = 0; c < insitu.size(); ++c) {
        if (insitu[c].empty()) continue;
        auto v = insitu[c];
        std::sort(v.begin(), v.end());
        g->cands[c].cost = std::max<int64_t>(1, (int64_t)(v[v.size() / 2] * 1e6 + 0.5));
    }
    for (int32_t i = 1; i < n - 1; ++i)
        for (int32_t lam = 0; lam < ns; ++lam) {
            const auto &v = ranked[i][lam];
            if (v.empty() || insitu[v[0]].empty() || unit[v[0]].cost <= 0 || unit[v[0]].cost == kInf) continue;
            const double ratio = (double)g->cands[v[0]].cost / (double)unit[v[0]].cost;
            for (int32_t c : v)
                if (insitu[c].empty() && unit[c].cost != kInf)
                    g->cands[c].cost = std::max<int64_t>(1, (int64_t)(unit[c].cost * ratio + 0.5));
        }
    g->has_path = had_path;
    g->path_cand = saved_path;
    g->path_total = saved_total;
    invalidate_plan(g);
    return rc;
}

// ---------------------------------------------------------------------------
// qint8 calibration (post-training, symmetric, one scale per blob)
// ---------------------------------------------------------------------------
sn_status calibrate(Graph *g, const void *in, cudaStream_t st) {
    const int32_t n = g->n_layers();
    // the cheapest float path: DPRS over the current costs without the qint8
    // candidates
    const std::vector<Candidate> saved_costs = g->cands;
    for (auto &c : g->cands)
        if (g->schemas[c.schema].dtype == SN_QI8 || g->schemas[cand_out(c)].dtype == SN_QI8) c.cost = kInf;
    std::vector<int32_t> pc;
    int64_t total = kInf;
    sn_status rc = select_path(*g, SN_SELECT_DPRS, pc, total);
    g->cands = saved_costs;
    if (rc != SN_OK || total == kInf)
        return fail(SN_ESTATE, "sn_calibrate: no float path of finite cost (profile or set the costs first)");

    const bool had_path = g->has_path;
    const std::vector<int32_t> saved_path = g->path_cand;
    const int64_t saved_total = g->path_total;
    g->path_cand = pc;
    g->has_path = true;
    std::vector<Buffer> outs;
    Buffer dmax;
    auto finish = [&](sn_status r) {
        for (auto &b : outs) dev_free(g, &b);
        dev_free(g, &dmax);
        g->has_path = had_path;
        g->path_cand = saved_path;
        g->path_total = saved_total;
        invalidate_plan(g);
        return r;
    };
    if ((rc = build_plan(g, st)) != SN_OK) return finish(rc);
    IoPtrs io;
    io.in.push_back(in);
    for (int32_t j : g->layers[n - 1].inputs) {
        Buffer b;
        if ((rc = dev_alloc(g, (size_t)g->layers[j].out.numel() * dtype_size(g->out_schema.dtype), &b)) != SN_OK)
            return finish(rc);
        outs.push_back(b);
        io.out.push_back(b.ptr);
    }
    if ((rc = dev_alloc(g, (size_t)n * sizeof(unsigned), &dmax)) != SN_OK) return finish(rc);
    unsigned *dm = static_cast<unsigned *>(dmax.ptr);
    if (cudaMemsetAsync(dm, 0, (size_t)n * sizeof(unsigned), st) != cudaSuccess ||
        k::absmax(in, g->in_schema.dtype, g->in_shape.numel(), dm, st) != cudaSuccess)
        return finish(fail(SN_ECUDA, "sn_calibrate: input reduction failed"));
    for (const PlanOp &op : g->plan) {
        if ((rc = launch_op(g, op, io, st)) != SN_OK) return finish(rc);
        if (op.kind != PlanOp::LAYER) continue;
        const int32_t so = op.out_slot;
        const void *y = so < 1 ? in : so < g->n_ext ? io.out[so - 1] : g->slots[so].ptr;
        if (k::absmax(y, g->slot_schema[so].dtype, g->slot_shape[so].numel(), dm + op.layer, st) != cudaSuccess)
            return finish(fail(SN_ECUDA, "sn_calibrate: reduction failed"));
    }
    std::vector<unsigned> hm(n);
    if (cudaMemcpyAsync(hm.data(), dm, (size_t)n * sizeof(unsigned), cudaMemcpyDeviceToHost, st) != cudaSuccess ||
        cudaStreamSynchronize(st) != cudaSuccess)
        return finish(fail(SN_ECUDA, "sn_calibrate: read-back failed"));
    for (int32_t i = 0; i < n - 1; ++i) {
        float m;
        std::memcpy(&m, &hm[i], sizeof(float));
        g->layers[i].qscale = m > 0.0f ? m / 127.0f : 1.0f;
    }
    return finish(SN_OK);
}

}  // namespace sn
