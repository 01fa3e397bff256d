// Net construction and finalisation (section III-B: net = DAG of layers with
// one input and one output; section IV-A: layers L_1..L_n in topological
// order; section IV-E: auxiliary zero-cost input/output layers).
#include <algorithm>
#include <cstring>

#include "sn_internal.h"

namespace sn {

static thread_local std::string g_last_error;

void set_error(const std::string &msg) { g_last_error = msg; }
sn_status fail(sn_status s, const std::string &msg) {
    g_last_error = msg;
    return s;
}
const char *last_error() { return g_last_error.c_str(); }

std::string schema_str(sn_schema s) {
    static const char *dt[] = {"f32", "f16", "bf16", "qi8"};
    static const char *ly[] = {"nchw", "nhwc"};
    if (!schema_valid(s)) return "invalid";
    return std::string(dt[s.dtype]) + "." + ly[s.layout];
}

static int64_t out_dim(int64_t in, int64_t k, int64_t s, int64_t p, int64_t d) {
    const int64_t span = d * (k - 1) + 1;
    if (in + 2 * p < span) return 0;
    return (in + 2 * p - span) / s + 1;
}

Graph::~Graph() {
    if (gexec) cudaGraphExecDestroy(gexec);
    for (auto &c : chains) {
        dev_free(this, &c.desc);
        dev_free(this, &c.done);
    }
    for (auto &b : slots) dev_free(this, &b);
    for (auto &kv : weight_cache) dev_free(this, &kv.second);
    for (auto &kv : bias_cache) dev_free(this, &kv.second);
    dev_free(this, &workspace);
    dev_free(this, &tile_counts);
    dev_free(this, &arena);
    if (copy_stream) cudaStreamSynchronize(copy_stream);  // no upload still writes a landing buffer
    for (int b = 0; b < 2; ++b) {
        dev_free(this, &host_land[b]);
        if (land_done[b]) cudaEventDestroy(land_done[b]);
        if (land_free[b]) cudaEventDestroy(land_free[b]);
    }
    if (copy_stream) cudaStreamDestroy(copy_stream);
    dev_free(this, &host_in);
    dev_free(this, &host_out);
}

sn_status dev_alloc(Graph *g, size_t bytes, Buffer *b) {
    b->bytes = bytes;
    b->ptr = nullptr;
    if (bytes == 0) return SN_OK;
    const size_t rounded = (bytes + 255) & ~size_t(255);
    if (g->alloc) {
        b->ptr = g->alloc(rounded, g->alloc_ctx);
        if (!b->ptr) return fail(SN_ENOMEM, "allocator returned NULL for " + std::to_string(rounded) + " bytes");
        if (reinterpret_cast<uintptr_t>(b->ptr) & 255u) {
            g->free_fn(b->ptr, g->alloc_ctx);
            b->ptr = nullptr;
            return fail(SN_EINVAL, "allocator returned a pointer not aligned to 256 bytes");
        }
        return SN_OK;
    }
    cudaError_t e = cudaMalloc(&b->ptr, rounded);
    if (e != cudaSuccess) {
        b->ptr = nullptr;
        return fail(e == cudaErrorMemoryAllocation ? SN_ENOMEM : SN_ECUDA,
                    std::string("cudaMalloc: ") + cudaGetErrorString(e));
    }
    return SN_OK;
}

void dev_free(Graph *g, Buffer *b) {
    if (b->view) {
        b->ptr = nullptr;
        b->view = false;
        return;
    }
    if (!b->ptr) return;
    if (g->free_fn) g->free_fn(b->ptr, g->alloc_ctx);
    else cudaFree(b->ptr);
    b->ptr = nullptr;
    b->bytes = 0;
}

void invalidate_plan(Graph *g) {
    g->plan_valid = false;
    g->plan.clear();
    for (auto &c : g->chains) {
        dev_free(g, &c.desc);
        dev_free(g, &c.done);
    }
    g->chains.clear();
    g->op_chain.clear();
    if (g->gexec) {
        cudaGraphExecDestroy(g->gexec);
        g->gexec = nullptr;
    }
}

// ---------------------------------------------------------------------------
// layer validation + shape inference
// ---------------------------------------------------------------------------
static sn_status infer_shape(Layer &L, const std::vector<Shape> &in) {
    switch (L.type) {
    case SN_L_CONV2:
    case SN_L_DWCONV2: {
        const sn_conv_params &p = L.conv;
        // conv2 may take a second input: a residual of the output's shape,
        // added after the bias and before the activation (a fused add)
        if (in.size() != 1 && !(L.type == SN_L_CONV2 && in.size() == 2))
            return fail(SN_EINVAL, "conv2 takes one input (or two: input, residual); dwconv2 takes one");
        if (p.kh < 1 || p.kw < 1 || p.sh < 1 || p.sw < 1 || p.ph < 0 || p.pw < 0 || p.dh < 1 ||
            p.dw < 1 || p.groups < 1 || p.c_in < 1 || p.c_out < 1)
            return fail(SN_EINVAL, "conv2: invalid parameter");
        if (p.act < SN_ACT_NONE || p.act > SN_ACT_HSIGMOID) return fail(SN_EINVAL, "conv2: bad act");
        if (in[0].c != p.c_in) return fail(SN_EINVAL, "conv2: input channels != c_in");
        if (p.c_in % p.groups || p.c_out % p.groups)
            return fail(SN_EINVAL, "conv2: groups must divide c_in and c_out");
        if (L.type == SN_L_DWCONV2 && !(p.groups == p.c_in && p.c_in == p.c_out))
            return fail(SN_EINVAL, "dwconv2: requires groups == c_in == c_out");
        const int64_t P = out_dim(in[0].h, p.kh, p.sh, p.ph, p.dh);
        const int64_t Q = out_dim(in[0].w, p.kw, p.sw, p.pw, p.dw);
        if (P < 1 || Q < 1) return fail(SN_EINVAL, "conv2: empty output");
        L.out = {in[0].n, p.c_out, P, Q};
        L.act = p.act;
        if (in.size() == 2 && !(in[1] == L.out))
            return fail(SN_EINVAL, "conv2: the residual input must have the output's shape");
        return SN_OK;
    }
    case SN_L_MAXPOOL: {
        const sn_pool_params &p = L.pool;
        if (in.size() != 1) return fail(SN_EINVAL, "maxpool takes one input");
        if (p.kh < 1 || p.kw < 1 || p.sh < 1 || p.sw < 1 || p.ph < 0 || p.pw < 0 ||
            p.ph >= p.kh || p.pw >= p.kw)
            return fail(SN_EINVAL, "maxpool: invalid parameter (padding must be < kernel)");
        const int64_t P = out_dim(in[0].h, p.kh, p.sh, p.ph, 1);
        const int64_t Q = out_dim(in[0].w, p.kw, p.sw, p.pw, 1);
        if (P < 1 || Q < 1) return fail(SN_EINVAL, "maxpool: empty output");
        L.out = {in[0].n, in[0].c, P, Q};
        return SN_OK;
    }
    case SN_L_GAP:
        if (in.size() != 1) return fail(SN_EINVAL, "gap takes one input");
        L.out = {in[0].n, in[0].c, 1, 1};
        return SN_OK;
    case SN_L_ADD:
        if (in.size() != 2) return fail(SN_EINVAL, "add takes two inputs");
        if (!(in[0] == in[1])) return fail(SN_EINVAL, "add: input shapes differ");
        if (L.act < SN_ACT_NONE || L.act > SN_ACT_HSIGMOID) return fail(SN_EINVAL, "add: bad act");
        L.out = in[0];
        return SN_OK;
    case SN_L_MUL:
        if (in.size() != 2) return fail(SN_EINVAL, "mul takes two inputs (blob, per-channel scale)");
        if (!(in[1] == Shape{in[0].n, in[0].c, 1, 1}))
            return fail(SN_EINVAL, "mul: the scale must be N x C x 1 x 1 of the blob's N and C");
        if (L.act < SN_ACT_NONE || L.act > SN_ACT_HSIGMOID) return fail(SN_EINVAL, "mul: bad act");
        L.out = in[0];
        return SN_OK;
    case SN_L_DENSE:
        if (in.size() != 1) return fail(SN_EINVAL, "dense takes one input");
        if (in[0].h != 1 || in[0].w != 1 || in[0].c != L.dense_in || L.dense_out < 1)
            return fail(SN_EINVAL, "dense: input must be N x in_features x 1 x 1");
        if (L.act < SN_ACT_NONE || L.act > SN_ACT_HSIGMOID) return fail(SN_EINVAL, "dense: bad act");
        L.out = {in[0].n, L.dense_out, 1, 1};
        return SN_OK;
    default:
        return fail(SN_EINVAL, "unknown layer type");
    }
}

sn_status add_layer(Graph *g, int32_t type, const void *params, const int32_t *inputs,
                    int32_t n_inputs, const float *weights, const float *bias, int32_t *out_id) {
    if (g->finalized) return fail(SN_ESTATE, "net already finalised; no more layers");
    if (n_inputs < 1 || n_inputs > 2 || !inputs) return fail(SN_EINVAL, "bad inputs");
    Layer L;
    L.type = type;
    std::vector<Shape> in;
    // internal indices: net input k (id -1 - k) is layer k, user layer u is
    // layer u + (number of net inputs)
    const int32_t m_in = 1 + (int32_t)g->extra_in.size();
    for (int32_t i = 0; i < n_inputs; ++i) {
        const int32_t id = inputs[i];
        if (id < -m_in || id >= (int32_t)g->user.size()) return fail(SN_EINVAL, "input id out of range");
        if (id < 0) {
            const int32_t k = -1 - id;
            L.inputs.push_back(k);
            in.push_back(k == 0 ? g->in_shape : g->extra_in[k - 1]);
        } else {
            L.inputs.push_back(id + m_in);
            in.push_back(g->user[id].out);
        }
    }
    int64_t wn = 0, bn = 0;
    switch (type) {
    case SN_L_CONV2:
    case SN_L_DWCONV2:
        if (!params) return fail(SN_EINVAL, "conv2 needs params");
        std::memcpy(&L.conv, params, sizeof(sn_conv_params));
        wn = (int64_t)L.conv.c_out * (L.conv.groups > 0 ? L.conv.c_in / L.conv.groups : 0) *
             L.conv.kh * L.conv.kw;
        bn = L.conv.c_out;
        break;
    case SN_L_MAXPOOL:
        if (!params) return fail(SN_EINVAL, "maxpool needs params");
        std::memcpy(&L.pool, params, sizeof(sn_pool_params));
        break;
    case SN_L_GAP:
        break;
    case SN_L_ADD:
    case SN_L_MUL:
        L.act = params ? static_cast<const sn_add_params *>(params)->act : SN_ACT_NONE;
        break;
    case SN_L_DENSE: {
        if (!params) return fail(SN_EINVAL, "dense needs params");
        auto *p = static_cast<const sn_dense_params *>(params);
        L.dense_in = p->in_features;
        L.dense_out = p->out_features;
        L.act = p->act;
        wn = (int64_t)L.dense_in * L.dense_out;
        bn = L.dense_out;
        break;
    }
    default:
        return fail(SN_EINVAL, "unknown layer type");
    }
    sn_status s = infer_shape(L, in);
    if (s != SN_OK) return s;
    if (wn > 0) {
        if (!weights) return fail(SN_EINVAL, "layer needs weights");
        L.weight.assign(weights, weights + wn);
        L.bias.assign(bn, 0.0f);
        if (bias) L.bias.assign(bias, bias + bn);
    }
    g->user.push_back(std::move(L));
    *out_id = (int32_t)g->user.size() - 1;
    return SN_OK;
}

// ---------------------------------------------------------------------------
// finalisation: internal layers, edges, candidates
// ---------------------------------------------------------------------------
sn_status add_input(Graph *g, const int64_t nchw[4], int32_t *id) {
    if (g->finalized) return fail(SN_ESTATE, "net already finalised");
    if (!g->user.empty()) return fail(SN_ESTATE, "declare every net input before the first layer");
    for (int k = 0; k < 4; ++k)
        if (nchw[k] < 1) return fail(SN_EINVAL, "input extents must be >= 1");
    g->extra_in.push_back(Shape{nchw[0], nchw[1], nchw[2], nchw[3]});
    g->extra_in_qscale.push_back(0.0f);
    *id = -1 - (int32_t)g->extra_in.size();
    return SN_OK;
}

sn_status set_outputs(Graph *g, const int32_t *ids, int32_t n) {
    if (g->finalized) return fail(SN_ESTATE, "net already finalised");
    if (n < 1 || !ids) return fail(SN_EINVAL, "at least one output");
    std::vector<int32_t> v;
    for (int32_t i = 0; i < n; ++i) {
        if (ids[i] < 0 || ids[i] >= (int32_t)g->user.size()) return fail(SN_EINVAL, "output id out of range");
        for (int32_t u : v)
            if (u == ids[i]) return fail(SN_EINVAL, "duplicate output id");
        v.push_back(ids[i]);
    }
    g->outputs = v;
    return SN_OK;
}

// Graph optimiser pass run before tuning (section III-A fuses layers ahead of
// tuning): every add whose input is a conv2 without activation, read by
// nothing else and not a net output, becomes that conv2 with the add's other
// input as a residual and the add's activation, y = act(conv(x) + b + r).
// The fused layer takes the add's place (after both of its inputs) and the
// conv2 is dropped; the user layers are renumbered.  new_id[old] = the new
// id of each old user layer (-1 for a conv2 folded into its add).
sn_status fuse_residual(Graph *g, std::vector<int32_t> &new_id, int32_t *n_fused) {
    if (g->finalized) return fail(SN_ESTATE, "sn_fuse_residual: the net is already finalised (fuse before tuning)");
    const int32_t m = (int32_t)g->user.size(), m_in = g->n_in();
    std::vector<std::vector<int32_t>> consumers(m);
    for (int32_t i = 0; i < m; ++i)
        for (int32_t j : g->user[i].inputs)
            if (j >= m_in) consumers[j - m_in].push_back(i);
    std::vector<char> is_output(m, 0);
    for (int32_t u : g->outputs) is_output[u] = 1;
    if (g->outputs.empty() && m > 0) is_output[m - 1] = 1;
    std::vector<int32_t> fold_conv(m, -1), fold_other(m, -1);  // per add: the folded conv2, the residual
    std::vector<char> dropped(m, 0);
    int32_t nf = 0;
    for (int32_t i = 0; i < m; ++i) {
        const Layer &a = g->user[i];
        if (a.type != SN_L_ADD || a.inputs.size() != 2) continue;
        for (int pos = 0; pos < 2; ++pos) {
            const int32_t jj = a.inputs[pos], other = a.inputs[1 - pos];
            if (jj < m_in || jj == other) continue;
            const int32_t j = jj - m_in;
            const Layer &c = g->user[j];
            if (c.type != SN_L_CONV2 || c.inputs.size() != 1 || c.conv.act != SN_ACT_NONE) continue;
            if (consumers[j].size() != 1 || consumers[j][0] != i || is_output[j] || dropped[j]) continue;
            fold_conv[i] = j;
            fold_other[i] = other;
            dropped[j] = 1;
            ++nf;
            break;
        }
    }
    new_id.assign(m, -1);
    std::vector<Layer> out;
    for (int32_t i = 0; i < m; ++i) {
        if (dropped[i]) continue;
        new_id[i] = (int32_t)out.size();
        if (fold_conv[i] >= 0) {
            Layer f = g->user[fold_conv[i]];
            f.inputs = {f.inputs[0], fold_other[i]};
            f.conv.act = g->user[i].act;
            f.act = g->user[i].act;
            f.out = g->user[i].out;
            f.qscale = g->user[i].qscale;
            out.push_back(std::move(f));
        } else {
            out.push_back(g->user[i]);
        }
    }
    for (Layer &l : out)
        for (int32_t &j : l.inputs)
            if (j >= m_in) j = new_id[j - m_in] + m_in;
    for (int32_t &u : g->outputs) u = new_id[u];
    g->user = std::move(out);
    if (n_fused) *n_fused = nf;
    return SN_OK;
}

sn_status graph_finalize(Graph *g) {
    if (g->finalized) return SN_OK;
    const int32_t m = (int32_t)g->user.size();
    const int32_t m_in = g->n_in();
    if (g->outputs.empty() && m > 0) g->outputs = {m - 1};
    std::vector<Layer> L;
    Layer in_l;
    in_l.type = -1;
    in_l.out = g->in_shape;
    in_l.qscale = g->in_qscale;
    L.push_back(in_l);
    // the other net inputs: input layers fed by the auxiliary input layer 0
    // (section IV-E), one zero-cost routine each
    for (size_t k = 0; k < g->extra_in.size(); ++k) {
        Layer x;
        x.type = -3;
        x.inputs = {0};
        x.out = g->extra_in[k];
        x.qscale = g->extra_in_qscale[k];
        L.push_back(x);
    }
    for (auto &u : g->user) L.push_back(u);
    // the auxiliary output layer merges every net output
    Layer out_l;
    out_l.type = -2;
    if (m == 0) {
        out_l.inputs = {0};
        out_l.out = g->in_shape;
    } else {
        for (int32_t u : g->outputs) out_l.inputs.push_back(u + m_in);
        out_l.out = g->user[g->outputs[0]].out;
    }
    L.push_back(out_l);
    const int32_t n = (int32_t)L.size();

    // 1-in-1-out: every layer must reach the output (section IV-A)
    std::vector<char> reach(n, 0);
    reach[n - 1] = 1;
    for (int32_t i = n - 1; i >= 0; --i)
        if (reach[i])
            for (int32_t j : L[i].inputs) reach[j] = 1;
    for (int32_t i = 0; i < n; ++i)
        if (!reach[i])
            return fail(SN_EINVAL, (L[i].type == -3 ? "net input " + std::to_string(i) + " feeds no layer"
                                                    : "layer " + std::to_string(i - m_in) +
                                                          " does not reach a net output (every layer must feed one)"));

    std::vector<std::pair<int32_t, int32_t>> edges;
    for (int32_t i = 0; i < n; ++i)
        for (int32_t j : L[i].inputs) edges.push_back({j, i});

    std::vector<Candidate> cands;
    std::vector<int32_t> begin(n + 1, 0);
    for (int32_t i = 0; i < n; ++i) {
        begin[i] = (int32_t)cands.size();
        if (i == 0 || L[i].type == -3) {  // net inputs: the caller's buffers, in in_schema
            cands.push_back({R_IO, 0, g->in_schema_idx, i, 0});
            continue;
        }
        if (i == n - 1) {
            cands.push_back({R_IO, 0, g->out_schema_idx, n - 1, 0});
            continue;
        }
        std::vector<Shape> in;
        for (int32_t j : L[i].inputs) in.push_back(L[j].out);
        for (int32_t r = 1; r < R_COUNT; ++r) {
            if (r == R_ADAPT) continue;
            for (int32_t s = 0; s < g->n_lambda; ++s) {
                const int32_t nv = routine_variants(r, L[i], in, g->schemas[s]);
                for (int32_t v = 0; v < nv; ++v) cands.push_back({r, v, s, i, kInf});
                if (nv == 0) continue;
                // the same routine writing another schema of Lambda (fused boundary)
                for (const sn_schema &o : fused_outputs(r, L[i], g->schemas[s]))
                    for (int32_t so = 0; so < g->n_lambda; ++so)
                        if (so != s && schema_eq(g->schemas[so], o))
                            for (int32_t v = 0; v < nv; ++v) {
                                if (!fused_variant_ok(r, L[i], in, g->schemas[s], v)) continue;
                                Candidate c{r, v, s, i, kInf};
                                c.out_schema = so;
                                cands.push_back(c);
                            }
            }
        }
        if ((int32_t)cands.size() == begin[i])
            return fail(SN_EINFEASIBLE, "layer " + std::to_string(i - m_in) +
                                            " has no routine in any schema of Lambda");
    }
    begin[n] = (int32_t)cands.size();

    const int32_t ns = g->n_schemas();
    std::vector<int64_t> ac((size_t)edges.size() * ns * ns, kInf);
    for (size_t e = 0; e < edges.size(); ++e)
        for (int32_t a = 0; a < ns; ++a) ac[(e * ns + a) * ns + a] = 0;  // void adapt

    g->layers = std::move(L);
    g->edges = std::move(edges);
    g->cands = std::move(cands);
    g->cand_begin = std::move(begin);
    g->adapt_cost = std::move(ac);
    g->finalized = true;
    return SN_OK;
}

}  // namespace sn
