// Routine path selection (section IV).
//
//   F_i(lambda) = argmin_{r in R_i(lambda)} T(r)                       (Eq. 1)
//   T(S) = sum_{r in S} T(r), with an adapt routine on every edge whose
//          endpoint schemas differ, void (T = 0) otherwise     (Def. 1-2, IV-F)
//   S*   = argmin_S T(S)                                                (Eq. 2)
//
// select_dprs implements Alg. 1 (DPRS): a sweep over the layers in
// topological order keeping, for every layer i, schema lambda and tuple
// lambda_C of schemas of the still-open branching layers C_i, the fastest
// routine subpath S_i(lambda; lambda_C) (Eq. 3 for straight nets, Eq. 4 for
// merges).  At a merging layer the constraints of every branching layer that
// the merging layer post-dominates are relaxed (Eq. 5, Prop. 3); a branching
// layer then adds its own schema to the constraint tuple.
//
// Readings where Alg. 1 is terse:
//   * C_i is the union of the predecessors' constraint sets (the listing says
//     they are all equal, which fails for nested branches; the union is what
//     the recurrence needs).  A predecessor's state is looked up with the
//     restriction of lambda_C to its own C_h.
//   * S_i is a *set* union (Eq. 4): subpaths that share ancestors count them
//     once.  Every state therefore keeps its schema assignment over the
//     layers it covers (the ancestors of L_i and L_i), and the time of a union
//     is evaluated from that assignment, so shared prefixes are never counted
//     twice.
//   * Ties: the first minimum in enumeration order wins (lower schema index
//     first, the predecessors' tuples in lexicographic order).
#include <algorithm>
#include <numeric>

#include "sn_internal.h"

namespace sn {

void fastest_per_schema(const Graph &g, std::vector<int64_t> &F, std::vector<int32_t> &argF) {
    const int32_t n = g.n_layers(), ns = g.n_schemas();
    F.assign((size_t)n * ns, kInf);
    argF.assign((size_t)n * ns, -1);
    for (int32_t i = 0; i < n; ++i)
        for (int32_t c = g.cand_begin[i]; c < g.cand_begin[i + 1]; ++c) {
            const Candidate &k = g.cands[c];
            const size_t idx = (size_t)i * ns + k.schema;
            if (argF[idx] < 0 || k.cost < F[idx]) {  // first minimum wins
                F[idx] = k.cost;
                argF[idx] = c;
            }
        }
}

namespace {

struct Ctx {
    const Graph &g;
    int32_t n, ns;
    std::vector<int64_t> F;
    std::vector<std::vector<int32_t>> preds, succs;     // distinct
    std::vector<std::vector<int32_t>> in_edges;         // edge ids into i
    std::vector<std::vector<char>> covered;             // ancestors + self
    std::vector<std::vector<char>> pdom;                // pdom[v][u]: u post-dominates v

    explicit Ctx(const Graph &gg) : g(gg), n(gg.n_layers()), ns(gg.n_schemas()) {
        std::vector<int32_t> argF;
        fastest_per_schema(g, F, argF);
        preds.assign(n, {});
        succs.assign(n, {});
        in_edges.assign(n, {});
        for (size_t e = 0; e < g.edges.size(); ++e) {
            auto [u, v] = g.edges[e];
            in_edges[v].push_back((int32_t)e);
            if (std::find(preds[v].begin(), preds[v].end(), u) == preds[v].end()) preds[v].push_back(u);
            if (std::find(succs[u].begin(), succs[u].end(), v) == succs[u].end()) succs[u].push_back(v);
        }
        for (auto &p : preds) std::sort(p.begin(), p.end());
        covered.assign(n, std::vector<char>(n, 0));
        for (int32_t i = 0; i < n; ++i) {
            covered[i][i] = 1;
            for (int32_t h : preds[i])
                for (int32_t v = 0; v < n; ++v)
                    if (covered[h][v]) covered[i][v] = 1;
        }
        // post-dominators on the 1-in-1-out DAG, output = n-1
        pdom.assign(n, std::vector<char>(n, 0));
        for (int32_t v = n - 1; v >= 0; --v) {
            if (succs[v].empty()) {
                pdom[v][v] = 1;
                continue;
            }
            std::vector<char> acc(n, 1);
            for (int32_t s : succs[v])
                for (int32_t u = 0; u < n; ++u) acc[u] = acc[u] && pdom[s][u];
            acc[v] = 1;
            pdom[v] = acc;
        }
    }

    // T of the subpath given by asg over the layers covered by layer i
    int64_t eval(int32_t i, const std::vector<int16_t> &asg) const {
        int64_t t = 0;
        for (int32_t v = 0; v < n; ++v) {
            if (!covered[i][v]) continue;
            t = sat_add(t, F[(size_t)v * ns + asg[v]]);
            if (t == kInf) return kInf;
            for (int32_t e : in_edges[v]) {
                const int32_t u = g.edges[e].first;
                t = sat_add(t, g.adapt(e, asg[u], asg[v]));  // 0 for a void adapt
                if (t == kInf) return kInf;
            }
        }
        return t;
    }
};

struct State {
    int64_t cost = kInf;
    std::vector<int16_t> asg;  // schema per layer, -1 = not covered
};

size_t ipow(int32_t b, size_t e) {
    size_t r = 1;
    while (e--) r *= (size_t)b;
    return r;
}

// tuple index (mixed radix ns, first constraint most significant)
void decode(size_t idx, int32_t ns, size_t len, std::vector<int32_t> &out) {
    out.assign(len, 0);
    for (size_t k = len; k-- > 0;) {
        out[k] = (int32_t)(idx % (size_t)ns);
        idx /= (size_t)ns;
    }
}
size_t encode(const std::vector<int32_t> &t, int32_t ns) {
    size_t idx = 0;
    for (int32_t v : t) idx = idx * (size_t)ns + (size_t)v;
    return idx;
}

}  // namespace

sn_status select_dprs(const Graph &g, std::vector<int32_t> &schema_of, int64_t &total) {
    Ctx cx(g);
    const int32_t n = cx.n, ns = cx.ns;
    std::vector<std::vector<int32_t>> Cset(n);
    std::vector<std::vector<State>> table(n);
    std::vector<int32_t> tup, sub, lamH;

    for (int32_t i = 0; i < n; ++i) {
        const auto &H = cx.preds[i];
        // C_i <- union of C_h
        std::vector<int32_t> C;
        for (int32_t h : H) C.insert(C.end(), Cset[h].begin(), Cset[h].end());
        std::sort(C.begin(), C.end());
        C.erase(std::unique(C.begin(), C.end()), C.end());
        const size_t nt = ipow(ns, C.size());
        std::vector<State> T((size_t)ns * nt);
        // positions of each predecessor's constraints inside C
        std::vector<std::vector<int32_t>> posmap(H.size());
        for (size_t hj = 0; hj < H.size(); ++hj)
            for (int32_t b : Cset[H[hj]])
                posmap[hj].push_back((int32_t)(std::lower_bound(C.begin(), C.end(), b) - C.begin()));
        const size_t nH = ipow(ns, H.size());

        for (int32_t lam = 0; lam < ns; ++lam) {
            if (cx.F[(size_t)i * ns + lam] == kInf) continue;
            for (size_t ti = 0; ti < nt; ++ti) {
                State &best = T[(size_t)lam * nt + ti];
                if (H.empty()) {
                    best.asg.assign(n, -1);
                    best.asg[i] = (int16_t)lam;
                    best.cost = cx.F[(size_t)i * ns + lam];
                    continue;
                }
                decode(ti, ns, C.size(), tup);
                std::vector<int16_t> merged;
                for (size_t hi = 0; hi < nH; ++hi) {
                    decode(hi, ns, H.size(), lamH);
                    merged.assign(n, -1);
                    bool ok = true;
                    for (size_t hj = 0; hj < H.size() && ok; ++hj) {
                        const int32_t h = H[hj];
                        sub.resize(posmap[hj].size());
                        for (size_t k = 0; k < posmap[hj].size(); ++k) sub[k] = tup[posmap[hj][k]];
                        const size_t ntH = ipow(ns, Cset[h].size());
                        const State &sh = table[h][(size_t)lamH[hj] * ntH + encode(sub, ns)];
                        if (sh.cost == kInf) {
                            ok = false;
                            break;
                        }
                        for (int32_t v = 0; v < n; ++v) {
                            if (sh.asg[v] < 0) continue;
                            if (merged[v] >= 0 && merged[v] != sh.asg[v]) {
                                ok = false;  // subpaths disagree on a shared layer
                                break;
                            }
                            merged[v] = sh.asg[v];
                        }
                    }
                    if (!ok) continue;
                    merged[i] = (int16_t)lam;
                    const int64_t t = cx.eval(i, merged);
                    if (t < best.cost) {
                        best.cost = t;
                        best.asg = merged;
                    }
                }
            }
        }

        // merging layer: relax the constraints of branching layers it post-dominates
        if (H.size() >= 2 && !C.empty()) {
            std::vector<int32_t> keep, relax_pos, keep_pos;
            for (size_t k = 0; k < C.size(); ++k) {
                if (cx.pdom[C[k]][i]) relax_pos.push_back((int32_t)k);
                else {
                    keep.push_back(C[k]);
                    keep_pos.push_back((int32_t)k);
                }
            }
            if (!relax_pos.empty()) {
                const size_t nk = ipow(ns, keep.size());
                std::vector<State> R((size_t)ns * nk);
                for (int32_t lam = 0; lam < ns; ++lam)
                    for (size_t ti = 0; ti < nt; ++ti) {  // lexicographic over the full tuple
                        decode(ti, ns, C.size(), tup);
                        sub.resize(keep.size());
                        for (size_t k = 0; k < keep.size(); ++k) sub[k] = tup[keep_pos[k]];
                        State &dst = R[(size_t)lam * nk + encode(sub, ns)];
                        const State &src = T[(size_t)lam * nt + ti];
                        if (src.cost < dst.cost) dst = src;
                    }
                T.swap(R);
                C = keep;
            }
        }
        // branching layer: push its own schema into the constraint tuple
        if (cx.succs[i].size() >= 2) {
            const size_t ntc = ipow(ns, C.size());
            std::vector<State> B((size_t)ns * ntc * ns);
            for (int32_t lam = 0; lam < ns; ++lam)
                for (size_t ti = 0; ti < ntc; ++ti)
                    B[(size_t)lam * ntc * ns + ti * ns + lam] = T[(size_t)lam * ntc + ti];
            T.swap(B);
            C.push_back(i);  // i exceeds every earlier index: C stays sorted
        }
        Cset[i] = std::move(C);
        table[i] = std::move(T);
    }

    // S* = fastest over lambda of S_n(lambda; {}) (the constraint set is empty
    // at the output by Prop. 3; take the best over any leftover tuple anyway)
    const int32_t o = n - 1;
    const size_t nto = ipow(ns, Cset[o].size());
    const State *best = nullptr;
    for (int32_t lam = 0; lam < ns; ++lam)
        for (size_t ti = 0; ti < nto; ++ti) {
            const State &s = table[o][(size_t)lam * nto + ti];
            if (s.cost < kInf && (!best || s.cost < best->cost)) best = &s;
        }
    if (!best) return fail(SN_EINFEASIBLE, "no routine path with finite cost");
    schema_of.assign(n, 0);
    for (int32_t v = 0; v < n; ++v) schema_of[v] = best->asg[v];
    total = best->cost;
    return SN_OK;
}

sn_status select_brute(const Graph &g, std::vector<int32_t> &schema_of, int64_t &total) {
    Ctx cx(g);
    const int32_t n = cx.n, ns = cx.ns;
    std::vector<std::vector<int16_t>> opts(n);
    double space = 1.0;
    for (int32_t i = 0; i < n; ++i) {
        for (int32_t l = 0; l < ns; ++l)
            if (cx.F[(size_t)i * ns + l] != kInf) opts[i].push_back((int16_t)l);
        if (opts[i].empty()) return fail(SN_EINFEASIBLE, "a layer has no feasible schema");
        space *= (double)opts[i].size();
    }
    if (space > (double)(1u << 26))
        return fail(SN_EUNSUPPORTED, "too many schema assignments for brute force");
    std::vector<int32_t> ctr(n, 0);
    std::vector<int16_t> asg(n), best_asg;
    int64_t best = kInf;
    for (;;) {
        for (int32_t i = 0; i < n; ++i) asg[i] = opts[i][ctr[i]];
        const int64_t t = cx.eval(n - 1, asg);  // the output covers every layer
        if (t < best) {
            best = t;
            best_asg = asg;
        }
        int32_t i = n - 1;
        while (i >= 0 && ctr[i] == (int32_t)opts[i].size() - 1) ctr[i--] = 0;
        if (i < 0) break;
        ctr[i]++;
    }
    if (best == kInf) return fail(SN_EINFEASIBLE, "no routine path with finite cost");
    schema_of.assign(best_asg.begin(), best_asg.end());
    total = best;
    return SN_OK;
}

// ---------------------------------------------------------------------------
// fused boundaries: the same algorithm over (read, written) schema pairs
// ---------------------------------------------------------------------------
// The pair problem has |Lambda|^2 schemas p = read * ns + written; candidate c
// of layer i sits at its pair, and edge (u, v) costs the adapt from u's
// written schema to v's read one (void when they agree).  Pairs no routine
// has keep F = INF, so DPRS never enters them.
static void expand_pairs(const Graph &g, Graph &x) {
    const int32_t ns = g.n_schemas(), np = ns * ns;
    x.layers.resize(g.layers.size());
    x.schemas.assign((size_t)np, sn_schema{SN_F32, SN_NCHW});
    x.edges = g.edges;
    x.cand_begin = g.cand_begin;
    x.cands = g.cands;
    for (auto &c : x.cands) {
        c.schema = c.schema * ns + cand_out(c);
        c.out_schema = -1;
    }
    x.adapt_cost.assign(g.edges.size() * (size_t)np * np, kInf);
    for (size_t e = 0; e < g.edges.size(); ++e)
        for (int32_t p = 0; p < np; ++p)
            for (int32_t q = 0; q < np; ++q)
                x.adapt((int32_t)e, p, q) = g.adapt((int32_t)e, p % ns, q / ns);
    x.finalized = true;
}

sn_status select_path(const Graph &g, int32_t method, std::vector<int32_t> &cand_of, int64_t &total) {
    bool fused = false;
    for (const auto &c : g.cands) fused = fused || cand_out(c) != c.schema;
    Graph xg;
    const Graph *pg = &g;
    if (fused) {
        expand_pairs(g, xg);
        pg = &xg;
    }
    std::vector<int32_t> schema_of;
    sn_status rc = method == SN_SELECT_BRUTE ? select_brute(*pg, schema_of, total) : select_dprs(*pg, schema_of, total);
    if (rc != SN_OK) return rc;
    std::vector<int64_t> F;
    std::vector<int32_t> argF;
    fastest_per_schema(*pg, F, argF);
    const int32_t n = pg->n_layers(), ns = pg->n_schemas();
    cand_of.assign(n, -1);
    for (int32_t i = 0; i < n; ++i) {
        cand_of[i] = argF[(size_t)i * ns + schema_of[i]];
        if (cand_of[i] < 0) return fail(SN_EINFEASIBLE, "selected schema has no routine");
    }
    return SN_OK;
}

}  // namespace sn
