"""Exact optimal-routine-path search for nets too large to enumerate whole.

TEST INFRASTRUCTURE ONLY (see the package docstring).

The problem is Def. 2 / Eq. 2 of the paper: minimise
    T(S) = sum_i F_i(lambda_i) + sum_{(j,i) in E} F^a_{j,i}(lambda_j -> lambda_i)
over schema assignments (void adapt = 0).  `brute_force` in the package
enumerates Lambda^n and is the reference for small nets.  ResNet- and
MobileNet-shaped nets are series compositions of two-terminal blocks
between *articulation* layers (layers every input-to-output path crosses),
so the same minimum is reached by a different exact algorithm:
  1. brute-force every block's interior for each (entry, exit) schema pair;
  2. run a chain dynamic program over the articulation layers.
This is textbook decomposition, deliberately unlike DPRS's constrained
states (section IV-C/D), so agreement between the two is evidence.

Also here: enumeration of the full routine product prod_i |R_i| for tiny
nets, which checks that reducing each layer to F_i(lambda) (Eq. 1) loses
nothing.
"""
from __future__ import annotations

import itertools

import numpy as np

INF = np.iinfo(np.int64).max


def _reach(n, succ, start, banned=-1):
    seen = [False] * n
    if start == banned:
        return seen
    stack = [start]
    seen[start] = True
    while stack:
        u = stack.pop()
        for v in succ[u]:
            if v != banned and not seen[v]:
                seen[v] = True
                stack.append(v)
    return seen


def articulation_layers(n, edges):
    """Layers that every path from layer 0 to layer n-1 passes through."""
    succ = [[] for _ in range(n)]
    for u, v in edges:
        succ[u].append(v)
    arts = []
    for v in range(n):
        if v in (0, n - 1) or not _reach(n, succ, 0, banned=v)[n - 1]:
            arts.append(v)
    return arts


def blockwise_search(layer_cost, edges, adapt_cost, max_interior=16, pairs=None):
    """Exact min of T(S) by block brute force + chain DP.

    layer_cost: int64 [n, ns] of F_i(lambda) (INF where infeasible);
    edges: (src, dst) pairs; adapt_cost: int64 [n_edges, ns, ns].
    Returns (cost, assignment).  Raises ValueError if a block is too large.

    pairs (routines that write a schema other than the one they read): the
    states of a layer are then the (read, written) schema pairs pairs[k] and
    layer_cost is [n, len(pairs)]; an edge (u, v) costs the adapt from u's
    written schema to v's read schema, nothing when they agree (Def. 1 read
    for fused boundaries).  adapt_cost stays indexed by schemas.
    """
    lc = np.asarray(layer_cost, dtype=np.int64)
    n, ns = lc.shape
    edges = [tuple(map(int, e)) for e in np.asarray(edges).reshape(-1, 2)]
    ac = np.asarray(adapt_cost, dtype=np.int64)
    nsch = ns if pairs is None else ac.shape[-1]
    ac = ac.reshape(len(edges), nsch, nsch)
    succ = [[] for _ in range(n)]
    for u, v in edges:
        succ[u].append(v)
    arts = articulation_layers(n, edges)  # ascending = topological along the chain
    pos = {a: k for k, a in enumerate(arts)}

    def add(a, b):
        return INF if a == INF or b == INF else a + b

    def adapt(e, x, y):
        if pairs is not None:
            x, y = pairs[x][1], pairs[y][0]  # written by the producer, read by the consumer
        return 0 if x == y else int(ac[e, x, y])

    # assign every layer and edge to the block that contains it
    fwd0 = _reach(n, succ, 0)
    blocks = []  # (entry, exit, interior layers, edge ids)
    for k in range(len(arts) - 1):
        a, b = arts[k], arts[k + 1]
        from_a = _reach(n, succ, a)
        interior = [v for v in range(a + 1, b) if from_a[v] and v not in pos]
        blocks.append((a, b, interior, []))
    block_of_layer = {}
    for k, (a, b, interior, _) in enumerate(blocks):
        for v in interior:
            block_of_layer[v] = k
    for e, (u, v) in enumerate(edges):
        if v in pos:
            k = pos[v] - 1
        else:
            k = block_of_layer[v]
        blocks[k][3].append(e)
    if not all(fwd0):
        raise ValueError("net has layers unreachable from the input")

    # 1. block tables B_k[x, y] and their argmin interiors
    tables = []
    for a, b, interior, eids in blocks:
        if len(interior) > max_interior:
            raise ValueError("block interior too large for brute force")
        idx = {v: t for t, v in enumerate(interior)}
        B = np.full((ns, ns), INF, dtype=np.int64)
        arg = {}
        for x in range(ns):
            for y in range(ns):
                best, best_asg = INF, None
                # only states a layer can take (finite F): the others give INF anyway
                for asg in itertools.product(*[[z for z in range(ns) if lc[v, z] < INF] for v in interior]):
                    t = 0
                    for v, lam in zip(interior, asg):
                        t = add(t, int(lc[v, lam]))
                    for e in eids:
                        u, v = edges[e]
                        lu = x if u == a else asg[idx[u]]
                        lv = y if v == b else asg[idx[v]]
                        t = add(t, adapt(e, lu, lv))
                    if t < best:
                        best, best_asg = t, asg
                B[x, y] = best
                arg[(x, y)] = best_asg
        tables.append((B, arg))

    # 2. chain DP over articulation layers
    D = np.array([int(lc[arts[0], x]) for x in range(ns)], dtype=object)
    back = []
    for k in range(1, len(arts)):
        B, _ = tables[k - 1]
        Dn = [INF] * ns
        bk = [0] * ns
        for y in range(ns):
            for x in range(ns):
                t = add(add(int(D[x]), int(B[x, y])), int(lc[arts[k], y]))
                if t < Dn[y]:
                    Dn[y], bk[y] = t, x
        back.append(bk)
        D = Dn
    y = int(np.argmin([d if d != INF else np.iinfo(np.int64).max for d in D]))
    cost = int(D[y])
    assign = np.zeros(n, np.int32)
    if cost == INF:
        return INF, assign
    for k in range(len(arts) - 1, 0, -1):
        x = back[k - 1][y]
        assign[arts[k]] = y
        a, b, interior, _ = blocks[k - 1]
        asg = tables[k - 1][1][(x, y)]
        for v, lam in zip(interior, asg):
            assign[v] = lam
        y = x
    assign[arts[0]] = y
    return cost, assign


def full_routine_product(cands, edges, adapt_cost, ns):
    """min over every routine combination (not reduced to F_i) of T(S).

    cands[i] = list of (schema, cost) for layer i.  Tiny nets only.
    """
    edges = [tuple(map(int, e)) for e in np.asarray(edges).reshape(-1, 2)]
    ac = np.asarray(adapt_cost, dtype=np.int64).reshape(len(edges), ns, ns)
    best = INF
    for combo in itertools.product(*[range(len(c)) for c in cands]):
        t = 0
        for i, j in enumerate(combo):
            c = cands[i][j][1]
            t = INF if (t == INF or c == INF) else t + c
        for e, (u, v) in enumerate(edges):
            su, sv = cands[u][combo[u]][0], cands[v][combo[v]][0]
            if su != sv:
                c = int(ac[e, su, sv])
                t = INF if (t == INF or c == INF) else t + c
        best = min(best, t)
    return best


def brute_force_candidates(cands, edges, adapt_cost):
    """Exact optimum when a routine may write a schema other than the one it
    reads (a fused boundary): enumerate one candidate per layer, with
    T = sum of candidate times + sum over edges (u, v) of the adapt from u's
    written schema to v's read schema (0 when they agree).

    cands: per layer a list of (cost, read_schema, written_schema); adapt_cost
    [n_edges, ns, ns].  Returns (T*, [chosen index per layer]) — the first
    minimum in lexicographic order of the choices; INF when none is finite.
    """
    n = len(cands)
    best, best_pick = INF, None
    for pick in itertools.product(*[range(len(c)) for c in cands]):
        t = 0
        for i, k in enumerate(pick):
            t = INF if cands[i][k][0] >= INF else t + int(cands[i][k][0])
            if t >= INF:
                break
        if t >= INF:
            continue
        for e, (u, v) in enumerate(edges):
            w, r = cands[u][pick[u]][2], cands[v][pick[v]][1]
            if w != r:
                a = int(adapt_cost[e][w][r])
                if a >= INF:
                    t = INF
                    break
                t += a
        if t < best:
            best, best_pick = t, list(pick)
    return best, best_pick

