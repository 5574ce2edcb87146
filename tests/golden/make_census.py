"""Writes census_<workload>.json: the oracle's count of the exact Earley chart
of each sampled sequence x of a benchmark batch (Alg. 3 run to its fixpoint
over the whole partial-output graph of x, not stopped at acceptance): graph
nodes, gap nodes, (node, origin) pairs holding at least one item, and items.
The benchmark's roofline takes its algorithmic work from these counts (a
forward chart stores one item bitset of ceil(D/32) words per (node, origin)
pair), never from the kernels' own counters.

With --checks it also counts the chart of every check x (+) (i, t) of the
batch (the whole-graph walks compute exactly those charts); only for
workloads whose charts are small.

Calls only the oracle.  Usage:
    python tests/golden/make_census.py WORKLOAD [n_sample] [procs] [--checks]
"""
import json
import multiprocessing as mp
import os
import sys
import time

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(os.path.dirname(HERE))
sys.path.insert(0, ROOT)


def _one(args):
    name, seed, b = args
    import numpy as np
    import oracle
    from synth import make_workload
    w = make_workload(name, seed)
    O = oracle.Oracle(w.grammar, w.vocab)
    t0 = time.time()
    items, origins, gap = O.chart_census(w.x[b])
    return dict(b=int(b), nodes=int(len(items)), gaps=int(gap.sum()), pairs=int(origins.sum()),
                items=int(items.sum()), max_origins=int(origins.max(initial=0)),
                oracle_s=round(time.time() - t0, 1))


def _checks(args):
    name, seed, b = args
    import oracle
    from synth import make_workload
    w = make_workload(name, seed)
    O = oracle.Oracle(w.grammar, w.vocab)
    pairs = 0
    for j in range(w.k):
        for c in range(w.K):
            y = w.x[b].copy()
            y[w.pos[b, j]] = w.cand[b, j, c]
            items, origins, gap = O.chart_census(y)
            pairs += int(origins.sum())
    return pairs


def reduced_items(g):
    """Dotted items (sum of |rhs| + 1, plus S' -> S) of the grammar reduced to
    its useful productions: a nonterminal is productive when some production
    of it has only terminals and productive nonterminals on its right side,
    reachable when the start symbol reaches it through productive
    productions; only productions with a reachable left side and a productive
    right side take part in any derivation."""
    T = g.T
    prods = g.productions
    productive = set()
    changed = True
    while changed:
        changed = False
        for lhs, rhs in prods:
            if lhs not in productive and all(s < T or (s - T) in productive for s in rhs):
                productive.add(lhs)
                changed = True
    useful = [(lhs, rhs) for lhs, rhs in prods if lhs in productive and all(s < T or (s - T) in productive for s in rhs)]
    reach = {g.start}
    changed = True
    while changed:
        changed = False
        for lhs, rhs in useful:
            if lhs in reach:
                for s in rhs:
                    if s >= T and (s - T) not in reach:
                        reach.add(s - T)
                        changed = True
    return sum(len(rhs) + 1 for lhs, rhs in useful if lhs in reach) + 2


def main():
    argv = [a for a in sys.argv[1:] if not a.startswith('--')]
    with_checks = '--checks' in sys.argv
    name = argv[0]
    n_sample = int(argv[1]) if len(argv) > 1 else 8
    procs = int(argv[2]) if len(argv) > 2 else min(8, os.cpu_count() or 1)
    seed = 42
    from synth import make_workload
    w = make_workload(name, seed)
    g = w.grammar
    D = reduced_items(g)
    B = w.B
    sample = list(range(min(n_sample, B)))
    checks_pairs = None
    with mp.get_context('spawn').Pool(procs) as pool:
        per = pool.map(_one, [(name, seed, b) for b in sample])
        if with_checks:
            checks_pairs = sum(pool.map(_checks, [(name, seed, b) for b in range(B)]))
    out = dict(workload=name, seed=seed, batch=B, n=int(w.x.shape[1]), D=D, words=(D + 31) // 32,
               sampled=sample, per_seq=per,
               note='oracle chart census of x per sampled sequence; batch totals scale the sample mean by '
                    'batch / len(sampled)')
    if checks_pairs is not None:
        out['checks_pairs'] = checks_pairs
        out['checks'] = int(B * w.k * w.K)
    path = os.path.join(HERE, 'census_%s.json' % name)
    with open(path, 'w') as f:
        json.dump(out, f, indent=1)
    print(path)


if __name__ == '__main__':
    main()
