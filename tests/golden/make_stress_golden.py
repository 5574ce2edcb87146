"""Writes stress1024_checks.json: the oracle's validity bits for a sample of
full-length checks of the random-stress-1024 workload (one 1,024-token row,
a few proposed positions x K candidates, the row's witness token among
them), so that the GPU test can compare against them without running oracle
charts of a thousand tokens (tens of minutes each on one core).

Calls only the oracle.  Usage:
    python tests/golden/make_stress_golden.py [procs]
"""
import json
import multiprocessing as mp
import os
import sys
import time

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(os.path.dirname(HERE))
sys.path.insert(0, ROOT)

CASE = dict(name='random-stress-1024', seed=42, batch=1, k=4, K=4)


def rows():
    """The row, its proposed positions and candidates (witness first)."""
    import numpy as np
    from synth import make_workload
    w = make_workload(CASE['name'], CASE['seed'], batch=CASE['batch'], k=CASE['k'], K=CASE['K'])
    cand = w.cand.copy()
    for j in range(w.k):
        wt = w.witness[0, w.pos[0, j]]
        if wt >= 0 and wt not in cand[0, j]:
            cand[0, j, 0] = wt
    return w, cand


def _one(args):
    j, c = args
    import numpy as np
    import oracle
    w, cand = rows()
    O = oracle.Oracle(w.grammar, w.vocab)
    t0 = time.time()
    v = O.validate_batch(w.x, w.pos[:, j:j + 1], cand[:, j:j + 1, c:c + 1])
    return j, c, int(v[0, 0, 0]), round(time.time() - t0, 1)


def main():
    procs = int(sys.argv[1]) if len(sys.argv) > 1 else min(8, os.cpu_count() or 1)
    w, cand = rows()
    jobs = [(j, c) for j in range(w.k) for c in range(w.K)]
    with mp.get_context('spawn').Pool(procs) as pool:
        res = pool.map(_one, jobs)
    valid = [[0] * w.K for _ in range(w.k)]
    secs = {}
    for j, c, v, s in res:
        valid[j][c] = v
        secs['%d,%d' % (j, c)] = s
    out = dict(case=CASE, pos=w.pos[0].tolist(), cand=cand[0].tolist(), valid=valid, oracle_seconds=secs,
               note='oracle validate_batch, one check per call; candidates with the witness token first')
    path = os.path.join(HERE, 'stress1024_checks.json')
    with open(path, 'w') as f:
        json.dump(out, f, indent=1)
    print(path)


if __name__ == '__main__':
    main()
