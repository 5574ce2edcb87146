"""Writes sample_<workload>.json: the oracle's validity bits for a sample of the
checks of a full benchmark batch (seed 42, the batch bench.py times), so that
a GPU test can run the whole batch in that launch configuration and compare
the sampled checks without running oracle charts of hundreds of tokens
during the test.

Calls only the oracle.  Usage:
    python tests/golden/make_sample_golden.py WORKLOAD "b:j,b:j,..." [procs]
(every candidate of each sampled (sequence, position) pair is checked).
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
    name, b, j, c = args
    import oracle
    from synth import make_workload
    w = make_workload(name, 42)
    O = oracle.Oracle(w.grammar, w.vocab)
    t0 = time.time()
    v = O.validate_batch(w.x[b:b + 1], w.pos[b:b + 1, j:j + 1], w.cand[b:b + 1, j:j + 1, c:c + 1])
    return b, j, c, int(v[0, 0, 0]), round(time.time() - t0, 1)


def main():
    name = sys.argv[1]
    pairs = [tuple(int(v) for v in p.split(':')) for p in sys.argv[2].split(',')]
    procs = int(sys.argv[3]) if len(sys.argv) > 3 else min(8, os.cpu_count() or 1)
    from synth import make_workload
    w = make_workload(name, 42)
    jobs = [(name, b, j, c) for (b, j) in pairs for c in range(w.K)]
    with mp.get_context('spawn').Pool(procs) as pool:
        res = pool.map(_one, jobs, chunksize=1)
    out = dict(workload=name, seed=42, batch=w.B, n=int(w.x.shape[1]), k=w.k, K=w.K,
               checks=[dict(b=b, j=j, c=c, valid=v, oracle_s=s) for (b, j, c, v, s) in res],
               note='oracle validate_batch, one check per call, on the full batch of bench.py')
    path = os.path.join(HERE, 'sample_%s.json' % name)
    with open(path, 'w') as f:
        json.dump(out, f, indent=1)
    print(path)


if __name__ == '__main__':
    main()
