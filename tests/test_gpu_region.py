"""GPU parity of the checks by region (one forward chart and good-item masks
per sequence, then only each candidate's region walked per check) against the
oracle, bit-exact.  The region path is the default for wide item sets; here
it is also forced on the small grammars, whose every position shape (runs of
one mask between spans, leading and trailing runs, dead lexings, candidates
at the first and last position) the tests below cover."""
import os

import numpy as np
import pytest

import oracle
from synth import grammars as G
from synth import make_workload

from test_gpu_edges import rows_with_all_positions, run_gpu, words_grammar

pytestmark = pytest.mark.gpu
NTHREADS = os.cpu_count() or 1


@pytest.fixture
def region(monkeypatch):
    monkeypatch.setenv('EPIC_REGION', '1')


@pytest.mark.parametrize('gname', ['expr', 'words'])
def test_region_random_rows(cuda, region, gname):
    """Short random rows (mostly not completable: every check of such a row is
    0 without a walk) with every masked position proposed."""
    spec = G.expr_grammar() if gname == 'expr' else words_grammar()
    extra = ['1+', '(2', '3)', '*(', ' 4', '^-'] if gname == 'expr' else ['if', '<<', 'a ', '1.', 'f<', '<<=']
    vocab = list(dict.fromkeys([c.encode() for c in sorted(set(spec.charset))] + [e.encode() for e in extra]))
    rng = np.random.default_rng(23)
    O = oracle.Oracle(spec, vocab)
    for n in (1, 2, 3, 5, 9, 14):
        X, P = rows_with_all_positions(rng, len(vocab), n, 0.45, 6)
        cand = rng.integers(0, len(vocab), (X.shape[0], P.shape[1], 6)).astype(np.int32)
        got, st = run_gpu(spec, vocab, X, P, cand, cuda)
        assert st['overflow'] == 0
        np.testing.assert_array_equal(got, O.validate_batch(X, P, cand, nthreads=NTHREADS))


@pytest.mark.parametrize('path', ['region', 'walk'])
@pytest.mark.parametrize('name,n', [('expr-tiny', 32), ('json-schema', 40), ('json-schema', 96),
                                    ('smiles-256', 48)])
def test_every_masked_position(cuda, monkeypatch, path, name, n):
    """Completable rows (masked witnesses) with EVERY masked position proposed:
    candidates at the first and last position, inside long runs, at both ends
    of a run and in runs of one; the witness's own token is among them.  Both
    the checks by region and the whole-graph walks."""
    monkeypatch.setenv('EPIC_REGION', '1' if path == 'region' else '0')
    w = make_workload(name, 11, batch=4, n=n)
    rng = np.random.default_rng(5)
    masks = [np.flatnonzero(w.x[b] < 0) for b in range(w.B)]
    k = max(len(m) for m in masks)
    K = 6
    P = np.zeros((w.B, k), np.int32)
    cand = rng.integers(0, len(w.vocab), (w.B, k, K)).astype(np.int32)
    for b, m in enumerate(masks):
        P[b, :len(m)] = m
        P[b, len(m):] = m[0]
        wt = w.witness[b, P[b]]  # -1 on the masked padding after the witness
        cand[b, :, 0] = np.where(wt >= 0, wt, cand[b, :, 0])
    has_witness = np.stack([w.witness[b, P[b]] >= 0 for b in range(w.B)])
    got, st = run_gpu(w.grammar, w.vocab, w.x, P, cand, cuda)
    assert st['overflow'] == 0
    ref = oracle.Oracle(w.grammar, w.vocab).validate_batch(w.x, P, cand, nthreads=NTHREADS)
    np.testing.assert_array_equal(got, ref)
    assert ref[:, :, 0][has_witness].all(), 'the witness token is always a valid single update'


@pytest.mark.parametrize('name,seed,kw', [
    ('expr-tiny', 42, {}), ('expr-tiny', 45, {}),
    ('json-schema', 42, dict(batch=4)), ('json-schema', 46, dict(batch=3, k=3)),
    ('smiles-256', 42, dict(batch=6, k=4)),
])
def test_region_workload_parity(cuda, region, name, seed, kw):
    w = make_workload(name, seed, **kw)
    got, st = run_gpu(w.grammar, w.vocab, w.x, w.pos, w.cand, cuda)
    ref = oracle.Oracle(w.grammar, w.vocab).validate_batch(w.x, w.pos, w.cand, nthreads=NTHREADS)
    assert st['overflow'] == 0
    np.testing.assert_array_equal(got, ref)
    assert ref.any(), 'the case should hold valid candidates'


def test_region_json_full_batch(cuda, region):
    """The json-schema benchmark batch (16 x 256, k = 4, K = 16) by regions."""
    w = make_workload('json-schema', 42)
    got, st = run_gpu(w.grammar, w.vocab, w.x, w.pos, w.cand, cuda)
    assert st['overflow'] == 0
    ref = oracle.Oracle(w.grammar, w.vocab).validate_batch(w.x, w.pos, w.cand, nthreads=NTHREADS)
    np.testing.assert_array_equal(got, ref)


@pytest.mark.parametrize('name,seed,kw', [
    ('clike-512', 42, dict(batch=2, k=4, K=8)),
    ('clike-512', 43, dict(batch=2, k=4, K=8, n=128)),
    ('random-stress-1024', 42, dict(batch=2, k=4, K=4, n=96)),
])
def test_wide_grammars_by_region(cuda, name, seed, kw):
    """Wide item sets take the region path by default."""
    w = make_workload(name, seed, **kw)
    got, st = run_gpu(w.grammar, w.vocab, w.x, w.pos, w.cand, cuda)
    assert st['overflow'] == 0
    ref = oracle.Oracle(w.grammar, w.vocab).validate_batch(w.x, w.pos, w.cand, nthreads=NTHREADS)
    np.testing.assert_array_equal(got, ref)


def test_clike_full_length_row(cuda):
    """clike-512 at its full row length (512 tokens) on one row, 4 positions x
    8 candidates, by region (the default for its item width), against the
    oracle."""
    w = make_workload('clike-512', 44, batch=1, k=4, K=8)
    got, st = run_gpu(w.grammar, w.vocab, w.x, w.pos, w.cand, cuda)
    assert st['overflow'] == 0
    assert st['region_checks'] == w.cand.size
    ref = oracle.Oracle(w.grammar, w.vocab).validate_batch(w.x, w.pos, w.cand, nthreads=NTHREADS)
    np.testing.assert_array_equal(got, ref)


def test_random_stress_full_length_row(cuda):
    """random-stress-1024 (400 nonterminals, 1,500 productions, 213 item words)
    on a whole 1,024-token row: 4 positions x 4 candidates, the row's witness
    token among them, against the oracle's bits stored by
    tests/golden/make_stress_golden.py (an oracle chart of a thousand tokens
    takes up to tens of minutes, too long to run here)."""
    import json
    here = os.path.dirname(os.path.abspath(__file__))
    with open(os.path.join(here, 'golden', 'stress1024_checks.json')) as f:
        gold = json.load(f)
    c = gold['case']
    w = make_workload(c['name'], c['seed'], batch=c['batch'], k=c['k'], K=c['K'])
    pos = np.array([gold['pos']], np.int32)
    cand = np.array([gold['cand']], np.int32)
    assert np.array_equal(pos, w.pos)
    got, st = run_gpu(w.grammar, w.vocab, w.x, pos, cand, cuda)
    assert st['overflow'] == 0
    assert st['region_checks'] == cand.size
    np.testing.assert_array_equal(got[0], np.array(gold['valid'], np.uint8))


def test_clike_full_batch_sampled(cuda):
    """The clike-512 benchmark batch (32 x 512, k = 8, K = 32) in one
    epic_validate_batch call, the launch bench.py times, against the oracle's
    bits for a sample of 128 of its checks (every candidate of four
    (sequence, position) pairs), stored by tests/golden/make_sample_golden.py
    (the whole batch is about 8,000 oracle checks of 512-token rows)."""
    import json
    here = os.path.dirname(os.path.abspath(__file__))
    with open(os.path.join(here, 'golden', 'sample_clike-512.json')) as f:
        gold = json.load(f)
    w = make_workload(gold['workload'], gold['seed'])
    assert (w.B, w.x.shape[1], w.k, w.K) == (gold['batch'], gold['n'], gold['k'], gold['K'])
    got, st = run_gpu(w.grammar, w.vocab, w.x, w.pos, w.cand, cuda)
    assert st['overflow'] == 0
    assert st['checks'] == w.cand.size
    for c in gold['checks']:
        assert got[c['b'], c['j'], c['c']] == c['valid'], c
    assert any(c['valid'] for c in gold['checks']) and not all(c['valid'] for c in gold['checks'])
